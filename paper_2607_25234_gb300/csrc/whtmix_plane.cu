// One-plane-per-CTA forward (planes of 2^14 .. 2^16 elements in tensor memory): host-side launcher,
// fp32 and bf16 I/O.
#include <cuda_runtime.h>

#include <map>
#include <mutex>

#include "whtmix_plane.cuh"

namespace whtmix {
namespace pln {

// Per device and kernel: raise the dynamic shared memory limit once.
inline cudaError_t prepare(const void* k) {
  static std::mutex mu;
  static std::map<std::pair<int, const void*>, cudaError_t> done;
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  std::lock_guard<std::mutex> lk(mu);
  auto it = done.find({dev, k});
  if (it != done.end()) return it->second;
  e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(SMEM_BYTES));
  done[{dev, k}] = e;
  return e;
}

template <int D, int CB>
cudaError_t launch_cb(const Params& P, cudaStream_t stream) {
  const void* k = reinterpret_cast<const void*>(k_forward_plane<D, CB>);
  cudaError_t e = prepare(k);
  if (e != cudaSuccess) return e;
  Params p = P;
  void* args[] = {&p};
  return launch_pdl(k, static_cast<unsigned>(P.B), THREADS, SMEM_BYTES, stream, args);
}

template <int D>
cudaError_t launch(const Params& P, cudaStream_t stream) {
  switch (P.m) {
    case 14: return launch_cb<D, 0>(P, stream);
    case 15: return launch_cb<D, 1>(P, stream);
    case 16: return launch_cb<D, 2>(P, stream);
    default: return cudaErrorInvalidValue;
  }
}

cudaError_t forward_f32(const Params& P, cudaStream_t stream) { return launch<DT_F32>(P, stream); }
cudaError_t forward_bf16(const Params& P, cudaStream_t stream) { return launch<DT_BF16>(P, stream); }

}  // namespace pln
}  // namespace whtmix
