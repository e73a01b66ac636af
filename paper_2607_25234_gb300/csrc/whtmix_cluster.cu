// Cluster forward, host-side launcher, fp32 and bf16 I/O.  Instantiated for planes of 2^14 .. 2^16
// elements (clusters of 1 or 2 CTAs); the kernel is written for up to 2^19 (clusters of 16), where
// the three-phase kernel measured faster.
#include <cuda_runtime.h>

#include <map>
#include <mutex>

#include "whtmix_cluster.cuh"

namespace whtmix {
namespace clu {

// Per device and kernel: raise the dynamic shared memory limit (and allow 16-CTA clusters) once,
// and check that at least one cluster fits on the device.
inline cudaError_t prepare(const void* k, int cluster) {
  static std::mutex mu;
  static std::map<std::pair<int, const void*>, cudaError_t> done;
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  std::lock_guard<std::mutex> lk(mu);
  auto it = done.find({dev, k});
  if (it != done.end()) return it->second;
  e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(SMEM_BYTES));
  if (e == cudaSuccess && cluster > 8) e = cudaFuncSetAttribute(k, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
  if (e == cudaSuccess) {
    cudaLaunchConfig_t cfg = {};
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = static_cast<unsigned>(cluster);
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.gridDim = dim3(static_cast<unsigned>(cluster));
    cfg.blockDim = dim3(THREADS);
    cfg.dynamicSmemBytes = SMEM_BYTES;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    int n = 0;
    e = cudaOccupancyMaxActiveClusters(&n, k, &cfg);
    if (e == cudaSuccess && n < 1) e = cudaErrorInvalidConfiguration;
  }
  done[{dev, k}] = e;
  return e;
}

template <int D, int CB>
cudaError_t launch_cb(const Params& P, cudaStream_t stream) {
  constexpr int NR = 1 << CB;
  constexpr int K = NR > 1 ? NR / 2 : 1;
  const void* k = reinterpret_cast<const void*>(k_forward_cluster<D, CB>);
  cudaError_t e = prepare(k, K);
  if (e != cudaSuccess) return e;
  cudaLaunchConfig_t cfg = {};
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = K;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.gridDim = dim3(static_cast<unsigned>(P.B * K));
  cfg.blockDim = dim3(THREADS);
  cfg.dynamicSmemBytes = SMEM_BYTES;
  cfg.stream = stream;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, k_forward_cluster<D, CB>, P);
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

template <int D>
bool usable_d(int m) {
  switch (m) {
    case 14: return prepare(reinterpret_cast<const void*>(k_forward_cluster<D, 0>), 1) == cudaSuccess;
    case 15: return prepare(reinterpret_cast<const void*>(k_forward_cluster<D, 1>), 1) == cudaSuccess;
    case 16: return prepare(reinterpret_cast<const void*>(k_forward_cluster<D, 2>), 2) == cudaSuccess;
    default: return false;
  }
}
bool usable(int m, bool bf16) { return bf16 ? usable_d<DT_BF16>(m) : usable_d<DT_F32>(m); }

}  // namespace clu
}  // namespace whtmix
