// whtmix_noalloc.cu -- a forward entry point that allocates no device memory.
//
// Who needs this: code that must not call cudaMalloc / cudaMallocAsync while it runs -- for
// example a host whose memory budget is fixed up front by an outside allocator or framework that
// forbids other allocations, a real-time loop where an allocation could block or fail at the
// worst moment, or a plugin that is handed only input and output buffers.  The plain
// whtmix_forward allocates its workspace the first time it sees a stream, and whtmix_forward_ex
// needs the caller to own a workspace; this entry point needs neither.
//
// How: the scratch the forward kernels keep between their phases (a device-wide barrier header
// and a plane group of fp32 intermediates) lives in one fixed array in device memory, defined
// below.  Every device that loads this library holds that array until the process exits, whether
// or not this entry point is ever called.  The call runs exactly the kernels whtmix_forward picks
// for the shape, with plane groups limited to what the array holds, so its results are the same
// bit for bit.  All calls share the array, so two calls whose kernels overlap on a GPU (different
// streams, or different host threads) race on it; order them on one stream.
#include <cuda_runtime.h>

#include <map>
#include <mutex>

#include "whtmix.h"
#include "whtmix_kernels.cuh"

// Fixed scratch: a 256-byte device-wide barrier header followed by 16 MiB of fp32 / uint32
// plane-group workspace (4 Mi elements: planes of up to N*C = 2^22 elements).
#define WHTMIX_NOALLOC_HEADER_BYTES 256
#define WHTMIX_NOALLOC_DATA_BYTES (16u << 20)
static __device__ __align__(256) unsigned char g_noalloc_scratch[WHTMIX_NOALLOC_HEADER_BYTES + WHTMIX_NOALLOC_DATA_BYTES];

namespace whtmix {
// whtmix_capi.cu: the forward with a fixed scratch as its workspace
int forward_in_fixed_scratch(const void* x, const void* gains, void* y, int64_t B, int64_t N, int64_t C, int dtype,
                             void* scratch, size_t scratch_bytes, void* stream);
}  // namespace whtmix

namespace {

std::mutex g_noalloc_mu;
std::map<int, void*> g_noalloc_addr;  // device -> device address of g_noalloc_scratch

// In host code g_noalloc_scratch names a host-side stand-in, not device memory, so its device
// address is looked up once per device (with that device current) and cached.  The array starts
// zeroed, like every device variable without an initializer, so its barrier header is ready.
int noalloc_setup(void** scratch_out) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return WHTMIX_ERR_NO_DEVICE;
  std::lock_guard<std::mutex> lk(g_noalloc_mu);
  auto it = g_noalloc_addr.find(dev);
  if (it == g_noalloc_addr.end()) {
    int major = 0, minor = 0;
    if (cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev) != cudaSuccess)
      return WHTMIX_ERR_CUDA;
    if (major != 10 || minor != 3) return WHTMIX_ERR_NO_DEVICE;
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_noalloc_scratch) != cudaSuccess || p == nullptr) return WHTMIX_ERR_CUDA;
    it = g_noalloc_addr.emplace(dev, p).first;
  }
  *scratch_out = it->second;
  return WHTMIX_OK;
}

}  // namespace

namespace whtmix {
// Read by whtmix_sync: the fixed scratch of device `dev` once a call has set it up there.
void* noalloc_scratch_of(int dev) {
  std::lock_guard<std::mutex> lk(g_noalloc_mu);
  auto it = g_noalloc_addr.find(dev);
  return it == g_noalloc_addr.end() ? nullptr : it->second;
}
}  // namespace whtmix

extern "C" WHTMIX_API int whtmix_forward_noalloc(const void* x, const void* gains, void* y, int64_t B, int64_t N,
                                                 int64_t C, int dtype, void* stream) {
  // The argument checks (shape, dtype, pointers, aliasing, scratch size) run in the shared path
  // before anything is enqueued; only a valid call reaches the device.  A shape that is invalid
  // for every entry point is rejected here before the scratch is looked up, so such a call needs
  // no device at all.
  if (B < 0 || N < 1 || C < 1) return WHTMIX_ERR_INVALID_ARG;
  if (dtype != WHTMIX_F32 && dtype != WHTMIX_BF16 && dtype != WHTMIX_I32) return WHTMIX_ERR_BAD_DTYPE;
  if ((N & (N - 1)) || (C & (C - 1))) return WHTMIX_ERR_BAD_SHAPE;
  int n_bits = 0, c_bits = 0;
  while ((int64_t{1} << n_bits) < N) ++n_bits;
  while ((int64_t{1} << c_bits) < C) ++c_bits;
  const int m = n_bits + c_bits;  // log2(N C) without forming the product (it could overflow)
  if (m > whtmix::MAX_PLANE_BITS || B > (int64_t{1} << (60 - m))) return WHTMIX_ERR_BAD_SHAPE;
  if (m > whtmix::TILE_BITS && (size_t{4} << m) > WHTMIX_NOALLOC_DATA_BYTES) return WHTMIX_ERR_WORKSPACE;
  if (B == 0) return WHTMIX_OK;
  void* scratch = nullptr;
  const int rc = noalloc_setup(&scratch);
  if (rc != WHTMIX_OK) return rc;
  return whtmix::forward_in_fixed_scratch(x, gains, y, B, N, C, dtype, scratch,
                                          WHTMIX_NOALLOC_HEADER_BYTES + WHTMIX_NOALLOC_DATA_BYTES, stream);
}
