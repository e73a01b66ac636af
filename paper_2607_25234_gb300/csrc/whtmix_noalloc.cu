// whtmix_noalloc.cu -- a forward entry point that allocates no device memory.
//
// Who needs this: code that must not call cudaMalloc / cudaMallocAsync while it runs -- for
// example a host whose memory budget is fixed up front by an outside allocator or framework that
// forbids other allocations, a real-time loop where an allocation could block or fail at the
// worst moment, or a plugin that is handed only input and output buffers.  The plain
// whtmix_forward allocates its workspace the first time it sees a stream, and whtmix_forward_ex
// needs the caller to own a workspace; this entry point needs neither.
//
// How: the scratch that the three-phase forward kernel (k_forward_m) keeps between its phases
// lives in one fixed array in device memory, defined below.  Every device that loads this library
// holds that array until the process exits, whether or not this entry point is ever called.
// All calls share it, so two calls whose kernels overlap on a GPU (different streams, or
// different host threads) race on it; order them on one stream.
#include <cuda_runtime.h>

#include <map>
#include <mutex>

#include "whtmix.h"
#include "whtmix_kernels.cuh"

// Fixed scratch: a 256-byte device-wide barrier header followed by 16 MiB of fp32 / uint32
// plane-group workspace (4 Mi elements: planes of up to N*C = 2^22 elements, one plane at a time).
#define WHTMIX_NOALLOC_HEADER_BYTES 256
#define WHTMIX_NOALLOC_DATA_BYTES (16u << 20)
static __device__ __align__(256) unsigned char g_noalloc_scratch[WHTMIX_NOALLOC_HEADER_BYTES + WHTMIX_NOALLOC_DATA_BYTES];

using namespace whtmix;

namespace {

std::mutex g_noalloc_mu;
std::map<int, void*> g_noalloc_addr;  // device -> device address of g_noalloc_scratch
std::map<int, int> g_noalloc_sms;      // device -> SM count (0: not an sm_103 device)

// In host code g_noalloc_scratch names a host-side stand-in, not device memory, so its device
// address is looked up once per device (with that device current) and cached.
int noalloc_setup(int* dev_out, void** scratch_out, int* sms_out) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return WHTMIX_ERR_NO_DEVICE;
  std::lock_guard<std::mutex> lk(g_noalloc_mu);
  auto it = g_noalloc_addr.find(dev);
  if (it == g_noalloc_addr.end()) {
    int major = 0, minor = 0, sms = 0;
    if (cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
      return WHTMIX_ERR_CUDA;
    if (major != 10 || minor != 3) return WHTMIX_ERR_NO_DEVICE;
    void* p = nullptr;
    e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
    if (e != cudaSuccess || p == nullptr) return WHTMIX_ERR_CUDA;
    it = g_noalloc_addr.emplace(dev, p).first;
    g_noalloc_sms[dev] = sms;
  }
  *dev_out = dev;
  *scratch_out = it->second;
  *sms_out = g_noalloc_sms[dev];
  return WHTMIX_OK;
}

bool pow2(int64_t v) { return v > 0 && (v & (v - 1)) == 0; }

template <class K>
int noalloc_launch(K kernel, bool cooperative, int sms, long long max_units, const Params& P, cudaStream_t stream) {
  int occ = 0;
  if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&occ, kernel, THREADS, TILE * 4) != cudaSuccess || occ < 1)
    return WHTMIX_ERR_CUDA;
  long long grid = static_cast<long long>(occ) * sms;
  if (max_units < grid) grid = max_units < 1 ? 1 : max_units;
  Params p = P;
  void* args[] = {&p};
  const cudaError_t e = cooperative
      ? cudaLaunchCooperativeKernel(reinterpret_cast<const void*>(kernel), dim3(static_cast<unsigned>(grid)), dim3(THREADS), args, TILE * 4, stream)
      : cudaLaunchKernel(reinterpret_cast<const void*>(kernel), dim3(static_cast<unsigned>(grid)), dim3(THREADS), args, TILE * 4, stream);
  return e == cudaSuccess ? WHTMIX_OK : WHTMIX_ERR_CUDA;
}

template <int D>
int noalloc_dispatch(const Params& P, int sms, cudaStream_t stream) {
  if (P.m <= TILE_BITS) {
    const long long ppt = 1ll << (TILE_BITS - P.m);
    return noalloc_launch(k_forward_s<D>, false, sms, (P.B + ppt - 1) / ppt, P, stream);
  }
  return noalloc_launch(k_forward_m<D>, true, sms, static_cast<long long>(P.gp) << (P.m - TILE_BITS), P, stream);
}

}  // namespace

extern "C" WHTMIX_API int whtmix_forward_noalloc(const void* x, const void* gains, void* y, int64_t B, int64_t N,
                                                 int64_t C, int dtype, void* stream_v) {
  if (B < 0 || N < 1 || C < 1) return WHTMIX_ERR_INVALID_ARG;
  if (dtype != WHTMIX_F32 && dtype != WHTMIX_BF16 && dtype != WHTMIX_I32) return WHTMIX_ERR_BAD_DTYPE;
  if (!pow2(N) || !pow2(C)) return WHTMIX_ERR_BAD_SHAPE;
  int m = 0;
  while ((int64_t{1} << m) < N * C) ++m;
  if (m > MAX_PLANE_BITS || B > (int64_t{1} << (60 - m))) return WHTMIX_ERR_BAD_SHAPE;
  const size_t plane_ws = (size_t{1} << m) * 4;
  if (m > TILE_BITS && plane_ws > WHTMIX_NOALLOC_DATA_BYTES) return WHTMIX_ERR_WORKSPACE;
  if (B == 0) return WHTMIX_OK;
  if (!x || !gains || !y) return WHTMIX_ERR_INVALID_ARG;
  const uintptr_t px = reinterpret_cast<uintptr_t>(x), pg = reinterpret_cast<uintptr_t>(gains),
                  py = reinterpret_cast<uintptr_t>(y);
  if ((px | pg | py) & 15u) return WHTMIX_ERR_MISALIGNED;
  const size_t nb = static_cast<size_t>(B) * (size_t{1} << m) * (dtype == WHTMIX_BF16 ? 2 : 4);
  const size_t gb = (size_t{1} << m) * 4;
  if ((py != px && py < px + nb && px < py + nb) || (py < pg + gb && pg < py + nb)) return WHTMIX_ERR_ALIAS;

  int dev = 0, sms = 0;
  void* scratch = nullptr;
  int rc = noalloc_setup(&dev, &scratch, &sms);
  if (rc != WHTMIX_OK) return rc;
  cudaStream_t stream = static_cast<cudaStream_t>(stream_v);

  Params P{};
  P.x = x;
  P.g = gains;
  P.y = y;
  P.B = B;
  P.m = m;
  P.scale = 1.0f / static_cast<float>(size_t{1} << m);
  P.bar = static_cast<GridBarrier*>(scratch);
  P.ws = static_cast<unsigned char*>(scratch) + WHTMIX_NOALLOC_HEADER_BYTES;
  long long gp = m > TILE_BITS ? static_cast<long long>(WHTMIX_NOALLOC_DATA_BYTES / plane_ws) : 1;
  if (gp > B) gp = B;
  P.gp = static_cast<int>(gp);
  if (m > TILE_BITS) {
    // The barrier's arrival counts and error word must start at zero; a call that gave up
    // part-way could have left them set, so clear the header before every launch (a memset
    // on the stream, no allocation).  The workspace itself is fully written before it is read.
    if (cudaMemsetAsync(scratch, 0, WHTMIX_NOALLOC_HEADER_BYTES, stream) != cudaSuccess) return WHTMIX_ERR_CUDA;
  }
  switch (dtype) {
    case WHTMIX_F32: return noalloc_dispatch<DT_F32>(P, sms, stream);
    case WHTMIX_BF16: return noalloc_dispatch<DT_BF16>(P, sms, stream);
    default: return noalloc_dispatch<DT_I32>(P, sms, stream);
  }
}
