// whtmix_capi.cu -- host side of the C ABI declared in include/whtmix.h.
//
// Every check runs before anything is enqueued; a failing call enqueues and writes nothing.
// The plain calls take their workspace from a per-(device, stream) cache; the _ex calls use the
// caller's buffer.  Each call is one kernel launch (cooperative when the plan needs device-wide
// barriers), plus a stream-ordered allocation the first time a cached workspace grows.
#include <cuda_runtime.h>

#include <cstring>
#include <map>
#include <mutex>
#include <utility>

#include "whtmix.h"
#include "whtmix_fast_launch.cuh"
#include "whtmix_kernels.cuh"

using namespace whtmix;

namespace {

thread_local int g_last_cuda_error = 0;

constexpr size_t HEADER_BYTES = sizeof(GridBarrier);
constexpr size_t WS_TARGET_BYTES = 32ull << 20;  // plane-group workspace kept L2-resident

int cuda_fail(cudaError_t e) {
  g_last_cuda_error = static_cast<int>(e);
  return WHTMIX_ERR_CUDA;
}

int ilog2_pow2(int64_t v) {
  int r = 0;
  while ((int64_t{1} << r) < v) ++r;
  return r;
}

bool is_pow2(int64_t v) { return v > 0 && (v & (v - 1)) == 0; }

size_t elem_size(int dtype) { return dtype == WHTMIX_BF16 ? 2 : 4; }

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

bool overlap(const void* a, size_t na, const void* b, size_t nb) {
  const uintptr_t pa = reinterpret_cast<uintptr_t>(a), pb = reinterpret_cast<uintptr_t>(b);
  return na && nb && pa < pb + nb && pb < pa + na;
}

// Shape/dtype checks shared by every entry point.  On success sets m = log2(N C).
int check_shape(int64_t B, int64_t N, int64_t C, int dtype, int* m) {
  if (B < 0 || N < 1 || C < 1) return WHTMIX_ERR_INVALID_ARG;
  if (dtype != WHTMIX_F32 && dtype != WHTMIX_BF16 && dtype != WHTMIX_I32) return WHTMIX_ERR_BAD_DTYPE;
  if (!is_pow2(N) || !is_pow2(C)) return WHTMIX_ERR_BAD_SHAPE;
  const int mm = ilog2_pow2(N) + ilog2_pow2(C);
  if (mm > MAX_PLANE_BITS) return WHTMIX_ERR_BAD_SHAPE;
  if (B > (int64_t{1} << (62 - mm))) return WHTMIX_ERR_BAD_SHAPE;
  *m = mm;
  return WHTMIX_OK;
}

int planes_per_group(int64_t B, int m, int backward) {
  if (B == 0) return 1;
  const size_t per = (size_t{1} << m) * 4 * (backward && m > TILE_BITS ? 2 : 1);
  int64_t gp = static_cast<int64_t>(WS_TARGET_BYTES / per);
  if (gp < 1) gp = 1;
  if (gp > B) gp = B;
  return static_cast<int>(gp);
}

size_t workspace_bytes(int64_t B, int m, int backward) {
  if (m <= TILE_BITS && !backward) return HEADER_BYTES;
  const int gp = planes_per_group(B, m, backward);
  const size_t per = (size_t{1} << m) * 4 * (backward && m > TILE_BITS ? 2 : 1);
  return HEADER_BYTES + per * static_cast<size_t>(gp);
}

struct DevInfo {
  bool init = false;
  bool ok = false;
  int sms = 0;
};
std::mutex g_mu;
std::map<int, DevInfo> g_dev;

int device_check(int* dev_out, int* sms_out) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) {
    g_last_cuda_error = static_cast<int>(e);
    return WHTMIX_ERR_NO_DEVICE;
  }
  std::lock_guard<std::mutex> lk(g_mu);
  DevInfo& di = g_dev[dev];
  if (!di.init) {
    cudaDeviceProp prop;
    e = cudaGetDeviceProperties(&prop, dev);
    if (e != cudaSuccess) return cuda_fail(e);
    di.ok = prop.major == 10 && prop.minor == 3;
    di.sms = prop.multiProcessorCount;
    di.init = true;
  }
  if (!di.ok) return WHTMIX_ERR_NO_DEVICE;
  *dev_out = dev;
  *sms_out = di.sms;
  return WHTMIX_OK;
}

// ---- library-managed workspaces, one per (device, stream) ----
struct WsEntry {
  void* ptr = nullptr;
  size_t bytes = 0;
};
std::map<std::pair<int, cudaStream_t>, WsEntry> g_ws;

int cached_workspace(int dev, cudaStream_t stream, size_t need, void** out) {
  std::lock_guard<std::mutex> lk(g_mu);
  WsEntry& w = g_ws[{dev, stream}];
  if (w.bytes < need) {
    if (w.ptr) {
      cudaError_t e = cudaFreeAsync(w.ptr, stream);
      if (e != cudaSuccess) return cuda_fail(e);
      w.ptr = nullptr;
      w.bytes = 0;
    }
    void* p = nullptr;
    cudaError_t e = cudaMallocAsync(&p, need, stream);
    if (e != cudaSuccess) return cuda_fail(e);
    e = cudaMemsetAsync(p, 0, HEADER_BYTES, stream);
    if (e != cudaSuccess) {
      cudaFreeAsync(p, stream);
      return cuda_fail(e);
    }
    w.ptr = p;
    w.bytes = need;
  }
  *out = w.ptr;
  return WHTMIX_OK;
}

// ---- kernel selection and launch ----
// Resident CTAs per SM of a kernel at a given dynamic smem size, per device; the first query
// also raises the kernel's dynamic-smem limit.  Cached: the answer never changes.
std::map<std::pair<int, const void*>, int> g_occ;

int occupancy(const void* kernel, size_t smem, int* occ_out) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return cuda_fail(e);
  std::lock_guard<std::mutex> lk(g_mu);
  auto it = g_occ.find({dev, kernel});
  if (it != g_occ.end()) {
    *occ_out = it->second;
    return WHTMIX_OK;
  }
  if (smem > 48 * 1024) {
    e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
    if (e != cudaSuccess) return cuda_fail(e);
  }
  int occ = 0;
  e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&occ, kernel, THREADS, smem);
  if (e != cudaSuccess) return cuda_fail(e);
  if (occ < 1) return cuda_fail(cudaErrorInvalidConfiguration);
  g_occ[{dev, kernel}] = occ;
  *occ_out = occ;
  return WHTMIX_OK;
}

template <class K>
int launch(K kernel, bool cooperative, int sms, long long max_units, size_t smem, const Params& P, cudaStream_t stream) {
  cudaError_t e;
  int occ = 0;
  const int rc = occupancy(reinterpret_cast<const void*>(kernel), smem, &occ);
  if (rc != WHTMIX_OK) return rc;
  long long grid = static_cast<long long>(occ) * sms;
  if (max_units < grid) grid = max_units < 1 ? 1 : max_units;
  Params p = P;
  void* args[] = {&p};
  if (cooperative)
    e = cudaLaunchCooperativeKernel(reinterpret_cast<const void*>(kernel), dim3(static_cast<unsigned>(grid)), dim3(THREADS), args, smem, stream);
  else
    e = cudaLaunchKernel(reinterpret_cast<const void*>(kernel), dim3(static_cast<unsigned>(grid)), dim3(THREADS), args, smem, stream);
  if (e != cudaSuccess) return cuda_fail(e);
  return WHTMIX_OK;
}

// The fast forward (whtmix_fast.cuh) covers fp32 / bf16 planes with 2^14 <= N*C <= 2^23.
bool use_fast_forward(int dtype, int m) {
  return (dtype == WHTMIX_F32 || dtype == WHTMIX_BF16) && m >= 14 && m <= 23;
}

// The fast backward (whtmix_fast_bwd.cuh) covers fp32 / bf16 planes with 2^14 <= N*C <= 2^21.
bool use_fast_backward(int dtype, int m) {
  return (dtype == WHTMIX_F32 || dtype == WHTMIX_BF16) && m >= 14 && m <= 21;
}

template <int D>
int dispatch(bool backward, const Params& P, int sms, cudaStream_t stream) {
  using A = typename Tr<D>::A;
  const int m = P.m;
  const size_t tile_bytes = sizeof(A) * TILE;
  if (!backward) {
    if constexpr (D != DT_I32) {
      if (use_fast_forward(D, m)) {
        const cudaError_t e = D == DT_BF16 ? fast::forward_bf16(P, sms, stream) : fast::forward_f32(P, sms, stream);
        return e == cudaSuccess ? WHTMIX_OK : cuda_fail(e);
      }
    }
    if (m <= TILE_BITS) {
      const long long ppt = 1ll << (TILE_BITS - m);
      return launch(k_forward_s<D>, false, sms, (P.B + ppt - 1) / ppt, tile_bytes, P, stream);
    }
    return launch(k_forward_m<D>, true, sms, static_cast<long long>(P.gp) << (m - TILE_BITS), tile_bytes, P, stream);
  }
  if constexpr (D != DT_I32) {
    if (use_fast_backward(D, m)) {
      const cudaError_t e = D == DT_BF16 ? fast::backward_bf16(P, sms, stream) : fast::backward_f32(P, sms, stream);
      return e == cudaSuccess ? WHTMIX_OK : cuda_fail(e);
    }
  }
  if (m <= TILE_BITS) {
    const long long ppt = 1ll << (TILE_BITS - m);
    long long units = (P.gp + ppt - 1) / ppt;
    const long long lunits = ((1ll << m) + THREADS - 1) / THREADS;
    if (lunits > units) units = lunits;
    return launch(k_backward_s<D>, true, sms, units, 2 * tile_bytes, P, stream);
  }
  return launch(k_backward_m<D>, true, sms, 2ll * (static_cast<long long>(P.gp) << (m - TILE_BITS)), 3 * tile_bytes, P, stream);
}

int run(bool backward, const void* x, const void* g, const void* dy, void* y_or_dx, void* dg,
        int64_t B, int64_t N, int64_t C, int dtype, void* user_ws, size_t user_ws_bytes, bool use_user_ws,
        void* stream_v) {
  int m = 0;
  int rc = check_shape(B, N, C, dtype, &m);
  if (rc != WHTMIX_OK) return rc;
  if (B == 0) {
    // Empty batch: the forward has nothing to do (any pointers, even null, are accepted); the
    // backward's dG is a sum over no planes, so it is set to zero.
    if (!backward) return WHTMIX_OK;
    if (!dg) return WHTMIX_ERR_INVALID_ARG;
    if (!aligned16(dg)) return WHTMIX_ERR_MISALIGNED;
    int dev = 0, sms = 0;
    rc = device_check(&dev, &sms);
    if (rc != WHTMIX_OK) return rc;
    cudaError_t e = cudaMemsetAsync(dg, 0, (size_t{1} << m) * 4, static_cast<cudaStream_t>(stream_v));
    return e == cudaSuccess ? WHTMIX_OK : cuda_fail(e);
  }
  if (!x || !g || !y_or_dx || (backward && (!dy || !dg))) return WHTMIX_ERR_INVALID_ARG;
  if (!aligned16(x) || !aligned16(g) || !aligned16(y_or_dx) || (backward && (!aligned16(dy) || !aligned16(dg))))
    return WHTMIX_ERR_MISALIGNED;
  const size_t L = size_t{1} << m;
  const size_t plane_bytes = static_cast<size_t>(B) * L * elem_size(dtype);
  const size_t g_bytes = L * 4;
  if (!backward) {
    if (y_or_dx != x && overlap(y_or_dx, plane_bytes, x, plane_bytes)) return WHTMIX_ERR_ALIAS;
    if (overlap(y_or_dx, plane_bytes, g, g_bytes)) return WHTMIX_ERR_ALIAS;
  } else {
    void* dx = y_or_dx;
    if (dx != dy && overlap(dx, plane_bytes, dy, plane_bytes)) return WHTMIX_ERR_ALIAS;
    if (overlap(dx, plane_bytes, x, plane_bytes) || overlap(dx, plane_bytes, g, g_bytes)) return WHTMIX_ERR_ALIAS;
    if (overlap(dg, g_bytes, x, plane_bytes) || overlap(dg, g_bytes, dy, plane_bytes) ||
        overlap(dg, g_bytes, dx, plane_bytes) || overlap(dg, g_bytes, g, g_bytes))
      return WHTMIX_ERR_ALIAS;
  }
  const size_t need = workspace_bytes(B, m, backward);
  if (use_user_ws) {
    if (!user_ws || (reinterpret_cast<uintptr_t>(user_ws) & 255u) || user_ws_bytes < need) return WHTMIX_ERR_WORKSPACE;
  }
  int dev = 0, sms = 0;
  rc = device_check(&dev, &sms);
  if (rc != WHTMIX_OK) return rc;
  cudaStream_t stream = static_cast<cudaStream_t>(stream_v);
  void* ws = user_ws;
  if (!use_user_ws) {
    rc = cached_workspace(dev, stream, need, &ws);
    if (rc != WHTMIX_OK) return rc;
  }
  Params P{};
  P.x = x;
  P.g = g;
  P.dy = dy;
  if (backward) {
    P.dx = y_or_dx;
    P.dg = dg;
  } else {
    P.y = y_or_dx;
  }
  P.bar = static_cast<GridBarrier*>(ws);
  P.ws = static_cast<char*>(ws) + HEADER_BYTES;
  P.B = B;
  P.m = m;
  P.gp = planes_per_group(B, m, backward);
  P.scale = 1.0f / static_cast<float>(L);
  switch (dtype) {
    case WHTMIX_F32: return dispatch<DT_F32>(backward, P, sms, stream);
    case WHTMIX_BF16: return dispatch<DT_BF16>(backward, P, sms, stream);
    default: return dispatch<DT_I32>(backward, P, sms, stream);
  }
}

}  // namespace

extern "C" {

int whtmix_forward(const void* x, const void* gains, void* y, int64_t B, int64_t N, int64_t C, int dtype, void* stream) {
  return run(false, x, gains, nullptr, y, nullptr, B, N, C, dtype, nullptr, 0, false, stream);
}

int whtmix_backward(const void* x, const void* gains, const void* dy, void* dx, void* dgains, int64_t B, int64_t N,
                    int64_t C, int dtype, void* stream) {
  return run(true, x, gains, dy, dx, dgains, B, N, C, dtype, nullptr, 0, false, stream);
}

int whtmix_forward_ex(const void* x, const void* gains, void* y, int64_t B, int64_t N, int64_t C, int dtype,
                      void* workspace, size_t workspace_bytes_, void* stream) {
  return run(false, x, gains, nullptr, y, nullptr, B, N, C, dtype, workspace, workspace_bytes_, true, stream);
}

int whtmix_backward_ex(const void* x, const void* gains, const void* dy, void* dx, void* dgains, int64_t B, int64_t N,
                       int64_t C, int dtype, void* workspace, size_t workspace_bytes_, void* stream) {
  return run(true, x, gains, dy, dx, dgains, B, N, C, dtype, workspace, workspace_bytes_, true, stream);
}

int whtmix_workspace_bytes(int64_t B, int64_t N, int64_t C, int dtype, int backward, size_t* out_bytes) {
  if (!out_bytes) return WHTMIX_ERR_INVALID_ARG;
  int m = 0;
  const int rc = check_shape(B, N, C, dtype, &m);
  if (rc != WHTMIX_OK) return rc;
  *out_bytes = workspace_bytes(B, m, backward != 0);
  return WHTMIX_OK;
}

int whtmix_sync(void* stream_v) {
  cudaStream_t stream = static_cast<cudaStream_t>(stream_v);
  cudaError_t e = cudaStreamSynchronize(stream);
  if (e != cudaSuccess) return cuda_fail(e);
  int dev = 0;
  e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return cuda_fail(e);
  void* ptr = nullptr;
  {
    std::lock_guard<std::mutex> lk(g_mu);
    auto it = g_ws.find({dev, stream});
    if (it != g_ws.end()) ptr = it->second.ptr;
  }
  if (!ptr) return WHTMIX_OK;
  GridBarrier h;
  e = cudaMemcpy(&h, ptr, sizeof(h), cudaMemcpyDeviceToHost);
  if (e != cudaSuccess) return cuda_fail(e);
  if (h.err == 0) return WHTMIX_OK;
  e = cudaMemset(ptr, 0, HEADER_BYTES);
  if (e != cudaSuccess) return cuda_fail(e);
  return WHTMIX_ERR_TIMEOUT;
}

int whtmix_release_workspaces(void) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return cuda_fail(e);
  e = cudaDeviceSynchronize();
  if (e != cudaSuccess) return cuda_fail(e);
  std::lock_guard<std::mutex> lk(g_mu);
  for (auto it = g_ws.begin(); it != g_ws.end();) {
    if (it->first.first == dev) {
      if (it->second.ptr) cudaFree(it->second.ptr);
      it = g_ws.erase(it);
    } else {
      ++it;
    }
  }
  return WHTMIX_OK;
}

const char* whtmix_status_string(int status) {
  switch (status) {
    case WHTMIX_OK: return "ok";
    case WHTMIX_ERR_INVALID_ARG: return "invalid argument (null pointer, B < 0, N < 1 or C < 1)";
    case WHTMIX_ERR_BAD_SHAPE: return "bad shape (N and C must be powers of two, N*C <= 2^26)";
    case WHTMIX_ERR_BAD_DTYPE: return "bad dtype (expected WHTMIX_F32, WHTMIX_BF16 or WHTMIX_I32)";
    case WHTMIX_ERR_MISALIGNED: return "pointer not 16-byte aligned";
    case WHTMIX_ERR_ALIAS: return "output partially overlaps another buffer";
    case WHTMIX_ERR_CUDA: return "CUDA runtime error (see whtmix_last_cuda_error)";
    case WHTMIX_ERR_TIMEOUT: return "a bounded device-wide wait expired";
    case WHTMIX_ERR_NO_DEVICE: return "no usable CUDA device (sm_103 required)";
    case WHTMIX_ERR_WORKSPACE: return "workspace null, not 256-byte aligned, or too small";
    default: return "unknown status";
  }
}

int whtmix_last_cuda_error(void) { return g_last_cuda_error; }

int whtmix_plan(int64_t N, int64_t C) {
  int m = 0;
  if (check_shape(1, N, C, WHTMIX_F32, &m) != WHTMIX_OK) return 0;
  return m <= TILE_BITS ? 1 : 2;
}

}  // extern "C"
