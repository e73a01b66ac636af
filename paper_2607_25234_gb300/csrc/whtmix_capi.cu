// whtmix_capi.cu -- host side of the C ABI declared in include/whtmix.h.
//
// Every check runs before anything is enqueued; a failing call enqueues and writes nothing.
// The plain calls take their workspace from a per-(device, stream) cache; the _ex calls use the
// caller's buffer.  Each call is one kernel launch for most shapes (five per plane group for planes
// of more than 2^26 elements), with programmatic stream serialisation, plus a stream-ordered
// allocation the first time a cached workspace grows.
#include <cuda_runtime.h>

#include <cstring>
#include <map>
#include <mutex>
#include <tuple>
#include <utility>

#include "whtmix.h"
#include "whtmix_fast_launch.cuh"
#include "whtmix_kernels.cuh"

namespace whtmix {
namespace pln {
// One plane per CTA in tensor memory (whtmix_plane.cu): fp32 / bf16 planes of 2^14 .. 2^16 elements.
cudaError_t forward_f32(const Params& P, cudaStream_t stream);
cudaError_t forward_bf16(const Params& P, cudaStream_t stream);
}  // namespace pln
namespace blk {
// Fused block (whtmix_block.cu): bf16, C = 128, 2^21 <= N C <= 2^23, full gains, N_valid = N.
cudaError_t forward_bf16(const Params& P, const void* w_in, const void* w_out, int sms, cudaStream_t stream);
}  // namespace blk
namespace proj {
// whtmix_proj.cu: Z = X W^T on the tensor cores (C = 64, 128, 256; bf16 in, bf16 or fp32 out)
cudaError_t project(const void* x, const void* w, void* z, long long T, int C, bool out_f32, unsigned int* err, int sms,
                    cudaStream_t s);
}  // namespace proj
namespace bbwd {
// whtmix_block_bwd.cu: the block backward's weight transposes and weight gradients on the tensor cores
int wgrad_chunks(long long T, int sms);
cudaError_t transpose(const void* in, void* out, long long T, int C, long long Tp, int sms, cudaStream_t stream);
cudaError_t wgrad(const void* a_tok, const void* b_tok, float* part, float* out, long long T, int C, int sms,
                  unsigned int* err, cudaStream_t stream);
}  // namespace bbwd
}  // namespace whtmix

using namespace whtmix;

namespace {

thread_local int g_last_cuda_error = 0;

constexpr size_t HEADER_BYTES = sizeof(GridBarrier);
constexpr size_t WS_TARGET_BYTES = 64ull << 20;  // plane-group workspace, L2-resident (126 MiB L2)
constexpr int64_t PLANE_MIN_BATCH_16 = 80;
// Smallest batch for which the one-plane-per-CTA forward beats the three-phase kernel: a plane of
// 2^16 elements is four rows for one CTA (two per worker, one after the other), so a small batch
// leaves most SMs idle (measured on [B, 512, 128] bf16, back to back: B = 64 three-phase 24.6 us
// against 26.6, B = 96 30.8 against 26.7, B = 128 36.0 against 28.7); 2^14 and 2^15 planes are one
// row per worker.
int64_t plane_kernel_min_batch(int m) { return m == 16 ? PLANE_MIN_BATCH_16 : 1; }

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
  // B*N*C <= 2^60, so that every byte count of the call (up to three padded copies of the batch
  // at 4 bytes an element) stays far below 2^64
  if (B > (int64_t{1} << (60 - mm))) return WHTMIX_ERR_BAD_SHAPE;
  *m = mm;
  return WHTMIX_OK;
}

// Planes per group: as many as fit in `target` bytes of plane-group workspace (at least one);
// `es` bytes per workspace element (2 for the bf16 exchange of whtmix_forward_x16).
int planes_per_group(int64_t B, int m, int backward, size_t target = WS_TARGET_BYTES, size_t es = 4) {
  if (B == 0) return 1;
  const size_t per = (size_t{1} << m) * es * (backward && m > TILE_BITS ? 2 : 1);
  int64_t gp = static_cast<int64_t>(target / per);
  if (gp < 1) gp = 1;
  if (gp > B) gp = B;
  return static_cast<int>(gp);
}

size_t workspace_bytes(int64_t B, int m, int backward, size_t target = WS_TARGET_BYTES, size_t es = 4) {
  if (m <= TILE_BITS && !backward) return HEADER_BYTES;
  const int gp = planes_per_group(B, m, backward, target, es);
  const size_t per = (size_t{1} << m) * es * (backward && m > TILE_BITS ? 2 : 1);
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
  // Bind the device's primary context to this host thread (a no-op where it is already current):
  // a thread that never set a device -- an autograd worker, a fresh thread of the caller -- then
  // sees the same context as the one that allocated its buffers.
  e = cudaSetDevice(dev);
  if (e != cudaSuccess) return cuda_fail(e);
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

// ---- library-managed workspaces, one per (device, stream, slot) ----
// Slot 0 is the kernels' workspace (barrier header + plane group); slot 1 holds the block
// backward's intermediates, which must survive the slot-0 calls made in between.
struct WsEntry {
  void* ptr = nullptr;
  size_t bytes = 0;
};
std::map<std::tuple<int, cudaStream_t, int>, WsEntry> g_ws;

int cached_workspace(int dev, cudaStream_t stream, size_t need, void** out, int slot = 0) {
  std::lock_guard<std::mutex> lk(g_mu);
  WsEntry& w = g_ws[std::make_tuple(dev, stream, slot)];
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

// One launch of a generic-engine kernel: a grid of at most the resident CTAs (so that with
// device-wide barriers, plans M and the backward, every CTA is resident at once).
template <class K>
int launch(K kernel, int sms, long long max_units, size_t smem, const Params& P, cudaStream_t stream) {
  cudaError_t e;
  int occ = 0;
  const int rc = occupancy(reinterpret_cast<const void*>(kernel), smem, &occ);
  if (rc != WHTMIX_OK) return rc;
  long long grid = static_cast<long long>(occ) * sms;
  if (max_units < grid) grid = max_units < 1 ? 1 : max_units;
  Params p = P;
  void* args[] = {&p};
  e = launch_pdl(reinterpret_cast<const void*>(kernel), static_cast<unsigned>(grid), THREADS, smem, stream, args);
  if (e != cudaSuccess) return cuda_fail(e);
  return WHTMIX_OK;
}

// One launch of a plan-L pass kernel (whtmix_kernels.cuh) over `units` tiles: a grid-stride grid of
// at most the resident CTAs, programmatic stream serialisation, arguments converted to the kernel's
// parameter types by the typed cudaLaunchKernelEx.
template <class... KArgs, class... Args>
int launch_pass(void (*kernel)(KArgs...), int sms, long long units, size_t smem, cudaStream_t stream, Args... args) {
  int occ = 0;
  const int rc = occupancy(reinterpret_cast<const void*>(kernel), smem, &occ);
  if (rc != WHTMIX_OK) return rc;
  long long grid = static_cast<long long>(occ) * sms;
  if (units < grid) grid = units < 1 ? 1 : units;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(static_cast<unsigned>(grid));
  cfg.blockDim = dim3(THREADS);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  const cudaError_t e = cudaLaunchKernelEx(&cfg, kernel, args...);
  return e == cudaSuccess ? WHTMIX_OK : cuda_fail(e);
}

// Plan L (2^26 < N*C <= 2^30): per plane group five passes (forward) or seven (backward), one
// launch each; the high bits [13, m) are split into [13, 13 + k1) and [13 + k1, m).
template <int D>
int dispatch_plan_l(bool backward, const Params& P, int sms, cudaStream_t stream) {
  using A = typename Tr<D>::A;
  const int m = P.m, kt = m - TILE_BITS, k1 = kt / 2, k2 = kt - k1;
  const size_t tb = sizeof(A) * TILE;
  A* wsx = static_cast<A*>(P.ws);
  A* wsd = wsx + (static_cast<long long>(P.gp) << m);
  const long long tiles = 1ll << kt;
  int rc = WHTMIX_OK;
#define WHTMIX_PASS(...)                         \
  do {                                          \
    rc = launch_pass(__VA_ARGS__);              \
    if (rc != WHTMIX_OK) return rc;             \
  } while (0)
  for (long long b0 = 0; b0 < P.B; b0 += P.gp) {
    const long long nb = P.B - b0 < P.gp ? P.B - b0 : P.gp;
    const long long units = nb * tiles;
    if (!backward) {
      WHTMIX_PASS(k_pass_rows_in<D>, sms, units, tb, stream, P.x, wsx, b0, nb, m);
      WHTMIX_PASS(k_pass_cols<D>, sms, units, tb, stream, wsx, nb, m, TILE_BITS, k1, P.g, P.scale, 0);
      WHTMIX_PASS(k_pass_cols<D>, sms, units, tb, stream, wsx, nb, m, TILE_BITS + k1, k2, P.g, P.scale, 1);
      WHTMIX_PASS(k_pass_cols<D>, sms, units, tb, stream, wsx, nb, m, TILE_BITS, k1, P.g, P.scale, 0);
      WHTMIX_PASS(k_pass_rows_out<D>, sms, units, tb, stream, static_cast<const A*>(wsx), P.y, b0, nb, m);
    } else {
      WHTMIX_PASS(k_pass_rows_in<D>, sms, units, tb, stream, P.x, wsx, b0, nb, m);
      WHTMIX_PASS(k_pass_rows_in<D>, sms, units, tb, stream, P.dy, wsd, b0, nb, m);
      WHTMIX_PASS(k_pass_cols<D>, sms, units, tb, stream, wsx, nb, m, TILE_BITS, k1, P.g, P.scale, 0);
      WHTMIX_PASS(k_pass_cols<D>, sms, units, tb, stream, wsd, nb, m, TILE_BITS, k1, P.g, P.scale, 0);
      WHTMIX_PASS(k_pass_cols_bwd<D>, sms, tiles, 3 * tb, stream, wsx, wsd, static_cast<A*>(P.dg), nb, m,
                  TILE_BITS + k1, k2, P.g, P.scale, b0 == 0 ? 1 : 0);
      WHTMIX_PASS(k_pass_cols<D>, sms, units, tb, stream, wsd, nb, m, TILE_BITS, k1, P.g, P.scale, 0);
      WHTMIX_PASS(k_pass_rows_out<D>, sms, units, tb, stream, static_cast<const A*>(wsd), P.dx, b0, nb, m);
    }
  }
#undef WHTMIX_PASS
  return rc;
}

// The fast forward (whtmix_fast.cuh) covers fp32 / bf16 planes with 2^14 <= N*C <= 2^23.
bool use_fast_forward(int dtype, int m) {
  return (dtype == WHTMIX_F32 || dtype == WHTMIX_BF16) && m >= 14 && m <= 23;
}

// The fast backward (whtmix_fast_bwd.cuh) covers fp32 / bf16 planes with 2^14 <= N*C <= 2^23.
bool use_fast_backward(int dtype, int m) {
  return (dtype == WHTMIX_F32 || dtype == WHTMIX_BF16) && m >= 14 && m <= 23;
}

// ws16: the three-phase forward exchanges bf16 (whtmix_forward_x16); P.ws is then sized for it.
template <int D>
int dispatch(bool backward, const Params& P, int sms, cudaStream_t stream, bool ws16 = false) {
  using A = typename Tr<D>::A;
  const int m = P.m;
  const size_t tile_bytes = sizeof(A) * TILE;
  if (m > MAX_PLANE_BITS_M) return dispatch_plan_l<D>(backward, P, sms, stream);
  if (!backward) {
    if constexpr (D != DT_I32) {
      if (use_fast_forward(D, m)) {
        const cudaError_t e = ws16 ? (D == DT_BF16 ? fast::forward_x16_bf16(P, sms, stream) : fast::forward_x16_f32(P, sms, stream))
                                   : (D == DT_BF16 ? fast::forward_bf16(P, sms, stream) : fast::forward_f32(P, sms, stream));
        return e == cudaSuccess ? WHTMIX_OK : cuda_fail(e);
      }
    }
    if (m <= TILE_BITS) {
      const long long ppt = 1ll << (TILE_BITS - m);
      return launch(k_forward_s<D>, sms, (P.B + ppt - 1) / ppt, tile_bytes, P, stream);
    }
    return launch(k_forward_m<D>, sms, static_cast<long long>(P.gp) << (m - TILE_BITS), tile_bytes, P, stream);
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
    return launch(k_backward_s<D>, sms, units, 2 * tile_bytes, P, stream);
  }
  return launch(k_backward_m<D>, sms, 2ll * (static_cast<long long>(P.gp) << (m - TILE_BITS)), 3 * tile_bytes, P, stream);
}

// ---- separable log gains (Section III-B, Eq. 2-3): G[n, c] = exp(g_t[n]) exp(g_c[c]) ----

constexpr int SEP_THREADS = 256;

size_t align256(size_t v) { return (v + 255) & ~size_t{255}; }

// G[e] = exp(g_t[e >> cbits]) * exp(g_c[e mod C]) over one plane: the same two expf values and
// the same single rounding of their product as the separable fast forward's tables.
__global__ void k_sep_gains(float* G, const float* gt, const float* gc, int m, int cbits) {
  const long long L = 1ll << m, cm = (1ll << cbits) - 1;
  for (long long e = static_cast<long long>(blockIdx.x) * blockDim.x + threadIdx.x; e < L;
       e += static_cast<long long>(gridDim.x) * blockDim.x)
    G[e] = expf(gt[e >> cbits]) * expf(gc[e & cm]);
}

// dg_t[n] = sum over c of dG[n, c] G[n, c] (the chain rule through G = exp(g_t) exp(g_c)): one warp
// per token, each lane over channels lane, lane + 32, ... in order, then a fixed shuffle tree.
// These sums run over up to 2^30 products with cancellation, so they accumulate in float64 (the
// products of two floats are exact there) and round once; they are outside the mixer's hot path.
__global__ void k_sep_reduce_t(float* dgt, const float* dG, const float* G, int m, int cbits) {
  const long long N = 1ll << (m - cbits);
  const int C = 1 << cbits, lane = threadIdx.x & 31;
  const long long warps = (static_cast<long long>(gridDim.x) * blockDim.x) >> 5;
  for (long long n = (static_cast<long long>(blockIdx.x) * blockDim.x + threadIdx.x) >> 5; n < N; n += warps) {
    double acc = 0.0;
    for (int c = lane; c < C; c += 32)
      acc += static_cast<double>(dG[(n << cbits) + c]) * static_cast<double>(G[(n << cbits) + c]);
    for (int o = 16; o > 0; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
    if (lane == 0) dgt[n] = static_cast<float>(acc);
  }
}

// dg_c[c] = sum over n of dG[n, c] G[n, c], in two fixed-order steps (float64 as above):
// part[k][c] over the tokens of chunk k in ascending n, then the chunks in ascending k.
__global__ void k_sep_reduce_c_part(double* part, const float* dG, const float* G, int m, int cbits,
                                    long long rows_per_chunk, long long nchunks) {
  const long long N = 1ll << (m - cbits);
  const int C = 1 << cbits;
  for (long long i = static_cast<long long>(blockIdx.x) * blockDim.x + threadIdx.x; i < (nchunks << cbits);
       i += static_cast<long long>(gridDim.x) * blockDim.x) {
    const long long k = i >> cbits, c = i & (C - 1);
    const long long n0 = k * rows_per_chunk, n1 = min(N, n0 + rows_per_chunk);
    double acc = 0.0;
    for (long long n = n0; n < n1; ++n)
      acc += static_cast<double>(dG[(n << cbits) + c]) * static_cast<double>(G[(n << cbits) + c]);
    part[i] = acc;
  }
}
__global__ void k_sep_reduce_c_final(float* dgc, const double* part, int cbits, long long nchunks) {
  const long long C = 1ll << cbits;
  for (long long c = static_cast<long long>(blockIdx.x) * blockDim.x + threadIdx.x; c < C;
       c += static_cast<long long>(gridDim.x) * blockDim.x) {
    double acc = 0.0;
    for (long long k = 0; k < nchunks; ++k) acc += part[(k << cbits) + c];
    dgc[c] = static_cast<float>(acc);
  }
}

unsigned grid_for(long long work, int sms) {
  const long long blocks = (work + SEP_THREADS - 1) / SEP_THREADS;
  const long long cap = 8ll * sms;
  return static_cast<unsigned>(blocks < 1 ? 1 : blocks > cap ? cap : blocks);
}

// Token chunks of the dg_c reduction: enough (chunk, channel) pairs to fill the GPU.
long long sep_chunks(int m, int cbits) {
  const long long N = 1ll << (m - cbits);
  long long k = (1ll << 16) >> cbits;
  if (k < 1) k = 1;
  return k < N ? k : N;
}

bool use_fast_separable(int dtype, int m, int cbits) {
  return use_fast_forward(dtype, m) && cbits >= 1 && cbits <= fast::forward_row_bits(m);
}

// Zero padding / crop on the token axis for the shapes the fast kernels do not pad themselves:
// planes of lv stored elements <-> planes of 2^m elements (element size es bytes).
__global__ void k_pad_planes(void* dst, const void* src, long long B, long long lv, int m, int es) {
  const long long L = 1ll << m;
  for (long long i = static_cast<long long>(blockIdx.x) * blockDim.x + threadIdx.x; i < B * L;
       i += static_cast<long long>(gridDim.x) * blockDim.x) {
    const long long b = i >> m, e = i & (L - 1);
    if (es == 2)
      static_cast<unsigned short*>(dst)[i] = e < lv ? static_cast<const unsigned short*>(src)[b * lv + e] : 0;
    else
      static_cast<unsigned int*>(dst)[i] = e < lv ? static_cast<const unsigned int*>(src)[b * lv + e] : 0u;
  }
}
__global__ void k_crop_planes(void* dst, const void* src, long long B, long long lv, int m, int es) {
  for (long long i = static_cast<long long>(blockIdx.x) * blockDim.x + threadIdx.x; i < B * lv;
       i += static_cast<long long>(gridDim.x) * blockDim.x) {
    const long long b = i / lv, e = i - b * lv;
    if (es == 2)
      static_cast<unsigned short*>(dst)[i] = static_cast<const unsigned short*>(src)[(b << m) + e];
    else
      static_cast<unsigned int*>(dst)[i] = static_cast<const unsigned int*>(src)[(b << m) + e];
  }
}

// One call of the C ABI, after its arguments are named: full gains (g, dg) or separable log gains
// (gt, gc, dgt, dgc); x, y / dx and dy hold n_valid of the N rows of each plane.
struct Call {
  bool backward = false;
  bool separable = false;
  const void* x = nullptr;
  const void* g = nullptr;
  const float* gt = nullptr;
  const float* gc = nullptr;
  const void* dy = nullptr;
  void* out = nullptr;  // y (forward) or dx (backward)
  void* dg = nullptr;
  float* dgt = nullptr;
  float* dgc = nullptr;
  int64_t B = 0, n_valid = 0, N = 0, C = 0;
  int dtype = 0;
  // the mixer block's projections (Eq. 1 and 4), fused into the forward; null for the mixer alone
  const void* w_in = nullptr;
  const void* w_out = nullptr;
  // bytes of plane-group workspace a group may fill (smaller for a fixed-size scratch)
  size_t group_target = WS_TARGET_BYTES;
  // clear the barrier's arrival counts before the launch, keeping its error word (a fixed
  // scratch shared by every call: a wait that gave up in an earlier call must not leave counts
  // behind, and its error stays set until whtmix_sync reports it)
  bool reset_arrivals = false;
  // whtmix_forward_x16: where the three-phase fast forward runs, it exchanges bf16 between its
  // phases (every other kernel keeps its fp32 intermediate)
  bool ws16 = false;
};

// The call runs the three-phase fast forward with the bf16 exchange workspace.
bool x16_applies(const Call& c, int m) {
  return c.ws16 && !c.backward && !c.separable && !c.w_in && use_fast_forward(c.dtype, m);
}

// Workspace layout of a call: the kernel workspace (barrier header + plane group) first, then
// the separable tables or G / dG / partial sums, then the zero-padded copies.
struct Layout {
  size_t base = 0, g = 0, dg = 0, part = 0, pad = 0, total = 0;
  bool fast_sep = false, pad_copy = false;
  int pad_planes = 0;
};

Layout plan_call(const Call& c, int m) {
  Layout l;
  const size_t L = size_t{1} << m;
  const int cbits = ilog2_pow2(c.C);
  const size_t es = elem_size(c.dtype);
  const size_t lv = static_cast<size_t>(c.n_valid) * static_cast<size_t>(c.C);
  // the fast kernels pad and crop in their row passes when every stored plane starts 16-byte aligned
  const bool fast = c.backward ? use_fast_backward(c.dtype, m) : use_fast_forward(c.dtype, m);
  l.pad_copy = lv < L && !(fast && (lv * es) % 16 == 0);
  l.fast_sep = c.separable && !c.backward && !l.pad_copy && use_fast_separable(c.dtype, m, cbits);
  // whtmix_workspace_bytes for a plain call
  l.base = workspace_bytes(c.B, m, c.backward, c.group_target, x16_applies(c, m) ? 2 : 4);
  size_t off = l.base;
  if (c.separable || l.pad_copy) off = align256(off);
  if (l.fast_sep) {
    off += align256((L >> cbits) * 4 + (size_t{1} << cbits) * 4);  // exp tables, right after the plane group
  } else if (c.separable) {
    l.g = off;
    off += align256(L * 4);
    if (c.backward) {
      l.dg = off;
      off += align256(L * 4);
      l.part = off;
      off += align256(static_cast<size_t>(sep_chunks(m, cbits) << cbits) * 8);
    }
  }
  if (l.pad_copy) {
    l.pad = off;
    l.pad_planes = c.backward ? 3 : 2;  // x, y  |  x, dy, dx
    off += l.pad_planes * align256(static_cast<size_t>(c.B) * L * es);
  }
  l.total = off;
  return l;
}

int run(const Call& c, void* user_ws, size_t user_ws_bytes, bool use_user_ws, void* stream_v) {
  int m = 0;
  int rc = check_shape(c.B, c.N, c.C, c.dtype, &m);
  if (rc != WHTMIX_OK) return rc;
  if (c.n_valid < 0 || c.n_valid > c.N) return WHTMIX_ERR_INVALID_ARG;
  if (c.separable && c.dtype == WHTMIX_I32) return WHTMIX_ERR_BAD_DTYPE;  // log-domain gains are real
  cudaStream_t stream = static_cast<cudaStream_t>(stream_v);
  const size_t L = size_t{1} << m;
  const size_t es = elem_size(c.dtype);
  const size_t lv = static_cast<size_t>(c.n_valid) * static_cast<size_t>(c.C);
  const size_t plane_bytes = static_cast<size_t>(c.B) * lv * es;
  const size_t g_bytes = L * 4, t_bytes = static_cast<size_t>(c.N) * 4, ch_bytes = static_cast<size_t>(c.C) * 4;
  auto aligned4 = [](const void* p) { return (reinterpret_cast<uintptr_t>(p) & 3u) == 0; };
  if (c.B == 0 || lv == 0) {
    // No stored elements: the forward has nothing to do (any pointers, even null, are accepted);
    // the backward's gain gradients are sums over nothing, so they are set to zero.
    if (!c.backward) return WHTMIX_OK;
    if (c.separable) {
      if (!c.dgt || !c.dgc) return WHTMIX_ERR_INVALID_ARG;
      if (!aligned4(c.dgt) || !aligned4(c.dgc)) return WHTMIX_ERR_MISALIGNED;
      if (overlap(c.dgt, t_bytes, c.dgc, ch_bytes)) return WHTMIX_ERR_ALIAS;
    } else {
      if (!c.dg) return WHTMIX_ERR_INVALID_ARG;
      if (!aligned16(c.dg)) return WHTMIX_ERR_MISALIGNED;
    }
    int dev = 0, sms = 0;
    rc = device_check(&dev, &sms);
    if (rc != WHTMIX_OK) return rc;
    cudaError_t e = c.separable ? cudaMemsetAsync(c.dgt, 0, t_bytes, stream) : cudaMemsetAsync(c.dg, 0, g_bytes, stream);
    if (e == cudaSuccess && c.separable) e = cudaMemsetAsync(c.dgc, 0, ch_bytes, stream);
    return e == cudaSuccess ? WHTMIX_OK : cuda_fail(e);
  }
  // pointers, alignment, aliasing
  if (!c.x || !c.out || (c.backward && !c.dy)) return WHTMIX_ERR_INVALID_ARG;
  if (c.separable ? (!c.gt || !c.gc || (c.backward && (!c.dgt || !c.dgc))) : (!c.g || (c.backward && !c.dg)))
    return WHTMIX_ERR_INVALID_ARG;
  if (!aligned16(c.x) || !aligned16(c.out) || (c.backward && !aligned16(c.dy))) return WHTMIX_ERR_MISALIGNED;
  if (c.separable) {
    if (!aligned4(c.gt) || !aligned4(c.gc) || (c.backward && (!aligned4(c.dgt) || !aligned4(c.dgc))))
      return WHTMIX_ERR_MISALIGNED;
  } else if (!aligned16(c.g) || (c.backward && !aligned16(c.dg))) {
    return WHTMIX_ERR_MISALIGNED;
  }
  // read-only inputs the output must not touch; the output may equal its own input exactly
  const void* in = c.backward ? c.dy : c.x;
  if (c.out != in && overlap(c.out, plane_bytes, in, plane_bytes)) return WHTMIX_ERR_ALIAS;
  const void* ro[4];
  size_t ro_bytes[4];
  int nro = 0;
  if (c.separable) {
    ro[nro] = c.gt, ro_bytes[nro++] = t_bytes;
    ro[nro] = c.gc, ro_bytes[nro++] = ch_bytes;
  } else {
    ro[nro] = c.g, ro_bytes[nro++] = g_bytes;
  }
  if (c.backward) ro[nro] = c.x, ro_bytes[nro++] = plane_bytes;
  for (int i = 0; i < nro; ++i)
    if (overlap(c.out, plane_bytes, ro[i], ro_bytes[i])) return WHTMIX_ERR_ALIAS;
  if (c.backward) {
    // gain gradients: disjoint from every other buffer of the call
    const void* all[6] = {c.x, c.dy, c.out, c.separable ? static_cast<const void*>(c.gt) : c.g, c.gc, c.dgc};
    const size_t all_bytes[6] = {plane_bytes, plane_bytes, plane_bytes, c.separable ? t_bytes : g_bytes,
                                 c.separable ? ch_bytes : 0, c.separable ? ch_bytes : 0};
    const void* gout = c.separable ? static_cast<const void*>(c.dgt) : c.dg;
    const size_t gout_bytes = c.separable ? t_bytes : g_bytes;
    for (int i = 0; i < 6; ++i)
      if (overlap(gout, gout_bytes, all[i], all_bytes[i])) return WHTMIX_ERR_ALIAS;
    if (c.separable)
      for (int i = 0; i < 5; ++i)
        if (overlap(c.dgc, ch_bytes, all[i], all_bytes[i])) return WHTMIX_ERR_ALIAS;
  }
  const Layout lay = plan_call(c, m);
  if (use_user_ws) {
    if (!user_ws || (reinterpret_cast<uintptr_t>(user_ws) & 255u) || user_ws_bytes < lay.total) return WHTMIX_ERR_WORKSPACE;
  }
  // Planes of 2^14 .. 2^16 elements: one plane per CTA, the fp32 intermediate in the SM's tensor
  // memory, no workspace and no device-wide barrier.
  if (!c.backward && !c.separable && !c.w_in && c.dtype != WHTMIX_I32 && m >= 14 && m <= 16 &&
      c.B >= plane_kernel_min_batch(m) && (lv == L || (lv * es) % 16 == 0) &&
      c.B <= 0x7fffffff) {  // one CTA per plane: B fits a grid
    int dev = 0, sms = 0;
    rc = device_check(&dev, &sms);
    if (rc != WHTMIX_OK) return rc;
    Params P{};
    P.x = c.x;
    P.g = c.g;
    P.y = c.out;
    P.B = c.B;
    P.m = m;
    P.scale = 1.0f / static_cast<float>(L);
    P.lv = static_cast<long long>(lv);
    const cudaError_t e = c.dtype == WHTMIX_BF16 ? pln::forward_bf16(P, stream) : pln::forward_f32(P, stream);
    return e == cudaSuccess ? WHTMIX_OK : cuda_fail(e);
  }
  int dev = 0, sms = 0;
  rc = device_check(&dev, &sms);
  if (rc != WHTMIX_OK) return rc;
  void* ws = user_ws;
  if (!use_user_ws) {
    rc = cached_workspace(dev, stream, lay.total, &ws);
    if (rc != WHTMIX_OK) return rc;
  }
  char* wsb = static_cast<char*>(ws);
  if (c.reset_arrivals) {
    GridBarrier* h = static_cast<GridBarrier*>(ws);
    cudaError_t e0 = cudaMemsetAsync(h->slot01, 0, sizeof(h->slot01), stream);
    if (e0 == cudaSuccess) e0 = cudaMemsetAsync(h->slot23, 0, sizeof(h->slot23), stream);
    if (e0 != cudaSuccess) return cuda_fail(e0);
  }
  const int cbits = ilog2_pow2(c.C);
  Params P{};
  P.x = c.x;
  P.g = c.g;
  P.dy = c.dy;
  if (c.backward) {
    P.dx = c.out;
    P.dg = c.dg;
  } else {
    P.y = c.out;
  }
  P.bar = static_cast<GridBarrier*>(ws);
  P.ws = wsb + HEADER_BYTES;
  P.B = c.B;
  P.m = m;
  const bool ws16 = x16_applies(c, m);
  P.gp = planes_per_group(c.B, m, c.backward, c.group_target, ws16 ? 2 : 4);
  P.scale = 1.0f / static_cast<float>(L);
  P.gt = c.gt;
  P.gc = c.gc;
  P.cbits = cbits;
  P.lv = static_cast<long long>(lv);
  cudaError_t e = cudaSuccess;
  if (c.w_in) {
    e = blk::forward_bf16(P, c.w_in, c.w_out, sms, stream);
    return e == cudaSuccess ? WHTMIX_OK : cuda_fail(e);
  }
  if (lay.fast_sep) {
    e = c.dtype == WHTMIX_BF16 ? fast::forward_sep_bf16(P, sms, stream) : fast::forward_sep_f32(P, sms, stream);
    return e == cudaSuccess ? WHTMIX_OK : cuda_fail(e);
  }
  if (c.separable) {
    // the separable gains as a G plane in the workspace, for the full-gain kernels
    float* G = reinterpret_cast<float*>(wsb + lay.g);
    k_sep_gains<<<grid_for(static_cast<long long>(L), sms), SEP_THREADS, 0, stream>>>(G, c.gt, c.gc, m, cbits);
    P.g = G;
    if (c.backward) P.dg = wsb + lay.dg;
  }
  void* out_pad = nullptr;
  if (lay.pad_copy) {
    const size_t pb = align256(static_cast<size_t>(c.B) * L * es);
    void* xpad = wsb + lay.pad;
    out_pad = wsb + lay.pad + pb;
    const unsigned grid = grid_for(c.B * static_cast<long long>(L), sms);
    k_pad_planes<<<grid, SEP_THREADS, 0, stream>>>(xpad, c.x, c.B, static_cast<long long>(lv), m, static_cast<int>(es));
    P.x = xpad;
    if (c.backward) {
      void* dypad = wsb + lay.pad + 2 * pb;
      k_pad_planes<<<grid, SEP_THREADS, 0, stream>>>(dypad, c.dy, c.B, static_cast<long long>(lv), m, static_cast<int>(es));
      P.dy = dypad;
      P.dx = out_pad;
    } else {
      P.y = out_pad;
    }
    P.lv = static_cast<long long>(L);
    e = cudaGetLastError();
    if (e != cudaSuccess) return cuda_fail(e);
  }
  switch (c.dtype) {
    case WHTMIX_F32: rc = dispatch<DT_F32>(c.backward, P, sms, stream, ws16); break;
    case WHTMIX_BF16: rc = dispatch<DT_BF16>(c.backward, P, sms, stream, ws16); break;
    default: rc = dispatch<DT_I32>(c.backward, P, sms, stream); break;
  }
  if (rc != WHTMIX_OK) return rc;
  if (lay.pad_copy)
    k_crop_planes<<<grid_for(c.B * static_cast<long long>(lv), sms), SEP_THREADS, 0, stream>>>(
        c.out, out_pad, c.B, static_cast<long long>(lv), m, static_cast<int>(es));
  if (c.separable && c.backward) {
    const float* G = static_cast<const float*>(P.g);
    const float* dG = reinterpret_cast<const float*>(wsb + lay.dg);
    double* part = reinterpret_cast<double*>(wsb + lay.part);
    const long long nchunks = sep_chunks(m, cbits), Nn = 1ll << (m - cbits);
    k_sep_reduce_t<<<grid_for(Nn * 32, sms), SEP_THREADS, 0, stream>>>(c.dgt, dG, G, m, cbits);
    k_sep_reduce_c_part<<<grid_for(nchunks << cbits, sms), SEP_THREADS, 0, stream>>>(part, dG, G, m, cbits,
                                                                                      (Nn + nchunks - 1) / nchunks, nchunks);
    k_sep_reduce_c_final<<<grid_for(1ll << cbits, sms), SEP_THREADS, 0, stream>>>(c.dgc, part, cbits, nchunks);
  }
  e = cudaGetLastError();
  return e == cudaSuccess ? WHTMIX_OK : cuda_fail(e);
}

Call full_call(bool backward, const void* x, const void* g, const void* dy, void* out, void* dg, int64_t B,
               int64_t n_valid, int64_t N, int64_t C, int dtype) {
  Call c;
  c.backward = backward;
  c.x = x;
  c.g = g;
  c.dy = dy;
  c.out = out;
  c.dg = dg;
  c.B = B;
  c.n_valid = n_valid;
  c.N = N;
  c.C = C;
  c.dtype = dtype;
  return c;
}

Call separable_call(bool backward, const void* x, const float* gt, const float* gc, const void* dy, void* out,
                    float* dgt, float* dgc, int64_t B, int64_t n_valid, int64_t N, int64_t C, int dtype) {
  Call c;
  c.backward = backward;
  c.separable = true;
  c.x = x;
  c.gt = gt;
  c.gc = gc;
  c.dy = dy;
  c.out = out;
  c.dgt = dgt;
  c.dgc = dgc;
  c.B = B;
  c.n_valid = n_valid;
  c.N = N;
  c.C = C;
  c.dtype = dtype;
  return c;
}

// The fused block kernel covers 128 channels and planes of 2^21 to 2^23 elements (rows of 128
// tokens x 128 channels, columns of 128 to 512 rows).
bool use_fused_block(int64_t C, int m) { return C == 128 && m >= 21 && m <= 23; }

}  // namespace

namespace whtmix {
// The forward of whtmix_forward_noalloc (whtmix_noalloc.cu): whtmix_forward's kernel choice with
// the fixed scratch as the workspace, plane groups limited to what it holds.  A plane that needs
// more scratch than that returns WHTMIX_ERR_WORKSPACE; nothing is allocated.
int forward_in_fixed_scratch(const void* x, const void* gains, void* y, int64_t B, int64_t N, int64_t C, int dtype,
                             void* scratch, size_t scratch_bytes, void* stream) {
  Call c = full_call(false, x, gains, nullptr, y, nullptr, B, N, N, C, dtype);
  c.group_target = scratch_bytes - HEADER_BYTES;
  c.reset_arrivals = true;
  return run(c, scratch, scratch_bytes, true, stream);
}
// Device address of the fixed scratch on device `dev`, or null if no call has set it up there.
void* noalloc_scratch_of(int dev);
}  // namespace whtmix

extern "C" {

int whtmix_forward(const void* x, const void* gains, void* y, int64_t B, int64_t N, int64_t C, int dtype, void* stream) {
  return run(full_call(false, x, gains, nullptr, y, nullptr, B, N, N, C, dtype), nullptr, 0, false, stream);
}

int whtmix_forward_x16(const void* x, const void* gains, void* y, int64_t B, int64_t N, int64_t C, int dtype,
                       void* stream) {
  Call c = full_call(false, x, gains, nullptr, y, nullptr, B, N, N, C, dtype);
  c.ws16 = true;
  return run(c, nullptr, 0, false, stream);
}

int whtmix_backward(const void* x, const void* gains, const void* dy, void* dx, void* dgains, int64_t B, int64_t N,
                    int64_t C, int dtype, void* stream) {
  return run(full_call(true, x, gains, dy, dx, dgains, B, N, N, C, dtype), nullptr, 0, false, stream);
}

int whtmix_forward_ex(const void* x, const void* gains, void* y, int64_t B, int64_t N, int64_t C, int dtype,
                      void* workspace, size_t workspace_bytes_, void* stream) {
  return run(full_call(false, x, gains, nullptr, y, nullptr, B, N, N, C, dtype), workspace, workspace_bytes_, true,
             stream);
}

int whtmix_backward_ex(const void* x, const void* gains, const void* dy, void* dx, void* dgains, int64_t B, int64_t N,
                       int64_t C, int dtype, void* workspace, size_t workspace_bytes_, void* stream) {
  return run(full_call(true, x, gains, dy, dx, dgains, B, N, N, C, dtype), workspace, workspace_bytes_, true, stream);
}

int whtmix_forward_padded(const void* x, const void* gains, void* y, int64_t B, int64_t N_valid, int64_t N, int64_t C,
                          int dtype, void* stream) {
  return run(full_call(false, x, gains, nullptr, y, nullptr, B, N_valid, N, C, dtype), nullptr, 0, false, stream);
}

int whtmix_backward_padded(const void* x, const void* gains, const void* dy, void* dx, void* dgains, int64_t B,
                           int64_t N_valid, int64_t N, int64_t C, int dtype, void* stream) {
  return run(full_call(true, x, gains, dy, dx, dgains, B, N_valid, N, C, dtype), nullptr, 0, false, stream);
}

int whtmix_forward_separable(const void* x, const float* g_t, const float* g_c, void* y, int64_t B, int64_t N_valid,
                             int64_t N, int64_t C, int dtype, void* stream) {
  return run(separable_call(false, x, g_t, g_c, nullptr, y, nullptr, nullptr, B, N_valid, N, C, dtype), nullptr, 0,
             false, stream);
}

int whtmix_backward_separable(const void* x, const float* g_t, const float* g_c, const void* dy, void* dx,
                              float* dg_t, float* dg_c, int64_t B, int64_t N_valid, int64_t N, int64_t C, int dtype,
                              void* stream) {
  return run(separable_call(true, x, g_t, g_c, dy, dx, dg_t, dg_c, B, N_valid, N, C, dtype), nullptr, 0, false,
             stream);
}

int whtmix_project(const void* x, const void* w, void* z, int64_t T, int64_t C, int out_dtype, void* stream_v) {
  if (T < 0 || C < 1) return WHTMIX_ERR_INVALID_ARG;
  if (C != 64 && C != 128 && C != 256) return WHTMIX_ERR_BAD_SHAPE;
  if (T > (int64_t{1} << 60) / C) return WHTMIX_ERR_BAD_SHAPE;  // T*C <= 2^60: byte counts stay below 2^64
  if (out_dtype != WHTMIX_F32 && out_dtype != WHTMIX_BF16) return WHTMIX_ERR_BAD_DTYPE;
  if (T == 0) return WHTMIX_OK;
  if (!x || !w || !z) return WHTMIX_ERR_INVALID_ARG;
  if (!aligned16(x) || !aligned16(w) || !aligned16(z)) return WHTMIX_ERR_MISALIGNED;
  const size_t xb = static_cast<size_t>(T) * C * 2, wb = static_cast<size_t>(C) * C * 2;
  const size_t zb = static_cast<size_t>(T) * C * (out_dtype == WHTMIX_F32 ? 4 : 2);
  // z may be x itself (bf16 out: each tile is read whole before it is written), nothing else
  if (!(z == x && out_dtype == WHTMIX_BF16) && overlap(z, zb, x, xb)) return WHTMIX_ERR_ALIAS;
  if (overlap(z, zb, w, wb)) return WHTMIX_ERR_ALIAS;
  int dev = 0, sms = 0;
  int rc = device_check(&dev, &sms);
  if (rc != WHTMIX_OK) return rc;
  cudaStream_t stream = static_cast<cudaStream_t>(stream_v);
  void* ws = nullptr;
  rc = cached_workspace(dev, stream, HEADER_BYTES, &ws);
  if (rc != WHTMIX_OK) return rc;
  const cudaError_t e = proj::project(x, w, z, T, static_cast<int>(C), out_dtype == WHTMIX_F32,
                                      &static_cast<GridBarrier*>(ws)->err, sms, stream);
  return e == cudaSuccess ? WHTMIX_OK : cuda_fail(e);
}

int whtmix_block_forward(const void* x, const void* w_in, const void* gains, const void* w_out, void* y, int64_t B,
                         int64_t N, int64_t C, int dtype, void* stream) {
  int m = 0;
  int rc = check_shape(B, N, C, dtype, &m);
  if (rc != WHTMIX_OK) return rc;
  if (dtype != WHTMIX_BF16) return WHTMIX_ERR_BAD_DTYPE;
  if (C != 64 && C != 128 && C != 256) return WHTMIX_ERR_BAD_SHAPE;
  if (B == 0) return WHTMIX_OK;
  if (!x || !w_in || !gains || !w_out || !y) return WHTMIX_ERR_INVALID_ARG;
  if (!aligned16(x) || !aligned16(w_in) || !aligned16(gains) || !aligned16(w_out) || !aligned16(y))
    return WHTMIX_ERR_MISALIGNED;
  const size_t plane_bytes = static_cast<size_t>(B) * N * C * 2, wb = static_cast<size_t>(C) * C * 2;
  const size_t g_bytes = static_cast<size_t>(N) * C * 4;
  // y is written three times (projection, mixer, projection), so it may not hold any input except x
  if (y != x && overlap(y, plane_bytes, x, plane_bytes)) return WHTMIX_ERR_ALIAS;
  if (overlap(y, plane_bytes, w_in, wb) || overlap(y, plane_bytes, w_out, wb) || overlap(y, plane_bytes, gains, g_bytes))
    return WHTMIX_ERR_ALIAS;
  if (use_fused_block(C, m)) {
    // one launch: the projections are the prologue and epilogue of the mixer's row phases
    Call c = full_call(false, x, gains, nullptr, y, nullptr, B, N, N, C, dtype);
    c.w_in = w_in;
    c.w_out = w_out;
    return run(c, nullptr, 0, false, stream);
  }
  const long long T = B * N;
  // Eq. 1: Z = X W_in^T, into y; Eq. 2-3: the mixer, in place; Eq. 4: Y = M W_out^T, in place
  rc = whtmix_project(x, w_in, y, T, C, WHTMIX_BF16, stream);
  if (rc != WHTMIX_OK) return rc;
  rc = run(full_call(false, y, gains, nullptr, y, nullptr, B, N, N, C, dtype), nullptr, 0, false, stream);
  if (rc != WHTMIX_OK) return rc;
  return whtmix_project(y, w_out, y, T, C, WHTMIX_BF16, stream);
}

int whtmix_block_backward(const void* x, const void* w_in, const void* gains, const void* w_out, const void* dy,
                          void* dx, void* dw_in, void* dgains, void* dw_out, int64_t B, int64_t N, int64_t C, int dtype,
                          void* stream_v) {
  int m = 0;
  int rc = check_shape(B, N, C, dtype, &m);
  if (rc != WHTMIX_OK) return rc;
  if (dtype != WHTMIX_BF16) return WHTMIX_ERR_BAD_DTYPE;
  if (C != 64 && C != 128 && C != 256) return WHTMIX_ERR_BAD_SHAPE;
  if (!dw_in || !dgains || !dw_out) return WHTMIX_ERR_INVALID_ARG;
  if (!aligned16(dw_in) || !aligned16(dgains) || !aligned16(dw_out)) return WHTMIX_ERR_MISALIGNED;
  const size_t wgb = static_cast<size_t>(C) * C * 4, gb = static_cast<size_t>(N) * C * 4;
  if (overlap(dw_in, wgb, dgains, gb) || overlap(dw_in, wgb, dw_out, wgb) || overlap(dgains, gb, dw_out, wgb))
    return WHTMIX_ERR_ALIAS;
  cudaStream_t stream = static_cast<cudaStream_t>(stream_v);
  int dev = 0, sms = 0;
  if (B == 0) {  // sums over no tokens
    rc = device_check(&dev, &sms);
    if (rc != WHTMIX_OK) return rc;
    cudaError_t e = cudaMemsetAsync(dw_in, 0, wgb, stream);
    if (e == cudaSuccess) e = cudaMemsetAsync(dgains, 0, gb, stream);
    if (e == cudaSuccess) e = cudaMemsetAsync(dw_out, 0, wgb, stream);
    return e == cudaSuccess ? WHTMIX_OK : cuda_fail(e);
  }
  if (!x || !w_in || !gains || !w_out || !dy || !dx) return WHTMIX_ERR_INVALID_ARG;
  if (!aligned16(x) || !aligned16(w_in) || !aligned16(gains) || !aligned16(w_out) || !aligned16(dy) || !aligned16(dx))
    return WHTMIX_ERR_MISALIGNED;
  const long long T = B * N;
  const size_t pb = static_cast<size_t>(T) * C * 2, wb = static_cast<size_t>(C) * C * 2;
  // dx may be dy itself (dY is consumed before dZ is written there); no other overlap
  const void* ins[5] = {x, w_in, gains, w_out, dy};
  const size_t in_bytes[5] = {pb, wb, gb, wb, pb};
  void* outs[4] = {dx, dw_in, dgains, dw_out};
  const size_t out_bytes[4] = {pb, wgb, gb, wgb};
  for (int o = 0; o < 4; ++o) {
    for (int i = 0; i < 5; ++i)
      if (!(o == 0 && i == 4 && outs[o] == ins[i]) && overlap(outs[o], out_bytes[o], ins[i], in_bytes[i]))
        return WHTMIX_ERR_ALIAS;
    for (int p = o + 1; p < 4; ++p)
      if (overlap(outs[o], out_bytes[o], outs[p], out_bytes[p])) return WHTMIX_ERR_ALIAS;
  }
  rc = device_check(&dev, &sms);
  if (rc != WHTMIX_OK) return rc;
  // slot-1 layout: Z, M, dM [T, C] bf16; a transposed weight [C, C] bf16; the per-chunk partials
  // [chunks, C, C] fp32 of a weight gradient
  const int chunks = bbwd::wgrad_chunks(T, sms);
  size_t off[5], total = 0;
  const size_t sizes[5] = {pb, pb, pb, wb, static_cast<size_t>(chunks) * wgb};
  for (int i = 0; i < 5; ++i) {
    off[i] = total;
    total += align256(sizes[i]);
  }
  void* w1 = nullptr;
  rc = cached_workspace(dev, stream, total, &w1, 1);
  if (rc != WHTMIX_OK) return rc;
  char* base = static_cast<char*>(w1);
  void *Z = base + off[0], *M = base + off[1], *dM = base + off[2], *WT = base + off[3];
  float* part = reinterpret_cast<float*>(base + off[4]);
  auto err_word = [&](unsigned int** e) -> int {  // the slot-0 header's error word, read by whtmix_sync
    void* w0 = nullptr;
    const int r = cached_workspace(dev, stream, HEADER_BYTES, &w0, 0);
    *e = &static_cast<GridBarrier*>(w0)->err;
    return r;
  };
  unsigned int* err = nullptr;
  cudaError_t e = cudaSuccess;
#define WHTMIX_STEP(call)                  \
  do {                                     \
    rc = (call);                           \
    if (rc != WHTMIX_OK) return rc;        \
  } while (0)
#define WHTMIX_CUDA_STEP(call)             \
  do {                                     \
    e = (call);                            \
    if (e != cudaSuccess) return cuda_fail(e); \
  } while (0)
  // Eq. 1 and the mixer: Z = X W_in^T, M = mix(Z) (bf16 activations, as the forward's)
  WHTMIX_STEP(whtmix_project(x, w_in, Z, T, C, WHTMIX_BF16, stream));
  WHTMIX_STEP(run(full_call(false, Z, gains, nullptr, M, nullptr, B, N, N, C, dtype), nullptr, 0, false, stream));
  // Eq. 4 backward: dM = dY W_out (the projection with W_out^T), dW_out = dY^T M
  WHTMIX_CUDA_STEP(bbwd::transpose(w_out, WT, C, static_cast<int>(C), C, sms, stream));
  WHTMIX_STEP(whtmix_project(dy, WT, dM, T, C, WHTMIX_BF16, stream));
  WHTMIX_STEP(err_word(&err));
  WHTMIX_CUDA_STEP(bbwd::wgrad(dy, M, part, static_cast<float*>(dw_out), T, static_cast<int>(C), sms, err, stream));
  // the mixer's backward: dZ (into dx) and dG
  WHTMIX_STEP(run(full_call(true, Z, gains, dM, dx, dgains, B, N, N, C, dtype), nullptr, 0, false, stream));
  // Eq. 1 backward: dW_in = dZ^T X, then dX = dZ W_in in place
  WHTMIX_STEP(err_word(&err));
  WHTMIX_CUDA_STEP(bbwd::wgrad(dx, x, part, static_cast<float*>(dw_in), T, static_cast<int>(C), sms, err, stream));
  WHTMIX_CUDA_STEP(bbwd::transpose(w_in, WT, C, static_cast<int>(C), C, sms, stream));
  WHTMIX_STEP(whtmix_project(dx, WT, dx, T, C, WHTMIX_BF16, stream));
#undef WHTMIX_STEP
#undef WHTMIX_CUDA_STEP
  return WHTMIX_OK;
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
  void* ptrs[2] = {nullptr, whtmix::noalloc_scratch_of(dev)};
  {
    std::lock_guard<std::mutex> lk(g_mu);
    auto it = g_ws.find(std::make_tuple(dev, stream, 0));
    if (it != g_ws.end()) ptrs[0] = it->second.ptr;
  }
  // the stream's library-managed workspace, then the no-allocation scratch of this device (both
  // keep a set error word until it is reported here)
  int rc = WHTMIX_OK;
  for (void* ptr : ptrs) {
    if (!ptr) continue;
    GridBarrier h;
    e = cudaMemcpy(&h, ptr, sizeof(h), cudaMemcpyDeviceToHost);
    if (e != cudaSuccess) return cuda_fail(e);
    if (h.err == 0) continue;
    e = cudaMemset(ptr, 0, HEADER_BYTES);
    if (e != cudaSuccess) return cuda_fail(e);
    rc = WHTMIX_ERR_TIMEOUT;
  }
  return rc;
}

int whtmix_release_workspaces(void) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return cuda_fail(e);
  e = cudaDeviceSynchronize();
  if (e != cudaSuccess) return cuda_fail(e);
  std::lock_guard<std::mutex> lk(g_mu);
  for (auto it = g_ws.begin(); it != g_ws.end();) {
    if (std::get<0>(it->first) == dev) {
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
    case WHTMIX_ERR_BAD_SHAPE: return "bad shape (N and C must be powers of two, N*C <= 2^30)";
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
  return m <= TILE_BITS ? 1 : m <= MAX_PLANE_BITS_M ? 2 : 3;
}

}  // extern "C"
