// whtmix_kernels.cuh -- CUDA kernels of the WHTMix token mixer for sm_103a (generic tile engine).
//
// The map (Section III-B, Eq. 1-4): Y_b = H_N (G (.) H_N X_b H_C) H_C / (N C), with H the
// Sylvester-Hadamard matrix.  Row-major flattening of a plane puts the channel index in the low
// log2(C) bits and the token index in the high log2(N) bits of the flat index, and
// H_N (x) H_C = H_{NC} in Sylvester order, so the 2D transform of a plane is the 1D transform of
// length L = N C over all m = log2(L) bits of the flat index.  Butterfly stages on different
// bits commute, which lets each kernel phase transform whichever bits its data layout holds.
//
// Plans (chosen per shape by the host):
//   S (m <= 13): a tile of 2^13 elements holds one or more whole planes; one pass reads X, runs
//     all m bits forward, multiplies by G/L, runs all m bits again, writes Y.
//   M (13 < m <= 26): three phases over a plane group kept in an fp32 (uint32) workspace, with a
//     device-wide barrier between phases:
//       phase 1  each row tile (2^13 contiguous elements): bits [0, 13)            X  -> ws
//       phase 2  each column tile (W = 2^(26-m) adjacent columns x 2^(m-13) rows): bits
//                [13, m) forward, gain, bits [13, m) inverse                       ws -> ws
//       phase 3  each row tile: bits [0, 13) again                                 ws -> Y
//   L (26 < m <= 30): the high bits no longer fit one column tile, so they are split in two
//     groups [13, 13 + k1) and [13 + k1, m) and the transform runs as five passes, one launch
//     each (the kernel boundary is the barrier): rows, columns over the first group, columns over
//     the second with the gain in the middle, the first group again, rows again.
// Inside a tile the data sits in shared memory (XOR-swizzled) and every round loads 2^e <= 32
// elements per thread into registers, runs e butterfly stages there and stores them back.
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

namespace whtmix {

constexpr int TILE_BITS = 13;
constexpr int TILE = 1 << TILE_BITS;
constexpr int THREADS = 256;
constexpr int MAX_PLANE_BITS_M = 2 * TILE_BITS;  // plan M: one column tile holds the high bits
constexpr int MAX_PLANE_BITS = 30;               // plan L up to 2^30 elements per plane
constexpr int ROUND_BITS = 5;
constexpr unsigned long long BARRIER_TIMEOUT_NS = 1000000000ull;  // 1 s

enum DType { DT_F32 = 0, DT_BF16 = 1, DT_I32 = 2 };

// Host: launch a kernel that begins with pdl_wait() (and ends with pdl_trigger()) with programmatic
// stream serialisation, so that its launch and prologue overlap the previous kernel's tail.
inline cudaError_t launch_pdl(const void* kernel, unsigned int grid, unsigned int block, size_t smem,
                              cudaStream_t stream, void** args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(grid);
  cfg.blockDim = dim3(block);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelExC(&cfg, kernel, args);
}

// Device-wide barrier state; lives in the first 256 bytes of the workspace.  Barriers are numbered
// on from call to call (seq); barrier k counts its arrivals in slot k mod 4.
struct GridBarrier {
  unsigned int slot01[2];  // words 0, 1: arrival counts of slots 0 and 1
  unsigned int err;        // word 2: non-zero once a wait gave up
  unsigned int slot23[2];  // words 3, 4: arrival counts of slots 2 and 3
  unsigned int seq;        // word 5: number of the next barrier
  unsigned int pad[58];
};
static_assert(sizeof(GridBarrier) == 256, "barrier header is 256 bytes");

struct Params {
  const void* x;
  const void* dy;
  const void* g;
  void* y;
  void* dx;
  void* dg;
  void* ws;          // plane-group workspace (accumulator type), after the barrier header
  GridBarrier* bar;  // device-wide barrier
  long long B;       // planes
  int m;             // log2(N C)
  int gp;            // planes per group
  float scale;       // 1 / (N C) for the floating-point dtypes
  // separable log gains (fast forward only): g_t [N], g_c [C], C = 2^cbits; g is unused then
  const float* gt;
  const float* gc;
  int cbits;
  // elements of a plane held in x, y, dy, dx (planes stored back to back, lv each); the plane the
  // mixer transforms is those followed by 2^m - lv zeros (the token-axis zero padding).  Only the
  // fast kernels read it; everything else runs with lv = 2^m.
  long long lv;
};

// ---- dtype traits: storage <-> accumulator (fp32 for F32/BF16, uint32 for I32) ----
template <int D> struct Tr;
template <> struct Tr<DT_F32> {
  using A = float;
  __device__ static __forceinline__ float ld(const void* p, long long i) { return __ldcg(static_cast<const float*>(p) + i); }
  __device__ static __forceinline__ void st(void* p, long long i, float v) { static_cast<float*>(p)[i] = v; }
  __device__ static __forceinline__ float gain(const void* g, long long i, float s) { return __ldg(static_cast<const float*>(g) + i) * s; }
};
template <> struct Tr<DT_BF16> {
  using A = float;
  __device__ static __forceinline__ float ld(const void* p, long long i) {
    unsigned short u = __ldcg(static_cast<const unsigned short*>(p) + i);
    return __uint_as_float(static_cast<unsigned int>(u) << 16);
  }
  __device__ static __forceinline__ void st(void* p, long long i, float v) { static_cast<__nv_bfloat16*>(p)[i] = __float2bfloat16_rn(v); }
  __device__ static __forceinline__ float gain(const void* g, long long i, float s) { return __ldg(static_cast<const float*>(g) + i) * s; }
};
template <> struct Tr<DT_I32> {
  using A = unsigned int;
  __device__ static __forceinline__ unsigned int ld(const void* p, long long i) { return static_cast<unsigned int>(__ldcg(static_cast<const int*>(p) + i)); }
  __device__ static __forceinline__ void st(void* p, long long i, unsigned int v) { static_cast<int*>(p)[i] = static_cast<int>(v); }
  __device__ static __forceinline__ unsigned int gain(const void* g, long long i, float) { return static_cast<unsigned int>(__ldg(static_cast<const int*>(g) + i)); }
};

// accumulator-typed workspace / dG access (L2-coherent loads: other CTAs wrote these)
__device__ __forceinline__ float ld_ws(const float* p, long long i) { return __ldcg(p + i); }
__device__ __forceinline__ unsigned int ld_ws(const unsigned int* p, long long i) { return __ldcg(p + i); }
__device__ __forceinline__ float mul_scale(float a, float s) { return a * s; }
__device__ __forceinline__ unsigned int mul_scale(unsigned int a, float) { return a; }

// XOR swizzle of the 2^13-element tile: every round below touches 32 distinct banks per warp.
__device__ __forceinline__ int swz(int i) { return i ^ ((i >> 5) & 31); }

// e butterfly stages over the 2^e values of one thread: (a, b) -> (a + b, a - b) on each pair
// (j, j + h), h = 1, 2, ..., 2^(e-1).
template <class A, int E>
__device__ __forceinline__ void bfly_regs(A (&v)[1 << E]) {
#pragma unroll
  for (int h = 1; h < (1 << E); h <<= 1) {
#pragma unroll
    for (int i = 0; i < (1 << E); ++i) {
      if ((i & h) == 0) {
        const A a = v[i], b = v[i + h];
        v[i] = a + b;
        v[i + h] = a - b;
      }
    }
  }
}

struct NoMid {
  template <class A, int E>
  __device__ __forceinline__ void apply(A (&)[1 << E], int, int, int) const {}
};

// One round: butterflies over tile bits [s, s + E).  `mid` runs on the registers after them.
template <class A, int E, class Mid>
__device__ __forceinline__ void round_e(A* tile, int s, const Mid& mid) {
  constexpr int R = 1 << E;
  for (int gi = threadIdx.x; gi < (TILE >> E); gi += THREADS) {
    const int lo = gi & ((1 << s) - 1);
    const int hi = (gi >> s) << (s + E);
    A v[R];
#pragma unroll
    for (int r = 0; r < R; ++r) v[r] = tile[swz(hi | (r << s) | lo)];
    bfly_regs<A, E>(v);
    mid.template apply<A, E>(v, hi, lo, s);
#pragma unroll
    for (int r = 0; r < R; ++r) tile[swz(hi | (r << s) | lo)] = v[r];
  }
  __syncthreads();
}

template <class A, class Mid>
__device__ __forceinline__ void round_any(A* tile, int s, int e, const Mid& mid) {
  switch (e) {
    case 0: round_e<A, 0>(tile, s, mid); break;
    case 1: round_e<A, 1>(tile, s, mid); break;
    case 2: round_e<A, 2>(tile, s, mid); break;
    case 3: round_e<A, 3>(tile, s, mid); break;
    case 4: round_e<A, 4>(tile, s, mid); break;
    default: round_e<A, 5>(tile, s, mid); break;
  }
}

// Forward transform over tile bits [s0, s1).
template <class A>
__device__ __forceinline__ void xform(A* tile, int s0, int s1) {
  for (int s = s0; s < s1; s += ROUND_BITS) round_any(tile, s, min(ROUND_BITS, s1 - s), NoMid{});
}

// Transform over [s0, s1), then `mid` (gain), then the same transform again.  The last round
// carries the mid step and the repeated stages of its own bits; the other rounds repeat after.
template <class A, class Mid>
__device__ __forceinline__ void xform_mid_xform(A* tile, int s0, int s1, const Mid& mid) {
  const int n = s1 - s0;
  const int nr = n == 0 ? 1 : (n + ROUND_BITS - 1) / ROUND_BITS;
  for (int r = 0; r + 1 < nr; ++r) round_any(tile, s0 + r * ROUND_BITS, ROUND_BITS, NoMid{});
  const int sl = s0 + (nr - 1) * ROUND_BITS;
  round_any(tile, sl, s1 - sl, mid);
  for (int r = nr - 2; r >= 0; --r) round_any(tile, s0 + r * ROUND_BITS, ROUND_BITS, NoMid{});
}

// Tile-local index -> index into G / dG ([N, C] flattened) for the two tile shapes.
struct PlaneMap {  // plan S: tile = consecutive whole planes
  int lmask;
  __device__ __forceinline__ long long operator()(int i) const { return i & lmask; }
};
struct ColMap {  // column tile: i = (row << w) | c  ->  (row << s) + col0 + c (s = 13 in plan M)
  int w;
  long long col0;
  int s = TILE_BITS;
  __device__ __forceinline__ long long operator()(int i) const {
    return (static_cast<long long>(i >> w) << s) + col0 + (i & ((1 << w) - 1));
  }
};

// Gain step: v *= G[map(i)] / (N C), then the same butterfly stages again.
template <int D, class Map>
struct GainMid {
  const void* g;
  float scale;
  Map map;
  template <class A, int E>
  __device__ __forceinline__ void apply(A (&v)[1 << E], int hi, int lo, int s) const {
#pragma unroll
    for (int r = 0; r < (1 << E); ++r) v[r] = v[r] * Tr<D>::gain(g, map(hi | (r << s) | lo), scale);
    bfly_regs<A, E>(v);
  }
};

// Backward, plan S: at the gain step of the dY tile, write the partial (W X)(W dY)/L for dG,
// then continue as the forward does.
template <int D>
struct BwdMidS {
  const typename Tr<D>::A* tx;  // transformed X tile (smem)
  typename Tr<D>::A* part;      // group partials, at this tile's first plane
  int nvalid;                   // valid elements in the tile
  const void* g;
  float scale;
  int lmask;
  template <class A, int E>
  __device__ __forceinline__ void apply(A (&v)[1 << E], int hi, int lo, int s) const {
#pragma unroll
    for (int r = 0; r < (1 << E); ++r) {
      const int i = hi | (r << s) | lo;
      if (i < nvalid) part[i] = mul_scale(tx[swz(i)] * v[r], scale);
      v[r] = v[r] * Tr<D>::gain(g, i & lmask, scale);
    }
    bfly_regs<A, E>(v);
  }
};

// Backward, plan M column tile: accumulate (W X)(W dY)/L into the dG tile, then the gain step.
template <int D>
struct BwdMidM {
  const typename Tr<D>::A* tx;
  typename Tr<D>::A* acc;
  const void* g;
  float scale;
  ColMap map;
  template <class A, int E>
  __device__ __forceinline__ void apply(A (&v)[1 << E], int hi, int lo, int s) const {
#pragma unroll
    for (int r = 0; r < (1 << E); ++r) {
      const int i = hi | (r << s) | lo;
      acc[swz(i)] = acc[swz(i)] + mul_scale(tx[swz(i)] * v[r], scale);
      v[r] = v[r] * Tr<D>::gain(g, map(i), scale);
    }
    bfly_regs<A, E>(v);
  }
};

// ---- global <-> tile movement ----
template <int D>
__device__ __forceinline__ void load_contig(typename Tr<D>::A* tile, const void* src, long long base, int n) {
  using A = typename Tr<D>::A;
  for (int i = threadIdx.x; i < TILE; i += THREADS) tile[swz(i)] = i < n ? Tr<D>::ld(src, base + i) : A(0);
}
template <int D>
__device__ __forceinline__ void store_contig(const typename Tr<D>::A* tile, void* dst, long long base, int n) {
  for (int i = threadIdx.x; i < n; i += THREADS) Tr<D>::st(dst, base + i, tile[swz(i)]);
}
template <class A>
__device__ __forceinline__ void load_ws_contig(A* tile, const A* src, long long base) {
  for (int i = threadIdx.x; i < TILE; i += THREADS) tile[swz(i)] = ld_ws(src, base + i);
}
template <class A>
__device__ __forceinline__ void store_ws_contig(const A* tile, A* dst, long long base) {
  for (int i = threadIdx.x; i < TILE; i += THREADS) dst[base + i] = tile[swz(i)];
}
// column tile: i = (row << w) | c  <->  base + (row << s) + c (rows of stride 2^s, s = 13 in plan M)
template <class A>
__device__ __forceinline__ void load_ws_col(A* tile, const A* src, long long base, int w, int s = TILE_BITS) {
  for (int i = threadIdx.x; i < TILE; i += THREADS)
    tile[swz(i)] = ld_ws(src, base + (static_cast<long long>(i >> w) << s) + (i & ((1 << w) - 1)));
}
template <class A>
__device__ __forceinline__ void store_ws_col(const A* tile, A* dst, long long base, int w, int s = TILE_BITS) {
  for (int i = threadIdx.x; i < TILE; i += THREADS)
    dst[base + (static_cast<long long>(i >> w) << s) + (i & ((1 << w) - 1))] = tile[swz(i)];
}

// ---- device-wide barrier with a bounded wait ----
__device__ __forceinline__ unsigned long long global_ns() {
  unsigned long long t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}
__device__ __forceinline__ unsigned int ld_acquire(const unsigned int* p) {
  unsigned int v;
  asm volatile("ld.acquire.gpu.global.b32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}

__device__ __forceinline__ void st_relaxed(unsigned int* p, unsigned int v) {
  asm volatile("st.relaxed.gpu.global.b32 [%0], %1;" ::"l"(p), "r"(v) : "memory");
}
__device__ __forceinline__ void red_release_add(unsigned int* p, unsigned int v) {
  asm volatile("red.release.gpu.global.add.u32 [%0], %1;" ::"l"(p), "r"(v) : "memory");
}
__device__ __forceinline__ unsigned int* barrier_slot(GridBarrier* b, unsigned int k) {
  k &= 3u;
  return k < 2 ? &b->slot01[k] : &b->slot23[k - 2];
}

// Programmatic dependent launch.  The kernels are launched with programmatic stream
// serialisation, so a kernel's CTAs may start (allocate tensor memory, set up shared memory) while
// the previous kernel in the stream is finishing.  Before touching global memory every such kernel
// waits (pdl_wait) until that kernel has completed and its writes are visible; when its own work is
// done it lets the next kernel begin launching (pdl_trigger).  Triggering only at the end measured
// best: an early trigger slowed a forward/backward pair by ~35 us (512 against 477 us at
// [16, 8192, 256]) while the late one keeps the gain on back-to-back forwards (44.2 against 47.0 us
// at [1, 65536, 128]).  Without the launch attribute both are no-ops.
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void pdl_trigger() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }

// Device-wide barrier of a persistent grid of at most the resident-CTA count (every CTA becomes
// resident as SMs free up; kernels that occupied SMs for ever would make the wait run out instead
// of hanging); every CTA calls it the same number of times.  Returns false (and sets bar->err) if this CTA gave up after BARRIER_TIMEOUT_NS; the
// caller then returns.
// Barrier k: thread 0 of each CTA adds one (release) to slot k mod 4 and polls (acquire) until
// the slot holds gridDim.x -- the arrivals themselves release the waiters, with no second word
// to publish.  A slot is cleared by CTA 0 once it has passed the barrier after the slot's (every
// CTA has then left the slot's barrier), which is three barriers before the slot is used again.
// The barrier number continues from call to call (seq, read once at kernel start and updated by
// CTA 0 after each barrier; every CTA has read it by the time CTA 0 passes its first barrier), so
// the slot left full by a call's last barrier is cleared at the next call's first one.  Must be
// constructed after pdl_wait().
struct GridSync {
  GridBarrier* bar;
  int* flag;          // shared: thread 0's verdict for the CTA
  unsigned int k;     // thread 0: number of the next barrier
  __device__ __forceinline__ GridSync(GridBarrier* b, int* f) : bar(b), flag(f), k(0) {
    if (threadIdx.x == 0) k = ld_acquire(&b->seq);
  }
  __device__ __forceinline__ bool operator()() {
    __syncthreads();
    if (threadIdx.x == 0) {
      int ok = 1;
      unsigned int* c = barrier_slot(bar, k);
      red_release_add(c, 1u);
      // Poll without sleeping (the wait is ~1 us and a sleep quantum would add to it); the clock
      // is read once per 256 polls to bound the wait.
      const unsigned long long t0 = global_ns();
      for (unsigned int polls = 1; ld_acquire(c) != gridDim.x; ++polls) {
        if ((polls & 255u) == 0 && global_ns() - t0 > BARRIER_TIMEOUT_NS) {
          atomicOr(&bar->err, 1u);
          ok = 0;
          break;
        }
      }
      ++k;
      if (ok && blockIdx.x == 0) {
        // plain stores: nobody else writes these words now, and the next arrival's release
        // orders them before any later use of the slot
        st_relaxed(barrier_slot(bar, k - 2), 0u);  // the slot of the barrier before this one
        st_relaxed(&bar->seq, k);
      }
      *flag = ok;
    }
    __syncthreads();
    return *flag != 0;
  }
};

// ---------------------------------------------------------------------------------------------
// Forward, plan S (no device-wide barrier: launched as an ordinary persistent grid).
template <int D>
__global__ void __launch_bounds__(THREADS) k_forward_s(Params P) {
  using A = typename Tr<D>::A;
  extern __shared__ __align__(16) unsigned char smem_raw[];
  pdl_wait();
  A* tA = reinterpret_cast<A*>(smem_raw);
  const int m = P.m;
  const long long ppt = 1ll << (TILE_BITS - m);
  const long long ntiles = (P.B + ppt - 1) / ppt;
  const GainMid<D, PlaneMap> mid{P.g, P.scale, PlaneMap{(1 << m) - 1}};
  for (long long t = blockIdx.x; t < ntiles; t += gridDim.x) {
    const long long b0 = t * ppt;
    const int n = static_cast<int>(min(ppt, P.B - b0) << m);
    load_contig<D>(tA, P.x, b0 << m, n);
    __syncthreads();
    xform_mid_xform(tA, 0, m, mid);
    store_contig<D>(tA, P.y, b0 << m, n);
    __syncthreads();
  }
  pdl_trigger();
}

// Forward, plan M (a grid of resident CTAs: device-wide barriers between phases).
template <int D>
__global__ void __launch_bounds__(THREADS) k_forward_m(Params P) {
  using A = typename Tr<D>::A;
  extern __shared__ __align__(16) unsigned char smem_raw[];
  __shared__ int flag;
  pdl_wait();
  GridSync gsync(P.bar, &flag);
  A* tA = reinterpret_cast<A*>(smem_raw);
  A* ws = static_cast<A*>(P.ws);
  const int m = P.m, q = m - TILE_BITS, w = TILE_BITS - q;
  const long long L = 1ll << m;
  for (long long b0 = 0; b0 < P.B; b0 += P.gp) {
    const long long nb = min(static_cast<long long>(P.gp), P.B - b0);
    const long long units = nb << q;
    // phase 1: bits [0, 13) of each row tile, X -> ws
    for (long long u = blockIdx.x; u < units; u += gridDim.x) {
      const long long b = u >> q, rt = u & ((1ll << q) - 1);
      load_contig<D>(tA, P.x, ((b0 + b) << m) + (rt << TILE_BITS), TILE);
      __syncthreads();
      xform(tA, 0, TILE_BITS);
      store_ws_contig(tA, ws, (b << m) + (rt << TILE_BITS));
      __syncthreads();
    }
    if (!gsync()) return;
    // phase 2: bits [13, m) forward, gain, inverse on each column tile, ws -> ws
    for (long long u = blockIdx.x; u < units; u += gridDim.x) {
      const long long b = u >> q, col0 = (u & ((1ll << q) - 1)) << w;
      load_ws_col(tA, ws, (b << m) + col0, w);
      __syncthreads();
      xform_mid_xform(tA, w, TILE_BITS, GainMid<D, ColMap>{P.g, P.scale, ColMap{w, col0}});
      store_ws_col(tA, ws, (b << m) + col0, w);
      __syncthreads();
    }
    if (!gsync()) return;
    // phase 3: bits [0, 13) again, ws -> Y
    for (long long u = blockIdx.x; u < units; u += gridDim.x) {
      const long long b = u >> q, rt = u & ((1ll << q) - 1);
      load_ws_contig(tA, ws, (b << m) + (rt << TILE_BITS));
      __syncthreads();
      xform(tA, 0, TILE_BITS);
      store_contig<D>(tA, P.y, ((b0 + b) << m) + (rt << TILE_BITS), TILE);
      __syncthreads();
    }
    if (b0 + P.gp < P.B && !gsync()) return;
    (void)L;
  }
  pdl_trigger();
}

// Backward, plan S: dX per tile, partial products per plane, then dG summed over b ascending.
template <int D>
__global__ void __launch_bounds__(THREADS) k_backward_s(Params P) {
  using A = typename Tr<D>::A;
  extern __shared__ __align__(16) unsigned char smem_raw[];
  __shared__ int flag;
  pdl_wait();
  GridSync gsync(P.bar, &flag);
  A* tA = reinterpret_cast<A*>(smem_raw);
  A* tB = tA + TILE;
  A* ws = static_cast<A*>(P.ws);
  A* dg = static_cast<A*>(P.dg);
  const int m = P.m;
  const long long L = 1ll << m;
  const long long ppt = 1ll << (TILE_BITS - m);
  for (long long b0 = 0; b0 < P.B; b0 += P.gp) {
    const long long nb = min(static_cast<long long>(P.gp), P.B - b0);
    const long long ntiles = (nb + ppt - 1) / ppt;
    for (long long t = blockIdx.x; t < ntiles; t += gridDim.x) {
      const long long tb = t * ppt;  // first plane of the tile, within the group
      const int n = static_cast<int>(min(ppt, nb - tb) << m);
      load_contig<D>(tA, P.x, (b0 + tb) << m, n);
      load_contig<D>(tB, P.dy, (b0 + tb) << m, n);
      __syncthreads();
      xform(tA, 0, m);
      xform_mid_xform(tB, 0, m, BwdMidS<D>{tA, ws + (tb << m), n, P.g, P.scale, static_cast<int>(L - 1)});
      store_contig<D>(tB, P.dx, (b0 + tb) << m, n);
      __syncthreads();
    }
    if (!gsync()) return;
    for (long long l = blockIdx.x * (long long)THREADS + threadIdx.x; l < L; l += (long long)gridDim.x * THREADS) {
      A acc = b0 == 0 ? A(0) : ld_ws(dg, l);
      for (long long b = 0; b < nb; ++b) acc = acc + ld_ws(ws, (b << m) + l);
      dg[l] = acc;
    }
    if (b0 + P.gp < P.B && !gsync()) return;
  }
  pdl_trigger();
}

// Backward, plan M: phase 1 row tiles of X and dY -> workspaces; phase 2 each column tile loops
// over the group's planes in ascending b, accumulating dG and running the gain step; phase 3
// row tiles -> dX.
template <int D>
__global__ void __launch_bounds__(THREADS) k_backward_m(Params P) {
  using A = typename Tr<D>::A;
  extern __shared__ __align__(16) unsigned char smem_raw[];
  __shared__ int flag;
  pdl_wait();
  GridSync gsync(P.bar, &flag);
  A* tA = reinterpret_cast<A*>(smem_raw);
  A* tB = tA + TILE;
  A* tC = tB + TILE;
  const int m = P.m, q = m - TILE_BITS, w = TILE_BITS - q;
  A* wsx = static_cast<A*>(P.ws);
  A* wsd = wsx + (static_cast<long long>(P.gp) << m);
  A* dg = static_cast<A*>(P.dg);
  for (long long b0 = 0; b0 < P.B; b0 += P.gp) {
    const long long nb = min(static_cast<long long>(P.gp), P.B - b0);
    const long long units = nb << q;
    for (long long u = blockIdx.x; u < 2 * units; u += gridDim.x) {
      const bool is_dy = u >= units;
      const long long uu = is_dy ? u - units : u;
      const long long b = uu >> q, rt = uu & ((1ll << q) - 1);
      load_contig<D>(tA, is_dy ? P.dy : P.x, ((b0 + b) << m) + (rt << TILE_BITS), TILE);
      __syncthreads();
      xform(tA, 0, TILE_BITS);
      store_ws_contig(tA, is_dy ? wsd : wsx, (b << m) + (rt << TILE_BITS));
      __syncthreads();
    }
    if (!gsync()) return;
    for (long long ct = blockIdx.x; ct < (1ll << q); ct += gridDim.x) {
      const long long col0 = ct << w;
      if (b0 == 0) {
        for (int i = threadIdx.x; i < TILE; i += THREADS) tC[i] = A(0);
      } else {
        load_ws_col(tC, dg, col0, w);
      }
      for (long long b = 0; b < nb; ++b) {
        load_ws_col(tA, wsx, (b << m) + col0, w);
        load_ws_col(tB, wsd, (b << m) + col0, w);
        __syncthreads();
        xform(tA, w, TILE_BITS);
        xform_mid_xform(tB, w, TILE_BITS, BwdMidM<D>{tA, tC, P.g, P.scale, ColMap{w, col0}});
        store_ws_col(tB, wsd, (b << m) + col0, w);
        __syncthreads();
      }
      store_ws_col(tC, dg, col0, w);
      __syncthreads();
    }
    if (!gsync()) return;
    for (long long u = blockIdx.x; u < units; u += gridDim.x) {
      const long long b = u >> q, rt = u & ((1ll << q) - 1);
      load_ws_contig(tA, wsd, (b << m) + (rt << TILE_BITS));
      __syncthreads();
      xform(tA, 0, TILE_BITS);
      store_contig<D>(tA, P.dx, ((b0 + b) << m) + (rt << TILE_BITS), TILE);
      __syncthreads();
    }
    if (b0 + P.gp < P.B && !gsync()) return;
  }
  pdl_trigger();
}

// ---------------------------------------------------------------------------------------------
// Plan L passes (26 < m <= 30), each its own launch over nb planes of the group (planes b0 ... of
// X, Y, dY, dX; planes 0 ... of the workspaces).
//
// Row pass in: each row tile (2^13 contiguous elements) of `src` (dtype D), bits [0, 13) -> ws.
template <int D>
__global__ void __launch_bounds__(THREADS) k_pass_rows_in(const void* src, typename Tr<D>::A* ws, long long b0,
                                                          long long nb, int m) {
  using A = typename Tr<D>::A;
  extern __shared__ __align__(16) unsigned char smem_raw[];
  pdl_wait();
  A* tA = reinterpret_cast<A*>(smem_raw);
  const int q = m - TILE_BITS;
  for (long long u = blockIdx.x; u < (nb << q); u += gridDim.x) {
    const long long b = u >> q, rt = u & ((1ll << q) - 1);
    load_contig<D>(tA, src, ((b0 + b) << m) + (rt << TILE_BITS), TILE);
    __syncthreads();
    xform(tA, 0, TILE_BITS);
    store_ws_contig(tA, ws, (b << m) + (rt << TILE_BITS));
    __syncthreads();
  }
  pdl_trigger();
}

// Row pass out: each row tile of ws, bits [0, 13) -> `dst` (dtype D).
template <int D>
__global__ void __launch_bounds__(THREADS) k_pass_rows_out(const typename Tr<D>::A* ws, void* dst, long long b0,
                                                           long long nb, int m) {
  using A = typename Tr<D>::A;
  extern __shared__ __align__(16) unsigned char smem_raw[];
  pdl_wait();
  A* tA = reinterpret_cast<A*>(smem_raw);
  const int q = m - TILE_BITS;
  for (long long u = blockIdx.x; u < (nb << q); u += gridDim.x) {
    const long long b = u >> q, rt = u & ((1ll << q) - 1);
    load_ws_contig(tA, ws, (b << m) + (rt << TILE_BITS));
    __syncthreads();
    xform(tA, 0, TILE_BITS);
    store_contig<D>(tA, dst, ((b0 + b) << m) + (rt << TILE_BITS), TILE);
    __syncthreads();
  }
  pdl_trigger();
}

// A column tile of the bit group [s, s + k) (k + w = 13): 2^w adjacent elements of each of 2^k rows
// of stride 2^s, i.e. varying bits [0, w) and [s, s + k); tile t fixes bits [w, s) and [s + k, m).
__device__ __forceinline__ long long col_tile_base(long long t, int w, int s, int k) {
  return ((t & ((1ll << (s - w)) - 1)) << w) | ((t >> (s - w)) << (s + k));
}

// Column pass: bits [s, s + k) of every column tile of nb planes of ws, in place; with gain != 0
// the forward bits, the gain G/L (no scale for int32) and the same bits again.
template <int D>
__global__ void __launch_bounds__(THREADS) k_pass_cols(typename Tr<D>::A* ws, long long nb, int m, int s, int k,
                                                       const void* g, float scale, int gain) {
  using A = typename Tr<D>::A;
  extern __shared__ __align__(16) unsigned char smem_raw[];
  pdl_wait();
  A* tA = reinterpret_cast<A*>(smem_raw);
  const int q = m - TILE_BITS, w = TILE_BITS - k;
  for (long long u = blockIdx.x; u < (nb << q); u += gridDim.x) {
    const long long b = u >> q, base = col_tile_base(u & ((1ll << q) - 1), w, s, k);
    load_ws_col(tA, ws, (b << m) + base, w, s);
    __syncthreads();
    if (gain)
      xform_mid_xform(tA, w, TILE_BITS, GainMid<D, ColMap>{g, scale, ColMap{w, base, s}});
    else
      xform(tA, w, TILE_BITS);
    store_ws_col(tA, ws, (b << m) + base, w, s);
    __syncthreads();
  }
  pdl_trigger();
}

// Backward gain pass: bits [s, s + k) of the X and dY planes of the group; each column tile owns
// its dG positions and, in ascending b, adds the planes' (W X)(W dY)/L to them (starting from 0
// for the first group, else from dG), applies the gain to dY and runs dY's bits back.
template <int D>
__global__ void __launch_bounds__(THREADS) k_pass_cols_bwd(typename Tr<D>::A* wsx, typename Tr<D>::A* wsd,
                                                           typename Tr<D>::A* dg, long long nb, int m, int s, int k,
                                                           const void* g, float scale, int first) {
  using A = typename Tr<D>::A;
  extern __shared__ __align__(16) unsigned char smem_raw[];
  pdl_wait();
  A* tA = reinterpret_cast<A*>(smem_raw);
  A* tB = tA + TILE;
  A* tC = tB + TILE;
  const int q = m - TILE_BITS, w = TILE_BITS - k;
  for (long long t = blockIdx.x; t < (1ll << q); t += gridDim.x) {
    const long long base = col_tile_base(t, w, s, k);
    if (first) {
      for (int i = threadIdx.x; i < TILE; i += THREADS) tC[i] = A(0);
    } else {
      load_ws_col(tC, dg, base, w, s);
    }
    for (long long b = 0; b < nb; ++b) {
      load_ws_col(tA, wsx, (b << m) + base, w, s);
      load_ws_col(tB, wsd, (b << m) + base, w, s);
      __syncthreads();
      xform(tA, w, TILE_BITS);
      xform_mid_xform(tB, w, TILE_BITS, BwdMidM<D>{tA, tC, g, scale, ColMap{w, base, s}});
      store_ws_col(tB, wsd, (b << m) + base, w, s);
      __syncthreads();
    }
    store_ws_col(tC, dg, base, w, s);
    __syncthreads();
  }
  pdl_trigger();
}

}  // namespace whtmix
