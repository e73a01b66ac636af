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
constexpr int MAX_PLANE_BITS = 2 * TILE_BITS;
constexpr int ROUND_BITS = 5;
constexpr unsigned long long BARRIER_TIMEOUT_NS = 1000000000ull;  // 1 s

enum DType { DT_F32 = 0, DT_BF16 = 1, DT_I32 = 2 };

// Device-wide barrier state; lives in the first 256 bytes of the workspace.
struct GridBarrier {
  unsigned int count;      // arrivals at a barrier of even generation (back to 0 after it)
  unsigned int gen;        // generation, bumped by the last arrival
  unsigned int err;        // non-zero once a wait gave up
  unsigned int count_odd;  // arrivals at a barrier of odd generation (back to 0 after it)
  unsigned int pad[60];
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
struct ColMap {  // plan M column tile: i = (row << w) | c  ->  (row << 13) + col0 + c
  int w;
  long long col0;
  __device__ __forceinline__ long long operator()(int i) const {
    return (static_cast<long long>(i >> w) << TILE_BITS) + col0 + (i & ((1 << w) - 1));
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
// column tile: i = (row << w) | c  <->  base + (row << 13) + c
template <class A>
__device__ __forceinline__ void load_ws_col(A* tile, const A* src, long long base, int w) {
  for (int i = threadIdx.x; i < TILE; i += THREADS)
    tile[swz(i)] = ld_ws(src, base + (static_cast<long long>(i >> w) << TILE_BITS) + (i & ((1 << w) - 1)));
}
template <class A>
__device__ __forceinline__ void store_ws_col(const A* tile, A* dst, long long base, int w) {
  for (int i = threadIdx.x; i < TILE; i += THREADS)
    dst[base + (static_cast<long long>(i >> w) << TILE_BITS) + (i & ((1 << w) - 1))] = tile[swz(i)];
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

// Device-wide barrier of a cooperative launch; every CTA calls it the same number of times.
// Returns false (and sets bar->err) if this CTA gave up after BARRIER_TIMEOUT_NS; the caller
// then returns.  Thread 0 of each CTA reads the generation word once, at kernel start (it cannot
// advance before this CTA arrives), and counts the barriers itself afterwards, so an arrival is
// one fence and one atomic.  Barriers of even and odd generation count arrivals in separate words:
// the last arrival releases the others first and clears its counter afterwards, off the critical
// path, since that counter is next used two barriers later, which no CTA reaches before the last
// arrival has passed the barrier in between.
struct GridSync {
  GridBarrier* bar;
  int* flag;          // shared: thread 0's verdict for the CTA
  unsigned int gen;   // thread 0: generation of the next barrier
  __device__ __forceinline__ GridSync(GridBarrier* b, int* f) : bar(b), flag(f), gen(0) {
    if (threadIdx.x == 0) gen = ld_acquire(&b->gen);
  }
  __device__ __forceinline__ bool operator()() {
    __syncthreads();
    if (threadIdx.x == 0) {
      int ok = 1;
      unsigned int* count = (gen & 1u) ? &bar->count_odd : &bar->count;
      __threadfence();
      const unsigned int arrived = atomicAdd(count, 1u);
      if (arrived == gridDim.x - 1) {
        __threadfence();
        atomicAdd(&bar->gen, 1u);
        atomicExch(count, 0u);
      } else {
        // Spin on the generation word (no sleep: the wait is ~1 us and a sleep quantum would add
        // to it); the clock is read once per 256 polls to bound the wait.
        const unsigned long long t0 = global_ns();
        for (unsigned int polls = 1; ld_acquire(&bar->gen) == gen; ++polls) {
          if ((polls & 255u) == 0 && global_ns() - t0 > BARRIER_TIMEOUT_NS) {
            atomicOr(&bar->err, 1u);
            ok = 0;
            break;
          }
        }
      }
      __threadfence();
      ++gen;
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
}

// Forward, plan M (cooperative launch: device-wide barriers between phases).
template <int D>
__global__ void __launch_bounds__(THREADS) k_forward_m(Params P) {
  using A = typename Tr<D>::A;
  extern __shared__ __align__(16) unsigned char smem_raw[];
  __shared__ int flag;
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
}

// Backward, plan S: dX per tile, partial products per plane, then dG summed over b ascending.
template <int D>
__global__ void __launch_bounds__(THREADS) k_backward_s(Params P) {
  using A = typename Tr<D>::A;
  extern __shared__ __align__(16) unsigned char smem_raw[];
  __shared__ int flag;
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
}

// Backward, plan M: phase 1 row tiles of X and dY -> workspaces; phase 2 each column tile loops
// over the group's planes in ascending b, accumulating dG and running the gain step; phase 3
// row tiles -> dX.
template <int D>
__global__ void __launch_bounds__(THREADS) k_backward_m(Params P) {
  using A = typename Tr<D>::A;
  extern __shared__ __align__(16) unsigned char smem_raw[];
  __shared__ int flag;
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
}

}  // namespace whtmix
