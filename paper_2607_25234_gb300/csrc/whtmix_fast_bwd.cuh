// whtmix_fast_bwd.cuh -- register/TMEM backward kernel for planes of 2^14 <= N*C <= 2^23 elements,
// fp32 and bf16 I/O.
//
// The backward of the Section III-B mixer Y = W (G o W X) with W = H_N . H_C / sqrt(NC):
//   dX_b = W (G o W dY_b)                       (W is symmetric, the map is its own adjoint)
//   dG   = sum_b (W X_b) o (W dY_b)             (summed over b = 0, 1, ..., B-1 in that order)
// Both need the 2D transforms of X_b and dY_b up to the gain step, so one kernel runs the fast
// forward's three phases over X and dY together, per group of planes:
//   phase 1  rows of X_b and dY_b: R bits forward                      X, dY -> wsx, wsd
//   phase 2  every column of both: Q bits forward; the product
//            (W X)(W dY) (unnormalised, times 1/L) replaces the X column
//            in wsx; the dY column takes the gain G/L and its Q bits
//            again                                                       wsx, wsd -> wsx, wsd
//   phase 3  rows of wsd: R bits again -> dX; then dG at this CTA's
//            positions: dG (0 for the first group) + the group's products in ascending b
// with the bounded device-wide barrier between phases and between groups.  A thread owns one
// column of 2^Q rows as 2^(Q-1) register pairs (j, j + 2^(Q-1)).  For Q <= 6 the transformed X
// column stays in registers beside the dY column; for Q = 7 (128 rows) it is parked in the
// thread's TMEM lane (the two warps w and w+4 that share a lane quarter use columns [0, 128) and
// [128, 256)) while the dY column is transformed.  Columns of 256 and 512 rows (Q = 8, 9, rows of
// 2^14) take the forward's TMEM column pass twice: the X columns' bits forward in place, then the
// dY columns, whose gain step also turns the X column into the product.  Because each thread
// reduces the same dG positions in every group, dG's summation order is exactly b = 0, 1, ..., B-1.
#pragma once

#include "whtmix_fast.cuh"

namespace whtmix {
namespace fast {

// Phase 2 of the backward for 2^Q-row columns (Q <= 7).  Units are storage positions of the
// group's planes, u = (b << R) + sp; a thread takes units u_begin + threadIdx.x + k * THREADS.
template <int Q, int R>
__device__ __forceinline__ void col_pass_bwd(float* wsx, float* wsd, const float* g, float scale, int m,
                                             long long u_begin, long long u_end, uint32_t tcol) {
  constexpr int NP = 1 << (Q - 1);    // register pairs per column
  constexpr bool STASH = Q == 7;      // transformed X column parked in TMEM
  static_assert(Q >= 1 && Q <= 7, "column height");
  const float2 sc = make_float2(scale, scale);
  for (long long u0 = u_begin; u0 < u_end; u0 += THREADS) {
    const long long u = u0 + threadIdx.x;
    const bool active = u < u_end;
    // TMEM loads and stores are warp-collective: with STASH every lane runs every pass (idle lanes
    // on a valid column, storing nothing); without it idle lanes leave
    if (!STASH && !active) break;
    const long long uu = active ? u : u_begin;
    const long long b = uu >> R;
    const int sp = static_cast<int>(uu & ((1 << R) - 1));
    float* xc = wsx + (b << m) + sp;
    float* dc = wsd + (b << m) + sp;
    const float* gb = g + sigma_inv(sp);
    float2 v[NP];
    float2 xh[NP];
#pragma unroll
    for (int j = 0; j < NP; ++j)
      v[j] = make_float2(__ldcg(xc + (static_cast<long long>(j) << R)), __ldcg(xc + (static_cast<long long>(j + NP) << R)));
    bfly_all<NP>(v);
#pragma unroll
    for (int j = 0; j < NP; ++j) bf_in(v[j]);
    if constexpr (STASH) {
#pragma unroll
      for (int q = 0; q < NP / 16; ++q) {
        float lo[16], hi[16];
#pragma unroll
        for (int i = 0; i < 16; ++i) {
          lo[i] = v[16 * q + i].x;
          hi[i] = v[16 * q + i].y;
        }
        tmem_st16(tcol + 16 * q, lo);
        tmem_st16(tcol + NP + 16 * q, hi);
      }
    } else {
#pragma unroll
      for (int j = 0; j < NP; ++j) xh[j] = v[j];
    }
#pragma unroll
    for (int j = 0; j < NP; ++j)
      v[j] = make_float2(__ldcg(dc + (static_cast<long long>(j) << R)), __ldcg(dc + (static_cast<long long>(j + NP) << R)));
    bfly_all<NP>(v);
#pragma unroll
    for (int j = 0; j < NP; ++j) bf_in(v[j]);
    if constexpr (STASH) tmem_wait_st();
#pragma unroll
    for (int q = 0; q < (NP + 15) / 16; ++q) {
      float lo[16], hi[16];
      if constexpr (STASH) {
        tmem_ld16(tcol + 16 * q, lo);
        tmem_ld16(tcol + NP + 16 * q, hi);
        tmem_wait_ld();
      }
#pragma unroll
      for (int i = 0; i < 16; ++i) {
        const int j = 16 * q + i;
        if (j < NP) {
          float2 xj;
          if constexpr (STASH) xj = make_float2(lo[i], hi[i]);
          else xj = xh[j];
          const float2 p = mul2(mul2(xj, v[j]), sc);
          if (active) {
            __stcg(xc + (static_cast<long long>(j) << R), p.x);
            __stcg(xc + (static_cast<long long>(j + NP) << R), p.y);
          }
          const float2 gg = make_float2(__ldg(gb + (static_cast<long long>(j) << R)), __ldg(gb + (static_cast<long long>(j + NP) << R)));
          v[j] = mul2(v[j], mul2(gg, sc));
        }
      }
    }
#pragma unroll
    for (int j = 0; j < NP; ++j) bf_in(v[j]);
    bfly_all<NP>(v);
    if (active) {
#pragma unroll
      for (int j = 0; j < NP; ++j) {
        __stcg(dc + (static_cast<long long>(j) << R), v[j].x);
        __stcg(dc + (static_cast<long long>(j + NP) << R), v[j].y);
      }
    }
  }
}

// dG at plane positions [lb, le) (multiples of 4): dG (or 0 for the first group) plus the
// group's nb product planes in ascending b.  Position l of a workspace row is storage position
// l mod 2^R; dG is indexed by the logical position sigma_inv of it (r0, r1 map to themselves, so
// four consecutive storage positions are four consecutive dG entries).
template <int R>
__device__ __forceinline__ void dg_reduce(float* dg, const float* wsx, int m, long long nb, bool first,
                                          long long lb, long long le) {
  for (long long l = lb + 4 * threadIdx.x; l < le; l += 4 * THREADS) {
    const long long row = l >> R;
    const int sp = static_cast<int>(l & ((1 << R) - 1));
    float4* dp = reinterpret_cast<float4*>(dg + (row << R) + sigma_inv(sp));
    float4 acc = first ? make_float4(0.f, 0.f, 0.f, 0.f) : __ldcg(dp);
    for (long long b = 0; b < nb; ++b) {
      const float4 p = __ldcg(reinterpret_cast<const float4*>(wsx + (b << m) + l));
      acc.x += p.x;
      acc.y += p.y;
      acc.z += p.z;
      acc.w += p.w;
    }
    __stcg(dp, acc);
  }
}

// Backward kernel: persistent grid (one CTA per SM, all resident).  P.ws holds wsx (P.gp planes)
// followed by wsd (P.gp planes).
template <int D, int R, int Q>
__global__ void __launch_bounds__(THREADS, 1) k_backward_fast(Params P) {
  static_assert((R == 13 && Q >= 1 && Q <= 7) || (R == 14 && Q >= 7 && Q <= 9), "supported row/column split");
  extern __shared__ __align__(16) unsigned char smem_raw[];
  __shared__ int flag;
  __shared__ uint32_t tmem_slot;
  constexpr bool USE_TMEM = Q >= 7;
  using RW = Row<R>;
  float* sm = reinterpret_cast<float*>(smem_raw);
  const int worker = threadIdx.x / RW::WORKER, wt = threadIdx.x % RW::WORKER;
  float* xbuf = sm + worker * RW::LEN;
  float* stg = sm + SMEM_XBUF_BYTES / sizeof(float) + worker * RW::STAGE;
  const int m = R + Q;
  float* wsx = static_cast<float*>(P.ws);
  float* wsd = wsx + (static_cast<long long>(P.gp) << m);
  const float* g = static_cast<const float*>(P.g);
  float* dg = static_cast<float*>(P.dg);
  uint32_t tcol = 0;
  if constexpr (USE_TMEM) {
    if (threadIdx.x < 32) tmem_alloc_512(&tmem_slot);
    tmem_fence_before();
    __syncthreads();
    tmem_fence_after();
    // lane quarter of this warp; for Q = 7 warps w and w + 4 take TMEM columns [0, 128) and
    // [128, 256); the column passes of Q = 8, 9 split the lane between the two warps themselves
    tcol = tmem_slot + (static_cast<uint32_t>(32 * ((threadIdx.x >> 5) & 3)) << 16) + (Q == 7 ? 128u * (threadIdx.x >> 7) : 0u);
  }
  // tensor memory is allocated before the wait: the previous kernel's CTA on this SM has left
  pdl_wait();
  GridSync gsync(P.bar, &flag);
  const long long L = 1ll << m;
  const long long lb = ((L >> 2) * blockIdx.x / gridDim.x) << 2, le = ((L >> 2) * (blockIdx.x + 1) / gridDim.x) << 2;
  for (long long b0 = 0; b0 < P.B; b0 += P.gp) {
    const long long nb = min(static_cast<long long>(P.gp), P.B - b0);
    const long long rows = nb << Q;
    // phase 1: units [0, rows) are rows of X, [rows, 2 rows) rows of dY; balanced per CTA
    {
      const long long ub = 2 * rows * blockIdx.x / gridDim.x, ue = 2 * rows * (blockIdx.x + 1) / gridDim.x;
      auto src_of = [&](long long u) -> const void* { return u < rows ? P.x : P.dy; };
      if (ub + worker < ue) {
        long long e0;
        int lim;
        const long long u = ub + worker;
        row_loc<R, Q>(b0, u < rows ? u : u - rows, P.lv, &e0, &lim);
        stage_row_in<D, R>(src_of(u), e0, stg, wt, lim);
      }
      for (long long u = ub + worker; u < ue; u += RW::NWORKERS) {
        const long long un = u + RW::NWORKERS;
        // G is first read in phase 2: its fetch into L2 is spread over the first group's rows
        if (b0 == 0 && wt == 0) l2_prefetch_piece(g, 4ll << m, u - ub, ue - ub);
        float* dst = u < rows ? wsx + (u << R) : wsd + ((u - rows) << R);
        long long e0, e0n;
        int lim, limn;
        row_loc<R, Q>(b0, u < rows ? u : u - rows, P.lv, &e0, &lim);
        row_loc<R, Q>(b0, un < rows ? un : un - rows, P.lv, &e0n, &limn);
        row_forward_in<D, R>(src_of(u), e0, lim, dst, xbuf, stg, wt, worker, un < ue ? src_of(un) : nullptr, e0n, limn);
      }
    }
    if (!gsync()) break;
    // phase 2: columns of both, product, gain
    {
      const long long cols = nb << R;
      const long long cb = ((cols * blockIdx.x / gridDim.x) + 4) & ~7ll;
      const long long ce = blockIdx.x + 1 == gridDim.x ? cols : ((cols * (blockIdx.x + 1) / gridDim.x) + 4) & ~7ll;
      if constexpr (Q >= 8) {
        // columns of 256 or 512 rows: the X columns' bits forward (stored in place), then the dY
        // columns with the products written over the X columns at the gain step
        const FullGain<R> gain{g};
        col_pass_tmem<Q, R, FullGain<R>, 1>(wsx, gain, P.scale, m, cb, ce, tcol);
        col_pass_tmem<Q, R, FullGain<R>, 2>(wsd, gain, P.scale, m, cb, ce, tcol, wsx);
      } else {
        col_pass_bwd<Q, R>(wsx, wsd, g, P.scale, m, cb, ce, tcol);
      }
    }
    if (!gsync()) break;
    // phase 3: wsd -> dX, row bits; then this CTA's dG positions
    {
      const long long rb = rows * blockIdx.x / gridDim.x, re = rows * (blockIdx.x + 1) / gridDim.x;
      if (rb + worker < re) stage_row_out<R>(wsd + ((rb + worker) << R), stg, wt);
      for (long long r = rb + worker; r < re; r += RW::NWORKERS) {
        const long long rn = r + RW::NWORKERS;
        long long e0;
        int lim;
        row_loc<R, Q>(b0, r, P.lv, &e0, &lim);
        row_forward_out<D, R>(wsd + (r << R), P.dx, e0, lim, xbuf, stg, wt, worker, rn < re ? wsd + (rn << R) : nullptr);
      }
      dg_reduce<R>(dg, wsx, m, nb, b0 == 0, lb, le);
    }
    if (b0 + P.gp < P.B && !gsync()) break;
  }
  pdl_trigger();
  if constexpr (USE_TMEM) {
    tmem_fence_before();
    __syncthreads();
    tmem_fence_after();
    if (threadIdx.x < 32) tmem_dealloc_512(tmem_slot);
  }
}

}  // namespace fast
}  // namespace whtmix
