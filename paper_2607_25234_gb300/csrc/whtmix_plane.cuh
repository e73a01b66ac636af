// whtmix_plane.cuh -- forward for planes of 2^14 <= N*C <= 2^16 elements, one plane per CTA, the
// whole fp32 plane held in the SM's tensor memory (Section III-B, Eq. 2-3:
// Y = H_N (G o (H_N X H_C)) H_C / (N C), flattened to one 2^m-point transform).
//
// A plane is NR = 2^CB rows of 2^14 elements (CB = m - 14 <= 2); a CTA has two row workers of 128
// threads and TMEM's 512 columns x 128 lanes (256 KiB) hold up to four fp32 rows: row r lives in
// columns [256 (r mod 2) + 128 (r / 2), +128) of the lanes of worker r mod 2, thread wt in lane wt.
//   phase 1  each worker, for each of its rows (the next one prefetched by cp.async): X row -> 14
//            row bits in registers and one exchange through its shared-memory buffer -> the
//            thread's 64 pairs into its TMEM lane;
//   phase 2  thread wt of either worker meets the same 128 row positions of every row of the
//            plane in its lane (both workers' warps w and w + 4 reach the lane): the CB column
//            bits, the gain G/L and the CB bits back, half the pairs each;
//   phase 3  each worker, for each of its rows: TMEM -> 14 row bits -> Y row.
// Nothing crosses HBM but X, G and Y, and nothing crosses L2 twice; a batch of B planes is B CTAs.
#pragma once

#include "whtmix_fast.cuh"

namespace whtmix {
namespace pln {

// X rows with zero padding past `n` elements (the padding is a whole 16-byte chunk).
template <int D>
__device__ __forceinline__ void ld8_pad(const void* p, long long e, float2 (&o)[4], long long n) {
  if constexpr (D == DT_BF16) {
    if (n > 0) {
      fast::IOv<DT_BF16>::ld8(p, e, o);
    } else {
#pragma unroll
      for (int i = 0; i < 4; ++i) o[i] = make_float2(0.f, 0.f);
    }
  } else {
    fast::IOv<DT_F32>::ld8_lim(p, e, o, n);
  }
}

using fast::THREADS;          // 256: workers 0 (warps 0-3) and 1 (warps 4-7)
constexpr int R = 14;         // row bits
constexpr int WK = 128;       // threads per row worker
constexpr int ROW = 1 << R;   // elements per row
constexpr int STG = 64 * WK;   // staging floats per worker: a bf16 row, or the first half of an fp32 row
// an exchange buffer and a staging area per worker (more than half an SM: one CTA per SM)
constexpr size_t SMEM_BYTES = 2 * (ROW + STG) * sizeof(float);

// TMEM column of pair s's x (y at + 64) for row r of the plane, in this thread's lane.
__device__ __forceinline__ uint32_t row_col(int r) { return 256u * (r & 1) + 128u * (r >> 1); }

// A row's 64 pairs (row elements pbase + 8 s, pbase + 8 s + 1) <-> TMEM: x of pair s at column s,
// y at column 64 + s.
__device__ __forceinline__ void pairs_to_tmem(uint32_t ta, const float2 (&b)[64]) {
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    float lo[16], hi[16];
#pragma unroll
    for (int i = 0; i < 16; ++i) {
      lo[i] = b[16 * q + i].x;
      hi[i] = b[16 * q + i].y;
    }
    fast::tmem_st16(ta + 16 * q, lo);
    fast::tmem_st16(ta + 64 + 16 * q, hi);
  }
}
__device__ __forceinline__ void pairs_from_tmem(uint32_t ta, float2 (&b)[64]) {
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    float lo[16], hi[16];
    fast::tmem_ld16(ta + 16 * q, lo);
    fast::tmem_ld16(ta + 64 + 16 * q, hi);
#pragma unroll
    for (int i = 0; i < 16; ++i) b[16 * q + i] = make_float2(lo[i], hi[i]);
  }
  fast::tmem_wait_ld();
}

// Phase 1 row: X (elements e0 ..., lim of them stored; a whole bf16 row or the first half of an
// fp32 row already staged in stg by cp.async) -> the 14 row bits -> this thread's pairs into TMEM
// at ta (rounds as the three-phase forward's rows).  Once the row is in registers the worker's
// next row (src_next, if not null) is staged behind it.  Each thread reads back only the chunks it
// copied, so the staging area needs no barrier.
template <int D>
__device__ __forceinline__ void row_in(const void* src, long long e0, int lim, float* buf, float* stg, int wt,
                                       int worker, uint32_t ta, const void* src_next, long long e0_next, int lim_next) {
  constexpr int VS = ROW / 16;
  float2 a[16][4];
  if constexpr (D == DT_F32) {
#pragma unroll
    for (int v = 8; v < 16; ++v) {
      const int o = 8 * wt + VS * v;
      ld8_pad<D>(src, e0 + (o < lim ? o : 0), a[v], lim - o);
    }
  }
  fast::cp_async_wait_all();
  if constexpr (D == DT_BF16) {
#pragma unroll
    for (int v = 0; v < 16; ++v) {
      const uint4 u = *reinterpret_cast<const uint4*>(stg + (v * WK + wt) * 4);
      const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
      for (int i = 0; i < 4; ++i) a[v][i] = make_float2(__uint_as_float(w[i] << 16), __uint_as_float(w[i] & 0xFFFF0000u));
    }
  } else {
#pragma unroll
    for (int v = 0; v < 8; ++v) {
      const float4 q0 = *reinterpret_cast<const float4*>(stg + ((2 * v) * WK + wt) * 4);
      const float4 q1 = *reinterpret_cast<const float4*>(stg + ((2 * v + 1) * WK + wt) * 4);
      a[v][0] = make_float2(q0.x, q0.y);
      a[v][1] = make_float2(q0.z, q0.w);
      a[v][2] = make_float2(q1.x, q1.y);
      a[v][3] = make_float2(q1.z, q1.w);
    }
  }
  fast::round_v(a);
  if (src_next != nullptr) fast::stage_row_in<D, R>(src_next, e0_next, stg, wt, lim_next);
#pragma unroll
  for (int v = 0; v < 16; ++v)
#pragma unroll
    for (int r2 = 0; r2 < 2; ++r2) {
      const int r = 8 * wt + VS * v + 4 * r2;
      *reinterpret_cast<float4*>(buf + fast::xswz(r)) =
          make_float4(a[v][2 * r2].x, a[v][2 * r2].y, a[v][2 * r2 + 1].x, a[v][2 * r2 + 1].y);
    }
  fast::worker_sync<R>(worker);
  const int pbase = fast::pbase_of(wt);
  float2 b[64];
#pragma unroll
  for (int s = 0; s < 64; ++s) b[s] = *reinterpret_cast<const float2*>(buf + fast::xswz(pbase + 8 * s));
  fast::worker_sync<R>(worker);  // the buffer is free for the worker's next row
#pragma unroll
  for (int s = 0; s < 64; ++s) fast::bf_in(b[s]);
  fast::bfly_all<64>(b);
  fast::bfly_lane4(b);
  pairs_to_tmem(ta, b);
}

// Phase 3 row: this thread's pairs from TMEM at ta -> the 14 row bits -> Y (elements e0 ..., only
// the first lim stored).
template <int D>
__device__ __forceinline__ void row_out(uint32_t ta, float* buf, void* dst, long long e0, int lim, int wt, int worker) {
  constexpr int VS = ROW / 16;
  const int pbase = fast::pbase_of(wt);
  float2 b[64];
  pairs_from_tmem(ta, b);
  fast::bfly_all<64>(b);
  fast::bfly_lane4(b);
#pragma unroll
  for (int s = 0; s < 64; ++s) *reinterpret_cast<float2*>(buf + fast::xswz(pbase + 8 * s)) = b[s];
  fast::worker_sync<R>(worker);
  float2 a[16][4];
#pragma unroll
  for (int v = 0; v < 16; ++v)
#pragma unroll
    for (int r2 = 0; r2 < 2; ++r2) {
      const float4 q = *reinterpret_cast<const float4*>(buf + fast::xswz(8 * wt + VS * v + 4 * r2));
      a[v][2 * r2] = make_float2(q.x, q.y);
      a[v][2 * r2 + 1] = make_float2(q.z, q.w);
    }
  fast::worker_sync<R>(worker);  // the buffer is free for the worker's next row
#pragma unroll
  for (int v = 0; v < 16; ++v)
#pragma unroll
    for (int i = 0; i < 4; ++i) fast::bf_in(a[v][i]);
  fast::round_v(a);
#pragma unroll
  for (int v = 0; v < 16; ++v) fast::IOv<D>::st8_lim(dst, e0 + 8 * wt + VS * v, a[v], lim - (8 * wt + VS * v));
}

// Phase 2: pairs [32 worker, 32 worker + 32) of this lane's 64 positions, in two chunks of 16,
// across the NR rows of the plane.
template <int CB>
__device__ __forceinline__ void columns(uint32_t lane_ta, const float* __restrict__ g, float scale, int wt, int worker) {
  constexpr int NR = 1 << CB;
  const int pbase = fast::pbase_of(wt);
  const float2 sc = make_float2(scale, scale);
#pragma unroll 1
  for (int k = 2 * worker; k < 2 * worker + 2; ++k) {
    float2 v[NR][16];
#pragma unroll
    for (int r = 0; r < NR; ++r) {
      float lo[16], hi[16];
      fast::tmem_ld16(lane_ta + row_col(r) + 16 * k, lo);
      fast::tmem_ld16(lane_ta + row_col(r) + 64 + 16 * k, hi);
#pragma unroll
      for (int i = 0; i < 16; ++i) v[r][i] = make_float2(lo[i], hi[i]);
    }
    fast::tmem_wait_ld();
#pragma unroll
    for (int h = 1; h < NR; h <<= 1)
#pragma unroll
      for (int r = 0; r < NR; ++r)
        if ((r & h) == 0)
#pragma unroll
          for (int i = 0; i < 16; ++i) fast::bf2(v[r][i], v[r + h][i]);
#pragma unroll
    for (int r = 0; r < NR; ++r)
#pragma unroll
      for (int i = 0; i < 16; ++i) {
        // pair s = 16 k + i: the row's elements pbase + 8 s and + 1 (the pairs are in row order)
        const int s = 16 * k + i;
        const float2 gg = __ldg(reinterpret_cast<const float2*>(g + (r << R) + pbase + 8 * s));
        v[r][i] = fast::mul2(v[r][i], fast::mul2(gg, sc));
      }
#pragma unroll
    for (int h = 1; h < NR; h <<= 1)
#pragma unroll
      for (int r = 0; r < NR; ++r)
        if ((r & h) == 0)
#pragma unroll
          for (int i = 0; i < 16; ++i) fast::bf2(v[r][i], v[r + h][i]);
#pragma unroll
    for (int r = 0; r < NR; ++r) {
      float lo[16], hi[16];
#pragma unroll
      for (int i = 0; i < 16; ++i) {
        lo[i] = v[r][i].x;
        hi[i] = v[r][i].y;
      }
      fast::tmem_st16(lane_ta + row_col(r) + 16 * k, lo);
      fast::tmem_st16(lane_ta + row_col(r) + 64 + 16 * k, hi);
    }
  }
}

// TMEM is allocated by warp 0 for the whole CTA; both phase boundaries order TMEM stores before
// the other warps' loads (wait::st, fence, CTA barrier, fence).
__device__ __forceinline__ void tmem_cta_sync() {
  fast::tmem_wait_st();
  fast::tmem_fence_before();
  __syncthreads();
  fast::tmem_fence_after();
}

template <int D, int CB>
__global__ void __launch_bounds__(THREADS, 1) k_forward_plane(Params P) {
  constexpr int NR = 1 << CB;
  static_assert(CB >= 0 && CB <= 2, "planes of 2^14 to 2^16 elements");
  extern __shared__ __align__(16) float pl_smem[];
  __shared__ uint32_t tmem_slot;
  const long long b = blockIdx.x;
  const int worker = threadIdx.x / WK, wt = threadIdx.x % WK;
  float* buf = pl_smem + worker * ROW;
  float* stg = pl_smem + 2 * ROW + worker * STG;
  if (threadIdx.x < 32) fast::tmem_alloc_512(&tmem_slot);
  fast::tmem_fence_before();
  __syncthreads();
  fast::tmem_fence_after();
  pdl_wait();  // tensor memory first: the previous kernel's CTA on this SM has left
  // this thread's lane: warps w and w + 4 (thread wt of either worker) share lane wt
  const uint32_t lane_ta = tmem_slot + (static_cast<uint32_t>(32 * ((threadIdx.x >> 5) & 3)) << 16);
  if (worker < NR) {
    long long e0;
    int lim;
    fast::row_loc<R, CB>(0, b * NR + worker, P.lv, &e0, &lim);
    fast::stage_row_in<D, R>(P.x, e0, stg, wt, lim);
  }
  for (int r = worker; r < NR; r += 2) {
    long long e0, e0n = 0;
    int lim, limn = 0;
    fast::row_loc<R, CB>(0, b * NR + r, P.lv, &e0, &lim);
    if (r + 2 < NR) fast::row_loc<R, CB>(0, b * NR + r + 2, P.lv, &e0n, &limn);
    row_in<D>(P.x, e0, lim, buf, stg, wt, worker, lane_ta + row_col(r), r + 2 < NR ? P.x : nullptr, e0n, limn);
  }
  tmem_cta_sync();  // every row of the plane is in TMEM
  columns<CB>(lane_ta, static_cast<const float*>(P.g), P.scale, wt, worker);
  tmem_cta_sync();  // every column is back
  for (int r = worker; r < NR; r += 2) {
    long long e0;
    int lim;
    fast::row_loc<R, CB>(0, b * NR + r, P.lv, &e0, &lim);
    row_out<D>(lane_ta + row_col(r), buf, P.y, e0, lim, wt, worker);
  }
  pdl_trigger();
  fast::tmem_fence_before();
  __syncthreads();
  fast::tmem_fence_after();
  if (threadIdx.x < 32) fast::tmem_dealloc_512(tmem_slot);
}

}  // namespace pln
}  // namespace whtmix
