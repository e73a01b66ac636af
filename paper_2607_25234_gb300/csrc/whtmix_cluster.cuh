// whtmix_cluster.cuh -- forward for planes of 2^14 <= N*C <= 2^19 elements, one plane per thread-block
// cluster, with the whole fp32 plane held in the cluster's shared memory (Section III-B, Eq. 2-3:
// Y = H_N (G o (H_N X H_C)) H_C / (N C), flattened to one 2^m-point transform).
//
// A plane is 2^CB rows of 2^14 elements (CB = m - 14 column bits); a CTA of two row workers (128
// threads each) holds two rows, so a plane takes K = max(1, 2^(CB-1)) CTAs, launched as a cluster
// of K (up to 16).  Three phases, as in the three-phase forward, but the workspace is the cluster's
// distributed shared memory instead of L2, and the phase barriers are cluster barriers:
//   phase 1  each worker: its X row -> 14 row bits in registers and one exchange through its row
//            buffer -> the row buffer in storage order;
//   phase 2  each thread: four consecutive storage positions of every row of the plane (16-byte
//            loads from the cluster's row buffers, local or remote) -> CB column bits, gain G/L,
//            CB column bits -> back;
//   phase 3  each worker: its row buffer -> 14 row bits -> Y row.
// Nothing touches HBM but X, G and Y, so the plane's fp32 intermediate never crosses L2.
#pragma once

#include <cooperative_groups.h>

#include "whtmix_fast.cuh"

namespace whtmix {
namespace clu {

namespace cg = cooperative_groups;
using fast::THREADS;            // 256: workers 0 (threads 0-127) and 1 (128-255)
constexpr int R = 14;           // row bits
constexpr int WK = 128;         // threads per row worker
constexpr int ROW = 1 << R;     // elements per row
constexpr size_t SMEM_BYTES = 2 * ROW * sizeof(float);  // one fp32 row buffer per worker

// bf16 X rows with zero padding past `n` elements (the padding is a whole 16-byte chunk).
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

// Phase 1 row: X (elements e0 ..., lim of them stored) -> buf in storage order (sigma), all 14 row
// bits.  Layouts and rounds as the three-phase forward's rows: layout V (thread wt holds 8-vectors
// at 8 wt + 1024 v), round over r1, r2 and the vector bits, one exchange through buf (XOR-swizzled),
// layout P, round over r0, r3..r8 and r9 by one shuffle stage.
template <int D>
__device__ __forceinline__ void row_in(const void* src, long long e0, int lim, float* buf, int wt, int worker) {
  constexpr int VS = ROW / 16;
  float2 a[16][4];
#pragma unroll
  for (int v = 0; v < 16; ++v) {
    const int o = 8 * wt + VS * v;
    ld8_pad<D>(src, e0 + (o < lim ? o : 0), a[v], lim - o);
  }
  fast::round_v(a);
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
  fast::worker_sync<R>(worker);  // every thread has its pairs: the buffer takes the result
#pragma unroll
  for (int s = 0; s < 64; ++s) fast::bf_in(b[s]);
  fast::bfly_all<64>(b);
  fast::bfly_lane4(b);
#pragma unroll
  for (int s = 0; s < 64; ++s) *reinterpret_cast<float2*>(buf + fast::sigma(pbase + 8 * s)) = b[s];
}

// Phase 3 row: buf (storage order) -> Y (elements e0 ..., only the first lim stored), all 14 row
// bits: the mirror of row_in.
template <int D>
__device__ __forceinline__ void row_out(float* buf, void* dst, long long e0, int lim, int wt, int worker) {
  constexpr int VS = ROW / 16;
  const int pbase = fast::pbase_of(wt);
  float2 b[64];
#pragma unroll
  for (int s = 0; s < 64; ++s) b[s] = *reinterpret_cast<const float2*>(buf + fast::sigma(pbase + 8 * s));
  fast::bfly_all<64>(b);
  fast::bfly_lane4(b);
  fast::worker_sync<R>(worker);  // every thread has read its pairs: the buffer takes the exchange
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
#pragma unroll
  for (int v = 0; v < 16; ++v)
#pragma unroll
    for (int i = 0; i < 4; ++i) fast::bf_in(a[v][i]);
  fast::round_v(a);
#pragma unroll
  for (int v = 0; v < 16; ++v) fast::IOv<D>::st8_lim(dst, e0 + 8 * wt + VS * v, a[v], lim - (8 * wt + VS * v));
}

__device__ __forceinline__ void bf4(float4& a, float4& b) {
  float2 a0 = make_float2(a.x, a.y), a1 = make_float2(a.z, a.w);
  float2 b0 = make_float2(b.x, b.y), b1 = make_float2(b.z, b.w);
  fast::bf2(a0, b0);
  fast::bf2(a1, b1);
  a = make_float4(a0.x, a0.y, a1.x, a1.y);
  b = make_float4(b0.x, b0.y, b1.x, b1.y);
}

// Phase 2: storage positions [k SPC, (k + 1) SPC) of every row (SPC = 2^14 / K), four consecutive
// positions per thread and group; a thread's groups (16 / K of them, NR = 2^CB rows each: 32
// 16-byte values in all) are loaded at once, so each thread waits for one round of loads.
template <int CB>
__device__ __forceinline__ void columns(const cg::cluster_group& cl, float* smem, const float* __restrict__ g,
                                        float scale, int k) {
  constexpr int NR = 1 << CB;                    // rows per plane
  constexpr int K = NR > 1 ? NR / 2 : 1;         // CTAs per plane
  constexpr int SPC = ROW / K;                   // positions per CTA
  constexpr int NG = SPC / (4 * THREADS);        // groups of four positions per thread
  static_assert(NG >= 1 && NG * NR <= 32, "32 vectors per thread");
  float* rowbuf[NR];
#pragma unroll
  for (int r = 0; r < NR; ++r) rowbuf[r] = cl.map_shared_rank(smem + (r & 1) * ROW, r >> 1);
  float4 v[NG][NR];
#pragma unroll
  for (int q = 0; q < NG; ++q) {
    const int sp = k * SPC + 4 * (threadIdx.x + q * THREADS);
#pragma unroll
    for (int r = 0; r < NR; ++r) v[q][r] = *reinterpret_cast<const float4*>(rowbuf[r] + sp);
  }
  const float4 sc = make_float4(scale, scale, scale, scale);
#pragma unroll
  for (int q = 0; q < NG; ++q) {
    const int sp = k * SPC + 4 * (threadIdx.x + q * THREADS);
#pragma unroll
    for (int h = 1; h < NR; h <<= 1)
#pragma unroll
      for (int r = 0; r < NR; ++r)
        if ((r & h) == 0) bf4(v[q][r], v[q][r + h]);
    // the four positions are four consecutive plane elements (sigma keeps bits 0..2)
    const float* gq = g + fast::sigma_inv(sp);
#pragma unroll
    for (int r = 0; r < NR; ++r) {
      const float4 gg = __ldg(reinterpret_cast<const float4*>(gq + (static_cast<long long>(r) << R)));
      v[q][r] = make_float4(v[q][r].x * gg.x * sc.x, v[q][r].y * gg.y * sc.y, v[q][r].z * gg.z * sc.z,
                            v[q][r].w * gg.w * sc.w);
    }
#pragma unroll
    for (int h = 1; h < NR; h <<= 1)
#pragma unroll
      for (int r = 0; r < NR; ++r)
        if ((r & h) == 0) bf4(v[q][r], v[q][r + h]);
#pragma unroll
    for (int r = 0; r < NR; ++r) *reinterpret_cast<float4*>(rowbuf[r] + sp) = v[q][r];
  }
}

// One plane per cluster of K CTAs: CTA k of the cluster for plane b holds rows 2k and 2k + 1.
template <int D, int CB>
__global__ void __launch_bounds__(THREADS, 1) k_forward_cluster(Params P) {
  constexpr int NR = 1 << CB;
  constexpr int K = NR > 1 ? NR / 2 : 1;
  extern __shared__ __align__(16) float cl_smem[];
  cg::cluster_group cl = cg::this_cluster();
  const int k = static_cast<int>(cl.block_rank());
  const long long b = blockIdx.x / K;
  const int worker = threadIdx.x / WK, wt = threadIdx.x % WK;
  const int r = 2 * k + worker;  // this worker's row of the plane
  float* buf = cl_smem + worker * ROW;
  long long e0 = 0;
  int lim = 0;
  if (r < NR) fast::row_loc<R, CB>(0, b * NR + r, P.lv, &e0, &lim);
  if (r < NR) row_in<D>(P.x, e0, lim, buf, wt, worker);
  cl.sync();  // every row of the plane is in the cluster's shared memory
  columns<CB>(cl, cl_smem, static_cast<const float*>(P.g), P.scale, k);
  cl.sync();  // every column is back
  if (r < NR) row_out<D>(buf, P.y, e0, lim, wt, worker);
}

}  // namespace clu
}  // namespace whtmix
