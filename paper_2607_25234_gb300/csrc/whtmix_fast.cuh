// whtmix_fast.cuh -- register/TMEM forward kernel for large planes (2^14 <= N*C <= 2^23), fp32 and
// bf16 I/O.
//
// Same three phases as the generic plan M (Section III-B map; see whtmix_kernels.cuh), written
// for the instruction and latency budget of the path: the butterflies need 2 log2(NC) fp32 adds
// per element, which at N*C = 2^23 on 152 SMs is about as long as streaming X, G and Y through
// HBM.  A plane of 2^m elements is viewed as 2^Q rows of 2^R contiguous elements (R = 13 for the
// forward launches, Q <= 10; the row code also serves R = 14, used by the backward and the fused
// block):
//   phase 1  every row: its R bits forward                              X  -> workspace
//   phase 2  every column: its Q bits forward, gain G/L, Q bits again   workspace -> workspace
//   phase 3  every row: its R bits again                                workspace -> Y
// with a bounded device-wide barrier between phases.  Design points:
//   * butterflies run on register pairs with packed add/sub.f32x2 (half the instructions);
//   * one CTA of 8 warps per SM; a row is one worker's (2^(R-7) threads, 128 elements each):
//     one round in registers, one conflict-free XOR-swizzled shared-memory exchange, a second
//     round (plus one warp-shuffle stage for R = 14); each worker's next row is prefetched with
//     cp.async; rows are spread as balanced contiguous ranges per SM;
//   * the workspace stores rows bit-permuted (sigma) so that every row access of phases 1 and 3
//     is one contiguous 256-byte span per warp instruction;
//   * phase 2 gives columns to threads: whole columns in registers when a column has <= 128
//     elements; otherwise the two warps (w, w+4) that share a TMEM lane quarter hold one column
//     per lane (Blackwell tensor memory as per-thread storage, up to 256 fp32 per thread) and
//     trade the bit between their halves through TMEM; 1024-row columns take two lanes of a warp;
//   * column ranges are balanced and aligned to 8 columns (32-byte sectors).
#pragma once

#include <type_traits>

#include "whtmix_kernels.cuh"

namespace whtmix {
namespace fast {

constexpr int THREADS = 256;  // 8 warps; warps w and w+4 share a TMEM lane quarter
// shared memory: row exchange buffers (128 KiB) and row staging areas for the cp.async prefetch
// (64 KiB).  More than half an SM, so exactly one CTA runs per SM.
constexpr size_t SMEM_XBUF_BYTES = 128 * 1024;
constexpr size_t SMEM_STAGE_BYTES = 64 * 1024;
constexpr size_t SMEM_BYTES = SMEM_XBUF_BYTES + SMEM_STAGE_BYTES;
static_assert(SMEM_BYTES <= 227 * 1024, "shared memory per CTA");

// Row geometry for R row bits: 128 elements per thread.
template <int R>
struct Row {
  static constexpr int LEN = 1 << R;
  static constexpr int WORKER = 1 << (R - 7);          // threads per row
  static constexpr int NWORKERS = THREADS / WORKER;
  static constexpr int VSTRIDE = 1 << (R - 4);         // element stride between a thread's 16 vectors
  static constexpr int STAGE = SMEM_STAGE_BYTES / sizeof(float) / NWORKERS;  // staging floats per worker
  static_assert(NWORKERS * LEN * sizeof(float) == SMEM_XBUF_BYTES, "one exchange buffer per worker");
  static_assert(STAGE >= 64 * WORKER, "staging holds 16 bf16 vectors or 32 fp32 pairs per thread");
};

// ---------------------------------------------------------------------------------------------
// packed fp32 pairs
__device__ __forceinline__ float2 add2(float2 a, float2 b) {
  float2 r;
  asm("{.reg .b64 pa, pb, pd;\n\t"
      "mov.b64 pa, {%2, %3};\n\tmov.b64 pb, {%4, %5};\n\t"
      "add.rn.f32x2 pd, pa, pb;\n\tmov.b64 {%0, %1}, pd;}"
      : "=f"(r.x), "=f"(r.y) : "f"(a.x), "f"(a.y), "f"(b.x), "f"(b.y));
  return r;
}
__device__ __forceinline__ float2 sub2(float2 a, float2 b) {
  float2 r;
  asm("{.reg .b64 pa, pb, pd;\n\t"
      "mov.b64 pa, {%2, %3};\n\tmov.b64 pb, {%4, %5};\n\t"
      "sub.rn.f32x2 pd, pa, pb;\n\tmov.b64 {%0, %1}, pd;}"
      : "=f"(r.x), "=f"(r.y) : "f"(a.x), "f"(a.y), "f"(b.x), "f"(b.y));
  return r;
}
__device__ __forceinline__ float2 mul2(float2 a, float2 b) {
  float2 r;
  asm("{.reg .b64 pa, pb, pd;\n\t"
      "mov.b64 pa, {%2, %3};\n\tmov.b64 pb, {%4, %5};\n\t"
      "mul.rn.f32x2 pd, pa, pb;\n\tmov.b64 {%0, %1}, pd;}"
      : "=f"(r.x), "=f"(r.y) : "f"(a.x), "f"(a.y), "f"(b.x), "f"(b.y));
  return r;
}
// a * s + b with s = +-1 (exact)
__device__ __forceinline__ float2 fma2(float2 a, float2 s, float2 b) {
  float2 r;
  asm("{.reg .b64 pa, ps, pb, pd;\n\t"
      "mov.b64 pa, {%2, %3};\n\tmov.b64 ps, {%4, %5};\n\tmov.b64 pb, {%6, %7};\n\t"
      "fma.rn.f32x2 pd, pa, ps, pb;\n\tmov.b64 {%0, %1}, pd;}"
      : "=f"(r.x), "=f"(r.y) : "f"(a.x), "f"(a.y), "f"(s.x), "f"(s.y), "f"(b.x), "f"(b.y));
  return r;
}

// butterfly on two pairs: (a, b) -> (a + b, a - b), elementwise
__device__ __forceinline__ void bf2(float2& a, float2& b) {
  const float2 s = add2(a, b), d = sub2(a, b);
  a = s;
  b = d;
}
// butterfly inside one pair: (x, y) -> (x + y, x - y)
__device__ __forceinline__ void bf_in(float2& a) {
  const float s = a.x + a.y, d = a.x - a.y;
  a.x = s;
  a.y = d;
}

// Butterflies over the bits of an index into v[]: for every h = 1, 2, ..., N/2 pair (i, i + h).
template <int N>
__device__ __forceinline__ void bfly_all(float2 (&v)[N]) {
#pragma unroll
  for (int h = 1; h < N; h <<= 1)
#pragma unroll
    for (int i = 0; i < N; ++i)
      if ((i & h) == 0) bf2(v[i], v[i + h]);
}

// ---------------------------------------------------------------------------------------------
// TMEM (tensor memory) as per-thread storage: thread t of warp w owns lane 32*(w%4) + t.
__device__ __forceinline__ void tmem_alloc_512(uint32_t* smem_slot) {
  const uint32_t dst = static_cast<uint32_t>(__cvta_generic_to_shared(smem_slot));
  asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], 512;" ::"r"(dst) : "memory");
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void tmem_dealloc_512(uint32_t taddr) {
  asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, 512;" ::"r"(taddr) : "memory");
}
__device__ __forceinline__ void tmem_fence_before() { asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void tmem_fence_after() { asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void tmem_wait_ld() { asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory"); }
__device__ __forceinline__ void tmem_wait_st() { asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory"); }

// 16 consecutive 32-bit columns of this thread's lane <-> registers
__device__ __forceinline__ void tmem_ld16(uint32_t ta, float (&r)[16]) {
  asm volatile("tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15}, [%16];"
               : "=f"(r[0]), "=f"(r[1]), "=f"(r[2]), "=f"(r[3]), "=f"(r[4]), "=f"(r[5]), "=f"(r[6]), "=f"(r[7]),
                 "=f"(r[8]), "=f"(r[9]), "=f"(r[10]), "=f"(r[11]), "=f"(r[12]), "=f"(r[13]), "=f"(r[14]), "=f"(r[15])
               : "r"(ta) : "memory");
}
__device__ __forceinline__ void tmem_st16(uint32_t ta, const float (&r)[16]) {
  asm volatile("tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16};"
               ::"r"(ta), "f"(r[0]), "f"(r[1]), "f"(r[2]), "f"(r[3]), "f"(r[4]), "f"(r[5]), "f"(r[6]), "f"(r[7]),
                 "f"(r[8]), "f"(r[9]), "f"(r[10]), "f"(r[11]), "f"(r[12]), "f"(r[13]), "f"(r[14]), "f"(r[15])
               : "memory");
}

// ---------------------------------------------------------------------------------------------
// Row exchange buffer: word address of row element r, XOR-swizzled so that both access patterns
// below are bank-conflict free:
//   layout V (16-byte vectors of r0..r1, lanes on r3..r7): bits 2..4 = (r2^r5, r3^r9, r4^r10)
//   layout P (8-byte pairs of r0, lanes on r1, r2, r9, r10, r11): bits 1..4 = (r1, r2^r5, r3^r9, r4^r10)
__device__ __forceinline__ int xswz(int r) {
  return r ^ (((r >> 5) & 1) << 2) ^ (((r >> 9) & 1) << 3) ^ (((r >> 10) & 1) << 4);
}

// Workspace rows are stored with their index bits permuted (sigma), so that layout P's lanes
// (r1, r2, r9, r10, r11, plus the in-register pair bit r0) cover 64 consecutive floats: phase 1's
// stores and phase 3's loads are one 256-byte span per warp instruction.  Storage position s of
// row element r: s = (r0, r1, r2, r9, r10, r11, r3, r4, r5, r6, r7, r8, r12, r13) from bit 0 up.
// Phase 2 works in storage positions and maps back to the logical column only to index G.
__device__ __forceinline__ int sigma(int r) {
  return (r & 7) | (((r >> 9) & 7) << 3) | (((r >> 3) & 63) << 6) | (r & ~4095);
}
__device__ __forceinline__ int sigma_inv(int s) {
  return (s & 7) | (((s >> 6) & 63) << 3) | (((s >> 3) & 7) << 9) | (s & ~4095);
}

template <int R>
__device__ __forceinline__ void worker_sync(int worker) {
  asm volatile("bar.sync %0, %1;" ::"r"(worker + 1), "r"(Row<R>::WORKER) : "memory");
}

// Butterfly on a row bit held by lane bit 2 (r9 in layout P when R = 14): lane pairs (l, l ^ 4).
__device__ __forceinline__ void bfly_lane4(float2 (&b)[64]) {
  const float2 sgn = (threadIdx.x & 4) ? make_float2(-1.f, -1.f) : make_float2(1.f, 1.f);
#pragma unroll
  for (int s = 0; s < 64; ++s) {
    const float2 p = make_float2(__shfl_xor_sync(0xffffffffu, b[s].x, 4), __shfl_xor_sync(0xffffffffu, b[s].y, 4));
    b[s] = fma2(b[s], sgn, p);
  }
}

// Storage <-> fp32 for the two floating dtypes.
template <int D> struct IOv;
// (ld8_lim / st8_lim: only the first `n` of the 8 elements exist in memory, n a multiple of the
// 16-byte chunk's element count; the others read as zero and are not written.)
template <> struct IOv<DT_BF16> {
  // 8 consecutive elements at element index e (16-byte aligned): 4 pairs (r0 = 0, 1)
  __device__ static __forceinline__ void ld8(const void* p, long long e, float2 (&o)[4]) {
    const uint4 u = __ldcs(reinterpret_cast<const uint4*>(static_cast<const unsigned short*>(p) + e));
    const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
    for (int i = 0; i < 4; ++i) o[i] = make_float2(__uint_as_float(w[i] << 16), __uint_as_float(w[i] & 0xFFFF0000u));
  }
  __device__ static __forceinline__ void st8(void* p, long long e, const float2 (&v)[4]) {
    uint32_t w[4];
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      __nv_bfloat162 h = __floats2bfloat162_rn(v[i].x, v[i].y);
      w[i] = *reinterpret_cast<uint32_t*>(&h);
    }
    __stcs(reinterpret_cast<uint4*>(static_cast<unsigned short*>(p) + e), make_uint4(w[0], w[1], w[2], w[3]));
  }
  __device__ static __forceinline__ void st8_lim(void* p, long long e, const float2 (&v)[4], long long n) {
    if (n > 0) st8(p, e, v);
  }
};
template <> struct IOv<DT_F32> {
  __device__ static __forceinline__ void ld8(const void* p, long long e, float2 (&o)[4]) {
    const float4* q = reinterpret_cast<const float4*>(static_cast<const float*>(p) + e);
    const float4 a = __ldcs(q), b = __ldcs(q + 1);
    o[0] = make_float2(a.x, a.y);
    o[1] = make_float2(a.z, a.w);
    o[2] = make_float2(b.x, b.y);
    o[3] = make_float2(b.z, b.w);
  }
  __device__ static __forceinline__ void st8(void* p, long long e, const float2 (&v)[4]) {
    float4* q = reinterpret_cast<float4*>(static_cast<float*>(p) + e);
    __stcs(q, make_float4(v[0].x, v[0].y, v[1].x, v[1].y));
    __stcs(q + 1, make_float4(v[2].x, v[2].y, v[3].x, v[3].y));
  }
  __device__ static __forceinline__ void ld8_lim(const void* p, long long e, float2 (&o)[4], long long n) {
    const float4* q = reinterpret_cast<const float4*>(static_cast<const float*>(p) + e);
    const float4 z = make_float4(0.f, 0.f, 0.f, 0.f);
    const float4 a = n > 0 ? __ldcs(q) : z, b = n > 4 ? __ldcs(q + 1) : z;
    o[0] = make_float2(a.x, a.y);
    o[1] = make_float2(a.z, a.w);
    o[2] = make_float2(b.x, b.y);
    o[3] = make_float2(b.z, b.w);
  }
  __device__ static __forceinline__ void st8_lim(void* p, long long e, const float2 (&v)[4], long long n) {
    float4* q = reinterpret_cast<float4*>(static_cast<float*>(p) + e);
    if (n > 0) __stcs(q, make_float4(v[0].x, v[0].y, v[1].x, v[1].y));
    if (n > 4) __stcs(q + 1, make_float4(v[2].x, v[2].y, v[3].x, v[3].y));
  }
};

// ---------------------------------------------------------------------------------------------
// Workspace element: fp32 (the exact exchange), or bf16 for whtmix_forward_x16, where every value
// that crosses between SMs is rounded to the nearest bf16 (ties to even) where it is written and
// widened exactly where it is read; every butterfly and the gain stay fp32.  ld2/st2: elements
// p[0], p[1] (p even).  The phase-3 staging holds a pair per slot (an fp32 pair, or one 32-bit
// word of two bf16).
struct WsF32 {
  using T = float;
  __device__ static __forceinline__ float ld(const float* p) { return __ldcg(p); }
  __device__ static __forceinline__ void st(float* p, float v) { __stcg(p, v); }
  __device__ static __forceinline__ float2 ld2(const float* p) { return __ldcg(reinterpret_cast<const float2*>(p)); }
  __device__ static __forceinline__ void st2(float* p, float2 v) { __stcg(reinterpret_cast<float2*>(p), v); }
  __device__ static __forceinline__ float2 staged(const float* stg, int slot) {
    return *reinterpret_cast<const float2*>(stg + 2 * slot);
  }
};
struct WsB16 {
  using T = unsigned short;
  __device__ static __forceinline__ float2 widen2(uint32_t w) {
    return make_float2(__uint_as_float(w << 16), __uint_as_float(w & 0xFFFF0000u));
  }
  __device__ static __forceinline__ float ld(const unsigned short* p) {
    return __uint_as_float(static_cast<uint32_t>(__ldcg(p)) << 16);
  }
  __device__ static __forceinline__ void st(unsigned short* p, float v) {
    __stcg(p, __bfloat16_as_ushort(__float2bfloat16_rn(v)));
  }
  __device__ static __forceinline__ float2 ld2(const unsigned short* p) {
    return widen2(__ldcg(reinterpret_cast<const unsigned int*>(p)));
  }
  __device__ static __forceinline__ void st2(unsigned short* p, float2 v) {
    const __nv_bfloat162 h = __floats2bfloat162_rn(v.x, v.y);
    __stcg(reinterpret_cast<unsigned int*>(p), *reinterpret_cast<const unsigned int*>(&h));
  }
  __device__ static __forceinline__ float2 staged(const float* stg, int slot) {
    return widen2(reinterpret_cast<const uint32_t*>(stg)[slot]);
  }
};

// ---------------------------------------------------------------------------------------------
// Asynchronous global -> shared copies (no registers held while in flight).
__device__ __forceinline__ void cp_async16(float* smem_dst, const void* gsrc) {
  const uint32_t s = static_cast<uint32_t>(__cvta_generic_to_shared(smem_dst));
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(s), "l"(gsrc) : "memory");
}
// 16-byte copy of which only the first src_bytes (0 or 16) are read; the rest is zero-filled.
__device__ __forceinline__ void cp_async16_zfill(float* smem_dst, const void* gsrc, int src_bytes) {
  const uint32_t s = static_cast<uint32_t>(__cvta_generic_to_shared(smem_dst));
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(s), "l"(gsrc), "r"(src_bytes) : "memory");
}
__device__ __forceinline__ void cp_async8(float* smem_dst, const void* gsrc) {
  const uint32_t s = static_cast<uint32_t>(__cvta_generic_to_shared(smem_dst));
  asm volatile("cp.async.ca.shared.global [%0], [%1], 8;" ::"r"(s), "l"(gsrc) : "memory");
}
__device__ __forceinline__ void cp_async4(float* smem_dst, const float* gsrc) {
  const uint32_t s = static_cast<uint32_t>(__cvta_generic_to_shared(smem_dst));
  asm volatile("cp.async.ca.shared.global [%0], [%1], 4;" ::"r"(s), "l"(gsrc) : "memory");
}
// Bulk prefetch into L2 of piece i of n of this CTA's 1/gridDim.x share of a buffer (16-byte
// chunks).
__device__ __forceinline__ void l2_prefetch_piece(const void* base, long long bytes, long long i, long long n) {
  const long long chunks = bytes >> 4;
  const long long s0 = chunks * blockIdx.x / gridDim.x, s1 = chunks * (blockIdx.x + 1) / gridDim.x;
  const long long c0 = s0 + (s1 - s0) * i / n, c1 = s0 + (s1 - s0) * (i + 1) / n;
  if (c1 > c0)
    asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(static_cast<const char*>(base) + (c0 << 4)),
                 "r"(static_cast<unsigned>((c1 - c0) << 4))
                 : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
__device__ __forceinline__ void cp_async_wait_all() { asm volatile("cp.async.wait_group 0;" ::: "memory"); }

// Row prefetch.  Every thread copies exactly the 16-byte (8-byte) chunks it will read back
// itself, so the staging area needs no barrier; chunk k of thread wt sits at (k * WORKER + wt),
// which makes each warp's read-back one contiguous span.
// Phase 1 stages a whole bf16 row (16 vectors of 8 elements) or the first half of an fp32 row.
// Elements of the row at offsets >= lim are padding: not read, staged as zeros.
template <int D, int R>
__device__ __forceinline__ void stage_row_in(const void* src, long long e0, float* stg, int wt, int lim) {
  constexpr int WK = Row<R>::WORKER, VS = Row<R>::VSTRIDE;
  if constexpr (D == DT_BF16) {
#pragma unroll
    for (int v = 0; v < 16; ++v) {
      const int o = 8 * wt + VS * v;
      cp_async16_zfill(stg + (v * WK + wt) * 4, static_cast<const unsigned short*>(src) + e0 + (o < lim ? o : 0),
                       o < lim ? 16 : 0);
    }
  } else {
#pragma unroll
    for (int v = 0; v < 8; ++v)
#pragma unroll
      for (int h2 = 0; h2 < 2; ++h2) {
        const int o = 8 * wt + VS * v + 4 * h2;
        cp_async16_zfill(stg + ((2 * v + h2) * WK + wt) * 4, static_cast<const float*>(src) + e0 + (o < lim ? o : 0),
                         o < lim ? 16 : 0);
      }
  }
  cp_async_commit();
}
// Phase 3 stages the first 32 of the 64 pairs each thread reads in layout P.
__device__ __forceinline__ int pbase_of(int wt) { return 2 * (wt & 1) + 4 * ((wt >> 1) & 1) + 512 * (wt >> 2); }
template <int R, class WS = WsF32>
__device__ __forceinline__ void stage_row_out(const typename WS::T* src_ws, float* stg, int wt) {
  const int pbase = pbase_of(wt);
#pragma unroll
  for (int s = 0; s < 32; ++s) {
    if constexpr (sizeof(typename WS::T) == 4) cp_async8(stg + (s * Row<R>::WORKER + wt) * 2, src_ws + sigma(pbase + 8 * s));
    else cp_async4(stg + s * Row<R>::WORKER + wt, reinterpret_cast<const float*>(src_ws + sigma(pbase + 8 * s)));
  }
  cp_async_commit();
}

// round over the layout-V register bits: r1, r2 (inside a vector) and the 4 vector bits
__device__ __forceinline__ void round_v(float2 (&a)[16][4]) {
#pragma unroll
  for (int v = 0; v < 16; ++v) {
    bf2(a[v][0], a[v][1]);
    bf2(a[v][2], a[v][3]);
    bf2(a[v][0], a[v][2]);
    bf2(a[v][1], a[v][3]);
  }
#pragma unroll
  for (int h = 1; h < 16; h <<= 1)
#pragma unroll
    for (int v = 0; v < 16; ++v)
      if ((v & h) == 0)
#pragma unroll
        for (int i = 0; i < 4; ++i) bf2(a[v][i], a[v + h][i]);
}

// ---------------------------------------------------------------------------------------------
// Phase 1 row: X (dtype D) -> workspace (fp32), butterflies on all R row bits.
//   layout V: thread wt holds r0..r2 (8-vectors) x 16 vectors (bits R-4..R-1); wt = r3..r(R-5).
//     round A: bits r1, r2 and the vector bits (pairs on r0).
//   exchange through smem, then layout P: thread holds pairs (r0) x r3..r8; wt bits = (r1, r2,
//     r9, ...) with lanes on (r1, r2, r9, r10, r11).  round B: r0 (inside the pairs), r3..r8,
//     and for R = 14 r9 by one shuffle stage.
// The row arrives through the staging area (prefetched while the previous row was processed);
// the next row's prefetch (element e0_next of src_next, lim_next of its elements stored, if
// src_next is not null) is issued as soon as this row is in registers.  Elements of a row at
// offsets >= lim are zero padding (never read).
template <int D, int R, class WS = WsF32>
__device__ __forceinline__ void row_forward_in(const void* src, long long e0, int lim, typename WS::T* dst_ws, float* xbuf,
                                               float* stg, int wt, int worker, const void* src_next, long long e0_next,
                                               int lim_next) {
  constexpr int WK = Row<R>::WORKER, VS = Row<R>::VSTRIDE;
  float2 a[16][4];  // [vector][r1 + 2 r2]
  if constexpr (D == DT_F32) {
#pragma unroll
    for (int v = 8; v < 16; ++v) {
      const int o = 8 * wt + VS * v;
      IOv<D>::ld8_lim(src, e0 + (o < lim ? o : 0), a[v], lim - o);
    }
  }
  cp_async_wait_all();
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
  round_v(a);
  if (src_next != nullptr) stage_row_in<D, R>(src_next, e0_next, stg, wt, lim_next);
  // exchange V -> P
#pragma unroll
  for (int v = 0; v < 16; ++v)
#pragma unroll
    for (int r2 = 0; r2 < 2; ++r2) {
      const int r = 8 * wt + VS * v + 4 * r2;
      *reinterpret_cast<float4*>(xbuf + xswz(r)) = make_float4(a[v][2 * r2].x, a[v][2 * r2].y, a[v][2 * r2 + 1].x, a[v][2 * r2 + 1].y);
    }
  worker_sync<R>(worker);
  const int pbase = pbase_of(wt);
  float2 b[64];  // [s = r3..r8]
#pragma unroll
  for (int s = 0; s < 64; ++s) b[s] = *reinterpret_cast<const float2*>(xbuf + xswz(pbase + 8 * s));
  worker_sync<R>(worker);  // buffer free for the next row
  // round B
#pragma unroll
  for (int s = 0; s < 64; ++s) bf_in(b[s]);
  bfly_all<64>(b);
  if constexpr (R == 14) bfly_lane4(b);
#pragma unroll
  for (int s = 0; s < 64; ++s) WS::st2(dst_ws + sigma(pbase + 8 * s), b[s]);
}

// Phase 3 row: workspace (fp32) -> Y (dtype D), butterflies on all R row bits (mirror of phase 1).
// The first half of the row's pairs arrives through the staging area; src_next (if not null) is
// the next row, whose prefetch is issued once this row is in registers.
// Only the row's first lim elements are stored (the rest is the cropped padding).
template <int D, int R, class WS = WsF32>
__device__ __forceinline__ void row_forward_out(const typename WS::T* src_ws, void* dst, long long e0, int lim, float* xbuf,
                                                float* stg, int wt, int worker, const typename WS::T* src_next) {
  constexpr int WK = Row<R>::WORKER, VS = Row<R>::VSTRIDE;
  const int pbase = pbase_of(wt);
  float2 b[64];
#pragma unroll
  for (int s = 32; s < 64; ++s) b[s] = WS::ld2(src_ws + sigma(pbase + 8 * s));
  cp_async_wait_all();
#pragma unroll
  for (int s = 0; s < 32; ++s) b[s] = WS::staged(stg, s * WK + wt);
  bfly_all<64>(b);  // round A: r3..r8 (and r9 for R = 14)
  if constexpr (R == 14) bfly_lane4(b);
  if (src_next != nullptr) stage_row_out<R, WS>(src_next, stg, wt);
#pragma unroll
  for (int s = 0; s < 64; ++s) *reinterpret_cast<float2*>(xbuf + xswz(pbase + 8 * s)) = b[s];
  worker_sync<R>(worker);
  float2 a[16][4];
#pragma unroll
  for (int v = 0; v < 16; ++v)
#pragma unroll
    for (int r2 = 0; r2 < 2; ++r2) {
      const float4 q = *reinterpret_cast<const float4*>(xbuf + xswz(8 * wt + VS * v + 4 * r2));
      a[v][2 * r2] = make_float2(q.x, q.y);
      a[v][2 * r2 + 1] = make_float2(q.z, q.w);
    }
  worker_sync<R>(worker);
  // round B: r0, r1, r2 and the vector bits
#pragma unroll
  for (int v = 0; v < 16; ++v)
#pragma unroll
    for (int i = 0; i < 4; ++i) bf_in(a[v][i]);
  round_v(a);
#pragma unroll
  for (int v = 0; v < 16; ++v) IOv<D>::st8_lim(dst, e0 + 8 * wt + VS * v, a[v], lim - (8 * wt + VS * v));
}

// Where row r of the plane group that starts at plane b0 lives in X / Y (planes of lv stored
// elements, back to back): its first element and how many of its 2^R elements are stored.
// Rows wholly in the padding get lim = 0 and the plane's first element (never accessed).
template <int R, int Q>
__device__ __forceinline__ void row_loc(long long b0, long long r, long long lv, long long* e0, int* lim) {
  const long long b = r >> Q, start = (r & ((1ll << Q) - 1)) << R;
  long long n = lv - start;
  n = n < 0 ? 0 : n > (1ll << R) ? (1ll << R) : n;
  *e0 = (b0 + b) * lv + (n > 0 ? start : 0);
  *lim = static_cast<int>(n);
}

// Issued before pdl_wait(): asks L2 for the X rows [rb, re) of the first plane group that this
// CTA's phase 1 reads, at most PREFETCH_BYTES of them, so that their HBM reads overlap the
// previous kernel's tail.  A cache hint only: L2 is the point of coherence, so a line fetched
// before the previous kernel's last writes to it still returns those writes.
constexpr long long PREFETCH_BYTES = 128 * 1024;
template <int D, int R, int Q>
__device__ __forceinline__ void l2_prefetch_first_rows(const void* src, long long rb, long long re, long long lv) {
  constexpr long long ES = D == DT_BF16 ? 2 : 4;
  const long long r = rb + threadIdx.x;
  if (r >= re || (r - rb) * (ES << R) >= PREFETCH_BYTES) return;
  long long e0;
  int lim;
  row_loc<R, Q>(0, r, lv, &e0, &lim);
  if (lim > 0)
    asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(static_cast<const char*>(src) + e0 * ES),
                 "r"(static_cast<unsigned>(lim * ES))
                 : "memory");
}

// ---------------------------------------------------------------------------------------------
// Gains as phase 2 reads them, per column: storage position sp of a workspace row, whose element
// j is logical plane element (j << R) + sigma_inv(sp).  at() is one element of the column, at2()
// the elements of the storage positions sp and sp + 1 (sp even), which sigma_inv keeps adjacent.
// NAT: the workspace rows are in natural order (storage position sp is plane element (j << R) + sp).
template <int R, bool NAT = false>
struct FullGain {  // G [N, C] as given
  static constexpr bool SEPARABLE = false;
  const float* g;
  struct Col {
    const float* p;
  };
  __device__ __forceinline__ Col col(int sp) const { return {g + (NAT ? sp : sigma_inv(sp))}; }
  __device__ __forceinline__ float at(const Col& c, long long j) const { return __ldg(c.p + (j << R)); }
  __device__ __forceinline__ float2 at2(const Col& c, long long j) const {
    return __ldg(reinterpret_cast<const float2*>(c.p + (j << R)));
  }
};
// Separable log gains (Section III-B, Eq. 2-3): G[n, c] = exp(g_t[n]) exp(g_c[c]), from two tables
// phase 1 builds in the workspace.  With C = 2^cb, 1 <= cb <= R, a column holds one channel
// c = s mod C (s = sigma_inv(sp)) and the tokens n = (j << (R - cb)) + (s >> cb), so the token
// table is stored column-major, etT[(n mod 2^(R-cb)) * 2^Q + (n >> (R-cb))] = exp(g_t[n]): a column's
// gains are then consecutive floats (compile-time offsets from one pointer), and ec[c] = exp(g_c[c]).
// at2's second position is channel c + 1 of the same token.  The tables are written during the
// launch, before the barrier that opens phase 2, so they are read with ordinary (coherent) loads.
template <int R, int Q>
struct SepGain {
  static constexpr bool SEPARABLE = true;
  const float* etT;
  const float* ec;
  int cb;
  struct Col {
    const float* p;
    float e0, e1;
  };
  __device__ __forceinline__ Col col(int sp) const {
    const int s = sigma_inv(sp), c = s & ((1 << cb) - 1);
    return {etT + (static_cast<long long>(s >> cb) << Q), ec[c], ec[c | 1]};
  }
  __device__ __forceinline__ float at(const Col& c, long long j) const { return c.p[j] * c.e0; }
  __device__ __forceinline__ float2 at2(const Col& c, long long j) const {
    const float t = c.p[j];
    return make_float2(t * c.e0, t * c.e1);
  }
  // rows j and j + 1 (j even: one 8-byte load)
  __device__ __forceinline__ float2 rows2(const Col& c, long long j) const {
    return mul2(*reinterpret_cast<const float2*>(c.p + j), make_float2(c.e0, c.e0));
  }
};
// Entry i of the column-major token table built by phase 1: exp(g_t[n]) for the token n it holds.
template <int R, int Q>
__device__ __forceinline__ long long sep_token_of(long long i, int cb) {
  return ((i & ((1ll << Q) - 1)) << (R - cb)) | (i >> Q);
}

// ---------------------------------------------------------------------------------------------
// Phase 2, register variant (Q <= 6): a thread owns two adjacent storage positions (one logical
// column pair) x 2^Q rows.
template <int Q, int R, class GainT, class WS = WsF32>
__device__ __forceinline__ void col_pass_pairs(typename WS::T* ws, const GainT& gain, float scale, int m, long long u_begin,
                                               long long u_end) {
  constexpr int NR = 1 << Q;
  const float2 sc = make_float2(scale, scale);
  for (long long u0 = u_begin; u0 < u_end; u0 += 2 * THREADS) {
    const long long u = u0 + 2 * threadIdx.x;  // even: the pair never straddles a plane
    if (u >= u_end) break;
    const long long b = u >> R;
    const int sp = static_cast<int>(u & ((1 << R) - 1));  // storage position (even); sp + 1 is column c + 1
    typename WS::T* base = ws + (b << m) + sp;
    const auto gc = gain.col(sp);
    float2 v[NR];
#pragma unroll
    for (int j = 0; j < NR; ++j) v[j] = WS::ld2(base + (static_cast<long long>(j) << R));
    bfly_all<NR>(v);
#pragma unroll
    for (int j = 0; j < NR; ++j) v[j] = mul2(v[j], mul2(gain.at2(gc, j), sc));
    bfly_all<NR>(v);
#pragma unroll
    for (int j = 0; j < NR; ++j) WS::st2(base + (static_cast<long long>(j) << R), v[j]);
  }
}

// Phase 2, register variant for Q = 7: a thread owns one column of 128 rows as 64 pairs (j, j + 64).
template <int R, class GainT, class WS = WsF32>
__device__ __forceinline__ void col_pass_single128(typename WS::T* ws, const GainT& gain, float scale, int m, long long u_begin,
                                                   long long u_end) {
  for (long long u0 = u_begin; u0 < u_end; u0 += THREADS) {
    const long long u = u0 + threadIdx.x;
    if (u >= u_end) break;
    const long long b = u >> R;
    const int sp = static_cast<int>(u & ((1 << R) - 1));
    typename WS::T* base = ws + (b << m) + sp;
    const auto gc = gain.col(sp);
    float2 v[64];
#pragma unroll
    for (int j = 0; j < 64; ++j)
      v[j] = make_float2(WS::ld(base + (static_cast<long long>(j) << R)), WS::ld(base + (static_cast<long long>(j + 64) << R)));
    bfly_all<64>(v);
#pragma unroll
    for (int j = 0; j < 64; ++j) bf_in(v[j]);
#pragma unroll
    for (int j = 0; j < 64; ++j) {
      float2 gg;
      if constexpr (GainT::SEPARABLE) gg = make_float2(gain.at(gc, j), gain.at(gc, j + 64));
      else gg = make_float2(__ldg(gc.p + (static_cast<long long>(j) << R)), __ldg(gc.p + (static_cast<long long>(j + 64) << R)));
      v[j] = mul2(v[j], mul2(gg, make_float2(scale, scale)));
    }
#pragma unroll
    for (int j = 0; j < 64; ++j) bf_in(v[j]);
    bfly_all<64>(v);
#pragma unroll
    for (int j = 0; j < 64; ++j) {
      WS::st(base + (static_cast<long long>(j) << R), v[j].x);
      WS::st(base + (static_cast<long long>(j + 64) << R), v[j].y);
    }
  }
}

// The two warps (w, w + 4) that share a TMEM lane quarter meet here; TMEM stores made before the
// barrier are visible to the other warp's loads after it.
__device__ __forceinline__ void pair_sync(int quarter) {
  tmem_wait_st();
  tmem_fence_before();
  asm volatile("bar.sync %0, %1;" ::"r"(5 + quarter), "r"(64) : "memory");
  tmem_fence_after();
}

// Column bit 9 for Q = 10, held by lane bit 4: lanes l and l ^ 16 hold the two halves of one
// column at the same register positions (combinations s = 0..7 of bits 6..8).  A swap trades half
// of them so that each lane holds both halves for four combinations: afterwards lane bit 4 = h
// holds combinations 4h + t, t = 0..3, with bit 9 = 0 in v[t] and bit 9 = 1 in v[t + 4].  The
// same swap restores the layout.  (Half the shuffles of a butterfly across the lanes.)
template <int W>
__device__ __forceinline__ void lane16_swap(float2 (&v)[8][W], int h) {
#pragma unroll
  for (int t = 0; t < 4; ++t)
#pragma unroll
    for (int w = 0; w < W; ++w) {
      const float2 a = v[t][w], b = v[t + 4][w];
      const float2 snd = h ? a : b;
      const float2 r = make_float2(__shfl_xor_sync(0xffffffffu, snd.x, 16), __shfl_xor_sync(0xffffffffu, snd.y, 16));
      v[t][w] = h ? r : a;
      v[t + 4][w] = h ? b : r;
    }
}

// Phase 2, TMEM variant (Q = 8, 9, 10).  Per TMEM lane: 2^Q rows of one column (Q = 8, 9), or
// half of a 1024-row column (Q = 10: lanes l and l ^ 16 of a warp share a column, lane bit 4 =
// column bit 9, so a pass covers 64 columns).  The lane's 2*ET columns hold element k of warp
// half hw at column hw*ET + k (ET = 2^(Q-1) elements per thread, 2^8 for Q = 10).
// Bits: k0..k(et-1) local to a thread, k(et) = warp half (traded through TMEM), k9 = lane bit 4.
//   round A: own ET elements, bits k0..k5 forward (pairs on the top local bit), global -> TMEM
//   round B: bits k6..k(et) (and k9 after a half swap between the lanes) forward, gain, back;
//            each warp half takes k5 = hw
//   round C: own ET elements, bits k0..k5 again, TMEM -> global
// MODE 0 is the forward's column pass.  The backward (Q = 8, 9) runs two more: MODE 1 takes the
// column bits forward only and stores the transformed column straight from round B (no gain, no
// round C); MODE 2 is MODE 0 on the dY workspace, and at the gain step also reads the MODE 1
// result at the same positions of xws, the transformed X column, and replaces it with the product
// (W X)(W dY) times `scale` (the dG term of the plane).
template <int Q, int R, class GainT, int MODE = 0, class WS = WsF32>
__device__ __forceinline__ void col_pass_tmem(typename WS::T* ws, const GainT& gain, float scale, int m, long long u_begin,
                                              long long u_end, uint32_t tlane, float* xws = nullptr) {
  constexpr bool LANE_BIT = Q == 10;
  static_assert(MODE == 0 || std::is_same<WS, WsF32>::value, "the backward modes: fp32 workspace");
  static_assert(MODE == 0 || (!LANE_BIT && !GainT::SEPARABLE), "the backward modes: Q = 8, 9, full gains");
  constexpr int ET_BITS = LANE_BIT ? 8 : Q - 1;        // 8, 7 for Q = 9, 8; 8 for Q = 10
  constexpr int ET = 1 << ET_BITS;
  constexpr int PER_PASS = LANE_BIT ? 64 : 128;        // columns per pass
  constexpr int ITA = ET / 128;                        // round A/C iterations (64 pairs each)
  constexpr int NH = 1 << (ET_BITS - 5);               // high combinations in round B (incl. warp half)
  constexpr int W = 64 / NH;                           // pairs per high combination
  constexpr int ITB = 16 / W;                          // round B iterations
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int quarter = warp & 3, hw = warp >> 2;
  const int slot = LANE_BIT ? quarter * 16 + (lane & 15) : quarter * 32 + lane;
  const int l4 = LANE_BIT ? (lane >> 4) & 1 : 0;     // column half (rows 512 l4 ...)
  const float2 sc = make_float2(scale, scale);
  for (long long u0 = u_begin; u0 < u_end; u0 += PER_PASS) {
    const long long u = u0 + slot;
    const bool active = u < u_end;
    const long long uu = active ? u : u_begin;  // inactive lanes compute on a valid column, never store
    const long long b = uu >> R;
    const int sp = static_cast<int>(uu & ((1 << R) - 1));  // storage position of the column
    typename WS::T* colp = ws + (b << m) + sp;
    const auto gcol = gain.col(sp);
    typename WS::T* own = colp + (static_cast<long long>(l4 * 2 * ET + hw * ET) << R);
    // round A
#pragma unroll 1
    for (int it = 0; it < ITA; ++it) {
      float2 v[64];
#pragma unroll
      for (int k = 0; k < 64; ++k) {
        const long long k0 = k + 64 * it, k1 = k0 + ET / 2;
        v[k] = make_float2(WS::ld(own + (k0 << R)), WS::ld(own + (k1 << R)));
      }
      bfly_all<64>(v);
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        float lo[16], hi[16];
#pragma unroll
        for (int i = 0; i < 16; ++i) {
          lo[i] = v[16 * q + i].x;
          hi[i] = v[16 * q + i].y;
        }
        tmem_st16(tlane + hw * ET + 64 * it + 16 * q, lo);
        tmem_st16(tlane + hw * ET + ET / 2 + 64 * it + 16 * q, hi);
      }
    }
    pair_sync(quarter);
    // round B
#pragma unroll 1
    for (int it = 0; it < ITB; ++it) {
      float2 v[NH][W];
#pragma unroll
      for (int s = 0; s < NH; ++s) {
        const int s_local = s & (NH / 2 - 1), s_hw = s / (NH / 2);
        const uint32_t col = s_hw * ET + s_local * 64 + 32 * hw + 2 * W * it;
#pragma unroll
        for (int q = 0; q < 2 * W / 16; ++q) {
          float t[16];
          tmem_ld16(tlane + col + 16 * q, t);
#pragma unroll
          for (int i = 0; i < 8; ++i) v[s][8 * q + i] = make_float2(t[2 * i], t[2 * i + 1]);
        }
      }
      tmem_wait_ld();
#pragma unroll
      for (int hh = 1; hh < NH; hh <<= 1)
#pragma unroll
        for (int s = 0; s < NH; ++s)
          if ((s & hh) == 0)
#pragma unroll
            for (int w = 0; w < W; ++w) bf2(v[s][w], v[s + hh][w]);
      if constexpr (LANE_BIT) {
        lane16_swap(v, l4);
#pragma unroll
        for (int t = 0; t < 4; ++t)
#pragma unroll
          for (int w = 0; w < W; ++w) bf2(v[t][w], v[t + 4][w]);
      }
      if constexpr (MODE == 1) {  // the transformed column, rows j and j + 1 of each pair
        if (active) {
#pragma unroll
          for (int s = 0; s < NH; ++s) {
            const int s_local = s & (NH / 2 - 1), s_hw = s / (NH / 2);
            const long long j0 = s_hw * ET + s_local * 64 + 32 * hw + 2 * W * it;
#pragma unroll
            for (int w = 0; w < W; ++w) {
              const long long j = j0 + 2 * w;
              __stcg(colp + (j << R), v[s][w].x);
              __stcg(colp + ((j + 1) << R), v[s][w].y);
            }
          }
        }
      } else {
#pragma unroll
        for (int s = 0; s < NH; ++s) {
          const int s_local = s & (NH / 2 - 1), s_hw = s / (NH / 2);
          // (Q = 10: after the swap, s / 4 is column bit 9 and the warp-half bit is this lane's l4)
          const long long j0 = LANE_BIT ? s_hw * 2 * ET + l4 * ET + s_local * 64 + 32 * hw + 2 * W * it
                                        : s_hw * ET + s_local * 64 + 32 * hw + 2 * W * it;
#pragma unroll
          for (int w = 0; w < W; ++w) {
            const long long j = j0 + 2 * w;
            float2 gg;
            // (the full gain's loads are written out here: through at() the compiler spills in this loop)
            if constexpr (GainT::SEPARABLE) gg = gain.rows2(gcol, j);
            else gg = make_float2(__ldg(gcol.p + (j << R)), __ldg(gcol.p + ((j + 1) << R)));
            if constexpr (MODE == 2) {  // dG term: the transformed X column times this one, at rows j, j + 1
              float* xp = xws + (b << m) + sp + (j << R);
              const float2 xh = make_float2(__ldcg(xp), __ldcg(xp + (1ll << R)));
              const float2 pr = mul2(mul2(xh, v[s][w]), sc);
              if (active) {
                __stcg(xp, pr.x);
                __stcg(xp + (1ll << R), pr.y);
              }
            }
            v[s][w] = mul2(v[s][w], mul2(gg, sc));
          }
        }
        if constexpr (LANE_BIT) {
#pragma unroll
          for (int t = 0; t < 4; ++t)
#pragma unroll
            for (int w = 0; w < W; ++w) bf2(v[t][w], v[t + 4][w]);
          lane16_swap(v, l4);
        }
#pragma unroll
        for (int hh = 1; hh < NH; hh <<= 1)
#pragma unroll
          for (int s = 0; s < NH; ++s)
            if ((s & hh) == 0)
#pragma unroll
              for (int w = 0; w < W; ++w) bf2(v[s][w], v[s + hh][w]);
#pragma unroll
        for (int s = 0; s < NH; ++s) {
          const int s_local = s & (NH / 2 - 1), s_hw = s / (NH / 2);
          const uint32_t col = s_hw * ET + s_local * 64 + 32 * hw + 2 * W * it;
#pragma unroll
          for (int q = 0; q < 2 * W / 16; ++q) {
            float t[16];
#pragma unroll
            for (int i = 0; i < 8; ++i) {
              t[2 * i] = v[s][8 * q + i].x;
              t[2 * i + 1] = v[s][8 * q + i].y;
            }
            tmem_st16(tlane + col + 16 * q, t);
          }
        }
      }  // MODE != 1
    }
    pair_sync(quarter);
    // round C (MODE 1 stored its column from round B)
#pragma unroll 1
    for (int it = 0; it < (MODE == 1 ? 0 : ITA); ++it) {
      float2 v[64];
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        float lo[16], hi[16];
        tmem_ld16(tlane + hw * ET + 64 * it + 16 * q, lo);
        tmem_ld16(tlane + hw * ET + ET / 2 + 64 * it + 16 * q, hi);
#pragma unroll
        for (int i = 0; i < 16; ++i) v[16 * q + i] = make_float2(lo[i], hi[i]);
      }
      tmem_wait_ld();
      bfly_all<64>(v);
      if (active) {
#pragma unroll
        for (int k = 0; k < 64; ++k) {
          const long long k0 = k + 64 * it, k1 = k0 + ET / 2;
          WS::st(own + (k0 << R), v[k].x);
          WS::st(own + (k1 << R), v[k].y);
        }
      }
    }
    // the next pass's round A overwrites only this thread's own columns, which the other warp
    // of the pair stopped reading at the second pair_sync
  }
}

// ---------------------------------------------------------------------------------------------
// Forward kernel: persistent grid (one CTA per SM, all resident), plane groups of P.gp planes,
// three phases.  R and Q are template parameters so that every register array has a static size.
// WS: the workspace element (WsF32, or WsB16 for whtmix_forward_x16; full gains only).
template <int D, int R, int Q, bool SEP, class WS = WsF32>
__global__ void __launch_bounds__(THREADS, 1) k_forward_fast(Params P) {
  static_assert((R == 13 && Q >= 1 && Q <= 10) || (R == 14 && (Q == 7 || Q == 9)), "supported row/column split");
  static_assert(!SEP || std::is_same<WS, WsF32>::value, "separable gains: fp32 workspace (it holds the gain tables)");
  extern __shared__ __align__(16) unsigned char smem_raw[];
  __shared__ int flag;
  __shared__ uint32_t tmem_slot;
  constexpr bool USE_TMEM = Q >= 8;
  using RW = Row<R>;
  float* sm = reinterpret_cast<float*>(smem_raw);
  const int worker = threadIdx.x / RW::WORKER, wt = threadIdx.x % RW::WORKER;
  float* xbuf = sm + worker * RW::LEN;
  float* stg = sm + SMEM_XBUF_BYTES / sizeof(float) + worker * RW::STAGE;
  typename WS::T* ws = static_cast<typename WS::T*>(P.ws);
  const float* g = static_cast<const float*>(P.g);
  const int m = R + Q;
  uint32_t tlane = 0;
  if constexpr (USE_TMEM) {
    if (threadIdx.x < 32) tmem_alloc_512(&tmem_slot);
    tmem_fence_before();
    __syncthreads();
    tmem_fence_after();
    tlane = tmem_slot + (static_cast<uint32_t>(32 * ((threadIdx.x >> 5) & 3)) << 16);
  }
  {
    const long long rows = min(static_cast<long long>(P.gp), P.B) << Q;
    l2_prefetch_first_rows<D, R, Q>(P.x, rows * blockIdx.x / gridDim.x, rows * (blockIdx.x + 1) / gridDim.x, P.lv);
  }
  // tensor memory is allocated before the wait: the previous kernel's CTA on this SM has left
  pdl_wait();
  GridSync gsync(P.bar, &flag);
  for (long long b0 = 0; b0 < P.B; b0 += P.gp) {
    const long long nb = min(static_cast<long long>(P.gp), P.B - b0);
    const long long rows = nb << Q;
    const long long rb = rows * blockIdx.x / gridDim.x, re = rows * (blockIdx.x + 1) / gridDim.x;
    // phase-2 column range: balanced, aligned to 8 columns
    const long long cols = nb << R;
    const long long cb = ((cols * blockIdx.x / gridDim.x) + 4) & ~7ll;
    const long long ce = blockIdx.x + 1 == gridDim.x ? cols : ((cols * (blockIdx.x + 1) / gridDim.x) + 4) & ~7ll;
    // phase 1: X -> ws, row bits (and, once, the separable gain tables exp(g_t), exp(g_c))
    if constexpr (SEP) {
      if (b0 == 0) {
        float* tab = reinterpret_cast<float*>(ws) + (static_cast<long long>(P.gp) << m);
        const long long n_t = 1ll << (m - P.cbits), n_tab = n_t + (1ll << P.cbits);
        for (long long i = static_cast<long long>(blockIdx.x) * THREADS + threadIdx.x; i < n_tab;
             i += static_cast<long long>(gridDim.x) * THREADS)
          tab[i] = expf(i < n_t ? P.gt[sep_token_of<R, Q>(i, P.cbits)] : P.gc[i - n_t]);
      }
    }
    if (rb + worker < re) {
      long long e0;
      int lim;
      row_loc<R, Q>(b0, rb + worker, P.lv, &e0, &lim);
      stage_row_in<D, R>(P.x, e0, stg, wt, lim);
    }
    for (long long r = rb + worker; r < re; r += RW::NWORKERS) {
      const long long rn = r + RW::NWORKERS;
      // G is first read in phase 2; its fetch into L2 is spread over phase 1 (one bulk prefetch
      // per row, together the CTA's share of G), where HBM carries only X.
      if (!SEP && b0 == 0 && wt == 0) l2_prefetch_piece(g, 4ll << m, r - rb, re - rb);
      long long e0, e0n;
      int lim, limn;
      row_loc<R, Q>(b0, r, P.lv, &e0, &lim);
      row_loc<R, Q>(b0, rn, P.lv, &e0n, &limn);
      row_forward_in<D, R, WS>(P.x, e0, lim, ws + (r << R), xbuf, stg, wt, worker, rn < re ? P.x : nullptr, e0n, limn);
    }
    if (!gsync()) break;
    // phase 2: column bits, gain, column bits
    {
      using GainT = typename std::conditional<SEP, SepGain<R, Q>, FullGain<R>>::type;
      GainT gain;
      if constexpr (SEP) {
        const float* tab = reinterpret_cast<const float*>(ws) + (static_cast<long long>(P.gp) << m);
        gain = GainT{tab, tab + (1ll << (m - P.cbits)), P.cbits};
      } else {
        gain = GainT{g};
      }
      if constexpr (USE_TMEM) col_pass_tmem<Q, R, GainT, 0, WS>(ws, gain, P.scale, m, cb, ce, tlane);
      else if constexpr (Q == 7) col_pass_single128<R, GainT, WS>(ws, gain, P.scale, m, cb, ce);
      else col_pass_pairs<Q, R, GainT, WS>(ws, gain, P.scale, m, cb, ce);
    }
    if (!gsync()) break;
    // phase 3: ws -> Y, row bits
    if (rb + worker < re) stage_row_out<R, WS>(ws + ((rb + worker) << R), stg, wt);
    for (long long r = rb + worker; r < re; r += RW::NWORKERS) {
      const long long rn = r + RW::NWORKERS;
      long long e0;
      int lim;
      row_loc<R, Q>(b0, r, P.lv, &e0, &lim);
      row_forward_out<D, R, WS>(ws + (r << R), P.y, e0, lim, xbuf, stg, wt, worker, rn < re ? ws + (rn << R) : nullptr);
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
