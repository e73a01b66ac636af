// whtmix_block.cuh -- the whole mixer block of Section III-B, Eq. 1-4, as one persistent kernel for
// bf16 planes of 128 channels and 2^21..2^23 elements:
//   Y_b = ( H_N (G o (H_N (X_b W_in^T) H_C)) H_C / (N C) ) W_out^T
// The two projections are the prologue of the first row phase and the epilogue of the last, on the
// tensor cores, so X and Y cross HBM once (the unfused block is three launches).
//
// A row is a tile of 128 tokens x 128 channels (2^14 elements), handled by a worker of 128 threads
// (two per CTA); thread t of the worker owns TMEM lane t.
//   phase 1, per row: X tile -> shared memory (the tensor core's 128-byte-swizzled K-major layout)
//     -> tcgen05.mma with W_in -> TMEM (lane = token, column = channel) -> thread t holds token t's
//     128 channels: the channel transform in registers -> a swizzled shared-memory transpose ->
//     thread c holds channel c's 128 tokens: the token transform in registers -> the workspace in
//     natural order (a warp's stores are 128 contiguous bytes).
//   phase 2: the fast forward's column pass (columns of 2^(m-14) rows, gain G/L, natural order).
//   phase 3, per row: the mirror image, ending with the tile rounded to bf16 (the block's
//     activations) as the A operand of tcgen05.mma with W_out; the output tile leaves through a
//     shared-memory staging area in coalesced stores.
// The arithmetic between the projections is fp32; Z = X W_in^T is not rounded.
#pragma once

#include "whtmix_fast.cuh"

namespace whtmix {
namespace blk {

using fast::THREADS;   // 8 warps: workers 0 (warps 0-3) and 1 (warps 4-7)
constexpr int R = 14;  // 128 tokens x 128 channels per row
constexpr int WORKER = 128;
constexpr int BUF_BYTES = 128 * 132 * 4;  // per worker: the transpose buffer (its first 32 KiB also stage the A operand)
constexpr size_t SMEM_BYTES = 1024 + 2 * 32768 + 2 * BUF_BYTES;  // alignment slack, W_in, W_out, the workers' buffers
constexpr long long WAIT_LIMIT = 1ll << 26;

__device__ __forceinline__ uint32_t smem_u32(const void* p) { return static_cast<uint32_t>(__cvta_generic_to_shared(p)); }
// 128 x 128 bf16 K-major operand, 128-byte swizzle: two atoms of 64 elements along K
__device__ __forceinline__ uint32_t sw_off(int r, int k) {
  return static_cast<uint32_t>((k >> 6) * 16384 + r * 128 + ((((k >> 3) & 7) ^ (r & 7)) << 4) + (k & 7) * 2);
}
__device__ __forceinline__ uint64_t op_desc(uint32_t base, int ks) {
  const uint32_t a = base + (ks >> 2) * 16384 + (ks & 3) * 32;
  return static_cast<uint64_t>((a & 0x3FFFFu) >> 4) | (1ull << 16) | (static_cast<uint64_t>(1024 >> 4) << 32) |
         (1ull << 46) | (2ull << 61);
}
constexpr uint32_t IDESC = (1u << 4) | (1u << 7) | (1u << 10) | ((128u >> 3) << 17) | ((128u >> 4) << 24);

// (a rolled loop: unrolled, the 16 descriptors of each operand pair are loop invariants the
// compiler keeps in registers for the whole kernel)
__device__ __forceinline__ void mma_tile(uint32_t d, uint32_t a_base, uint32_t b_base) {
#pragma unroll 1
  for (int ks = 0; ks < 8; ++ks)
    asm volatile("{\n\t.reg .pred p;\n\tsetp.ne.b32 p, %4, 0;\n\ttcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}"
                 ::"r"(d), "l"(op_desc(a_base, ks)), "l"(op_desc(b_base, ks)), "r"(IDESC), "r"(ks > 0 ? 1u : 0u) : "memory");
}
__device__ __forceinline__ void mma_commit(uint64_t* bar) {
  asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(smem_u32(bar)) : "memory");
}
__device__ __forceinline__ bool mbar_wait(uint64_t* bar, uint32_t parity) {
  const uint32_t a = smem_u32(bar);
  for (long long i = 0; i < WAIT_LIMIT; ++i) {
    uint32_t done;
    asm volatile("{\n\t.reg .pred p;\n\tmbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\tselp.u32 %0, 1, 0, p;\n\t}"
                 : "=r"(done) : "r"(a), "r"(parity) : "memory");
    if (done) return true;
  }
  return false;
}
__device__ __forceinline__ void wsync(int worker) { asm volatile("bar.sync %0, %1;" ::"r"(worker + 1), "r"(WORKER) : "memory"); }

// Transpose buffer (fp32 128 x 128, rows padded to 132 floats): a quarter warp writing 16-byte
// chunks of 8 consecutive rows, or a warp reading one float of 32 consecutive columns, touches every
// bank once, and a thread's addresses are its own base plus compile-time offsets.
constexpr int TSTRIDE = 132;
__device__ __forceinline__ int tpos(int t, int c) { return t * TSTRIDE + c; }

// The 128 projected values of this thread's TMEM lane (its token), as pairs (c, c + 64).
__device__ __forceinline__ void tmem_row(uint32_t ta, float2 (&v)[64]) {
  float t[128];
#pragma unroll
  for (int c = 0; c < 128; c += 16) fast::tmem_ld16(ta + c, *reinterpret_cast<float(*)[16]>(t + c));
  fast::tmem_wait_ld();
#pragma unroll
  for (int k = 0; k < 64; ++k) v[k] = make_float2(t[k], t[k + 64]);
}

// 128-point transform of the pairs (k, k + 64): bits 0..5 across the pairs, bit 6 inside.
__device__ __forceinline__ void fwht128(float2 (&v)[64]) {
  fast::bfly_all<64>(v);
#pragma unroll
  for (int k = 0; k < 64; ++k) fast::bf_in(v[k]);
}

// An opaque copy of v: what is computed from it is computed where it is used, not hoisted out of
// the persistent loop into registers held across all three phases.
__device__ __forceinline__ uint32_t fresh(uint32_t v) {
  uint32_t r;
  asm volatile("mov.b32 %0, %1;" : "=r"(r) : "r"(v));
  return r;
}
template <class T>
__device__ __forceinline__ T* fresh(T* p) {
  uint64_t r;
  asm volatile("mov.b64 %0, %1;" : "=l"(r) : "l"(reinterpret_cast<uint64_t>(p)));
  return reinterpret_cast<T*>(r);
}

// Shared state of the kernel, at namespace scope so that the tile functions reach it directly.
extern __shared__ __align__(1024) unsigned char blk_smem_raw[];
__shared__ uint32_t blk_tmem_slot;
__shared__ uint64_t blk_mbar[2];

// Tile context of one worker: its buffer, the resident B operand, its accumulator, its mbarrier.
// Rebuilt at the start of each tile from the thread index and the shared symbols (through fresh(),
// so that it is not hoisted into registers held across the whole kernel).
struct Tile {
  unsigned char* buf;
  uint32_t w;      // shared address of W (W_in or W_out), 128-byte swizzled
  uint32_t acc;    // this thread's TMEM lane of the worker's accumulator columns
  uint32_t acc_d;  // the accumulator (lane 0) as the MMA's D
  uint64_t* bar;
  int worker, wt;
};
// Operands start on 1024-byte boundaries (the 128-byte swizzle is a function of the address):
// W_in at 0, W_out at 32 KiB, worker buffers from 64 KiB.
__device__ __forceinline__ unsigned char* block_smem() {
  return blk_smem_raw + ((1024u - (smem_u32(blk_smem_raw) & 1023u)) & 1023u);
}
template <bool OUT>
__device__ __forceinline__ Tile make_tile() {
  const uint32_t tid = fresh(static_cast<uint32_t>(threadIdx.x));
  const int worker = static_cast<int>(tid / WORKER), wt = static_cast<int>(tid % WORKER);
  unsigned char* smem = block_smem();
  const uint32_t slot = blk_tmem_slot;
  return {smem + 65536 + worker * BUF_BYTES, smem_u32(smem) + (OUT ? 32768u : 0u),
          slot + (static_cast<uint32_t>(32 * ((tid >> 5) & 3)) << 16) + 128u * worker, slot + 128u * worker,
          &blk_mbar[worker], worker, wt};
}

// One MMA tile: elected thread issues C / 16 MMAs into the worker's accumulator; every thread of
// the worker waits for their commit (bounded).  False if the wait gave up.
__device__ __forceinline__ bool tile_mma(const Tile& T, uint32_t parity) {
  if (T.wt == 0) {
    fast::tmem_fence_after();
    mma_tile(T.acc_d, smem_u32(T.buf), T.w);
    mma_commit(T.bar);
  }
  const bool ok = __all_sync(0xffffffffu, mbar_wait(T.bar, parity));
  fast::tmem_fence_after();
  return ok;
}

// Staging of a worker's next tile into its buffer, by cp.async (16-byte chunks, consecutive
// threads on consecutive chunks); the tile that consumes it waits for the copies.
// X tile (128 tokens x 128 channels, bf16) in the MMA's A-operand layout.
__device__ __forceinline__ void stage_x(unsigned char* buf, const __nv_bfloat16* __restrict__ xt, int wt) {
#pragma unroll
  for (int i = 0; i < 16; ++i) {
    const int q = wt + WORKER * i, t = q >> 4, c = (q & 15) * 8;
    fast::cp_async16(reinterpret_cast<float*>(buf + sw_off(t, c)), xt + t * 128 + c);
  }
  fast::cp_async_commit();
}
// Workspace row (2^14 fp32: token t, channel c at t * 128 + c) in the transpose layout.
__device__ __forceinline__ void stage_ws(float* fbuf, const float* __restrict__ wsr, int wt) {
#pragma unroll
  for (int i = 0; i < 32; ++i) {
    const int q = wt + WORKER * i, t = q >> 5, c = (q & 31) * 4;
    fast::cp_async16(fbuf + tpos(t, c), wsr + t * 128 + c);
  }
  fast::cp_async_commit();
}
__device__ __forceinline__ unsigned char* worker_buf(int worker) { return block_smem() + 65536 + worker * BUF_BYTES; }

// Phase 1 for one row: X tile (staged by the previous call or the phase's prologue) -> Z = X W_in^T
// -> channel transform -> token transform -> 2^14 fp32 workspace values in natural order.  Once the
// buffer is free, the next tile's X (xt_next, if any) is staged behind the token transform and
// the stores.  A worker without a row (active false) only takes part in the worker's barriers.
// After a failed MMA wait the tile still runs to the end (on whatever TMEM holds) so that the
// barriers stay matched; the caller records the error.
__device__ __forceinline__ bool tile_in(float* __restrict__ wsr, const __nv_bfloat16* xt_next, uint32_t parity,
                                        bool active) {
  if (!active) {
    const int worker = threadIdx.x / WORKER;
    wsync(worker);
    wsync(worker);
    wsync(worker);
    return true;
  }
  const Tile T = make_tile<false>();
  float* fbuf = reinterpret_cast<float*>(T.buf);
  const int wt = T.wt;
  fast::cp_async_wait_all();
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
  wsync(T.worker);
  const bool ok = tile_mma(T, parity);
  float2 v[64];
  tmem_row(T.acc, v);  // token wt's 128 channels
  fast::tmem_fence_before();
  fwht128(v);          // channels
#pragma unroll
  for (int j = 0; j < 16; ++j) {
    *reinterpret_cast<float4*>(fbuf + tpos(wt, 4 * j)) = make_float4(v[4 * j].x, v[4 * j + 1].x, v[4 * j + 2].x, v[4 * j + 3].x);
    *reinterpret_cast<float4*>(fbuf + tpos(wt, 64 + 4 * j)) =
        make_float4(v[4 * j].y, v[4 * j + 1].y, v[4 * j + 2].y, v[4 * j + 3].y);
  }
  wsync(T.worker);
#pragma unroll
  for (int k = 0; k < 64; ++k) v[k] = make_float2(fbuf[tpos(k, wt)], fbuf[tpos(k + 64, wt)]);  // channel wt's tokens
  wsync(T.worker);  // the buffer is free: the next tile's X streams in behind this one's stores
  if (xt_next) stage_x(T.buf, xt_next, wt);
  fwht128(v);       // tokens
  float* out = wsr + wt;
#pragma unroll
  for (int k = 0; k < 64; ++k) {
    __stcg(out + k * 128, v[k].x);
    __stcg(out + (k + 64) * 128, v[k].y);
  }
  return ok;
}

// Phase 3 for one row: 2^14 workspace values (staged by the previous call or the phase's
// prologue) -> token transform -> channel transform -> M (bf16) -> Y = M W_out^T (bf16, 128
// tokens x 128 channels).  The next row (wsr_next, if any) is staged once the MMA has read the
// buffer, behind this tile's output.  Inactive workers and failed waits as in tile_in.
__device__ __forceinline__ bool tile_out(const float* wsr_next, __nv_bfloat16* __restrict__ yt, uint32_t parity,
                                         bool active) {
  if (!active) {
    const int worker = threadIdx.x / WORKER;
#pragma unroll 1
    for (int i = 0; i < 8; ++i) wsync(worker);  // as many as an active tile
    return true;
  }
  const Tile T = make_tile<true>();
  float* fbuf = reinterpret_cast<float*>(T.buf);
  const int wt = T.wt;
  fast::cp_async_wait_all();
  wsync(T.worker);
  float2 v[64];
  // channel wt's 128 tokens, transformed in place: each thread reads and writes only its column
#pragma unroll
  for (int k = 0; k < 64; ++k) v[k] = make_float2(fbuf[tpos(k, wt)], fbuf[tpos(k + 64, wt)]);
  fwht128(v);  // tokens
#pragma unroll
  for (int k = 0; k < 64; ++k) {
    fbuf[tpos(k, wt)] = v[k].x;
    fbuf[tpos(k + 64, wt)] = v[k].y;
  }
  wsync(T.worker);
#pragma unroll
  for (int j = 0; j < 16; ++j) {
    const float4 lo = *reinterpret_cast<const float4*>(fbuf + tpos(wt, 4 * j));
    const float4 hi = *reinterpret_cast<const float4*>(fbuf + tpos(wt, 64 + 4 * j));
    v[4 * j] = make_float2(lo.x, hi.x);
    v[4 * j + 1] = make_float2(lo.y, hi.y);
    v[4 * j + 2] = make_float2(lo.z, hi.z);
    v[4 * j + 3] = make_float2(lo.w, hi.w);
  }
  wsync(T.worker);
  fwht128(v);  // channels of token wt: v[k] = (channel k, channel k + 64)
  // M (bf16, the block's activations) as the A operand: row = token, K = channel
#pragma unroll
  for (int j = 0; j < 8; ++j) {
    uint32_t lo4[4], hi4[4];
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      __nv_bfloat162 a = __floats2bfloat162_rn(v[8 * j + 2 * q].x, v[8 * j + 2 * q + 1].x);
      __nv_bfloat162 b = __floats2bfloat162_rn(v[8 * j + 2 * q].y, v[8 * j + 2 * q + 1].y);
      lo4[q] = *reinterpret_cast<uint32_t*>(&a);
      hi4[q] = *reinterpret_cast<uint32_t*>(&b);
    }
    *reinterpret_cast<uint4*>(T.buf + sw_off(wt, 8 * j)) = make_uint4(lo4[0], lo4[1], lo4[2], lo4[3]);
    *reinterpret_cast<uint4*>(T.buf + sw_off(wt, 64 + 8 * j)) = make_uint4(hi4[0], hi4[1], hi4[2], hi4[3]);
  }
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
  wsync(T.worker);
  const bool ok = tile_mma(T, parity);
  if (wsr_next) stage_ws(fbuf, wsr_next, wt);  // the MMA has read the buffer
  // Y in two halves of 64 channels through a 16 KiB staging area (rows of 128 bytes, 16-byte
  // chunks XOR-swizzled by the row): thread t writes token t's half row, then the worker stores
  // the half tile with 8 consecutive threads on each token's 128 bytes.
  unsigned char* ystg = block_smem() + T.worker * 16384;  // the W_in region, unused in this phase
#pragma unroll
  for (int h = 0; h < 2; ++h) {
    float y[64];
#pragma unroll
    for (int c = 0; c < 64; c += 16) fast::tmem_ld16(T.acc + 64 * h + c, *reinterpret_cast<float(*)[16]>(y + c));
    fast::tmem_wait_ld();
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      uint32_t q4[4];
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        __nv_bfloat162 b = __floats2bfloat162_rn(y[8 * j + 2 * q], y[8 * j + 2 * q + 1]);
        q4[q] = *reinterpret_cast<uint32_t*>(&b);
      }
      *reinterpret_cast<uint4*>(ystg + wt * 128 + ((j ^ (wt & 7)) << 4)) = make_uint4(q4[0], q4[1], q4[2], q4[3]);
    }
    wsync(T.worker);
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      const int q = wt + WORKER * i, t = q >> 3, c = q & 7;
      const uint4 val = *reinterpret_cast<const uint4*>(ystg + t * 128 + ((c ^ (t & 7)) << 4));
      __stcs(reinterpret_cast<uint4*>(yt + t * 128 + 64 * h + 8 * c), val);
    }
    wsync(T.worker);  // the staging area is free
  }
  fast::tmem_fence_before();
  return ok;
}

template <int Q>
__global__ void __launch_bounds__(THREADS, 1) k_block_fast(Params P, const __nv_bfloat16* __restrict__ w_in,
                                                            const __nv_bfloat16* __restrict__ w_out) {
  static_assert(Q >= 7 && Q <= 9, "columns of 128 to 512 rows");
  __shared__ int flag;
  pdl_wait();
  GridSync gsync(P.bar, &flag);
  const int m = R + Q;
  const int worker = threadIdx.x / WORKER, wt = threadIdx.x % WORKER;
  unsigned char* sWin = block_smem();
  unsigned char* sWout = sWin + 32768;
  float* ws = static_cast<float*>(P.ws);
  const float* g = static_cast<const float*>(P.g);
  // W_in and W_out (out, in) as the B operand: rows = output channels, K = input channels.  Phase 3
  // stages Y in W_in's place, so W_in is loaded again for every later plane group.
  for (int q = threadIdx.x; q < 128 * 16; q += THREADS) {
    const int r = q >> 4, k = (q & 15) * 8;
    *reinterpret_cast<uint4*>(sWin + sw_off(r, k)) = __ldg(reinterpret_cast<const uint4*>(w_in + r * 128 + k));
    *reinterpret_cast<uint4*>(sWout + sw_off(r, k)) = __ldg(reinterpret_cast<const uint4*>(w_out + r * 128 + k));
  }
  if (threadIdx.x < 32) fast::tmem_alloc_512(&blk_tmem_slot);
  if (threadIdx.x == 0) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], 1;" ::"r"(smem_u32(&blk_mbar[0])) : "memory");
    asm volatile("mbarrier.init.shared::cta.b64 [%0], 1;" ::"r"(smem_u32(&blk_mbar[1])) : "memory");
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
  fast::tmem_fence_before();
  __syncthreads();
  fast::tmem_fence_after();
  uint32_t parity = 0;
  bool ok = true;
  const __nv_bfloat16* x = static_cast<const __nv_bfloat16*>(P.x);
  __nv_bfloat16* y = static_cast<__nv_bfloat16*>(P.y);
  for (long long b0 = 0; b0 < P.B; b0 += P.gp) {
    const long long nb = min(static_cast<long long>(P.gp), P.B - b0);
    const long long rows = nb << Q;
    const long long rb = rows * blockIdx.x / gridDim.x, re = rows * (blockIdx.x + 1) / gridDim.x;
    const long long cols = nb << R;
    const long long cb = ((cols * blockIdx.x / gridDim.x) + 4) & ~7ll;
    const long long ce = blockIdx.x + 1 == gridDim.x ? cols : ((cols * (blockIdx.x + 1) / gridDim.x) + 4) & ~7ll;
    if (b0 > 0) {
      for (int q = threadIdx.x; q < 128 * 16; q += THREADS) {
        const int r = q >> 4, k = (q & 15) * 8;
        *reinterpret_cast<uint4*>(sWin + sw_off(r, k)) = __ldg(reinterpret_cast<const uint4*>(w_in + r * 128 + k));
      }
      asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
      __syncthreads();
    }
    // phase 1: X -> (W_in) -> channel and token transforms -> workspace (row r of the group is
    // plane b0 + (r >> Q), tokens 128 (r mod 2^Q) ...)
    // G, first read in phase 2, is fetched into L2 in pieces, one per tile.  (Fetching the
    // worker's later X tiles into L2 up front as well: 4 us slower in the phase probe, no change in
    // the steady-state bench; left out.)
    if (rb + worker < re) stage_x(worker_buf(worker), x + (b0 << m) + ((rb + worker) << R), wt);
    for (long long r = rb + worker; r < re + worker; r += 2) {
      const bool active = r < re && ok;
      const __nv_bfloat16* xn = r + 2 < re ? x + (b0 << m) + ((r + 2) << R) : nullptr;
      if (b0 == 0 && wt == 0 && r < re) fast::l2_prefetch_piece(g, 4ll << m, r - rb, re - rb);
      if (!tile_in(ws + (r << R), xn, parity, active)) ok = false;
      if (active) parity ^= 1u;
    }
    fast::tmem_fence_before();
    if (__syncthreads_or(!ok) || !gsync()) break;
    fast::tmem_fence_after();
    // phase 2: column bits, gain, column bits (natural-order workspace)
    {
      // natural order: column sp holds channel sp % 128 of token (j << 7) + sp / 128
      const fast::FullGain<R, true> gain{g};
      const uint32_t lane_ta = blk_tmem_slot + (static_cast<uint32_t>(32 * ((threadIdx.x >> 5) & 3)) << 16);
      if constexpr (Q >= 8) fast::col_pass_tmem<Q, R>(ws, gain, P.scale, m, cb, ce, lane_ta);
      else fast::col_pass_single128<R>(ws, gain, P.scale, m, cb, ce);
    }
    fast::tmem_fence_before();
    if (!gsync()) break;
    fast::tmem_fence_after();
    // phase 3: token and channel transforms -> bf16 -> (W_out) -> Y
    if (rb + worker < re) stage_ws(reinterpret_cast<float*>(worker_buf(worker)), ws + ((rb + worker) << R), wt);
    for (long long r = rb + worker; r < re + worker; r += 2) {
      const bool active = r < re && ok;
      const float* wn = r + 2 < re ? ws + ((r + 2) << R) : nullptr;
      if (!tile_out(wn, y + (b0 << m) + (r << R), parity, active)) ok = false;
      if (active) parity ^= 1u;
    }
    if (__syncthreads_or(!ok) || (b0 + P.gp < P.B && !gsync())) break;
  }
  if (!ok && threadIdx.x == 0) atomicOr(&P.bar->err, 1u << 12);
  fast::cp_async_wait_all();  // staging left in flight by an early exit
  fast::tmem_fence_before();
  __syncthreads();
  fast::tmem_fence_after();
  pdl_trigger();
  if (threadIdx.x < 32) fast::tmem_dealloc_512(blk_tmem_slot);
}

}  // namespace blk
}  // namespace whtmix
