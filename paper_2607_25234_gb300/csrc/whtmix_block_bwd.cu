// whtmix_block_bwd.cu -- the pieces of the mixer block's backward (Section III-B, Eq. 1-4) that the
// forward kernels do not already provide: the weight gradients
//     dW[o, i] = sum over tokens t of A[t, o] B[t, i]      (dW_out = dY^T M, dW_in = dZ^T X)
// on the 5th-generation tensor cores, and the transposes that feed them.
//
// A and B are [T, C] bf16 token rows; the contraction runs over the tokens, so both are first
// transposed into [C, Tp] (Tp = T rounded up to 64, zero past T) -- K-major operands for the MMA.
// k_wgrad splits the tokens into one chunk per CTA (one persistent CTA per SM, 128 threads): per
// K tile of 64 tokens the CTA stages the A rows (output channels o, 128 per MMA tile) and the B rows
// (input channels i) in the tensor core's no-swizzle K-major canonical layout, double-buffered,
// and one thread issues tcgen05.mma (kind::f16, M = 128, N = C, K = 16) into a TMEM accumulator
// per 128 rows of o, committed to an mbarrier per buffer.  Each thread then reads its row o of the
// accumulator (tcgen05.ld) into the chunk's fp32 partial [C, C]; k_wgrad_reduce adds the partials
// in ascending chunk order, so dW is the same bit for bit on every run.
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "whtmix_kernels.cuh"
#include "whtmix_tc.cuh"

namespace whtmix {
namespace bbwd {

using namespace tc;

constexpr int KT = 64;             // tokens per K tile (one 128-byte row of bf16 per operand row)
constexpr int WG_THREADS = 128;    // one thread per TMEM lane = per output row o of an MMA tile
constexpr int TR_THREADS = 256;
constexpr size_t SMEM_MIN = 120 * 1024;  // more than half an SM: one CTA per SM, so TMEM allocation never waits

// out[c, t] = in[t, c] for t < T, 0 for T <= t < Tp (both bf16; C a multiple of 64, Tp of 64).
__global__ void __launch_bounds__(TR_THREADS) k_transpose(const uint16_t* __restrict__ in, uint16_t* __restrict__ out,
                                                          long long T, int C, long long Tp) {
  __shared__ uint16_t tile[64][66];
  pdl_wait();
  const long long ntt = Tp / 64;
  const int nct = C / 64, tx = threadIdx.x & 63, ty = threadIdx.x >> 6;
  for (long long blk = blockIdx.x; blk < ntt * nct; blk += gridDim.x) {
    const long long tt = blk / nct;
    const int ct = static_cast<int>(blk - tt * nct);
    for (int r = ty; r < 64; r += TR_THREADS / 64) {
      const long long t = tt * 64 + r;
      tile[r][tx] = t < T ? in[t * C + ct * 64 + tx] : static_cast<uint16_t>(0);
    }
    __syncthreads();
    for (int r = ty; r < 64; r += TR_THREADS / 64) out[static_cast<long long>(ct * 64 + r) * Tp + tt * 64 + tx] = tile[tx][r];
    __syncthreads();
  }
  pdl_trigger();
}

// Partial weight gradient of token chunk blockIdx.x: part[chunk][o][i] = sum over the chunk's
// tokens of At[o][t] Bt[i][t].  C in {64, 128, 256}.
template <int C>
__global__ void __launch_bounds__(WG_THREADS, 1) k_wgrad(const __nv_bfloat16* __restrict__ At,
                                                         const __nv_bfloat16* __restrict__ Bt, float* __restrict__ part,
                                                         long long Tp, int nchunk, unsigned int* err) {
  constexpr int MT = C > 128 ? C / 128 : 1;          // MMA tiles of 128 output rows
  constexpr int AR = MT * 128;                       // staged A rows (rows >= C are zero)
  constexpr uint32_t A_BYTES = AR * KT * 2, B_BYTES = C * KT * 2, STAGE = A_BYTES + B_BYTES;
  constexpr uint32_t TCOLS = MT * C;                 // 64, 128 or 512 TMEM columns
  static_assert(C == 64 || C == 128 || C == 256, "channels");
  extern __shared__ __align__(1024) unsigned char smem[];
  __shared__ uint64_t mbar[2];
  __shared__ uint32_t tmem_slot;
  const int tid = threadIdx.x, warp = tid >> 5;
  if (tid < 32) tmem_alloc(&tmem_slot, TCOLS);
  if (tid == 0) {
    mbar_init(&mbar[0], 1);
    mbar_init(&mbar[1], 1);
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
  __syncthreads();
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
  pdl_wait();
  const uint32_t tmem = tmem_slot;
  const long long ntiles = Tp / KT;
  const long long k0 = ntiles * blockIdx.x / nchunk, k1 = ntiles * (blockIdx.x + 1) / nchunk;

  // K tile kt of both operands into buffer `buf`, canonical layout (8-row x 16-byte core matrices,
  // the K-adjacent one 128 bytes on, the next 8 rows KT / 8 x 128 bytes on)
  auto stage = [&](long long kt, int buf) {
    unsigned char* sa = smem + buf * STAGE;
    unsigned char* sb = sa + A_BYTES;
    const long long t0 = kt * KT;
    for (int q = tid; q < AR * (KT / 8); q += WG_THREADS) {
      const int r = q / (KT / 8), k = (q % (KT / 8)) * 8;
      uint4 v = make_uint4(0u, 0u, 0u, 0u);
      if (r < C) v = __ldcs(reinterpret_cast<const uint4*>(At + r * Tp + t0 + k));
      *reinterpret_cast<uint4*>(sa + core_off(r, k, KT)) = v;
    }
    for (int q = tid; q < C * (KT / 8); q += WG_THREADS) {
      const int r = q / (KT / 8), k = (q % (KT / 8)) * 8;
      *reinterpret_cast<uint4*>(sb + core_off(r, k, KT)) = __ldcs(reinterpret_cast<const uint4*>(Bt + r * Tp + t0 + k));
    }
    // generic-proxy shared-memory writes -> visible to the tensor core (async proxy)
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
  };

  const uint32_t idesc = instr_desc(128, C);
  uint32_t parity[2] = {0u, 0u};
  bool ok = true;
  stage(k0, 0);
  __syncthreads();
  for (long long kt = k0; kt < k1; ++kt) {
    const int buf = static_cast<int>((kt - k0) & 1);
    if (tid == 0) {
      asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
      const uint32_t sa = smem_u32(smem + buf * STAGE), sb = sa + A_BYTES;
#pragma unroll
      for (int mt = 0; mt < MT; ++mt)
#pragma unroll
        for (int ks = 0; ks < KT / 16; ++ks)  // K steps of 16: two core matrices along K
          mma_bf16(tmem + mt * C, smem_desc(sa + mt * (128 * KT * 2) + ks * 256, 128, (KT / 8) * 128),
                   smem_desc(sb + ks * 256, 128, (KT / 8) * 128), idesc, (kt > k0 || ks > 0) ? 1u : 0u);
      mma_commit(&mbar[buf]);
    }
    if (kt + 1 < k1) {
      const int nb = buf ^ 1;
      if (kt > k0) {  // buffer nb is free once the MMAs of tile kt - 1 (its last reader) completed
        ok = __syncthreads_and(mbar_wait(&mbar[nb], parity[nb]) ? 1 : 0) != 0;
        parity[nb] ^= 1u;
        if (!ok) break;
      }
      stage(kt + 1, nb);
      __syncthreads();
    }
  }
  if (ok && k1 > k0) {  // the last tile's commit covers every MMA issued before it
    const int lb = static_cast<int>((k1 - 1 - k0) & 1);
    ok = __syncthreads_and(mbar_wait(&mbar[lb], parity[lb]) ? 1 : 0) != 0;
  }
  if (!ok && tid == 0) atomicOr(err, 1u << 13);
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
  // row o = mt * 128 + tid of the accumulator -> this chunk's partial (zeros for an empty chunk)
  float* pc = part + static_cast<long long>(blockIdx.x) * C * C;
#pragma unroll 1
  for (int mt = 0; mt < MT; ++mt) {
    const int o = mt * 128 + tid;
#pragma unroll 1
    for (int c0 = 0; c0 < C; c0 += 16) {
      float v[16];
      tmem_ld16(tmem + (static_cast<uint32_t>(32 * warp) << 16) + mt * C + c0, v);
      asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
      if (o < C) {
        float4* dst = reinterpret_cast<float4*>(pc + static_cast<long long>(o) * C + c0);
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          const bool live = ok && k1 > k0;
          dst[q] = live ? make_float4(v[4 * q], v[4 * q + 1], v[4 * q + 2], v[4 * q + 3]) : make_float4(0.f, 0.f, 0.f, 0.f);
        }
      }
    }
  }
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
  __syncthreads();
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
  pdl_trigger();
  if (tid < 32) tmem_dealloc(tmem, TCOLS);
}

// dW[o][i] = sum of the chunks' partials in ascending chunk order (float32).
__global__ void __launch_bounds__(TR_THREADS) k_wgrad_reduce(const float* __restrict__ part, float* __restrict__ out,
                                                             int cc, int nchunk) {
  pdl_wait();
  for (int q = blockIdx.x * blockDim.x + threadIdx.x; q < cc; q += gridDim.x * blockDim.x) {
    float acc = 0.f;
    for (int c = 0; c < nchunk; ++c) acc += part[static_cast<long long>(c) * cc + q];
    out[q] = acc;
  }
  pdl_trigger();
}

// ---- host ----

// Token chunks of one weight gradient: one per SM, at most one per K tile.
int wgrad_chunks(long long Tp, int sms) {
  const long long nt = Tp / KT;
  return static_cast<int>(nt < sms ? (nt < 1 ? 1 : nt) : sms);
}

cudaError_t transpose(const void* in, void* out, long long T, int C, long long Tp, int sms, cudaStream_t stream) {
  const long long blocks = (Tp / 64) * (C / 64);
  const unsigned grid = static_cast<unsigned>(blocks < 8ll * sms ? (blocks < 1 ? 1 : blocks) : 8ll * sms);
  const uint16_t* i = static_cast<const uint16_t*>(in);
  uint16_t* o = static_cast<uint16_t*>(out);
  void* args[] = {&i, &o, &T, &C, &Tp};
  return launch_pdl(reinterpret_cast<const void*>(k_transpose), grid, TR_THREADS, 0, stream, args);
}

template <int C>
cudaError_t wgrad_c(const void* at, const void* bt, float* part, float* out, long long Tp, int sms, unsigned int* err,
                    cudaStream_t stream) {
  constexpr int MT = C > 128 ? C / 128 : 1;
  constexpr size_t need = 2ull * (MT * 128 + C) * KT * 2;
  const size_t smem = need > SMEM_MIN ? need : SMEM_MIN;
  const void* k = reinterpret_cast<const void*>(k_wgrad<C>);
  cudaError_t e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
  if (e != cudaSuccess) return e;
  int nchunk = wgrad_chunks(Tp, sms);
  const __nv_bfloat16* a = static_cast<const __nv_bfloat16*>(at);
  const __nv_bfloat16* b = static_cast<const __nv_bfloat16*>(bt);
  void* args[] = {&a, &b, &part, &Tp, &nchunk, &err};
  e = launch_pdl(k, static_cast<unsigned>(nchunk), WG_THREADS, smem, stream, args);
  if (e != cudaSuccess) return e;
  int cc = C * C;
  const float* pc = part;
  void* rargs[] = {&pc, &out, &cc, &nchunk};
  return launch_pdl(reinterpret_cast<const void*>(k_wgrad_reduce), static_cast<unsigned>((cc + TR_THREADS - 1) / TR_THREADS),
                    TR_THREADS, 0, stream, rargs);
}

// dW = A^T B over the tokens, from the transposed operands at, bt [C, Tp]; part holds
// wgrad_chunks(Tp, sms) partial [C, C] fp32 planes.
cudaError_t wgrad(const void* at, const void* bt, float* part, float* out, long long Tp, int C, int sms,
                  unsigned int* err, cudaStream_t stream) {
  switch (C) {
    case 64: return wgrad_c<64>(at, bt, part, out, Tp, sms, err, stream);
    case 128: return wgrad_c<128>(at, bt, part, out, Tp, sms, err, stream);
    case 256: return wgrad_c<256>(at, bt, part, out, Tp, sms, err, stream);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace bbwd
}  // namespace whtmix
