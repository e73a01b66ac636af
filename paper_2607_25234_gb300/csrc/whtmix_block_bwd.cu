// whtmix_block_bwd.cu -- the pieces of the mixer block's backward (Section III-B, Eq. 1-4) that the
// forward kernels do not already provide: the weight gradients
//     dW[o, i] = sum over tokens t of A[t, o] B[t, i]      (dW_out = dY^T M, dW_in = dZ^T X)
// on the 5th-generation tensor cores, and the weight transposes the projections need.
//
// A and B are [T, C] bf16 token rows; the contraction runs over the tokens.  k_wgrad splits the
// tokens into one chunk per CTA (one persistent CTA per SM, 128 threads): per K tile of 64 tokens
// the CTA reads the token rows of both operands, transposes 8 x 8 blocks in registers and stages
// the A rows (output channels o, 128 per MMA tile) and the B rows (input channels i) in the tensor
// core's 128-byte-swizzled K-major layout, double-buffered, with the next tile's loads in flight;
// one thread issues tcgen05.mma (kind::f16, M = 128, N = C, K = 16) into a TMEM accumulator per
// 128 rows of o, committed to an mbarrier per buffer.  Each thread then reads its row o of the
// accumulator (tcgen05.ld) into the chunk's fp32 partial [C, C]; k_wgrad_reduce adds the partials
// in a fixed order, so dW is the same bit for bit on every run.
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

// out[c, t] = in[t, c] for t < T, 0 for T <= t < Tp (both bf16; C a multiple of 64, Tp of 64):
// the weights' transposes.
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
// tokens t of A[t][o] B[t][i], with A and B the [T, C] token rows as given.  C in {64, 128, 256}.
//
// A K tile of KT = 64 tokens of an operand becomes C rows (channels) of 128 bytes (64 tokens) in
// the tensor core's 128-byte-swizzled K-major layout: in each 1024-byte group of 8 rows, the
// 16-byte chunk j (tokens 8j .. 8j + 7) of row r sits at chunk position j ^ (r mod 8).  Thread
// work item (r8, k) reads the 8 x 8 block of channels 8 r8 .. + 7 and tokens 8 k .. + 7 as eight
// 16-byte token rows, transposes it in registers (byte permutes of token pairs) and writes the
// eight 16-byte channel rows; the eight items of a row group land in eight different bank groups.
template <int C>
__global__ void __launch_bounds__(WG_THREADS, 1) k_wgrad(const uint16_t* __restrict__ A, const uint16_t* __restrict__ B,
                                                         float* __restrict__ part, long long T, int nchunk,
                                                         unsigned int* err) {
  constexpr int MT = C > 128 ? C / 128 : 1;          // MMA tiles of 128 output rows
  constexpr int AR = MT * 128;                       // staged A rows (rows >= C stay zero)
  constexpr uint32_t A_BYTES = AR * KT * 2, B_BYTES = C * KT * 2, STAGE = A_BYTES + B_BYTES;
  constexpr uint32_t TCOLS = MT * C;                 // 64, 128 or 512 TMEM columns
  constexpr int ITEMS = C / WG_THREADS > 0 ? C / WG_THREADS : 1;  // 8 x 8 blocks per operand per thread
  static_assert(C == 64 || C == 128 || C == 256, "channels");
  extern __shared__ __align__(1024) unsigned char smem_raw[];
  __shared__ uint64_t mbar[2];
  __shared__ uint32_t tmem_slot;
  // the swizzle pattern is a function of the address: stage buffers start on 1024-byte boundaries
  unsigned char* smem = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);
  const int tid = threadIdx.x, warp = tid >> 5;
  if (tid < 32) tmem_alloc(&tmem_slot, TCOLS);
  if (tid == 0) {
    mbar_init(&mbar[0], 1);
    mbar_init(&mbar[1], 1);
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if constexpr (AR > C) {  // A rows C .. AR - 1 of both buffers: zero once, never written again
    for (int q = tid; q < 2 * (AR - C) * 8; q += WG_THREADS) {
      const int b = q / ((AR - C) * 8), rem = q % ((AR - C) * 8);
      *reinterpret_cast<uint4*>(smem + b * STAGE + C * 128 + rem * 16) = make_uint4(0u, 0u, 0u, 0u);
    }
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
  }
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
  __syncthreads();
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
  pdl_wait();
  const uint32_t tmem = tmem_slot;
  const long long ntiles = (T + KT - 1) / KT;
  const long long k0 = ntiles * blockIdx.x / nchunk, k1 = ntiles * (blockIdx.x + 1) / nchunk;
  const bool has_item = tid < C;  // C work items per operand and tile: C = 64 leaves threads 64 .. 127 idle

  // the 8 x 8 blocks of tile kt, item n of this thread: n-th work item tid + 128 n = 8 r8 + k
  uint4 ra[ITEMS][8], rb[ITEMS][8];
  auto load = [&](long long kt) {
#pragma unroll
    for (int n = 0; n < ITEMS; ++n) {
      const int item = tid + WG_THREADS * n, r8 = item >> 3, k = item & 7;
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        const long long t = kt * KT + 8 * k + j;
        const bool live = has_item && t < T;
        const long long off = (live ? t : 0) * C + 8 * r8;
        ra[n][j] = live ? __ldcs(reinterpret_cast<const uint4*>(A + off)) : make_uint4(0u, 0u, 0u, 0u);
        rb[n][j] = live ? __ldcs(reinterpret_cast<const uint4*>(B + off)) : make_uint4(0u, 0u, 0u, 0u);
      }
    }
  };
  // transpose one 8 x 8 block (v[j] = token j's 8 channels) and store its 8 channel rows
  auto put = [&](unsigned char* base, const uint4 (&v)[8], int r8, int k) {
    uint32_t o[8][4];
#pragma unroll
    for (int j = 0; j < 8; j += 2) {
      const uint32_t a[4] = {v[j].x, v[j].y, v[j].z, v[j].w}, b[4] = {v[j + 1].x, v[j + 1].y, v[j + 1].z, v[j + 1].w};
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        o[2 * q][j / 2] = __byte_perm(a[q], b[q], 0x5410);      // channel 2q, tokens j, j + 1
        o[2 * q + 1][j / 2] = __byte_perm(a[q], b[q], 0x7632);  // channel 2q + 1, tokens j, j + 1
      }
    }
#pragma unroll
    for (int c = 0; c < 8; ++c)
      *reinterpret_cast<uint4*>(base + (r8 * 8 + c) * 128 + ((k ^ c) << 4)) = make_uint4(o[c][0], o[c][1], o[c][2], o[c][3]);
  };
  auto store = [&](int buf) {
    unsigned char* sa = smem + buf * STAGE;
    unsigned char* sb = sa + A_BYTES;
    if (has_item) {
#pragma unroll
      for (int n = 0; n < ITEMS; ++n) {
        const int item = tid + WG_THREADS * n;
        put(sa, ra[n], item >> 3, item & 7);
        put(sb, rb[n], item >> 3, item & 7);
      }
    }
    // generic-proxy shared-memory writes -> visible to the tensor core (async proxy)
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
  };

  const uint32_t idesc = instr_desc(128, C);
  uint32_t parity[2] = {0u, 0u};
  bool ok = true;
  if (k1 > k0) load(k0);
  for (long long kt = k0; kt < k1; ++kt) {
    const int buf = static_cast<int>((kt - k0) & 1);
    if (kt - k0 >= 2) {  // buffer buf is free once the MMAs of tile kt - 2 (its last reader) completed
      ok = __syncthreads_and(mbar_wait(&mbar[buf], parity[buf]) ? 1 : 0) != 0;
      parity[buf] ^= 1u;
      if (!ok) break;
    }
    store(buf);
    if (kt + 1 < k1) load(kt + 1);  // in flight while this tile is handed to the tensor core
    __syncthreads();
    if (tid == 0) {
      asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
      const uint32_t sa = smem_u32(smem + buf * STAGE), sb = sa + A_BYTES;
#pragma unroll
      for (int mt = 0; mt < MT; ++mt)
#pragma unroll
        for (int ks = 0; ks < KT / 16; ++ks)  // K steps of 16 tokens: 32 bytes along the swizzled rows
          mma_bf16(tmem + mt * C, sw128_desc(sa + mt * (128 * 128) + ks * 32), sw128_desc(sb + ks * 32), idesc,
                   (kt > k0 || ks > 0) ? 1u : 0u);
      mma_commit(&mbar[buf]);
    }
  }
  if (ok && k1 > k0) {  // the last two tiles' commits cover every MMA issued
    const long long n = k1 - k0;
    for (long long kt = (n >= 2 ? k1 - 2 : k0); kt < k1 && ok; ++kt) {
      const int b = static_cast<int>((kt - k0) & 1);
      ok = __syncthreads_and(mbar_wait(&mbar[b], parity[b]) ? 1 : 0) != 0;
      parity[b] ^= 1u;
    }
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

// dW = the sum of the chunks' partials (float32) in a fixed order: RG runs of consecutive chunks,
// each summed in ascending order by one thread, then the RG run sums in ascending order.  A CTA
// covers 32 float4 outputs x RG runs.
constexpr int RG = TR_THREADS / 32;
__global__ void __launch_bounds__(TR_THREADS) k_wgrad_reduce(const float4* __restrict__ part, float4* __restrict__ out,
                                                             int cc4, int nchunk) {
  __shared__ float4 sums[RG][32];
  pdl_wait();
  const int o = blockIdx.x * 32 + (threadIdx.x & 31), g = threadIdx.x >> 5;
  const int c0 = nchunk * g / RG, c1 = nchunk * (g + 1) / RG;
  float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
  if (o < cc4) {
    int c = c0;
    for (; c + 4 <= c1; c += 4) {
      float4 v[4];
#pragma unroll
      for (int u = 0; u < 4; ++u) v[u] = __ldcs(part + static_cast<long long>(c + u) * cc4 + o);
#pragma unroll
      for (int u = 0; u < 4; ++u) acc = make_float4(acc.x + v[u].x, acc.y + v[u].y, acc.z + v[u].z, acc.w + v[u].w);
    }
    for (; c < c1; ++c) {
      const float4 v = __ldcs(part + static_cast<long long>(c) * cc4 + o);
      acc = make_float4(acc.x + v.x, acc.y + v.y, acc.z + v.z, acc.w + v.w);
    }
  }
  sums[g][threadIdx.x & 31] = acc;
  __syncthreads();
  if (g == 0 && o < cc4) {
    float4 s = sums[0][threadIdx.x];
#pragma unroll
    for (int r = 1; r < RG; ++r) {
      const float4 v = sums[r][threadIdx.x];
      s = make_float4(s.x + v.x, s.y + v.y, s.z + v.z, s.w + v.w);
    }
    out[o] = s;
  }
  pdl_trigger();
}

// ---- host ----

// Token chunks of one weight gradient over T tokens: one per SM, at most one per K tile.
int wgrad_chunks(long long T, int sms) {
  const long long nt = (T + KT - 1) / KT;
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
cudaError_t wgrad_c(const void* a_tok, const void* b_tok, float* part, float* out, long long T, int sms, unsigned int* err,
                    cudaStream_t stream) {
  constexpr int MT = C > 128 ? C / 128 : 1;
  constexpr size_t need = 2ull * (MT * 128 + C) * KT * 2 + 1024;  // two stages, 1024-byte alignment slack
  const size_t smem = need > SMEM_MIN ? need : SMEM_MIN;
  const void* k = reinterpret_cast<const void*>(k_wgrad<C>);
  cudaError_t e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
  if (e != cudaSuccess) return e;
  int nchunk = wgrad_chunks(T, sms);
  const uint16_t* a = static_cast<const uint16_t*>(a_tok);
  const uint16_t* b = static_cast<const uint16_t*>(b_tok);
  void* args[] = {&a, &b, &part, &T, &nchunk, &err};
  e = launch_pdl(k, static_cast<unsigned>(nchunk), WG_THREADS, smem, stream, args);
  if (e != cudaSuccess) return e;
  int cc4 = C * C / 4;
  const float4* pc = reinterpret_cast<const float4*>(part);
  float4* o4 = reinterpret_cast<float4*>(out);
  void* rargs[] = {&pc, &o4, &cc4, &nchunk};
  return launch_pdl(reinterpret_cast<const void*>(k_wgrad_reduce), static_cast<unsigned>((cc4 + 31) / 32), TR_THREADS, 0,
                    stream, rargs);
}

// dW = A^T B over the T tokens of the [T, C] bf16 operands a_tok, b_tok; part holds
// wgrad_chunks(T, sms) partial [C, C] fp32 planes; out is 16-byte aligned.
cudaError_t wgrad(const void* a_tok, const void* b_tok, float* part, float* out, long long T, int C, int sms,
                  unsigned int* err, cudaStream_t stream) {
  switch (C) {
    case 64: return wgrad_c<64>(a_tok, b_tok, part, out, T, sms, err, stream);
    case 128: return wgrad_c<128>(a_tok, b_tok, part, out, T, sms, err, stream);
    case 256: return wgrad_c<256>(a_tok, b_tok, part, out, T, sms, err, stream);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace bbwd
}  // namespace whtmix
