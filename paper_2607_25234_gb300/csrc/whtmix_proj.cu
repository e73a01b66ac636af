// whtmix_proj.cu -- token-wise channel projection on the 5th-generation tensor cores:
//   Z[t, :] = X[t, :] W^T        X [T, C] bf16, W [C, C] bf16 (out, in), Z [T, C] bf16 or fp32
// the W_in and W_out projections around the mixer (Section III-B, Eq. 1 and Eq. 4).
//
// One persistent CTA per SM (the shared-memory request leaves room for one), 128 threads: tiles
// of 128 tokens.  W is staged in shared memory once per CTA; each tile of X is staged next to it;
// one thread issues C/16 tcgen05.mma (kind::f16, bf16 x bf16 -> fp32, M = 128, N = C, K = 16) with
// the accumulator in TMEM (lane = token of the tile, column = output channel) and commits them to
// an mbarrier; every thread then reads its token's row of the accumulator with tcgen05.ld and
// stores it.  Both operands are K-major (X rows are tokens with their channels contiguous, W rows
// are output channels with their input channels contiguous), laid out in shared memory as the
// tensor core's no-swizzle canonical form: 8-row x 16-byte core matrices, the K-adjacent core
// matrix 128 bytes on, the next group of 8 rows (C / 8) x 128 bytes on.  bf16 output at C = 64 and
// 128 takes the pipelined, warp-specialised k_proj_pipe below instead (TMA in and out).
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "whtmix_kernels.cuh"
#include "whtmix_tc.cuh"

namespace whtmix {
namespace proj {

constexpr int THREADS = 128;   // one thread per TMEM lane = per token of a tile
constexpr int TILE_T = 128;    // tokens per tile (the MMA's M)
constexpr size_t SMEM_MIN = 120 * 1024;  // more than half an SM: one CTA per SM, so TMEM allocation never waits

using namespace tc;

// C in {64, 128, 256}; OUT_F32: fp32 output (else bf16, round to nearest even).
template <int C, bool OUT_F32>
__global__ void __launch_bounds__(THREADS, 1) k_proj(const __nv_bfloat16* x, const __nv_bfloat16* __restrict__ w,
                                                     void* z, long long T, unsigned int* err) {  // z may be x
  static_assert(C == 64 || C == 128 || C == 256, "channels");
  extern __shared__ __align__(1024) unsigned char smem[];
  __shared__ uint64_t mbar;
  __shared__ uint32_t tmem_slot;
  unsigned char* sw = smem;                     // W: C x C bf16, canonical layout
  unsigned char* sx = smem + C * C * 2;         // X tile: 128 x C bf16, canonical layout
  const int tid = threadIdx.x;
  // W once per CTA
  for (int i = tid; i < C * C / 8; i += THREADS) {
    const int r = i / (C / 8), k = (i % (C / 8)) * 8;
    *reinterpret_cast<uint4*>(sw + core_off(r, k, C)) = *reinterpret_cast<const uint4*>(w + static_cast<long long>(r) * C + k);
  }
  if (tid < 32) tmem_alloc(&tmem_slot, C);
  if (tid == 0) {
    mbar_init(&mbar, 1);
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
  __syncthreads();
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
  const uint32_t tmem = tmem_slot;
  const uint32_t idesc = instr_desc(TILE_T, C);
  const uint32_t lane_base = static_cast<uint32_t>(32 * (tid >> 5)) << 16;
  const long long ntiles = (T + TILE_T - 1) / TILE_T;
  uint32_t parity = 0;
  bool ok = true;
  for (long long tile = blockIdx.x; tile < ntiles && ok; tile += gridDim.x) {
    const long long t0 = tile * TILE_T;
    // X tile; tokens past T are zero
    for (int i = tid; i < TILE_T * C / 8; i += THREADS) {
      const int r = i / (C / 8), k = (i % (C / 8)) * 8;
      uint4 v = make_uint4(0u, 0u, 0u, 0u);
      if (t0 + r < T) v = *reinterpret_cast<const uint4*>(x + (t0 + r) * C + k);
      *reinterpret_cast<uint4*>(sx + core_off(r, k, C)) = v;
    }
    // generic-proxy shared-memory writes -> visible to the tensor core (async proxy)
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
    __syncthreads();
    if (tid == 0) {
      asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
      const uint32_t ax = smem_u32(sx), aw = smem_u32(sw);
#pragma unroll
      for (int ks = 0; ks < C / 16; ++ks)  // K steps of 16: two core matrices along K
        mma_bf16(tmem, smem_desc(ax + ks * 256, 128, (C / 8) * 128), smem_desc(aw + ks * 256, 128, (C / 8) * 128), idesc,
                 ks > 0 ? 1u : 0u);
      mma_commit(&mbar);
    }
    // every thread waits; the CTA goes on only if all saw the MMAs complete (a uniform decision,
    // so that no thread is left at a later barrier)
    ok = __syncthreads_and(mbar_wait(&mbar, parity) ? 1 : 0) != 0;
    if (!ok) {
      if (tid == 0) atomicOr(err, 1u);
      break;
    }
    parity ^= 1u;
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
    // row tid of the tile: C accumulator columns of TMEM lane tid
    const long long t = t0 + tid;
#pragma unroll
    for (int c0 = 0; c0 < C; c0 += 16) {
      float v[16];
      tmem_ld16(tmem + lane_base + c0, v);
      asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
      if (t < T) {
        if constexpr (OUT_F32) {
          float4* o = reinterpret_cast<float4*>(static_cast<float*>(z) + t * C + c0);
#pragma unroll
          for (int q = 0; q < 4; ++q) o[q] = make_float4(v[4 * q], v[4 * q + 1], v[4 * q + 2], v[4 * q + 3]);
        } else {
          uint32_t h[8];
#pragma unroll
          for (int q = 0; q < 8; ++q) {
            __nv_bfloat162 b = __floats2bfloat162_rn(v[2 * q], v[2 * q + 1]);
            h[q] = *reinterpret_cast<uint32_t*>(&b);
          }
          uint4* o = reinterpret_cast<uint4*>(static_cast<__nv_bfloat16*>(z) + t * C + c0);
          o[0] = make_uint4(h[0], h[1], h[2], h[3]);
          o[1] = make_uint4(h[4], h[5], h[6], h[7]);
        }
      }
    }
    // every thread's TMEM reads are done before the next tile's MMAs overwrite the accumulator,
    // and the MMAs (complete, per the mbarrier) no longer read the X tile
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
    __syncthreads();
  }
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
  if (tid < 32) tmem_dealloc(tmem, C);
}

// ---------------------------------------------------------------------------------------------
// Pipelined projection for C = 64, 128 with bf16 output: tiles of 128 tokens stream through TMA
// (128-byte swizzled boxes of 64 channels = the tensor core's K-major canonical layout), two
// slots per stage, with fixed warp roles handing tiles on through mbarriers:
//   warp 0  TMA producer of X tiles;  warp 1  MMA issuer (C / 16 MMAs per tile into TMEM slot s);
//   warps 2-5  epilogue: TMEM row -> bf16 -> swizzled staging -> TMA tensor store.
// Tokens past T are zero-filled by the loads and dropped by the stores (the tensor maps' bounds).
constexpr int P2_THREADS = 192;

// K step ks (16 bf16) of an R-row K-major operand stored as 64-element atoms of R x 128 bytes
template <int R>
__device__ __forceinline__ uint64_t sw_op_desc(uint32_t base, int ks) {
  return sw128_desc(base + (ks >> 2) * (R * 128) + (ks & 3) * 32);
}
__device__ __forceinline__ void mbar_arrive(uint64_t* b) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(b)) : "memory");
}
__device__ __forceinline__ void mbar_expect_tx(uint64_t* b, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(b)), "r"(bytes) : "memory");
}
__device__ __forceinline__ void tma_load_2d(void* sdst, const CUtensorMap* tm, int x, int y, uint64_t* bar) {
  asm volatile("cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3}], [%4];"
               ::"r"(smem_u32(sdst)), "l"(tm), "r"(x), "r"(y), "r"(smem_u32(bar)) : "memory");
}
__device__ __forceinline__ void tma_store_2d(const CUtensorMap* tm, int x, int y, const void* ssrc) {
  asm volatile("cp.async.bulk.tensor.2d.global.shared::cta.bulk_group [%0, {%1, %2}], [%3];"
               ::"l"(tm), "r"(x), "r"(y), "r"(smem_u32(ssrc)) : "memory");
}

struct ProjBars {
  uint64_t wfull, xfull[2], xempty[2], dfull[2], dempty[2], sfree[2];
};

template <int C>
__global__ void __launch_bounds__(P2_THREADS, 1) k_proj_pipe(const __grid_constant__ CUtensorMap tmx,
                                                             const __grid_constant__ CUtensorMap tmw,
                                                             const __grid_constant__ CUtensorMap tmz, long long ntiles,
                                                             unsigned int* err) {
  static_assert(C == 64 || C == 128, "channels");
  constexpr int A = C / 64;                     // 64-channel atoms per row
  constexpr uint32_t TILE_BYTES = 128 * C * 2;  // one 128-token tile, bf16
  constexpr uint32_t IDESC = (1u << 4) | (1u << 7) | (1u << 10) | ((C >> 3) << 17) | ((128u >> 4) << 24);
  extern __shared__ __align__(1024) unsigned char smem[];
  __shared__ ProjBars bars;
  __shared__ uint32_t tmem_slot;
  unsigned char* sW = smem;                                        // C x C
  unsigned char* sX[2] = {smem + C * C * 2, smem + C * C * 2 + TILE_BYTES};
  unsigned char* sS[2] = {smem + C * C * 2 + 2 * TILE_BYTES, smem + C * C * 2 + 3 * TILE_BYTES};
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  if (warp == 0) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(&tmem_slot)), "r"(2 * C)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  if (tid == 32) {
    mbar_init(&bars.wfull, 1);
    for (int s = 0; s < 2; ++s) {
      mbar_init(&bars.xfull[s], 1);
      mbar_init(&bars.xempty[s], 1);
      mbar_init(&bars.dfull[s], 1);
      mbar_init(&bars.dempty[s], 4);
      mbar_init(&bars.sfree[s], 1);
    }
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
  __syncthreads();
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
  const uint32_t tmem = tmem_slot;
  const long long first = blockIdx.x, step = gridDim.x;
  const long long mine = first < ntiles ? (ntiles - first + step - 1) / step : 0;
  unsigned bad = 0;
  if (warp == 0) {
    if (lane == 0) {
      mbar_expect_tx(&bars.wfull, C * C * 2);
#pragma unroll
      for (int a = 0; a < A; ++a) tma_load_2d(sW + a * C * 128, &tmw, 64 * a, 0, &bars.wfull);
      for (long long i = 0; i < mine; ++i) {
        const int s = static_cast<int>(i & 1);
        const uint32_t u = static_cast<uint32_t>(i >> 1);
        if (!mbar_wait(&bars.xempty[s], (u & 1) ^ 1)) {
          bad |= 1;
          break;
        }
        mbar_expect_tx(&bars.xfull[s], TILE_BYTES);
        const int y = static_cast<int>((first + i * step) * TILE_T);
#pragma unroll
        for (int a = 0; a < A; ++a) tma_load_2d(sX[s] + a * 16384, &tmx, 64 * a, y, &bars.xfull[s]);
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      if (!mbar_wait(&bars.wfull, 0)) bad |= 2;
      const uint32_t aw = smem_u32(sW);
      for (long long i = 0; i < mine && !bad; ++i) {
        const int s = static_cast<int>(i & 1);
        const uint32_t u = static_cast<uint32_t>(i >> 1);
        if (!mbar_wait(&bars.xfull[s], u & 1) || !mbar_wait(&bars.dempty[s], (u & 1) ^ 1)) {
          bad |= 4;
          break;
        }
        asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
        const uint32_t ax = smem_u32(sX[s]);
#pragma unroll
        for (int ks = 0; ks < C / 16; ++ks)
          mma_bf16(tmem + static_cast<uint32_t>(C * s), sw_op_desc<128>(ax, ks), sw_op_desc<C>(aw, ks), IDESC, ks > 0 ? 1u : 0u);
        mma_commit(&bars.dfull[s]);
        mma_commit(&bars.xempty[s]);
      }
    }
  } else {
    // epilogue: thread = TMEM lane = token of the tile; staged as A boxes of 128 rows x 64 bf16
    const int row = 32 * (warp & 3) + lane;
    const uint32_t lane_base = static_cast<uint32_t>(32 * (warp & 3)) << 16;
    for (long long i = 0; i < mine; ++i) {
      const int s = static_cast<int>(i & 1);
      const uint32_t u = static_cast<uint32_t>(i >> 1);
      const bool ok = __all_sync(0xffffffffu, mbar_wait(&bars.dfull[s], u & 1)) &&
                      __all_sync(0xffffffffu, mbar_wait(&bars.sfree[s], (u & 1) ^ 1));
      if (!ok) bad |= 8;
      if (ok) {
        asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
        float v[C];
#pragma unroll
        for (int c = 0; c < C; c += 16) {
          float t[16];
          tmem_ld16(tmem + lane_base + static_cast<uint32_t>(C * s + c), t);
#pragma unroll
          for (int j = 0; j < 16; ++j) v[c + j] = t[j];
        }
        asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
        asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
        __syncwarp();
        if (lane == 0) mbar_arrive(&bars.dempty[s]);
#pragma unroll
        for (int q = 0; q < C / 8; ++q) {  // 16-byte chunk q = channels 8q .. 8q + 7
          uint32_t h[4];
#pragma unroll
          for (int j = 0; j < 4; ++j) {
            __nv_bfloat162 b = __floats2bfloat162_rn(v[8 * q + 2 * j], v[8 * q + 2 * j + 1]);
            h[j] = *reinterpret_cast<uint32_t*>(&b);
          }
          *reinterpret_cast<uint4*>(sS[s] + (q >> 3) * 16384 + row * 128 + (((q & 7) ^ (row & 7)) << 4)) =
              make_uint4(h[0], h[1], h[2], h[3]);
        }
        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
      }
      asm volatile("bar.sync 1, 128;" ::: "memory");
      if (ok && warp == 2 && lane == 0) {
        const int y = static_cast<int>((first + i * step) * TILE_T);
#pragma unroll
        for (int a = 0; a < A; ++a) tma_store_2d(&tmz, 64 * a, y, sS[s] + a * 16384);
        asm volatile("cp.async.bulk.commit_group;" ::: "memory");
        asm volatile("cp.async.bulk.wait_group.read 0;" ::: "memory");
        mbar_arrive(&bars.sfree[s]);
      }
    }
    if (warp == 2 && lane == 0) asm volatile("cp.async.bulk.wait_group 0;" ::: "memory");
  }
  if (bad) atomicOr(err, bad << 8);
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
  __syncthreads();
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
  if (warp == 0) asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(2 * C) : "memory");
}

// cuTensorMapEncodeTiled through the runtime's driver entry point (no link against libcuda).
typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                  const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                  CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);
static EncodeTiledFn encode_fn() {
  static EncodeTiledFn fn = nullptr;
  static bool tried = false;
  if (!tried) {
    tried = true;
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFn>(p);
  }
  return fn;
}
// bf16 [rows, C] row-major, boxes of box_rows rows x 64 channels, 128-byte swizzle.
static bool encode_bf16_rows(CUtensorMap* tm, const void* base, long long rows, int C, int box_rows) {
  EncodeTiledFn f = encode_fn();
  if (!f) return false;
  const cuuint64_t dims[2] = {static_cast<cuuint64_t>(C), static_cast<cuuint64_t>(rows)};
  const cuuint64_t strides[1] = {static_cast<cuuint64_t>(C) * 2};
  const cuuint32_t box[2] = {64, static_cast<cuuint32_t>(box_rows)};
  const cuuint32_t es[2] = {1, 1};
  return f(tm, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box, es,
           CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_128B,
           CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

template <int C>
cudaError_t launch_pipe(const void* x, const void* w, void* z, long long T, unsigned int* err, int sms, cudaStream_t s) {
  CUtensorMap tmx, tmw, tmz;
  if (!encode_bf16_rows(&tmx, x, T, C, TILE_T) || !encode_bf16_rows(&tmw, w, C, C, C) ||
      !encode_bf16_rows(&tmz, z, T, C, TILE_T))
    return cudaErrorInvalidValue;
  const size_t smem = static_cast<size_t>(C) * C * 2 + 4 * static_cast<size_t>(TILE_T) * C * 2;
  cudaError_t e = cudaFuncSetAttribute(k_proj_pipe<C>, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
  if (e != cudaSuccess) return e;
  const long long ntiles = (T + TILE_T - 1) / TILE_T;
  const unsigned grid = static_cast<unsigned>(ntiles < sms ? ntiles : sms);
  k_proj_pipe<C><<<grid, P2_THREADS, smem, s>>>(tmx, tmw, tmz, ntiles, err);
  return cudaGetLastError();
}

template <int C, bool OUT_F32>
cudaError_t launch_c(const void* x, const void* w, void* z, long long T, unsigned int* err, int sms, cudaStream_t s) {
  const size_t need = static_cast<size_t>(C) * C * 2 + static_cast<size_t>(TILE_T) * C * 2;
  const size_t smem = need > SMEM_MIN ? need : SMEM_MIN;
  auto k = k_proj<C, OUT_F32>;
  cudaError_t e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
  if (e != cudaSuccess) return e;
  const long long ntiles = (T + TILE_T - 1) / TILE_T;
  const unsigned grid = static_cast<unsigned>(ntiles < sms ? ntiles : sms);
  k<<<grid, THREADS, smem, s>>>(static_cast<const __nv_bfloat16*>(x), static_cast<const __nv_bfloat16*>(w), z, T, err);
  return cudaGetLastError();
}

// Z = X W^T for T tokens of C channels (C = 64, 128 or 256); err: device word set on a timeout.
cudaError_t project(const void* x, const void* w, void* z, long long T, int C, bool out_f32, unsigned int* err, int sms,
                    cudaStream_t s) {
  if (T <= 0) return cudaSuccess;
  // bf16 output at C = 64, 128: the pipelined kernel (its TMA tensor maps need 16-byte aligned bases)
  const bool aligned = ((reinterpret_cast<uintptr_t>(x) | reinterpret_cast<uintptr_t>(w) | reinterpret_cast<uintptr_t>(z)) & 15u) == 0;
  if (!out_f32 && aligned && C == 64) return launch_pipe<64>(x, w, z, T, err, sms, s);
  if (!out_f32 && aligned && C == 128) return launch_pipe<128>(x, w, z, T, err, sms, s);
  switch (C) {
    case 64: return out_f32 ? launch_c<64, true>(x, w, z, T, err, sms, s) : launch_c<64, false>(x, w, z, T, err, sms, s);
    case 128: return out_f32 ? launch_c<128, true>(x, w, z, T, err, sms, s) : launch_c<128, false>(x, w, z, T, err, sms, s);
    case 256: return out_f32 ? launch_c<256, true>(x, w, z, T, err, sms, s) : launch_c<256, false>(x, w, z, T, err, sms, s);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace proj
}  // namespace whtmix
