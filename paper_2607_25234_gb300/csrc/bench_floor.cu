// bench_floor.cu -- memory-only model of the three-phase forward, for the bench's floor measurement.
//
// Not part of the mixer: a separate library (libwhtmix_floor.so) that bench.py --floor loads to
// measure how fast this GPU moves the data of the three-phase design (Section III-B map, one plane
// of 2^m elements, bf16 X / Y, fp32 G, fp32 exchange workspace) when no butterflies are computed:
//   phase 1  each CTA's rows of X (bf16)  -> fp32 workspace rows           (HBM read, L2 write)
//            with each CTA's share of G fetched into L2 during the phase, as the mixer does
//   phase 2  each CTA's columns: workspace and G read, workspace written   (L2 read, L2 write)
//   phase 3  each CTA's rows of the workspace -> Y (bf16)                  (L2 read, HBM write)
// with the same row and column ownership per CTA (rows of 2^13 elements, balanced ranges; column
// ranges balanced and aligned to 8), the same bounded device-wide barrier between phases, one
// persistent CTA of 256 threads per SM, and every access a coalesced 16-byte vector.  Each phase
// stamps the global timer per CTA so the host can split the time.  The values are carried through
// (widened, multiplied by G, narrowed) so that no access can be optimised away.
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "whtmix_kernels.cuh"

namespace {

using namespace whtmix;

constexpr int FT = 256;      // threads per CTA
constexpr int ROWB = 13;     // row bits
constexpr int ROWL = 1 << ROWB;

struct FloorArgs {
  const uint16_t* x;         // [2^m] bf16
  const float* g;            // [2^m]
  uint16_t* y;               // [2^m] bf16
  float* ws;                 // [2^m] fp32
  GridBarrier* bar;
  unsigned long long* stamps;  // [gridDim.x][4]: start, end of phase 1, 2, 3
  int m;
};

__device__ __forceinline__ void prefetch_l2(const void* p, unsigned bytes) {
  asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(p), "r"(bytes) : "memory");
}

__global__ void __launch_bounds__(FT, 1) k_floor_three_phase(FloorArgs A) {
  __shared__ int flag;
  pdl_wait();
  GridSync gsync(A.bar, &flag);
  const int m = A.m, q = m - ROWB;
  const long long rows = 1ll << q, cols = ROWL;
  const long long rb = rows * blockIdx.x / gridDim.x, re = rows * (blockIdx.x + 1) / gridDim.x;
  unsigned long long* st = A.stamps + 4ull * blockIdx.x;
  if (threadIdx.x == 0) {
    st[0] = global_ns();
    // this CTA's share of G into L2, in 8 pieces (the mixer spreads the same share over its rows)
    const long long gb = (4ll << m) / gridDim.x;
    for (int k = 0; k < 8; ++k) {
      const long long a0 = (gb * blockIdx.x + gb * k / 8) & ~15ll, a1 = (gb * blockIdx.x + gb * (k + 1) / 8) & ~15ll;
      if (a1 > a0) prefetch_l2(reinterpret_cast<const char*>(A.g) + a0, static_cast<unsigned>(a1 - a0));
    }
  }
  // Each phase loads a batch of UNR items per thread into registers before storing any of them,
  // so that UNR loads per thread are in flight (stores and loads could alias as far as the
  // compiler knows, which would otherwise serialise every item on its load).
  constexpr int UNR = 8;
  // phase 1: rows [rb, re) of X -> workspace, 8 bf16 (16 bytes) per item
  {
    const long long v0 = rb << (ROWB - 3), v1 = re << (ROWB - 3);
    const uint4* __restrict__ xs = reinterpret_cast<const uint4*>(A.x);
    float4* __restrict__ wd = reinterpret_cast<float4*>(A.ws);
    for (long long vb = v0 + threadIdx.x; vb < v1; vb += UNR * FT) {
      uint4 u[UNR];
#pragma unroll
      for (int j = 0; j < UNR; ++j) {
        const long long v = vb + j * FT;
        u[j] = v < v1 ? __ldcs(xs + v) : make_uint4(0u, 0u, 0u, 0u);
      }
#pragma unroll
      for (int j = 0; j < UNR; ++j) {
        const long long v = vb + j * FT;
        if (v >= v1) continue;
        const uint32_t w[4] = {u[j].x, u[j].y, u[j].z, u[j].w};
        float f[8];
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          f[2 * i] = __uint_as_float(w[i] << 16);
          f[2 * i + 1] = __uint_as_float(w[i] & 0xFFFF0000u);
        }
        __stcg(wd + 2 * v, make_float4(f[0], f[1], f[2], f[3]));
        __stcg(wd + 2 * v + 1, make_float4(f[4], f[5], f[6], f[7]));
      }
    }
  }
  if (threadIdx.x == 0) st[1] = global_ns();
  if (!gsync()) return;
  // phase 2: this CTA's columns (balanced, aligned to 8) of every row: ws * G -> ws, 4 per item
  {
    const long long cb = ((cols * blockIdx.x / gridDim.x) + 4) & ~7ll;
    const long long ce = blockIdx.x + 1 == gridDim.x ? cols : ((cols * (blockIdx.x + 1) / gridDim.x) + 4) & ~7ll;
    const long long nv = (ce - cb) / 4;  // float4 vectors per row in this CTA's range
    const long long items = nv * rows;
    for (long long ib = threadIdx.x; ib < items; ib += UNR * FT) {
      float4 a[UNR], gg[UNR];
      long long off[UNR];
#pragma unroll
      for (int j = 0; j < UNR; ++j) {
        const long long it = ib + j * FT;
        const long long r = it / nv;
        off[j] = (r << ROWB) + cb + 4 * (it - r * nv);
        if (it < items) {
          a[j] = __ldcg(reinterpret_cast<const float4*>(A.ws + off[j]));
          gg[j] = __ldg(reinterpret_cast<const float4*>(A.g + off[j]));
        }
      }
#pragma unroll
      for (int j = 0; j < UNR; ++j)
        if (ib + j * FT < items)
          __stcg(reinterpret_cast<float4*>(A.ws + off[j]),
                 make_float4(a[j].x * gg[j].x, a[j].y * gg[j].y, a[j].z * gg[j].z, a[j].w * gg[j].w));
    }
  }
  if (threadIdx.x == 0) st[2] = global_ns();
  if (!gsync()) return;
  // phase 3: rows [rb, re) of the workspace -> Y, 8 elements per item
  {
    const long long v0 = rb << (ROWB - 3), v1 = re << (ROWB - 3);
    const float4* __restrict__ ws = reinterpret_cast<const float4*>(A.ws);
    uint4* __restrict__ yd = reinterpret_cast<uint4*>(A.y);
    for (long long vb = v0 + threadIdx.x; vb < v1; vb += UNR * FT) {
      float4 a[UNR], b[UNR];
#pragma unroll
      for (int j = 0; j < UNR; ++j) {
        const long long v = vb + j * FT;
        if (v < v1) {
          a[j] = __ldcg(ws + 2 * v);
          b[j] = __ldcg(ws + 2 * v + 1);
        }
      }
#pragma unroll
      for (int j = 0; j < UNR; ++j) {
        const long long v = vb + j * FT;
        if (v >= v1) continue;
        const float f[8] = {a[j].x, a[j].y, a[j].z, a[j].w, b[j].x, b[j].y, b[j].z, b[j].w};
        uint32_t w[4];
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          __nv_bfloat162 h = __floats2bfloat162_rn(f[2 * i], f[2 * i + 1]);
          w[i] = *reinterpret_cast<uint32_t*>(&h);
        }
        __stcs(yd + v, make_uint4(w[0], w[1], w[2], w[3]));
      }
    }
  }
  if (threadIdx.x == 0) st[3] = global_ns();
  pdl_trigger();
}

}  // namespace

// Launches the floor kernel once on `stream` over one plane of 2^m elements (14 <= m <= 30), one
// CTA on each of `sms` SMs.
// workspace: 256-byte barrier header (zero before first use) followed by 4 * 2^m bytes;
// stamps: 4 * sms 64-bit words.  Returns a cudaError_t.
extern "C" __attribute__((visibility("default"))) int whtmix_floor_three_phase(
    const void* x, const void* g, void* y, void* workspace, void* stamps, int m, int sms, void* stream) {
  if (m < 14 || m > 30) return static_cast<int>(cudaErrorInvalidValue);
  FloorArgs a;
  a.x = static_cast<const uint16_t*>(x);
  a.g = static_cast<const float*>(g);
  a.y = static_cast<uint16_t*>(y);
  a.bar = static_cast<GridBarrier*>(workspace);
  a.ws = reinterpret_cast<float*>(static_cast<char*>(workspace) + sizeof(GridBarrier));
  a.stamps = static_cast<unsigned long long*>(stamps);
  a.m = m;
  // more than half an SM's shared memory (unused) so that one CTA runs per SM, as in the mixer
  constexpr int kSmem = 160 * 1024;
  const void* k = reinterpret_cast<const void*>(k_floor_three_phase);
  cudaError_t e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, kSmem);
  if (e != cudaSuccess) return static_cast<int>(e);
  void* args[] = {&a};
  return static_cast<int>(launch_pdl(k, static_cast<unsigned>(sms), FT, kSmem, static_cast<cudaStream_t>(stream), args));
}
