// whtmix_fast_launch.cuh -- host-side launcher of the fast forward and backward kernels for one I/O dtype.
// Included by whtmix_fast_f32.cu and whtmix_fast_bf16.cu (one translation unit each, compiled in
// parallel).  Returns a cudaError_t; the C ABI maps it to a status.
#pragma once

#include <cuda_runtime.h>

#include <map>
#include <mutex>

#include "whtmix_fast.cuh"
#include "whtmix_fast_bwd.cuh"

namespace whtmix {
namespace fast {

// Resident CTAs per SM for one kernel and smem size, per device (first query also raises the
// kernel's dynamic shared memory limit).
inline cudaError_t occupancy_cached(const void* kernel, size_t smem, int* occ) {
  static std::mutex mu;
  static std::map<std::pair<int, const void*>, int> cache;
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  std::lock_guard<std::mutex> lk(mu);
  auto it = cache.find({dev, kernel});
  if (it != cache.end()) {
    *occ = it->second;
    return cudaSuccess;
  }
  e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
  if (e != cudaSuccess) return e;
  e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(occ, kernel, THREADS, smem);
  if (e != cudaSuccess) return e;
  if (*occ < 1) return cudaErrorInvalidConfiguration;
  cache[{dev, kernel}] = *occ;
  return cudaSuccess;
}

// Every variant requests more than half an SM's shared memory, so exactly one CTA runs per SM:
// two CTAs on one SM would both ask for all 512 TMEM columns, and the second would wait in
// tcgen05.alloc while the first waits for it at the device-wide barrier.  The grid is one CTA per
// SM, all resident at once; it is launched with programmatic stream serialisation (launch_pdl),
// which lets its launch and tensor-memory allocation overlap the previous kernel's tail.
inline cudaError_t launch_persistent(const void* k, const Params& P, int sms, cudaStream_t stream) {
  const size_t smem = SMEM_BYTES;
  int occ = 0;
  cudaError_t e = occupancy_cached(k, smem, &occ);
  if (e != cudaSuccess) return e;
  if (occ != 1) return cudaErrorInvalidConfiguration;
  Params p = P;
  void* args[] = {&p};
  return launch_pdl(k, static_cast<unsigned>(sms), THREADS, smem, stream, args);
}
template <int D, int R, int Q, bool SEP, class WS = WsF32>
cudaError_t launch_one(const Params& P, int sms, cudaStream_t stream) {
  return launch_persistent(reinterpret_cast<const void*>(k_forward_fast<D, R, Q, SEP, WS>), P, sms, stream);
}
template <int D, int R, int Q>
cudaError_t launch_bwd_one(const Params& P, int sms, cudaStream_t stream) {
  return launch_persistent(reinterpret_cast<const void*>(k_backward_fast<D, R, Q>), P, sms, stream);
}

// Rows of 2^13 elements at every size but 2^21; 2^23-element planes take 1024-row columns (two
// lanes per column).  With 152 SMs, 1024 rows of 2^13 spread as 7 or 6 per CTA, where 512 rows of
// 2^14 give 56 CTAs four rows against three; measured on the 2^22 planes, 2^13 rows with 512-row
// columns beat 2^14 rows.  2^21-element planes take rows of 2^14 and 128-row columns, one column
// per thread in registers, instead of 256-row columns in tensor memory: measured on sixteen such
// planes (bf16), 138 us against 146 us per call.
// SEP: separable log gains (P.gt, P.gc) instead of G; needs 1 <= P.cbits <= row bits.
// WS: the workspace element (WsB16: whtmix_forward_x16).
template <int D, bool SEP, class WS = WsF32>
cudaError_t launch_forward(const Params& P, int sms, cudaStream_t stream) {
  switch (P.m) {
    case 14: return launch_one<D, 13, 1, SEP, WS>(P, sms, stream);
    case 15: return launch_one<D, 13, 2, SEP, WS>(P, sms, stream);
    case 16: return launch_one<D, 13, 3, SEP, WS>(P, sms, stream);
    case 17: return launch_one<D, 13, 4, SEP, WS>(P, sms, stream);
    case 18: return launch_one<D, 13, 5, SEP, WS>(P, sms, stream);
    case 19: return launch_one<D, 13, 6, SEP, WS>(P, sms, stream);
    case 20: return launch_one<D, 13, 7, SEP, WS>(P, sms, stream);
    case 21: return launch_one<D, 14, 7, SEP, WS>(P, sms, stream);
    case 22: return launch_one<D, 13, 9, SEP, WS>(P, sms, stream);
    case 23: return launch_one<D, 13, 10, SEP, WS>(P, sms, stream);
    default: return cudaErrorInvalidValue;
  }
}
// Row bits of the fast forward for a 2^m-element plane.
inline int forward_row_bits(int m) { return m == 21 ? 14 : 13; }

// Backward: rows of 2^13 up to 2^20-element planes (columns of at most 128 rows, the transformed X
// column of a 128-row column parked in TMEM) and rows of 2^14 from 2^21 (columns of 128, 256 and
// 512 rows; the TMEM column pass for 256 and 512).
template <int D>
cudaError_t launch_backward(const Params& P, int sms, cudaStream_t stream) {
  switch (P.m) {
    case 14: return launch_bwd_one<D, 13, 1>(P, sms, stream);
    case 15: return launch_bwd_one<D, 13, 2>(P, sms, stream);
    case 16: return launch_bwd_one<D, 13, 3>(P, sms, stream);
    case 17: return launch_bwd_one<D, 13, 4>(P, sms, stream);
    case 18: return launch_bwd_one<D, 13, 5>(P, sms, stream);
    case 19: return launch_bwd_one<D, 13, 6>(P, sms, stream);
    case 20: return launch_bwd_one<D, 13, 7>(P, sms, stream);
    case 21: return launch_bwd_one<D, 14, 7>(P, sms, stream);
    case 22: return launch_bwd_one<D, 14, 8>(P, sms, stream);
    case 23: return launch_bwd_one<D, 14, 9>(P, sms, stream);
    default: return cudaErrorInvalidValue;
  }
}

// Entry points defined in whtmix_fast_f32.cu / whtmix_fast_bf16.cu.
cudaError_t forward_f32(const Params& P, int sms, cudaStream_t stream);
cudaError_t forward_bf16(const Params& P, int sms, cudaStream_t stream);
cudaError_t backward_f32(const Params& P, int sms, cudaStream_t stream);
cudaError_t backward_bf16(const Params& P, int sms, cudaStream_t stream);
// whtmix_fast_x16.cu: the forward with a bf16 exchange workspace
cudaError_t forward_x16_f32(const Params& P, int sms, cudaStream_t stream);
cudaError_t forward_x16_bf16(const Params& P, int sms, cudaStream_t stream);
// whtmix_fast_sep_f32.cu / whtmix_fast_sep_bf16.cu
cudaError_t forward_sep_f32(const Params& P, int sms, cudaStream_t stream);
cudaError_t forward_sep_bf16(const Params& P, int sms, cudaStream_t stream);

}  // namespace fast
}  // namespace whtmix
