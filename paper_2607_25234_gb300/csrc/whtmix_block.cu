// Fused mixer block (Section III-B, Eq. 1-4) for bf16 planes of 128 channels and 2^21..2^23
// elements: one persistent launch (one CTA per SM, all resident; programmatic stream serialisation).
#include "whtmix_block.cuh"
#include "whtmix_fast_launch.cuh"

namespace whtmix {
namespace blk {

template <int Q>
cudaError_t launch(const Params& P, const void* w_in, const void* w_out, int sms, cudaStream_t stream) {
  const void* k = reinterpret_cast<const void*>(k_block_fast<Q>);
  int occ = 0;
  cudaError_t e = fast::occupancy_cached(k, SMEM_BYTES, &occ);
  if (e != cudaSuccess) return e;
  if (occ != 1) return cudaErrorInvalidConfiguration;  // all 512 TMEM columns per CTA: one CTA per SM
  Params p = P;
  const __nv_bfloat16* wi = static_cast<const __nv_bfloat16*>(w_in);
  const __nv_bfloat16* wo = static_cast<const __nv_bfloat16*>(w_out);
  void* args[] = {&p, &wi, &wo};
  return launch_pdl(k, static_cast<unsigned>(sms), THREADS, SMEM_BYTES, stream, args);
}

cudaError_t forward_bf16(const Params& P, const void* w_in, const void* w_out, int sms, cudaStream_t stream) {
  switch (P.m) {
    case 21: return launch<7>(P, w_in, w_out, sms, stream);
    case 22: return launch<8>(P, w_in, w_out, sms, stream);
    case 23: return launch<9>(P, w_in, w_out, sms, stream);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace blk
}  // namespace whtmix
