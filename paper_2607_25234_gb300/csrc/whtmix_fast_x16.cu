// Three-phase forward with a bf16 exchange workspace (whtmix_forward_x16), both I/O dtypes
// (instantiated in a translation unit of its own so the build compiles it in parallel).
#include "whtmix_fast_launch.cuh"

namespace whtmix {
namespace fast {
cudaError_t forward_x16_f32(const Params& P, int sms, cudaStream_t stream) {
  return launch_forward<DT_F32, false, WsB16>(P, sms, stream);
}
cudaError_t forward_x16_bf16(const Params& P, int sms, cudaStream_t stream) {
  return launch_forward<DT_BF16, false, WsB16>(P, sms, stream);
}
}  // namespace fast
}  // namespace whtmix
