// Fast forward kernels with separable log gains, fp32 I/O (a translation unit of its own so the
// build compiles the variants in parallel).
#include "whtmix_fast_launch.cuh"

namespace whtmix {
namespace fast {
cudaError_t forward_sep_f32(const Params& P, int sms, cudaStream_t stream) { return launch_forward<DT_F32, true>(P, sms, stream); }
}  // namespace fast
}  // namespace whtmix
