// Fast forward and backward kernels, fp32 I/O (instantiated here so the build compiles dtypes in parallel).
#include "whtmix_fast_launch.cuh"

namespace whtmix {
namespace fast {
cudaError_t forward_f32(const Params& P, int sms, cudaStream_t stream) { return launch_forward<DT_F32, false>(P, sms, stream); }
cudaError_t backward_f32(const Params& P, int sms, cudaStream_t stream) { return launch_backward<DT_F32>(P, sms, stream); }
}  // namespace fast
}  // namespace whtmix
