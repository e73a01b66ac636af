// Fast forward and backward kernels, bf16 I/O (instantiated here so the build compiles dtypes in parallel).
#include "whtmix_fast_launch.cuh"

namespace whtmix {
namespace fast {
cudaError_t forward_bf16(const Params& P, int sms, cudaStream_t stream) { return launch_forward<DT_BF16, false>(P, sms, stream); }
cudaError_t backward_bf16(const Params& P, int sms, cudaStream_t stream) { return launch_backward<DT_BF16>(P, sms, stream); }
}  // namespace fast
}  // namespace whtmix
