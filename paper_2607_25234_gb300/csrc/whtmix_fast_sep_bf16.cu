// Fast forward kernels with separable log gains, bf16 I/O (a translation unit of its own so the
// build compiles the variants in parallel).
#include "whtmix_fast_launch.cuh"

namespace whtmix {
namespace fast {
cudaError_t forward_sep_bf16(const Params& P, int sms, cudaStream_t stream) { return launch_forward<DT_BF16, true>(P, sms, stream); }
}  // namespace fast
}  // namespace whtmix
