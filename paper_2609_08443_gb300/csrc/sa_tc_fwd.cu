// tcgen05 forward kernel (sm_103a).  Not yet enabled: every shape takes the
// CUDA-core path until this kernel passes its parity tests.
#include "sa_tc.cuh"

namespace sa {

bool tc_fwd_supported(int, int, sa_dtype) { return false; }
const char* tc_fwd_name(int, int) { return "tc_fwd"; }
int tc_tile_tokens() { return 128; }
int tc_fwd_workers(int num_sms, int, int) { return num_sms; }
cudaError_t launch_tc_fwd(const Args&, int, float*, float*, cudaStream_t) { return cudaErrorNotSupported; }

}  // namespace sa
