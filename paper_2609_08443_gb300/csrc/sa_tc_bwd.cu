// tcgen05 backward kernel (sm_103a).  Not yet enabled.
#include "sa_tc.cuh"

namespace sa {

bool tc_bwd_supported(int, int, sa_dtype) { return false; }
const char* tc_bwd_name(int, int) { return "tc_bwd"; }
int tc_bwd_workers(int num_sms, int, int) { return num_sms; }
cudaError_t launch_tc_bwd(const Args&, int, const float*, const float*, void*, void*, cudaStream_t) {
  return cudaErrorNotSupported;
}

}  // namespace sa
