// Tensor-core (tcgen05 / TMEM / TMA) passes for sm_103a.
#include "dblast_internal.cuh"

namespace dblast {

bool tc_supported(const dblast_head* h) {
  (void)h;
  return false;
}

cudaError_t launch_draft_pass_tc(const StepCtx& c) {
  (void)c;
  return cudaErrorNotSupported;
}

cudaError_t launch_verify_pass_tc(const StepCtx& c) {
  (void)c;
  return cudaErrorNotSupported;
}

}  // namespace dblast
