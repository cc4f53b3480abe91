// router_fwd_var.cu -- the tensor-core router forward with the router variants compiled in
// (sigmoid gate with a selection bias, top-k-masked bin sums of eq. (12)); the kernel and its
// epilogue are in router_fwd_tc.cuh.
#include "router_fwd_tc.cuh"

namespace smoes {

cudaError_t launch_router_fwd_bf16_var(const FwdParams& p, const CUtensorMap& tmX,
                                       const CUtensorMap& tmW, const CUtensorMap* tmG, int n_sms,
                                       cudaStream_t s) {
  return launch_fwd_tc<true>(p, tmX, tmW, tmG, n_sms, s);
}

}  // namespace smoes
