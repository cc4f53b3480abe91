// attn_mass.cu -- attention-accumulated vision score, eqs. (2)-(4).
#include "smoes_internal.cuh"

namespace smoes {

cudaError_t launch_attn_mass(const AttnParams&, const CUtensorMap&, const CUtensorMap&, int, cudaStream_t) {
  return cudaErrorNotSupported;
}

}  // namespace smoes
