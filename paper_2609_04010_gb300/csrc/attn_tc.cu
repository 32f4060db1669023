// Part (a) of the verify step on tcgen05 tensor cores (not built yet in this file).
#include "attn_common.cuh"

namespace specv {

cudaError_t launch_attn_tc(const spec_attn_args_t&, const AttnPlan&, char*, cudaStream_t) {
  return cudaErrorNotSupported;
}

}  // namespace specv
