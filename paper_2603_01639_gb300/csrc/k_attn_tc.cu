// Tensor-core (tcgen05) tree attention for bf16, head_dim 128.  Not enabled
// yet: every call routes to the CUDA-core kernel until this path is validated.
#include "ltd_common.cuh"
#include "ltd_internal.h"

namespace ltd {

bool attn_tc_supported(const AttnParams&, ltd_dtype) { return false; }

size_t attn_tc_workspace(int32_t, int32_t, int32_t, int32_t, int32_t, int32_t) { return 0; }

cudaError_t launch_attn_tc(const AttnParams&, cudaStream_t) { return cudaErrorNotSupported; }

int32_t attn_tc_launches() { return 1; }

}  // namespace ltd
