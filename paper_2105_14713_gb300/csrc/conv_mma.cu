// Tensor-core (bf16) kernels of the 1xN-pruned convolution.  Not built yet:
// every request is reported as unsupported, so AUTO falls back to FFMA.
#include "conv_common.cuh"
#include "onexn_internal.h"

namespace onexn {

bool mma_supports(const ConvArgs &) { return false; }

cudaError_t launch_mma(const ConvArgs &, cudaStream_t) { return cudaErrorNotSupported; }

}  // namespace onexn
