// Tree verification attention on the tcgen05 tensor cores.
// Not yet available: every call falls back to the CUDA-core kernel.
#include "kernels.h"

namespace glide {

cudaError_t launch_tree_attn_tc(const AttnArgs&, cudaStream_t) { return cudaErrorNotSupported; }

}  // namespace glide
