// Chunked gated linear attention on tcgen05 tensor cores (not yet built).
#include "hs_internal.cuh"

namespace hs {

cudaError_t launch_gla_chunked_tc(const GlaParams &, int, cudaStream_t)
{
    return cudaErrorNotSupported;
}

}  // namespace hs
