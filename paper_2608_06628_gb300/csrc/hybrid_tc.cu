// hybrid_tc.cu -- tensor-core (tcgen05) block-attention kernel.
#include "hybrid_common.cuh"
#include "hybrid_tc.h"

namespace hyb {

bool tc_attn_supported(const hybrid_cfg &) { return false; }

cudaError_t launch_attn_tc(const hybrid_cfg &, const void *, const void *, const void *, const void *,
                           const float *, void *const *, int, void *, unsigned *, cudaStream_t)
{
    return cudaErrorNotSupported;
}

}  // namespace hyb
