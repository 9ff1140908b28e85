// hybrid_tc.h -- launchers of the tensor-core (tcgen05) kernels.
#pragma once

#include <cuda_runtime.h>

#include "hybrid.h"

namespace hyb {

// True when hybrid_block_attn for this cfg runs on the tcgen05 kernel.
bool tc_attn_supported(const hybrid_cfg &c);
cudaError_t launch_attn_tc(const hybrid_cfg &c, const void *Q, const void *K, const void *V,
                           const void *W, const float *alpha, void *const *states, int n_req,
                           void *O, unsigned *err, cudaStream_t st);

// True when hybrid_commit_block for this cfg runs on the tcgen05 kernel.
bool tc_commit_supported(const hybrid_cfg &c);
cudaError_t launch_commit_tc(const hybrid_cfg &c, const void *K, const void *V, int n_tok, const void *W,
                             void *const *states, int n_req, unsigned *err, cudaStream_t st);

}  // namespace hyb
