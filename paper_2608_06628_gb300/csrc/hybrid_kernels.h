// hybrid_kernels.h -- internal launchers (host side), one per kernel family.
#pragma once

#include <cuda_runtime.h>

#include "hybrid.h"

namespace hyb {

// CUDA-core kernels (hybrid_generic.cu)
cudaError_t launch_feature_map(hybrid_dtype dt, const void *X, int n_rows, int nh, int Hkv, int d,
                               int F, const void *W, float *Phi, cudaStream_t st);
cudaError_t launch_attn_generic(const hybrid_cfg &c, const void *Q, const void *K, const void *V,
                                const void *W, const float *alpha, void *const *states, int n_req,
                                void *O, unsigned *err, cudaStream_t st);
cudaError_t launch_commit_generic(const hybrid_cfg &c, const void *K, const void *V, int n_tok,
                                  const void *W, void *const *states, int n_req, unsigned *err,
                                  cudaStream_t st);

// state utilities (hybrid_state.cu)
cudaError_t launch_state_init(const hybrid_cfg &c, void *const *states, int n_req, cudaStream_t st);
cudaError_t launch_state_unpack(const hybrid_cfg &c, void *const *states, int n_req, float *S,
                                float *z, unsigned *err, cudaStream_t st);
cudaError_t launch_state_pack(const hybrid_cfg &c, const float *S, const float *z,
                              void *const *states, int n_req, unsigned *err, cudaStream_t st);

}  // namespace hyb
