// hybrid_tc.h -- launchers of the tensor-core (tcgen05) kernels.
#pragma once

#include <cuda_runtime.h>

#include <atomic>

#include "hybrid.h"

namespace hyb {

// Test hook (hybrid_debug_arm_wait_timeout): when nonzero, the next launch of the
// persistent step kernel takes it as its wait limit in nanoseconds and withholds
// one barrier arrival; the launch consumes it.
extern std::atomic<unsigned long long> g_armed_wait_ns;

// True when hybrid_block_attn for this cfg runs on the tcgen05 kernel.
bool tc_attn_supported(const hybrid_cfg &c);
cudaError_t launch_attn_tc(const hybrid_cfg &c, const void *Q, const void *K, const void *V,
                           const void *W, const float *alpha, void *const *states, int n_req,
                           void *O, unsigned *err, cudaStream_t st);

// Persistent step kernel, one unit at a time with both feature halves read out
// at once (hybrid_step.cu).
bool step_supported(const hybrid_cfg &c);
cudaError_t launch_step(const hybrid_cfg &c, const void *Q, const void *K, const void *V, const void *W,
                        const float *alpha, void *const *states, int n_req, void *O, unsigned *err,
                        cudaStream_t st);

// Persistent warp-specialised step fused with the block commit (hybrid_fused.cu):
// the readout uses the pre-commit state and the block's K/V are folded into the
// state in the same pass.
bool fused_supported(const hybrid_cfg &c);
cudaError_t launch_fused(const hybrid_cfg &c, const void *Q, const void *K, const void *V, const void *W,
                         const float *alpha, void *const *states, int n_req, void *O, unsigned *err,
                         cudaStream_t st);

// Commit / prefill as a reduction (hybrid_commit_red.cu): S += dS and z += dz are
// added into the state in global memory by bulk reduce-adds; any n_tok >= 1.
bool commit_red_supported(const hybrid_cfg &c);
// Commit / prefill with the key feature map computed token-major
// (hybrid_prefill.cu): 128-token chunks, ranges of chunks balanced across SMs,
// increments added by bulk reduce-adds; any n_tok >= 1.
bool prefill_supported(const hybrid_cfg &c);
cudaError_t launch_prefill(const hybrid_cfg &c, const void *K, const void *V, int n_tok, const void *W,
                           void *const *states, int n_req, unsigned *err, cudaStream_t st);
cudaError_t launch_commit_red(const hybrid_cfg &c, const void *K, const void *V, int n_tok, const void *W,
                              void *const *states, int n_req, unsigned *err, cudaStream_t st);

// Ragged prompts: request r folds tokens [tok[r], tok[r + 1]) of the packed K, V
// [tok[n_req]][Hkv][d]; tok is a host array read at launch (its values travel in
// the kernel parameters), so at most kMaxRaggedRequests requests per launch.
constexpr int kMaxRaggedRequests = 2048;
cudaError_t launch_prefill_ragged(const hybrid_cfg &c, const void *K, const void *V, const int *tok, const void *W,
                                  void *const *states, int n_req, unsigned *err, cudaStream_t st);
cudaError_t launch_commit_red_ragged(const hybrid_cfg &c, const void *K, const void *V, const int *tok,
                                     const void *W, void *const *states, int n_req, unsigned *err, cudaStream_t st);

}  // namespace hyb
