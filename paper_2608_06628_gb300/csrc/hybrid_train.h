// hybrid_train.h -- launchers of the training-form kernels (hybrid_train.cu).
#pragma once

#include <cuda_runtime.h>

#include "hybrid.h"

namespace hyb {

// bf16 I/O, d in {64, 128}, F in {64, 128}, B in {16, 32, 64}, G*B <= 128, B | seq_len.
bool train_supported(const hybrid_cfg &c, int seq_len);
size_t train_workspace_bytes(const hybrid_cfg &c, int n_seq, int seq_len);
// Device array (inside the workspace) of the n_seq * n_blk block states: entry
// s * n_blk + n points at S_{n-1}, z_{n-1} of sequence s in decode-image layout.
void *const *train_state_ptrs(const hybrid_cfg &c, int n_seq, int seq_len, void *workspace);
// The states of every block: the pointer array, dS per block, running sums.
cudaError_t launch_train_states(const hybrid_cfg &c, const void *K, const void *V, const void *W, int n_seq,
                                int seq_len, void *workspace, unsigned *err, cudaStream_t st);
cudaError_t launch_train_backward(const hybrid_cfg &c, const void *Q, const void *K, const void *V, const void *W,
                                  const float *alpha, const void *dO, int n_seq, int seq_len,
                                  void *workspace, float *dW, float *dalpha, unsigned *err, cudaStream_t st);

}  // namespace hyb
