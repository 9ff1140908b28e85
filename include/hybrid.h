/*
 * hybrid.h -- C ABI of the block-hybrid attention library (sm_103a).
 *
 * Block-hybrid attention ("Retrofitting Linear Attention into Diffusion
 * Language Models", Section 3.1): during blockwise semi-autoregressive
 * decoding, each query of the active block of B tokens attends
 *   (1) to every token of its own block with exact, unmasked softmax
 *       (a_j = exp(q.k_j / sqrt(d)); sm_num = sum_j a_j v_j; sm_den = sum_j a_j), and
 *   (2) to all committed blocks through a fixed-size linear-attention state
 *       S = sum_t phi(k_t) v_t^T in R^{2F x d} and z = sum_t phi(k_t) in R^{2F}
 *       (lin_num = phi(q)^T S, lin_den = phi(q)^T z),
 * merged through a shared normaliser with the gate w = sigmoid(alpha):
 *       out = (w sm_num + lin_num) / (w sm_den + lin_den).
 * The feature map is Hedgehog's: phi(x) = [softmax(xW), softmax(-xW)],
 * W in R^{d x F}.  When a block commits, its tokens are folded into (S, z).
 *
 * Conventions shared by every entry point
 * ---------------------------------------
 * Notation: n = n_req requests, B = block size, Hq query heads, Hkv state
 * (key/value) heads, G = Hq / Hkv, d = head_dim, F = feat_dim (phi has 2F
 * entries).
 *
 * Ownership: the caller allocates every buffer (inputs, outputs, states and
 * the device array of state pointers).  The library allocates no memory in
 * any call.  Its own static device memory, per device, is one 4-byte error word
 * (read back by hybrid_check()) and the HYBRID_LOGICAL_SCRATCH_BYTES scratch
 * array used only by hybrid_block_attn_commit_logical().
 *
 * Pointers: every tensor argument is a DEVICE pointer unless stated.  Tensor
 * pointers must be 16-byte aligned (alpha: 4-byte).  d_state_ptrs is a device
 * array of n_req device pointers, one per request, each to a state buffer of
 * hybrid_state_bytes(cfg) bytes, 16-byte aligned.  A batch may name any
 * subset of live requests in any order (ragged concurrent batches); the same
 * state must not appear twice in one commit call.
 *
 * Streams: every call is asynchronous and ordered on the given stream
 * (a cudaStream_t; 0 is the legacy default stream).  The calling thread's
 * current device must own all pointers.
 *
 * Layouts (row-major, innermost last):
 *   Q, O        [n][B][Hq][d]     io_dtype
 *   K, V        [n][T][Hkv][d]    io_dtype   (T = B in hybrid_block_attn)
 *   W           [Hkv][d][F]       io_dtype   query head h uses W[h / G]
 *   alpha       [Hq]              float32    w_h = sigmoid(alpha[h]); +-inf allowed
 *   state       per request: Hkv head blocks of (2F*d + 2F) float32 each.
 *               Within a head block, S is kept transposed (S^T, d rows of 2F
 *               features) and cut into 2F/32 tiles of d rows x 32 features
 *               (128 bytes per row).  Logical element S[f][e] lives at float
 *               offset
 *                   (f/32)*32*d + e*32 + 4*(((f%32)/4) ^ (e%8)) + f%4,
 *               i.e. each 128-byte row is stored with its eight 16-byte
 *               granules permuted by XOR with (e mod 8).  This is the byte
 *               image that the tensor-core kernels consume directly (a
 *               1024-byte-aligned linear copy of a tile is a valid 128-byte-
 *               swizzled K-major operand), so a state is streamed from HBM
 *               with plain bulk copies.  z[f] follows at float offset
 *               2F*d + f.  hybrid_state_unpack / hybrid_state_pack convert
 *               to and from the logical [Hkv][2F][d] / [Hkv][2F] layout.
 *
 * Supported sizes: head_dim d in {64, 128}; feat_dim F in {16, 32, 64, 128,
 * 256}; 1 <= B <= 128; 1 <= Hkv <= Hq <= 256 with Hq % Hkv == 0; io_dtype
 * float32 or bfloat16.  The state is always float32.  Arithmetic is float32
 * throughout.  With bfloat16 inputs and F >= 64 the contractions of the
 * step (B a multiple of 16, G * B <= 128) and of the commit run on the
 * tensor cores (bf16 and tf32 operands, float32 accumulation); other shapes
 * and float32 inputs run float32 FMA kernels.
 *
 * Errors: argument checks run synchronously on the host and return
 * HYBRID_ERR_INVALID_ARG (null or misaligned pointer, inconsistent sizes) or
 * HYBRID_ERR_UNSUPPORTED (a size outside the supported set).  A failed
 * launch returns HYBRID_ERR_CUDA.  Problems found on the device (a null or
 * misaligned state pointer in d_state_ptrs, a wait that gave up) never trap:
 * the affected unit is skipped, a bit is set in the device error word, and
 * hybrid_check() reports it.
 */
#ifndef HYBRID_H_
#define HYBRID_H_

#include <stddef.h>
#include <cuda_runtime_api.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
    HYBRID_OK = 0,
    HYBRID_ERR_INVALID_ARG = 1,
    HYBRID_ERR_UNSUPPORTED = 2,
    HYBRID_ERR_CUDA = 3,
    HYBRID_ERR_TIMEOUT = 4,   /* a bounded device-side wait gave up */
    HYBRID_ERR_DEVICE = 5     /* a device-side argument check failed */
} hybrid_status;

typedef enum { HYBRID_F32 = 0, HYBRID_BF16 = 1 } hybrid_dtype;

typedef struct {
    int head_dim;          /* d */
    int feat_dim;          /* F: columns of W; phi(x) has 2F entries */
    int n_q_heads;         /* Hq */
    int n_kv_heads;        /* Hkv: state heads (GQA group G = Hq / Hkv) */
    int block_size;        /* B: tokens of the active block */
    hybrid_dtype io_dtype; /* dtype of Q, K, V, O, W */
} hybrid_cfg;

/* Bytes of one request's state: Hkv * (2F*d + 2F) * 4.  Returns 0 for an
 * invalid or unsupported cfg.  Cf. Section 3.1 (S_n in R^{2F x d},
 * Z_n in R^{2F}); the size is independent of the number of tokens absorbed. */
size_t hybrid_state_bytes(const hybrid_cfg *cfg);

/* Zero the states of n_req requests (an empty prefix: S_0 = 0, z_0 = 0). */
hybrid_status hybrid_state_init(const hybrid_cfg *cfg, void *const *d_state_ptrs, int n_req,
                                 cudaStream_t stream);

/* Feature map of Section 3.1: Phi = [softmax(X W_g), softmax(-X W_g)].
 *   X    [n_rows][n_heads_x][d] io_dtype (device); row head h uses
 *        W[h / (n_heads_x / Hkv)], so n_heads_x must be a multiple of Hkv
 *        (pass Hq for queries, Hkv for keys).
 *   Phi  [n_rows][n_heads_x][2F] float32 (device, written).
 * n_rows >= 0. */
hybrid_status hybrid_feature_map(const hybrid_cfg *cfg, const void *X, int n_rows, int n_heads_x,
                                 const void *W, float *Phi, cudaStream_t stream);

/* One denoising step of block-hybrid attention over the active block of every
 * request (Section 3.1: in-block softmax branch, linear readout from the
 * committed state, gated shared-normaliser merge).
 *   Q [n][B][Hq][d], K, V [n][B][Hkv][d], W [Hkv][d][F]: inputs (io_dtype)
 *   alpha [Hq] float32
 *   d_state_ptrs [n]: device array of state pointers; read, never written
 *   O [n][B][Hq][d]: output (io_dtype); must not alias an input
 * Query head h of request r reads state head h / G of request r. */
hybrid_status hybrid_block_attn(const hybrid_cfg *cfg, const void *Q, const void *K, const void *V,
                                const void *W, const float *alpha, void *const *d_state_ptrs,
                                int n_req, void *O, cudaStream_t stream);

/* One denoising step followed by the commit of the same block, in one pass
 * over the states (Section 3.1's step and state update; the paper's serving
 * section computes both in a single kernel launch).  O is computed from the
 * pre-commit state, then the block's K, V are folded into (S, z): equivalent to
 * hybrid_block_attn followed by hybrid_commit_block with n_tok = B, reading
 * and writing each state element once.  Arguments and layouts as in
 * hybrid_block_attn; the states are updated in place, so d_state_ptrs must not
 * name the same state twice. */
hybrid_status hybrid_block_attn_commit(const hybrid_cfg *cfg, const void *Q, const void *K,
                                       const void *V, const void *W, const float *alpha,
                                       void *const *d_state_ptrs, int n_req, void *O,
                                       cudaStream_t stream);

/* Bytes of the library's static scratch for hybrid_block_attn_commit_logical
 * (64 MiB, part of the library's device image on every device it runs on). */
#define HYBRID_LOGICAL_SCRATCH_BYTES (64u << 20)

/* hybrid_block_attn_commit on states held in the LOGICAL layout, for callers
 * that cannot allocate device memory.  The paper has no counterpart.  Some
 * callers keep S [n][Hkv][2F][d] and z [n][Hkv][2F] float32 in their own
 * buffers and cannot call cudaMalloc: a host application that owns all device
 * memory through its own pool or budget, so that a library may not take any;
 * a latency-critical decode loop, where an allocation can stall the loop
 * (cudaFree synchronises the device).  Such callers cannot provide the pointer
 * array and the operand-image states that hybrid_block_attn_commit reads.
 * This entry point brings its own device memory instead: one file-scope array
 * of HYBRID_LOGICAL_SCRATCH_BYTES per device, part of the library's device
 * image and held by every GPU that loads the library until the process exits.
 * One call packs the n_req states into that scratch (with the state-pointer
 * array), runs the fused step and commit there, and unpacks the updated states
 * back in place:
 *   Q, K, V, W, alpha, O  as in hybrid_block_attn (device pointers)
 *   S_logical, z_logical  device, read and overwritten with the committed state
 * It allocates nothing: no cudaMalloc, cudaFree or allocating library call.
 * Errors (the size and pointer checks run on the host before anything is
 * queued on the stream):
 * HYBRID_ERR_UNSUPPORTED when n_req * (hybrid_state_bytes(cfg) + 8) + 255
 * exceeds HYBRID_LOGICAL_SCRATCH_BYTES (up to 127 requests of 528 KB at c3's
 * shape, 15 of 4.2 MB at c5's); HYBRID_ERR_INVALID_ARG for a null or misaligned
 * pointer (S_logical, z_logical: 4-byte); otherwise as hybrid_block_attn_commit.
 * Races: the scratch is one per device, shared by every call, and keeps the
 * last call's contents (each call overwrites every byte it reads).  Calls that
 * overlap on the GPU race on it: issue them on one stream, or synchronise.
 * Set-up: the first call on a device, with that device current, looks the
 * scratch address up with cudaGetSymbolAddress (n_req = 0 does only that). */
hybrid_status hybrid_block_attn_commit_logical(const hybrid_cfg *cfg, const void *Q, const void *K,
                                               const void *V, const void *W, const float *alpha,
                                               float *S_logical, float *z_logical, int n_req, void *O,
                                               cudaStream_t stream);

/* Block commit of Section 3.1: S += sum_t phi(k_t) v_t^T, z += sum_t phi(k_t)
 * over the n_tok tokens of K, V [n][n_tok][Hkv][d] (io_dtype), for every
 * request and state head.  n_tok = B folds a decoded block; any n_tok >= 0
 * folds a prompt (prefill).  The states are updated in place. */
hybrid_status hybrid_commit_block(const hybrid_cfg *cfg, const void *K, const void *V, int n_tok,
                                  const void *W, void *const *d_state_ptrs, int n_req,
                                  cudaStream_t stream);

/* Prompt prefill with a different length per request (the state update of
 * Section 3.1, folding a prompt's tokens): request r folds tokens
 * [tok_offsets[r], tok_offsets[r + 1]) of the packed K, V
 * [tok_offsets[n_req]][Hkv][d] (io_dtype) into its state d_state_ptrs[r].
 *   tok_offsets  HOST array of n_req + 1 ints, tok_offsets[0] = 0, non-decreasing
 *                (a request with no tokens is left unchanged); read during the
 *                call, so the caller may reuse it on return
 *   K, V         device, 16-byte aligned, packed token-major as above
 * Equivalent to one hybrid_commit_block per request with n_tok = its length,
 * in one launch per 2048 requests (the offsets travel in the kernel
 * parameters, so the call can be captured in a CUDA graph).  Errors:
 * HYBRID_ERR_INVALID_ARG for null or misaligned pointers or offsets that do not
 * start at 0 or decrease; otherwise as hybrid_commit_block. */
hybrid_status hybrid_commit_ragged(const hybrid_cfg *cfg, const void *K, const void *V, const int *tok_offsets,
                                   int n_req, const void *W, void *const *d_state_ptrs, cudaStream_t stream);

/* Convert states to / from the logical layout (device buffers):
 *   S_logical [n][Hkv][2F][d] float32 (S[f][e] as in Section 3.1)
 *   z_logical [n][Hkv][2F]    float32 */
hybrid_status hybrid_state_unpack(const hybrid_cfg *cfg, void *const *d_state_ptrs, int n_req,
                                  float *S_logical, float *z_logical, cudaStream_t stream);
hybrid_status hybrid_state_pack(const hybrid_cfg *cfg, const float *S_logical,
                                const float *z_logical, void *const *d_state_ptrs, int n_req,
                                cudaStream_t stream);

/* ------------------------------------------------------------------------
 * Training form (Section 3.2, Stage 1 attention transfer).
 *
 * A batch of n_seq training sequences of seq_len = n_blk * B tokens, cut into
 * blocks B_0 .. B_{n_blk-1} of B = cfg->block_size tokens.  Teacher forcing
 * supplies every block's queries, keys and values; block n attends to itself
 * with the exact softmax branch and to blocks 0 .. n-1 through
 * S_{n-1} = sum_{m<n} sum_{t in B_m} phi(k_t) v_t^T and z_{n-1} likewise
 * (Section 3.1 applied to every block of the sequence; S_{-1} = 0).  Stage 1
 * trains only psi = {W, alpha} to match a frozen softmax teacher's output
 * under a squared-error loss; the caller forms dO = dL/dO from its loss.
 *
 *   Q, O, dO  [n_seq][seq_len][Hq][d]    bf16  (O: output of the forward)
 *   K, V      [n_seq][seq_len][Hkv][d]   bf16
 *   W         [Hkv][d][F] bf16;  alpha [Hq] float32
 *   dW        [Hkv][d][F] float32;  dalpha [Hq] float32  (overwritten)
 *   workspace device, 1024-byte aligned, >= hybrid_train_workspace_bytes bytes;
 *             hybrid_train_forward fills it with the states of every block, and
 *             hybrid_train_backward reads them (and then reuses the space), so
 *             one forward precedes each backward on the same workspace.
 * Supported: bf16 I/O, d in {64, 128}, F in {64, 128}, B in {16, 32, 64},
 * (Hq / Hkv) * B <= 128, seq_len a multiple of B; otherwise
 * HYBRID_ERR_UNSUPPORTED (seq_len not a multiple of B: HYBRID_ERR_INVALID_ARG).
 * Both calls are asynchronous on the stream; device-side wait failures are
 * reported by hybrid_check. */

/* Bytes of workspace for n_seq sequences of seq_len tokens; 0 when the shape is
 * not supported.  It holds the state of every block in two layouts, du of every
 * query and key row, the block-state pointers, and the partial sums of dW (at
 * most 256 slices of d x F) and of dalpha (one per block and query head) that
 * the backward adds in a fixed order. */
size_t hybrid_train_workspace_bytes(const hybrid_cfg *cfg, int n_seq, int seq_len);

/* O = block-hybrid attention of every block against the states of the blocks
 * before it; leaves those states in the workspace. */
hybrid_status hybrid_train_forward(const hybrid_cfg *cfg, const void *Q, const void *K, const void *V,
                                   const void *W, const float *alpha, int n_seq, int seq_len, void *O,
                                   void *workspace, size_t workspace_bytes, cudaStream_t stream);

/* Gradient of sum(dO * O) with respect to W and alpha, O being the output of
 * the preceding hybrid_train_forward on this workspace (O itself is not read:
 * dO . O is re-formed in fp32 from the merge's terms):
 *   dN = dO / D, dD = -(dO . O) / D (D = the merge's denominator),
 *   dw_h = sum (dN . sm_num + dD sm_den), dalpha_h = dw_h w_h (1 - w_h),
 *   dphi(q) = S_{n-1} dN + z_{n-1} dD,  dphi(k_t in B_m) = sum_{n>m} dS_{n-1} v_t + dz_{n-1},
 *   dW = sum over query and key rows of x du^T through phi's two softmaxes.
 * Partial sums are added in a fixed order (no floating-point atomics), so the
 * same inputs give the same dW and dalpha bits on every call. */
hybrid_status hybrid_train_backward(const hybrid_cfg *cfg, const void *Q, const void *K, const void *V,
                                    const void *W, const float *alpha, const void *dO, int n_seq,
                                    int seq_len, void *workspace, size_t workspace_bytes, float *dW,
                                    float *dalpha, cudaStream_t stream);

/* Testing hook for the device-side failure path; the paper has no counterpart.
 * Every wait inside the tensor-core kernels is bounded (1 s of the device's
 * global timer); when a bound runs out the kernel sets a bit in the device
 * error word, leaves its remaining work, waits (bounded) for its own copies in
 * flight, frees its Tensor Memory and returns, and hybrid_check() then reports
 * HYBRID_ERR_TIMEOUT.  Arming makes the NEXT launch of the persistent step
 * kernel (hybrid_block_attn on bf16 shapes with d, F in {64, 128}, B in
 * {16, 32}, G*B <= 128) exercise that path without faulting anything: its
 * waits give up after wait_ns nanoseconds instead of 1 s, and its math warps
 * never signal the barrier that releases the readout of the first feature
 * half (a barrier that no asynchronous copy targets), so the tensor-core
 * issuer's wait on it runs out.  The launch consumes the setting; later
 * launches run normally.  wait_ns = 0 disarms.  Errors: HYBRID_ERR_INVALID_ARG
 * for wait_ns above 10 s.  Host-only; touches no device. */
hybrid_status hybrid_debug_arm_wait_timeout(unsigned long long wait_ns);

/* Synchronise the stream, then read and clear this device's error word.
 * Returns HYBRID_OK, HYBRID_ERR_DEVICE (a state pointer failed its device
 * check), HYBRID_ERR_TIMEOUT (a bounded wait gave up) or HYBRID_ERR_CUDA. */
hybrid_status hybrid_check(cudaStream_t stream);

/* Static, human-readable name of a status code. */
const char *hybrid_status_str(hybrid_status status);

#ifdef __cplusplus
}
#endif

#endif /* HYBRID_H_ */
