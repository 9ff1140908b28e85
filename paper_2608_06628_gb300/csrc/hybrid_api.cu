// hybrid_api.cu -- the extern "C" entry points declared in include/hybrid.h:
// argument validation, kernel selection and launch, and the device error word.
#include <atomic>
#include <mutex>

#include "hybrid_common.cuh"
#include "hybrid_kernels.h"
#include "hybrid_tc.h"
#include "hybrid_train.h"

namespace {

// One error word per device, in the library's own static device memory.
__device__ unsigned g_error_word;

constexpr int kMaxDevices = 64;
std::mutex g_mu;
std::atomic<unsigned *> g_err_ptr[kMaxDevices];

// Device address of this device's error word, looked up once per device
// (with that device current, as cudaGetSymbolAddress requires).
unsigned *error_word()
{
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return nullptr;
    unsigned *p = g_err_ptr[dev].load(std::memory_order_acquire);
    if (p) return p;
    std::lock_guard<std::mutex> lock(g_mu);
    p = g_err_ptr[dev].load(std::memory_order_relaxed);
    if (!p) {
        void *sym = nullptr;
        if (cudaGetSymbolAddress(&sym, g_error_word) != cudaSuccess) return nullptr;
        p = static_cast<unsigned *>(sym);
        g_err_ptr[dev].store(p, std::memory_order_release);
    }
    return p;
}

// Scratch of hybrid_block_attn_commit_logical: the pointer array and the packed
// (operand-image) states of one call, in the library's own static device memory.
constexpr size_t kScratchBytes = (size_t)HYBRID_LOGICAL_SCRATCH_BYTES;
__device__ __align__(256) unsigned char g_scratch[kScratchBytes];
std::atomic<unsigned char *> g_scratch_ptr[kMaxDevices];

// Device address of this device's scratch, looked up once per device.
unsigned char *scratch()
{
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return nullptr;
    unsigned char *p = g_scratch_ptr[dev].load(std::memory_order_acquire);
    if (p) return p;
    std::lock_guard<std::mutex> lock(g_mu);
    p = g_scratch_ptr[dev].load(std::memory_order_relaxed);
    if (!p) {
        void *sym = nullptr;
        if (cudaGetSymbolAddress(&sym, g_scratch) != cudaSuccess) return nullptr;
        p = static_cast<unsigned char *>(sym);
        g_scratch_ptr[dev].store(p, std::memory_order_release);
    }
    return p;
}

// ptrs[i] = base + i * stride (the state pointers of the scratch slots).
__global__ void k_fill_ptrs(void **ptrs, unsigned char *base, size_t stride, int n)
{
    const int i = blockIdx.x * blockDim.x + threadIdx.x;
    if (i < n) ptrs[i] = base + (size_t)i * stride;
}

bool aligned(const void *p, uintptr_t a) { return (reinterpret_cast<uintptr_t>(p) & (a - 1)) == 0; }

hybrid_status check_cfg(const hybrid_cfg *c)
{
    if (!c) return HYBRID_ERR_INVALID_ARG;
    if (c->io_dtype != HYBRID_F32 && c->io_dtype != HYBRID_BF16) return HYBRID_ERR_UNSUPPORTED;
    if (c->head_dim != 64 && c->head_dim != 128) return HYBRID_ERR_UNSUPPORTED;
    const int F = c->feat_dim;
    if (F != 16 && F != 32 && F != 64 && F != 128 && F != 256) return HYBRID_ERR_UNSUPPORTED;
    if (c->block_size < 1 || c->block_size > 128) return HYBRID_ERR_UNSUPPORTED;
    if (c->n_kv_heads < 1 || c->n_q_heads < 1 || c->n_q_heads > 256) return HYBRID_ERR_UNSUPPORTED;
    if (c->n_kv_heads > c->n_q_heads || c->n_q_heads % c->n_kv_heads != 0) return HYBRID_ERR_INVALID_ARG;
    return HYBRID_OK;
}

hybrid_status from_cuda(cudaError_t e) { return e == cudaSuccess ? HYBRID_OK : HYBRID_ERR_CUDA; }

}  // namespace

namespace hyb {
std::atomic<unsigned long long> g_armed_wait_ns{0};
}

extern "C" {

size_t hybrid_state_bytes(const hybrid_cfg *cfg)
{
    if (check_cfg(cfg) != HYBRID_OK) return 0;
    return (size_t)cfg->n_kv_heads * hyb::head_floats(cfg->head_dim, cfg->feat_dim) * sizeof(float);
}

hybrid_status hybrid_state_init(const hybrid_cfg *cfg, void *const *d_state_ptrs, int n_req,
                                cudaStream_t stream)
{
    hybrid_status s = check_cfg(cfg);
    if (s != HYBRID_OK) return s;
    if (n_req < 0) return HYBRID_ERR_INVALID_ARG;
    if (n_req == 0) return HYBRID_OK;
    if (!d_state_ptrs || !aligned(d_state_ptrs, 8)) return HYBRID_ERR_INVALID_ARG;
    return from_cuda(hyb::launch_state_init(*cfg, d_state_ptrs, n_req, stream));
}

hybrid_status hybrid_feature_map(const hybrid_cfg *cfg, const void *X, int n_rows, int n_heads_x,
                                 const void *W, float *Phi, cudaStream_t stream)
{
    hybrid_status s = check_cfg(cfg);
    if (s != HYBRID_OK) return s;
    if (n_rows < 0 || n_heads_x < 1 || n_heads_x % cfg->n_kv_heads != 0) return HYBRID_ERR_INVALID_ARG;
    if (n_rows == 0) return HYBRID_OK;
    if (!X || !W || !Phi || !aligned(X, 16) || !aligned(W, 16) || !aligned(Phi, 16))
        return HYBRID_ERR_INVALID_ARG;
    return from_cuda(hyb::launch_feature_map(cfg->io_dtype, X, n_rows, n_heads_x, cfg->n_kv_heads,
                                             cfg->head_dim, cfg->feat_dim, W, Phi, stream));
}

hybrid_status hybrid_block_attn(const hybrid_cfg *cfg, const void *Q, const void *K, const void *V,
                                const void *W, const float *alpha, void *const *d_state_ptrs,
                                int n_req, void *O, cudaStream_t stream)
{
    hybrid_status s = check_cfg(cfg);
    if (s != HYBRID_OK) return s;
    if (n_req < 0) return HYBRID_ERR_INVALID_ARG;
    if (n_req == 0) return HYBRID_OK;
    if (!Q || !K || !V || !W || !alpha || !d_state_ptrs || !O) return HYBRID_ERR_INVALID_ARG;
    if (!aligned(Q, 16) || !aligned(K, 16) || !aligned(V, 16) || !aligned(W, 16) || !aligned(O, 16) ||
        !aligned(alpha, 4) || !aligned(d_state_ptrs, 8))
        return HYBRID_ERR_INVALID_ARG;
    unsigned *err = error_word();
    if (!err) return HYBRID_ERR_CUDA;
    if (hyb::step_supported(*cfg))
        return from_cuda(hyb::launch_step(*cfg, Q, K, V, W, alpha, d_state_ptrs, n_req, O, err, stream));
    if (hyb::tc_attn_supported(*cfg))
        return from_cuda(hyb::launch_attn_tc(*cfg, Q, K, V, W, alpha, d_state_ptrs, n_req, O, err, stream));
    return from_cuda(hyb::launch_attn_generic(*cfg, Q, K, V, W, alpha, d_state_ptrs, n_req, O, err, stream));
}

hybrid_status hybrid_block_attn_commit(const hybrid_cfg *cfg, const void *Q, const void *K, const void *V,
                                       const void *W, const float *alpha, void *const *d_state_ptrs,
                                       int n_req, void *O, cudaStream_t stream)
{
    hybrid_status s = check_cfg(cfg);
    if (s != HYBRID_OK) return s;
    if (n_req < 0) return HYBRID_ERR_INVALID_ARG;
    if (n_req == 0) return HYBRID_OK;
    if (!Q || !K || !V || !W || !alpha || !d_state_ptrs || !O) return HYBRID_ERR_INVALID_ARG;
    if (!aligned(Q, 16) || !aligned(K, 16) || !aligned(V, 16) || !aligned(W, 16) || !aligned(O, 16) ||
        !aligned(alpha, 4) || !aligned(d_state_ptrs, 8))
        return HYBRID_ERR_INVALID_ARG;
    unsigned *err = error_word();
    if (!err) return HYBRID_ERR_CUDA;
    if (hyb::fused_supported(*cfg))
        return from_cuda(hyb::launch_fused(*cfg, Q, K, V, W, alpha, d_state_ptrs, n_req, O, err, stream));
    // other shapes: the step, then the commit, on the same stream
    s = hybrid_block_attn(cfg, Q, K, V, W, alpha, d_state_ptrs, n_req, O, stream);
    if (s != HYBRID_OK) return s;
    return hybrid_commit_block(cfg, K, V, cfg->block_size, W, d_state_ptrs, n_req, stream);
}

hybrid_status hybrid_block_attn_commit_logical(const hybrid_cfg *cfg, const void *Q, const void *K,
                                               const void *V, const void *W, const float *alpha,
                                               float *S_logical, float *z_logical, int n_req, void *O,
                                               cudaStream_t stream)
{
    hybrid_status s = check_cfg(cfg);
    if (s != HYBRID_OK) return s;
    if (n_req < 0) return HYBRID_ERR_INVALID_ARG;
    // Size first, on the host, in a form that cannot wrap: the pointer array takes
    // at most 8 n_req + 255 bytes once rounded up to 256, so
    //   n_req (8 + sb) + 255 <= kScratchBytes  implies  ceil256(8 n_req) + n_req sb <= kScratchBytes.
    const size_t sb = hybrid_state_bytes(cfg);   // a multiple of 16 bytes
    if (sb == 0) return HYBRID_ERR_UNSUPPORTED;
    if ((size_t)n_req > (kScratchBytes - 255) / (sb + sizeof(void *))) return HYBRID_ERR_UNSUPPORTED;
    // every pointer is checked before any work is queued on the stream
    if (n_req > 0) {
        if (!Q || !K || !V || !W || !alpha || !O || !S_logical || !z_logical) return HYBRID_ERR_INVALID_ARG;
        if (!aligned(Q, 16) || !aligned(K, 16) || !aligned(V, 16) || !aligned(W, 16) || !aligned(O, 16) ||
            !aligned(alpha, 4) || !aligned(S_logical, 4) || !aligned(z_logical, 4))
            return HYBRID_ERR_INVALID_ARG;
    }
    // the scratch address is looked up here, also for n_req = 0 (set-up call)
    unsigned char *base = scratch();
    if (!base) return HYBRID_ERR_CUDA;
    if (n_req == 0) return HYBRID_OK;
    const size_t ptr_bytes = ((size_t)n_req * sizeof(void *) + 255) & ~(size_t)255;
    void **d_ptrs = reinterpret_cast<void **>(base);
    unsigned char *states = base + ptr_bytes;
    {
        // the launch's own status (not an error left over from earlier work)
        size_t stride = sb;
        int n = n_req;
        void *args[] = {&d_ptrs, &states, &stride, &n};
        const cudaError_t e = cudaLaunchKernel(reinterpret_cast<const void *>(&k_fill_ptrs),
                                               dim3((unsigned)((n_req + 127) / 128)), dim3(128), args, 0, stream);
        if (e != cudaSuccess) return HYBRID_ERR_CUDA;
    }
    s = hybrid_state_pack(cfg, S_logical, z_logical, d_ptrs, n_req, stream);
    if (s != HYBRID_OK) return s;
    s = hybrid_block_attn_commit(cfg, Q, K, V, W, alpha, d_ptrs, n_req, O, stream);
    if (s != HYBRID_OK) return s;
    return hybrid_state_unpack(cfg, d_ptrs, n_req, S_logical, z_logical, stream);
}

// Commits of more tokens than this run the prefill kernel (measured crossover
// on the batch-64 shape: 64 tokens per request).
constexpr int kPrefillMinTokens = 64;

hybrid_status hybrid_commit_block(const hybrid_cfg *cfg, const void *K, const void *V, int n_tok,
                                  const void *W, void *const *d_state_ptrs, int n_req,
                                  cudaStream_t stream)
{
    hybrid_status s = check_cfg(cfg);
    if (s != HYBRID_OK) return s;
    if (n_req < 0 || n_tok < 0) return HYBRID_ERR_INVALID_ARG;
    if (n_req == 0 || n_tok == 0) return HYBRID_OK;
    if (!K || !V || !W || !d_state_ptrs) return HYBRID_ERR_INVALID_ARG;
    if (!aligned(K, 16) || !aligned(V, 16) || !aligned(W, 16) || !aligned(d_state_ptrs, 8))
        return HYBRID_ERR_INVALID_ARG;
    unsigned *err = error_word();
    if (!err) return HYBRID_ERR_CUDA;
    // block commits (a few dozen tokens) run the per-unit reduction kernel; longer
    // prompts the token-major prefill kernel, which balances chunks across SMs
    if (n_tok > kPrefillMinTokens && hyb::prefill_supported(*cfg))
        return from_cuda(hyb::launch_prefill(*cfg, K, V, n_tok, W, d_state_ptrs, n_req, err, stream));
    if (hyb::commit_red_supported(*cfg))
        return from_cuda(hyb::launch_commit_red(*cfg, K, V, n_tok, W, d_state_ptrs, n_req, err, stream));
    return from_cuda(hyb::launch_commit_generic(*cfg, K, V, n_tok, W, d_state_ptrs, n_req, err, stream));
}

hybrid_status hybrid_commit_ragged(const hybrid_cfg *cfg, const void *K, const void *V, const int *tok_offsets,
                                   int n_req, const void *W, void *const *d_state_ptrs, cudaStream_t stream)
{
    hybrid_status s = check_cfg(cfg);
    if (s != HYBRID_OK) return s;
    if (n_req < 0) return HYBRID_ERR_INVALID_ARG;
    if (n_req == 0) return HYBRID_OK;
    if (!tok_offsets || tok_offsets[0] != 0) return HYBRID_ERR_INVALID_ARG;
    for (int r = 0; r < n_req; ++r)
        if (tok_offsets[r + 1] < tok_offsets[r]) return HYBRID_ERR_INVALID_ARG;
    if (tok_offsets[n_req] == 0) return HYBRID_OK;
    if (!K || !V || !W || !d_state_ptrs) return HYBRID_ERR_INVALID_ARG;
    if (!aligned(K, 16) || !aligned(V, 16) || !aligned(W, 16) || !aligned(d_state_ptrs, 8))
        return HYBRID_ERR_INVALID_ARG;
    unsigned *err = error_word();
    if (!err) return HYBRID_ERR_CUDA;
    const size_t row_bytes = (size_t)cfg->n_kv_heads * cfg->head_dim * (cfg->io_dtype == HYBRID_BF16 ? 2 : 4);
    const unsigned char *Kb = static_cast<const unsigned char *>(K);
    const unsigned char *Vb = static_cast<const unsigned char *>(V);
    const bool red = hyb::commit_red_supported(*cfg), pre = hyb::prefill_supported(*cfg);
    if (!red && !pre) {
        // FMA kernels: one launch per request that has tokens
        for (int r = 0; r < n_req; ++r) {
            const int T = tok_offsets[r + 1] - tok_offsets[r];
            if (T == 0) continue;
            const size_t off = (size_t)tok_offsets[r] * row_bytes;
            const cudaError_t e =
                hyb::launch_commit_generic(*cfg, Kb + off, Vb + off, T, W, d_state_ptrs + r, 1, err, stream);
            if (e != cudaSuccess) return from_cuda(e);
        }
        return HYBRID_OK;
    }
    // tensor-core kernels, up to kMaxRaggedRequests requests per launch (offsets rebased)
    static thread_local int tok[hyb::kMaxRaggedRequests + 1];
    for (int r0 = 0; r0 < n_req; r0 += hyb::kMaxRaggedRequests) {
        const int nb = n_req - r0 < hyb::kMaxRaggedRequests ? n_req - r0 : hyb::kMaxRaggedRequests;
        int longest = 0;
        for (int i = 0; i <= nb; ++i) tok[i] = tok_offsets[r0 + i] - tok_offsets[r0];
        for (int i = 0; i < nb; ++i) longest = tok[i + 1] - tok[i] > longest ? tok[i + 1] - tok[i] : longest;
        if (tok[nb] == 0) continue;
        const size_t off = (size_t)tok_offsets[r0] * row_bytes;
        // as for uniform prompts: the token-major kernel once a prompt is longer than a
        // block commit (it balances chunks across SMs), else the per-unit reduction kernel
        const cudaError_t e =
            pre && (longest > kPrefillMinTokens || !red)
                ? hyb::launch_prefill_ragged(*cfg, Kb + off, Vb + off, tok, W, d_state_ptrs + r0, nb, err, stream)
                : hyb::launch_commit_red_ragged(*cfg, Kb + off, Vb + off, tok, W, d_state_ptrs + r0, nb, err, stream);
        if (e != cudaSuccess) return from_cuda(e);
    }
    return HYBRID_OK;
}

hybrid_status hybrid_state_unpack(const hybrid_cfg *cfg, void *const *d_state_ptrs, int n_req,
                                  float *S_logical, float *z_logical, cudaStream_t stream)
{
    hybrid_status s = check_cfg(cfg);
    if (s != HYBRID_OK) return s;
    if (n_req < 0) return HYBRID_ERR_INVALID_ARG;
    if (n_req == 0) return HYBRID_OK;
    if (!d_state_ptrs || !S_logical || !z_logical || !aligned(d_state_ptrs, 8) ||
        !aligned(S_logical, 4) || !aligned(z_logical, 4))
        return HYBRID_ERR_INVALID_ARG;
    unsigned *err = error_word();
    if (!err) return HYBRID_ERR_CUDA;
    return from_cuda(hyb::launch_state_unpack(*cfg, d_state_ptrs, n_req, S_logical, z_logical, err, stream));
}

hybrid_status hybrid_state_pack(const hybrid_cfg *cfg, const float *S_logical,
                                const float *z_logical, void *const *d_state_ptrs, int n_req,
                                cudaStream_t stream)
{
    hybrid_status s = check_cfg(cfg);
    if (s != HYBRID_OK) return s;
    if (n_req < 0) return HYBRID_ERR_INVALID_ARG;
    if (n_req == 0) return HYBRID_OK;
    if (!d_state_ptrs || !S_logical || !z_logical || !aligned(d_state_ptrs, 8) ||
        !aligned(S_logical, 4) || !aligned(z_logical, 4))
        return HYBRID_ERR_INVALID_ARG;
    unsigned *err = error_word();
    if (!err) return HYBRID_ERR_CUDA;
    return from_cuda(hyb::launch_state_pack(*cfg, S_logical, z_logical, d_state_ptrs, n_req, err, stream));
}

size_t hybrid_train_workspace_bytes(const hybrid_cfg *cfg, int n_seq, int seq_len)
{
    if (check_cfg(cfg) != HYBRID_OK || n_seq < 1 || !hyb::train_supported(*cfg, seq_len)) return 0;
    return hyb::train_workspace_bytes(*cfg, n_seq, seq_len);
}

namespace {
hybrid_status check_train(const hybrid_cfg *cfg, int n_seq, int seq_len, const void *workspace,
                          size_t workspace_bytes)
{
    hybrid_status s = check_cfg(cfg);
    if (s != HYBRID_OK) return s;
    if (n_seq < 1 || seq_len < 1) return HYBRID_ERR_INVALID_ARG;
    if (seq_len % cfg->block_size != 0) return HYBRID_ERR_INVALID_ARG;
    if (!hyb::train_supported(*cfg, seq_len)) return HYBRID_ERR_UNSUPPORTED;
    if (!workspace || !aligned(workspace, 1024)) return HYBRID_ERR_INVALID_ARG;
    if (workspace_bytes < hyb::train_workspace_bytes(*cfg, n_seq, seq_len)) return HYBRID_ERR_INVALID_ARG;
    return HYBRID_OK;
}
}  // namespace

hybrid_status hybrid_train_forward(const hybrid_cfg *cfg, const void *Q, const void *K, const void *V,
                                   const void *W, const float *alpha, int n_seq, int seq_len, void *O,
                                   void *workspace, size_t workspace_bytes, cudaStream_t stream)
{
    hybrid_status s = check_train(cfg, n_seq, seq_len, workspace, workspace_bytes);
    if (s != HYBRID_OK) return s;
    if (!Q || !K || !V || !W || !alpha || !O) return HYBRID_ERR_INVALID_ARG;
    if (!aligned(Q, 16) || !aligned(K, 16) || !aligned(V, 16) || !aligned(W, 16) || !aligned(O, 16) ||
        !aligned(alpha, 4))
        return HYBRID_ERR_INVALID_ARG;
    unsigned *err = error_word();
    if (!err) return HYBRID_ERR_CUDA;
    const cudaError_t e = hyb::launch_train_states(*cfg, K, V, W, n_seq, seq_len, workspace, err, stream);
    if (e != cudaSuccess) return HYBRID_ERR_CUDA;
    // every block of every sequence is one decode step against the state of its prefix
    const int n_blk = seq_len / cfg->block_size;
    return hybrid_block_attn(cfg, Q, K, V, W, alpha, hyb::train_state_ptrs(*cfg, n_seq, seq_len, workspace),
                             n_seq * n_blk, O, stream);
}

hybrid_status hybrid_train_backward(const hybrid_cfg *cfg, const void *Q, const void *K, const void *V,
                                    const void *W, const float *alpha, const void *dO, int n_seq,
                                    int seq_len, void *workspace, size_t workspace_bytes, float *dW,
                                    float *dalpha, cudaStream_t stream)
{
    hybrid_status s = check_train(cfg, n_seq, seq_len, workspace, workspace_bytes);
    if (s != HYBRID_OK) return s;
    if (!Q || !K || !V || !W || !alpha || !dO || !dW || !dalpha) return HYBRID_ERR_INVALID_ARG;
    if (!aligned(Q, 16) || !aligned(K, 16) || !aligned(V, 16) || !aligned(W, 16) || !aligned(dO, 16) ||
        !aligned(alpha, 4) || !aligned(dW, 16) || !aligned(dalpha, 4))
        return HYBRID_ERR_INVALID_ARG;
    unsigned *err = error_word();
    if (!err) return HYBRID_ERR_CUDA;
    return from_cuda(hyb::launch_train_backward(*cfg, Q, K, V, W, alpha, dO, n_seq, seq_len, workspace, dW, dalpha,
                                                err, stream));
}

hybrid_status hybrid_debug_arm_wait_timeout(unsigned long long wait_ns)
{
    if (wait_ns > 10000000000ull) return HYBRID_ERR_INVALID_ARG;
    hyb::g_armed_wait_ns.store(wait_ns);
    return HYBRID_OK;
}

hybrid_status hybrid_check(cudaStream_t stream)
{
    unsigned *err = error_word();
    if (!err) return HYBRID_ERR_CUDA;
    if (cudaStreamSynchronize(stream) != cudaSuccess) return HYBRID_ERR_CUDA;
    unsigned word = 0;
    if (cudaMemcpy(&word, err, sizeof word, cudaMemcpyDeviceToHost) != cudaSuccess) return HYBRID_ERR_CUDA;
    if (word != 0) {
        const unsigned zero = 0;
        if (cudaMemcpy(err, &zero, sizeof zero, cudaMemcpyHostToDevice) != cudaSuccess)
            return HYBRID_ERR_CUDA;
    }
    if (word & hyb::ERR_WAIT_TIMEOUT) return HYBRID_ERR_TIMEOUT;
    if (word & hyb::ERR_BAD_STATE_PTR) return HYBRID_ERR_DEVICE;
    return HYBRID_OK;
}

const char *hybrid_status_str(hybrid_status status)
{
    switch (status) {
    case HYBRID_OK: return "HYBRID_OK";
    case HYBRID_ERR_INVALID_ARG: return "HYBRID_ERR_INVALID_ARG: invalid argument";
    case HYBRID_ERR_UNSUPPORTED: return "HYBRID_ERR_UNSUPPORTED: size or dtype outside the supported set";
    case HYBRID_ERR_CUDA: return "HYBRID_ERR_CUDA: CUDA runtime error";
    case HYBRID_ERR_TIMEOUT: return "HYBRID_ERR_TIMEOUT: a bounded device wait gave up";
    case HYBRID_ERR_DEVICE: return "HYBRID_ERR_DEVICE: a device-side argument check failed";
    }
    return "HYBRID_ERR_UNKNOWN";
}

}  // extern "C"
