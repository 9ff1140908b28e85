// hybrid_state.cu -- zeroing and layout conversion of the per-request state.
//
// The state of one request is Hkv head blocks of S (2F x d) and z (2F),
// Section 3.1's S_n and Z_n, stored as documented in hybrid.h.
#include "hybrid_common.cuh"
#include "hybrid_kernels.h"

namespace hyb {

// grid.x = n_req * chunks; zero 16-byte granules of each request's buffer
__global__ void k_state_init(void *const *__restrict__ states, int chunks, size_t n_gran)
{
    const int r = blockIdx.x / chunks;
    const size_t base = (size_t)(blockIdx.x % chunks) * blockDim.x * 8;
    float4 *p = reinterpret_cast<float4 *>(states[r]);
    if (!state_ptr_ok(p)) return;
    const float4 zero = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
    for (int k = 0; k < 8; ++k) {
        const size_t i = base + (size_t)k * blockDim.x + threadIdx.x;
        if (i < n_gran) p[i] = zero;
    }
}

cudaError_t launch_state_init(const hybrid_cfg &c, void *const *states, int n_req, cudaStream_t st)
{
    const size_t n_gran = (size_t)c.n_kv_heads * head_floats(c.head_dim, c.feat_dim) / 4;
    const int threads = 256;
    const int chunks = (int)((n_gran + threads * 8 - 1) / (threads * 8));
    k_state_init<<<(unsigned)((long long)n_req * chunks), threads, 0, st>>>(states, chunks, n_gran);
    return cudaGetLastError();
}

// one thread per logical (request, head, f, e) element, plus z
template <bool kPack>
__global__ void k_state_convert(void *const *__restrict__ states, int n_req, int Hkv, int d, int F,
                                float *__restrict__ S, float *__restrict__ z, unsigned *err)
{
    const int P2 = 2 * F;
    const size_t per_head = (size_t)P2 * d + P2;
    const size_t total = (size_t)n_req * Hkv * per_head;
    for (size_t i = (size_t)blockIdx.x * blockDim.x + threadIdx.x; i < total;
         i += (size_t)gridDim.x * blockDim.x) {
        const size_t rh = i / per_head;
        const size_t w = i % per_head;
        const int r = (int)(rh / Hkv), g = (int)(rh % Hkv);
        float *st = reinterpret_cast<float *>(states[r]);
        if (!state_ptr_ok(st)) {
            raise_error(err, ERR_BAD_STATE_PTR);
            continue;
        }
        float *hb = st + (size_t)g * head_floats(d, F);
        if (w < (size_t)P2 * d) {
            const int f = (int)(w / d), e = (int)(w % d);
            float *logical = S + rh * (size_t)P2 * d + w;
            if (kPack) hb[s_offset(f, e, d)] = *logical;
            else *logical = hb[s_offset(f, e, d)];
        } else {
            const int f = (int)(w - (size_t)P2 * d);
            float *logical = z + rh * (size_t)P2 + f;
            if (kPack) hb[z_offset(f, d, F)] = *logical;
            else *logical = hb[z_offset(f, d, F)];
        }
    }
}

cudaError_t launch_state_unpack(const hybrid_cfg &c, void *const *states, int n_req, float *S,
                                float *z, unsigned *err, cudaStream_t st)
{
    k_state_convert<false><<<1024, 256, 0, st>>>(states, n_req, c.n_kv_heads, c.head_dim, c.feat_dim,
                                                 S, z, err);
    return cudaGetLastError();
}

cudaError_t launch_state_pack(const hybrid_cfg &c, const float *S, const float *z,
                              void *const *states, int n_req, unsigned *err, cudaStream_t st)
{
    k_state_convert<true><<<1024, 256, 0, st>>>(states, n_req, c.n_kv_heads, c.head_dim, c.feat_dim,
                                                const_cast<float *>(S), const_cast<float *>(z), err);
    return cudaGetLastError();
}

}  // namespace hyb
