// hybrid_common.cuh -- device helpers shared by the block-hybrid kernels.
//
// Notation follows Section 3.1 of "Retrofitting Linear Attention into
// Diffusion Language Models": d = head dim, F = columns of the Hedgehog map
// W (phi has 2F entries), S in R^{2F x d}, z in R^{2F}.
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "hybrid.h"

namespace hyb {

// Bits of the per-device error word (read and cleared by hybrid_check).
enum : unsigned {
    ERR_BAD_STATE_PTR = 1u,   // null or misaligned entry in d_state_ptrs
    ERR_WAIT_TIMEOUT = 2u,    // a bounded mbarrier / flag wait gave up
};

__device__ __forceinline__ void raise_error(unsigned *err, unsigned bit)
{
    if (err) atomicOr(err, bit);
}

// ---------------------------------------------------------------------------
// State layout (documented in hybrid.h).  Per head block: S^T cut into 2F/32
// tiles of d rows x 32 features, each 128-byte row with its 16-byte granules
// permuted by XOR with (row mod 8); then z[2F].
// ---------------------------------------------------------------------------
__host__ __device__ __forceinline__ size_t head_floats(int d, int F)
{
    return (size_t)2 * F * d + (size_t)2 * F;
}

// float offset of logical S[f][e] inside a head block
__host__ __device__ __forceinline__ size_t s_offset(int f, int e, int d)
{
    return (size_t)(f >> 5) * 32 * d + (size_t)e * 32 + (size_t)((((f & 31) >> 2) ^ (e & 7)) << 2) + (f & 3);
}

// float offset of z[f] inside a head block
__host__ __device__ __forceinline__ size_t z_offset(int f, int d, int F)
{
    return (size_t)2 * F * d + f;
}

// For granule p (16 bytes) of tile `tile` (d rows x 8 granules, in storage
// order): the row e and the first logical feature f of the 4 floats it holds.
__host__ __device__ __forceinline__ void granule_coords(int p_in_tile, int tile, int &e, int &f0)
{
    e = p_in_tile >> 3;
    const int j = (p_in_tile & 7) ^ (e & 7);
    f0 = tile * 32 + 4 * j;
}

__device__ __forceinline__ bool state_ptr_ok(const void *p)
{
    return p != nullptr && (reinterpret_cast<uintptr_t>(p) & 15u) == 0;
}

// ---------------------------------------------------------------------------
// io dtype loads / stores
// ---------------------------------------------------------------------------
__device__ __forceinline__ float to_f32(float x) { return x; }
__device__ __forceinline__ float to_f32(__nv_bfloat16 x) { return __bfloat162float(x); }

template <typename T> __device__ __forceinline__ T from_f32(float x);
template <> __device__ __forceinline__ float from_f32<float>(float x) { return x; }
template <> __device__ __forceinline__ __nv_bfloat16 from_f32<__nv_bfloat16>(float x)
{
    return __float2bfloat16_rn(x);
}

__device__ __forceinline__ float warp_max(float v)
{
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
    return v;
}
__device__ __forceinline__ float warp_min(float v)
{
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v = fminf(v, __shfl_xor_sync(0xffffffffu, v, o));
    return v;
}
__device__ __forceinline__ float warp_sum(float v)
{
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}

// log(sigmoid(alpha)) = -softplus(-alpha), finite for finite alpha, -inf at -inf.
__device__ __forceinline__ float log_sigmoid(float alpha)
{
    const float x = -alpha;
    if (x > 20.f) return -(x + log1pf(expf(-x)));
    return -log1pf(expf(x));
}

// Gated shared-normaliser merge of Section 3.1,
//     out = (w sm_num + lin_num) / (w sm_den + lin_den),
// evaluated from the shifted softmax sums sm_num = e^m * num_s, sm_den = e^m * l
// (num_s, l computed with max-shift m).  Writing A = w sm_den and L = lin_den,
//     out = A/(A+L) * (num_s / l) + L/(A+L) * (lin_num / L),
// which is the same quantity with both masses compared in log space, so no
// exponential of the unshifted scores is ever formed.
struct MergeWeights {
    float ws;   // weight of num_s  (= A/(A+L) / l)
    float wl;   // weight of lin_num (= L/(A+L) / L)
};
__device__ __forceinline__ MergeWeights merge_weights(float log_w, float m, float l, float lin_den)
{
    MergeWeights r;
    if (lin_den > 0.f) {
        // x = log A - log L
        const float x = log_w + m + logf(l) - logf(lin_den);
        const float rho = 1.f / (1.f + expf(-x));          // A / (A + L)
        const float rho_l = 1.f / (1.f + expf(x));         // L / (A + L)
        r.ws = rho / l;
        r.wl = rho_l / lin_den;
    } else {
        // empty prefix: the softmax branch alone (w cancels); w = 0 gives 0/0
        r.ws = (log_w == -INFINITY) ? __int_as_float(0x7fc00000) : 1.f / l;
        r.wl = 0.f;
    }
    return r;
}

}  // namespace hyb
