// hybrid_generic.cu -- CUDA-core kernels for every supported shape and dtype.
//
// These kernels do all arithmetic in float32 on the FMA pipes.  They are the
// exact path for float32 I/O and the path for shapes that the tensor-core
// kernels do not take.  Section 3.1 of "Retrofitting Linear Attention into
// Diffusion Language Models" defines every quantity computed here.
#include "hybrid_common.cuh"
#include "hybrid_kernels.h"

namespace hyb {

constexpr int kMaxFWarp = 8;   // F <= 256 -> at most 8 features per lane and half

// ---------------------------------------------------------------------------
// phi of one row, one warp (Sec. 3.1):  u = x W_g,
//   pos[k] = softmax(u)[f],  neg[k] = softmax(-u)[f],  f = lane + 32 k.
// x is float32 in shared memory (broadcast reads), W_g is [d][F] in global.
// Both softmaxes are max-shifted, which leaves them unchanged.
// ---------------------------------------------------------------------------
template <typename T>
__device__ __forceinline__ void warp_phi_row(const float *x, const T *__restrict__ Wg, int d, int F,
                                             float (&pos)[kMaxFWarp], float (&neg)[kMaxFWarp])
{
    const int lane = threadIdx.x & 31;
    float u[kMaxFWarp];
#pragma unroll
    for (int k = 0; k < kMaxFWarp; ++k) u[k] = 0.f;
    for (int e = 0; e < d; ++e) {
        const float xe = x[e];
        const T *wrow = Wg + (size_t)e * F;
#pragma unroll
        for (int k = 0; k < kMaxFWarp; ++k) {
            const int f = lane + 32 * k;
            if (f < F) u[k] = fmaf(xe, to_f32(wrow[f]), u[k]);
        }
    }
    float mx = -INFINITY, mn = INFINITY;
#pragma unroll
    for (int k = 0; k < kMaxFWarp; ++k) {
        if (lane + 32 * k < F) { mx = fmaxf(mx, u[k]); mn = fminf(mn, u[k]); }
    }
    mx = warp_max(mx);
    mn = warp_min(mn);
    float sp = 0.f, sn = 0.f;
#pragma unroll
    for (int k = 0; k < kMaxFWarp; ++k) {
        if (lane + 32 * k < F) {
            pos[k] = expf(u[k] - mx);
            neg[k] = expf(mn - u[k]);
            sp += pos[k];
            sn += neg[k];
        } else {
            pos[k] = 0.f;
            neg[k] = 0.f;
        }
    }
    sp = warp_sum(sp);
    sn = warp_sum(sn);
    const float ip = 1.f / sp, in = 1.f / sn;
#pragma unroll
    for (int k = 0; k < kMaxFWarp; ++k) { pos[k] *= ip; neg[k] *= in; }
}

// ---------------------------------------------------------------------------
// Feature map: one warp per (row, head).
// ---------------------------------------------------------------------------
template <typename T>
__global__ void __launch_bounds__(256) k_feature_map(const T *__restrict__ X, int n_rows, int nh,
                                                     int group, int d, int F,
                                                     const T *__restrict__ W, float *__restrict__ Phi)
{
    extern __shared__ float smem[];
    const int warp_in_cta = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const long long item = (long long)blockIdx.x * (blockDim.x >> 5) + warp_in_cta;
    float *xs = smem + warp_in_cta * d;
    const bool active = item < (long long)n_rows * nh;
    if (!active) return;
    const int h = (int)(item % nh);
    const T *x = X + (size_t)item * d;
    for (int e = lane; e < d; e += 32) xs[e] = to_f32(x[e]);
    __syncwarp();
    float pos[kMaxFWarp], neg[kMaxFWarp];
    warp_phi_row<T>(xs, W + (size_t)(h / group) * d * F, d, F, pos, neg);
    float *out = Phi + (size_t)item * 2 * F;
#pragma unroll
    for (int k = 0; k < kMaxFWarp; ++k) {
        const int f = lane + 32 * k;
        if (f < F) { out[f] = pos[k]; out[F + f] = neg[k]; }
    }
}

// ---------------------------------------------------------------------------
// Block attention, generic: one CTA per (request, query head, tile of RT rows).
// ---------------------------------------------------------------------------
constexpr int kRT = 16;            // query rows per CTA
constexpr int kGenThreads = 256;   // 8 warps, 2 rows each

size_t generic_attn_smem_bytes(int d, int F, int B)
{
    const size_t fl = (size_t)B * (d + 1) + (size_t)B * d + (size_t)kRT * d + (size_t)kRT * 2 * F +
                      (size_t)kRT * B + (size_t)d * 33 + 3 * kRT;
    return fl * sizeof(float);
}

template <typename T>
__global__ void __launch_bounds__(kGenThreads) k_attn_generic(
    const T *__restrict__ Q, const T *__restrict__ K, const T *__restrict__ V, const T *__restrict__ W,
    const float *__restrict__ alpha, void *const *__restrict__ states, int n_req, int B, int Hq,
    int Hkv, int d, int F, T *__restrict__ O, unsigned *err)
{
    extern __shared__ float smem[];
    const int P2 = 2 * F;
    float *Ks = smem;                       // [B][d+1]
    float *Vs = Ks + B * (d + 1);           // [B][d]
    float *qs = Vs + B * d;                 // [RT][d]
    float *phis = qs + kRT * d;             // [RT][2F]
    float *ps = phis + kRT * P2;            // [RT][B]
    float *St = ps + kRT * B;               // [d][33] one S tile, feature-contiguous
    float *row_m = St + d * 33;             // [RT]
    float *row_l = row_m + kRT;             // [RT]
    float *row_ld = row_l + kRT;            // [RT]

    const int n_tiles_rows = (B + kRT - 1) / kRT;
    const int r = blockIdx.x / (Hq * n_tiles_rows);
    const int rem = blockIdx.x % (Hq * n_tiles_rows);
    const int h = rem / n_tiles_rows;
    const int i0 = (rem % n_tiles_rows) * kRT;
    const int G = Hq / Hkv, g = h / G;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int rows = min(kRT, B - i0);

    const float *state = reinterpret_cast<const float *>(states[r]);
    if (!state_ptr_ok(state)) {
        if (tid == 0) raise_error(err, ERR_BAD_STATE_PTR);
        return;
    }
    const float *Sg = state + (size_t)g * head_floats(d, F);
    const float *zg = Sg + (size_t)P2 * d;

    // active-block keys/values of state head g, queries of head h
    for (int idx = tid; idx < B * d; idx += kGenThreads) {
        const int j = idx / d, e = idx % d;
        const size_t src = (((size_t)r * B + j) * Hkv + g) * d + e;
        Ks[j * (d + 1) + e] = to_f32(K[src]);
        Vs[j * d + e] = to_f32(V[src]);
    }
    for (int idx = tid; idx < kRT * d; idx += kGenThreads) {
        const int i = idx / d, e = idx % d;
        qs[idx] = (i < rows) ? to_f32(Q[(((size_t)r * B + i0 + i) * Hq + h) * d + e]) : 0.f;
    }
    __syncthreads();

    const T *Wg = W + (size_t)g * d * F;
    const float inv_sqrt_d = rsqrtf((float)d);
    for (int ii = 0; ii < 2; ++ii) {
        const int i = warp * 2 + ii;
        // phi(q_i)
        float pos[kMaxFWarp], neg[kMaxFWarp];
        warp_phi_row<T>(qs + i * d, Wg, d, F, pos, neg);
#pragma unroll
        for (int k = 0; k < kMaxFWarp; ++k) {
            const int f = lane + 32 * k;
            if (f < F) { phis[i * P2 + f] = pos[k]; phis[i * P2 + F + f] = neg[k]; }
        }
        // in-block scores s_ij = q_i . k_j / sqrt(d), every j (no mask)
        float m = -INFINITY;
        for (int j = lane; j < B; j += 32) {
            float s = 0.f;
            for (int e = 0; e < d; ++e) s = fmaf(qs[i * d + e], Ks[j * (d + 1) + e], s);
            s *= inv_sqrt_d;
            ps[i * B + j] = s;
            m = fmaxf(m, s);
        }
        m = warp_max(m);
        float l = 0.f;
        for (int j = lane; j < B; j += 32) {
            const float p = expf(ps[i * B + j] - m);
            ps[i * B + j] = p;
            l += p;
        }
        l = warp_sum(l);
        __syncwarp();
        // lin_den = phi(q_i) . z
        float ld = 0.f;
        for (int f = lane; f < P2; f += 32) ld = fmaf(phis[i * P2 + f], zg[f], ld);
        ld = warp_sum(ld);
        if (lane == 0) { row_m[i] = m; row_l[i] = l; row_ld[i] = ld; }
    }
    __syncthreads();

    // numerators: warp owns rows 2w, 2w+1; lane owns e = lane + 32 k
    constexpr int kMaxE = 4;   // d <= 128
    float acc_s[2][kMaxE], acc_l[2][kMaxE];
#pragma unroll
    for (int ii = 0; ii < 2; ++ii)
#pragma unroll
        for (int k = 0; k < kMaxE; ++k) { acc_s[ii][k] = 0.f; acc_l[ii][k] = 0.f; }
    const int nE = d / 32;
    for (int j = 0; j < B; ++j) {
        const float p0 = ps[(warp * 2) * B + j], p1 = ps[(warp * 2 + 1) * B + j];
#pragma unroll
        for (int k = 0; k < kMaxE; ++k) {
            if (k < nE) {
                const float v = Vs[j * d + lane + 32 * k];
                acc_s[0][k] = fmaf(p0, v, acc_s[0][k]);
                acc_s[1][k] = fmaf(p1, v, acc_s[1][k]);
            }
        }
    }
    // linear readout lin_num = phi(q)^T S, one S tile (32 features) at a time
    const int n_tiles = P2 / 32;
    for (int t = 0; t < n_tiles; ++t) {
        __syncthreads();
        const float4 *src = reinterpret_cast<const float4 *>(Sg + (size_t)t * 32 * d);
        for (int p = tid; p < 8 * d; p += kGenThreads) {
            int e, f0;
            granule_coords(p, 0, e, f0);
            const float4 v = src[p];
            float *dst = St + e * 33 + f0;
            dst[0] = v.x; dst[1] = v.y; dst[2] = v.z; dst[3] = v.w;
        }
        __syncthreads();
        for (int fl = 0; fl < 32; ++fl) {
            const float a0 = phis[(warp * 2) * P2 + t * 32 + fl];
            const float a1 = phis[(warp * 2 + 1) * P2 + t * 32 + fl];
#pragma unroll
            for (int k = 0; k < kMaxE; ++k) {
                if (k < nE) {
                    const float s = St[(lane + 32 * k) * 33 + fl];
                    acc_l[0][k] = fmaf(a0, s, acc_l[0][k]);
                    acc_l[1][k] = fmaf(a1, s, acc_l[1][k]);
                }
            }
        }
    }

    // gated shared-normaliser merge and store
    const float lw = log_sigmoid(alpha[h]);
#pragma unroll
    for (int ii = 0; ii < 2; ++ii) {
        const int i = warp * 2 + ii;
        if (i >= rows) continue;
        const MergeWeights mw = merge_weights(lw, row_m[i], row_l[i], row_ld[i]);
        T *o = O + (((size_t)r * B + i0 + i) * Hq + h) * d;
#pragma unroll
        for (int k = 0; k < kMaxE; ++k) {
            if (k < nE) {
                const float val = mw.ws * acc_s[ii][k] + (mw.wl == 0.f ? 0.f : mw.wl * acc_l[ii][k]);
                o[lane + 32 * k] = from_f32<T>(val);
            }
        }
    }
}

// ---------------------------------------------------------------------------
// Commit, generic: one CTA per (request, state head, group of TPC S tiles).
// Each CTA folds every token into its own tiles; phi(k_t) is recomputed per
// CTA (only this CTA's features are kept).  Accumulation runs in registers in
// token order and the state is read-modified-written once.
// ---------------------------------------------------------------------------
constexpr int kTC = 32;            // tokens per smem chunk
constexpr int kComThreads = 256;

size_t generic_commit_smem_bytes(int d, int F)
{
    const int tpc = (d == 64) ? 4 : 2;
    const int nt = (2 * F) / 32;
    const int tiles = tpc < nt ? tpc : nt;
    const size_t fl = (size_t)kTC * d /*ks*/ + (size_t)kTC * d /*vs*/ + (size_t)kTC * tiles * 32;
    return fl * sizeof(float);
}

int generic_commit_tiles_per_cta(int d, int F)
{
    const int tpc = (d == 64) ? 4 : 2;
    const int nt = (2 * F) / 32;
    return tpc < nt ? tpc : nt;
}

template <typename T>
__global__ void __launch_bounds__(kComThreads) k_commit_generic(
    const T *__restrict__ K, const T *__restrict__ V, int n_tok, const T *__restrict__ W,
    void *const *__restrict__ states, int n_req, int Hkv, int d, int F, int tpc, unsigned *err)
{
    extern __shared__ float smem[];
    const int P2 = 2 * F;
    const int n_tiles = P2 / 32;
    const int n_groups = (n_tiles + tpc - 1) / tpc;
    const int r = blockIdx.x / (Hkv * n_groups);
    const int g = (blockIdx.x / n_groups) % Hkv;
    const int tile0 = (blockIdx.x % n_groups) * tpc;
    const int tiles = min(tpc, n_tiles - tile0);
    const int f_lo = tile0 * 32, nf = tiles * 32;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;

    float *ks = smem;                 // [TC][d]
    float *vs = ks + kTC * d;         // [TC][d]
    float *ph = vs + kTC * d;         // [TC][nf]   phi features f_lo .. f_lo+nf-1

    float *state = reinterpret_cast<float *>(states[r]);
    if (!state_ptr_ok(state)) {
        if (tid == 0) raise_error(err, ERR_BAD_STATE_PTR);
        return;
    }
    float *Sg = state + (size_t)g * head_floats(d, F);
    const T *Wg = W + (size_t)g * d * F;

    // this thread's granules: p = tid + 256 k over tiles x d rows x 8 granules
    const int n_gran = tiles * d * 8;
    constexpr int kMaxG = 8;          // tiles*d*8/256 <= 8 (tpc = 256/d)
    float4 acc[kMaxG];
    int g_e[kMaxG], g_f[kMaxG];
#pragma unroll
    for (int k = 0; k < kMaxG; ++k) {
        acc[k] = make_float4(0.f, 0.f, 0.f, 0.f);
        const int p = tid + kComThreads * k;
        if (p < n_gran) {
            int e, f0;
            granule_coords(p % (8 * d), tile0 + p / (8 * d), e, f0);
            g_e[k] = e;
            g_f[k] = f0 - f_lo;
        } else {
            g_e[k] = 0;
            g_f[k] = -1;
        }
    }
    float dz = 0.f;   // z increment of feature f_lo + tid (tid < nf)

    for (int t0 = 0; t0 < n_tok; t0 += kTC) {
        const int tc = min(kTC, n_tok - t0);
        __syncthreads();
        for (int idx = tid; idx < kTC * d; idx += kComThreads) {
            const int t = idx / d, e = idx % d;
            float kv = 0.f, vv = 0.f;
            if (t < tc) {
                const size_t src = (((size_t)r * n_tok + t0 + t) * Hkv + g) * d + e;
                kv = to_f32(K[src]);
                vv = to_f32(V[src]);
            }
            ks[idx] = kv;
            vs[idx] = vv;
        }
        __syncthreads();
        for (int t = warp; t < kTC; t += kComThreads / 32) {
            float pos[kMaxFWarp], neg[kMaxFWarp];
            if (t < tc) {
                warp_phi_row<T>(ks + t * d, Wg, d, F, pos, neg);
            } else {
#pragma unroll
                for (int k = 0; k < kMaxFWarp; ++k) { pos[k] = 0.f; neg[k] = 0.f; }
            }
#pragma unroll
            for (int k = 0; k < kMaxFWarp; ++k) {
                const int f = lane + 32 * k;
                if (f < F) {
                    if (f >= f_lo && f < f_lo + nf) ph[t * nf + f - f_lo] = pos[k];
                    if (F + f >= f_lo && F + f < f_lo + nf) ph[t * nf + F + f - f_lo] = neg[k];
                }
            }
        }
        __syncthreads();
        for (int t = 0; t < tc; ++t) {
#pragma unroll
            for (int k = 0; k < kMaxG; ++k) {
                if (g_f[k] >= 0) {
                    const float v = vs[t * d + g_e[k]];
                    const float4 p = *reinterpret_cast<const float4 *>(ph + t * nf + g_f[k]);
                    acc[k].x = fmaf(p.x, v, acc[k].x);
                    acc[k].y = fmaf(p.y, v, acc[k].y);
                    acc[k].z = fmaf(p.z, v, acc[k].z);
                    acc[k].w = fmaf(p.w, v, acc[k].w);
                }
            }
            if (tid < nf) dz += ph[t * nf + tid];
        }
    }

    // read-modify-write this CTA's tiles and z entries
    float4 *dst = reinterpret_cast<float4 *>(Sg + (size_t)tile0 * 32 * d);
#pragma unroll
    for (int k = 0; k < kMaxG; ++k) {
        if (g_f[k] >= 0) {
            const int p = tid + kComThreads * k;
            float4 s = dst[p];
            s.x += acc[k].x; s.y += acc[k].y; s.z += acc[k].z; s.w += acc[k].w;
            dst[p] = s;
        }
    }
    if (tid < nf) Sg[z_offset(f_lo + tid, d, F)] += dz;
}

// ---------------------------------------------------------------------------
// host-side launchers
// ---------------------------------------------------------------------------
template <typename T>
cudaError_t launch_feature_map_t(const void *X, int n_rows, int nh, int Hkv, int d, int F,
                                 const void *W, float *Phi, cudaStream_t st)
{
    const long long items = (long long)n_rows * nh;
    if (items == 0) return cudaSuccess;
    const int warps = 8;
    const long long blocks = (items + warps - 1) / warps;
    k_feature_map<T><<<(unsigned)blocks, warps * 32, warps * d * sizeof(float), st>>>(
        (const T *)X, n_rows, nh, nh / Hkv, d, F, (const T *)W, Phi);
    return cudaGetLastError();
}

cudaError_t launch_feature_map(hybrid_dtype dt, const void *X, int n_rows, int nh, int Hkv, int d,
                               int F, const void *W, float *Phi, cudaStream_t st)
{
    if (dt == HYBRID_F32) return launch_feature_map_t<float>(X, n_rows, nh, Hkv, d, F, W, Phi, st);
    return launch_feature_map_t<__nv_bfloat16>(X, n_rows, nh, Hkv, d, F, W, Phi, st);
}

template <typename T>
cudaError_t launch_attn_generic_t(const hybrid_cfg &c, const void *Q, const void *K, const void *V,
                                  const void *W, const float *alpha, void *const *states, int n_req,
                                  void *O, unsigned *err, cudaStream_t st)
{
    const int d = c.head_dim, F = c.feat_dim, B = c.block_size;
    const size_t smem = generic_attn_smem_bytes(d, F, B);
    cudaError_t e = cudaFuncSetAttribute(k_attn_generic<T>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)smem);
    if (e != cudaSuccess) return e;
    const long long blocks = (long long)n_req * c.n_q_heads * ((B + kRT - 1) / kRT);
    k_attn_generic<T><<<(unsigned)blocks, kGenThreads, smem, st>>>(
        (const T *)Q, (const T *)K, (const T *)V, (const T *)W, alpha, states, n_req, B, c.n_q_heads,
        c.n_kv_heads, d, F, (T *)O, err);
    return cudaGetLastError();
}

cudaError_t launch_attn_generic(const hybrid_cfg &c, const void *Q, const void *K, const void *V,
                                const void *W, const float *alpha, void *const *states, int n_req,
                                void *O, unsigned *err, cudaStream_t st)
{
    if (c.io_dtype == HYBRID_F32)
        return launch_attn_generic_t<float>(c, Q, K, V, W, alpha, states, n_req, O, err, st);
    return launch_attn_generic_t<__nv_bfloat16>(c, Q, K, V, W, alpha, states, n_req, O, err, st);
}

template <typename T>
cudaError_t launch_commit_generic_t(const hybrid_cfg &c, const void *K, const void *V, int n_tok,
                                    const void *W, void *const *states, int n_req, unsigned *err,
                                    cudaStream_t st)
{
    const int d = c.head_dim, F = c.feat_dim;
    const int tpc = generic_commit_tiles_per_cta(d, F);
    const int n_groups = ((2 * F) / 32 + tpc - 1) / tpc;
    const size_t smem = generic_commit_smem_bytes(d, F);
    cudaError_t e = cudaFuncSetAttribute(k_commit_generic<T>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    const long long blocks = (long long)n_req * c.n_kv_heads * n_groups;
    k_commit_generic<T><<<(unsigned)blocks, kComThreads, smem, st>>>(
        (const T *)K, (const T *)V, n_tok, (const T *)W, states, n_req, c.n_kv_heads, d, F, tpc, err);
    return cudaGetLastError();
}

cudaError_t launch_commit_generic(const hybrid_cfg &c, const void *K, const void *V, int n_tok,
                                  const void *W, void *const *states, int n_req, unsigned *err,
                                  cudaStream_t st)
{
    if (c.io_dtype == HYBRID_F32)
        return launch_commit_generic_t<float>(c, K, V, n_tok, W, states, n_req, err, st);
    return launch_commit_generic_t<__nv_bfloat16>(c, K, V, n_tok, W, states, n_req, err, st);
}

}  // namespace hyb
