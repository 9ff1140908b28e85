// hybrid_tc_commit.cu -- the block commit of Section 3.1 of "Retrofitting
// Linear Attention into Diffusion Language Models" on the tensor cores:
//     S_g += sum_t phi(k_t) v_t^T,    z_g += sum_t phi(k_t).
//
// One CTA per (request r, state head g); tokens in chunks of 32.
//   U^T   = W_g^T K^T          bf16 x bf16 -> f32 (TMEM lanes = features f, columns = tokens t)
//   phi   : per token t, softmax over f of U^T[:, t] and of -U^T[:, t]
//           (cross-lane reductions; each thread then owns the phi^T row of its feature)
//   dS^T  = V^T phi^T           tf32 x tf32 -> f32 (TMEM lanes = e, columns = f)
// The state (already in the swizzled tile image) is bulk-copied into shared
// memory at the start, updated in place row by row from TMEM, and bulk-copied
// back; each state element is read and written exactly once.
#include "hybrid_common.cuh"
#include "hybrid_tc.h"
#include "tc_ptx.cuh"

namespace hyb {

namespace {

constexpr int kThreads = 256;
constexpr int kTok = 32;                      // tokens per chunk (one 128-byte tf32 row)
constexpr uint32_t kColU = 0;                 // U^T: 32 token columns per 128 features (2 blocks for F=256)
constexpr uint32_t kColD = 256;               // dS^T: 2F columns (2F <= 256)
constexpr uint64_t kWaitNs = 1000000000ull;
constexpr float kLog2e = 1.4426950408889634f;
constexpr int kSmemLimit = 232448;
constexpr int kOneCtaPerSm = 118 * 1024;

struct CommitArgs {
    const __nv_bfloat16 *K, *V, *W;
    void *const *states;
    unsigned *err;
    int T, Hkv, d, F;
    uint32_t off_s, off_w, off_k, off_vt, off_pt, off_z, off_red, off_bar;
};

struct CLayout {
    uint32_t off_s, off_w, off_k, off_vt, off_pt, off_z, off_red, off_bar, bytes;
};

CLayout make_clayout(int d, int F)
{
    CLayout L{};
    uint32_t off = 0;
    const int Fp = F < 128 ? 128 : F;    // W region sized for M = 128 feature rows
    L.off_s = off; off += (uint32_t)2 * F * d * 4;
    L.off_w = off; off += (uint32_t)d * Fp * 2;
    L.off_k = off; off += (uint32_t)kTok * d * 2;
    L.off_vt = off; off += 128u * 128;                  // V^T: 128 rows (e, padded) x 32 tokens f32
    L.off_pt = off; off += (uint32_t)2 * F * 128;       // phi^T: 2F rows x 32 tokens f32
    L.off_z = off; off += (((uint32_t)2 * F * 4) + 1023) & ~1023u;
    L.off_red = off; off += 8u * 4 * 32 * 4 + 1024;     // cross-warp reductions [8][4][32] + dz
    L.off_bar = off; off += 1024;
    L.bytes = off + 1024;
    if ((int)L.bytes < kOneCtaPerSm) L.bytes = kOneCtaPerSm;
    return L;
}

__device__ __forceinline__ float ex2(float x)
{
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

__global__ void __launch_bounds__(kThreads, 1) k_commit_tc(const __grid_constant__ CommitArgs a)
{
    using namespace ptx;
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int r = blockIdx.x / a.Hkv, g = blockIdx.x % a.Hkv;
    const int d = a.d, F = a.F, T = a.T;
    const int P2 = 2 * F, NC = P2 / 32;
    const uint32_t chunk_bytes = (uint32_t)d * 128;

    float *state = reinterpret_cast<float *>(a.states[r]);
    if (!state_ptr_ok(state)) {
        if (tid == 0) raise_error(a.err, ERR_BAD_STATE_PTR);
        return;
    }
    float *Sg = state + (size_t)g * head_floats(d, F);
    float *zg = Sg + (size_t)P2 * d;

    uint64_t *bar_s = reinterpret_cast<uint64_t *>(smem + a.off_bar);
    uint64_t *bar_u = bar_s + 1;
    uint64_t *bar_m = bar_s + 2;
    uint32_t *tmem_holder = reinterpret_cast<uint32_t *>(bar_s + 3);
    int *fail = reinterpret_cast<int *>(tmem_holder + 1);
    float *red = reinterpret_cast<float *>(smem + a.off_red);   // [8 slots][4 warps][32 tokens]
    float *dzs = red + 8 * 4 * 32;                              // [2F]

    if (tid == 0) {
        mbar_init(bar_s, 1);
        mbar_init(bar_u, 1);
        mbar_init(bar_m, 1);
        *fail = 0;
        fence_mbar_init();
    }
    if (warp == 0) {
        tmem_alloc(tmem_holder, 512);
        tmem_relinquish();
    }
    for (int f = tid; f < P2; f += kThreads) dzs[f] = 0.f;
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_holder;

    // the whole state head (S tiles, then z) in one transaction group
    if (tid == 0) {
        mbar_arrive_expect_tx(bar_s, (uint32_t)P2 * d * 4 + (uint32_t)P2 * 4);
        for (int c = 0; c < NC; ++c)
            bulk_g2s(smem + a.off_s + (size_t)c * chunk_bytes, Sg + (size_t)c * 32 * d, chunk_bytes, bar_s);
        bulk_g2s(smem + a.off_z, zg, (uint32_t)P2 * 4, bar_s);
    }
    // W_g as the MN-major operand [e][f]
    {
        const int gw = F / 8;
        const int natoms = F < 128 ? 2 : F / 64;   // M = 128 rows even for F = 64
        for (int idx = tid; idx < d * gw; idx += kThreads) {
            const int e = idx / gw, c = idx % gw;
            cp_async16(smem + a.off_w + (e >> 3) * (natoms * 1024) + (c >> 3) * 1024 + (e & 7) * 128 +
                           (((c & 7) ^ (e & 7)) << 4),
                       a.W + ((size_t)g * d + e) * F + 8 * c);
        }
    }

    const int q4 = warp & 3, th = warp >> 2;     // th: which 16 tokens of the chunk
    const int nfb = F > 128 ? 2 : 1;             // 128-feature blocks of U^T
    const int natoms_w = F < 128 ? 2 : F / 64;
    float dzp[2] = {0.f, 0.f}, dzn[2] = {0.f, 0.f};
    int n_chunks = (T + kTok - 1) / kTok;

    for (int ch = 0; ch < n_chunks; ++ch) {
        const int t0 = ch * kTok;
        const int tv = min(kTok, T - t0);
        if (ch > 0) {
            // the previous chunk's dS MMA must be done reading K, V^T and phi^T
            if (!mbar_wait(bar_m, (uint32_t)(ch - 1) & 1u, kWaitNs)) atomicOr(fail, 1);
            tc_fence_after();
        }
        // K chunk: K-major [t][e]; rows beyond T are zero
        {
            const int gpr = d / 8;
            for (int idx = tid; idx < kTok * gpr; idx += kThreads) {
                const int t = idx / gpr, c = idx % gpr;
                uint8_t *dst = smem + a.off_k + (c >> 3) * (kTok * 128) + t * 128 + (((c & 7) ^ (t & 7)) << 4);
                if (t < tv)
                    cp_async16(dst, a.K + (((size_t)r * T + t0 + t) * a.Hkv + g) * d + 8 * c);
                else
                    *reinterpret_cast<uint4 *>(dst) = make_uint4(0, 0, 0, 0);
            }
            // V^T in f32: row e, column t (K-major, 128-byte swizzle); zero for t >= tv and e >= d
            for (int idx = tid; idx < 16 * kTok; idx += kThreads) {
                const int ec = idx / kTok, t = idx % kTok;    // ec: 8-wide group of e
                float v[8];
                if (t < tv && ec * 8 < d) {
                    const uint4 raw = *reinterpret_cast<const uint4 *>(
                        a.V + (((size_t)r * T + t0 + t) * a.Hkv + g) * d + 8 * ec);
                    const __nv_bfloat162 *b2 = reinterpret_cast<const __nv_bfloat162 *>(&raw);
#pragma unroll
                    for (int i = 0; i < 4; ++i) { v[2 * i] = __low2float(b2[i]); v[2 * i + 1] = __high2float(b2[i]); }
                } else {
#pragma unroll
                    for (int i = 0; i < 8; ++i) v[i] = 0.f;
                }
#pragma unroll
                for (int i = 0; i < 8; ++i) {
                    const int e = ec * 8 + i;
                    float *dst = reinterpret_cast<float *>(smem + a.off_vt + e * 128 + ((((t >> 2) ^ (e & 7))) << 4)) + (t & 3);
                    *dst = v[i];
                }
            }
        }
        cp_async_wait_all();
        fence_proxy_async_smem();
        __syncthreads();

        // U^T = W^T K^T: M = 128 features per block, N = 32 tokens, K = d
        if (tid == 0) {
            tc_fence_after();
            const uint32_t w_u = smem_u32(smem + a.off_w), k_u = smem_u32(smem + a.off_k);
            const uint32_t idU = instr_desc(FMT_BF16, FMT_BF16, true, false, 128, kTok);
            for (int fb = 0; fb < nfb; ++fb) {
                for (int k = 0; k < d / 16; ++k) {
                    const uint64_t ad = smem_desc(w_u + fb * 2 * 1024 + 2 * k * (natoms_w * 1024), 1024,
                                                  natoms_w * 1024, SWZ_128B);
                    const uint64_t bd = smem_desc(k_u + (k >> 2) * (kTok * 128) + (k & 3) * 32, 16, 1024, SWZ_128B);
                    mma_bf16_ss(tmem + kColU + fb * kTok, ad, bd, idU, k > 0);
                }
            }
            mma_commit(bar_u);
        }
        if (!mbar_wait(bar_u, (uint32_t)ch & 1u, kWaitNs)) atomicOr(fail, 1);
        tc_fence_after();

        // phi for 16 tokens per thread group; thread = feature (lane) of block fb
        const uint32_t lane_off = (uint32_t)(32 * q4) << 16;
        float u[2][16];
        for (int fb = 0; fb < nfb; ++fb) {
            tmem_ld16(tmem + lane_off + kColU + fb * kTok + 16 * th, u[fb]);
        }
        tmem_wait_ld();
        const int fbase = 32 * q4 + lane;
        float mx[16], mn[16];
#pragma unroll
        for (int i = 0; i < 16; ++i) { mx[i] = -INFINITY; mn[i] = INFINITY; }
        for (int fb = 0; fb < nfb; ++fb) {
            if (fb * 128 + fbase < F) {
#pragma unroll
                for (int i = 0; i < 16; ++i) { mx[i] = fmaxf(mx[i], u[fb][i]); mn[i] = fminf(mn[i], u[fb][i]); }
            }
        }
#pragma unroll
        for (int i = 0; i < 16; ++i) { mx[i] = warp_max(mx[i]); mn[i] = warp_min(mn[i]); }
        if (lane < 16) {
            // lane i publishes token i of this warp's half
            float vmx = mx[0], vmn = mn[0];
#pragma unroll
            for (int i = 1; i < 16; ++i) if (lane == i) { vmx = mx[i]; vmn = mn[i]; }
            red[(0 * 4 + q4) * 32 + 16 * th + lane] = vmx;
            red[(1 * 4 + q4) * 32 + 16 * th + lane] = vmn;
        }
        __syncthreads();
#pragma unroll
        for (int i = 0; i < 16; ++i) {
            const int t = 16 * th + i;
            mx[i] = fmaxf(fmaxf(red[(0 * 4 + 0) * 32 + t], red[(0 * 4 + 1) * 32 + t]),
                          fmaxf(red[(0 * 4 + 2) * 32 + t], red[(0 * 4 + 3) * 32 + t]));
            mn[i] = fminf(fminf(red[(1 * 4 + 0) * 32 + t], red[(1 * 4 + 1) * 32 + t]),
                          fminf(red[(1 * 4 + 2) * 32 + t], red[(1 * 4 + 3) * 32 + t]));
        }
        float ep[2][16], en[2][16], sp[16], sn[16];
#pragma unroll
        for (int i = 0; i < 16; ++i) { sp[i] = 0.f; sn[i] = 0.f; }
        for (int fb = 0; fb < nfb; ++fb) {
            const bool fv = fb * 128 + fbase < F;
#pragma unroll
            for (int i = 0; i < 16; ++i) {
                ep[fb][i] = fv ? ex2((u[fb][i] - mx[i]) * kLog2e) : 0.f;
                en[fb][i] = fv ? ex2((mn[i] - u[fb][i]) * kLog2e) : 0.f;
                sp[i] += ep[fb][i];
                sn[i] += en[fb][i];
            }
        }
#pragma unroll
        for (int i = 0; i < 16; ++i) { sp[i] = warp_sum(sp[i]); sn[i] = warp_sum(sn[i]); }
        if (lane < 16) {
            float vsp = sp[0], vsn = sn[0];
#pragma unroll
            for (int i = 1; i < 16; ++i) if (lane == i) { vsp = sp[i]; vsn = sn[i]; }
            red[(2 * 4 + q4) * 32 + 16 * th + lane] = vsp;
            red[(3 * 4 + q4) * 32 + 16 * th + lane] = vsn;
        }
        __syncthreads();
        // phi^T rows: feature f (phi+) and F + f (phi-), columns = tokens
        for (int fb = 0; fb < nfb; ++fb) {
            const int f = fb * 128 + fbase;
            if (f >= F) continue;
            float pp[16], pn[16];
#pragma unroll
            for (int i = 0; i < 16; ++i) {
                const int t = 16 * th + i;
                const float tsp = red[(2 * 4 + 0) * 32 + t] + red[(2 * 4 + 1) * 32 + t] +
                                  red[(2 * 4 + 2) * 32 + t] + red[(2 * 4 + 3) * 32 + t];
                const float tsn = red[(3 * 4 + 0) * 32 + t] + red[(3 * 4 + 1) * 32 + t] +
                                  red[(3 * 4 + 2) * 32 + t] + red[(3 * 4 + 3) * 32 + t];
                const bool tvld = t < tv;
                pp[i] = tvld ? ep[fb][i] / tsp : 0.f;
                pn[i] = tvld ? en[fb][i] / tsn : 0.f;
                dzp[fb] += pp[i];
                dzn[fb] += pn[i];
            }
            uint8_t *rp = smem + a.off_pt + f * 128;
            uint8_t *rn = smem + a.off_pt + (F + f) * 128;
#pragma unroll
            for (int gq = 0; gq < 4; ++gq) {
                const int gidx = 4 * th + gq;   // 16-byte granule of the 128-byte row
                *reinterpret_cast<float4 *>(rp + ((gidx ^ (f & 7)) << 4)) =
                    make_float4(pp[4 * gq], pp[4 * gq + 1], pp[4 * gq + 2], pp[4 * gq + 3]);
                *reinterpret_cast<float4 *>(rn + ((gidx ^ ((F + f) & 7)) << 4)) =
                    make_float4(pn[4 * gq], pn[4 * gq + 1], pn[4 * gq + 2], pn[4 * gq + 3]);
            }
        }
        fence_proxy_async_smem();
        tc_fence_before();
        __syncthreads();

        // dS^T += V^T phi^T: M = 128 (e), N = 2F, K = 32 tokens
        if (tid == 0) {
            tc_fence_after();
            const uint32_t v_u = smem_u32(smem + a.off_vt), p_u = smem_u32(smem + a.off_pt);
            const uint32_t idD = instr_desc(FMT_TF32, FMT_TF32, false, false, 128, P2);
#pragma unroll
            for (int kk = 0; kk < 4; ++kk)
                mma_tf32_ss(tmem + kColD, smem_desc(v_u + 32 * kk, 16, 1024, SWZ_128B),
                            smem_desc(p_u + 32 * kk, 16, 1024, SWZ_128B), idD, (ch | kk) != 0);
            mma_commit(bar_m);
        }
    }

    // z increments: two token halves per feature
    for (int fb = 0; fb < nfb; ++fb) {
        const int f = fb * 128 + 32 * q4 + lane;
        if (f < F) {
            atomicAdd(&dzs[f], dzp[fb]);
            atomicAdd(&dzs[F + f], dzn[fb]);
        }
    }
    if (!mbar_wait(bar_m, (uint32_t)(n_chunks - 1) & 1u, kWaitNs)) atomicOr(fail, 1);
    if (!mbar_wait(bar_s, 0, kWaitNs)) atomicOr(fail, 1);
    tc_fence_after();
    __syncthreads();
    const bool failed = *fail != 0;

    // S^T tile rows += dS^T rows (thread = row e; two thread groups split the tiles)
    if (!failed) {
        const int e = 32 * q4 + lane;
        const uint32_t lane_off = (uint32_t)(32 * q4) << 16;
        for (int c = th; c < NC; c += 2) {
            float v[32];
            tmem_ld32(tmem + lane_off + kColD + 32 * c, v);
            tmem_wait_ld();
            if (e < d) {
                uint8_t *rowp = smem + a.off_s + (size_t)c * chunk_bytes + e * 128;
#pragma unroll
                for (int j = 0; j < 8; ++j) {
                    float4 *p = reinterpret_cast<float4 *>(rowp + ((j ^ (e & 7)) << 4));
                    float4 s = *p;
                    s.x += v[4 * j]; s.y += v[4 * j + 1]; s.z += v[4 * j + 2]; s.w += v[4 * j + 3];
                    *p = s;
                }
            }
        }
        float *zs = reinterpret_cast<float *>(smem + a.off_z);
        for (int f = tid; f < P2; f += kThreads) zs[f] += dzs[f];
    }
    fence_proxy_async_smem();
    tc_fence_before();
    __syncthreads();
    if (tid == 0) {
        if (!failed) {
            for (int c = 0; c < NC; ++c)
                bulk_s2g(Sg + (size_t)c * 32 * d, smem + a.off_s + (size_t)c * chunk_bytes, chunk_bytes);
            bulk_s2g(zg, smem + a.off_z, (uint32_t)P2 * 4);
            bulk_commit();
            bulk_wait_all();
        } else {
            raise_error(a.err, ERR_WAIT_TIMEOUT);
        }
    }
    __syncthreads();
    if (warp == 0) {
        tc_fence_after();
        tmem_dealloc(tmem, 512);
    }
}

}  // namespace

bool tc_commit_supported(const hybrid_cfg &c)
{
    if (c.io_dtype != HYBRID_BF16) return false;
    if (c.head_dim != 64 && c.head_dim != 128) return false;
    if (c.feat_dim != 64 && c.feat_dim != 128) return false;
    const CLayout L = make_clayout(c.head_dim, c.feat_dim);
    return (int)L.bytes <= kSmemLimit;
}

cudaError_t launch_commit_tc(const hybrid_cfg &c, const void *K, const void *V, int n_tok, const void *W,
                             void *const *states, int n_req, unsigned *err, cudaStream_t st)
{
    const CLayout L = make_clayout(c.head_dim, c.feat_dim);
    CommitArgs a;
    a.K = static_cast<const __nv_bfloat16 *>(K);
    a.V = static_cast<const __nv_bfloat16 *>(V);
    a.W = static_cast<const __nv_bfloat16 *>(W);
    a.states = states;
    a.err = err;
    a.T = n_tok;
    a.Hkv = c.n_kv_heads;
    a.d = c.head_dim;
    a.F = c.feat_dim;
    a.off_s = L.off_s;
    a.off_w = L.off_w;
    a.off_k = L.off_k;
    a.off_vt = L.off_vt;
    a.off_pt = L.off_pt;
    a.off_z = L.off_z;
    a.off_red = L.off_red;
    a.off_bar = L.off_bar;
    cudaError_t e = cudaFuncSetAttribute(k_commit_tc, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)L.bytes);
    if (e != cudaSuccess) return e;
    k_commit_tc<<<(unsigned)((long long)n_req * c.n_kv_heads), kThreads, L.bytes, st>>>(a);
    return cudaGetLastError();
}

}  // namespace hyb
