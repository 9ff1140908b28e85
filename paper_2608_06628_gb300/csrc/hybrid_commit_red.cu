// hybrid_commit_red.cu -- block commit and prompt prefill (Section 3.1's state
// update S += sum_t phi(k_t) v_t^T, z += sum_t phi(k_t)) as a reduction: the
// increments are formed on the tensor cores for each (request, state head) and
// added into the state in global memory by bulk reduce-adds, which the L2 applies
// (one float32 add per element, as S + dS).  The state never passes through the
// SM, so the SM streams only K, V and W.
//
// Work unit = (request r, state head g) with T tokens, taken in chunks of 32
// token slots (the last chunk masked).  One CTA per SM walks a contiguous range
// of units.  Warp roles (12 warps):
//   warp 0      producer: W of the unit by TMA; per chunk V by TMA and K^T
//               (transposed by the warp from global K) into a two-chunk ring
//   warp 1      MMA issuer (one thread); owns the Tensor Memory allocation
//   warp 2      storer: bulk reduce-adds of the dS^T tiles and of dz
//   warps 4-11  math: phi(K) per chunk (thread = one feature of one half for the
//               chunk's 32 tokens), dz, and the dS^T tiles into a staging ring
// Per chunk the tensor cores form U_k^T = W^T K^T (features on TMEM lanes) and,
// once phi(K) is written, dS^T += V^T phi(K)^T for both feature halves, so dS^T
// accumulates over the unit's chunks in Tensor Memory:
//   [0,32) and [32,64)   U_k^T of the two chunk buffers
//   [256,256+F)          dS^T of phi+ features,  [384,384+F) of phi- features
// With F = 256 the two halves of dS^T (512 columns) do not fit: the unit is then
// taken in two passes, one per sign of the feature map, each re-forming U_k^T as
// two 128-feature tiles ([0,32) and [64,96) for buffer 0, +32 for buffer 1), with
// the math warps' two parts on the two feature tiles instead of the two signs,
// and dS^T of the pass's sign in [256,512).
#include <atomic>

#include "hybrid_common.cuh"
#include "hybrid_tc.h"
#include "tc_pipeline.cuh"

namespace hyb {

namespace {

using namespace pipe;

constexpr int kWarps = 12;
constexpr int kThreads = kWarps * 32;
constexpr int kMathThreads = 256;
constexpr int kChunk = 32;          // token slots per chunk
constexpr int kStage = 4;           // staging slots for dS^T tiles
constexpr uint32_t kBarMath = 1;
constexpr int kSmemLimit = 232448;
constexpr int kOneCtaPerSm = 118 * 1024;
constexpr uint32_t kColDSp = 256, kColDSm = 384;

struct CommitArgs {
    CUtensorMap tmV, tmW;   // V [n*T][Hkv][d], W [Hkv*d][F]; 128-byte swizzle, 64-element panels
                            // as the outermost box dimension (one copy for all of them)
    CUtensorMap tmK;        // K as V (used only to prefetch K into L2; K is read by the warps)
    const bf16 *K;
    void *const *states;
    unsigned *err;
    int n_units, T, Hkv, d, F;
    int n_pass;             // passes per (request, head): 1, or 2 for F = 256 (one per sign)
    uint32_t off_w, off_c, off_s, off_dz, off_tk, off_bar, chunk_stride;
};

// Shared memory: [W: 2 atoms of d rows][chunk ring x2: K^T atom | V | phi(K)]
// [staging x kStage: d rows x 128 B][dz][token stats][barriers].  W always has two
// atoms so that the M = 128 operand W^T stays inside the allocation for F = 64.
struct CLayout {
    uint32_t off_w, off_c, chunk, off_s, off_dz, off_tk, off_bar, bytes;
};

CLayout make_clayout(int d, int F)
{
    CLayout L{};
    const uint32_t atom = (uint32_t)d * 128;
    const uint32_t v = (uint32_t)(d / 64) * kChunk * 128;
    const int nf = F > 128 ? F : 2 * F;   // phi(K) features of one pass
    const uint32_t pk = (uint32_t)(nf / 64) * kChunk * 128;
    uint32_t off = 0;
    L.off_w = off; off += (uint32_t)(F / 64 > 2 ? F / 64 : 2) * atom;
    L.chunk = atom + v + pk;
    L.off_c = off; off += 2 * L.chunk;
    L.off_s = off; off += kStage * atom;
    L.off_dz = off; off += (((uint32_t)2 * F * 4) + 1023) & ~1023u;
    L.off_tk = off; off += 512 * 4;
    L.off_bar = off; off += 1024;
    L.bytes = off + 1024;
    if ((int)L.bytes < kOneCtaPerSm) L.bytes = kOneCtaPerSm;
    return L;
}

// unit u = pass (u % n_pass) of state head g of request r, (r, g) = (u / n_pass) / Hkv, % Hkv
// Ragged prompts: request r owns tokens [tok[r], tok[r + 1]) of the packed K and V;
// carried in the parameters.
struct CommitRaggedArgs : CommitArgs {
    int n_req;
    int tok[kMaxRaggedRequests + 1];
};
// tokens of unit u and the K/V row of its first token, uniform or ragged
__device__ __forceinline__ int unit_len(const CommitArgs &a, int) { return a.T; }
__device__ __forceinline__ long long unit_tok0(const CommitArgs &a, int u)
{
    return (long long)((u / a.n_pass) / a.Hkv) * a.T;
}
__device__ __forceinline__ int unit_len(const CommitRaggedArgs &a, int u)
{
    const int r = (u / a.n_pass) / a.Hkv;
    return a.tok[r + 1] - a.tok[r];
}
__device__ __forceinline__ long long unit_tok0(const CommitRaggedArgs &a, int u) { return a.tok[(u / a.n_pass) / a.Hkv]; }

__device__ __forceinline__ float *unit_head(const CommitArgs &a, int u)
{
    const int hu = u / a.n_pass;
    float *st = reinterpret_cast<float *>(a.states[hu / a.Hkv]);
    if (!state_ptr_ok(st)) return nullptr;
    return st + (size_t)(hu % a.Hkv) * head_floats(a.d, a.F);
}

template <class A>
__global__ void __launch_bounds__(kThreads, 1) k_commit_red(const __grid_constant__ A a)
{
    using namespace ptx;
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int d = a.d, F = a.F;
    const bool wide = a.n_pass > 1;       // F = 256: one sign per pass
    const int NH = F / 32;                 // dS^T tiles per half
    const int NCP = wide ? NH : 2 * NH;    // dS^T tiles per pass
    const uint32_t atom = (uint32_t)d * 128;
    const uint32_t vbytes = (uint32_t)(d / 64) * kChunk * 128;
    const int per = a.n_units / (int)gridDim.x, rem = a.n_units % (int)gridDim.x;
    const int u_begin = (int)blockIdx.x * per + min((int)blockIdx.x, rem);
    const int u_end = u_begin + per + ((int)blockIdx.x < rem ? 1 : 0);

    uint64_t *bars = reinterpret_cast<uint64_t *>(smem + a.off_bar);
    uint64_t *cfull = bars;            // [2] K^T and V of a chunk buffer are in place
    uint64_t *cfree = cfull + 2;       // [2] the chunk buffer has been consumed by the MMAs
    uint64_t *ukready = cfree + 2;     // [2] U_k^T of a chunk buffer is in Tensor Memory
    uint64_t *pkready = ukready + 2;   // [2] phi(K) of a chunk buffer is written
    uint64_t *sfull = pkready + 2;     // [kStage] a staging slot holds a dS^T tile
    uint64_t *sempty = sfull + kStage;
    uint64_t *wfull = sempty + kStage;
    uint64_t *wfree = wfull + 1;
    uint64_t *dsready = wfree + 1;     // the unit's dS^T is complete
    uint64_t *dsfree = dsready + 1;    // the math warps have staged the unit's dS^T
    uint64_t *dzready = dsfree + 1;
    uint64_t *dzfree = dzready + 1;
    uint64_t *mmadone = dzfree + 1;
    const int n_bars = 8 + 2 * kStage + 7;
    uint32_t *tmem_holder = reinterpret_cast<uint32_t *>(bars + n_bars);
    volatile int *fail = reinterpret_cast<volatile int *>(tmem_holder + 1);

    if (warp == 0 && lane == 0) {
        prefetch_tensormap(&a.tmV);
        prefetch_tensormap(&a.tmW);
    }
    if (tid == 0) {
        for (int i = 0; i < n_bars; ++i) mbar_init(&bars[i], 1);
        for (int b = 0; b < 2; ++b) {
            mbar_init(&cfull[b], 2);
            mbar_init(&pkready[b], 8);
        }
        for (int s = 0; s < kStage; ++s) mbar_init(&sfull[s], 4);   // the four warps of one part
        mbar_init(dsfree, 8);
        mbar_init(dzready, 8);
        *fail = 0;
        fence_mbar_init();
    }
    if (warp == 1) {
        tmem_alloc(tmem_holder, 512);
        tmem_relinquish();
    }
    __syncthreads();
    tc_fence_after();
    if (tid == 0) griddep_launch_dependents();
    // the first chunks of K and V of the CTA's first units into L2 while the previous kernel
    // drains: a prefetch brings no value into the SM, so it needs no ordering after it
    if (tid == 64)
        for (int u = u_begin; u < u_end && u < u_begin + 2; ++u) {
            const int Tu = unit_len(a, u), g = (u / a.n_pass) % a.Hkv;
            const int tok0 = (int)unit_tok0(a, u);
            for (int j = 0; j * kChunk < Tu && j < 2; ++j) {
                tma_prefetch_4d(&a.tmK, 0, g, tok0 + j * kChunk, 0);
                tma_prefetch_4d(&a.tmV, 0, g, tok0 + j * kChunk, 0);
            }
        }
    griddep_wait();
    const uint32_t tmem = *tmem_holder;
    uint8_t *wsm = smem + a.off_w;
    uint8_t *stage = smem + a.off_s;
    float *dzs = reinterpret_cast<float *>(smem + a.off_dz);

    if (warp == 0) {
        // ------------------------------------------------------------- producer
        uint32_t kp = 0, cc = 0;
        int nw = 0, nv = 0;
        bool ok = true;
        for (int u = u_begin; u < u_end && ok; ++u) {
            const int Tu = unit_len(a, u);   // a request without tokens has no work
            if (Tu == 0 || !unit_head(a, u)) continue;
            const int n_chunks = (Tu + kChunk - 1) / kChunk;
            const long long tok0 = unit_tok0(a, u);
            const int g = (u / a.n_pass) % a.Hkv;
            if (kp > 0) ok = wait_bar(wfree, (kp - 1) & 1u, fail);
            if (__any_sync(0xffffffffu, !ok)) break;
            if (lane == 0) {
                mbar_arrive_expect_tx(wfull, (uint32_t)(F / 64) * atom);
                tma_load_3d(wsm, &a.tmW, 0, g * d, 0, wfull);
            }
            ++nw;
            for (int j = 0; j < n_chunks; ++j, ++cc) {
                const int b = cc & 1;
                uint8_t *cb = smem + a.off_c + b * a.chunk_stride;
                KtRegs kr;
                kt_load(a.K, (size_t)tok0 + (size_t)j * kChunk, min(kChunk, Tu - j * kChunk), a.Hkv, g, d, kr, lane);
                ok = wait_bar(&cfree[b], ((cc >> 1) & 1u) ^ 1u, fail);
                if (__any_sync(0xffffffffu, !ok)) break;
                if (lane == 0) {
                    mbar_arrive_expect_tx(&cfull[b], vbytes);
                    tma_load_4d(cb + atom, &a.tmV, 0, g, (int)tok0 + j * kChunk, 0, &cfull[b]);
                }
                ++nv;
                kt_store(kr, d, cb, lane);
                fence_proxy_async_smem();
                __syncwarp();
                if (lane == 0) mbar_arrive(&cfull[b]);
            }
            ++kp;
        }
        if (lane == 0 && *fail) {
            if (nw) mbar_wait(wfull, (uint32_t)(nw - 1) & 1u, kWaitNs);
            if (nv) {
                for (int b = 0; b < 2; ++b) mbar_wait(&cfull[b], 0, 1000000ull);
            }
        }
    } else if (warp == 1) {
        // ------------------------------------------------------- MMA issuer
        if (lane == 0) {
            const uint32_t w_u = smem_u32(wsm), c_u = smem_u32(smem + a.off_c);
            const uint32_t idKT = instr_desc(FMT_BF16, FMT_BF16, true, true, 128, kChunk);
            const uint32_t idDS = instr_desc(FMT_BF16, FMT_BF16, true, true, 128, F);
            uint32_t kp = 0, cc = 0;
            bool ok = true;
            // U_k^T of chunk cc into buffer cc & 1 (F = 256: two 128-feature tiles)
            auto ukt = [&](uint32_t ci) {
                const uint32_t kt_u = c_u + (ci & 1) * a.chunk_stride;
                for (int t = 0; t < (wide ? 2 : 1); ++t)
                    for (int k = 0; k < d / 16; ++k) {
                        const uint64_t aw = smem_desc(w_u + 2 * t * atom + 2 * k * 1024, d * 128, 1024, SWZ_128B);
                        const uint64_t bk = smem_desc(kt_u + 2 * k * 1024, d * 128, 1024, SWZ_128B);
                        mma_bf16_ss(tmem + 32 * (ci & 1) + 64 * t, aw, bk, idKT, k > 0);
                    }
                mma_commit(&ukready[ci & 1]);
            };
            // dS^T (+)= V^T phi(K)^T of chunk ci for both halves
            auto dst = [&](uint32_t ci, bool first) {
                const uint32_t cb = c_u + (ci & 1) * a.chunk_stride;
                const uint32_t v_u = cb + atom, pk_u = cb + atom + vbytes;
                for (int h = 0; h < (wide ? 1 : 2); ++h)
                    for (int ks = 0; ks < kChunk / 16; ++ks) {
                        const uint64_t av = smem_desc(v_u + ks * 2048, kChunk * 128, 1024, SWZ_128B);
                        const uint64_t bp = smem_desc(pk_u + (uint32_t)h * (F / 64) * (kChunk * 128) + ks * 2048,
                                                      kChunk * 128, 1024, SWZ_128B);
                        mma_bf16_ss(tmem + (h == 0 ? kColDSp : kColDSm), av, bp, idDS, !(first && ks == 0));
                    }
                mma_commit(&cfree[ci & 1]);
            };
            for (int u = u_begin; u < u_end && ok; ++u) {
                const int Tu = unit_len(a, u);
                if (Tu == 0 || !unit_head(a, u)) continue;
                const int n_chunks = (Tu + kChunk - 1) / kChunk;
                if (!wait_bar(wfull, kp & 1u, fail)) { ok = false; break; }
                for (int j = 0; j <= n_chunks && ok; ++j) {
                    // U_k^T of chunk j ahead of dS^T of chunk j - 1 (its phi(K) is on the math warps)
                    if (j < n_chunks) {
                        const uint32_t ci = cc + j;
                        if (!wait_bar(&cfull[ci & 1], (ci >> 1) & 1u, fail)) { ok = false; break; }
                        tc_fence_after();
                        ukt(ci);
                    }
                    if (j >= 1) {
                        const uint32_t ci = cc + j - 1;
                        if (!wait_bar(&pkready[ci & 1], (ci >> 1) & 1u, fail)) { ok = false; break; }
                        // the previous unit's dS^T has been staged before it is overwritten
                        if (j == 1 && kp > 0 && !wait_bar(dsfree, (kp - 1) & 1u, fail)) { ok = false; break; }
                        tc_fence_after();
                        dst(ci, j == 1);
                    }
                }
                if (!ok) break;
                mma_commit(wfree);
                mma_commit(dsready);
                cc += n_chunks;
                ++kp;
            }
            mma_commit(mmadone);
            mbar_wait(mmadone, 0, kWaitNs);
        }
    } else if (warp == 2) {
        // --------------------------------------------------------------- storer
        if (lane == 0) {
            uint32_t kp = 0, sg = 0;
            bool ok = true;
            for (int u = u_begin; u < u_end && ok; ++u) {
                if (unit_len(a, u) == 0) continue;
                float *Sg = unit_head(a, u);
                if (!Sg) continue;
                const int pass = u % a.n_pass;
                if (!wait_bar(dzready, kp & 1u, fail)) break;
                bulk_reduce_add_f32(Sg + (size_t)2 * F * d + (size_t)pass * F, dzs, (uint32_t)NCP * 32 * 4);
                bulk_commit();
                bulk_wait_read_all();
                mbar_arrive(dzfree);
                for (int c = 0; c < NCP; ++c, ++sg) {
                    const int slot = sg % kStage;
                    if (!wait_bar(&sfull[slot], (sg / kStage) & 1u, fail)) { ok = false; break; }
                    bulk_reduce_add_f32(Sg + (size_t)(pass * NCP + c) * 32 * d, stage + (size_t)slot * atom, atom);
                    bulk_commit();
                    bulk_wait_read_all();
                    mbar_arrive(&sempty[slot]);
                }
                ++kp;
            }
            bulk_wait_all();
        }
    } else if (warp >= 4) {
        // ------------------------------------------------------------- math
        const int mt = tid - 128;
        const int q4 = warp & 3, part = (warp - 4) >> 2;
        const int row = 32 * q4 + lane;
        const uint32_t lane_off = (uint32_t)(32 * q4) << 16;
        const bool fval = row < F;
        // the thread's feature within the pass: one per part (the sign) for F <= 128;
        // for F = 256 the parts are the two 128-feature tiles of the pass's sign
        const int fp = wide ? 128 * part + row : part * F + row;
        // per-token partial extrema and sums: [token][quarter] per part, or, for
        // F = 256, [token][part][quarter] shared by both parts
        float *tk = reinterpret_cast<float *>(smem + a.off_tk);
        const int tk_m = wide ? 8 * lane : (part * 32 + lane) * 4;
        const int tk_w = wide ? 4 * part + q4 : q4;
        uint32_t kp = 0, cc = 0, sg = 0;
        bool ok = true;
        for (int u = u_begin; u < u_end && ok; ++u) {
            const int Tu = unit_len(a, u);
            if (Tu == 0) continue;
            if (!unit_head(a, u)) {
                if (mt == 0) raise_error(a.err, ERR_BAD_STATE_PTR);
                continue;
            }
            const int n_chunks = (Tu + kChunk - 1) / kChunk;
            const float sgn = (wide ? u % a.n_pass : part) == 0 ? kLog2e : -kLog2e;
            const bool neg = sgn < 0.f;
            float dz = 0.f;
            for (int j = 0; j < n_chunks; ++j, ++cc) {
                const int b = cc & 1;
                const int nt = min(kChunk, Tu - j * kChunk);
                uint8_t *pkb = smem + a.off_c + b * a.chunk_stride + atom + vbytes;
                bool bad = !wait_bar(&ukready[b], (cc >> 1) & 1u, fail);
                tc_fence_after();
                // per-token maximum of +-U_k over this warp's 32 features
                float uk[32], ek[32];
                tmem_ld32(tmem + 32 * b + (wide ? 64 * part : 0) + lane_off, uk);
                tmem_wait_ld();
#pragma unroll
                for (int t = 0; t < 32; ++t) ek[t] = (fval && t < nt) ? (neg ? -uk[t] : uk[t]) : -INFINITY;
                tk[tk_m + tk_w] = warp_reduce32<1>(ek, lane);
                if (group_sync_failed(kBarMath, kMathThreads, bad)) { ok = false; break; }
                float m_l;
                {
                    const float4 x = *reinterpret_cast<const float4 *>(&tk[tk_m]);
                    m_l = fmaxf(fmaxf(x.x, x.y), fmaxf(x.z, x.w));
                    if (wide) {
                        const float4 y = *reinterpret_cast<const float4 *>(&tk[tk_m + 4]);
                        m_l = fmaxf(m_l, fmaxf(fmaxf(y.x, y.y), fmaxf(y.z, y.w)));
                    }
                    m_l *= kLog2e;
                }
#pragma unroll
                for (int t = 0; t < 32; ++t) {
                    const float m = __shfl_sync(0xffffffffu, m_l, t);
                    ek[t] = (fval && t < nt) ? ex2(fmaf(uk[t], sgn, -m)) : 0.f;
                    uk[t] = ek[t];
                }
                tk[256 + tk_m + tk_w] = warp_reduce32<0>(uk, lane);
                if (group_sync_failed(kBarMath, kMathThreads, false)) { ok = false; break; }
                // phi(K) normalised into the bf16 MN-major operand [token][feature];
                // lane t holds token t's normaliser (0 for an empty slot)
                float inv_l;
                {
                    const float4 v = *reinterpret_cast<const float4 *>(&tk[256 + tk_m]);
                    float sum = (v.x + v.y) + (v.z + v.w);
                    if (wide) {
                        const float4 y = *reinterpret_cast<const float4 *>(&tk[256 + tk_m + 4]);
                        sum += (y.x + y.y) + (y.z + y.w);
                    }
                    inv_l = sum > 0.f ? 1.f / sum : 0.f;
                }
                const int f = fp;
                uint8_t *bf = pkb + (f >> 6) * (kChunk * 128) + ((f & 7) << 1);
                const int gf = (f & 63) >> 3;
#pragma unroll
                for (int t = 0; t < 32; ++t) {
                    const float v = ek[t] * __shfl_sync(0xffffffffu, inv_l, t);
                    dz += v;
                    if (fval) *reinterpret_cast<bf16 *>(bf + t * 128 + ((gf ^ (t & 7)) << 4)) = __float2bfloat16_rn(v);
                }
                fence_proxy_async_smem();
                __syncwarp();
                if (lane == 0) mbar_arrive(&pkready[b]);
            }
            if (!ok) break;
            // dz of this thread's feature, then the dS^T tiles into the staging ring
            bool bad = !wait_bar(dzfree, (kp & 1u) ^ 1u, fail);
            if (fval && !bad) dzs[fp] = dz;
            fence_proxy_async_smem();
            __syncwarp();
            if (lane == 0 && !bad) mbar_arrive(dzready);
            bad = !wait_bar(dsready, kp & 1u, fail) || bad;
            tc_fence_after();
            const int e = row;
#pragma unroll 1
            for (int i = 0; i < NCP / 2; ++i) {
                // tiles of this part: chunks part, part + 2, ... of each half, in storer order
                const int hp = NH / 2 > 0 ? NH / 2 : 1;   // tiles per half and part
                const int h = i / hp;
                const int k = part + 2 * (i % hp);
                if (k >= NH) continue;
                const int c = h * NH + k;
                const uint32_t sgc = sg + c;
                const int slot = sgc % kStage;
                bool okc = wait_bar(&sempty[slot], ((sgc / kStage) & 1u) ^ 1u, fail) && !bad;
                float v[32];
                tmem_ld32(tmem + (h == 0 ? kColDSp : kColDSm) + lane_off + 32 * k, v);
                tmem_wait_ld();
                if (okc && e < d) {
                    uint8_t *rowp = stage + (size_t)slot * atom + e * 128;
#pragma unroll
                    for (int gq = 0; gq < 8; ++gq)
                        *reinterpret_cast<float4 *>(rowp + ((gq ^ (e & 7)) << 4)) =
                            make_float4(v[4 * gq], v[4 * gq + 1], v[4 * gq + 2], v[4 * gq + 3]);
                }
                fence_proxy_async_smem();
                __syncwarp();
                if (lane == 0 && okc) mbar_arrive(&sfull[slot]);
                bad = bad || !okc;
            }
            tc_fence_before();
            __syncwarp();
            if (lane == 0 && !bad) mbar_arrive(dsfree);
            sg += NCP;
            ++kp;
        }
        if (mt == 0 && *fail) raise_error(a.err, ERR_WAIT_TIMEOUT);
    }

    __syncthreads();
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc(tmem, 512);
    }
}

}  // namespace

bool commit_red_supported(const hybrid_cfg &c)
{
    if (c.io_dtype != HYBRID_BF16) return false;
    if (c.head_dim != 64 && c.head_dim != 128) return false;
    if (c.feat_dim != 64 && c.feat_dim != 128 && c.feat_dim != 256) return false;
    return (int)make_clayout(c.head_dim, c.feat_dim).bytes <= kSmemLimit;
}

namespace {

// Tensor maps and sizes shared by the uniform and the ragged launch; rows = tokens of K and V.
bool fill_commit_args(const hybrid_cfg &c, const void *K, const void *V, long long rows, const void *W,
                      void *const *states, int n_req, unsigned *err, CommitArgs &a)
{
    const CLayout L = make_clayout(c.head_dim, c.feat_dim);
    const int d = c.head_dim, F = c.feat_dim, Hkv = c.n_kv_heads;
    // V: [panel][row][head][64], a box of kChunk rows of one head; W: [panel][row][64]
    const cuuint64_t dv[4] = {64, (cuuint64_t)Hkv, (cuuint64_t)rows, (cuuint64_t)d / 64};
    const cuuint64_t sv[3] = {(cuuint64_t)d * 2, (cuuint64_t)Hkv * d * 2, 128};
    const cuuint32_t bv[4] = {64, 1, (cuuint32_t)kChunk, (cuuint32_t)d / 64};
    const cuuint64_t dw[3] = {64, (cuuint64_t)Hkv * d, (cuuint64_t)F / 64};
    const cuuint64_t sw[2] = {(cuuint64_t)F * 2, 128};
    const cuuint32_t bw[3] = {64, (cuuint32_t)d, (cuuint32_t)F / 64};
    if (!encode_bf16(&a.tmV, V, 4, dv, sv, bv) || !encode_bf16(&a.tmK, K, 4, dv, sv, bv) ||
        !encode_bf16(&a.tmW, W, 3, dw, sw, bw))
        return false;
    a.K = static_cast<const bf16 *>(K);
    a.states = states;
    a.err = err;
    a.n_pass = F > 128 ? 2 : 1;
    a.n_units = n_req * Hkv * a.n_pass;
    a.Hkv = Hkv;
    a.d = d;
    a.F = F;
    a.off_w = L.off_w;
    a.off_c = L.off_c;
    a.off_s = L.off_s;
    a.off_dz = L.off_dz;
    a.off_tk = L.off_tk;
    a.off_bar = L.off_bar;
    a.chunk_stride = L.chunk;
    return true;
}

template <class A>
cudaError_t run_commit_red(const hybrid_cfg &c, const A &a, cudaStream_t st)
{
    const CLayout L = make_clayout(c.head_dim, c.feat_dim);
    const int grid = a.n_units < sm_count() ? a.n_units : sm_count();
    static std::atomic<unsigned long long> opted;
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
    const unsigned long long bit = 1ull << dev;
    if (!(opted.load(std::memory_order_acquire) & bit)) {
        const cudaError_t e =
            cudaFuncSetAttribute(k_commit_red<A>, cudaFuncAttributeMaxDynamicSharedMemorySize, kSmemLimit);
        if (e != cudaSuccess) return e;
        opted.fetch_or(bit, std::memory_order_release);
    }
    cudaLaunchConfig_t lc = {};
    lc.gridDim = dim3(grid);
    lc.blockDim = dim3(kThreads);
    lc.dynamicSmemBytes = L.bytes;
    lc.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    lc.attrs = attr;
    lc.numAttrs = 1;
    return cudaLaunchKernelEx(&lc, k_commit_red<A>, a);
}

}  // namespace

cudaError_t launch_commit_red(const hybrid_cfg &c, const void *K, const void *V, int n_tok, const void *W,
                              void *const *states, int n_req, unsigned *err, cudaStream_t st)
{
    CommitArgs a;
    if (!fill_commit_args(c, K, V, (long long)n_req * n_tok, W, states, n_req, err, a)) return cudaErrorInvalidValue;
    a.T = n_tok;
    return run_commit_red(c, a, st);
}

cudaError_t launch_commit_red_ragged(const hybrid_cfg &c, const void *K, const void *V, const int *tok,
                                     const void *W, void *const *states, int n_req, unsigned *err, cudaStream_t st)
{
    if (n_req < 1 || n_req > kMaxRaggedRequests) return cudaErrorInvalidValue;
    static thread_local CommitRaggedArgs a;   // 8 KB of offsets: kept off the stack
    if (!fill_commit_args(c, K, V, tok[n_req] > 0 ? tok[n_req] : 1, W, states, n_req, err, a))
        return cudaErrorInvalidValue;
    a.T = 0;
    a.n_req = n_req;
    for (int r = 0; r <= n_req; ++r) a.tok[r] = tok[r];
    return run_commit_red(c, a, st);
}

}  // namespace hyb
