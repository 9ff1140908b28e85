// hybrid_fused.cu -- persistent, warp-specialised block-hybrid step on the
// tcgen05 tensor cores, optionally fused with the block commit.
//
// Section 3.1 of "Retrofitting Linear Attention into Diffusion Language
// Models" defines the step (in-block softmax, linear readout from the committed
// state, gated shared-normaliser merge) and the state update; its serving
// section computes both in one kernel launch, which kCommit = true does here:
// every state tile is read once, used for the readout with the pre-commit
// state, updated with this block's phi(k) v^T and written back.
//
// Work unit = (request r, state head g).  One CTA per SM loops over a
// contiguous range of units.  Warp roles (12 warps):
//   warp 0     S producer: z and the 2F/32 state tiles of each unit, by 1-D bulk
//              copies, through an NS-slot ring (the state layout is the MMA
//              operand image, see hybrid.h).
//   warp 1     MMA issuer (one thread).
//   warp 2     producer: TMA of Q, W, K (region X) and V of the next unit; V^T in
//              f32 (commit operand) into region X once Q, W, K are spent.
//   warp 3     storer: TMA stores of the output tile and, with the commit, bulk
//              stores of the updated state tiles and z, releasing ring slots
//              once they have been read out.  The output tile (128 rows x d
//              bf16) is staged in the ring slots of the unit's last two state
//              tiles, which are held back for it.
//   warps 4-11 math: row statistics and phi(Q) (one thread per TMEM lane and
//              column half), P, phi(K)^T, the state-tile update and the output.
// Tensor Memory (512 columns):
//   [0,256)    U = Q W, then phi(Q) = [phi+, phi-] (A operand of the readout);
//              with the commit, each half is reused for dS^T = V^T phi(K)^T of
//              the same features once the readout has consumed it.
//   [256,384), [384,512)  two output accumulators (alternating units): first
//              the scores Q K^T (and U_k^T = W^T K^T), then
//              D = phi'(Q) S + P' V, the merged numerator.
// Merge: with sigma = log of the larger branch mass, phi' = phi e^-sigma and
// P' = w e^(s - sigma), so D / den = (w sm_num + lin_num) / (w sm_den + lin_den)
// exactly, with den = e^(log lin_den - sigma) + e^(log(w sm_den) - sigma) in [1, 2].
//
// MMA cost note: on this part a tcgen05.mma with M = 128 costs about the same
// time for any N up to 128-256, so contractions are shaped for few, wide
// instructions (dS^T as two N = F products rather than per-tile N = 32 ones).
#include <cuda.h>
#include <cudaTypedefs.h>

#include <atomic>
#include <mutex>

#include "hybrid_common.cuh"
#include "hybrid_tc.h"
#include "tc_ptx.cuh"

namespace hyb {

namespace {

using bf16 = __nv_bfloat16;

constexpr int kWarps = 12;
constexpr int kThreads = kWarps * 32;
constexpr int kMathThreads = 256;
constexpr uint32_t kColA = 0, kColD0 = 256;
constexpr int kMaxSlots = 16;
constexpr uint64_t kWaitNs = 1000000000ull;
constexpr float kLog2e = 1.4426950408889634f;
constexpr int kSmemLimit = 232448;
constexpr int kOneCtaPerSm = 118 * 1024;
constexpr uint32_t kBarMath = 1;

struct FusedArgs {
    CUtensorMap tmQ, tmK, tmV, tmW, tmO;   // Q, O [n*B][Hq][d], K and V [n*B][Hkv][d], W [Hkv*d][F]; 128-byte swizzle
    const bf16 *Q, *K, *V, *W;
    const float *alpha;
    void *const *states;
    bf16 *O;
    unsigned *err;
    int n_units, B, Hq, Hkv, G, d, F, NS;
    float scale;
    uint32_t off_q, off_w, off_k, off_vb, off_p, off_z, off_st, off_bar;
};

// Shared memory: [ring NS x d*128][X: Q | W | K][Vb][P][z x2][stats][barriers].
// With the commit, V^T (128 x 32 f32) and phi(K)^T (2F x 32 f32) reuse region X
// after the unit's first MMA group has consumed Q, W and K.  Q, K, V and W land
// by TMA with the 128-byte swizzle: Q as two 64-column atoms of 128 rows
// (16 KB apart), K as two atoms of B rows, V as two 64-column atoms of B rows
// (MN-major B operand: j-groups 1 KB apart, atoms B*128 apart), W as F/64
// atoms of d rows (MN-major: e-groups 1 KB apart, atoms d*128 apart).
struct FLayout {
    uint32_t off_q, off_w, off_k, off_vb, off_p, off_z, off_st, off_bar, bytes;
    int NS;
};

FLayout make_flayout(int d, int F, int B)
{
    FLayout L{};
    const uint32_t chunk = (uint32_t)d * 128;
    const uint32_t zb = (((uint32_t)2 * F * 4) + 1023) & ~1023u;
    const uint32_t q = (uint32_t)d * 256, w = (uint32_t)d * (F < 128 ? 128 : F) * 2, k = (uint32_t)B * d * 2,
                   vb = (uint32_t)B * d * 2, p = 128u * B * 2;
    const uint32_t st = 16 * 1024, bar = 1024;
    const uint32_t fixed = q + w + k + vb + p + 2 * zb + st + bar + 1024;
    int ns = ((int)kSmemLimit - (int)fixed) / (int)chunk;
    if (ns > kMaxSlots) ns = kMaxSlots;
    L.NS = ns;
    uint32_t off = (uint32_t)(ns > 0 ? ns : 0) * chunk;
    L.off_q = off; off += q;
    L.off_w = off; off += w;
    L.off_k = off; off += k;
    L.off_vb = off; off += vb;
    L.off_p = off; off += p;
    L.off_z = off; off += 2 * zb;
    L.off_st = off; off += st;
    L.off_bar = off; off += bar;
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

__device__ __forceinline__ uint32_t pack_bf16x2(float a, float b)
{
    const __nv_bfloat162 v = __floats2bfloat162_rn(a, b);
    return *reinterpret_cast<const uint32_t *>(&v);
}

// Bounded wait that also gives up as soon as another role has failed.
__device__ __forceinline__ bool wait_bar(uint64_t *bar, uint32_t parity, volatile int *fail)
{
    if (ptx::mbar_try_wait(bar, parity)) return true;
    const uint64_t t0 = ptx::global_timer_ns();
    while (true) {
        if (ptx::mbar_try_wait_sleep(bar, parity, 200000u)) return true;
        if (*fail) return false;
        if (ptx::global_timer_ns() - t0 > kWaitNs) {
            atomicOr(const_cast<int *>(fail), 1);
            return false;
        }
    }
}

// Barrier over one warp group that also ORs a failure flag across it, so that
// every thread of the group takes the same branch afterwards.
__device__ __forceinline__ bool group_sync_failed(uint32_t id, uint32_t nthreads, bool local_fail)
{
    uint32_t r;
    asm volatile(
        "{\n\t.reg .pred p, q;\n\t"
        "setp.ne.u32 p, %1, 0;\n\t"
        "bar.red.or.pred q, %2, %3, p;\n\t"
        "selp.u32 %0, 1, 0, q;\n\t}"
        : "=r"(r)
        : "r"((uint32_t)local_fail), "r"(id), "r"(nthreads)
        : "memory");
    return r != 0;
}
__device__ __forceinline__ bool math_sync_failed(bool local_fail)
{
    return group_sync_failed(kBarMath, kMathThreads, local_fail);
}


// Reduce 16 per-lane values across the 32 lanes of a warp (op = add / max /
// min) by halving the set each step; on return lane L holds the total of
// value index tok(L) = 8*b4 + 4*b3 + 2*b2 + b1 (b_i = bit i of L).
template <int kOp>
__device__ __forceinline__ float comb(float a, float b)
{
    return kOp == 0 ? a + b : (kOp == 1 ? fmaxf(a, b) : fminf(a, b));
}
template <int kOp>
__device__ __forceinline__ float warp_reduce16(float (&v)[16], int lane)
{
#pragma unroll
    for (int i = 0; i < 8; ++i) {
        const bool up = lane & 16;
        const float send = up ? v[i] : v[i + 8], keep = up ? v[i + 8] : v[i];
        v[i] = comb<kOp>(keep, __shfl_xor_sync(0xffffffffu, send, 16));
    }
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const bool up = lane & 8;
        const float send = up ? v[i] : v[i + 4], keep = up ? v[i + 4] : v[i];
        v[i] = comb<kOp>(keep, __shfl_xor_sync(0xffffffffu, send, 8));
    }
#pragma unroll
    for (int i = 0; i < 2; ++i) {
        const bool up = lane & 4;
        const float send = up ? v[i] : v[i + 2], keep = up ? v[i + 2] : v[i];
        v[i] = comb<kOp>(keep, __shfl_xor_sync(0xffffffffu, send, 4));
    }
    {
        const bool up = lane & 2;
        const float send = up ? v[0] : v[1], keep = up ? v[1] : v[0];
        v[0] = comb<kOp>(keep, __shfl_xor_sync(0xffffffffu, send, 2));
    }
    return comb<kOp>(v[0], __shfl_xor_sync(0xffffffffu, v[0], 1));
}
__device__ __forceinline__ int reduce16_token(int lane)
{
    return ((lane >> 4) & 1) * 8 + ((lane >> 3) & 1) * 4 + ((lane >> 2) & 1) * 2 + ((lane >> 1) & 1);
}

__device__ __forceinline__ float *unit_state(const FusedArgs &a, int u)
{
    const int r = u / a.Hkv, g = u % a.Hkv;
    float *st = reinterpret_cast<float *>(a.states[r]);
    if (!state_ptr_ok(st)) return nullptr;
    return st + (size_t)g * head_floats(a.d, a.F);
}

// TMA of unit (r, g)'s Q, W, K into region X (one thread), completing on bar.
__device__ __forceinline__ void tma_x(const FusedArgs &a, uint8_t *smem, int r, int g, uint64_t *bar)
{
    using namespace ptx;
    const int d = a.d, F = a.F, B = a.B, G = a.G;
    const uint32_t bytes = (uint32_t)(d / 64) * (G * B * 128) + (uint32_t)(F / 64) * (d * 128) + (uint32_t)(d / 64) * (B * 128);
    mbar_arrive_expect_tx(bar, bytes);
    for (int e = 0; e < d / 64; ++e) {
        tma_load_3d(smem + a.off_q + e * (128 * 128), &a.tmQ, 64 * e, g * G, r * B, bar);
        tma_load_3d(smem + a.off_k + e * (B * 128), &a.tmK, 64 * e, g, r * B, bar);
    }
    for (int f = 0; f < F / 64; ++f) tma_load_2d(smem + a.off_w + f * (d * 128), &a.tmW, 64 * f, g * d, bar);
}
__device__ __forceinline__ void tma_v(const FusedArgs &a, uint8_t *smem, int r, int g, uint64_t *bar)
{
    using namespace ptx;
    const int d = a.d, B = a.B;
    mbar_arrive_expect_tx(bar, (uint32_t)(d / 64) * (B * 128));
    for (int e = 0; e < d / 64; ++e) tma_load_3d(smem + a.off_vb + e * (B * 128), &a.tmV, 64 * e, g, r * B, bar);
}

template <bool kCommit>
__global__ void __launch_bounds__(kThreads, 1) k_fused(const __grid_constant__ FusedArgs a)
{
    using namespace ptx;
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int d = a.d, F = a.F, B = a.B, G = a.G, NS = a.NS;
    const int NC = (2 * F) / 32;
    // with the commit, the output tile is staged in the slots of tiles ocm, ocm + 1
    const int ocm = NC > NS ? NC - NS : 0;
    const uint32_t chunk_bytes = (uint32_t)d * 128;
    const int per = a.n_units / (int)gridDim.x, rem = a.n_units % (int)gridDim.x;
    const int u_begin = (int)blockIdx.x * per + min((int)blockIdx.x, rem);
    const int u_end = u_begin + per + ((int)blockIdx.x < rem ? 1 : 0);

    uint64_t *bars = reinterpret_cast<uint64_t *>(smem + a.off_bar);
    uint64_t *full = bars;
    uint64_t *empty = full + NS;
    uint64_t *zfull = empty + NS;
    uint64_t *zempty = zfull + 2;
    uint64_t *dready = zempty + 2;   // [2]
    uint64_t *dfree = dready + 2;    // [2]
    uint64_t *hread = dfree + 2;     // [2]
    uint64_t *dsready = hread + 2;   // [2]
    uint64_t *xfull = dsready + 2;
    uint64_t *xfree = xfull + 1;
    uint64_t *vfull = xfree + 1;
    uint64_t *vfree = vfull + 1;
    uint64_t *vtready = vfree + 1;
    uint64_t *uready = vtready + 1;
    uint64_t *phiready = uready + 1;
    uint64_t *efree = phiready + 1;
    uint64_t *rdone = efree + 1;
    uint64_t *mmadone = rdone + 1;
    uint64_t *tready = mmadone + 1;  // [2] math -> storer: a feature half of the tiles is updated
    uint64_t *zdone = tready + 2;    // math -> storer: z is updated
    uint64_t *ofree = zdone + 1;     // the last two slots of the unit may take the output tile
    uint64_t *ostaged = ofree + 1;   // math -> storer: the output tile is in the slots
    const int n_bars = 2 * NS + 14 + 15;
    uint32_t *tmem_holder = reinterpret_cast<uint32_t *>(bars + n_bars);
    volatile int *fail = reinterpret_cast<volatile int *>(tmem_holder + 1);

    if (tid == 0) {
        for (int i = 0; i < n_bars; ++i) {
            uint64_t *b = &bars[i];
            const uint32_t cnt = b == vtready ? 2u : 1u;
            mbar_init(b, cnt);
        }
        *fail = 0;
        fence_mbar_init();
    }
    if (warp == 1) {
        tmem_alloc(tmem_holder, 512);
        tmem_relinquish();
    }
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_holder;
    uint8_t *ring = smem;
    float *zbuf0 = reinterpret_cast<float *>(smem + a.off_z);
    const int zstride = ((2 * F * 4 + 1023) & ~1023) / 4;
    uint8_t *vt_s = smem + a.off_q;                     // V^T: 128 rows x 128 B (commit)
    uint8_t *pt_s = smem + a.off_q + 128 * 128;         // phi(K)^T: 2F rows x 128 B (commit)

    if (warp == 0) {
        // ------------------------------------------------------- S producer
        if (lane == 0) {
            uint32_t q = 0, kp = 0;
            int issued_slot[kMaxSlots];
            int issued_z[2] = {0, 0};
            for (int i = 0; i < kMaxSlots; ++i) issued_slot[i] = 0;
            bool ok = true;
            for (int u = u_begin; u < u_end && ok; ++u) {
                float *Sg = unit_state(a, u);
                if (!Sg) continue;
                const int zb = kp & 1;
                if (!wait_bar(&zempty[zb], ((kp >> 1) & 1u) ^ 1u, fail)) break;
                mbar_arrive_expect_tx(&zfull[zb], 2 * F * 4);
                bulk_g2s(zbuf0 + zb * zstride, Sg + (size_t)2 * F * d, 2 * F * 4, &zfull[zb]);
                ++issued_z[zb];
                for (int c = 0; c < NC; ++c, ++q) {
                    const int slot = q % NS;
                    if (!wait_bar(&empty[slot], ((q / NS) & 1u) ^ 1u, fail)) { ok = false; break; }
                    mbar_arrive_expect_tx(&full[slot], chunk_bytes);
                    bulk_g2s(ring + (size_t)slot * chunk_bytes, Sg + (size_t)c * 32 * d, chunk_bytes, &full[slot]);
                    ++issued_slot[slot];
                }
                ++kp;
            }
            if (*fail) {
                for (int s = 0; s < NS; ++s)
                    if (issued_slot[s]) mbar_wait(&full[s], (uint32_t)(issued_slot[s] - 1) & 1u, kWaitNs);
                for (int s = 0; s < 2; ++s)
                    if (issued_z[s]) mbar_wait(&zfull[s], (uint32_t)(issued_z[s] - 1) & 1u, kWaitNs);
            }
        }
    } else if (warp == 1) {
        // ------------------------------------------------------- MMA issuer
        if (lane == 0) {
            const uint32_t q_u = smem_u32(smem + a.off_q), w_u = smem_u32(smem + a.off_w),
                           k_u = smem_u32(smem + a.off_k), vb_u = smem_u32(smem + a.off_vb),
                           vt_u = smem_u32(vt_s), pt_u = smem_u32(pt_s), p_u = smem_u32(smem + a.off_p),
                           ring_u = smem_u32(ring);
            const uint32_t idU = instr_desc(FMT_BF16, FMT_BF16, false, true, 128, F);
            const uint32_t idS = instr_desc(FMT_BF16, FMT_BF16, false, false, 128, B);
            const uint32_t idK = instr_desc(FMT_BF16, FMT_BF16, true, false, 128, B);
            const uint32_t idR = instr_desc(FMT_TF32, FMT_TF32, false, false, 128, d);
            const uint32_t idDS = instr_desc(FMT_TF32, FMT_TF32, false, false, 128, F);
            const uint32_t idP = instr_desc(FMT_BF16, FMT_BF16, false, true, 128, d);
            uint32_t q = 0, kp = 0;
            bool ok = true;
            for (int u = u_begin; u < u_end && ok; ++u) {
                if (!unit_state(a, u)) continue;
                const uint32_t dcol = tmem + kColD0 + 128 * (kp & 1);
                const uint32_t dother = tmem + kColD0 + 128 * ((kp + 1) & 1);
                if (!wait_bar(xfull, kp & 1u, fail)) break;
                if (kp > 0) {
                    // Tensor Memory of the previous unit: phi columns (and, with the
                    // commit, the dS^T halves) must be consumed before U is rewritten
                    if (kCommit) { if (!wait_bar(efree, (kp - 1) & 1u, fail)) break; }
                    else { if (!wait_bar(rdone, (kp - 1) & 1u, fail)) break; }
                }
                if (kp > 1 && !wait_bar(&dfree[kp & 1], ((kp - 2) >> 1) & 1u, fail)) break;
                tc_fence_after();
                // group 1: U = Q W, scores = Q K^T, U_k^T = W^T K^T
                for (int k = 0; k < d / 16; ++k) {
                    const uint64_t aq = smem_desc(q_u + (k >> 2) * (128 * 128) + (k & 3) * 32, 16, 1024, SWZ_128B);
                    const uint64_t bw = smem_desc(w_u + 2 * k * 1024, d * 128, 1024, SWZ_128B);
                    const uint64_t bk = smem_desc(k_u + (k >> 2) * (B * 128) + (k & 3) * 32, 16, 1024, SWZ_128B);
                    mma_bf16_ss(tmem + kColA, aq, bw, idU, k > 0);
                    mma_bf16_ss(dcol, aq, bk, idS, k > 0);
                    if (kCommit) mma_bf16_ss(dcol + B, bw, bk, idK, k > 0);
                }
                mma_commit(uready);
                mma_commit(xfree);
                // group 2: readout over the state tiles, dS^T per feature half, then P V
                if (!wait_bar(phiready, kp & 1u, fail)) break;
                tc_fence_after();
                for (int c = 0; c < NC; ++c, ++q) {
                    const int slot = q % NS;
                    if (!wait_bar(&full[slot], (q / NS) & 1u, fail)) { ok = false; break; }
                    const uint32_t s_u = ring_u + slot * chunk_bytes;
#pragma unroll
                    for (int kk = 0; kk < 4; ++kk)
                        mma_tf32_ts(dcol, tmem + kColA + 32 * c + 8 * kk, smem_desc(s_u + 32 * kk, 16, 1024, SWZ_128B),
                                    idR, (c | kk) != 0);
                    if (!kCommit) {
                        if (c < NC - 2) mma_commit(&empty[slot]);
                        else if (c == NC - 1) mma_commit(ofree);
                    }
                    if (kCommit && c == NC / 2 - 1) {
                        // phi+ has been read: its columns take dS^T for features [0, F);
                        // dS^T for [F, 2F) goes to the idle output accumulator
                        mma_commit(&hread[0]);
                        if (!wait_bar(&hread[0], kp & 1u, fail)) { ok = false; break; }
                        if (!wait_bar(vtready, kp & 1u, fail)) { ok = false; break; }
                        if (kp > 0 && !wait_bar(&dfree[(kp + 1) & 1], ((kp - 1) >> 1) & 1u, fail)) { ok = false; break; }
                        tc_fence_after();
#pragma unroll
                        for (int h = 0; h < 2; ++h) {
#pragma unroll
                            for (int kk = 0; kk < 4; ++kk)
                                mma_tf32_ss(h == 0 ? tmem + kColA : dother, smem_desc(vt_u + 32 * kk, 16, 1024, SWZ_128B),
                                            smem_desc(pt_u + h * F * 128 + 32 * kk, 16, 1024, SWZ_128B), idDS, kk != 0);
                            mma_commit(&dsready[h]);
                        }
                    }
                }
                if (!ok) break;
                mma_commit(rdone);
                if (!wait_bar(vfull, kp & 1u, fail)) break;
                tc_fence_after();
                for (int k = 0; k < B / 16; ++k) {
                    const uint64_t ap = smem_desc(p_u + k * 256, 128, (B / 8) * 128, SWZ_NONE);
                    const uint64_t bv = smem_desc(vb_u + 2 * k * 1024, B * 128, 1024, SWZ_128B);
                    mma_bf16_ss(dcol, ap, bv, idP, 1);
                }
                mma_commit(&dready[kp & 1]);
                mma_commit(vfree);
                ++kp;
            }
            mma_commit(mmadone);
            mbar_wait(mmadone, 0, kWaitNs);
        }
    } else if (warp == 2) {
        // ------------------------------------------------------------- producer
        uint32_t kp = 0;
        for (int u = u_begin; u < u_end; ++u) {
            if (!unit_state(a, u)) continue;
            const int r = u / a.Hkv, g = u % a.Hkv;
            bool ok = true;
            if (kp > 0) {
                // region X is free once the previous unit's last use of it has completed
                ok = kCommit ? wait_bar(&dsready[1], (kp - 1) & 1u, fail) : wait_bar(xfree, (kp - 1) & 1u, fail);
            }
            if (__any_sync(0xffffffffu, !ok)) break;
            if (lane == 0) tma_x(a, smem, r, g, xfull);
            if (kp > 0) ok = wait_bar(vfree, (kp - 1) & 1u, fail);
            if (__any_sync(0xffffffffu, !ok)) break;
            if (lane == 0) tma_v(a, smem, r, g, vfull);
            if (kCommit) {
                // V^T in f32 into region X once this unit's first MMA group is done with it
                ok = wait_bar(xfree, kp & 1u, fail);
                if (__any_sync(0xffffffffu, !ok)) break;
                for (int idx = lane; idx < 16 * 32; idx += 32) {
                    const int eg = idx >> 5, t = idx & 31;     // 8 rows e = 8*eg .. 8*eg+7, column t
                    float v[8];
                    if (eg * 8 < d) {
                        const uint4 raw = *reinterpret_cast<const uint4 *>(
                            a.V + (((size_t)r * B + t) * a.Hkv + g) * d + 8 * eg);
                        const __nv_bfloat162 *b2 = reinterpret_cast<const __nv_bfloat162 *>(&raw);
#pragma unroll
                        for (int i = 0; i < 4; ++i) { v[2 * i] = __low2float(b2[i]); v[2 * i + 1] = __high2float(b2[i]); }
                    } else {
#pragma unroll
                        for (int i = 0; i < 8; ++i) v[i] = 0.f;
                    }
#pragma unroll
                    for (int i = 0; i < 8; ++i) {
                        const int e = 8 * eg + i;
                        *(reinterpret_cast<float *>(vt_s + e * 128 + ((((t >> 2) ^ (e & 7))) << 4)) + (t & 3)) = v[i];
                    }
                }
                fence_proxy_async_smem();
                __syncwarp();
                if (lane == 0) mbar_arrive(vtready);
            }
            ++kp;
        }
    } else if (warp == 3) {
        // --------------------------------------------------------------- storer
        if (lane == 0) {
            uint32_t q = 0, kp = 0;
            for (int u = u_begin; u < u_end; ++u) {
                float *Sg = unit_state(a, u);
                if (!Sg) continue;
                const int r = u / a.Hkv, g = u % a.Hkv;
                bool ok = true;
                if (kCommit) {
                    const int zb = kp & 1;
                    if (!wait_bar(zdone, kp & 1u, fail)) break;
                    bulk_s2g(Sg + (size_t)2 * F * d, zbuf0 + zb * zstride, 2 * F * 4);
                    bulk_commit();
                    bulk_wait_read_all();
                    mbar_arrive(&zempty[zb]);
                    for (int h = 0; h < 2 && ok; ++h) {
                        if (!wait_bar(&tready[h], kp & 1u, fail)) { ok = false; break; }
                        for (int c = h * NC / 2; c < (h + 1) * NC / 2; ++c)
                            bulk_s2g(Sg + (size_t)c * 32 * d, ring + (size_t)((q + c) % NS) * chunk_bytes, chunk_bytes);
                        bulk_commit();
                        bulk_wait_read_all();
                        // with the commit, two slots of the first half are held for the
                        // output tile: tiles oc and oc + 1, whose slots no later tile of
                        // this unit reuses
                        for (int c = h * NC / 2; c < (h + 1) * NC / 2; ++c)
                            if (h == 1 || c < ocm || c > ocm + 1) mbar_arrive(&empty[(q + c) % NS]);
                        if (h == 0) mbar_arrive(ofree);
                    }
                    if (!ok) break;
                }
                // output tile: two TMA boxes from the two held-back slots
                if (!wait_bar(ostaged, kp & 1u, fail)) break;
                const int oc = kCommit ? ocm : NC - 2;   // first of the two slots holding the output
                uint8_t *s0 = ring + (size_t)((q + oc) % NS) * chunk_bytes;
                uint8_t *s1 = ring + (size_t)((q + oc + 1) % NS) * chunk_bytes;
                if (d == 128) {
                    tma_store_3d(&a.tmO, 0, g * G, r * B, s0);
                    tma_store_3d(&a.tmO, 64, g * G, r * B, s1);
                } else {
                    tma_store_3d(&a.tmO, 0, g * G, r * B, s0);
                    tma_store_3d(&a.tmO, 0, g * G, r * B + B / 2, s1);
                }
                bulk_commit();
                bulk_wait_read_all();
                mbar_arrive(&empty[(q + oc) % NS]);
                mbar_arrive(&empty[(q + oc + 1) % NS]);
                q += NC;
                ++kp;
            }
            bulk_wait_all();
        }
    } else {
        // ------------------------------------------------------------- math
        const int mt = tid - 128;
        const int q4 = warp & 3, half = (warp - 4) >> 2;
        const int row = 32 * q4 + lane;
        const uint32_t lane_off = (uint32_t)(32 * q4) << 16;
        const int nsc = B / 16, nfc = F / 32;
        const int Mv = G * B;
        const bool valid = row < Mv;
        const bool fval = row < F;
        float *ex = reinterpret_cast<float *>(smem + a.off_st);   // [8 slots][2 halves][128 rows]
        float *den_s = ex + 8 * 256;                                // [2][128]
        float *tk = den_s + 256;                                    // token stats (commit) [8][32][4]
        const float scale_l2 = a.scale * kLog2e;
        const int tok = reduce16_token(lane);
        uint32_t q = 0, kp = 0;
        for (int u = u_begin; u < u_end; ++u) {
            float *Sg = unit_state(a, u);
            if (!Sg) {
                if (mt == 0) raise_error(a.err, ERR_BAD_STATE_PTR);
                continue;
            }
            const int g = u % a.Hkv;
            const int zb = kp & 1;
            // gate of this row's query head, loaded now so the latency overlaps the first rounds
            const float alpha_row = valid ? a.alpha[g * G + row % G] : 0.f;
            float *zs = zbuf0 + zb * zstride;
            const uint32_t dcol = tmem + kColD0 + 128 * (kp & 1);
            float *den = den_s + 128 * (kp & 1);
            bool ok = wait_bar(uready, kp & 1u, fail);
            tc_fence_after();

            // ---- round 1: row extrema; per-token extrema of U_k^T (features on lanes)
            {
                float ms = -INFINITY, mx = -INFINITY, mn = INFINITY;
                for (int k = half; k < nsc; k += 2) {
                    float v[16];
                    tmem_ld16(dcol + lane_off + 16 * k, v);
                    tmem_wait_ld();
#pragma unroll
                    for (int i = 0; i < 16; ++i) ms = fmaxf(ms, v[i]);
                }
                for (int k = half; k < nfc; k += 2) {
                    float v[32];
                    tmem_ld32(tmem + lane_off + kColA + 32 * k, v);
                    tmem_wait_ld();
#pragma unroll
                    for (int i = 0; i < 32; ++i) { mx = fmaxf(mx, v[i]); mn = fminf(mn, v[i]); }
                }
                ex[(0 * 2 + half) * 128 + row] = ms;
                ex[(1 * 2 + half) * 128 + row] = mx;
                ex[(2 * 2 + half) * 128 + row] = mn;
                if (kCommit) {
                    float uk[16], vmx[16], vmn[16];
                    tmem_ld16(dcol + B + lane_off + 16 * half, uk);
                    tmem_wait_ld();
#pragma unroll
                    for (int t = 0; t < 16; ++t) { vmx[t] = fval ? uk[t] : -INFINITY; vmn[t] = fval ? uk[t] : INFINITY; }
                    const float rmx = warp_reduce16<1>(vmx, lane), rmn = warp_reduce16<2>(vmn, lane);
                    if (!(lane & 1)) {
                        tk[(0 * 32 + 16 * half + tok) * 4 + q4] = rmx;
                        tk[(1 * 32 + 16 * half + tok) * 4 + q4] = rmn;
                    }
                }
            }
            if (math_sync_failed(!ok)) break;
            if (kCommit) {
                if (mt < 64) {   // combine the four feature quarters per token
                    const int t = mt & 31, s = mt >> 5;
                    const float4 v = *reinterpret_cast<const float4 *>(&tk[(s * 32 + t) * 4]);
                    tk[(4 + s) * 128 + t] = s == 0 ? fmaxf(fmaxf(v.x, v.y), fmaxf(v.z, v.w))
                                                   : fminf(fminf(v.x, v.y), fminf(v.z, v.w));
                }
                if (math_sync_failed(false)) break;
            }
            ok = wait_bar(&zfull[zb], (kp >> 1) & 1u, fail);

            // ---- round 2: exponentials and partial sums
            const float m_raw = fmaxf(ex[0 * 256 + row], ex[0 * 256 + 128 + row]);
            {
                const float mx = fmaxf(ex[1 * 256 + row], ex[1 * 256 + 128 + row]);
                const float mn = fminf(ex[2 * 256 + row], ex[2 * 256 + 128 + row]);
                const float mxl = mx * kLog2e, mnl = mn * kLog2e, ml = m_raw * scale_l2;
                float l = 0.f, sp = 0.f, sn = 0.f, lp = 0.f, ln = 0.f;
                for (int k = half; k < nsc; k += 2) {
                    float v[16];
                    tmem_ld16(dcol + lane_off + 16 * k, v);
                    tmem_wait_ld();
#pragma unroll
                    for (int i = 0; i < 16; ++i) l += ex2(fmaf(v[i], scale_l2, -ml));
                }
                for (int k = half; k < nfc; k += 2) {
                    float uu[32], ep[32], en[32];
                    tmem_ld32(tmem + lane_off + kColA + 32 * k, uu);
                    tmem_wait_ld();
                    const float4 *zp = reinterpret_cast<const float4 *>(zs + 32 * k);
                    const float4 *zn = reinterpret_cast<const float4 *>(zs + F + 32 * k);
#pragma unroll
                    for (int i4 = 0; i4 < 8; ++i4) {
                        const float4 a4 = zp[i4], b4 = zn[i4];
                        const float za[4] = {a4.x, a4.y, a4.z, a4.w}, zb4[4] = {b4.x, b4.y, b4.z, b4.w};
#pragma unroll
                        for (int j = 0; j < 4; ++j) {
                            const int i = 4 * i4 + j;
                            ep[i] = ex2(fmaf(uu[i], kLog2e, -mxl));
                            en[i] = ex2(fmaf(-uu[i], kLog2e, mnl));
                            sp += ep[i];
                            sn += en[i];
                            lp = fmaf(ep[i], za[j], lp);
                            ln = fmaf(en[i], zb4[j], ln);
                        }
                    }
                    tmem_st32(tmem + lane_off + kColA + 32 * k, ep);
                    tmem_st32(tmem + lane_off + kColA + F + 32 * k, en);
                }
                ex[(3 * 2 + half) * 128 + row] = l;
                ex[(4 * 2 + half) * 128 + row] = sp;
                ex[(5 * 2 + half) * 128 + row] = sn;
                ex[(6 * 2 + half) * 128 + row] = lp;
                ex[(7 * 2 + half) * 128 + row] = ln;
                if (kCommit) {
                    // unnormalised phi(K) into the phi(K)^T tile (row f, this half's 16 token
                    // columns), per-token partial sums over this warp's features
                    float uk[16], ep16[16], en16[16];
                    tmem_ld16(dcol + B + lane_off + 16 * half, uk);
                    tmem_wait_ld();
                    const float4 *tmx = reinterpret_cast<const float4 *>(&tk[4 * 128 + 16 * half]);
                    const float4 *tmn = reinterpret_cast<const float4 *>(&tk[5 * 128 + 16 * half]);
#pragma unroll
                    for (int t4 = 0; t4 < 4; ++t4) {
                        const float4 x = tmx[t4], y = tmn[t4];
                        const float kx[4] = {x.x, x.y, x.z, x.w}, kn[4] = {y.x, y.y, y.z, y.w};
#pragma unroll
                        for (int j = 0; j < 4; ++j) {
                            const int t = 4 * t4 + j;
                            ep16[t] = fval ? ex2((uk[t] - kx[j]) * kLog2e) : 0.f;
                            en16[t] = fval ? ex2((kn[j] - uk[t]) * kLog2e) : 0.f;
                        }
                    }
                    if (fval) {
                        uint8_t *rp = pt_s + row * 128;
                        uint8_t *rn = pt_s + (F + row) * 128;
#pragma unroll
                        for (int gq = 0; gq < 4; ++gq) {
                            const int gi = 4 * half + gq;
                            *reinterpret_cast<float4 *>(rp + ((gi ^ (row & 7)) << 4)) =
                                make_float4(ep16[4 * gq], ep16[4 * gq + 1], ep16[4 * gq + 2], ep16[4 * gq + 3]);
                            *reinterpret_cast<float4 *>(rn + ((gi ^ ((F + row) & 7)) << 4)) =
                                make_float4(en16[4 * gq], en16[4 * gq + 1], en16[4 * gq + 2], en16[4 * gq + 3]);
                        }
                    }
                    const float rsp = warp_reduce16<0>(ep16, lane), rsn = warp_reduce16<0>(en16, lane);
                    if (!(lane & 1)) {
                        tk[(2 * 32 + 16 * half + tok) * 4 + q4] = rsp;
                        tk[(3 * 32 + 16 * half + tok) * 4 + q4] = rsn;
                    }
                }
                tmem_wait_st();
            }
            if (math_sync_failed(!ok)) break;
            if (kCommit) {
                if (mt < 64) {   // per-token normalisers of phi(K)
                    const int t = mt & 31, s = mt >> 5;
                    const float4 v = *reinterpret_cast<const float4 *>(&tk[((2 + s) * 32 + t) * 4]);
                    tk[(6 + s) * 128 + t] = 1.f / ((v.x + v.y) + (v.z + v.w));
                }
                if (math_sync_failed(false)) break;
            }

            // ---- round 3: sigma, scaled phi(Q) in place, P', den; phi(K) normalised, z update
            {
                const float l = ex[3 * 256 + row] + ex[3 * 256 + 128 + row];
                const float sp = ex[4 * 256 + row] + ex[4 * 256 + 128 + row];
                const float sn = ex[5 * 256 + row] + ex[5 * 256 + 128 + row];
                const float lp = ex[6 * 256 + row] + ex[6 * 256 + 128 + row];
                const float ln = ex[7 * 256 + row] + ex[7 * 256 + 128 + row];
                const float lin_den = lp / sp + ln / sn;
                const int hh = row % G;
                const float lw = valid ? log_sigmoid(alpha_row) : 0.f;
                const float log_s = lw + m_raw * a.scale + logf(l);   // log(w sm_den)
                const float log_l = logf(lin_den);                      // log(lin_den), -inf if empty
                const float sig = fmaxf(fmaxf(log_s, log_l), -60.f);
                const float esig = expf(-sig);
                const float cpos = lin_den > 0.f ? esig / sp : 0.f;
                const float cneg = lin_den > 0.f ? esig / sn : 0.f;
                for (int k = half; k < nfc; k += 2) {
                    float v[32], w[32];
                    tmem_ld32(tmem + lane_off + kColA + 32 * k, v);
                    tmem_ld32(tmem + lane_off + kColA + F + 32 * k, w);
                    tmem_wait_ld();
#pragma unroll
                    for (int i = 0; i < 32; ++i) { v[i] *= cpos; w[i] *= cneg; }
                    tmem_st32(tmem + lane_off + kColA + 32 * k, v);
                    tmem_st32(tmem + lane_off + kColA + F + 32 * k, w);
                }
                // P' = w e^(s - sigma): K-major, no swizzle (8-row x 16-byte core matrices)
                const float pofs = (lw - sig) * kLog2e;
                for (int k = half; k < nsc; k += 2) {
                    float v[16];
                    tmem_ld16(dcol + lane_off + 16 * k, v);
                    tmem_wait_ld();
                    uint32_t pk[8];
#pragma unroll
                    for (int i = 0; i < 16; i += 2)
                        pk[i / 2] = pack_bf16x2(ex2(fmaf(v[i], scale_l2, pofs)), ex2(fmaf(v[i + 1], scale_l2, pofs)));
                    uint8_t *prow = smem + a.off_p + (row >> 3) * (B / 8) * 128 + (row & 7) * 16;
                    *reinterpret_cast<uint4 *>(prow + (2 * k) * 128) = make_uint4(pk[0], pk[1], pk[2], pk[3]);
                    *reinterpret_cast<uint4 *>(prow + (2 * k + 1) * 128) = make_uint4(pk[4], pk[5], pk[6], pk[7]);
                }
                if (half == 0) den[row] = expf(log_l - sig) + expf(log_s - sig);
                if (kCommit && fval) {
                    const float4 *ip = reinterpret_cast<const float4 *>(&tk[6 * 128 + 16 * half]);
                    const float4 *in = reinterpret_cast<const float4 *>(&tk[7 * 128 + 16 * half]);
                    uint8_t *rp = pt_s + row * 128;
                    uint8_t *rn = pt_s + (F + row) * 128;
                    float dzp = 0.f, dzn = 0.f;
                    float4 x[4], y[4], a4[4], b4[4];
#pragma unroll
                    for (int gq = 0; gq < 4; ++gq) {
                        const int gi = 4 * half + gq;
                        x[gq] = *reinterpret_cast<const float4 *>(rp + ((gi ^ (row & 7)) << 4));
                        y[gq] = *reinterpret_cast<const float4 *>(rn + ((gi ^ ((F + row) & 7)) << 4));
                        a4[gq] = ip[gq];
                        b4[gq] = in[gq];
                    }
#pragma unroll
                    for (int gq = 0; gq < 4; ++gq) {
                        const int gi = 4 * half + gq;
                        x[gq].x *= a4[gq].x; x[gq].y *= a4[gq].y; x[gq].z *= a4[gq].z; x[gq].w *= a4[gq].w;
                        y[gq].x *= b4[gq].x; y[gq].y *= b4[gq].y; y[gq].z *= b4[gq].z; y[gq].w *= b4[gq].w;
                        *reinterpret_cast<float4 *>(rp + ((gi ^ (row & 7)) << 4)) = x[gq];
                        *reinterpret_cast<float4 *>(rn + ((gi ^ ((F + row) & 7)) << 4)) = y[gq];
                        dzp += (x[gq].x + x[gq].y) + (x[gq].z + x[gq].w);
                        dzn += (y[gq].x + y[gq].y) + (y[gq].z + y[gq].w);
                    }
                    atomicAdd(&zs[row], dzp);
                    atomicAdd(&zs[F + row], dzn);
                }
                tmem_wait_st();
            }
            fence_proxy_async_smem();
            tc_fence_before();
            if (math_sync_failed(!ok)) break;
            if (mt == 0) {
                mbar_arrive(phiready);
                if (kCommit) {
                    mbar_arrive(vtready);
                    mbar_arrive(zdone);
                } else {
                    mbar_arrive(&zempty[zb]);
                }
            }

            // ---- state update: S^T tile rows += dS^T rows (per feature half), then store
            if (kCommit) {
                const int e = row;
                const int fpt = F / 2;   // features per thread within a half
                bool brk = false;
                const uint32_t dother = tmem + kColD0 + 128 * ((kp + 1) & 1);
                for (int h = 0; h < 2; ++h) {
                    ok = wait_bar(&dsready[h], kp & 1u, fail);
                    // the second half's tiles are modified only after the readout has read them
                    if (h == 1 && ok) ok = wait_bar(rdone, kp & 1u, fail);
                    tc_fence_after();
                    for (int j = 0; j < fpt / 32; ++j) {
                        const int fl = half * fpt + 32 * j;           // feature offset within the half
                        const int c = (h * F + fl) / 32;              // state tile
                        const int slot = (q + c) % NS;
                        float v[32];
                        tmem_ld32((h == 0 ? tmem + kColA : dother) + lane_off + fl, v);
                        uint8_t *rowp = ring + (size_t)slot * chunk_bytes + e * 128;
                        float4 s[8];
                        if (e < d) {
#pragma unroll
                            for (int gq = 0; gq < 8; ++gq) s[gq] = *reinterpret_cast<const float4 *>(rowp + ((gq ^ (e & 7)) << 4));
                        }
                        tmem_wait_ld();
                        if (ok && e < d) {
#pragma unroll
                            for (int gq = 0; gq < 8; ++gq) {
                                s[gq].x += v[4 * gq];
                                s[gq].y += v[4 * gq + 1];
                                s[gq].z += v[4 * gq + 2];
                                s[gq].w += v[4 * gq + 3];
                            }
#pragma unroll
                            for (int gq = 0; gq < 8; ++gq) *reinterpret_cast<float4 *>(rowp + ((gq ^ (e & 7)) << 4)) = s[gq];
                        }
                    }
                    fence_proxy_async_smem();
                    tc_fence_before();
                    if (math_sync_failed(!ok)) { brk = true; break; }
                    if (mt == 0) {
                        mbar_arrive(&tready[h]);
                        if (h == 1) mbar_arrive(efree);
                    }
                }
                if (brk) break;
            }

            // ---- output epilogue: out = D / den, staged as the TMA box image in the
            // unit's last two ring slots (row i = t*G + hh, 128-byte swizzle)
            ok = wait_bar(&dready[kp & 1], (kp >> 1) & 1u, fail);
            if (ok) ok = wait_bar(ofree, kp & 1u, fail);
            tc_fence_after();
            {
                const int dh = d / 2;
                const float inv = 1.f / den[row];
                float v[2][32];
                tmem_ld32(dcol + lane_off + half * dh, v[0]);
                if (dh > 32) tmem_ld32(dcol + lane_off + half * dh + 32, v[1]);
                tmem_wait_ld();
                if (ok && valid) {
                    // d = 128: column half -> slot; d = 64: token half -> slot (one 64-column atom)
                    const int rows_half = G * B / 2;
                    const int sidx = d == 128 ? half : (row >= rows_half ? 1 : 0);
                    const int srow = d == 128 ? row : row - sidx * rows_half;
                    const int oc = kCommit ? ocm : NC - 2;
                    uint8_t *base = ring + (size_t)((q + oc + sidx) % NS) * chunk_bytes + srow * 128;
#pragma unroll
                    for (int hc = 0; hc < 2; ++hc) {
                        if (hc * 32 >= dh) break;
                        uint32_t pk[16];
#pragma unroll
                        for (int i = 0; i < 32; i += 2) pk[i / 2] = pack_bf16x2(v[hc][i] * inv, v[hc][i + 1] * inv);
#pragma unroll
                        for (int i = 0; i < 4; ++i) {
                            const int gi = 4 * hc + i + (d == 128 ? 0 : 4 * half);   // 16-byte granule in the 128-byte row
                            *reinterpret_cast<uint4 *>(base + ((gi ^ (srow & 7)) << 4)) =
                                make_uint4(pk[4 * i], pk[4 * i + 1], pk[4 * i + 2], pk[4 * i + 3]);
                        }
                    }
                }
            }
            fence_proxy_async_smem();
            tc_fence_before();
            if (math_sync_failed(!ok)) break;
            if (mt == 0) {
                mbar_arrive(ostaged);
                mbar_arrive(&dfree[kp & 1]);
            }
            q += NC;
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

// cuTensorMapEncodeTiled from the driver, looked up once through the runtime.
PFN_cuTensorMapEncodeTiled_v12000 encode_fn()
{
    static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
    static std::once_flag once;
    std::call_once(once, [] {
        void *p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
    });
    return fn;
}

// bf16 tensor map with the 128-byte swizzle; dims and box innermost first,
// strides (bytes) of dims 1..rank-1.
bool encode_bf16(CUtensorMap *m, const void *base, int rank, const cuuint64_t *dims, const cuuint64_t *strides,
                 const cuuint32_t *box)
{
    PFN_cuTensorMapEncodeTiled_v12000 fn = encode_fn();
    if (!fn) return false;
    const cuuint32_t es[3] = {1, 1, 1};
    return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, (cuuint32_t)rank, const_cast<void *>(base), dims, strides, box, es,
              CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_128B,
              CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

int sm_count()
{
    static int cached[64] = {0};
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 148;
    if (!cached[dev]) {
        int n = 0;
        if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n <= 0) n = 148;
        cached[dev] = n;
    }
    return cached[dev];
}

}  // namespace

bool fused_supported(const hybrid_cfg &c, bool commit)
{
    if (c.io_dtype != HYBRID_BF16) return false;
    if (c.head_dim != 64 && c.head_dim != 128) return false;
    if (c.feat_dim != 64 && c.feat_dim != 128) return false;
    if (c.block_size % 16 != 0) return false;
    const int G = c.n_q_heads / c.n_kv_heads;
    if (G * c.block_size > 128) return false;
    if (commit && c.block_size != 32) return false;
    const FLayout L = make_flayout(c.head_dim, c.feat_dim, c.block_size);
    const int NC = 2 * c.feat_dim / 32;
    // the commit keeps the first feature half resident while the second streams
    if (L.NS < (commit ? NC / 2 + 2 : 4)) return false;
    // region X must also hold V^T and phi(K)^T for the commit
    if (commit && (uint32_t)(128 * 128 + 2 * c.feat_dim * 128) > L.off_vb - L.off_q) return false;
    return (int)L.bytes <= kSmemLimit;
}

cudaError_t launch_fused(const hybrid_cfg &c, bool commit, const void *Q, const void *K, const void *V,
                         const void *W, const float *alpha, void *const *states, int n_req, void *O,
                         unsigned *err, cudaStream_t st)
{
    const FLayout L = make_flayout(c.head_dim, c.feat_dim, c.block_size);
    FusedArgs a;
    {
        const int d = c.head_dim, F = c.feat_dim, B = c.block_size, Hq = c.n_q_heads, Hkv = c.n_kv_heads;
        const int G = Hq / Hkv;
        const cuuint64_t rows = (cuuint64_t)n_req * B;
        const cuuint64_t dq[3] = {(cuuint64_t)d, (cuuint64_t)Hq, rows};
        const cuuint64_t sq[2] = {(cuuint64_t)d * 2, (cuuint64_t)Hq * d * 2};
        const cuuint32_t bq[3] = {64, (cuuint32_t)G, (cuuint32_t)B};
        const cuuint64_t dk[3] = {(cuuint64_t)d, (cuuint64_t)Hkv, rows};
        const cuuint64_t sk[2] = {(cuuint64_t)d * 2, (cuuint64_t)Hkv * d * 2};
        const cuuint32_t bk[3] = {64, 1, (cuuint32_t)B};
        const cuuint64_t dw[2] = {(cuuint64_t)F, (cuuint64_t)Hkv * d};
        const cuuint64_t sw[1] = {(cuuint64_t)F * 2};
        const cuuint32_t bw[2] = {64, (cuuint32_t)d};
        if (!encode_bf16(&a.tmQ, Q, 3, dq, sq, bq) || !encode_bf16(&a.tmK, K, 3, dk, sk, bk) ||
            !encode_bf16(&a.tmV, V, 3, dk, sk, bk) || !encode_bf16(&a.tmW, W, 2, dw, sw, bw))
            return cudaErrorInvalidValue;
        const cuuint32_t bo[3] = {64, (cuuint32_t)G, (cuuint32_t)(d == 128 ? B : B / 2)};
        if (!encode_bf16(&a.tmO, O, 3, dq, sq, bo))
            return cudaErrorInvalidValue;
    }
    a.Q = static_cast<const bf16 *>(Q);
    a.K = static_cast<const bf16 *>(K);
    a.V = static_cast<const bf16 *>(V);
    a.W = static_cast<const bf16 *>(W);
    a.alpha = alpha;
    a.states = states;
    a.O = static_cast<bf16 *>(O);
    a.err = err;
    a.n_units = n_req * c.n_kv_heads;
    a.B = c.block_size;
    a.Hq = c.n_q_heads;
    a.Hkv = c.n_kv_heads;
    a.G = c.n_q_heads / c.n_kv_heads;
    a.d = c.head_dim;
    a.F = c.feat_dim;
    a.NS = L.NS;
    a.scale = 1.f / sqrtf((float)c.head_dim);
    a.off_q = L.off_q;
    a.off_w = L.off_w;
    a.off_k = L.off_k;
    a.off_vb = L.off_vb;
    a.off_p = L.off_p;
    a.off_z = L.off_z;
    a.off_st = L.off_st;
    a.off_bar = L.off_bar;
    const int grid = a.n_units < sm_count() ? a.n_units : sm_count();
    // opt in to the full shared memory once per device and kernel (the attribute
    // is set to the maximum, so every layout fits)
    static std::atomic<unsigned long long> opted[2];
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
    const unsigned long long bit = 1ull << dev;
    if (!(opted[commit].load(std::memory_order_acquire) & bit)) {
        const cudaError_t e = commit ? cudaFuncSetAttribute(k_fused<true>, cudaFuncAttributeMaxDynamicSharedMemorySize, kSmemLimit)
                                     : cudaFuncSetAttribute(k_fused<false>, cudaFuncAttributeMaxDynamicSharedMemorySize, kSmemLimit);
        if (e != cudaSuccess) return e;
        opted[commit].fetch_or(bit, std::memory_order_release);
    }
    if (commit) k_fused<true><<<grid, kThreads, L.bytes, st>>>(a);
    else k_fused<false><<<grid, kThreads, L.bytes, st>>>(a);
    return cudaGetLastError();
}

}  // namespace hyb
