// hybrid_fused.cu -- persistent, warp-specialised block-hybrid step fused with
// the block commit, on the tcgen05 tensor cores.
//
// Section 3.1 of "Retrofitting Linear Attention into Diffusion Language
// Models" defines the step (in-block softmax, linear readout from the committed
// state, gated shared-normaliser merge) and the state update; its serving
// section computes both in one kernel launch, as this kernel does: every state
// tile is read once, used for the readout with the pre-commit state, and
// updated with this block's phi(k) v^T.
//
// Work unit = (request r, state head g): the G*B query rows of the unit share
// one state.  One CTA per SM loops over a contiguous range of units.  Warp
// roles (12 warps):
//   warp 0     S producer: z and the 2F/32 state tiles of each unit, by 1-D bulk
//              copies, through an NS-slot ring (the state layout is the MMA
//              operand image, see hybrid.h).
//   warp 1     MMA issuer (one thread); owns the Tensor Memory allocation.
//   warp 2     producer: TMA of Q, W, K and V.
//   warp 3     storer: bulk stores of the updated state tiles and of z, and TMA
//              stores of the output tile.
//   warps 4-11 math: two threads per query row (one per TMEM lane and "part");
//              a part owns every other 32-feature chunk of each half of phi.
//
// Per unit the tensor cores run, in this order,
//   g1   U = Q W, scores = Q K^T and U_k^T = W^T K^T (phi of the block's keys);
//        K, as loaded, is the K-major operand of the last two
//   R+   D  = phi+'(Q) S+             (tf32, A operand in Tensor Memory)
//   dS   dS^T = V^T phi(K)^T per feature half (bf16 from the TMA'd V)
//   PV   D += P' V                    (P' = w e^(s - sigma), bf16)
//   R-   D += phi-'(Q) S-
// The math warps publish phi+ as soon as its exponentials are in Tensor
// Memory (R+ then overlaps the rest of the feature map), then compute phi-,
// the row statistics, phi(K) (signalled first, so dS^T is formed meanwhile)
// and P', and out = D / den after R-.  Merge: with sigma the log of the
// larger branch mass, phi' = phi e^-sigma and P' = w e^(s - sigma), so
// D / den = (w sm_num + lin_num) / (w sm_den + lin_den) exactly, with
// den = e^(log lin_den - sigma) + e^(log(w sm_den) - sigma) in [1, 2].  While
// the unshifted softmax mass w sp e^s of a warp's rows stays below e^60, the
// kernel accumulates D / kappa (kappa = e^-sigma / sp) instead, so phi+ needs
// no rescaling in Tensor Memory; kappa is folded into 1 / den.
//
// Tensor Memory: [D | phi | dS+ | dS-].  phi+ is parked in the dS- columns
// while R+ reads it; phi- replaces U in the phi columns.  Once a half's tiles
// have been read out, each still sits in its ring slot as read: the math warps
// add that half's dS^T rows to it there (float32) and the storer writes the
// tiles back over the state with plain bulk stores (a bulk reduce-add at L2
// would do the same add, but with every SM committing at once L2 takes 2.8 TB/s
// of added data, against ~6 TB/s of plain stores).  V, P' and phi(K) share the
// Q region once g1 has consumed Q, so all 2F/32 state tiles of a unit fit in
// the ring.
//
// MMA cost note: on this part a tcgen05.mma with M = 128 costs its issuing thread
// about the same time for any N up to 128-256, so contractions are shaped for few,
// wide instructions (dS^T is two N = F products).
#include <cuda.h>
#include <cudaTypedefs.h>

#include <atomic>
#include <mutex>

#include "hybrid_common.cuh"
#include "hybrid_tc.h"
#include "tc_pipeline.cuh"

namespace hyb {

namespace {

using namespace pipe;

constexpr int kWarps = 12;
constexpr int kThreads = kWarps * 32;
constexpr int kMathThreads = 256;
constexpr int kMaxSlots = 16;
constexpr int kSmemLimit = 232448;
constexpr int kOneCtaPerSm = 118 * 1024;
constexpr uint32_t kBarMath = 1;      // named barrier over the 256 math threads
constexpr uint32_t kStatBytes = 14 * 1024;
// Tensor Memory columns with the commit (F <= 128, d <= 128)
constexpr uint32_t kCmD = 0, kCmP = 128, kCmDSp = 256, kCmK = 288, kCmDSm = 384;
// unnormalised phi(K) parked between the two exchanges of the math warps (free
// columns until dS+ is formed)
constexpr uint32_t kCmEK = 320;

struct FusedArgs {
    // Q, O [n*B][Hq][d], K, V [n*B][Hkv][d], W [Hkv*d][F]; 128-byte swizzle.  Q, K, V
    // and W with the 64-element panels as the outermost box dimension (one copy each);
    // Q's box is 128 / G tokens deep over a dimension of B, so the rows of a unit's
    // 128-row tile beyond G B are zero-filled.
    CUtensorMap tmQ, tmK, tmV, tmW, tmO;
    const float *alpha;
    void *const *states;
    unsigned *err;
    int n_units, B, Hq, Hkv, G, d, F, NS;
    float scale;
    uint32_t off_q, off_wk, off_vb, off_p, off_pk, off_z, off_st, off_bar;
};

// Shared memory: [ring NS x d*128][Q][W][K][V][P'][phi(K)][z x2][stats][barriers]
// (V, P' and phi(K) overlay the Q region once g1 has read Q).  Q, K, V and W land
// by TMA with the 128-byte swizzle: Q as d/64 atoms of 128 rows (16 KB apart;
// rows t*G + h), K and V as d/64 atoms of B rows (K the K-major operand, V the
// MN-major one: 8-row groups 1 KB apart, atoms B*128 apart), W as F/64 atoms of
// d rows (MN-major: e-groups 1 KB apart, atoms d*128 apart).
struct FLayout {
    uint32_t off_q, off_wk, off_vb, off_p, off_pk, off_z, off_st, off_bar, bytes;
    int NS;
};

FLayout make_flayout(int d, int F, int B)
{
    FLayout L{};
    const uint32_t chunk = (uint32_t)d * 128;
    const uint32_t zb = (((uint32_t)2 * F * 4) + 1023) & ~1023u;
    const uint32_t q = (uint32_t)d * 256;
    const uint32_t wk = (uint32_t)(F / 64) * d * 128 + ((((uint32_t)B * d * 2) + 1023) & ~1023u);
    const uint32_t vb = (((uint32_t)B * d * 2) + 1023) & ~1023u;
    const uint32_t p = (((uint32_t)128 * B * 2) + 1023) & ~1023u;
    const uint32_t pk = (((uint32_t)(2 * F / 64) * B * 128) + 1023) & ~1023u;
    const uint32_t bar = 1024;
    // V, P' and phi(K) live in the Q region once g1 has read Q (the next unit's
    // Q is loaded after the unit's dS^T and P V are done)
    const bool overlay = vb + p + pk <= q;
    const uint32_t fixed = q + wk + (overlay ? 0u : vb + p + pk) + 2 * zb + kStatBytes + bar + 1024;
    int ns = ((int)kSmemLimit - (int)fixed) / (int)chunk;
    if (ns > kMaxSlots) ns = kMaxSlots;
    L.NS = ns;
    uint32_t off = (uint32_t)(ns > 0 ? ns : 0) * chunk;
    L.off_q = off; off += q;
    L.off_wk = off; off += wk;
    if (overlay) {
        L.off_vb = L.off_q;
        L.off_p = L.off_q + vb;
        L.off_pk = L.off_q + vb + p;
    } else {
        L.off_vb = off; off += vb;
        L.off_p = off; off += p;
        L.off_pk = off; off += pk;
    }
    L.off_z = off; off += 2 * zb;
    L.off_st = off; off += kStatBytes;
    L.off_bar = off; off += bar;
    L.bytes = off + 1024;
    if ((int)L.bytes < kOneCtaPerSm) L.bytes = kOneCtaPerSm;
    return L;
}

// Every role walks the same units and skips those whose state pointer fails its
// check.  The pointer of the next unit is loaded one unit ahead (state_raw), so
// its latency hides behind the current unit; state_at checks it when it is used.
__device__ __forceinline__ void *state_raw(const FusedArgs &a, int u, int u_end)
{
    return u < u_end ? a.states[u / a.Hkv] : nullptr;
}
__device__ __forceinline__ float *state_at(const FusedArgs &a, void *raw, int u)
{
    float *st = reinterpret_cast<float *>(raw);
    if (!state_ptr_ok(st)) return nullptr;
    return st + (size_t)(u % a.Hkv) * head_floats(a.d, a.F);
}

__global__ void __launch_bounds__(kThreads, 1) k_fused(const __grid_constant__ FusedArgs a)
{
    using namespace ptx;
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int d = a.d, F = a.F, B = a.B, G = a.G, NS = a.NS;
    const uint64_t wlim = kWaitNs;
    const int NCH = F / 32;          // 32-feature chunks (state tiles) per half of phi
    const int NC = 2 * NCH;          // state tiles per unit
    // the output tile is staged in the slots of tiles ocm, ocm + 1 of its unit:
    // the first two second-half tiles (their updated copies are stored before the
    // epilogue), so the next unit's first-half tiles, needed first, can enter
    // the ring early; if a unit has more tiles than the ring, first-half tiles
    // that no later tile of the unit reuses
    const int ocm = NC > NS ? NC - NS : NCH;
    const uint32_t chunk_bytes = (uint32_t)d * 128;
    const int per = a.n_units / (int)gridDim.x, rem = a.n_units % (int)gridDim.x;
    const int u_begin = (int)blockIdx.x * per + min((int)blockIdx.x, rem);
    const int u_end = u_begin + per + ((int)blockIdx.x < rem ? 1 : 0);

    uint64_t *bars = reinterpret_cast<uint64_t *>(smem + a.off_bar);
    uint64_t *full = bars;
    uint64_t *empty = full + NS;
    uint64_t *zfull = empty + NS;     // [2]
    uint64_t *zempty = zfull + 2;     // [2]
    uint64_t *dready = zempty + 2;    // [2] MMA -> math: the unit's output accumulator is complete
    uint64_t *tready = dready + 2;    // [2] math -> storer: a feature half of the tiles is updated
    uint64_t *xfull = tready + 2;     // Q, W and K have landed
    uint64_t *uready = xfull + 1;     // MMA -> math: g1 done
    uint64_t *phip = uready + 1;      // math -> MMA: phi+ is in the dS- columns
    uint64_t *phim = phip + 1;        // math -> MMA: phi- in the phi columns
    uint64_t *pready = phim + 1;      // math -> MMA: P' is written
    uint64_t *mmadone = pready + 1;   // the issuing thread's MMAs have completed
    uint64_t *xfree = mmadone + 1;
    uint64_t *vfull = xfree + 1;
    uint64_t *kready = vfull + 1;     // math -> MMA: phi(K) is written
    uint64_t *dsdone = kready + 1;    // MMA -> math: dS^T is formed
    uint64_t *pvdone = dsdone + 1;    // MMA -> producer: P V has read V and P'
    uint64_t *efree = pvdone + 1;     // math -> MMA: the first-half update has read dS+
    uint64_t *zdone = efree + 1;      // math -> storer: z is updated
    uint64_t *ofree = zdone + 1;      // storer -> math: the output slots may be written
    uint64_t *ostaged = ofree + 1;    // math -> storer: the output tile is in its slots
    const int n_bars = 2 * NS + 8 + 15;
    uint32_t *tmem_holder = reinterpret_cast<uint32_t *>(bars + n_bars);
    volatile int *fail = reinterpret_cast<volatile int *>(tmem_holder + 1);

    if (warp == 2 && lane == 0) {
        prefetch_tensormap(&a.tmQ);
        prefetch_tensormap(&a.tmW);
        prefetch_tensormap(&a.tmK);
        prefetch_tensormap(&a.tmV);
    }
    if (warp == 3 && lane == 0) prefetch_tensormap(&a.tmO);
    if (tid == 0) {
        for (int i = 0; i < n_bars; ++i) mbar_init(&bars[i], 1);
        mbar_init(xfull, 2);
        mbar_init(phip, 8);
        mbar_init(phim, 8);
        mbar_init(pready, 8);
        for (int i = 0; i < 2; ++i) mbar_init(&tready[i], 8);
        mbar_init(kready, 8);
        mbar_init(efree, 8);
        mbar_init(zdone, 8);
        mbar_init(ostaged, 8);
        *fail = 0;
        fence_mbar_init();
    }
    if (warp == 1) {
        tmem_alloc(tmem_holder, 512);
        tmem_relinquish();
    }
    __syncthreads();
    tc_fence_after();
    // launched with programmatic stream serialisation: the set-up above may run
    // while the previous kernel of the stream drains; nothing below touches
    // global memory before that kernel has completed
    if (tid == 0) griddep_launch_dependents();
    // the Q, K and V boxes of the CTA's units into L2 while the previous kernel drains: a
    // prefetch brings no value into the SM, so it needs no ordering after that kernel
    if (tid == 64)
        for (int u = u_begin; u < u_end && u < u_begin + 2; ++u) {
            const int r = u / a.Hkv, g = u % a.Hkv;
            tma_prefetch_5d(&a.tmQ, 0, g * G, 0, r, 0);
            tma_prefetch_4d(&a.tmK, 0, g, r * B, 0);
            tma_prefetch_4d(&a.tmV, 0, g, r * B, 0);
        }
    griddep_wait();
    const uint32_t tmem = *tmem_holder;
    uint8_t *ring = smem;
    float *zbuf0 = reinterpret_cast<float *>(smem + a.off_z);
    const int zstride = ((2 * F * 4 + 1023) & ~1023) / 4;

    if (warp == 0) {
        // ------------------------------------------------------- S producer
        if (lane == 0) {
            uint32_t q = 0, kp = 0;
            int issued_slot[kMaxSlots];
            int issued_z[2] = {0, 0};
            for (int i = 0; i < kMaxSlots; ++i) issued_slot[i] = 0;
            bool ok = true;
            void *nraw = state_raw(a, u_begin, u_end);
            for (int u = u_begin; u < u_end && ok; ++u) {
                void *raw = nraw;
                nraw = state_raw(a, u + 1, u_end);
                float *Sg = state_at(a, raw, u);
                if (!Sg) continue;
                const int zb = kp & 1;
                if (!wait_bar(&zempty[zb], ((kp >> 1) & 1u) ^ 1u, fail, wlim)) break;
                mbar_arrive_expect_tx(&zfull[zb], 2 * F * 4);
                bulk_g2s(zbuf0 + zb * zstride, Sg + (size_t)2 * F * d, 2 * F * 4, &zfull[zb]);
                ++issued_z[zb];
                if (kp == 0 && !wait_bar(xfull, 0, fail, wlim)) break;
                for (int c = 0; c < NC; ++c, ++q) {
                    const int slot = q % NS;
                    if (!wait_bar(&empty[slot], ((q / NS) & 1u) ^ 1u, fail, wlim)) { ok = false; break; }
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
            const uint32_t q_u = smem_u32(smem + a.off_q), wk_u = smem_u32(smem + a.off_wk),
                           vb_u = smem_u32(smem + a.off_vb), p_u = smem_u32(smem + a.off_p),
                           pk_u = smem_u32(smem + a.off_pk), ring_u = smem_u32(ring);
            const uint32_t k_u = wk_u + (uint32_t)(F / 64) * d * 128;   // K: d/64 atoms of B rows
            const uint32_t idU = instr_desc(FMT_BF16, FMT_BF16, false, true, 128, F);
            const uint32_t idS = instr_desc(FMT_BF16, FMT_BF16, false, false, 128, B);
            const uint32_t idKT = instr_desc(FMT_BF16, FMT_BF16, true, false, 128, B);
            const uint32_t idR = instr_desc(FMT_TF32, FMT_TF32, false, false, 128, d);
            const uint32_t idP = instr_desc(FMT_BF16, FMT_BF16, false, true, 128, d);
            const uint32_t idDS = instr_desc(FMT_BF16, FMT_BF16, true, true, 128, F);
            // g1: U = Q W at column ucol and the scores Q K^T after it, U_k^T = W^T K^T at
            // column kcol; K as loaded is the K-major operand of both
            auto g1 = [&](uint32_t ucol, uint32_t kcol) {
                for (int k = 0; k < d / 16; ++k) {
                    const uint64_t aq = smem_desc(q_u + (k >> 2) * (128 * 128) + (k & 3) * 32, 16, 1024, SWZ_128B);
                    const uint64_t bw = smem_desc(wk_u + 2 * k * 1024, d * 128, 1024, SWZ_128B);
                    const uint64_t bk = smem_desc(k_u + (k >> 2) * (B * 128) + (k & 3) * 32, 16, 1024, SWZ_128B);
                    mma_bf16_ss(tmem + ucol, aq, bw, idU, k > 0);
                    mma_bf16_ss(tmem + ucol + F, aq, bk, idS, k > 0);
                    mma_bf16_ss(tmem + kcol, bw, bk, idKT, k > 0);
                }
            };
            // P'V accumulates onto the phi+ readout
            auto pv = [&](uint32_t dcol) {
                for (int k = 0; k < B / 16; ++k) {
                    const uint64_t ap = smem_desc(p_u + k * 256, 128, (B / 8) * 128, SWZ_NONE);
                    const uint64_t bv = smem_desc(vb_u + 2 * k * 1024, B * 128, 1024, SWZ_128B);
                    mma_bf16_ss(tmem + dcol, ap, bv, idP, 1);
                }
            };
            // readout of the next state tile in the ring with phi columns acol
            // (first: the tile's first MMA initialises the accumulator)
            uint32_t rs = 0, rph = 0;   // ring slot and phase of the next tile, read in ring order
            auto readout = [&](uint32_t dcol, uint32_t acol, bool first = false) -> int {
                const int slot = (int)rs;
                if (!wait_bar(&full[slot], rph, fail, wlim)) return -1;
                if (++rs == (uint32_t)NS) { rs = 0; rph ^= 1u; }
                tc_fence_after();
                const uint32_t s_u = ring_u + slot * chunk_bytes;
#pragma unroll
                for (int kk = 0; kk < 4; ++kk)
                    mma_tf32_ts(tmem + dcol, tmem + acol + 8 * kk, smem_desc(s_u + 32 * kk, 16, 1024, SWZ_128B), idR,
                                !(first && kk == 0));
                return slot;
            };
            auto ds = [&](uint32_t dcol, int h) {
                for (int ks = 0; ks < B / 16; ++ks) {
                    const uint64_t av = smem_desc(vb_u + ks * 2048, B * 128, 1024, SWZ_128B);
                    const uint64_t bp = smem_desc(pk_u + (uint32_t)h * (F / 64) * (B * 128) + ks * 2048, B * 128, 1024,
                                                  SWZ_128B);
                    mma_bf16_ss(tmem + dcol, av, bp, idDS, ks > 0);
                }
            };
            uint32_t kp = 0;
            bool ok = true;
            void *nraw = state_raw(a, u_begin, u_end);
            for (int u = u_begin; u < u_end; ++u) {
                void *raw = nraw;
                nraw = state_raw(a, u + 1, u_end);
                if (!state_at(a, raw, u)) continue;
                if (!wait_bar(xfull, kp & 1u, fail, wlim)) { ok = false; break; }
                // U_k^T and the scores land in the dS+ columns: the previous unit's
                // first-half update must have read them (its R- precedes in issue order)
                if (kp >= 1 && !wait_bar(efree, (kp - 1) & 1u, fail, wlim)) { ok = false; break; }
                tc_fence_after();
                g1(kCmP, kCmK);
                mma_commit(uready);
                mma_commit(xfree);
                // phip also covers the previous unit's output epilogue and second-half update
                if (!wait_bar(phip, kp & 1u, fail, wlim)) { ok = false; break; }
                tc_fence_after();
                for (int c = 0; c < NCH && ok; ++c) ok = readout(kCmD, kCmDSm + 32 * c, c == 0) >= 0;
                if (!ok) break;
                if (!wait_bar(kready, kp & 1u, fail, wlim) || !wait_bar(vfull, kp & 1u, fail, wlim)) { ok = false; break; }
                tc_fence_after();
                ds(kCmDSp, 0);
                ds(kCmDSm, 1);
                mma_commit(dsdone);
                if (!wait_bar(pready, kp & 1u, fail, wlim)) { ok = false; break; }
                tc_fence_after();
                pv(kCmD);
                mma_commit(pvdone);
                if (!wait_bar(phim, kp & 1u, fail, wlim)) { ok = false; break; }
                tc_fence_after();
                for (int c = NCH; c < NC && ok; ++c) ok = readout(kCmD, kCmP + 32 * (c - NCH)) >= 0;
                if (!ok) break;
                mma_commit(&dready[kp & 1]);
                ++kp;
            }
            mma_commit(mmadone);
            mbar_wait(mmadone, 0, kWaitNs);
        }
    } else if (warp == 2) {
        // ------------------------------------------------------------- producer
        uint32_t kp = 0;
        int nx = 0, nv = 0;
        const uint32_t xbytes =
            (uint32_t)(d / 64) * (128 * 128) + (uint32_t)(F / 64) * (d * 128) + (uint32_t)(d / 64) * (B * 128);
        uint8_t *kb = smem + a.off_wk + (F / 64) * d * 128;
        void *nraw = state_raw(a, u_begin, u_end);
        for (int u = u_begin; u < u_end; ++u) {
            void *raw = nraw;
            nraw = state_raw(a, u + 1, u_end);
            if (!state_at(a, raw, u)) continue;
            const int r = u / a.Hkv, g = u % a.Hkv;
            bool ok = true;
            if (kp > 0) ok = wait_bar(xfree, (kp - 1) & 1u, fail, wlim);
            if (__any_sync(0xffffffffu, !ok)) break;
            // the Q region holds the previous unit's V, P' and phi(K) until its dS^T
            // and P V have run, so Q follows W and K (except for the first unit)
            const bool q_early = kp == 0;
            uint64_t *xf = xfull;
            if (lane == 0) {
                mbar_arrive_expect_tx(xf, xbytes);
                if (q_early) tma_load_5d(smem + a.off_q, &a.tmQ, 0, g * G, 0, r, 0, xf);
                tma_load_3d(smem + a.off_wk, &a.tmW, 0, g * d, 0, xf);
                tma_load_4d(kb, &a.tmK, 0, g, r * B, 0, xf);
            }
            __syncwarp();
            if (!q_early && kp > 0) ok = wait_bar(pvdone, (kp - 1) & 1u, fail, wlim);
            if (__any_sync(0xffffffffu, !ok)) break;
            if (lane == 0) {
                if (!q_early) tma_load_5d(smem + a.off_q, &a.tmQ, 0, g * G, 0, r, 0, xf);
                mbar_arrive(xf);
            }
            ++nx;
            // V shares the Q region: after this unit's g1 has read Q
            ok = wait_bar(xfree, kp & 1u, fail, wlim);
            if (__any_sync(0xffffffffu, !ok)) break;
            if (lane == 0) {
                mbar_arrive_expect_tx(vfull, (uint32_t)(d / 64) * (B * 128));
                tma_load_4d(smem + a.off_vb, &a.tmV, 0, g, r * B, 0, vfull);
            }
            ++nv;
            ++kp;
        }
        if (lane == 0 && *fail) {
            // let copies in flight land before the CTA exits
            if (nx) mbar_wait(xfull, (uint32_t)(nx - 1) & 1u, kWaitNs);
            if (nv) mbar_wait(vfull, (uint32_t)(nv - 1) & 1u, kWaitNs);
        }
    } else if (warp == 3) {
        // --------------------------------------------------------------- storer
        if (lane == 0) {
            uint32_t q = 0, kp = 0;
            void *nraw = state_raw(a, u_begin, u_end);
            for (int u = u_begin; u < u_end; ++u) {
                void *raw = nraw;
                nraw = state_raw(a, u + 1, u_end);
                float *Sg = state_at(a, raw, u);
                if (!Sg) continue;
                const int r = u / a.Hkv, g = u % a.Hkv;
                bool ok = true;
                const int zb = kp & 1;
                if (!wait_bar(zdone, kp & 1u, fail, wlim)) break;
                bulk_s2g(Sg + (size_t)2 * F * d, zbuf0 + zb * zstride, 2 * F * 4);
                bulk_commit();
                bulk_wait_read_all();
                mbar_arrive(&zempty[zb]);
                for (int h = 0; h < 2 && ok; ++h) {
                    if (!wait_bar(&tready[h], kp & 1u, fail, wlim)) { ok = false; break; }
                    // one bulk group per tile; the two output slots are freed as
                    // soon as their stores have read them
                    for (int c = h * NCH; c < (h + 1) * NCH; ++c) {
                        bulk_s2g(Sg + (size_t)c * 32 * d, ring + (size_t)((q + c) % NS) * chunk_bytes, chunk_bytes);
                        bulk_commit();
                    }
                    if (h == ocm / NCH) {
                        // the output slots may be written once their stores have read them
                        if ((h + 1) * NCH - (ocm + 2) >= 2) bulk_wait_read_2();
                        else bulk_wait_read_all();
                        mbar_arrive(ofree);
                    }
                    bulk_wait_read_all();
                    for (int c = h * NCH; c < (h + 1) * NCH; ++c)
                        if (c < ocm || c > ocm + 1) mbar_arrive(&empty[(q + c) % NS]);
                }
                if (!ok) break;
                // output tile: two TMA boxes from the two held-back slots
                if (!wait_bar(ostaged, kp & 1u, fail, wlim)) break;
                uint8_t *s0 = ring + (size_t)((q + ocm) % NS) * chunk_bytes;
                uint8_t *s1 = ring + (size_t)((q + ocm + 1) % NS) * chunk_bytes;
                if (d == 128) {
                    tma_store_3d(&a.tmO, 0, g * G, r * B, s0);
                    tma_store_3d(&a.tmO, 64, g * G, r * B, s1);
                } else {
                    tma_store_3d(&a.tmO, 0, g * G, r * B, s0);
                    tma_store_3d(&a.tmO, 0, g * G, r * B + B / 2, s1);
                }
                bulk_commit();
                bulk_wait_read_all();
                mbar_arrive(&empty[(q + ocm) % NS]);
                mbar_arrive(&empty[(q + ocm + 1) % NS]);
                q += NC;
                ++kp;
            }
            bulk_wait_all();
        }
    } else {
        // ------------------------------------------------------------- math
        const int mt = tid - 128;
        const int q4 = warp & 3, part = (warp - 4) >> 2;
        const int row = 32 * q4 + lane;
        const uint32_t lane_off = (uint32_t)(32 * q4) << 16;
        const bool two = NCH >= 4;          // a part owns chunks part and part + 2 of each half
        const bool has_sc = part < B / 16;  // score columns [16 part, 16 part + 16)
        const int Mv = G * B;
        const bool valid = row < Mv;
        const bool fval = row < F;
        float *xa = reinterpret_cast<float *>(smem + a.off_st);   // [part][ms, mx, mn][128]
        float *xs = xa + 6 * 128;                                  // [part][sp][128]
        float *xb = xs + 2 * 128;                                  // [part][l, lp, sn, ln][128]
        float *tk = xb + 8 * 128;                                  // token statistics (commit)
        uint8_t *pkb = smem + a.off_pk;
        const float scale_l2 = a.scale * kLog2e;
        // exchange point of all math warps
        auto sync_failed = [&](bool local_fail) -> bool { return group_sync_failed(kBarMath, kMathThreads, local_fail); };

        // out = D / den, staged as the TMA box image in the unit's held-back ring
        // slots (row i = t*G + hh, 128-byte swizzle) for the storer
        auto epilogue = [&](uint32_t ek, uint32_t eq, float inv) -> bool {
            bool ok = wait_bar(&dready[ek & 1], (ek >> 1) & 1u, fail, wlim);
            if (ok) ok = wait_bar(ofree, ek & 1u, fail, wlim);
            tc_fence_after();
            const int dh = d / 2;
            // d = 128: column half -> slot; d = 64: token half -> slot (one 64-column atom)
            const int rows_half = G * B / 2;
            const int sidx = d == 128 ? part : (row >= rows_half ? 1 : 0);
            const int srow = d == 128 ? row : row - sidx * rows_half;
            uint8_t *base = ring + (size_t)((eq + ocm + sidx) % NS) * chunk_bytes + srow * 128;
            for (int hc = 0; hc < dh / 32; ++hc) {
                float v[32];
                tmem_ld32(tmem + kCmD + lane_off + part * dh + 32 * hc, v);
                tmem_wait_ld();
                if (ok && valid) {
                    uint32_t pk[16];
#pragma unroll
                    for (int i = 0; i < 32; i += 2) pk[i / 2] = pack_bf16x2(v[i] * inv, v[i + 1] * inv);
#pragma unroll
                    for (int i = 0; i < 4; ++i) {
                        const int gi = 4 * hc + i + (d == 128 ? 0 : 4 * part);   // 16-byte granule in the row
                        *reinterpret_cast<uint4 *>(base + ((gi ^ (srow & 7)) << 4)) =
                            make_uint4(pk[4 * i], pk[4 * i + 1], pk[4 * i + 2], pk[4 * i + 3]);
                    }
                }
            }
            fence_proxy_async_smem();
            tc_fence_before();
            __syncwarp();
            if (lane == 0 && ok) mbar_arrive(ostaged);
            return ok;
        };

        uint32_t q = 0, kp = 0;
        void *nraw = state_raw(a, u_begin, u_end);
        float nalpha = valid && u_begin < u_end ? a.alpha[(u_begin % a.Hkv) * G + row % G] : 0.f;
        for (int u = u_begin; u < u_end; ++u) {
            void *raw = nraw;
            nraw = state_raw(a, u + 1, u_end);
            // gate of this row's query head, loaded one unit ahead
            const float alpha_row = nalpha;
            nalpha = valid && u + 1 < u_end ? a.alpha[((u + 1) % a.Hkv) * G + row % G] : 0.f;
            float *Sg = state_at(a, raw, u);
            if (!Sg) {
                if (mt == 0) raise_error(a.err, ERR_BAD_STATE_PTR);
                continue;
            }
            const int zb = kp & 1;
            float *zs = zbuf0 + zb * zstride;
            const uint32_t pcol = tmem + kCmP + lane_off;    // U, then phi-
            const uint32_t scol = pcol + F;                  // scores
            const uint32_t kcol = tmem + kCmK + lane_off;    // U_k^T
            // phi+ in the dS- columns (free until dS^T is formed), so U stays in place
            // for phi- and no thread holds U in registers
            const uint32_t ppcol = tmem + kCmDSm + lane_off;

            // ---- phase A: row extrema of U and of the scores, and the per-token
            // extrema of U_k^T over this warp's 32 features
            bool bad = !wait_bar(uready, kp & 1u, fail, wlim);
            tc_fence_after();
            float sc[16];
            {
                // phi(K): thread (feature row, part) owns feature part*F + row of every
                // token; part 0 needs the per-token max of U_k over features, part 1
                // the min (features on lanes: reduce over the warp, then the quarters)
                float uk[32];
                tmem_ld32(kcol, uk);
                tmem_wait_ld();
#pragma unroll
                for (int t = 0; t < 32; ++t) uk[t] = fval ? (part == 0 ? uk[t] : -uk[t]) : -INFINITY;
                const float ext = warp_reduce32<1>(uk, lane);
                tk[(part * 32 + lane) * 4 + q4] = ext;   // max of +-U_k for token lane
            }
            if (has_sc) tmem_ld16(scol + 16 * part, sc);
            tmem_wait_ld();
            {
                float ms = -INFINITY, mx = -INFINITY, mn = INFINITY;
                if (has_sc) {
#pragma unroll
                    for (int i = 0; i < 16; ++i) ms = fmaxf(ms, sc[i]);
                }
                // this thread's 32-feature chunks of U, one at a time
#pragma unroll 1
                for (int k = part; k < NCH; k += 2) {
                    float x[32];
                    tmem_ld32(pcol + 32 * k, x);
                    tmem_wait_ld();
#pragma unroll
                    for (int i = 0; i < 32; ++i) { mx = fmaxf(mx, x[i]); mn = fminf(mn, x[i]); }
                }
                xa[(part * 3 + 0) * 128 + row] = ms;
                xa[(part * 3 + 1) * 128 + row] = mx;
                xa[(part * 3 + 2) * 128 + row] = mn;
            }
            if (sync_failed(bad)) break;
            const float ms = fmaxf(xa[0 * 128 + row], xa[3 * 128 + row]);
            const float mx = fmaxf(xa[1 * 128 + row], xa[4 * 128 + row]);
            const float mn = fminf(xa[2 * 128 + row], xa[5 * 128 + row]);

            // ---- phase B1: phi+ (unnormalised) into Tensor Memory; once the row sums are
            // exchanged, R+ may start on it (unless the warp needs the exact rescale)
            bad = !wait_bar(&zfull[zb], (kp >> 1) & 1u, fail, wlim);
            const float mxl = mx * kLog2e, mnl = mn * kLog2e, ml = ms * scale_l2;
            const float lw = valid ? log_sigmoid(alpha_row) : 0.f;
            float lp = 0.f;
            {
                float sp = 0.f;
                auto expp = [&](const float (&uu)[32], int k) {
                    float ep[32];
                    const float4 *zp = reinterpret_cast<const float4 *>(zs + 32 * k);
#pragma unroll
                    for (int i4 = 0; i4 < 8; ++i4) {
                        const float4 a4 = zp[i4];
                        const float za[4] = {a4.x, a4.y, a4.z, a4.w};
#pragma unroll
                        for (int j = 0; j < 4; ++j) {
                            const int i = 4 * i4 + j;
                            const float e = ex2(fmaf(uu[i], kLog2e, -mxl));
                            ep[i] = e;
                            sp += e;
                            lp = fmaf(e, za[j], lp);
                        }
                    }
                    tmem_st32(ppcol + 32 * k, ep);
                };
#pragma unroll 1
                for (int k = part; k < NCH; k += 2) {
                    float x[32];
                    tmem_ld32(pcol + 32 * k, x);
                    tmem_wait_ld();
                    expp(x, k);
                }
                xs[part * 128 + row] = sp;
            }
            if (sync_failed(bad)) break;
            const float sp = xs[row] + xs[128 + row];
            // Accumulate D / kappa with kappa = e^-sigma / sp: phi+ then stays
            // unnormalised in Tensor Memory (no rescale pass) and phi- (in registers)
            // and P' absorb the factor (phi- x sp/sn, P' = w sp e^s).  This needs the
            // unshifted softmax mass w sp e^(s) inside float range; a warp with any row
            // beyond e^60 rescales phi+ exactly once sigma is known (phase C).  Padding
            // lanes (rows beyond the unit's G B query rows) do not count.
            const bool fast = __all_sync(0xffffffffu, !valid || !(lw + ms * a.scale + __logf(sp) > 60.f));
            if (fast) {
                tmem_wait_st();
                tc_fence_before();
                __syncwarp();
                if (lane == 0) mbar_arrive(phip);
            }

            // ---- phase B2: phi- over U (unscaled), the score sums, unnormalised phi(K)
            {
                float l = 0.f, sn = 0.f, ln = 0.f;
                if (has_sc) {
                    tmem_ld16(scol + 16 * part, sc);
                    tmem_wait_ld();
#pragma unroll
                    for (int i = 0; i < 16; ++i) l += ex2(fmaf(sc[i], scale_l2, -ml));
                }
                auto expm = [&](float (&uu)[32], int k) {
                    const float4 *zn = reinterpret_cast<const float4 *>(zs + F + 32 * k);
#pragma unroll
                    for (int i4 = 0; i4 < 8; ++i4) {
                        const float4 b4 = zn[i4];
                        const float zn4[4] = {b4.x, b4.y, b4.z, b4.w};
#pragma unroll
                        for (int j = 0; j < 4; ++j) {
                            const int i = 4 * i4 + j;
                            const float en = ex2(fmaf(-uu[i], kLog2e, mnl));
                            uu[i] = en;
                            sn += en;
                            ln = fmaf(en, zn4[j], ln);
                        }
                    }
                };
                // phi- (unscaled) over U in its columns; scaled by cneg in phase D
#pragma unroll 1
                for (int k = part; k < NCH; k += 2) {
                    float x[32];
                    tmem_ld32(pcol + 32 * k, x);
                    tmem_wait_ld();
                    expm(x, k);
                    tmem_st32(pcol + 32 * k, x);
                }
                {
                    // unnormalised phi(K) of this thread's feature for every token
                    float uk[32];
                    tmem_ld32(kcol, uk);
                    // lane t combines token t's extremum over the four feature quarters
                    float m_l;
                    {
                        const float4 x = *reinterpret_cast<const float4 *>(&tk[(part * 32 + lane) * 4]);
                        m_l = fmaxf(fmaxf(x.x, x.y), fmaxf(x.z, x.w)) * kLog2e;
                    }
                    tmem_wait_ld();
                    const float sgn = part == 0 ? kLog2e : -kLog2e;
#pragma unroll
                    for (int t = 0; t < 32; ++t) {
                        const float m = __shfl_sync(0xffffffffu, m_l, t);
                        uk[t] = fval ? ex2(fmaf(uk[t], sgn, -m)) : 0.f;
                    }
                    // parked in Tensor Memory until the token sums are exchanged
                    tmem_st32(tmem + kCmEK + 32 * part + lane_off, uk);
                    const float ssum = warp_reduce32<0>(uk, lane);
                    tk[((2 + part) * 32 + lane) * 4 + q4] = ssum;
                }
                xb[(part * 4 + 0) * 128 + row] = l;
                xb[(part * 4 + 1) * 128 + row] = lp;
                xb[(part * 4 + 2) * 128 + row] = sn;
                xb[(part * 4 + 3) * 128 + row] = ln;
            }
            if (sync_failed(bad)) break;

            // ---- phase C: phi(K), z, sigma, P', den (and, off the fast path, phi+
            // rescaled)
            float cneg, inv_den;
            {
                // the scores share the dS+ columns, which dS^T may overwrite once
                // phi(K) is signalled: P' takes them from registers
                if (has_sc) tmem_ld16(scol + 16 * part, sc);
                {
                    // phi(K) normalised, as the bf16 MN-major operand [token][feature]
                    // (64-feature atoms of B rows), and z[part*F + row] += sum_t phi(k_t)
                    // (this thread is the only writer); lane t holds token t's normaliser
                    float inv_l;
                    {
                        const float4 v = *reinterpret_cast<const float4 *>(&tk[((2 + part) * 32 + lane) * 4]);
                        inv_l = __fdividef(1.f, (v.x + v.y) + (v.z + v.w));
                    }
                    float ek[32];   // unnormalised phi(K) of feature part*F + row, per token
                    tmem_wait_st();
                    tmem_ld32(tmem + kCmEK + 32 * part + lane_off, ek);
                    tmem_wait_ld();
                    const int f = part * F + row;
                    uint8_t *bf = pkb + (f >> 6) * (B * 128) + ((f & 7) << 1);
                    const int gf = (f & 63) >> 3;
                    float dz = 0.f;
#pragma unroll
                    for (int t = 0; t < 32; ++t) {
                        const float v = ek[t] * __shfl_sync(0xffffffffu, inv_l, t);
                        dz += v;
                        if (fval) *reinterpret_cast<bf16 *>(bf + t * 128 + ((gf ^ (t & 7)) << 4)) = __float2bfloat16_rn(v);
                    }
                    if (fval) zs[f] += dz;
                    // dS^T may be formed while P' is computed (it overwrites the
                    // scores and U_k^T this thread has read from Tensor Memory)
                    fence_proxy_async_smem();
                    tc_fence_before();
                    __syncwarp();
                    if (lane == 0) {
                        mbar_arrive(kready);
                        mbar_arrive(zdone);
                    }
                }
                const float l = xb[0 * 128 + row] + xb[4 * 128 + row];
                const float lpf = xb[1 * 128 + row] + xb[5 * 128 + row];
                const float sn = xb[2 * 128 + row] + xb[6 * 128 + row];
                const float ln = xb[3 * 128 + row] + xb[7 * 128 + row];
                // (approximate intrinsics: the result is rounded to bf16)
                const float rsp = __fdividef(1.f, sp), rsn = __fdividef(1.f, sn);
                const float lin_den = lpf * rsp + ln * rsn;
                const float log_s = lw + ms * a.scale + __logf(l);   // log(w sm_den)
                const float log_l = __logf(lin_den);                   // log(lin_den), -inf if empty
                const float sig = fmaxf(fmaxf(log_s, log_l), -60.f);
                const float esig = __expf(-sig);
                float kappa, pofs;
                if (fast) {
                    kappa = esig * rsp;
                    cneg = lin_den > 0.f ? sp * rsn : 0.f;
                    pofs = lw * kLog2e + __log2f(sp);
                } else {
                    const float cpos = lin_den > 0.f ? esig * rsp : 0.f;
                    cneg = lin_den > 0.f ? esig * rsn : 0.f;
                    kappa = 1.f;
                    pofs = (lw - sig) * kLog2e;
                    auto scale_chunk = [&](uint32_t col) {
                        float v[32];
                        tmem_ld32(col, v);
                        tmem_wait_ld();
#pragma unroll
                        for (int i = 0; i < 32; ++i) v[i] *= cpos;
                        tmem_st32(col, v);
                    };
                    scale_chunk(ppcol + 32 * part);
                    if (two) scale_chunk(ppcol + 32 * (part + 2));
                    tmem_wait_st();
                    tc_fence_before();
                    __syncwarp();
                    if (lane == 0) mbar_arrive(phip);
                }
                if (has_sc) {
                    // P' (w e^(s - sigma), or w sp e^s on the fast path): K-major, no swizzle
                    // (8-row x 16-byte core matrices)
                    uint32_t pk[8];
#pragma unroll
                    for (int i = 0; i < 16; i += 2)
                        pk[i / 2] = pack_bf16x2(ex2(fmaf(sc[i], scale_l2, pofs)), ex2(fmaf(sc[i + 1], scale_l2, pofs)));
                    uint8_t *prow = smem + a.off_p + (row >> 3) * (B / 8) * 128 + (row & 7) * 16;
                    *reinterpret_cast<uint4 *>(prow + (2 * part) * 128) = make_uint4(pk[0], pk[1], pk[2], pk[3]);
                    *reinterpret_cast<uint4 *>(prow + (2 * part + 1) * 128) = make_uint4(pk[4], pk[5], pk[6], pk[7]);
                }
                inv_den = __fdividef(kappa, __expf(log_l - sig) + __expf(log_s - sig));
            }
            fence_proxy_async_smem();
            __syncwarp();
            if (lane == 0) mbar_arrive(pready);

            // ---- phase D: phi- scaled by cneg in the phi columns
            {
                tmem_wait_st();
#pragma unroll 1
                for (int k = part; k < NCH; k += 2) {
                    float x[32];
                    tmem_ld32(pcol + 32 * k, x);
                    tmem_wait_ld();
#pragma unroll
                    for (int i = 0; i < 32; ++i) x[i] *= cneg;
                    tmem_st32(pcol + 32 * k, x);
                }
            }
            tmem_wait_st();
            tc_fence_before();
            __syncwarp();
            if (lane == 0 && !bad) mbar_arrive(phim);

            {
                // ---- state update: S^T += dS^T for a feature half as soon as the readout
                // has consumed its tiles (first half now, second after R-): each tile's slot
                // still holds the tile as read, dS^T is added to it there (float32), and the
                // storer writes the tiles back with plain bulk stores
                const int e = row;
#pragma unroll 1
                for (int h = 0; h < 2; ++h) {
                    const bool bad2 = h == 0 ? !wait_bar(dsdone, kp & 1u, fail, wlim) || bad
                                             : !wait_bar(&dready[kp & 1], (kp >> 1) & 1u, fail, wlim);
                    tc_fence_after();
                    const uint32_t src = tmem + (h == 0 ? kCmDSp : kCmDSm) + lane_off;
                    auto upd = [&](int k) {
                        // the readout has consumed the tile: S^T + dS^T replaces it in its
                        // slot, and the storer writes it over the state in global memory
                        uint8_t *rowp = ring + (size_t)((q + h * NCH + k) % NS) * chunk_bytes + e * 128;
                        float v[32];
                        tmem_ld32(src + 32 * k, v);
                        tmem_wait_ld();
                        if (!bad2 && e < d) {
#pragma unroll
                            for (int gq = 0; gq < 8; ++gq) {
                                float4 *p4 = reinterpret_cast<float4 *>(rowp + ((gq ^ (e & 7)) << 4));
                                const float4 s4 = *p4;
                                *p4 = make_float4(s4.x + v[4 * gq], s4.y + v[4 * gq + 1], s4.z + v[4 * gq + 2],
                                                  s4.w + v[4 * gq + 3]);
                            }
                        }
                    };
#pragma unroll 1
                    for (int k = part; k < NCH; k += 2) upd(k);
                    fence_proxy_async_smem();
                    tc_fence_before();
                    __syncwarp();
                    if (lane == 0 && !bad2) {
                        mbar_arrive(&tready[h]);
                        if (h == 0) mbar_arrive(efree);
                    }
                }
                epilogue(kp, q, inv_den);
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

}  // namespace

bool fused_supported(const hybrid_cfg &c)
{
    if (c.io_dtype != HYBRID_BF16) return false;
    if (c.head_dim != 64 && c.head_dim != 128) return false;
    if (c.feat_dim != 64 && c.feat_dim != 128) return false;
    // phi(K) is formed for 32 tokens on the 32 lanes of a warp; the scores ride in
    // one 16-column chunk per part
    if (c.block_size != 32) return false;
    const int G = c.n_q_heads / c.n_kv_heads;
    if (G * c.block_size > 128) return false;
    // a unit's Q arrives as one box of 128 / G tokens x G heads
    if (128 % G != 0) return false;
    const FLayout L = make_flayout(c.head_dim, c.feat_dim, c.block_size);
    const int NCH = c.feat_dim / 32;
    // a ring shorter than a unit stages the output in first-half slots that no
    // later tile of the unit reuses, which needs NCH + 2 slots
    if (L.NS < NCH + 2) return false;
    return (int)L.bytes <= kSmemLimit;
}

cudaError_t launch_fused(const hybrid_cfg &c, const void *Q, const void *K, const void *V, const void *W,
                         const float *alpha, void *const *states, int n_req, void *O, unsigned *err,
                         cudaStream_t st)
{
    const FLayout L = make_flayout(c.head_dim, c.feat_dim, c.block_size);
    FusedArgs a;
    {
        const int d = c.head_dim, F = c.feat_dim, B = c.block_size, Hq = c.n_q_heads, Hkv = c.n_kv_heads;
        const int G = Hq / Hkv;
        const cuuint64_t rows = (cuuint64_t)n_req * B;
        const cuuint64_t P = (cuuint64_t)d / 64;
        // Q: [panel][request][token][head][64]; a box of G heads x 128 / G tokens
        const cuuint64_t dq5[5] = {64, (cuuint64_t)Hq, (cuuint64_t)B, (cuuint64_t)n_req, P};
        const cuuint64_t sq5[4] = {(cuuint64_t)d * 2, (cuuint64_t)Hq * d * 2, (cuuint64_t)B * Hq * d * 2, 128};
        const cuuint32_t bq5[5] = {64, (cuuint32_t)G, (cuuint32_t)(128 / G), 1, (cuuint32_t)P};
        // K, V: [panel][row][head][64], a box of B rows of one head
        const cuuint64_t dv[4] = {64, (cuuint64_t)Hkv, rows, P};
        const cuuint64_t sv[3] = {(cuuint64_t)d * 2, (cuuint64_t)Hkv * d * 2, 128};
        const cuuint32_t bv[4] = {64, 1, (cuuint32_t)B, (cuuint32_t)P};
        // W: [panel][row][64], a box of d rows
        const cuuint64_t dw[3] = {64, (cuuint64_t)Hkv * d, (cuuint64_t)F / 64};
        const cuuint64_t sw[2] = {(cuuint64_t)F * 2, 128};
        const cuuint32_t bw[3] = {64, (cuuint32_t)d, (cuuint32_t)F / 64};
        // O: one box per staged slot
        const cuuint64_t dq[3] = {(cuuint64_t)d, (cuuint64_t)Hq, rows};
        const cuuint64_t sq[2] = {(cuuint64_t)d * 2, (cuuint64_t)Hq * d * 2};
        const cuuint32_t bo[3] = {64, (cuuint32_t)G, (cuuint32_t)(d == 128 ? B : B / 2)};
        if (!encode_bf16(&a.tmQ, Q, 5, dq5, sq5, bq5) || !encode_bf16(&a.tmK, K, 4, dv, sv, bv) ||
            !encode_bf16(&a.tmV, V, 4, dv, sv, bv) ||
            !encode_bf16(&a.tmW, W, 3, dw, sw, bw) || !encode_bf16(&a.tmO, O, 3, dq, sq, bo))
            return cudaErrorInvalidValue;
    }
    a.alpha = alpha;
    a.states = states;
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
    a.off_wk = L.off_wk;
    a.off_vb = L.off_vb;
    a.off_p = L.off_p;
    a.off_pk = L.off_pk;
    a.off_z = L.off_z;
    a.off_st = L.off_st;
    a.off_bar = L.off_bar;
    const int grid = a.n_units < sm_count() ? a.n_units : sm_count();
    // opt in to the full shared memory once per device and kernel (the attribute
    // is set to the maximum, so every layout fits)
    static std::atomic<unsigned long long> opted{0};
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
    const unsigned long long bit = 1ull << dev;
    if (!(opted.load(std::memory_order_acquire) & bit)) {
        const cudaError_t e = cudaFuncSetAttribute(k_fused, cudaFuncAttributeMaxDynamicSharedMemorySize, kSmemLimit);
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
    return cudaLaunchKernelEx(&lc, k_fused, a);
}

}  // namespace hyb
