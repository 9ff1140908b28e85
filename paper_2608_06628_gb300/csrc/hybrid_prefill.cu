// hybrid_prefill.cu -- block commit and prompt prefill (Section 3.1's state
// update S += sum_t phi(k_t) v_t^T, z += sum_t phi(k_t)) with the key feature
// map computed token-major.
//
// U_k = K W is formed on the tensor cores with the chunk's 128 tokens as the M
// dimension (K is loaded by TMA in its natural [token][d] layout, W is the
// MN-major B operand), so each Tensor Memory lane holds one token's F values of
// U_k: a thread takes the softmax of its token over its half of phi entirely in
// registers, with no exchange between threads.  dS^T = V^T phi(K)^T accumulates
// in Tensor Memory over a run of chunks; dz is the token sum of phi(K), reduced
// within each warp.  At the end of a run the increments are added into the
// state in global memory by bulk reduce-adds (the float32 add happens at L2), so
// runs of the same state may be split across CTAs.
//
// Work: the n_units * n_chunks chunks ((request, state head) units of T tokens,
// 128-token chunks, the last one masked) are split into contiguous ranges, one
// per CTA, so long prompts balance across SMs to within one chunk; a range
// covers whole or partial units ("runs").  Warp roles (12 warps):
//   warp 0      producer: W of each run, K and V of each chunk (TMA)
//   warp 1      MMA issuer (one thread); owns the Tensor Memory allocation
//   warp 2      storer: bulk reduce-adds of dz and the dS^T tiles
//   warps 4-11  math: thread = (token 32*q4 + lane, half "part"); phi(K) rows
//               into shared memory, dz; at the end of a run the dS^T tiles
// Tensor Memory: U_k of two chunks at columns [0, F) and [F, 2F) (lanes =
// tokens), dS^T at [256, 256 + 2F) (lanes = e, the index into d; phi+ features
// first), formed by one N = 2F product per 16 tokens.
#include <atomic>

#include "hybrid_common.cuh"
#include "hybrid_tc.h"
#include "tc_pipeline.cuh"

namespace hyb {

namespace {

using namespace pipe;

constexpr int kWarps = 12;
constexpr int kThreads = kWarps * 32;
constexpr int kCT = 128;             // tokens per chunk (the M of U_k = K W)
constexpr int kStage = 4;            // staging slots for dS^T tiles, inside the phi(K) buffer
constexpr int kSmemLimit = 232448;
constexpr int kOneCtaPerSm = 118 * 1024;
constexpr uint32_t kColDS = 256;      // dS^T: phi+ features at [256, 256 + F), phi- at [256 + F, 256 + 2F)
constexpr uint32_t kAtom = kCT * 128;   // one 64-column atom of a 128-row operand
constexpr int kMaxRaggedReq = kMaxRaggedRequests;

struct PrefillArgs {
    CUtensorMap tmK, tmV, tmW;   // K, V [tokens][Hkv][d] (box 64 x 1 x 128), W [Hkv*d][F] (box 64 x d); 128-byte swizzle
    void *const *states;
    unsigned *err;
    int n_units, T, Hkv, d, F, n_chunks;
    uint32_t off_w, off_k, off_v, off_p, off_s, off_dz, off_bar;
};
// Ragged prompts: request r owns tokens [tok[r], tok[r + 1]) of the packed K and V
// and chunks [ch[r], ch[r + 1]) of each of its heads; carried in the parameters.
struct PrefillRaggedArgs : PrefillArgs {
    int n_req;
    int tok[kMaxRaggedReq + 1];
    int ch[kMaxRaggedReq + 1];
};

// Per-request token ranges and chunk counts, uniform or ragged.
__device__ __forceinline__ int req_tok0(const PrefillArgs &a, int r) { return r * a.T; }
__device__ __forceinline__ int req_len(const PrefillArgs &a, int) { return a.T; }
__device__ __forceinline__ int req_nch(const PrefillArgs &a, int) { return a.n_chunks; }
__device__ __forceinline__ long long total_chunks(const PrefillArgs &a) { return (long long)a.n_units * a.n_chunks; }
__device__ __forceinline__ int req_tok0(const PrefillRaggedArgs &a, int r) { return a.tok[r]; }
__device__ __forceinline__ int req_len(const PrefillRaggedArgs &a, int r) { return a.tok[r + 1] - a.tok[r]; }
__device__ __forceinline__ int req_nch(const PrefillRaggedArgs &a, int r) { return a.ch[r + 1] - a.ch[r]; }
__device__ __forceinline__ long long total_chunks(const PrefillRaggedArgs &a) { return (long long)a.Hkv * a.ch[a.n_req]; }
// request of global chunk c: request r holds chunks [Hkv ch[r], Hkv ch[r + 1])
__device__ __forceinline__ int chunk_req(const PrefillArgs &a, long long c)
{
    return (int)(c / ((long long)a.Hkv * a.n_chunks));
}
__device__ __forceinline__ long long req_chunk0(const PrefillArgs &a, int r) { return (long long)r * a.Hkv * a.n_chunks; }
__device__ __forceinline__ int chunk_req(const PrefillRaggedArgs &a, long long c)
{
    int lo = 0, hi = a.n_req;   // the last r with Hkv ch[r] <= c (empty requests precede it)
    while (hi - lo > 1) {
        const int mid = (lo + hi) >> 1;
        if ((long long)a.Hkv * a.ch[mid] <= c) lo = mid;
        else hi = mid;
    }
    return lo;
}
__device__ __forceinline__ long long req_chunk0(const PrefillRaggedArgs &a, int r) { return (long long)a.Hkv * a.ch[r]; }

// Shared memory: [W: F/64 atoms of d rows][K: 2 atoms of 128 rows][V x 2: 2 atoms each]
// [phi(K): 2F/64 atoms of 128 rows][dz: 4 x 2F][barriers].  K and V always have
// two atoms so that the M = 128 operand V^T stays inside the allocation for
// d = 64 (its upper rows are never read back).  V is double-buffered so the next
// chunk's V streams in while this chunk's dS^T runs.  At the end of a run the
// phi(K) buffer, free once the run's last dS^T is done, stages the dS^T tiles
// (kStage slots of d rows x 128 B).
struct PLayout {
    uint32_t off_w, off_k, off_v, off_p, off_s, off_dz, off_bar, bytes;
};

PLayout make_playout(int d, int F)
{
    PLayout L{};
    uint32_t off = 0;
    L.off_w = off; off += (uint32_t)(F / 64) * (uint32_t)d * 128;
    L.off_k = off; off += 2 * kAtom;
    L.off_v = off; off += 2 * 2 * kAtom;
    L.off_p = off; off += (uint32_t)(2 * F / 64) * kAtom;
    L.off_s = L.off_p;
    L.off_dz = off; off += (((uint32_t)4 * 2 * F * 4) + 1023) & ~1023u;
    L.off_bar = off; off += 1024;
    L.bytes = off + 1024;
    if ((int)L.bytes < kOneCtaPerSm) L.bytes = kOneCtaPerSm;
    return L;
}

__device__ __forceinline__ float *unit_head(const PrefillArgs &a, int u)
{
    float *st = reinterpret_cast<float *>(a.states[u / a.Hkv]);
    if (!state_ptr_ok(st)) return nullptr;
    return st + (size_t)(u % a.Hkv) * head_floats(a.d, a.F);
}

// The state of the chunk's unit, loaded once per unit (a chunk range visits its
// units in order, so each role keeps the last unit's pointer).
struct UnitCache {
    int u = -1;
    float *head = nullptr;
    __device__ __forceinline__ float *get(const PrefillArgs &a, int unit)
    {
        if (unit != u) {
            u = unit;
            head = unit_head(a, unit);
        }
        return head;
    }
};

// Position of a chunk within its unit and run.  A role walks its CTA's chunk
// range in order: the request is located once at the start, then the head and
// the chunk index advance incrementally (skipping requests without tokens).
struct ChunkPos {
    int u, j;
    int row0, nt;       // first token row in K and V, valid tokens
    bool first, last;   // first / last chunk of its run in this CTA's range
};
template <class A>
struct ChunkWalk {
    long long c, lo, hi;
    int r, g, j, nch;
    __device__ __forceinline__ ChunkWalk(const A &a, long long lo_, long long hi_) : c(lo_), lo(lo_), hi(hi_)
    {
        r = lo_ < hi_ ? chunk_req(a, lo_) : 0;
        nch = lo_ < hi_ ? req_nch(a, r) : 1;
        const long long rem = lo_ - req_chunk0(a, r);
        g = (int)(rem / nch);
        j = (int)(rem % nch);
    }
    __device__ __forceinline__ bool more() const { return c < hi; }
    __device__ __forceinline__ ChunkPos pos(const A &a) const
    {
        ChunkPos p;
        p.u = r * a.Hkv + g;
        p.j = j;
        p.row0 = req_tok0(a, r) + j * kCT;
        p.nt = min(kCT, req_len(a, r) - j * kCT);
        p.first = c == lo || j == 0;
        p.last = c == hi - 1 || j == nch - 1;
        return p;
    }
    __device__ __forceinline__ void next(const A &a)
    {
        if (++c >= hi) return;
        if (++j < nch) return;
        j = 0;
        if (++g < a.Hkv) return;
        g = 0;
        do {
            ++r;
        } while (req_nch(a, r) == 0);
        nch = req_nch(a, r);
    }
};

template <class A>
__global__ void __launch_bounds__(kThreads, 1) k_prefill(const __grid_constant__ A a)
{
    using namespace ptx;
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int d = a.d, F = a.F;
    const int NCH = F / 32, NC = 2 * NCH;
    const uint32_t tile = (uint32_t)d * 128;
    // staging slots that fit in the phi(K) buffer (2 for d = 128, F = 64)
    const int NSS = min(kStage, (int)(((uint32_t)(2 * F / 64) * kAtom) / tile));
    const long long total = total_chunks(a);
    const long long lo = total * (long long)blockIdx.x / (long long)gridDim.x;
    const long long hi = total * (long long)(blockIdx.x + 1) / (long long)gridDim.x;

    uint64_t *bars = reinterpret_cast<uint64_t *>(smem + a.off_bar);
    uint64_t *wfull = bars;            // W of the run is in place
    uint64_t *wfree = wfull + 1;       // the run's U_k products have read W
    uint64_t *kfull = wfree + 1;       // K of the chunk is in place
    uint64_t *kfree = kfull + 1;       // U_k of the chunk has read K
    uint64_t *vfull = kfree + 1;       // [2] V of a chunk buffer is in place
    uint64_t *vfree = vfull + 2;       // [2] dS^T of the chunk has read that buffer
    uint64_t *ukready = vfree + 2;     // [2] U_k of a Tensor Memory buffer is complete
    uint64_t *ukfree = ukready + 2;    // [2] the math warps have read that buffer
    uint64_t *pready = ukfree + 2;     // the chunk's phi(K) is written
    uint64_t *dsdone = pready + 1;     // the chunk's dS^T products are complete (phi(K) may be rewritten)
    uint64_t *segdone = dsdone + 1;    // the run's dS^T is complete
    uint64_t *dsfree = segdone + 1;    // the math warps have read the run's dS^T
    uint64_t *sfull = dsfree + 1;      // [kStage] a staging slot holds a dS^T tile
    uint64_t *sempty = sfull + kStage;
    uint64_t *dzready = sempty + kStage;
    uint64_t *dzfree = dzready + 1;
    uint64_t *sdrain = dzfree + 1;     // the run's staged tiles have been read (phi(K) may be rewritten)
    uint64_t *mmadone = sdrain + 1;
    const int n_bars = 20 + 2 * kStage;   // wfull .. mmadone
    uint32_t *tmem_holder = reinterpret_cast<uint32_t *>(bars + n_bars);
    volatile int *fail = reinterpret_cast<volatile int *>(tmem_holder + 1);

    if (warp == 0 && lane == 0) {
        prefetch_tensormap(&a.tmK);
        prefetch_tensormap(&a.tmV);
        prefetch_tensormap(&a.tmW);
    }
    if (tid == 0) {
        for (int i = 0; i < n_bars; ++i) mbar_init(&bars[i], 1);
        mbar_init(pready, 8);
        mbar_init(&ukfree[0], 8);
        mbar_init(&ukfree[1], 8);
        mbar_init(dsfree, 8);
        mbar_init(dzready, 8);
        for (int s = 0; s < kStage; ++s) mbar_init(&sfull[s], 4);   // the four warps of one part
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
    griddep_wait();
    const uint32_t tmem = *tmem_holder;
    uint8_t *stage = smem + a.off_s;
    float *dzq = reinterpret_cast<float *>(smem + a.off_dz);   // [quarter][2F]

    if (warp == 0) {
        // ------------------------------------------------------------- producer
        if (lane == 0) {
            uint32_t s = 0, i = 0;
            int nw = 0, nk = 0, nv = 0;
            bool ok = true;
            UnitCache uc;
            for (ChunkWalk<A> w(a, lo, hi); w.more() && ok; w.next(a)) {
                const ChunkPos p = w.pos(a);
                if (!uc.get(a, p.u)) continue;
                const int g = p.u % a.Hkv;
                const int row0 = p.row0;
                if (p.first) {
                    if (s > 0 && !wait_bar(wfree, (s - 1) & 1u, fail)) break;
                    mbar_arrive_expect_tx(wfull, (uint32_t)(F / 64) * tile);
                    tma_load_3d(smem + a.off_w, &a.tmW, 0, g * d, 0, wfull);
                    ++nw;
                    ++s;
                }
                if (i > 0 && !wait_bar(kfree, (i - 1) & 1u, fail)) break;
                mbar_arrive_expect_tx(kfull, (uint32_t)(d / 64) * kAtom);
                tma_load_4d(smem + a.off_k, &a.tmK, 0, g, row0, 0, kfull);
                ++nk;
                const int vb = i & 1;
                if (i >= 2 && !wait_bar(&vfree[vb], ((i - 2) >> 1) & 1u, fail)) break;
                mbar_arrive_expect_tx(&vfull[vb], (uint32_t)(d / 64) * kAtom);
                tma_load_4d(smem + a.off_v + vb * 2 * kAtom, &a.tmV, 0, g, row0, 0, &vfull[vb]);
                ++nv;
                ++i;
            }
            if (*fail) {
                // copies in flight land before the CTA exits
                if (nw) mbar_wait(wfull, (uint32_t)(nw - 1) & 1u, kWaitNs);
                if (nk) mbar_wait(kfull, (uint32_t)(nk - 1) & 1u, kWaitNs);
                for (int b = 0; b < 2 && b < nv; ++b)
                    mbar_wait(&vfull[b], (uint32_t)((nv - 1 - b) >> 1) & 1u, kWaitNs);
            }
        }
    } else if (warp == 1) {
        // ------------------------------------------------------- MMA issuer
        if (lane == 0) {
            const uint32_t w_u = smem_u32(smem + a.off_w), k_u = smem_u32(smem + a.off_k),
                           v_u = smem_u32(smem + a.off_v), p_u = smem_u32(smem + a.off_p);
            const uint32_t idU = instr_desc(FMT_BF16, FMT_BF16, false, true, 128, F);
            const uint32_t idDS = instr_desc(FMT_BF16, FMT_BF16, true, true, 128, 2 * F);
            // U_k = K W of local chunk i into Tensor Memory buffer i & 1 (lanes = tokens)
            auto uk = [&](uint32_t i) {
                for (int k = 0; k < d / 16; ++k) {
                    const uint64_t ak = smem_desc(k_u + (k >> 2) * kAtom + (k & 3) * 32, 16, 1024, SWZ_128B);
                    const uint64_t bw = smem_desc(w_u + 2 * k * 1024, d * 128, 1024, SWZ_128B);
                    mma_bf16_ss(tmem + (i & 1) * F, ak, bw, idU, k > 0);
                }
            };
            // dS^T (+)= V^T phi(K)^T of a chunk with nt tokens: both halves of phi in one
            // N = 2F product per 16 tokens (the phi(K) atoms are contiguous)
            auto dst = [&](uint32_t ci, int nt, bool first) {
                const int nks = (nt + 15) / 16;
                const uint32_t vb_u = v_u + (ci & 1) * 2 * kAtom;
                for (int ks = 0; ks < nks; ++ks) {
                    const uint64_t av = smem_desc(vb_u + ks * 2048, kAtom, 1024, SWZ_128B);
                    const uint64_t bp = smem_desc(p_u + ks * 2048, kAtom, 1024, SWZ_128B);
                    mma_bf16_ss(tmem + kColDS, av, bp, idDS, !(first && ks == 0));
                }
            };
            uint32_t s = 0, i = 0, sd = 0;   // runs whose W has been waited, chunks, runs whose dS^T began
            bool ok = true;
            // dS^T of a chunk is issued after the next chunk's U_k, so the math warps
            // can start on that chunk while this one's phi(K) is finished
            bool pend = false;
            uint32_t pi = 0;
            ChunkPos pp{};
            UnitCache uc;
            auto issue_ds = [&]() -> bool {
                if (!wait_bar(pready, pi & 1u, fail) || !wait_bar(&vfull[pi & 1], (pi >> 1) & 1u, fail)) return false;
                // the previous run's dS^T has been read before this run overwrites it
                if (pp.first && sd > 0 && !wait_bar(dsfree, (sd - 1) & 1u, fail)) return false;
                if (pp.first) ++sd;
                tc_fence_after();
                dst(pi, pp.nt, pp.first);
                mma_commit(dsdone);
                mma_commit(&vfree[pi & 1]);
                if (pp.last) mma_commit(segdone);
                return true;
            };
            for (ChunkWalk<A> w(a, lo, hi); w.more() && ok; w.next(a)) {
                const ChunkPos p = w.pos(a);
                if (!uc.get(a, p.u)) continue;
                if (p.first) {
                    if (!wait_bar(wfull, s & 1u, fail)) { ok = false; break; }
                    ++s;
                }
                if (!wait_bar(kfull, i & 1u, fail)) { ok = false; break; }
                if (i >= 2 && !wait_bar(&ukfree[i & 1], ((i - 2) >> 1) & 1u, fail)) { ok = false; break; }
                tc_fence_after();
                uk(i);
                mma_commit(&ukready[i & 1]);
                mma_commit(kfree);
                if (p.last) mma_commit(wfree);
                if (pend && !issue_ds()) { ok = false; break; }
                pend = true;
                pi = i;
                pp = p;
                ++i;
            }
            if (ok && pend) issue_ds();
            mma_commit(mmadone);
            mbar_wait(mmadone, 0, kWaitNs);
        }
    } else if (warp == 2) {
        // --------------------------------------------------------------- storer
        if (lane == 0) {
            uint32_t s = 0, sg = 0;
            bool ok = true;
            UnitCache uc;
            for (ChunkWalk<A> w(a, lo, hi); w.more() && ok; w.next(a)) {
                const ChunkPos p = w.pos(a);
                float *Sg = uc.get(a, p.u);
                if (!Sg || !p.last) continue;
                // dz: the four quarters' token sums, each added into z
                if (!wait_bar(dzready, s & 1u, fail)) break;
                for (int q = 0; q < 4; ++q) {
                    bulk_reduce_add_f32(Sg + (size_t)2 * F * d, dzq + q * 2 * F, 2 * F * 4);
                    bulk_commit();
                }
                bulk_wait_read_all();
                mbar_arrive(dzfree);
                for (int t = 0; t < NC; ++t, ++sg) {
                    const int slot = sg % NSS;
                    if (!wait_bar(&sfull[slot], (sg / NSS) & 1u, fail)) { ok = false; break; }
                    bulk_reduce_add_f32(Sg + (size_t)t * 32 * d, stage + (size_t)slot * tile, tile);
                    bulk_commit();
                    bulk_wait_read_all();
                    mbar_arrive(&sempty[slot]);
                }
                if (!ok) break;
                mbar_arrive(sdrain);
                ++s;
            }
            bulk_wait_all();
        }
    } else if (warp >= 4) {
        // ------------------------------------------------------------- math
        const int mt = tid - 128;
        const int q4 = warp & 3, part = (warp - 4) >> 2;
        const int tok = 32 * q4 + lane;                       // token of this thread in the chunk; e at the end
        const uint32_t lane_off = (uint32_t)(32 * q4) << 16;
        const float sgn = part == 0 ? kLog2e : -kLog2e;
        uint8_t *pkb = smem + a.off_p;
        uint32_t s = 0, i = 0, sg = 0;
        float dzacc[4] = {0.f, 0.f, 0.f, 0.f};   // token sums of features part*F + 32*jj + lane
        bool ok = true;
        UnitCache uc;
        for (ChunkWalk<A> w(a, lo, hi); w.more() && ok; w.next(a)) {
            const ChunkPos p = w.pos(a);
            if (!uc.get(a, p.u)) {
                if (mt == 0) raise_error(a.err, ERR_BAD_STATE_PTR);
                continue;
            }
            const int nt = p.nt;
            const bool active = 32 * q4 < nt;      // warp-uniform: the warp holds a valid token
            const bool valid = tok < nt;
            const uint32_t ub = tmem + (i & 1) * F + lane_off;
            bool bad = !wait_bar(&ukready[i & 1], (i >> 1) & 1u, fail);
            tc_fence_after();
            // softmax of this token over its half: the extremum (max of u for phi+,
            // min for phi-), then the sum of exponentials.  U stays unchanged in Tensor
            // Memory: the token's other half is computed from the same columns by a
            // thread of another warp
            float m = 0.f, l = 0.f;
            if (active) {
                float ext = part == 0 ? -INFINITY : INFINITY;
#pragma unroll 1
                for (int jj = 0; jj < NCH; ++jj) {
                    float x[32];
                    tmem_ld32(ub + 32 * jj, x);
                    tmem_wait_ld();
                    if (part == 0) {
#pragma unroll
                        for (int t = 0; t < 32; ++t) ext = fmaxf(ext, x[t]);
                    } else {
#pragma unroll
                        for (int t = 0; t < 32; ++t) ext = fminf(ext, x[t]);
                    }
                }
                m = ext * sgn;   // max of sgn * u (log2 units)
#pragma unroll 1
                for (int jj = 0; jj < NCH; ++jj) {
                    float x[32];
                    tmem_ld32(ub + 32 * jj, x);
                    tmem_wait_ld();
#pragma unroll
                    for (int t = 0; t < 32; ++t) l += ex2(fmaf(x[t], sgn, -m));
                }
            }
            // phi = 2^(sgn u - m) / l = 2^(sgn u - (m + log2 l)): the normaliser folds
            // into the exponent's offset
            const float mo = m + __log2f(l);
            const bool full = 32 * q4 + 32 <= nt;   // warp-uniform: every token of the warp is valid
            // phi(K) is rewritten once the previous chunk's dS^T has read it and, after
            // a run's end, once the storer has read the tiles staged there
            if (i > 0) bad = !wait_bar(dsdone, (i - 1) & 1u, fail) || bad;
            if (p.first && s > 0) bad = !wait_bar(sdrain, (s - 1) & 1u, fail) || bad;
            if (active) {
#pragma unroll 1
                for (int jj = 0; jj < NCH; ++jj) {
                    float x[32];
                    tmem_ld32(ub + 32 * jj, x);
                    tmem_wait_ld();
                    if (full) {
#pragma unroll
                        for (int t = 0; t < 32; ++t) x[t] = ex2(fmaf(x[t], sgn, -mo));
                    } else {
#pragma unroll
                        for (int t = 0; t < 32; ++t) x[t] = valid ? ex2(fmaf(x[t], sgn, -mo)) : 0.f;
                    }
                    // row tok of the MN-major operand [token][feature], 64-feature atoms,
                    // 16-byte granules permuted by (tok mod 8)
                    const int f0 = part * F + 32 * jj;
                    uint8_t *rowp = pkb + (f0 >> 6) * kAtom + tok * 128;
                    const int g0 = (f0 & 63) >> 3;
#pragma unroll
                    for (int gq = 0; gq < 4; ++gq) {
                        const uint4 w = make_uint4(pack_bf16x2(x[8 * gq], x[8 * gq + 1]), pack_bf16x2(x[8 * gq + 2], x[8 * gq + 3]),
                                                   pack_bf16x2(x[8 * gq + 4], x[8 * gq + 5]), pack_bf16x2(x[8 * gq + 6], x[8 * gq + 7]));
                        *reinterpret_cast<uint4 *>(rowp + (((g0 + gq) ^ (tok & 7)) << 4)) = w;
                    }
                    // token sum over this warp's 32 tokens: lane L gets feature f0 + L
                    const float sum = warp_reduce32<0>(x, lane);
                    if (jj == 0) dzacc[0] += sum;
                    else if (jj == 1) dzacc[1] += sum;
                    else if (jj == 2) dzacc[2] += sum;
                    else dzacc[3] += sum;
                }
            } else {
                // a warp beyond the chunk's tokens writes zero rows (the dS^T products
                // read whole 16-token groups)
#pragma unroll 1
                for (int jj = 0; jj < NCH; ++jj) {
                    const int f0 = part * F + 32 * jj;
                    uint8_t *rowp = pkb + (f0 >> 6) * kAtom + tok * 128;
                    const int g0 = (f0 & 63) >> 3;
#pragma unroll
                    for (int gq = 0; gq < 4; ++gq)
                        *reinterpret_cast<uint4 *>(rowp + (((g0 + gq) ^ (tok & 7)) << 4)) = make_uint4(0, 0, 0, 0);
                }
            }
            fence_proxy_async_smem();
            tc_fence_before();
            __syncwarp();
            if (lane == 0) {
                mbar_arrive(&ukfree[i & 1]);
                mbar_arrive(pready);
            }
            ++i;
            if (p.last) {
                // dz of this run: each quarter's token sums, added into z by the storer
                bad = (s > 0 && !wait_bar(dzfree, (s - 1) & 1u, fail)) || bad;
#pragma unroll
                for (int jj = 0; jj < 4; ++jj)
                    if (jj < NCH) dzq[q4 * 2 * F + part * F + 32 * jj + lane] = dzacc[jj];
                dzacc[0] = dzacc[1] = dzacc[2] = dzacc[3] = 0.f;
                fence_proxy_async_smem();
                __syncwarp();
                if (lane == 0) mbar_arrive(dzready);
                // the run's dS^T tiles into the staging ring, in the storer's order
                bad = !wait_bar(segdone, s & 1u, fail) || bad;
                tc_fence_after();
                const int e = tok;
#pragma unroll 1
                for (int t = 0; t < NCH; ++t) {
                    // tiles of this part: chunks part, part + 2 of each half
                    const int h = t / (NCH / 2 > 0 ? NCH / 2 : 1);
                    const int k = part + 2 * (t % (NCH / 2 > 0 ? NCH / 2 : 1));
                    if (k >= NCH) continue;
                    const int cidx = h * NCH + k;
                    const uint32_t sgc = sg + cidx;
                    const int slot = sgc % NSS;
                    const bool okc = wait_bar(&sempty[slot], ((sgc / NSS) & 1u) ^ 1u, fail) && !bad;
                    float v[32];
                    tmem_ld32(tmem + kColDS + (uint32_t)(h * F) + lane_off + 32 * k, v);
                    tmem_wait_ld();
                    if (okc && e < d) {
                        uint8_t *rowp = stage + (size_t)slot * tile + e * 128;
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
                if (lane == 0) mbar_arrive(dsfree);
                sg += NC;
                ++s;
            }
            if (__any_sync(0xffffffffu, bad) && *fail) ok = false;
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

bool prefill_supported(const hybrid_cfg &c)
{
    if (c.io_dtype != HYBRID_BF16) return false;
    if (c.head_dim != 64 && c.head_dim != 128) return false;
    if (c.feat_dim != 64 && c.feat_dim != 128) return false;
    return (int)make_playout(c.head_dim, c.feat_dim).bytes <= kSmemLimit;
}

namespace {

// Tensor maps and sizes shared by the uniform and the ragged launch; rows = tokens of K and V.
bool fill_prefill_args(const hybrid_cfg &c, const void *K, const void *V, long long rows, const void *W,
                       void *const *states, int n_req, unsigned *err, PrefillArgs &a)
{
    const PLayout L = make_playout(c.head_dim, c.feat_dim);
    const int d = c.head_dim, F = c.feat_dim, Hkv = c.n_kv_heads;
    // K, V: [panel][row][head][64], a box of kCT rows of one head; W: [panel][row][64]
    // (the 64-element panels as the outermost box dimension: one copy for all of them)
    const cuuint64_t dk[4] = {64, (cuuint64_t)Hkv, (cuuint64_t)rows, (cuuint64_t)d / 64};
    const cuuint64_t sk[3] = {(cuuint64_t)d * 2, (cuuint64_t)Hkv * d * 2, 128};
    const cuuint32_t bk[4] = {64, 1, (cuuint32_t)kCT, (cuuint32_t)d / 64};
    const cuuint64_t dw[3] = {64, (cuuint64_t)Hkv * d, (cuuint64_t)F / 64};
    const cuuint64_t sw[2] = {(cuuint64_t)F * 2, 128};
    const cuuint32_t bw[3] = {64, (cuuint32_t)d, (cuuint32_t)F / 64};
    if (!encode_bf16(&a.tmK, K, 4, dk, sk, bk) || !encode_bf16(&a.tmV, V, 4, dk, sk, bk) ||
        !encode_bf16(&a.tmW, W, 3, dw, sw, bw))
        return false;
    a.states = states;
    a.err = err;
    a.n_units = n_req * Hkv;
    a.Hkv = Hkv;
    a.d = d;
    a.F = F;
    a.off_w = L.off_w;
    a.off_k = L.off_k;
    a.off_v = L.off_v;
    a.off_p = L.off_p;
    a.off_s = L.off_s;
    a.off_dz = L.off_dz;
    a.off_bar = L.off_bar;
    return true;
}

template <class A>
cudaError_t run_prefill(const hybrid_cfg &c, const A &a, long long total, cudaStream_t st)
{
    if (total <= 0) return cudaSuccess;
    const PLayout L = make_playout(c.head_dim, c.feat_dim);
    const int grid = total < sm_count() ? (int)total : sm_count();
    static std::atomic<unsigned long long> opted;
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
    const unsigned long long bit = 1ull << dev;
    if (!(opted.load(std::memory_order_acquire) & bit)) {
        const cudaError_t e =
            cudaFuncSetAttribute(k_prefill<A>, cudaFuncAttributeMaxDynamicSharedMemorySize, kSmemLimit);
        if (e != cudaSuccess) return e;
        opted.fetch_or(bit, std::memory_order_acq_rel);
    }
    cudaLaunchConfig_t lc = {};
    lc.gridDim = dim3(grid);
    lc.blockDim = dim3(kThreads);
    lc.dynamicSmemBytes = L.bytes;
    lc.stream = st;
    cudaLaunchAttribute at[1];
    at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    at[0].val.programmaticStreamSerializationAllowed = 1;
    lc.attrs = at;
    lc.numAttrs = 1;
    return cudaLaunchKernelEx(&lc, k_prefill<A>, a);
}

}  // namespace

cudaError_t launch_prefill(const hybrid_cfg &c, const void *K, const void *V, int n_tok, const void *W,
                           void *const *states, int n_req, unsigned *err, cudaStream_t st)
{
    PrefillArgs a;
    if (!fill_prefill_args(c, K, V, (long long)n_req * n_tok, W, states, n_req, err, a)) return cudaErrorInvalidValue;
    a.T = n_tok;
    a.n_chunks = (n_tok + kCT - 1) / kCT;
    return run_prefill(c, a, (long long)a.n_units * a.n_chunks, st);
}

cudaError_t launch_prefill_ragged(const hybrid_cfg &c, const void *K, const void *V, const int *tok, const void *W,
                                  void *const *states, int n_req, unsigned *err, cudaStream_t st)
{
    if (n_req < 1 || n_req > kMaxRaggedReq) return cudaErrorInvalidValue;
    static thread_local PrefillRaggedArgs a;   // 16 KB of offsets: kept off the stack
    if (!fill_prefill_args(c, K, V, tok[n_req] > 0 ? tok[n_req] : 1, W, states, n_req, err, a))
        return cudaErrorInvalidValue;
    a.T = 0;
    a.n_chunks = 0;
    a.n_req = n_req;
    a.ch[0] = 0;
    for (int r = 0; r <= n_req; ++r) a.tok[r] = tok[r];
    for (int r = 0; r < n_req; ++r) a.ch[r + 1] = a.ch[r] + (tok[r + 1] - tok[r] + kCT - 1) / kCT;
    return run_prefill(c, a, (long long)c.n_kv_heads * a.ch[n_req], st);
}

}  // namespace hyb
