// hybrid_tc.cu -- block-hybrid attention on the 5th-generation tensor cores.
//
// A unit is one (request r, state head g).  Its M = G*B query rows (the G query
// heads of the group times the B tokens of the active block, padded to 128)
// share the state (S_g, z_g) of Section 3.1 of "Retrofitting Linear Attention
// into Diffusion Language Models", so the state is streamed from HBM once per
// group.  One CTA per SM takes a contiguous range of units one after another; a
// unit's loads go out as soon as the previous unit's MMAs are complete and land
// during its epilogue.  Contractions (tcgen05.mma, accumulators in Tensor Memory):
//   U      = Q W_g              bf16 x bf16 -> f32   (feature-map projection)
//   scores = Q K^T              bf16 x bf16 -> f32   (in-block softmax logits)
//   D_lin  = phi(Q) S_g         tf32 x tf32 -> f32   (linear readout; phi(Q) in TMEM)
//   D_s    = P V                bf16 x bf16 -> f32   (softmax numerator)
// Per-row work (one thread per TMEM lane/row, two threads per row splitting
// the columns): phi = [softmax(U), softmax(-U)], lin_den = phi . z_g, the
// in-block softmax statistics, and the gated shared-normaliser merge.
// With F = 256, phi = [phi+, phi-] (512 columns) does not fit beside D_lin and D_s
// in Tensor Memory: phi+ is written over U and read out first, then phi- takes its
// place for the second half of the readout.  Both are held scaled by the row's sum sp
// of e^(u - max u) (phi+ unnormalised, no pass over it), and the epilogue divides the
// readout by sp.  phi- comes from phi+ by the identity
// e^(mn - u) = e^(mn - mx) / e^(u - mx) when every row's range of U is moderate (then
// W and Q are dead after U = Q W and their space holds six more state tiles, loaded
// while the feature map is computed); otherwise U = Q W is formed again.
//
// The state arrives by 1-D bulk copies: its HBM layout (hybrid.h) is already
// the 128-byte-swizzled K-major operand image, so each 32-feature tile is one
// copy straight into an MMA-ready buffer.  Q, K, V and W arrive by TMA as
// 128-byte-swizzled boxes, each 64-element panel of a row one 128-byte line:
// Q as the G x B rows of the group's heads over the block's tokens (row t G + hh),
// K and V as B token rows, W as its d rows.
#include "hybrid_common.cuh"
#include "hybrid_tc.h"
#include "tc_pipeline.cuh"
#include "tc_ptx.cuh"

namespace hyb {

namespace {

constexpr int kThreads = 256;
constexpr uint32_t kColA = 0;     // U, then phi = [phi+, phi-] (F <= 128); F = 256: phi+, then phi-;
                                  // then D_s = P V (d columns)
constexpr uint32_t kColD = 256;   // D_lin of issuer A's tiles (d columns)
constexpr uint32_t kColS = 384;   // scores (B columns), then D_lin of issuer B's tiles
constexpr uint64_t kWaitNs = 1000000000ull;   // 1 s per bounded wait
constexpr float kLog2e = 1.4426950408889634f;
constexpr int kSmemLimit = 232448;            // 227 KB opt-in per CTA
constexpr int kOneCtaPerSm = 118 * 1024;      // request at least this much: 1 CTA / SM (TMEM 512 cols)
constexpr int kExtraSlots = 6;                // F = 256: W (4 tiles) and Q (2 tiles) as ring slots
constexpr float kRecipRange = 64.f;           // largest row range of U for phi- from phi+

struct TcAttnArgs {
    CUtensorMap tmQ, tmK, tmV, tmW;   // Q [n B][Hq][d] box {64, G, B}; K, V box {64, 1, B, d / 64};
                                      // W box {64, d, F / 64} (panels outermost)
    const float *alpha;
    void *const *states;
    __nv_bfloat16 *O;
    unsigned *err;
    int B, Hq, Hkv, G, d, F;
    int n_units;        // n_req Hkv (request, state head) units, u = r Hkv + g
    int n_slots;
    float scale_log2;   // log2(e) / sqrt(d)
    float inv_sqrt_d;
    uint32_t off_q, off_w, off_k, off_v, off_p, off_z, off_st, off_bar;
};

struct Layout {
    uint32_t off_q, off_w, off_k, off_v, off_p, off_z, off_st, off_bar, bytes;
    int n_slots;
};

Layout make_layout(int d, int F, int B)
{
    Layout L{};
    const uint32_t chunk = (uint32_t)d * 128;
    const int NC = 2 * F / 32;
    const uint32_t q = (uint32_t)d * 256, w = (uint32_t)d * F * 2, k = (uint32_t)B * d * 2,
                   v = (uint32_t)B * d * 2, p = 128u * B * 2, z = ((uint32_t)2 * F * 4 + 1023) & ~1023u;
    // F = 256 keeps Q for a second U = Q W, so the row statistics get their own space
    const uint32_t stb = F > 128 ? 10u * 1024 : 0u;
    const uint32_t fixed = q + w + k + v + p + z + stb + 1024 /*barriers*/ + 1024 /*alignment slack*/;
    int slots = (int)((kSmemLimit - (int)fixed) / (int)chunk);
    if (slots > NC) slots = NC;
    L.n_slots = slots;
    uint32_t off = (uint32_t)slots * chunk;
    L.off_q = off; off += q;
    L.off_w = off; off += w;
    L.off_k = off; off += k;
    L.off_v = off; off += v;
    L.off_p = off; off += p;
    L.off_z = off; off += z;
    L.off_st = F > 128 ? off : L.off_q;
    off += stb;
    L.off_bar = off; off += 1024;
    L.bytes = off + 1024;
    if ((int)L.bytes < kOneCtaPerSm) L.bytes = kOneCtaPerSm;
    return L;
}

__device__ __forceinline__ float tf32_round(float x)
{
    uint32_t r;
    asm("cvt.rna.tf32.f32 %0, %1;" : "=r"(r) : "f"(x));
    return __uint_as_float(r);
}

__device__ __forceinline__ uint32_t pack_bf16x2(float a, float b)
{
    const __nv_bfloat162 v = __floats2bfloat162_rn(a, b);
    return *reinterpret_cast<const uint32_t *>(&v);
}

// Tensor Memory accesses of 16 lanes by a whole warp (shape 16x32bx2): threads 0-15
// read lanes base + t at columns c .. c + n - 1, threads 16-31 the same lanes at
// columns c + n .. c + 2n - 1 (the split offset equals the width n here).
__device__ __forceinline__ void tmem_ld16x2_32(uint32_t taddr, float (&v)[32])
{
    uint32_t r[32];
    asm volatile("tcgen05.ld.sync.aligned.16x32bx2.x32.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32], 32;"
                 : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]), "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
                 : "r"(taddr));
#pragma unroll
    for (int i = 0; i < 32; ++i) v[i] = __uint_as_float(r[i]);
}
__device__ __forceinline__ void tmem_ld16x2_16(uint32_t taddr, float (&v)[16])
{
    uint32_t r[16];
    asm volatile("tcgen05.ld.sync.aligned.16x32bx2.x16.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15}, [%16], 16;"
                 : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
                 : "r"(taddr));
#pragma unroll
    for (int i = 0; i < 16; ++i) v[i] = __uint_as_float(r[i]);
}
__device__ __forceinline__ void tmem_st16x2_32(uint32_t taddr, const float (&v)[32])
{
    asm volatile("tcgen05.st.sync.aligned.16x32bx2.x32.b32 [%0], 32, {%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31,%32};" ::"r"(taddr),
                 "r"(__float_as_uint(v[0])), "r"(__float_as_uint(v[1])), "r"(__float_as_uint(v[2])), "r"(__float_as_uint(v[3])), "r"(__float_as_uint(v[4])), "r"(__float_as_uint(v[5])), "r"(__float_as_uint(v[6])), "r"(__float_as_uint(v[7])), "r"(__float_as_uint(v[8])), "r"(__float_as_uint(v[9])), "r"(__float_as_uint(v[10])), "r"(__float_as_uint(v[11])), "r"(__float_as_uint(v[12])), "r"(__float_as_uint(v[13])), "r"(__float_as_uint(v[14])), "r"(__float_as_uint(v[15])), "r"(__float_as_uint(v[16])), "r"(__float_as_uint(v[17])), "r"(__float_as_uint(v[18])), "r"(__float_as_uint(v[19])), "r"(__float_as_uint(v[20])), "r"(__float_as_uint(v[21])), "r"(__float_as_uint(v[22])), "r"(__float_as_uint(v[23])), "r"(__float_as_uint(v[24])), "r"(__float_as_uint(v[25])), "r"(__float_as_uint(v[26])), "r"(__float_as_uint(v[27])), "r"(__float_as_uint(v[28])), "r"(__float_as_uint(v[29])), "r"(__float_as_uint(v[30])), "r"(__float_as_uint(v[31]))
                 : "memory");
}

// This thread's column chunk at taddr (lane quarter and column included): in the
// spread layout the warp addresses its low half's chunk, n columns before a high
// thread's own.
template <bool kSpread>
__device__ __forceinline__ void ld_chunk32(uint32_t taddr, int hi, float (&v)[32])
{
    if (kSpread) tmem_ld16x2_32(taddr - 32u * hi, v);
    else ptx::tmem_ld32(taddr, v);
}
template <bool kSpread>
__device__ __forceinline__ void ld_chunk16(uint32_t taddr, int hi, float (&v)[16])
{
    if (kSpread) tmem_ld16x2_16(taddr - 16u * hi, v);
    else ptx::tmem_ld16(taddr, v);
}
template <bool kSpread>
__device__ __forceinline__ void st_chunk32(uint32_t taddr, int hi, const float (&v)[32])
{
    if (kSpread) tmem_st16x2_32(taddr - 32u * hi, v);
    else ptx::tmem_st32(taddr, v);
}

template <bool kSpread>
__global__ void __launch_bounds__(kThreads, 1) k_attn_tc(const __grid_constant__ TcAttnArgs a)
{
    using namespace ptx;
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int d = a.d, F = a.F, B = a.B, G = a.G;
    const int NC = (2 * F) / 32;
    const int Mv = G * B;
    const uint32_t chunk_bytes = (uint32_t)d * 128;
    const bool wide = F > 128;   // phi+ and phi- take turns in U's columns
    const int RM = a.n_slots + (wide ? kExtraSlots : 0);   // ring slots at most
    // the CTA's contiguous range of units
    const int per = a.n_units / (int)gridDim.x, rem = a.n_units % (int)gridDim.x;
    const int u_begin = (int)blockIdx.x * per + min((int)blockIdx.x, rem);
    const int u_end = u_begin + per + ((int)blockIdx.x < rem ? 1 : 0);

    uint64_t *bars = reinterpret_cast<uint64_t *>(smem + a.off_bar);
    uint64_t *full = bars;
    uint64_t *empty = bars + RM;
    uint64_t *bar_z = bars + 2 * RM;
    uint64_t *bar_u = bar_z + 1;
    uint64_t *bar_d = bar_z + 2;    // both issuers: D_lin halves and D_s are complete (every
                                    // shared-memory operand of the unit has been read)
    uint64_t *bar_p = bar_z + 3;    // F = 256, both issuers: the phi+ readout is done
    uint64_t *bar_u2 = bar_z + 4;   // F = 256: U = Q W formed again, for phi-
    uint64_t *bar_ld = bar_z + 5;   // Q, K, V and W have landed
    uint64_t *bar_b = bar_z + 6;    // issuer B's readout is complete
    uint32_t *tmem_holder = reinterpret_cast<uint32_t *>(bar_z + 7);
    int *fail = reinterpret_cast<int *>(tmem_holder + 1);
    int *issued = fail + 1;   // S chunks of the unit issued so far (for draining after a failure)

    if (tid == 0) {
        for (int i = 0; i < 2 * RM + 7; ++i) mbar_init(&bars[i], 1);
        mbar_init(bar_d, 2);
        mbar_init(bar_p, 2);
        *fail = 0;
        fence_mbar_init();
    }
    if (warp == 0) {
        tmem_alloc(tmem_holder, 512);
        tmem_relinquish();
    }
    __syncthreads();
    tc_fence_after();
    // launched with programmatic stream serialisation: the set-up above may run while the
    // previous kernel of the stream drains, and so may L2 prefetches of the first unit's Q, K
    // and V (a prefetch binds no value); nothing below reads global memory before that kernel
    // has completed
    if (tid == 0) griddep_launch_dependents();
    if (tid == 32 && u_begin < u_end) {
        const int r = u_begin / a.Hkv, g = u_begin % a.Hkv;
        if (kSpread) tma_prefetch_5d(&a.tmQ, 0, g, 0, r * (B / 16), 0);
        tma_prefetch_4d(&a.tmK, 0, g, r * B, 0);
        tma_prefetch_4d(&a.tmV, 0, g, r * B, 0);
    }
    griddep_wait();
    const uint32_t tmem = *tmem_holder;

    // the first unit from u on whose state pointer is usable (u_end if none); each
    // unusable pointer is reported once and its unit skipped
    auto next_unit = [&](int u) -> int {
        for (; u < u_end; ++u) {
            if (state_ptr_ok(a.states[u / a.Hkv])) break;
            if (tid == 0) raise_error(a.err, ERR_BAD_STATE_PTR);
        }
        return u;
    };
    auto head_state = [&](int u) -> const float * {
        return reinterpret_cast<const float *>(a.states[u / a.Hkv]) + (size_t)(u % a.Hkv) * head_floats(d, F);
    };
    // ---- loads of unit u (one thread): Q, K, V, W (TMA), z and the first S tiles
    // (bulk copies of the state image)
    // part 1: K and z (their space is free once the unit's phi- has been formed); part 2:
    // Q, V, W and the first state tiles (free once the unit's MMAs are complete: W's space
    // holds state tiles of the phi- readout when phi- comes from phi+)
    auto issue_loads = [&](int u, const void *st, int part) {
        const int r = u / a.Hkv, g = u % a.Hkv;
        const float *Sg = reinterpret_cast<const float *>(st) + (size_t)g * head_floats(d, F);
        if (part != 2) {
            // the spread Q box brings 128 rows, its padding rows zero-filled
            mbar_arrive_expect_tx(bar_ld, (uint32_t)((kSpread ? 128 : Mv) + 2 * B + F) * d * 2);
            // K: all d / 64 panels in one box
            tma_load_4d(smem + a.off_k, &a.tmK, 0, g, r * B, 0, bar_ld);
            mbar_arrive_expect_tx(bar_z, 2 * F * 4);
            bulk_g2s(smem + a.off_z, Sg + (size_t)2 * F * d, 2 * F * 4, bar_z);
        }
        if (part == 1) return;
        if (kSpread) {
            // query rows 16 q .. 16 q + 15 onto lanes 32 q .. 32 q + 15 (G = 1), rows
            // 16 q + 16 .. 16 q + 31 zero: one box of 2 panels x 4 groups x 32 rows
            tma_load_5d(smem + a.off_q, &a.tmQ, 0, g, 0, r * (B / 16), 0, bar_ld);
        } else {
            for (int c = 0; c < d / 64; ++c)
                tma_load_3d(smem + a.off_q + c * (128 * 128), &a.tmQ, 64 * c, g * G, r * B, bar_ld);
        }
        // V: all d / 64 panels in one box; W: all F / 64 panels in one box
        tma_load_4d(smem + a.off_v, &a.tmV, 0, g, r * B, 0, bar_ld);
        tma_load_3d(smem + a.off_w, &a.tmW, 0, g * d, 0, bar_ld);
        const int pre = NC < a.n_slots ? NC : a.n_slots;
        for (int c = 0; c < pre; ++c) {
            mbar_arrive_expect_tx(&full[c], chunk_bytes);
            bulk_g2s(smem + (size_t)c * chunk_bytes, Sg + (size_t)c * 32 * d, chunk_bytes, &full[c]);
        }
        *issued = pre;
    };

    // row statistics: in Q's buffer once Q is no longer read (F <= 128), else their own
    float *stat = reinterpret_cast<float *>(smem + a.off_st);  // [3][128] m, l, lin_den
    float *ex = stat + 3 * 128;                                 // [8][2][128] exchange
    // Thread -> (TMEM lane, column subset).  Default: lane 32 q4 + lane and the warp's
    // half as subset, two threads per row.  Spread (G = 1, B = 64): query row i sits on
    // lane 32 (i / 16) + i % 16, so the rows occupy all four lane quarters (and SM
    // sub-partitions), and a warp's two 16-thread halves take the same 16 lanes at
    // different columns: four threads per row.
    const int q4 = warp & 3, half = warp >> 2;
    const int hi = kSpread ? lane >> 4 : 0;
    const int row = kSpread ? 32 * q4 + (lane & 15) : 32 * q4 + lane;   // TMEM lane of the query row
    const int qrow = kSpread ? 16 * q4 + (lane & 15) : row;              // query row t G + hh
    const uint32_t lane_off = (uint32_t)(32 * q4) << 16;
    const bool valid = qrow < Mv;
    constexpr int NS = kSpread ? 4 : 2;               // column subsets per row
    const int sub = kSpread ? 2 * half + hi : half;   // owns the chunks k with k % NS == sub
    const int nsc = B / 16;       // 16-column chunks of scores
    const int nfc = F / 32;       // 32-column chunks of U
    // in the spread layout a row's partial results meet across lanes l and l ^ 16 first
    auto comb_max = [&](float x) { return kSpread ? fmaxf(x, __shfl_xor_sync(0xffffffffu, x, 16)) : x; };
    auto comb_min = [&](float x) { return kSpread ? fminf(x, __shfl_xor_sync(0xffffffffu, x, 16)) : x; };
    auto comb_add = [&](float x) { return kSpread ? x + __shfl_xor_sync(0xffffffffu, x, 16) : x; };

    // Units run one after another; the barriers used once per unit complete with
    // the parity of the unit's index it in this CTA.  Ring slot s has had fills and
    // releases of earlier units; fmask / emask bit s hold the parity of their counts.
    uint32_t fmask = 0, emask = 0, it = 0, n_u2 = 0;
    // what one unit adds to them, for the two ring sizes (n_slots, and min(NC, RM) slots
    // when phi- comes from phi+): slot s holds ceil((NC - s) / R) tiles, each released
    // but the last
    auto ring_x = [&](int Rv, bool rel) -> uint32_t {
        uint32_t x = 0;
        for (int sl = 0; sl < Rv; ++sl) {
            const int cnt = (NC - sl + Rv - 1) / Rv;
            x ^= (uint32_t)((rel ? cnt - 1 : cnt) & 1) << sl;
        }
        return x;
    };
    const uint32_t xf0 = ring_x(a.n_slots, false), xe0 = ring_x(a.n_slots, true);
    const uint32_t xf1 = ring_x(min(NC, RM), false), xe1 = ring_x(min(NC, RM), true);
    int u = next_unit(u_begin);
    if (tid == 0 && u < u_end) issue_loads(u, a.states[u / a.Hkv], 0);
    while (u < u_end) {
        const uint32_t up = it & 1u;
        const int r = u / a.Hkv, g = u % a.Hkv;
        const float *Sg = head_state(u);
        // the next unit's state pointer and this row's gate, loaded now (used after the readout)
        const void *nstate = u + 1 < u_end ? a.states[(u + 1) / a.Hkv] : nullptr;
        const float alpha_row = valid ? a.alpha[g * G + qrow % G] : 0.f;
        // phase parity of fill j (or release j) of ring slot s in this unit
        auto fph = [&](int s, int j) -> uint32_t { return ((fmask >> s) & 1u) ^ ((uint32_t)j & 1u); };
        auto eph = [&](int s, int j) -> uint32_t { return ((emask >> s) & 1u) ^ ((uint32_t)j & 1u); };
        bool early = false;   // thread 32: the next unit's first loads went out during this unit

        // ---- U = Q W_g and scores = Q K^T.  W and V are MN-major: 64-wide panels of
        // d (W) or B (V) rows, 8-row groups 1024 bytes apart.
        if (tid == 0) {
            if (mbar_wait(bar_ld, up, kWaitNs)) {
                tc_fence_after();
                const uint32_t q_u = smem_u32(smem + a.off_q), w_u = smem_u32(smem + a.off_w),
                               k_u = smem_u32(smem + a.off_k);
                const uint32_t idU = instr_desc(FMT_BF16, FMT_BF16, false, true, 128, F);
                const uint32_t idS = instr_desc(FMT_BF16, FMT_BF16, false, false, 128, B);
                for (int k = 0; k < d / 16; ++k) {
                    const uint64_t ad = smem_desc(q_u + (k >> 2) * (128 * 128) + (k & 3) * 32, 16, 1024, SWZ_128B);
                    const uint64_t bw = smem_desc(w_u + 2 * k * 1024, d * 128, 1024, SWZ_128B);
                    const uint64_t bk = smem_desc(k_u + (k >> 2) * (B * 128) + (k & 3) * 32, 16, 1024, SWZ_128B);
                    mma_bf16_ss(tmem + kColA, ad, bw, idU, k > 0);
                    mma_bf16_ss(tmem + kColS, ad, bk, idS, k > 0);
                }
                mma_commit(bar_u);
            } else {
                atomicOr(fail, 1);
                mbar_arrive(bar_u);
            }
        }
        if (!mbar_wait(bar_u, up, kWaitNs)) atomicOr(fail, 1);
        tc_fence_after();

        // ring slot s: the dedicated slots, then (F = 256, phi- from phi+) W's and Q's space
        auto slot_ptr = [&](int sl) -> uint8_t * {
            if (sl < a.n_slots) return smem + (size_t)sl * chunk_bytes;
            sl -= a.n_slots;
            return sl < 4 ? smem + a.off_w + (size_t)sl * chunk_bytes : smem + a.off_q + (size_t)(sl - 4) * chunk_bytes;
        };

        // ---- pass 1: local extrema
        {
            float ms = -INFINITY, mx = -INFINITY, mn = INFINITY;
            for (int k = sub; k < nsc; k += NS) {
                float v[16];
                ld_chunk16<kSpread>(tmem + lane_off + kColS + 16 * k, hi, v);
                tmem_wait_ld();
#pragma unroll
                for (int i = 0; i < 16; ++i) ms = fmaxf(ms, v[i]);
            }
            for (int k = sub; k < nfc; k += NS) {
                float v[32];
                ld_chunk32<kSpread>(tmem + lane_off + kColA + 32 * k, hi, v);
                tmem_wait_ld();
#pragma unroll
                for (int i = 0; i < 32; ++i) { mx = fmaxf(mx, v[i]); mn = fminf(mn, v[i]); }
            }
            ex[0 * 256 + half * 128 + row] = comb_max(ms);
            ex[1 * 256 + half * 128 + row] = comb_max(mx);
            ex[2 * 256 + half * 128 + row] = comb_min(mn);
        }
        __syncthreads();
        // F = 256: while every valid row's range of U stays within kRecipRange, phi- follows
        // from phi+ (phi-_j = e^(mn - mx) / (sp sn phi+_j), both sides far from underflow), so
        // U = Q W is not formed again and W's and Q's space takes six more state tiles now
        bool recip = false;
        if (wide) {
            const float rng = fmaxf(ex[1 * 256 + row], ex[1 * 256 + 128 + row]) -
                              fminf(ex[2 * 256 + row], ex[2 * 256 + 128 + row]);
            recip = __syncthreads_and(!valid || rng <= kRecipRange) != 0;
        }
        const int R = recip ? min(NC, RM) : a.n_slots;   // ring slots in use
        if (tid == 0 && R > a.n_slots && *fail == 0) {
            for (int c = a.n_slots; c < R; ++c) {
                mbar_arrive_expect_tx(&full[c], chunk_bytes);
                bulk_g2s(slot_ptr(c), Sg + (size_t)c * 32 * d, chunk_bytes, &full[c]);
            }
            *issued = R;
        }
        if (!mbar_wait(bar_z, up, kWaitNs)) atomicOr(fail, 1);

        // ---- pass 2: exponentials, P, unnormalised phi halves, partial sums
        {
            const float m_raw = fmaxf(ex[0 * 256 + row], ex[0 * 256 + 128 + row]);
            const float mx = fmaxf(ex[1 * 256 + row], ex[1 * 256 + 128 + row]);
            const float mn = fminf(ex[2 * 256 + row], ex[2 * 256 + 128 + row]);
            float l = 0.f, sp = 0.f, sn = 0.f, lp = 0.f, ln = 0.f;
            for (int k = sub; k < nsc; k += NS) {
                float v[16];
                ld_chunk16<kSpread>(tmem + lane_off + kColS + 16 * k, hi, v);
                tmem_wait_ld();
                uint32_t pk[8];
#pragma unroll
                for (int i = 0; i < 16; i += 2) {
                    const float p0 = exp2f((v[i] - m_raw) * a.scale_log2);
                    const float p1 = exp2f((v[i + 1] - m_raw) * a.scale_log2);
                    pk[i / 2] = pack_bf16x2(p0, p1);
                    const __nv_bfloat162 b2 = *reinterpret_cast<const __nv_bfloat162 *>(&pk[i / 2]);
                    l += __low2float(b2) + __high2float(b2);   // sum what the MMA will use
                }
                // P is K-major without swizzle: core matrices of 8 rows x 16 bytes
                uint8_t *prow = smem + a.off_p + (row >> 3) * (B / 8) * 128 + (row & 7) * 16;
                *reinterpret_cast<uint4 *>(prow + (2 * k) * 128) = make_uint4(pk[0], pk[1], pk[2], pk[3]);
                *reinterpret_cast<uint4 *>(prow + (2 * k + 1) * 128) = make_uint4(pk[4], pk[5], pk[6], pk[7]);
            }
            const float *zs = reinterpret_cast<const float *>(smem + a.off_z);
            const float mxl = mx * kLog2e, mnl = mn * kLog2e;
            for (int k = sub; k < nfc; k += NS) {
                float u[32], ep[32], en[32];
                ld_chunk32<kSpread>(tmem + lane_off + kColA + 32 * k, hi, u);
                tmem_wait_ld();
#pragma unroll
                for (int i = 0; i < 32; ++i) {
                    ep[i] = exp2f(fmaf(u[i], kLog2e, -mxl));
                    en[i] = exp2f(fmaf(-u[i], kLog2e, mnl));
                    sp += ep[i];
                    sn += en[i];
                    lp = fmaf(ep[i], zs[32 * k + i], lp);
                    ln = fmaf(en[i], zs[F + 32 * k + i], ln);
                }
                if (wide) {
                    // F = 256: phi+ stays unnormalised (the readout is scaled by 1 / sp)
#pragma unroll
                    for (int i = 0; i < 32; ++i) ep[i] = tf32_round(ep[i]);
                }
                st_chunk32<kSpread>(tmem + lane_off + kColA + 32 * k, hi, ep);
                if (!wide) st_chunk32<kSpread>(tmem + lane_off + kColA + F + 32 * k, hi, en);   // F = 256: formed later
            }
            ex[3 * 256 + half * 128 + row] = comb_add(l);
            ex[4 * 256 + half * 128 + row] = comb_add(sp);
            ex[5 * 256 + half * 128 + row] = comb_add(sn);
            ex[6 * 256 + half * 128 + row] = comb_add(lp);
            ex[7 * 256 + half * 128 + row] = comb_add(ln);
            if (half == 0) stat[row] = m_raw * a.inv_sqrt_d;
            tmem_wait_st();
        }
        __syncthreads();

        // ---- pass 3: normalise phi in place (rounded to tf32; F <= 128), row statistics.
        // With F = 256 the readout accumulates sp phi+ and sp phi-, and lin_scale = 1 / sp
        // scales it back in the epilogue.
        float lin_scale = 1.f;
        {
            const float sp = ex[4 * 256 + row] + ex[4 * 256 + 128 + row];
            const float sn = ex[5 * 256 + row] + ex[5 * 256 + 128 + row];
            const float isp = 1.f / sp, isn = 1.f / sn;
            if (wide) lin_scale = isp;
            for (int k = sub; !wide && k < nfc; k += NS) {
                float v[32];
                ld_chunk32<kSpread>(tmem + lane_off + kColA + 32 * k, hi, v);
                tmem_wait_ld();
#pragma unroll
                for (int i = 0; i < 32; ++i) v[i] = tf32_round(v[i] * isp);
                st_chunk32<kSpread>(tmem + lane_off + kColA + 32 * k, hi, v);
                ld_chunk32<kSpread>(tmem + lane_off + kColA + F + 32 * k, hi, v);
                tmem_wait_ld();
#pragma unroll
                for (int i = 0; i < 32; ++i) v[i] = tf32_round(v[i] * isn);
                st_chunk32<kSpread>(tmem + lane_off + kColA + F + 32 * k, hi, v);
            }
            if (half == 0) {
                stat[128 + row] = ex[3 * 256 + row] + ex[3 * 256 + 128 + row];
                const float lp = ex[6 * 256 + row] + ex[6 * 256 + 128 + row];
                const float ln = ex[7 * 256 + row] + ex[7 * 256 + 128 + row];
                stat[256 + row] = lp * isp + ln * isn;
            }
            tmem_wait_st();
        }
        fence_proxy_async_smem();
        tc_fence_before();
        __syncthreads();

        // ---- readout D_lin = phi(Q) S_g over the 2F/32 state tiles, then D_s = P V.
        // Tile c of phi sits at column kColA + 32 (c - c0) of the phase [c0, c1) that reads
        // it: one phase for F <= 128; for F = 256 the phi+ tiles, then the phi- tiles.
        // Two threads issue the readout: a tcgen05.mma with M = 128 keeps its issuing thread
        // about as long as two tf32 products take on the tensor pipe.  Thread 0 (issuer A)
        // reads the first half of each phase's tiles into D_lin at kColD, thread 64 (issuer
        // B) the second half into kColS (the scores' columns, free once P is written); the
        // epilogue adds the two.  Each accumulator has a fixed issue order.
        const int NC1 = wide ? NC / 2 : NC;
        bool ok = true;   // issuers only
        const int iss = tid == 64 ? 1 : 0;
        // A slot whose tile c is read out in the first phase is refilled (tile c + R) by
        // thread 32 as soon as the tensor cores release it, so the issue loops never wait for
        // a tile to finish.  A second-phase tile's slot (F = 256 with the 4-slot ring) is
        // refilled by the thread that read it, after the tile's MMAs.
        auto issue_tiles = [&](int c0, int c1) {
            const uint32_t idR = instr_desc(FMT_TF32, FMT_TF32, false, false, 128, d);
            const int hn = (c1 - c0) / 2;
            const int cb = c0 + iss * hn, ce = cb + hn;
            const uint32_t dcol = iss ? kColS : kColD;
            for (int c = cb; c < ce && ok; ++c) {
                const int slot = c % R;
                if (!mbar_wait(&full[slot], fph(slot, c / R), kWaitNs)) { ok = false; break; }
                const uint32_t s_u = smem_u32(slot_ptr(slot));
#pragma unroll
                for (int kk = 0; kk < 4; ++kk)
                    mma_tf32_ts(tmem + dcol, tmem + kColA + 32 * (c - c0) + 8 * kk,
                                smem_desc(s_u + 32 * kk, 16, 1024, SWZ_128B), idR, (c0 != 0 || c != cb || kk != 0));
                if (c + R < NC) {
                    mma_commit(&empty[slot]);
                    if (c >= NC1) {
                        if (!mbar_wait(&empty[slot], eph(slot, c / R), kWaitNs)) { ok = false; break; }
                        mbar_arrive_expect_tx(&full[slot], chunk_bytes);
                        bulk_g2s(slot_ptr(slot), Sg + (size_t)(c + R) * 32 * d, chunk_bytes, &full[slot]);
                        atomicMax(issued, c + R + 1);
                    }
                }
            }
        };
        if (tid == 32 && *fail == 0) {
            for (int c = R; c < NC && c - R < NC1; ++c) {
                const int slot = c % R;
                if (!mbar_wait(&empty[slot], eph(slot, (c - R) / R), kWaitNs)) {
                    atomicOr(fail, 1);
                    break;
                }
                mbar_arrive_expect_tx(&full[slot], chunk_bytes);
                bulk_g2s(slot_ptr(slot), Sg + (size_t)c * 32 * d, chunk_bytes, &full[slot]);
                atomicMax(issued, c + 1);
            }
        }
        if (tid == 0 || tid == 64) {
            ok = *fail == 0;
            if (ok) {
                tc_fence_after();
                issue_tiles(0, NC1);
            }
            if (wide) {
                if (ok) mma_commit(bar_p);
                else mbar_arrive(bar_p);
            }
        }
        if (wide) {
            // the tensor cores are done with phi+; phi- takes its columns
            if (!mbar_wait(bar_p, up, kWaitNs)) atomicOr(fail, 1);
            if (recip) {
                // sp phi-_j = e^(mn - mx) sp isn / e^(u_j - mx), rounded to tf32 (the
                // unnormalised phi+ in Tensor Memory is e^(u_j - mx))
                tc_fence_after();
                const float mx = fmaxf(ex[1 * 256 + row], ex[1 * 256 + 128 + row]);
                const float mn = fminf(ex[2 * 256 + row], ex[2 * 256 + 128 + row]);
                const float sp = ex[4 * 256 + row] + ex[4 * 256 + 128 + row];
                const float isn = 1.f / (ex[5 * 256 + row] + ex[5 * 256 + 128 + row]);
                const float kr = exp2f((mn - mx) * kLog2e) * sp * isn;
                for (int k = sub; k < nfc; k += NS) {
                    float v[32];
                    ld_chunk32<kSpread>(tmem + lane_off + kColA + 32 * k, hi, v);
                    tmem_wait_ld();
#pragma unroll
                    for (int i = 0; i < 32; ++i) v[i] = tf32_round(__fdividef(kr, v[i]));
                    st_chunk32<kSpread>(tmem + lane_off + kColA + 32 * k, hi, v);
                }
                tmem_wait_st();
            } else {
                // form U = Q W_g again in phi+'s columns
                if (tid == 0) {
                    ok = ok && *fail == 0;
                    if (ok) {
                        tc_fence_after();
                        const uint32_t q_u = smem_u32(smem + a.off_q), w_u = smem_u32(smem + a.off_w);
                        const uint32_t idU = instr_desc(FMT_BF16, FMT_BF16, false, true, 128, F);
                        for (int k = 0; k < d / 16; ++k)
                            mma_bf16_ss(tmem + kColA,
                                        smem_desc(q_u + (k >> 2) * (128 * 128) + (k & 3) * 32, 16, 1024, SWZ_128B),
                                        smem_desc(w_u + 2 * k * 1024, d * 128, 1024, SWZ_128B), idU, k > 0);
                        mma_commit(bar_u2);
                    } else {
                        mbar_arrive(bar_u2);
                    }
                }
                if (!mbar_wait(bar_u2, n_u2 & 1u, kWaitNs)) atomicOr(fail, 1);
                ++n_u2;
                tc_fence_after();
                // sp phi- = sp softmax(-U), from the same extremum and sums as pass 2, rounded to tf32
                const float mnl = fminf(ex[2 * 256 + row], ex[2 * 256 + 128 + row]) * kLog2e;
                const float spn = (ex[4 * 256 + row] + ex[4 * 256 + 128 + row]) /
                                  (ex[5 * 256 + row] + ex[5 * 256 + 128 + row]);
                for (int k = sub; k < nfc; k += NS) {
                    float v[32];
                    ld_chunk32<kSpread>(tmem + lane_off + kColA + 32 * k, hi, v);
                    tmem_wait_ld();
#pragma unroll
                    for (int i = 0; i < 32; ++i) v[i] = tf32_round(exp2f(fmaf(-v[i], kLog2e, mnl)) * spn);
                    st_chunk32<kSpread>(tmem + lane_off + kColA + 32 * k, hi, v);
                }
                tmem_wait_st();
            }
            tc_fence_before();
            __syncthreads();
            // the next unit's K and z: K was read by the scores, z by pass 2
            if (tid == 32 && *fail == 0 && u + 1 < u_end && state_ptr_ok(nstate)) {
                early = true;
                fence_proxy_async_smem();
                issue_loads(u + 1, nstate, 1);
            }
        }
        if (tid == 0 || tid == 64) {
            ok = ok && *fail == 0;
            if (ok) {
                tc_fence_after();
                if (NC1 < NC) issue_tiles(NC1, NC);
                // D_s = P V over phi's first d columns.  Issuer B's tiles of the last phase sit
                // from column 32 (NC - NC1) / 2 on (F with F <= 128, 128 with F = 256); if d
                // reaches there, A waits for B's readout, else only A's own earlier (in-order)
                // MMAs read those columns
                if (iss == 1 && ok) mma_commit(bar_b);
                if (ok && iss == 0 && d > 16 * (wide ? NC - NC1 : NC) && !mbar_wait(bar_b, up, kWaitNs)) ok = false;
                if (ok && iss == 0) {
                    const uint32_t p_u = smem_u32(smem + a.off_p), v_u = smem_u32(smem + a.off_v);
                    const uint32_t idP = instr_desc(FMT_BF16, FMT_BF16, false, true, 128, d);
                    for (int k = 0; k < B / 16; ++k) {
                        const uint64_t ad = smem_desc(p_u + k * 256, 128, (B / 8) * 128, SWZ_NONE);
                        const uint64_t bd = smem_desc(v_u + 2 * k * 1024, B * 128, 1024, SWZ_128B);
                        mma_bf16_ss(tmem + kColA, ad, bd, idP, k > 0);
                    }
                }
                if (ok) mma_commit(bar_d);
            }
            if (!ok) {
                atomicOr(fail, 1);
                if (iss == 1) mbar_arrive(bar_b);
                mbar_arrive(bar_d);   // release the waiting threads
            }
        }
        if (!mbar_wait(bar_d, up, kWaitNs)) atomicOr(fail, 1);
        tc_fence_after();
        // the row's statistics (with F <= 128 in Q's buffer, which the next unit's Q overwrites)
        const float m = stat[row], l = stat[128 + row], ld = stat[256 + row];
        const int issued_now = *issued;   // the next unit's copies reset the count
        // (a unit whose first part of loads went out is completed even after a failure,
        // so that every barrier the drain waits on completes)
        const bool early_any = __syncthreads_or(early) != 0;
        const bool failed = *fail != 0;
        // every operand in shared memory has been read: the next unit's loads go out now and
        // land while this unit's epilogue runs
        const uint32_t fmask_n = fmask ^ (recip ? xf1 : xf0), emask_n = emask ^ (recip ? xe1 : xe0);
        const int un = early_any ? u + 1 : failed ? u_end : u + 1 < u_end && state_ptr_ok(nstate) ? u + 1
                                                                                      : next_unit(u + 1);
        if (tid == 32 && un < u_end) {
            fence_proxy_async_smem();
            issue_loads(un, un == u + 1 ? nstate : a.states[un / a.Hkv], early ? 2 : 0);
        }

        // ---- epilogue: out = ws * D_s + wl * D_lin, stored as bf16
        if (!failed) {
            const int t = qrow / G, hh = qrow % G;
            MergeWeights mw{0.f, 0.f};
            if (valid) mw = merge_weights(log_sigmoid(alpha_row), m, l, ld);
            mw.wl *= lin_scale;
            __nv_bfloat16 *orow0 = a.O + (((size_t)r * B + t) * a.Hq + g * G + hh) * d;
            for (int kd = sub; kd < d / 32; kd += NS) {
                const int c0 = 32 * kd;
                float dl[32], d2[32], ds[32];
                ld_chunk32<kSpread>(tmem + lane_off + kColD + c0, hi, dl);
                ld_chunk32<kSpread>(tmem + lane_off + kColS + c0, hi, d2);
                ld_chunk32<kSpread>(tmem + lane_off + kColA + c0, hi, ds);
                tmem_wait_ld();
#pragma unroll
                for (int i = 0; i < 32; ++i) dl[i] += d2[i];
                if (valid) {
                    uint32_t pk[16];
#pragma unroll
                    for (int i = 0; i < 32; i += 2) {
                        const float o0 = mw.ws * ds[i] + (mw.wl == 0.f ? 0.f : mw.wl * dl[i]);
                        const float o1 = mw.ws * ds[i + 1] + (mw.wl == 0.f ? 0.f : mw.wl * dl[i + 1]);
                        pk[i / 2] = pack_bf16x2(o0, o1);
                    }
                    uint4 *dst = reinterpret_cast<uint4 *>(orow0 + c0);
#pragma unroll
                    for (int i = 0; i < 4; ++i) dst[i] = make_uint4(pk[4 * i], pk[4 * i + 1], pk[4 * i + 2], pk[4 * i + 3]);
                }
            }
        } else if (tid == 0) {
            raise_error(a.err, ERR_WAIT_TIMEOUT);
            // drain bulk copies that may still be landing in this CTA's shared memory
            mbar_wait(bar_ld, up, kWaitNs);
            mbar_wait(bar_z, up, kWaitNs);
            for (int c = 0; c < issued_now; ++c) mbar_wait(&full[c % R], fph(c % R, c / R), kWaitNs);
            if (un < u_end) {
                // the next unit's loads, issued before the failure was seen
                mbar_wait(bar_ld, up ^ 1u, kWaitNs);
                mbar_wait(bar_z, up ^ 1u, kWaitNs);
                for (int c = 0; c < NC && c < a.n_slots; ++c) mbar_wait(&full[c], (fmask_n >> c) & 1u, kWaitNs);
            }
        }
        fmask = fmask_n;
        emask = emask_n;
        ++it;
        tc_fence_before();
        __syncthreads();
        if (failed) break;
        u = un;
    }
    if (warp == 0) {
        tc_fence_after();
        tmem_dealloc(tmem, 512);
    }
}

}  // namespace

bool tc_attn_supported(const hybrid_cfg &c)
{
    if (c.io_dtype != HYBRID_BF16) return false;
    if (c.head_dim != 64 && c.head_dim != 128) return false;
    if (c.feat_dim != 64 && c.feat_dim != 128 && c.feat_dim != 256) return false;
    if (c.block_size % 16 != 0) return false;
    const int G = c.n_q_heads / c.n_kv_heads;
    if (G * c.block_size > 128) return false;
    const Layout L = make_layout(c.head_dim, c.feat_dim, c.block_size);
    return L.n_slots >= 1 && (int)L.bytes <= kSmemLimit;
}

cudaError_t launch_attn_tc(const hybrid_cfg &c, const void *Q, const void *K, const void *V, const void *W,
                           const float *alpha, void *const *states, int n_req, void *O, unsigned *err,
                           cudaStream_t st)
{
    const Layout L = make_layout(c.head_dim, c.feat_dim, c.block_size);
    TcAttnArgs a;
    // G = 1 with B = 64: 64 query rows spread over the four TMEM lane quarters
    const bool spread = c.n_q_heads == c.n_kv_heads && c.block_size == 64;
    {
        const int d = c.head_dim, F = c.feat_dim, B = c.block_size, Hq = c.n_q_heads, Hkv = c.n_kv_heads;
        const cuuint64_t rows = (cuuint64_t)n_req * B;
        const cuuint64_t dq[3] = {(cuuint64_t)d, (cuuint64_t)Hq, rows};
        const cuuint64_t sq[2] = {(cuuint64_t)d * 2, (cuuint64_t)Hq * d * 2};
        const cuuint32_t bq[3] = {64, (cuuint32_t)(Hq / Hkv), (cuuint32_t)B};
        // spread (G = 1, B = 64): Q as [panel][16-token group][token in group][head][64],
        // the box 32 tokens deep over a dimension of 16, so that each group's 16 rows are
        // followed by 16 zero-filled ones (lanes 32 q .. 32 q + 31 of quarter q)
        const cuuint64_t dqs[5] = {64, (cuuint64_t)Hq, 16, rows / 16, (cuuint64_t)d / 64};
        const cuuint64_t sqs[4] = {(cuuint64_t)d * 2, (cuuint64_t)Hq * d * 2, (cuuint64_t)16 * Hq * d * 2, 128};
        const cuuint32_t bqs[5] = {64, 1, 32, (cuuint32_t)B / 16, (cuuint32_t)d / 64};
        // K, V [rows][Hkv][d] and W [Hkv d][F] with their 64-element panels as the
        // outermost box dimension (stride 128 bytes), so one copy brings every panel
        const cuuint64_t dk[4] = {64, (cuuint64_t)Hkv, rows, (cuuint64_t)d / 64};
        const cuuint64_t sk[3] = {(cuuint64_t)d * 2, (cuuint64_t)Hkv * d * 2, 128};
        const cuuint32_t bk[4] = {64, 1, (cuuint32_t)B, (cuuint32_t)d / 64};
        const cuuint64_t dw[3] = {64, (cuuint64_t)Hkv * d, (cuuint64_t)F / 64};
        const cuuint64_t sw[2] = {(cuuint64_t)F * 2, 128};
        const cuuint32_t bw[3] = {64, (cuuint32_t)d, (cuuint32_t)F / 64};
        if (!(spread ? pipe::encode_bf16(&a.tmQ, Q, 5, dqs, sqs, bqs) : pipe::encode_bf16(&a.tmQ, Q, 3, dq, sq, bq)) || !pipe::encode_bf16(&a.tmK, K, 4, dk, sk, bk) ||
            !pipe::encode_bf16(&a.tmV, V, 4, dk, sk, bk) || !pipe::encode_bf16(&a.tmW, W, 3, dw, sw, bw))
            return cudaErrorInvalidValue;
    }
    a.alpha = alpha;
    a.states = states;
    a.O = static_cast<__nv_bfloat16 *>(O);
    a.err = err;
    a.B = c.block_size;
    a.Hq = c.n_q_heads;
    a.Hkv = c.n_kv_heads;
    a.G = c.n_q_heads / c.n_kv_heads;
    a.d = c.head_dim;
    a.F = c.feat_dim;
    a.n_slots = L.n_slots;
    a.inv_sqrt_d = 1.f / sqrtf((float)c.head_dim);
    a.scale_log2 = kLog2e * a.inv_sqrt_d;
    a.off_q = L.off_q;
    a.off_w = L.off_w;
    a.off_k = L.off_k;
    a.off_v = L.off_v;
    a.off_p = L.off_p;
    a.off_z = L.off_z;
    a.off_st = L.off_st;
    a.off_bar = L.off_bar;
    auto kern = spread ? k_attn_tc<true> : k_attn_tc<false>;
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)L.bytes);
    if (e != cudaSuccess) return e;
    a.n_units = n_req * c.n_kv_heads;
    const int grid = a.n_units < pipe::sm_count() ? a.n_units : pipe::sm_count();
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
    return cudaLaunchKernelEx(&lc, kern, a);
}

}  // namespace hyb
