// hybrid_train.cu -- the training form of block-hybrid attention (Section 3.2,
// Stage 1 attention transfer): the states seen by every block of a training
// sequence, and the gradient of sum(dO * O) with respect to W and alpha.
//
// A training sequence of L = n_blk * B tokens is cut into blocks of B tokens;
// block n reads S_{n-1} = sum_{m < n} dS_m, z_{n-1} likewise (Section 3.1 applied
// to every block, S_{-1} = 0), with dS_m = sum_{t in B_m} phi(k_t) [v_t | 1]^T.
// Per query row i of block n (N, D = numerator and denominator of the merge,
// g = dO row, o = N / D):
//     dN = g / D,  dD = -(g . o) / D,  dw_h += dN . sm_num + dD sm_den,
//     dphi(q) = S_{n-1} dN + z_{n-1} dD,   dR_n += phi(q) [dN | dD]^T,
// and a key t of block m receives dphi(k_t) = R_m v_t + r_m with
// [R_m | r_m] = sum_{n > m} dR_n.  Through phi = [softmax(u), softmax(-u)],
// u = x W:  du = p+ (g+ - <g+, p+>) - p- (g- - <g-, p->),  dW += x du^T.
//
// Kernels (128 threads; thread r owns row r of a tile and Tensor Memory lane r):
//   k_prefix_states one CTA per (sequence, state head, 32-feature slice): sweeps
//                   the blocks in order with the slice of S^T accumulating in
//                   Tensor Memory (S^T += V^T phi(K), bf16 MMA) and writes
//                   S_{n-1}, z_{n-1} into slot n of the decode image P (S^T
//                   tiles, read by the decode readout kernel) and of the
//                   feature-row image PT (S tiles: row f holds 32 consecutive e,
//                   128-byte swizzle), whose d/32 tiles are K-major tf32
//                   operands for S dN
//   k_slot_scan     reverse exclusive running sums over the R slots of a
//                   sequence (one CTA per (sequence, block, state head) below)
//   k_phi_grad<Q>   query side: [U | scores] = Q [W | K^T], dO V^T, the merge
//                   terms, dN into Tensor Memory, then S dN streamed over the PT
//                   tiles; g . o = w g.sm_num/D + phi(q).(S dN) and the gate term
//                   are formed from these fp32 products (the forward's rounded O is
//                   not needed), then du_q and dR_n = phi(Q)^T [dN | dD];
//                   key side: U = K W, V into Tensor Memory, R v + r over the
//                   R tiles, du_k
//   k_dw            dW_g = sum over query and key rows of x du^T, split over
//                   row ranges; each CTA writes its partial sum
//   k_grad_reduce   dW and d alpha from the per-CTA and per-block partial sums,
//                   added in a fixed order, so the gradients are the same bits
//                   from run to run
#include <algorithm>
#include <atomic>

#include "hybrid_common.cuh"
#include "hybrid_train.h"
#include "tc_pipeline.cuh"

namespace hyb {

namespace {

using namespace pipe;

constexpr int kThreads = 128;
constexpr int kSmemLimit = 232448;
constexpr uint32_t kColS = 0, kColGv = 64, kColU = 256, kColY = 384, kColG = 0, kColDR = 0;
constexpr int kDwStages = 3;   // shared-memory stages of k_dw
constexpr int kGradThreads = 256;   // k_phi_grad: two threads (parts) per Tensor Memory lane
constexpr uint32_t kXchBytes = 14 * 1024;   // k_phi_grad: the parts' exchange of row partials

struct TrainArgs {
    // 128-byte-swizzled tensor maps: Q and dO [n*L][Hq][d] with box {64, G, B} (rows t*G + h),
    // K and V [n*L][Hkv][d] with box {64, 1, B} (a block) and {64, 1, GR} (a group of the prefix
    // sweep), W [Hkv*d][F] with box {64, d}
    CUtensorMap tmQ, tmdO, tmK, tmV, tmKg, tmVg, tmW;
    const bf16 *Q, *K, *V, *W, *dO;
    const float *alpha;
    float *P, *PT, *R;
    bf16 *dUq, *dUk;
    float *dalpha;
    float *dap;   // per (sequence, block, state head): the G gate terms, summed by k_grad_reduce
    unsigned *err;
    int n_seq, L, B, Hq, Hkv, d, F, n_blk;
};

// Partial sums of dW kept for the ordered reduction: at most this many CTAs of
// k_dw in all, kMaxDwParts / Hkv per state head.
constexpr int kMaxDwParts = 256;

__host__ __device__ __forceinline__ size_t slot_floats(int Hkv, int d, int F)
{
    return (size_t)Hkv * head_floats(d, F);
}

// Feature-row head block (PT and R): logical S[f][e] at float offset
//     (e/32)*64F + f*32 + 4*(((e%32)/4) ^ (f%8)) + e%4,
// i.e. d/32 tiles of 2F rows x 32 consecutive e, each 128-byte row with its
// 16-byte granules permuted by XOR with (f mod 8); then z[f] at 2F*d + f, as in
// the decode image.  A tile is a K-major tf32 operand [N = 2F rows, K = 32 e].

// byte offset of 16-byte granule j of row r inside a 128-byte-swizzled panel
__device__ __forceinline__ uint32_t swz(int r, int j)
{
    return (uint32_t)r * 128u + (uint32_t)((j ^ (r & 7)) << 4);
}

__device__ __forceinline__ void bulk_wait_read_1() { asm volatile("cp.async.bulk.wait_group.read 1;" ::: "memory"); }

// Write 32 consecutive columns [c0, c0 + 32) of row r (values x, converted to
// bf16) into a bf16 operand image with panel stride pstride.
__device__ __forceinline__ void store_row32_bf16(uint8_t *img, uint32_t pstride, int r, int c0, const float (&x)[32])
{
    uint8_t *base = img + (uint32_t)(c0 >> 6) * pstride;
    const int j0 = (c0 & 63) >> 3;
#pragma unroll
    for (int q = 0; q < 4; ++q) {
        uint4 v;
        v.x = pack_bf16x2(x[8 * q + 0], x[8 * q + 1]);
        v.y = pack_bf16x2(x[8 * q + 2], x[8 * q + 3]);
        v.z = pack_bf16x2(x[8 * q + 4], x[8 * q + 5]);
        v.w = pack_bf16x2(x[8 * q + 6], x[8 * q + 7]);
        *reinterpret_cast<uint4 *>(base + swz(r, j0 + q)) = v;
    }
}

// Row statistics of phi = [softmax(u), softmax(-u)] for the F values of u in
// Tensor Memory columns [col, col + F) of this thread's lane.
struct PhiStats {
    float mp, sp, mn, sn;   // max u, sum e^(u - mp), min u, sum e^(mn - u)
};
__device__ __forceinline__ PhiStats phi_stats(uint32_t taddr, int F)
{
    PhiStats s{-INFINITY, 0.f, INFINITY, 0.f};
    float x[32];
    for (int j = 0; j < F / 32; ++j) {
        ptx::tmem_ld32(taddr + 32 * j, x);
        ptx::tmem_wait_ld();
#pragma unroll
        for (int k = 0; k < 32; ++k) {
            s.mp = fmaxf(s.mp, x[k]);
            s.mn = fminf(s.mn, x[k]);
        }
    }
    for (int j = 0; j < F / 32; ++j) {
        ptx::tmem_ld32(taddr + 32 * j, x);
        ptx::tmem_wait_ld();
#pragma unroll
        for (int k = 0; k < 32; ++k) {
            s.sp += ex2((x[k] - s.mp) * kLog2e);
            s.sn += ex2((s.mn - x[k]) * kLog2e);
        }
    }
    return s;
}

// Partial statistics of the same over the 32-column chunks [j0, j1) only, to be
// combined with the other chunks' by combine_stats.
__device__ __forceinline__ PhiStats phi_stats_chunks(uint32_t taddr, int j0, int j1)
{
    PhiStats s{-INFINITY, 0.f, INFINITY, 0.f};
    float x[32];
    for (int j = j0; j < j1; ++j) {
        ptx::tmem_ld32(taddr + 32 * j, x);
        ptx::tmem_wait_ld();
#pragma unroll
        for (int k = 0; k < 32; ++k) {
            s.mp = fmaxf(s.mp, x[k]);
            s.mn = fminf(s.mn, x[k]);
        }
    }
    for (int j = j0; j < j1; ++j) {
        ptx::tmem_ld32(taddr + 32 * j, x);
        ptx::tmem_wait_ld();
#pragma unroll
        for (int k = 0; k < 32; ++k) {
            s.sp += ex2((x[k] - s.mp) * kLog2e);
            s.sn += ex2((s.mn - x[k]) * kLog2e);
        }
    }
    return s;
}
// Statistics of the whole row from the two halves' (a first, then b: both threads
// of a row combine in the same order and get the same bits).
__device__ __forceinline__ PhiStats combine_stats(const PhiStats &a, const PhiStats &b)
{
    PhiStats s;
    s.mp = fmaxf(a.mp, b.mp);
    s.mn = fminf(a.mn, b.mn);
    s.sp = a.sp * ex2((a.mp - s.mp) * kLog2e) + b.sp * ex2((b.mp - s.mp) * kLog2e);
    s.sn = a.sn * ex2((s.mn - a.mn) * kLog2e) + b.sn * ex2((s.mn - b.mn) * kLog2e);
    return s;
}

// Shared memory of the row kernels (bytes, all 1024-aligned)
struct RowLayout {
    uint32_t off_q, off_w, off_k, off_v, off_do, off_phi, off_y, off_z, off_x, off_bar, bytes;
    uint32_t off_ring, ring_slot;
};

// k_phi_grad: phase-one operands (Q, W, K, V) share their space with the ring of
// S / R tiles used afterwards; dO shares its space with phi(Q).
RowLayout make_grad_layout(int d, int F, int B)
{
    RowLayout Lr{};
    const uint32_t rows128 = (uint32_t)(d / 64) * 128 * 128;        // 128 rows x d bf16
    const uint32_t wbytes = (uint32_t)(F / 64) * d * 128;           // d rows x F bf16
    const uint32_t kvbytes = (uint32_t)(d / 64) * B * 128;          // B rows x d bf16
    uint32_t off = 0;
    Lr.off_q = off;
    Lr.off_w = Lr.off_q + rows128;
    Lr.off_k = Lr.off_w + wbytes;
    Lr.off_v = Lr.off_k + kvbytes;
    uint32_t phase1 = Lr.off_v + kvbytes;
    Lr.ring_slot = (uint32_t)2 * F * 128;                            // 2F rows x 32 floats
    Lr.off_ring = 0;
    const uint32_t ring = 2 * Lr.ring_slot;
    off = phase1 > ring ? phase1 : ring;
    Lr.off_phi = off;                                               // 128 rows x 2F bf16; dO first
    off += (uint32_t)(2 * F / 64) * 128 * 128;
    Lr.off_do = Lr.off_phi;
    Lr.off_y = off;                                                 // 128 rows x (d + 16) bf16
    off += (uint32_t)((d + 16 + 63) / 64) * 128 * 128;
    Lr.off_z = off;
    off += (((uint32_t)2 * F * 4) + 1023) & ~1023u;
    Lr.off_x = off;
    off += kXchBytes;
    Lr.off_bar = off;
    off += 1024;
    Lr.bytes = off + 1024;
    return Lr;
}

__device__ __forceinline__ uint8_t *aligned_smem(uint8_t *raw)
{
    return reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(raw) + 1023) & ~uintptr_t(1023));
}

// ---------------------------------------------------------------------------
// k_prefix_states: S_{n-1}, z_{n-1} of every block n of a sequence for one
// 32-feature slice of one state head, written into slot n of P and PT.  The CTA
// sweeps the blocks in order with the running slice S^T (row e per thread):
//                                S^T += V_n^T phi_slice(K_n)  (bf16 MMA, the
// slice of phi taken from the full-F softmaxes), z += sum_t phi_slice(k_t)
// (fp32).  Keys are processed min(4, 128 / B) blocks at a time: U = K W for
// the rows, phi of the slice into a K-major [feature][token] operand, the
// increments of the group's blocks into their own Tensor Memory columns (one
// commit), then per block: store the running state (registers, thread = e)
// into its slot and add the block's increment.
// Shared memory: W, K rows, V rows (two panels of 64 e, the second zero for
// d = 64, so that V^T is an M = 128 operand), phi slice, row scratch (in K's
// space); 107 KB and 256 Tensor Memory columns, so two CTAs share an SM.
// ---------------------------------------------------------------------------
struct PrefixLayout {
    uint32_t off_w, off_k, off_v, off_p, off_x, off_z, off_bar, bytes;
};

PrefixLayout make_prefix_layout(int d, int F)
{
    PrefixLayout Lp{};
    uint32_t off = 0;
    Lp.off_w = off;
    off += (uint32_t)(F / 64) * d * 128;
    Lp.off_k = off;
    off += (uint32_t)(d / 64) * 128 * 128;
    Lp.off_v = off;
    off += 2u * 128 * 128;
    Lp.off_p = off;                    // 32 feature rows x 128 tokens (two 64-token panels)
    off += 2u * 32 * 128;
    Lp.off_x = Lp.off_k;               // 128 tokens x 32 fp32 (the slice of phi, for z): K is
                                       // dead once U = K W is formed
    Lp.off_z = off;                    // running z of the slice and per-block dz (fp32)
    off += 1024;
    Lp.off_bar = off;
    off += 1024;
    Lp.bytes = off + 1024;
    return Lp;
}

__global__ void __launch_bounds__(kThreads, 1) k_prefix_states(const __grid_constant__ TrainArgs a, PrefixLayout Lp)
{
    using namespace ptx;
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = aligned_smem(smem_raw);
    const int tid = threadIdx.x, warp = tid >> 5;
    const int d = a.d, F = a.F, B = a.B, Hkv = a.Hkv, n_blk = a.n_blk;
    const int NSL = 2 * F / 32;
    const int j = blockIdx.x % NSL, g = (blockIdx.x / NSL) % Hkv, s = blockIdx.x / (NSL * Hkv);
    const bool neg = j >= F / 32;              // slice of phi- features
    const int fu = (j % (F / 32)) * 32;        // first column of u the slice reads
    const size_t hf = head_floats(d, F);
    const int GB = min(4, 128 / B);            // blocks per group (at most 128 key rows)
    uint64_t *bar = reinterpret_cast<uint64_t *>(smem + Lp.off_bar);
    uint32_t *tmem_holder = reinterpret_cast<uint32_t *>(bar + 2);
    volatile int *fail = reinterpret_cast<volatile int *>(tmem_holder + 1);
    float *dz = reinterpret_cast<float *>(smem + Lp.off_z);   // [GB][32] dz of the group's blocks
    float *xs = reinterpret_cast<float *>(smem + Lp.off_x);   // [128][32] phi slice of the rows
    uint64_t *tbar = &bar[1];   // a group's K and V rows (and, with the first, W) have landed
    if (tid == 0) {
        mbar_init(&bar[0], 1);
        mbar_init(tbar, 1);
        *fail = 0;
        fence_mbar_init();
        prefetch_tensormap(&a.tmKg);
        prefetch_tensormap(&a.tmVg);
        prefetch_tensormap(&a.tmW);
    }
    if (warp == 0) {
        tmem_alloc(tmem_holder, 256);
        tmem_relinquish();
    }
    // the second 64-e panel of V^T stays zero for d = 64
    if (d == 64)
        for (int i = tid; i < 1024; i += kThreads)
            reinterpret_cast<uint4 *>(smem + Lp.off_v + 128 * 128)[i] = make_uint4(0, 0, 0, 0);
    fence_proxy_async_smem();
    __syncthreads();
    griddep_wait();
    tc_fence_after();
    const uint32_t tmem = *tmem_holder;
    const uint32_t lane_off = (uint32_t)(warp & 3) * 32u << 16;
    constexpr uint32_t kAcc = 128;             // the group's dS^T slices: columns [128, 128 + 32 GB)
    uint32_t phase = 0;
    bool ok = true;
    float run[32];                             // S_{n-1}^T slice, row e = tid (e < d)
#pragma unroll
    for (int k = 0; k < 32; ++k) run[k] = 0.f;
    float zc = 0.f;                            // z_{n-1} of feature 32 j + tid (tid < 32)
    const uint32_t w_u = smem_u32(smem + Lp.off_w), k_u = smem_u32(smem + Lp.off_k),
                   v_u = smem_u32(smem + Lp.off_v), p_u = smem_u32(smem + Lp.off_p);
    for (int b0 = 0; b0 < n_blk && ok; b0 += GB) {
        const int nb = min(GB, n_blk - b0), nt = nb * B;
        const size_t t0 = (size_t)s * a.L + (size_t)b0 * B;
        // the group's K and V rows by TMA (boxes of GB*B rows; rows past the sequence or past
        // the tensor are not used: their phi is zeroed and no MMA reads them)
        if (tid == 0) {
            const uint32_t box = (uint32_t)(d / 64) * (uint32_t)(GB * B) * 128;
            mbar_arrive_expect_tx(tbar, 2 * box + (b0 == 0 ? (uint32_t)(F / 64) * d * 128 : 0u));
            for (int p = 0; p < d / 64; ++p) {
                tma_load_3d(smem + Lp.off_k + p * 128 * 128, &a.tmKg, 64 * p, g, (int)t0, tbar);
                tma_load_3d(smem + Lp.off_v + p * 128 * 128, &a.tmVg, 64 * p, g, (int)t0, tbar);
            }
            if (b0 == 0)
                for (int p = 0; p < F / 64; ++p)
                    tma_load_2d(smem + Lp.off_w + p * d * 128, &a.tmW, 64 * p, g * d, tbar);
        }
        ok = wait_bar(tbar, (uint32_t)(b0 / GB) & 1u, fail) && ok;
        tc_fence_before();
        __syncthreads();
        tc_fence_after();
        if (tid == 0) {
            const uint32_t idU = instr_desc(FMT_BF16, FMT_BF16, false, true, 128, F);
            for (int k = 0; k < d / 16; ++k)
                mma_bf16_ss(tmem, smem_desc(k_u + (k >> 2) * (128 * 128) + (k & 3) * 32, 16, 1024, SWZ_128B),
                            smem_desc(w_u + 2 * k * 1024, d * 128, 1024, SWZ_128B), idU, k > 0);
            mma_commit(&bar[0]);
        }
        ok = wait_bar(&bar[0], phase & 1u, fail);
        ++phase;
        tc_fence_after();
        // the slice of phi of row tid (full-F softmax statistics), bf16 into the
        // [feature][token] operand and fp32 into the row scratch
        {
            const PhiStats st = phi_stats(tmem + lane_off, F);
            const float inv = 1.f / (neg ? st.sn : st.sp);
            float x[32];
            tmem_ld32(tmem + lane_off + (uint32_t)fu, x);
            tmem_wait_ld();
            const bool valid = tid < nt;
#pragma unroll
            for (int k = 0; k < 32; ++k) {
                const float ph = valid ? ex2((neg ? (st.mn - x[k]) : (x[k] - st.mp)) * kLog2e) * inv : 0.f;
                xs[tid * 32 + ((k + tid) & 31)] = ph;   // rotated: conflict-free across the warp
                const __nv_bfloat16 hb = __float2bfloat16_rn(ph);
                uint8_t *row = smem + Lp.off_p + (uint32_t)(tid >> 6) * (32 * 128) + (uint32_t)k * 128u;
                *reinterpret_cast<__nv_bfloat16 *>(row + (((((tid & 63) >> 3) ^ (k & 7))) << 4) + (tid & 7) * 2) = hb;
            }
        }
        fence_proxy_async_smem();
        tc_fence_before();
        __syncthreads();
        tc_fence_after();
        // dz of each block of the group: sum over its B rows, feature tid % 32
        for (int q = tid; q < nb * 32; q += kThreads) {
            const int bl = q >> 5, f = q & 31;
            float acc = 0.f;
            for (int t = bl * B; t < bl * B + B; ++t) acc += xs[t * 32 + ((f + t) & 31)];
            dz[bl * 32 + f] = acc;
        }
        __syncthreads();
        // the group's increments dS_n = V_n^T phi_slice(K_n), block bl into columns
        // [128 + 32 bl, 160 + 32 bl) (not those of the sequence's last block)
        if (tid == 0) {
            const uint32_t idS = instr_desc(FMT_BF16, FMT_BF16, true, false, 128, 32);
            for (int bl = 0; bl < nb; ++bl) {
                if (b0 + bl == n_blk - 1) break;
                for (int ks = 0; ks < B / 16; ++ks) {
                    const int tk = bl * B + 16 * ks;   // first token row of this k-step
                    mma_bf16_ss(tmem + kAcc + 32u * bl,
                                smem_desc(v_u + (uint32_t)(tk / 16) * 2048, 128 * 128, 1024, SWZ_128B),
                                smem_desc(p_u + (uint32_t)(tk >> 6) * (32 * 128) + (uint32_t)(tk & 63) * 2, 16, 1024,
                                          SWZ_128B),
                                idS, ks > 0 ? 1u : 0u);
                }
            }
            mma_commit(&bar[0]);
        }
        ok = wait_bar(&bar[0], phase & 1u, fail);
        ++phase;
        tc_fence_after();
        if (group_sync_failed(1, kThreads, !ok)) {
            ok = false;
            break;
        }
        for (int bl = 0; bl < nb; ++bl) {
            const int n = b0 + bl;
            // slot n holds S_{n-1} (the running slice, in registers) and z_{n-1}.  The
            // slice's bytes are contiguous runs of both images: decode-image tile j (d
            // rows x 128 bytes) and, per e-tile c, feature rows 32 j .. 32 j + 31 (4 KB).
            // They are laid out in shared memory exactly as in global memory and stored
            // by bulk copies; K's space stages even blocks and V's space odd ones (both
            // idle until the next group), so a block's staging waits only for the bulk
            // stores of the block two before it.
            const size_t slot = ((size_t)s * n_blk + n) * Hkv + g;
            float *P = a.P + slot * hf, *PT = a.PT + slot * hf;
            uint8_t *stg = smem + ((bl & 1) ? Lp.off_v : Lp.off_k);
            if (tid == 0 && bl >= 2) bulk_wait_read_1();
            __syncthreads();
            const int e = tid;
            if (e < d) {
                // decode-image tile j: row e at e * 128 bytes, granules permuted by e mod 8
                float4 *row = reinterpret_cast<float4 *>(stg + (size_t)e * 128);
#pragma unroll
                for (int q = 0; q < 8; ++q)
                    row[q ^ (e & 7)] = make_float4(run[4 * q], run[4 * q + 1], run[4 * q + 2], run[4 * q + 3]);
                // feature-row piece of e-tile e / 32: row k (f = 32 j + k), column e mod 32
                float *pt = reinterpret_cast<float *>(stg + (size_t)d * 128 + (size_t)(e >> 5) * 4096) + (e & 3);
#pragma unroll
                for (int k = 0; k < 32; ++k) pt[k * 32 + ((((e & 31) >> 2) ^ (k & 7)) << 2)] = run[k];
            }
            if (tid < 32) {
                P[z_offset(32 * j + tid, d, F)] = zc;
                PT[z_offset(32 * j + tid, d, F)] = zc;
                zc += dz[bl * 32 + tid];
            }
            fence_proxy_async_smem();
            __syncthreads();
            if (tid == 0) {
                bulk_s2g(P + (size_t)j * 32 * d, stg, (uint32_t)d * 128);
                for (int c = 0; c < d / 32; ++c)
                    bulk_s2g(PT + (size_t)c * 64 * F + (size_t)(32 * j) * 32, stg + (size_t)d * 128 + (size_t)c * 4096,
                             4096);
                bulk_commit();
            }
            if (n == n_blk - 1) break;
            if (e < d) {
                float x[32];
                tmem_ld32(tmem + lane_off + kAcc + 32u * bl, x);
                tmem_wait_ld();
#pragma unroll
                for (int k = 0; k < 32; ++k) run[k] += x[k];
            }
        }
        // the next group's copies reuse K's and V's space
        if (tid == 0) bulk_wait_read_all();
        tc_fence_before();
        __syncthreads();
        tc_fence_after();
    }
    if (tid == 0) bulk_wait_all();
    if (!ok && tid == 0) raise_error(a.err, ERR_WAIT_TIMEOUT);
    tc_fence_before();
    __syncthreads();
    griddep_launch_dependents();
    if (warp == 0) tmem_dealloc(tmem, 256);
}

// ---------------------------------------------------------------------------
// k_slot_scan: per sequence, running sums over n_slots slots of nf floats.
// reverse = false: slot n += slot n-1 (inclusive, slot 0 unchanged);
// reverse = true : slot m = sum of slots n > m (exclusive, from the end; the
// backward's R_m = sum_{n > m} dR_n, the only use at present).
// ---------------------------------------------------------------------------
__global__ void k_slot_scan(float *buf0, float *buf1, int n_seq, int n_slots, size_t nf, bool reverse)
{
    float *buf = blockIdx.y == 0 ? buf0 : buf1;
    ptx::griddep_wait();
    if (!buf) return;
    const size_t n4 = nf / 4;
    const size_t i = (size_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (i >= n4 * (size_t)n_seq) return;
    const size_t s = i / n4, j = i % n4;
    float4 *p = reinterpret_cast<float4 *>(buf) + s * n4 * n_slots + j;
    if (!reverse) {
        float4 acc = p[0];
        float4 nxt = n_slots > 1 ? p[n4] : acc;
        for (int n = 1; n < n_slots; ++n) {
            const float4 v = nxt;
            if (n + 1 < n_slots) nxt = p[(size_t)(n + 1) * n4];
            acc.x += v.x; acc.y += v.y; acc.z += v.z; acc.w += v.w;
            p[(size_t)n * n4] = acc;
        }
    } else {
        float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
        float4 nxt = p[(size_t)(n_slots - 1) * n4];
        for (int n = n_slots - 1; n >= 0; --n) {
            const float4 v = nxt;
            if (n > 0) nxt = p[(size_t)(n - 1) * n4];
            p[(size_t)n * n4] = acc;
            acc.x += v.x; acc.y += v.y; acc.z += v.z; acc.w += v.w;
        }
    }
    ptx::griddep_launch_dependents();
}

// ---------------------------------------------------------------------------
// k_phi_grad<kQuery>: one (sequence s, block n, state head g).
// ---------------------------------------------------------------------------
template <bool kQuery>
__global__ void __launch_bounds__(kGradThreads, 1) k_phi_grad(const __grid_constant__ TrainArgs a, RowLayout Lr)
{
    using namespace ptx;
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = aligned_smem(smem_raw);
    const int tid = threadIdx.x, warp = tid >> 5;
    // two threads per Tensor Memory lane (row): lr = the lane, part = which half of each
    // row's columns the thread takes; warps w and w + 4 share lanes 32 (w & 3) ..
    const int lr = tid & 127, part = tid >> 7;
    const int d = a.d, F = a.F, B = a.B, Hkv = a.Hkv, Hq = a.Hq, G = Hq / Hkv;
    const int g = blockIdx.x % Hkv, n = (blockIdx.x / Hkv) % a.n_blk, s = blockIdx.x / (Hkv * a.n_blk);
    // Rows of the tile on Tensor Memory lanes: query side, lane r < G*B is token r / G,
    // head r % G of the group (the order the TMA box lands in); key side, lane r < B is
    // token r.  Lanes beyond are zero rows.
    const int rows = kQuery ? G * B : B;
    const size_t hf = head_floats(d, F);
    const size_t t0 = (size_t)s * a.L + (size_t)n * B;
    const size_t kv_row = (size_t)Hkv * d;
    // tile source: PT slot n (query side: S_{n-1}) or R slot n (key side: R_n)
    const float *src = (kQuery ? a.PT : a.R) + (((size_t)s * a.n_blk + n) * Hkv + g) * hf;

    uint64_t *bars = reinterpret_cast<uint64_t *>(smem + Lr.off_bar);
    uint64_t *mbar = bars;          // MMA groups complete
    uint64_t *full = bars + 1;      // [2] ring slot loaded
    uint64_t *empty = bars + 3;     // [2] ring slot consumed
    uint64_t *tbar = bars + 5;      // the phase-one operands have landed
    uint32_t *tmem_holder = reinterpret_cast<uint32_t *>(bars + 6);
    volatile int *fail = reinterpret_cast<volatile int *>(tmem_holder + 1);
    float *sRowDw = reinterpret_cast<float *>(tmem_holder + 2);  // [128] each query row's gate term
    float *sZ = reinterpret_cast<float *>(smem + Lr.off_z);     // z_{n-1} or r_n
    if (tid == 0) {
        for (int i = 0; i < 6; ++i) mbar_init(&bars[i], 1);
        *fail = 0;
        fence_mbar_init();
        prefetch_tensormap(&a.tmW);
        prefetch_tensormap(&a.tmK);
        if (kQuery) {
            prefetch_tensormap(&a.tmQ);
            prefetch_tensormap(&a.tmdO);
            prefetch_tensormap(&a.tmV);
        }
    }
    if (warp == 0) {
        tmem_alloc(tmem_holder, 512);
        tmem_relinquish();
    }
    // rows of the M = 128 operands beyond the tile stay zero (the TMA boxes fill rows < rows)
    for (int i = tid; i < (128 - rows) * (d / 8); i += kGradThreads) {
        const int r = rows + i / (d / 8), c8 = i % (d / 8);
        const uint32_t off = (uint32_t)(c8 >> 3) * (128 * 128) + swz(r, c8 & 7);
        *reinterpret_cast<uint4 *>(smem + Lr.off_q + off) = make_uint4(0, 0, 0, 0);
        if (kQuery) *reinterpret_cast<uint4 *>(smem + Lr.off_do + off) = make_uint4(0, 0, 0, 0);
    }
    __syncthreads();
    griddep_wait();

    // ring of S / R tiles: in the phase-one operands' space on the query side (free once
    // the first MMAs have run); the key side has phi's space to itself, so its first two
    // tiles are loaded right away, next to the operands
    const uint32_t ring_off = kQuery ? Lr.off_ring : Lr.off_phi;
    int loads_issued = 0;
    // phase one by TMA: [U | scores] = Q [W | K^T] and dO V^T (query side) or U = K W
    if (tid == 0) {
        const uint32_t qbytes = (uint32_t)(d / 64) * rows * 128, kvbytes = (uint32_t)(d / 64) * B * 128;
        const uint32_t wbytes = (uint32_t)(F / 64) * d * 128;
        mbar_arrive_expect_tx(tbar, kQuery ? 2 * qbytes + 2 * kvbytes + wbytes : kvbytes + wbytes);
        for (int p = 0; p < d / 64; ++p) {
            if (kQuery) {
                tma_load_3d(smem + Lr.off_q + p * 128 * 128, &a.tmQ, 64 * p, g * G, (int)t0, tbar);
                tma_load_3d(smem + Lr.off_do + p * 128 * 128, &a.tmdO, 64 * p, g * G, (int)t0, tbar);
                tma_load_3d(smem + Lr.off_k + p * B * 128, &a.tmK, 64 * p, g, (int)t0, tbar);
                tma_load_3d(smem + Lr.off_v + p * B * 128, &a.tmV, 64 * p, g, (int)t0, tbar);
            } else {
                tma_load_3d(smem + Lr.off_q + p * 128 * 128, &a.tmK, 64 * p, g, (int)t0, tbar);
            }
        }
        for (int p = 0; p < F / 64; ++p) tma_load_2d(smem + Lr.off_w + p * d * 128, &a.tmW, 64 * p, g * d, tbar);
        if (!kQuery)
            for (int c = 0; c < 2 && c < d / 32; ++c) {
                mbar_arrive_expect_tx(&full[c], Lr.ring_slot);
                bulk_g2s(smem + ring_off + c * Lr.ring_slot, src + (size_t)c * 64 * F, Lr.ring_slot, &full[c]);
                ++loads_issued;
            }
    }
    for (int f = tid; f < 2 * F; f += kGradThreads) sZ[f] = src[z_offset(f, d, F)];
    bool ok = wait_bar(tbar, 0, fail);
    fence_proxy_async_smem();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_holder;
    const uint32_t lane_off = (uint32_t)(warp & 3) * 32u << 16;
    const uint32_t tl = tmem + lane_off;
    const int NCHUNK = d / 32;
    const uint32_t ring_u = smem_u32(smem + ring_off);
    if (tid == 0) {
        const uint32_t q_u = smem_u32(smem + Lr.off_q), w_u = smem_u32(smem + Lr.off_w);
        const uint32_t idU = instr_desc(FMT_BF16, FMT_BF16, false, true, 128, F);
        for (int k = 0; k < d / 16; ++k) {
            const uint64_t aq = smem_desc(q_u + (k >> 2) * (128 * 128) + (k & 3) * 32, 16, 1024, SWZ_128B);
            mma_bf16_ss(tmem + kColU, aq, smem_desc(w_u + 2 * k * 1024, d * 128, 1024, SWZ_128B), idU, k > 0);
            if (kQuery) {
                const uint32_t k_u = smem_u32(smem + Lr.off_k), v_u = smem_u32(smem + Lr.off_v),
                               o_u = smem_u32(smem + Lr.off_do);
                const uint32_t idS = instr_desc(FMT_BF16, FMT_BF16, false, false, 128, B);
                const uint32_t kb = (uint32_t)(k >> 2) * B * 128 + (k & 3) * 32;
                mma_bf16_ss(tmem + kColS, aq, smem_desc(k_u + kb, 16, 1024, SWZ_128B), idS, k > 0);
                const uint64_t ao = smem_desc(o_u + (k >> 2) * (128 * 128) + (k & 3) * 32, 16, 1024, SWZ_128B);
                mma_bf16_ss(tmem + kColGv, ao, smem_desc(v_u + kb, 16, 1024, SWZ_128B), idS, k > 0);
            }
        }
        mma_commit(mbar);
    }
    ok = wait_bar(mbar, 0, fail) && ok;
    tc_fence_after();
    // query side: the phase-one operands are consumed, the first two tiles go into their space
    if (kQuery && tid == 0 && ok) {
        for (int c = 0; c < 2 && c < NCHUNK; ++c) {
            mbar_arrive_expect_tx(&full[c], Lr.ring_slot);
            bulk_g2s(smem + ring_off + c * Lr.ring_slot, src + (size_t)c * 64 * F, Lr.ring_slot, &full[c]);
            ++loads_issued;
        }
    }

    // ---- row statistics: the two parts of a row each take half of its columns and
    // exchange partial sums through shared memory (pair barrier of warps w, w + 4) ----
    const bool valid = lr < rows;
    const int hl = (kQuery && valid) ? lr % G : 0;                 // query head within the group
    const int tok = valid ? (kQuery ? lr / G : lr) : 0;            // token within the block
    const size_t q_row = (size_t)Hq * d;
    const uint32_t pair_bar = 2 + (uint32_t)(warp & 3);
    float *x1 = reinterpret_cast<float *>(smem + Lr.off_x);        // [2][128][8] statistics
    float *x2 = x1 + 2 * 128 * 8;                                  // [2][128]    lin_den
    float *x3 = x2 + 2 * 128;                                      // [2][128][4] pass-0 dots
    const int uj0 = part * (F / 64), uj1 = uj0 + F / 64;           // this part's 32-column chunks of U
    const float scale = rsqrtf((float)d);
    float w = 0.f;
    if (kQuery) {
        const float alpha = valid ? a.alpha[g * G + hl] : 0.f;
        w = 1.f / (1.f + expf(-alpha));
    }
    PhiStats st;
    {
        const PhiStats mine = phi_stats_chunks(tl + kColU, uj0, uj1);
        float *o = x1 + (part * 128 + lr) * 8;
        o[0] = mine.mp; o[1] = mine.sp; o[2] = mine.mn; o[3] = mine.sn;
        if (kQuery) {
            // scores: this part's 16-column chunks j = part, part + 2, ..: m, sum e^(s - m), sum e^(s - m) g.v
            float m = -INFINITY, l = 0.f, an = 0.f;
            for (int j = part; j < B / 16; j += 2) {
                float x[16];
                tmem_ld16(tl + kColS + 16 * j, x);
                tmem_wait_ld();
#pragma unroll
                for (int k = 0; k < 16; ++k) m = fmaxf(m, x[k] * scale);
            }
            for (int j = part; j < B / 16; j += 2) {
                float x[16], y[16];
                tmem_ld16(tl + kColS + 16 * j, x);
                tmem_ld16(tl + kColGv + 16 * j, y);
                tmem_wait_ld();
#pragma unroll
                for (int k = 0; k < 16; ++k) {
                    const float e = ex2((x[k] * scale - m) * kLog2e);
                    l += e;
                    an += e * y[k];
                }
            }
            o[4] = m; o[5] = l; o[6] = an;
        }
        named_bar(pair_bar, 64);
        const float *o0 = x1 + lr * 8, *o1 = x1 + (128 + lr) * 8;
        st = combine_stats(PhiStats{o0[0], o0[1], o0[2], o0[3]}, PhiStats{o1[0], o1[1], o1[2], o1[3]});
    }
    const float ip = 1.f / st.sp, in = 1.f / st.sn;
    // Query rows: 1/D and the merge terms A = g.sm_num / D, beta = sm_den / D,
    // lambda = lin_den / D; after S dN, Lambda = g.lin_num / D = phi(q).(S dN)
    // gives g.o = w A + Lambda and dw = lambda A - beta Lambda (= dN.sm_num + dD sm_den).
    float inv = 0.f, A = 0.f, beta = 0.f, lambda = 0.f;
    if (kQuery) {
        // phi(q) of this part's columns into its operand image; partial lin_den = phi(q) . z
        float ld = 0.f;
        {
            float x[32], yp[32], yn[32];
            for (int j = uj0; j < uj1; ++j) {
                tmem_ld32(tl + kColU + 32 * j, x);
                tmem_wait_ld();
#pragma unroll
                for (int k = 0; k < 32; ++k) {
                    yp[k] = valid ? ex2((x[k] - st.mp) * kLog2e) * ip : 0.f;
                    yn[k] = valid ? ex2((st.mn - x[k]) * kLog2e) * in : 0.f;
                    ld += yp[k] * sZ[32 * j + k] + yn[k] * sZ[F + 32 * j + k];
                }
                store_row32_bf16(smem + Lr.off_phi, 128 * 128, lr, 32 * j, yp);
                store_row32_bf16(smem + Lr.off_phi, 128 * 128, lr, F + 32 * j, yn);
            }
        }
        x2[part * 128 + lr] = ld;
        named_bar(pair_bar, 64);
        const float lin_den = x2[lr] + x2[128 + lr];
        // scores of the whole row: shift c, D' = w sum_j e^(s_j - c) + lin_den e^(-c) (D = e^c D')
        const float *o0 = x1 + lr * 8, *o1 = x1 + (128 + lr) * 8;
        const float m = fmaxf(o0[4], o1[4]);
        float c = m;
        if (lin_den > 0.f) c = w > 0.f ? fmaxf(m, logf(lin_den) - logf(w)) : logf(lin_den);
        const float e0 = ex2((o0[4] - c) * kLog2e), e1 = o1[4] == -INFINITY ? 0.f : ex2((o1[4] - c) * kLog2e);
        const float l = o0[5] * e0 + o1[5] * e1, an = o0[6] * e0 + o1[6] * e1;
        const float ec = ex2(-c * kLog2e);
        const float Dp = w * l + lin_den * ec;
        inv = valid ? ec / Dp : 0.f;              // 1 / D
        const float pw = valid ? 1.f / Dp : 0.f;  // e^(s_j - c) / D' = e^(s_j) / D
        beta = l * pw;
        lambda = lin_den * inv;
        A = an * pw;                              // sum_j (e^(s_j) / D) g.v_j
        // dN = g / D of this part's half of the columns: Tensor Memory (fp32, A operand
        // of S dN) and the operand image (bf16); its d/2 values are loaded at once
        const uint4 *grow = reinterpret_cast<const uint4 *>(a.dO + (t0 + tok) * q_row + (size_t)(g * G + hl) * d) +
                            part * (d / 16);
        uint4 graw[8];
#pragma unroll
        for (int i = 0; i < 8; ++i) graw[i] = (valid && i < d / 16) ? __ldg(grow + i) : make_uint4(0, 0, 0, 0);
#pragma unroll
        for (int cc = 0; cc < 2; ++cc) {
            if (cc < d / 64) {
                float gv[32];
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    const uint4 q4 = graw[4 * cc + i];
                    const uint32_t w4[4] = {q4.x, q4.y, q4.z, q4.w};
#pragma unroll
                    for (int jj = 0; jj < 4; ++jj) {
                        gv[8 * i + 2 * jj] = __uint_as_float(w4[jj] << 16) * inv;
                        gv[8 * i + 2 * jj + 1] = __uint_as_float(w4[jj] & 0xFFFF0000u) * inv;
                    }
                }
                const int col = part * (d / 2) + 32 * cc;
                tmem_st32(tl + kColY + col, gv);
                store_row32_bf16(smem + Lr.off_y, 128 * 128, lr, col, gv);
            }
        }
    } else {
        // V rows (fp32, this part's half of the columns) as the Tensor Memory A operand of
        // R v; r enters with coefficient 1
        const uint4 *vrow = reinterpret_cast<const uint4 *>(a.V + (t0 + tok) * kv_row + (size_t)g * d) + part * (d / 16);
        uint4 vraw[8];
#pragma unroll
        for (int i = 0; i < 8; ++i) vraw[i] = (valid && i < d / 16) ? __ldg(vrow + i) : make_uint4(0, 0, 0, 0);
#pragma unroll
        for (int cc = 0; cc < 2; ++cc) {
            if (cc < d / 64) {
                float vv[32];
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    const uint4 q4 = vraw[4 * cc + i];
                    const uint32_t w4[4] = {q4.x, q4.y, q4.z, q4.w};
#pragma unroll
                    for (int jj = 0; jj < 4; ++jj) {
                        vv[8 * i + 2 * jj] = __uint_as_float(w4[jj] << 16);
                        vv[8 * i + 2 * jj + 1] = __uint_as_float(w4[jj] & 0xFFFF0000u);
                    }
                }
                tmem_st32(tl + kColY + part * (d / 2) + 32 * cc, vv);
            }
        }
    }
    tmem_wait_st();
    fence_proxy_async_smem();
    tc_fence_before();
    const bool failed1 = group_sync_failed(1, kGradThreads, !ok);
    tc_fence_after();

    // ---- dphi = [S | z] [dN; dD] (query) or [R | r] [v; 1] (key): tiles of 32 e ----
    if (!failed1 && tid == 0) {
        const uint32_t idC = instr_desc(FMT_TF32, FMT_TF32, false, false, 128, 2 * F);
        for (int c = 0; c < NCHUNK && ok; ++c) {
            const int slot = c & 1;
            ok = wait_bar(&full[slot], (uint32_t)(c >> 1) & 1u, fail);
            if (!ok) break;
            tc_fence_after();
            const uint32_t s_u = ring_u + slot * Lr.ring_slot;
#pragma unroll
            for (int kk = 0; kk < 4; ++kk)
                mma_tf32_ts(tmem + kColG, tmem + kColY + 32 * c + 8 * kk, smem_desc(s_u + 32 * kk, 16, 1024, SWZ_128B),
                            idC, (c | kk) != 0);
            mma_commit(&empty[slot]);
            if (c + 2 < NCHUNK) {
                ok = wait_bar(&empty[slot], (uint32_t)(c >> 1) & 1u, fail);
                if (!ok) break;
                mbar_arrive_expect_tx(&full[slot], Lr.ring_slot);
                bulk_g2s(smem + ring_off + slot * Lr.ring_slot, src + (size_t)(c + 2) * 64 * F, Lr.ring_slot,
                         &full[slot]);
                ++loads_issued;
            }
        }
        mma_commit(mbar);
        if (!ok) atomicOr(const_cast<int *>(fail), 1);
    }
    if (!failed1) ok = wait_bar(mbar, 1, fail) && ok;
    tc_fence_before();
    // one decision for the whole CTA: the pair barriers below need both parts of a row
    const bool failedC = group_sync_failed(1, kGradThreads, failed1 || !ok || *fail);
    tc_fence_after();

    // ---- du = p+ (g+ - <g+, p+>) - p- (g- - <g-, p->) with g = G + zeta dD, where
    // G = S dN (query) or R v (key) and zeta = z_{n-1} (query) or r_m (key); each part
    // takes its half of the features ----
    if (!failedC) {
        float x[32], gp[32], gn[32];
        // pass 0: Lambda+- = <G+-, p+->, Z+- = <zeta+-, p+-> over this part's features
        float Lp = 0.f, Ln = 0.f, Zp = 0.f, Zn = 0.f;
        for (int j = uj0; j < uj1; ++j) {
            tmem_ld32(tl + kColU + 32 * j, x);
            tmem_ld32(tl + kColG + 32 * j, gp);
            tmem_ld32(tl + kColG + F + 32 * j, gn);
            tmem_wait_ld();
#pragma unroll
            for (int k = 0; k < 32; ++k) {
                const float pp = ex2((x[k] - st.mp) * kLog2e) * ip;
                const float pn = ex2((st.mn - x[k]) * kLog2e) * in;
                Lp += gp[k] * pp;
                Ln += gn[k] * pn;
                Zp += sZ[32 * j + k] * pp;
                Zn += sZ[F + 32 * j + k] * pn;
            }
        }
        {
            float *o = x3 + (part * 128 + lr) * 4;
            o[0] = Lp; o[1] = Ln; o[2] = Zp; o[3] = Zn;
            named_bar(pair_bar, 64);
            const float *o0 = x3 + lr * 4, *o1 = x3 + (128 + lr) * 4;
            Lp = o0[0] + o1[0];
            Ln = o0[1] + o1[1];
            Zp = o0[2] + o1[2];
            Zn = o0[3] + o1[3];
        }
        float dD = valid ? 1.f : 0.f;
        if (kQuery) {
            const float Lam = Lp + Ln;
            dD = -(w * A + Lam) * inv;   // -(g . o) / D
            if (part == 0) {
                sRowDw[lr] = valid ? lambda * A - beta * Lam : 0.f;
                // column d of [dN | dD | 0] (the rest of that 32-column group is never read)
                uint8_t *base = smem + Lr.off_y + (uint32_t)(d >> 6) * (128 * 128);
                uint4 v0;
                v0.x = pack_bf16x2(dD, 0.f);
                v0.y = v0.z = v0.w = 0u;
                *reinterpret_cast<uint4 *>(base + swz(lr, 0)) = v0;
                *reinterpret_cast<uint4 *>(base + swz(lr, 1)) = make_uint4(0, 0, 0, 0);
            }
        }
        const float dotp = Lp + dD * Zp, dotn = Ln + dD * Zn;
        // pass 1: du of this part's features
        for (int j = uj0; j < uj1; ++j) {
            tmem_ld32(tl + kColU + 32 * j, x);
            tmem_ld32(tl + kColG + 32 * j, gp);
            tmem_ld32(tl + kColG + F + 32 * j, gn);
            tmem_wait_ld();
            float du[32];
#pragma unroll
            for (int k = 0; k < 32; ++k) {
                const float pp = ex2((x[k] - st.mp) * kLog2e) * ip;
                const float pn = ex2((st.mn - x[k]) * kLog2e) * in;
                const float g1 = gp[k] + sZ[32 * j + k] * dD;
                const float g2 = gn[k] + sZ[F + 32 * j + k] * dD;
                du[k] = pp * (g1 - dotp) - pn * (g2 - dotn);
            }
            if (valid) {
                bf16 *out = kQuery ? a.dUq + ((t0 + tok) * Hq + (size_t)(g * G + hl)) * F
                                   : a.dUk + ((t0 + tok) * Hkv + (size_t)g) * F;
                uint4 *o4 = reinterpret_cast<uint4 *>(out + 32 * j);
#pragma unroll
                for (int q = 0; q < 4; ++q) {
                    uint4 v;
                    v.x = pack_bf16x2(du[8 * q + 0], du[8 * q + 1]);
                    v.y = pack_bf16x2(du[8 * q + 2], du[8 * q + 3]);
                    v.z = pack_bf16x2(du[8 * q + 4], du[8 * q + 5]);
                    v.w = pack_bf16x2(du[8 * q + 6], du[8 * q + 7]);
                    o4[q] = v;
                }
            }
        }
    }
    fence_proxy_async_smem();
    tc_fence_before();
    const bool failed2 = group_sync_failed(1, kGradThreads, failedC || !ok || *fail);
    tc_fence_after();

    // ---- query side: dR_n = phi(Q)^T [dN | dD], the gate, and the R slot ----
    if (kQuery && !failed2) {
        const int NY = d + 16, NYS = (NY + 31) & ~31, NM = 2 * F / 128;
        if (tid == 0) {
            const uint32_t p_u = smem_u32(smem + Lr.off_phi), y_u = smem_u32(smem + Lr.off_y);
            const uint32_t idDR = instr_desc(FMT_BF16, FMT_BF16, true, true, 128, NY);
            for (int i = 0; i < NM; ++i)
                for (int ks = 0; ks < 8; ++ks)   // all 128 lanes (rows of unused lanes are zero)
                    mma_bf16_ss(tmem + kColDR + (uint32_t)(i * NYS),
                                smem_desc(p_u + (uint32_t)(2 * i) * 128 * 128 + ks * 2048, 128 * 128, 1024, SWZ_128B),
                                smem_desc(y_u + ks * 2048, 128 * 128, 1024, SWZ_128B), idDR, ks > 0);
            mma_commit(mbar);
        }
        if (tid < G) {
            // rows t*G + h of head h, added in row order
            float sum = 0.f;
            for (int r = tid; r < 128; r += G) sum += sRowDw[r];
            const float al = a.alpha[g * G + tid];
            const float w = 1.f / (1.f + expf(-al));
            a.dap[(((size_t)s * a.n_blk + n) * Hkv + g) * G + tid] = sum * w * (1.f - w);
        }
        ok = wait_bar(mbar, 0, fail);
        tc_fence_after();
        // R's slot: per e-tile c the 2F feature rows (2F x 128 bytes, contiguous in global
        // memory) are staged in the space of phi(Q) and [dN | dD], which the dR MMAs have
        // consumed, laid out as in global memory, and written by bulk copies
        if (!group_sync_failed(1, kGradThreads, !ok)) {
            float *R = a.R + (((size_t)s * a.n_blk + n) * Hkv + g) * hf;
            const uint32_t tile_bytes = (uint32_t)2 * F * 128;
            for (int c = 0; c < d / 32; ++c) {
                // buffers: phi's space (two tiles), then [dN | dD]'s; tile 3 reuses the first
                uint8_t *buf = (c % 3 == 2) ? smem + Lr.off_y : smem + Lr.off_phi + (uint32_t)(c % 3) * tile_bytes;
                if (c == 3) {
                    if (tid == 0) bulk_wait_read_all();
                    __syncthreads();
                }
                // part p stages the features of M-block p (with one block, part 0 alone)
                for (int i = part; i < NM; i += 2) {
                    const int f = 128 * i + lr;
                    float x[32];
                    tmem_ld32(tl + kColDR + (uint32_t)(i * NYS + 32 * c), x);
                    tmem_wait_ld();
                    float4 *row = reinterpret_cast<float4 *>(buf + (size_t)f * 128);
#pragma unroll
                    for (int q = 0; q < 8; ++q)
                        row[q ^ (f & 7)] = make_float4(x[4 * q], x[4 * q + 1], x[4 * q + 2], x[4 * q + 3]);
                }
                fence_proxy_async_smem();
                __syncthreads();
                if (tid == 0) {
                    bulk_s2g(R + (size_t)c * 64 * F, buf, tile_bytes);
                    bulk_commit();
                }
            }
            for (int i = part; i < NM; i += 2) {
                float zz[16];
                tmem_ld16(tl + kColDR + (uint32_t)(i * NYS + d), zz);
                tmem_wait_ld();
                R[z_offset(128 * i + lr, d, F)] = zz[0];
            }
            if (tid == 0) bulk_wait_all();
        } else {
            ok = false;
        }
    }
    if (tid == 0 && (failed2 || !ok)) raise_error(a.err, ERR_WAIT_TIMEOUT);
    // no tile copy may still be landing when the CTA leaves
    if (tid == 0) {
        for (int c = 0; c < loads_issued; ++c) {
            // loads c and c+2 share slot c&1; the later one completes the later phase
            if (c + 2 >= loads_issued) mbar_wait(&full[c & 1], (uint32_t)(c >> 1) & 1u, kWaitNs);
        }
    }
    tc_fence_before();
    __syncthreads();
    griddep_launch_dependents();
    if (warp == 0) tmem_dealloc(tmem, 512);
}

// ---------------------------------------------------------------------------
// k_dw: dW_g += sum over a range of rows of x du^T.  The rows of group g come in
// 128-token chunks: G query tiles of 128 / G tokens x G heads (Q, dU_q) and one key
// tile of 128 tokens (K, dU_k), each a TMA box of 128 rows in (token, head) order
// for both operands (rows past the batch read zeros).  One thread runs a ring of
// three shared-memory stages (boxes in flight two steps ahead, each stage freed by
// the commit of its MMAs); the accumulator (d lanes x F columns) stays in Tensor
// Memory over the CTA's range of tiles.
// ---------------------------------------------------------------------------
struct DwArgs {
    // X and dU boxes of 128 rows in the same (token, head) order: Q / dU_q with box
    // {64, G, 128 / G}, K / dU_k with box {64, 1, 128}
    CUtensorMap tmXq, tmUq, tmXk, tmUk;
    float *dWp;   // [Hkv][ctas_per_group][d][F] partial sums, one per CTA
    unsigned *err;
    int n_chunks;      // 128-token chunks of the batch
    int G, d, F, tiles_per_cta, ctas_per_group;
};

__global__ void __launch_bounds__(kThreads, 1) k_dw(const __grid_constant__ DwArgs a)
{
    using namespace ptx;
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = aligned_smem(smem_raw);
    const int tid = threadIdx.x, warp = tid >> 5;
    const int d = a.d, F = a.F, G = a.G, K1 = G + 1;
    const int g = blockIdx.x / a.ctas_per_group, part = blockIdx.x % a.ctas_per_group;
    // tiles of group g: chunk c has G query tiles (kind < G) then the key tile (kind G)
    const int total = a.n_chunks * K1;
    const int t_begin = part * a.tiles_per_cta;
    const int n_tiles = max(0, min(a.tiles_per_cta, total - t_begin));
    const uint32_t xbytes = 2 * 128 * 128, ubytes = (uint32_t)(F / 64) * 128 * 128, stage = xbytes + ubytes;
    uint64_t *bars = reinterpret_cast<uint64_t *>(smem + kDwStages * stage);
    uint64_t *full = bars;                   // [kDwStages] a stage's boxes have landed
    uint64_t *empty = bars + kDwStages;      // [kDwStages] the MMAs of a stage are done
    uint64_t *done = bars + 2 * kDwStages;   // every MMA of the CTA is done
    uint32_t *tmem_holder = reinterpret_cast<uint32_t *>(bars + 2 * kDwStages + 1);
    volatile int *fail = reinterpret_cast<volatile int *>(tmem_holder + 1);
    if (tid == 0) {
        for (int i = 0; i < 2 * kDwStages + 1; ++i) mbar_init(&bars[i], 1);
        *fail = 0;
        fence_mbar_init();
        prefetch_tensormap(&a.tmXq);
        prefetch_tensormap(&a.tmUq);
        prefetch_tensormap(&a.tmXk);
        prefetch_tensormap(&a.tmUk);
    }
    if (warp == 0) {
        tmem_alloc(tmem_holder, 128);
        tmem_relinquish();
    }
    // for d = 64 the second half of the M = 128 operand X^T stays zero
    if (d == 64)
        for (int i = tid; i < kDwStages * 1024; i += kThreads) {
            const int st = i / 1024, k = i % 1024;
            reinterpret_cast<uint4 *>(smem + st * stage + 128 * 128)[k] = make_uint4(0, 0, 0, 0);
        }
    fence_proxy_async_smem();
    __syncthreads();
    griddep_wait();
    tc_fence_after();
    const uint32_t tmem = *tmem_holder;
    bool ok = true;
    int issued = 0;
    if (tid == 0 && n_tiles > 0) {
        const uint32_t idW = instr_desc(FMT_BF16, FMT_BF16, true, true, 128, F);
        // step k (tile t_begin + k) into stage k % kDwStages
        auto issue = [&](int k) {
            const int t = t_begin + k, c = t / K1, kind = t % K1;
            uint8_t *sx = smem + (k % kDwStages) * stage, *su = sx + xbytes;
            uint64_t *bar = &full[k % kDwStages];
            mbar_arrive_expect_tx(bar, (uint32_t)(d / 64) * 128 * 128 + ubytes);
            const bool q = kind < G;
            const int tok = c * 128 + (q ? kind * (128 / G) : 0);
            for (int p = 0; p < d / 64; ++p)
                tma_load_3d(sx + p * 128 * 128, q ? &a.tmXq : &a.tmXk, 64 * p, q ? g * G : g, tok, bar);
            for (int p = 0; p < F / 64; ++p)
                tma_load_3d(su + p * 128 * 128, q ? &a.tmUq : &a.tmUk, 64 * p, q ? g * G : g, tok, bar);
            ++issued;
        };
        for (int k = 0; k < kDwStages && k < n_tiles; ++k) issue(k);
        for (int k = 0; k < n_tiles && ok; ++k) {
            ok = wait_bar(&full[k % kDwStages], (uint32_t)(k / kDwStages) & 1u, fail);
            if (!ok) break;
            tc_fence_after();
            const uint32_t x_u = smem_u32(smem + (k % kDwStages) * stage), u_u = x_u + xbytes;
            for (int ks = 0; ks < 8; ++ks)
                mma_bf16_ss(tmem, smem_desc(x_u + ks * 2048, 128 * 128, 1024, SWZ_128B),
                            smem_desc(u_u + ks * 2048, 128 * 128, 1024, SWZ_128B), idW, (k | ks) != 0);
            mma_commit(&empty[k % kDwStages]);
            // refill the previous step's stage once its MMAs are done
            const int kn = k - 1 + kDwStages;
            if (k >= 1 && kn < n_tiles) {
                ok = wait_bar(&empty[(k - 1) % kDwStages], (uint32_t)((k - 1) / kDwStages) & 1u, fail);
                if (ok) issue(kn);
            }
        }
        mma_commit(done);
        if (!ok) atomicOr(const_cast<int *>(fail), 1);
    }
    if (n_tiles > 0) ok = wait_bar(done, 0, fail) && ok;
    tc_fence_after();
    const bool failed = group_sync_failed(1, kThreads, !ok);
    if (!failed && tid < d) {
        // this CTA's partial sum (zero without tiles); k_grad_reduce adds the parts in order
        float4 *dst = reinterpret_cast<float4 *>(a.dWp + (((size_t)g * a.ctas_per_group + part) * d + tid) * F);
        const uint32_t lane_off = (uint32_t)(warp & 3) * 32u << 16;
        float x[32];
        for (int j = 0; j < F / 32; ++j) {
            if (n_tiles > 0) {
                tmem_ld32(tmem + lane_off + 32 * j, x);
                tmem_wait_ld();
            } else {
#pragma unroll
                for (int k = 0; k < 32; ++k) x[k] = 0.f;
            }
#pragma unroll
            for (int k = 0; k < 8; ++k) dst[8 * j + k] = make_float4(x[4 * k], x[4 * k + 1], x[4 * k + 2], x[4 * k + 3]);
        }
    }
    if (tid == 0) {
        if (failed) raise_error(a.err, ERR_WAIT_TIMEOUT);
        // no box may still be landing when the CTA leaves
        for (int k = max(0, issued - kDwStages); k < issued; ++k)
            mbar_wait(&full[k % kDwStages], (uint32_t)(k / kDwStages) & 1u, kWaitNs);
    }
    tc_fence_before();
    __syncthreads();
    griddep_launch_dependents();
    if (warp == 0) tmem_dealloc(tmem, 128);
}

// ---------------------------------------------------------------------------
// k_grad_reduce: dW[g] = sum over parts p = 0, 1, ... of dWp[g][p] and
// d alpha[g G + h] = sum over blocks u = 0, 1, ... of dap[u][g][h], each in that order.
// ---------------------------------------------------------------------------
struct ReduceArgs {
    const float *dWp, *dap;
    float *dW, *dalpha;
    int Hkv, G, dF, parts, blocks;   // dF = d * F; blocks = n_seq * n_blk
};

__global__ void k_grad_reduce(const ReduceArgs a)
{
    using namespace ptx;
    griddep_wait();
    const long long i = (long long)blockIdx.x * blockDim.x + threadIdx.x;
    const long long nw = (long long)a.Hkv * a.dF;
    if (i < nw) {
        const int g = (int)(i / a.dF);
        const long long e = i % a.dF;
        const float *p = a.dWp + (long long)g * a.parts * a.dF + e;
        float sum = 0.f;
        for (int k = 0; k < a.parts; ++k) sum += p[(long long)k * a.dF];
        a.dW[i] = sum;
    } else if (i < nw + (long long)a.Hkv * a.G) {
        const int j = (int)(i - nw);   // g G + h
        float sum = 0.f;
        for (int u = 0; u < a.blocks; ++u) sum += a.dap[(long long)u * a.Hkv * a.G + j];
        a.dalpha[j] = sum;
    }
    griddep_launch_dependents();
}

// ---------------------------------------------------------------------------
// host side
// ---------------------------------------------------------------------------
__global__ void k_slot_ptrs(float *P, int n, size_t slot_floats, void **ptrs)
{
    const int i = blockIdx.x * blockDim.x + threadIdx.x;
    if (i < n) ptrs[i] = P + (size_t)i * slot_floats;
}

template <class Kern, class... Args>
cudaError_t launch_pdl(Kern k, dim3 grid, dim3 block, size_t smem, cudaStream_t st, Args... args)
{
    cudaLaunchConfig_t lc = {};
    lc.gridDim = grid;
    lc.blockDim = block;
    lc.dynamicSmemBytes = smem;
    lc.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    lc.attrs = attr;
    lc.numAttrs = 1;
    return cudaLaunchKernelEx(&lc, k, args...);
}

template <class Kern>
cudaError_t opt_in(Kern k, std::atomic<unsigned long long> &opted)
{
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
    const unsigned long long bit = 1ull << dev;
    if (!(opted.load(std::memory_order_acquire) & bit)) {
        const cudaError_t e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, kSmemLimit);
        if (e != cudaSuccess) return e;
        opted.fetch_or(bit, std::memory_order_release);
    }
    return cudaSuccess;
}

struct Workspace {
    float *P, *PT;
    bf16 *dUq, *dUk;
    void **ptrs;
    float *dWp, *dap;
    size_t bytes;
};

size_t align_up(size_t x) { return (x + 1023) & ~size_t(1023); }

Workspace carve(const hybrid_cfg &c, int n_seq, int L, void *base)
{
    const int d = c.head_dim, F = c.feat_dim, B = c.block_size, n_blk = L / B;
    const size_t slots = (size_t)n_seq * n_blk;
    const size_t buf = align_up(slots * slot_floats(c.n_kv_heads, d, F) * sizeof(float));
    const size_t uq = align_up((size_t)n_seq * L * c.n_q_heads * F * sizeof(bf16));
    const size_t uk = align_up((size_t)n_seq * L * c.n_kv_heads * F * sizeof(bf16));
    const size_t pt = align_up(slots * sizeof(void *));
    const size_t dwp = align_up((size_t)kMaxDwParts * d * F * sizeof(float));
    const size_t dap = align_up(slots * c.n_q_heads * sizeof(float));
    Workspace w{};
    uint8_t *p = static_cast<uint8_t *>(base);
    w.P = reinterpret_cast<float *>(p);
    w.PT = reinterpret_cast<float *>(p ? p + buf : nullptr);
    w.dUq = reinterpret_cast<bf16 *>(p ? p + 2 * buf : nullptr);
    w.dUk = reinterpret_cast<bf16 *>(p ? p + 2 * buf + uq : nullptr);
    w.ptrs = reinterpret_cast<void **>(p ? p + 2 * buf + uq + uk : nullptr);
    w.dWp = reinterpret_cast<float *>(p ? p + 2 * buf + uq + uk + pt : nullptr);
    w.dap = reinterpret_cast<float *>(p ? p + 2 * buf + uq + uk + pt + dwp : nullptr);
    w.bytes = 2 * buf + uq + uk + pt + dwp + dap;
    return w;
}

TrainArgs make_args(const hybrid_cfg &c, int n_seq, int L, const Workspace &w)
{
    TrainArgs a{};
    a.n_seq = n_seq;
    a.L = L;
    a.B = c.block_size;
    a.Hq = c.n_q_heads;
    a.Hkv = c.n_kv_heads;
    a.d = c.head_dim;
    a.F = c.feat_dim;
    a.n_blk = L / c.block_size;
    a.P = w.P;
    a.PT = w.PT;
    a.R = w.P;   // the backward reuses the decode image's space for R
    a.dUq = w.dUq;
    a.dUk = w.dUk;
    a.dap = w.dap;
    return a;
}

std::atomic<unsigned long long> g_opt_state, g_opt_q, g_opt_k, g_opt_dw;

// Tensor maps of [n*L][H][d] (box {64, bh, bt}) and of W [Hkv*d][F] (box {64, d}).
bool encode_rows(CUtensorMap *m, const void *base, long long n_tok, int H, int d, int bh, int bt)
{
    const cuuint64_t dims[3] = {(cuuint64_t)d, (cuuint64_t)H, (cuuint64_t)n_tok};
    const cuuint64_t strides[2] = {(cuuint64_t)d * 2, (cuuint64_t)H * d * 2};
    const cuuint32_t box[3] = {64, (cuuint32_t)bh, (cuuint32_t)bt};
    return encode_bf16(m, base, 3, dims, strides, box);
}
bool encode_w(CUtensorMap *m, const void *W, int Hkv, int d, int F)
{
    const cuuint64_t dims[2] = {(cuuint64_t)F, (cuuint64_t)Hkv * d};
    const cuuint64_t strides[1] = {(cuuint64_t)F * 2};
    const cuuint32_t box[2] = {64, (cuuint32_t)d};
    return encode_bf16(m, W, 2, dims, strides, box);
}

}  // namespace

bool train_supported(const hybrid_cfg &c, int seq_len)
{
    if (c.io_dtype != HYBRID_BF16) return false;
    if (c.head_dim != 64 && c.head_dim != 128) return false;
    if (c.feat_dim != 64 && c.feat_dim != 128) return false;
    const int B = c.block_size;
    if (B != 16 && B != 32 && B != 64) return false;
    if (c.n_kv_heads <= 0 || c.n_q_heads % c.n_kv_heads != 0) return false;
    if ((c.n_q_heads / c.n_kv_heads) * B > 128) return false;
    if (seq_len <= 0 || seq_len % B != 0) return false;
    return make_grad_layout(c.head_dim, c.feat_dim, B).bytes <= (uint32_t)kSmemLimit;
}

size_t train_workspace_bytes(const hybrid_cfg &c, int n_seq, int seq_len)
{
    return carve(c, n_seq, seq_len, nullptr).bytes;
}

void *const *train_state_ptrs(const hybrid_cfg &c, int n_seq, int seq_len, void *workspace)
{
    return carve(c, n_seq, seq_len, workspace).ptrs;
}

cudaError_t launch_train_states(const hybrid_cfg &c, const void *K, const void *V, const void *W, int n_seq,
                                int seq_len, void *workspace, unsigned *err, cudaStream_t st)
{
    const Workspace w = carve(c, n_seq, seq_len, workspace);
    TrainArgs a = make_args(c, n_seq, seq_len, w);
    a.K = static_cast<const bf16 *>(K);
    a.V = static_cast<const bf16 *>(V);
    a.W = static_cast<const bf16 *>(W);
    a.err = err;
    {
        const long long n_tok = (long long)n_seq * seq_len;
        const int GR = std::min(4, 128 / a.B) * a.B;   // rows of a prefix-sweep group (k_prefix_states' GB * B)
        if (!encode_rows(&a.tmKg, K, n_tok, a.Hkv, a.d, 1, GR) || !encode_rows(&a.tmVg, V, n_tok, a.Hkv, a.d, 1, GR) ||
            !encode_w(&a.tmW, W, a.Hkv, a.d, a.F))
            return cudaErrorInvalidValue;
    }
    const int slots = n_seq * a.n_blk;
    const size_t sf = slot_floats(a.Hkv, a.d, a.F);
    cudaError_t e = cudaSuccess;
    k_slot_ptrs<<<(slots + 255) / 256, 256, 0, st>>>(w.P, slots, sf, w.ptrs);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
    const PrefixLayout Lp = make_prefix_layout(a.d, a.F);
    if ((e = opt_in(k_prefix_states, g_opt_state)) != cudaSuccess) return e;
    return launch_pdl(k_prefix_states, dim3((unsigned)(n_seq * a.Hkv * (2 * a.F / 32))), dim3(kThreads), Lp.bytes,
                      st, a, Lp);
}

cudaError_t launch_train_backward(const hybrid_cfg &c, const void *Q, const void *K, const void *V, const void *W,
                                  const float *alpha, const void *dO, int n_seq, int seq_len,
                                  void *workspace, float *dW, float *dalpha, unsigned *err, cudaStream_t st)
{
    const Workspace w = carve(c, n_seq, seq_len, workspace);
    TrainArgs a = make_args(c, n_seq, seq_len, w);
    a.Q = static_cast<const bf16 *>(Q);
    a.K = static_cast<const bf16 *>(K);
    a.V = static_cast<const bf16 *>(V);
    a.W = static_cast<const bf16 *>(W);
    a.dO = static_cast<const bf16 *>(dO);
    a.alpha = alpha;
    a.dalpha = dalpha;
    a.err = err;
    {
        const long long n_tok = (long long)n_seq * seq_len;
        const int G = a.Hq / a.Hkv;
        if (!encode_rows(&a.tmQ, Q, n_tok, a.Hq, a.d, G, a.B) || !encode_rows(&a.tmdO, dO, n_tok, a.Hq, a.d, G, a.B) ||
            !encode_rows(&a.tmK, K, n_tok, a.Hkv, a.d, 1, a.B) || !encode_rows(&a.tmV, V, n_tok, a.Hkv, a.d, 1, a.B) ||
            !encode_w(&a.tmW, W, a.Hkv, a.d, a.F))
            return cudaErrorInvalidValue;
    }
    const int units = n_seq * a.n_blk * a.Hkv;
    const size_t sf = slot_floats(a.Hkv, a.d, a.F);
    cudaError_t e;
    const RowLayout Lg = make_grad_layout(a.d, a.F, a.B);
    if ((e = opt_in(k_phi_grad<true>, g_opt_q)) != cudaSuccess) return e;
    if ((e = opt_in(k_phi_grad<false>, g_opt_k)) != cudaSuccess) return e;
    if ((e = launch_pdl(k_phi_grad<true>, dim3((unsigned)units), dim3(kGradThreads), Lg.bytes, st, a, Lg)) !=
        cudaSuccess)
        return e;
    const size_t n4 = sf / 4 * (size_t)n_seq;
    if ((e = launch_pdl(k_slot_scan, dim3((unsigned)((n4 + 255) / 256), 1), dim3(256), 0, st, a.R,
                        static_cast<float *>(nullptr), n_seq, a.n_blk, sf, true)) != cudaSuccess)
        return e;
    if ((e = launch_pdl(k_phi_grad<false>, dim3((unsigned)units), dim3(kGradThreads), Lg.bytes, st, a, Lg)) !=
        cudaSuccess)
        return e;
    DwArgs b{};
    {
        const long long n_tok = (long long)n_seq * seq_len;
        const int G = a.Hq / a.Hkv;
        if (!encode_rows(&b.tmXq, Q, n_tok, a.Hq, a.d, G, 128 / G) ||
            !encode_rows(&b.tmUq, w.dUq, n_tok, a.Hq, a.F, G, 128 / G) ||
            !encode_rows(&b.tmXk, K, n_tok, a.Hkv, a.d, 1, 128) || !encode_rows(&b.tmUk, w.dUk, n_tok, a.Hkv, a.F, 1, 128))
            return cudaErrorInvalidValue;
        b.G = G;
        b.n_chunks = (int)((n_tok + 127) / 128);
    }
    b.dWp = w.dWp;
    b.err = err;
    b.d = a.d;
    b.F = a.F;
    const long long tiles = (long long)b.n_chunks * (b.G + 1);
    // one CTA per SM (three 64 KB stages each), the group's tiles split evenly
    int per_group = sm_count() / a.Hkv;
    if (per_group > kMaxDwParts / a.Hkv) per_group = kMaxDwParts / a.Hkv;
    if (per_group > tiles) per_group = (int)tiles;
    if (per_group < 1) per_group = 1;
    b.tiles_per_cta = (int)((tiles + per_group - 1) / per_group);
    b.ctas_per_group = per_group;
    const size_t dw_smem = kDwStages * ((size_t)2 * 128 * 128 + (size_t)(a.F / 64) * 128 * 128) + 1024 + 1024;
    if ((e = opt_in(k_dw, g_opt_dw)) != cudaSuccess) return e;
    if ((e = launch_pdl(k_dw, dim3((unsigned)(a.Hkv * per_group)), dim3(kThreads), dw_smem, st, b)) != cudaSuccess)
        return e;
    ReduceArgs rd{};
    rd.dWp = w.dWp;
    rd.dap = w.dap;
    rd.dW = dW;
    rd.dalpha = dalpha;
    rd.Hkv = a.Hkv;
    rd.G = a.Hq / a.Hkv;
    rd.dF = a.d * a.F;
    rd.parts = per_group;
    rd.blocks = a.n_seq * a.n_blk;
    const long long n_out = (long long)a.Hkv * rd.dF + a.Hq;
    return launch_pdl(k_grad_reduce, dim3((unsigned)((n_out + 255) / 256)), dim3(256), 0, st, rd);
}

}  // namespace hyb
