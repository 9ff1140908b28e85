// tc_pipeline.cuh -- pieces shared by the persistent warp-specialised tensor-core
// kernels (hybrid_fused.cu, hybrid_commit_red.cu): bounded mbarrier waits, group
// barriers that OR a failure flag, warp reductions, the transposed key tile, and
// the host-side tensor-map encoding.
#pragma once

#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <mutex>

#include "tc_ptx.cuh"

namespace hyb {
namespace pipe {

using bf16 = __nv_bfloat16;

constexpr uint64_t kWaitNs = 1000000000ull;   // every wait gives up after 1 s
constexpr float kLog2e = 1.4426950408889634f;

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

// Bounded wait that also gives up as soon as another role has failed (limit in
// nanoseconds of %globaltimer; kernels may take it from their arguments).
__device__ __forceinline__ bool wait_bar(uint64_t *bar, uint32_t parity, volatile int *fail,
                                         uint64_t limit_ns = kWaitNs)
{
    if (ptx::mbar_try_wait(bar, parity)) return true;
    const uint64_t t0 = ptx::global_timer_ns();
    while (true) {
        if (ptx::mbar_try_wait_sleep(bar, parity, 200000u)) return true;
        if (*fail) return false;
        if (ptx::global_timer_ns() - t0 > limit_ns) {
            atomicOr(const_cast<int *>(fail), 1);
            return false;
        }
    }
}

// Barrier over a group of warps that also ORs a failure flag across it, so
// that every thread of the group takes the same branch afterwards.
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

template <int kOp>
__device__ __forceinline__ float comb(float a, float b)
{
    return kOp == 0 ? a + b : (kOp == 1 ? fmaxf(a, b) : fminf(a, b));
}
// Reduce 32 per-lane values across the 32 lanes of a warp (op = add / max /
// min) by halving the set each step (31 shuffles); on return lane L holds the
// total of value index L.
template <int kOp>
__device__ __forceinline__ float warp_reduce32(float (&v)[32], int lane)
{
#pragma unroll
    for (int i = 0; i < 16; ++i) {
        const bool up = lane & 16;
        const float send = up ? v[i] : v[i + 16], keep = up ? v[i + 16] : v[i];
        v[i] = comb<kOp>(keep, __shfl_xor_sync(0xffffffffu, send, 16));
    }
#pragma unroll
    for (int i = 0; i < 8; ++i) {
        const bool up = lane & 8;
        const float send = up ? v[i] : v[i + 8], keep = up ? v[i + 8] : v[i];
        v[i] = comb<kOp>(keep, __shfl_xor_sync(0xffffffffu, send, 8));
    }
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const bool up = lane & 4;
        const float send = up ? v[i] : v[i + 4], keep = up ? v[i + 4] : v[i];
        v[i] = comb<kOp>(keep, __shfl_xor_sync(0xffffffffu, send, 4));
    }
#pragma unroll
    for (int i = 0; i < 2; ++i) {
        const bool up = lane & 2;
        const float send = up ? v[i] : v[i + 2], keep = up ? v[i + 2] : v[i];
        v[i] = comb<kOp>(keep, __shfl_xor_sync(0xffffffffu, send, 2));
    }
    const bool up = lane & 1;
    const float send = up ? v[0] : v[1], keep = up ? v[1] : v[0];
    return comb<kOp>(keep, __shfl_xor_sync(0xffffffffu, send, 1));
}

// Transposed key tile into a K^T atom (one warp): row e holds K[t][e] for the 32
// token slots t of a chunk, 128-byte swizzled like a W atom, so that it serves
// as an MN-major operand.  Token slot t is key row tok0 + t (row stride Hkv*d,
// head g) for t < nt and zero beyond.  Lane = (token pair, parity of the 8-dim
// group), so each store instruction writes 16 consecutive words of one row.
// The loads are issued first (kt_load, into registers, e.g. before the atom is
// free) and the stores later (kt_store).
struct KtRegs {
    uint4 r0[8], r1[8];
};
__device__ __forceinline__ void kt_load(const bf16 *K, size_t tok0, int nt, int Hkv, int g, int d, KtRegs &k,
                                        int lane)
{
    const int tp = lane & 15, eh = lane >> 4;
    const size_t tstride = (size_t)Hkv * d;
    const bool v0 = 2 * tp < nt, v1 = 2 * tp + 1 < nt;
    const uint4 *k0 = reinterpret_cast<const uint4 *>(K + (tok0 + 2 * tp) * tstride + (size_t)g * d);
    const uint4 *k1 = reinterpret_cast<const uint4 *>(reinterpret_cast<const bf16 *>(k0) + tstride);
#pragma unroll
    for (int i = 0; i < 8; ++i) {
        const int ec = eh + 2 * i;
        if (ec < d / 8) {
            k.r0[i] = v0 ? __ldg(k0 + ec) : make_uint4(0, 0, 0, 0);
            k.r1[i] = v1 ? __ldg(k1 + ec) : make_uint4(0, 0, 0, 0);
        }
    }
}
__device__ __forceinline__ void kt_store(const KtRegs &k, int d, uint8_t *kt_in, int lane)
{
    // the base is made opaque so the 64 store addresses, which depend only on
    // the lane, are formed at the stores rather than kept live across a caller's loop
    uint8_t *kt = kt_in;
    asm volatile("" : "+l"(kt));
    const int tp = lane & 15, eh = lane >> 4;
#pragma unroll
    for (int i = 0; i < 8; ++i) {
        const int ec = eh + 2 * i;
        if (ec < d / 8) {
            const uint32_t w0[4] = {k.r0[i].x, k.r0[i].y, k.r0[i].z, k.r0[i].w};
            const uint32_t w1[4] = {k.r1[i].x, k.r1[i].y, k.r1[i].z, k.r1[i].w};
#pragma unroll
            for (int j = 0; j < 8; ++j) {
                const uint32_t lo = (w0[j >> 1] >> (16 * (j & 1))) & 0xFFFFu;
                const uint32_t hi = (w1[j >> 1] >> (16 * (j & 1))) & 0xFFFFu;
                const int e = 8 * ec + j;
                *reinterpret_cast<uint32_t *>(kt + e * 128 + ((((tp >> 2) ^ (e & 7))) << 4) + (tp & 3) * 4) =
                    lo | (hi << 16);
            }
        }
    }
}

// cuTensorMapEncodeTiled from the driver, looked up once through the runtime.
inline PFN_cuTensorMapEncodeTiled_v12000 encode_fn()
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
inline bool encode_bf16(CUtensorMap *m, const void *base, int rank, const cuuint64_t *dims, const cuuint64_t *strides,
                 const cuuint32_t *box)
{
    PFN_cuTensorMapEncodeTiled_v12000 fn = encode_fn();
    if (!fn) return false;
    const cuuint32_t es[5] = {1, 1, 1, 1, 1};
    return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, (cuuint32_t)rank, const_cast<void *>(base), dims, strides, box, es,
              CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_128B,
              CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

inline int sm_count()
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

}  // namespace pipe
}  // namespace hyb
