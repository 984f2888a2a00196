// gemm_tc.cu -- the tensor-core path for batches of tokens (batched decode and
// prefill) on sm_103a: tcgen05.mma with TMEM accumulators, operands staged by
// TMA (cp.async.bulk.tensor, 128-byte swizzle) through an mbarrier ring.
//
// For a batch of M tokens with per-token threshold t_m (0 for tokens routed to
// the base path, Sec. 3.2), the thresholded gated MLP (Sec. 2, Eqs. 1-5) is
//   G = X W_gate,  U = X W_up           (one kernel, two accumulators)
//   h_mj = |SiLU(g_mj)| >= t_m ? SiLU(g_mj) * u_mj : 0        (its epilogue)
//   Y = h W_down                        (second kernel)
// X is bf16: the caller's bf16 activations, or fp32 activations (optionally
// RMS-normalised) split into a bf16 high part and a bf16 low part, both fed to
// the same accumulator, so that the gate values keep ~fp32 accuracy.  h is
// kept in bf16 between the two GEMMs.
//
// Kernel layout (one output tile per CTA, 192 threads): warp 0 lane 0 issues
// the TMA loads, warp 1 owns the TMEM allocation and lane 0 issues the MMAs,
// warps 2-5 run the epilogue (warp w reads TMEM lanes 32 (w mod 4) ..).
// Every wait is bounded in time and sets the status word when it gives up.
#include <cuda.h>
#include <cuda_bf16.h>
#include <cudaTypedefs.h>

#include <atomic>
#include <cmath>
#include <mutex>

#include "common.cuh"
#include "internal.h"

namespace sats {
namespace tc {
namespace {

constexpr int BM = 128;              // tokens per tile (MMA M)
constexpr int BK = 64;               // K per stage: one 128-byte swizzle row of bf16
constexpr int kThreads = 192;
constexpr int kSmemBudget = 196608;  // stage ring
constexpr uint32_t kTmemCols = 256;

// ---------------------------------------------------------------------- device helpers
// Shared-memory matrix descriptor of a K-major bf16 tile written by TMA with
// 128-byte swizzle: rows of 128 bytes, 8-row atoms 1024 bytes apart.
__device__ __forceinline__ uint64_t smem_desc(uint32_t saddr)
{
    uint64_t d = 0;
    d |= (uint64_t)((saddr & 0x3FFFFu) >> 4);     // start address
    d |= (uint64_t)(16u >> 4) << 16;               // leading byte offset (unused for swizzled K-major)
    d |= (uint64_t)(1024u >> 4) << 32;             // stride byte offset: one 8-row atom
    d |= (uint64_t)1 << 46;                        // descriptor version of this architecture
    d |= (uint64_t)2 << 61;                        // 128-byte swizzle
    return d;
}

// Instruction descriptor of kind::f16: bf16 A and B (K-major), fp32 D, M x N.
__host__ __device__ constexpr uint32_t instr_desc(int M, int N)
{
    return (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(N >> 3) << 17) | ((uint32_t)(M >> 4) << 24);
}

__device__ __forceinline__ void mma_bf16(uint32_t d_tmem, uint64_t a, uint64_t b, uint32_t idesc, uint32_t acc)
{
    asm volatile(
        "{\n\t.reg .pred p;\n\tsetp.ne.b32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}"
        ::"r"(d_tmem), "l"(a), "l"(b), "r"(idesc), "r"(acc)
        : "memory");
}

// The mbarrier receives one arrival when all previously issued MMAs are done.
__device__ __forceinline__ void mma_commit(uint64_t *bar)
{
    asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];"
                 ::"r"(smem_addr(bar)) : "memory");
}

__device__ __forceinline__ void tc_fence_after() { asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void tc_fence_before() { asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory"); }

__device__ __forceinline__ void tmem_alloc(uint32_t *slot, uint32_t ncols)
{
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_addr(slot)), "r"(ncols)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
}

__device__ __forceinline__ void tmem_dealloc(uint32_t taddr, uint32_t ncols)
{
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols) : "memory");
}

// 16 consecutive fp32 columns of this warp's 32 TMEM lanes (one row per thread).
__device__ __forceinline__ void tmem_ld16(uint32_t taddr, float (&v)[16])
{
    uint32_t r[16];
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15}, [%16];"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
          "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
        : "r"(taddr)
        : "memory");
#pragma unroll
    for (int i = 0; i < 16; ++i) v[i] = __uint_as_float(r[i]);
}

__device__ __forceinline__ void tmem_ld_wait() { asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory"); }

// Error path only (a role gave up waiting): before the CTA releases its TMEM
// and exits, wait -- again bounded -- for the tile loads still in flight
// (stages issued but never consumed) and for the MMAs already issued.
__device__ void drain_after_abort(uint64_t *full, int stages, int issued, int consumed, uint64_t *acc_full)
{
    int never = 0;
    for (int k = consumed; k < issued; ++k)
        mbar_wait(&full[k % stages], (uint32_t)((k / stages) & 1), &never);
    mbar_wait(acc_full, 0u, &never);
}

// One 2D TMA tile load: inner coordinate c0 (elements, a multiple of 64), row c1.
__device__ __forceinline__ void tma_load(void *dst, const CUtensorMap *map, int c0, int c1, uint64_t *bar)
{
    asm volatile(
        "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3}], [%4];"
        ::"r"(smem_addr(dst)), "l"(map), "r"(c0), "r"(c1), "r"(smem_addr(bar))
        : "memory");
}

__device__ __forceinline__ uint16_t bf16_bits(float v)
{
    const __nv_bfloat16 h = __float2bfloat16_rn(v);
    return *reinterpret_cast<const uint16_t *>(&h);
}

__device__ __forceinline__ uint8_t *align1024(uint8_t *p)
{
    return reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(p) + 1023) & ~(uintptr_t)1023);
}

// ---------------------------------------------------------------------- activations
// Row m of X (fp32, optionally RMS-normalised with gain w) -> bf16 hi + lo.
__global__ void __launch_bounds__(256) split_kernel(const float *__restrict__ x, int H, const float *__restrict__ w,
                                                    float eps, uint16_t *__restrict__ hi, uint16_t *__restrict__ lo)
{
    const int m = blockIdx.x;
    const float *xr = x + (size_t)m * H;
    __shared__ float red[8];
    float inv = 1.0f;
    if (w) {
        float s = 0.f;
        for (int i = threadIdx.x; i < H; i += 256) s = fmaf(xr[i], xr[i], s);
        s = warp_sum(s);
        if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = s;
        __syncthreads();
        float tot = 0.f;
        for (int i = 0; i < 8; ++i) tot += red[i];
        inv = 1.0f / sqrtf(tot / (float)H + eps);
    }
    for (int i = threadIdx.x; i < H; i += 256) {
        const float v = w ? xr[i] * inv * w[i] : xr[i];
        const uint16_t h = bf16_bits(v);
        const float hv = __uint_as_float((uint32_t)h << 16);
        hi[(size_t)m * H + i] = h;
        lo[(size_t)m * H + i] = bf16_bits(v - hv);
    }
}

// ---------------------------------------------------------------------- gate + up GEMM
struct GuParams {
    int M, N, H;
    float t_l;                    // threshold of sparse-path tokens
    const uint8_t *dense_flags;   // [M] (1 = base path, threshold 0) or nullptr
    uint16_t *hact;               // [M][ldh] bf16
    int ldh;
    uint8_t *keep;                // [M][keep_stride] or nullptr
    int keep_stride;              // a multiple of 16
    uint8_t *keep_trace;          // [M][N] or nullptr
    int *ctl;
};

template <int BN, bool SPLIT>
struct GuShape {
    static constexpr int kA = BM * 128, kB = BN * 128;
    static constexpr int kStage = kA * (SPLIT ? 2 : 1) + 2 * kB;
    static constexpr int kStages = (kSmemBudget / kStage) > 6 ? 6 : (kSmemBudget / kStage);
    static constexpr size_t kSmem = (size_t)kStages * kStage + 1024 + 256;
    static_assert(kStage % 1024 == 0, "stages keep the 1024-byte alignment of the swizzle atoms");
    static_assert(2 * BN <= (int)kTmemCols, "gate and up accumulators fit the TMEM allocation");
};

// One 128-token x BN-neuron tile of G = X W_gate and U = X W_up (K = H), then
// h = CATS(SiLU(G)) * U in the epilogue.  Grid: (ceil(N / BN), ceil(M / 128)).
template <int BN, bool SPLIT>
__global__ void __launch_bounds__(kThreads, 1)
    gu_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmA2,
              const __grid_constant__ CUtensorMap tmG, const __grid_constant__ CUtensorMap tmU, const GuParams p)
{
    using Sh = GuShape<BN, SPLIT>;
    extern __shared__ uint8_t smem_raw[];
    uint8_t *ring = align1024(smem_raw);
    uint64_t *full = reinterpret_cast<uint64_t *>(ring + (size_t)Sh::kStages * Sh::kStage);
    uint64_t *empty = full + Sh::kStages;
    uint64_t *acc_full = empty + Sh::kStages;
    uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(acc_full + 1);
    __shared__ int abort_flag, issued_s, consumed_s;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int m0 = blockIdx.y * BM, n0 = blockIdx.x * BN;
    const int KB = (p.H + BK - 1) / BK;

    if (threadIdx.x == 0) {
        for (int s = 0; s < Sh::kStages; ++s) {
            mbar_init(&full[s], 1);
            mbar_init(&empty[s], 1);
        }
        mbar_init(acc_full, 1);
        abort_flag = 0;
        issued_s = 0;
        consumed_s = 0;
        mbar_init_fence();
    }
    if (warp == 1) tmem_alloc(tmem_slot, kTmemCols);
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_slot;

    if (warp == 0 && lane == 0) {
        // TMA producer
        int kb = 0;
        for (uint32_t s = 0, ph = 0; kb < KB; ++kb) {
            if (!mbar_wait(&empty[s], ph ^ 1u, &abort_flag)) {
                abort_flag = 1;
                atomicOr(p.ctl + kCtlStatus, kStatusTimeout);
                break;
            }
            uint8_t *st = ring + (size_t)s * Sh::kStage;
            uint8_t *g = st + Sh::kA * (SPLIT ? 2 : 1);
            mbar_arrive_expect_tx(&full[s], (uint32_t)Sh::kStage);
            tma_load(st, &tmA, kb * BK, m0, &full[s]);
            if (SPLIT) tma_load(st + Sh::kA, &tmA2, kb * BK, m0, &full[s]);
            tma_load(g, &tmG, kb * BK, n0, &full[s]);
            tma_load(g + Sh::kB, &tmU, kb * BK, n0, &full[s]);
            if (++s == (uint32_t)Sh::kStages) { s = 0; ph ^= 1u; }
        }
        issued_s = kb;
    } else if (warp == 1 && lane == 0) {
        // MMA issuer: gate accumulator at TMEM column 0, up accumulator at column BN
        constexpr uint32_t idesc = instr_desc(BM, BN);
        int kb = 0;
        for (uint32_t s = 0, ph = 0; kb < KB; ++kb) {
            if (!mbar_wait(&full[s], ph, &abort_flag)) {
                abort_flag = 1;
                atomicOr(p.ctl + kCtlStatus, kStatusTimeout);
                break;
            }
            tc_fence_after();
            const uint32_t st = smem_addr(ring + (size_t)s * Sh::kStage);
            const uint32_t ga = st + Sh::kA * (SPLIT ? 2 : 1);
#pragma unroll
            for (int kk = 0; kk < BK / 16; ++kk) {
                const uint32_t acc = (kb | kk) ? 1u : 0u;
                const uint64_t a = smem_desc(st + kk * 32);
                const uint64_t g = smem_desc(ga + kk * 32);
                const uint64_t u = smem_desc(ga + Sh::kB + kk * 32);
                mma_bf16(tmem, a, g, idesc, acc);
                mma_bf16(tmem + BN, a, u, idesc, acc);
                if (SPLIT) {
                    const uint64_t a2 = smem_desc(st + Sh::kA + kk * 32);
                    mma_bf16(tmem, a2, g, idesc, 1u);
                    mma_bf16(tmem + BN, a2, u, idesc, 1u);
                }
            }
            mma_commit(&empty[s]);   // the stage is free once these MMAs have read it
            if (++s == (uint32_t)Sh::kStages) { s = 0; ph ^= 1u; }
        }
        consumed_s = kb;
        mma_commit(acc_full);
    } else if (warp >= 2) {
        // epilogue: thread = one token row of the tile
        const bool ok = mbar_wait(acc_full, 0u, &abort_flag);
        tc_fence_after();
        const int lb = 32 * (warp & 3);
        const int m = m0 + lb + lane;
        const bool row_ok = ok && m < p.M;
        float thr = INFINITY;
        if (row_ok) thr = (p.dense_flags && p.dense_flags[m]) ? 0.f : p.t_l;
        for (int c0 = 0; c0 < BN; c0 += 16) {
            float g[16], u[16];
            tmem_ld16(tmem + ((uint32_t)lb << 16) + (uint32_t)c0, g);
            tmem_ld16(tmem + ((uint32_t)lb << 16) + (uint32_t)(BN + c0), u);
            tmem_ld_wait();
            const int n = n0 + c0;
            if (!row_ok || n >= p.N) continue;
            uint32_t hw[8], kw[4] = {0u, 0u, 0u, 0u};
#pragma unroll
            for (int e = 0; e < 16; e += 2) {
                const float a0 = g[e] / (1.0f + expf(-g[e]));            // SiLU, Eq. 2
                const float a1 = g[e + 1] / (1.0f + expf(-g[e + 1]));
                const bool k0 = fabsf(a0) >= thr, k1 = fabsf(a1) >= thr;  // Eqs. 4-5
                hw[e / 2] = (uint32_t)bf16_bits(k0 ? a0 * u[e] : 0.f) |
                            ((uint32_t)bf16_bits(k1 ? a1 * u[e + 1] : 0.f) << 16);
                kw[e / 4] |=((k0 ? 1u : 0u) << (8 * (e % 4))) | ((k1 ? 1u : 0u) << (8 * (e % 4) + 8));
            }
            uint16_t *hrow = p.hact + (size_t)m * p.ldh + n;
            uint8_t *krow = p.keep ? p.keep + (size_t)m * p.keep_stride + n : nullptr;
            if (n + 16 <= p.N) {
                reinterpret_cast<uint4 *>(hrow)[0] = make_uint4(hw[0], hw[1], hw[2], hw[3]);
                reinterpret_cast<uint4 *>(hrow)[1] = make_uint4(hw[4], hw[5], hw[6], hw[7]);
                if (krow) *reinterpret_cast<uint4 *>(krow) = make_uint4(kw[0], kw[1], kw[2], kw[3]);
            } else {
#pragma unroll
                for (int e = 0; e < 16; ++e) {
                    if (n + e < p.N) {
                        hrow[e] = (uint16_t)(hw[e / 2] >> (16 * (e & 1)));
                        if (krow) krow[e] = (uint8_t)(kw[e / 4] >> (8 * (e & 3)));
                    }
                }
            }
            if (p.keep_trace) {
                uint8_t *trow = p.keep_trace + (size_t)m * p.N + n;
#pragma unroll
                for (int e = 0; e < 16; ++e)
                    if (n + e < p.N) trow[e] = (uint8_t)(kw[e / 4] >> (8 * (e & 3)));
            }
        }
        tc_fence_before();
    }
    __syncthreads();
    if (abort_flag && threadIdx.x == 0) drain_after_abort(full, Sh::kStages, issued_s, consumed_s, acc_full);
    __syncthreads();
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc(tmem, kTmemCols);
    }
}

// ---------------------------------------------------------------------- down GEMM
struct DownParams {
    int M, N, H;          // tokens, K (neurons), output columns
    int kb_per_split;     // K blocks of 64 neurons per split (blockIdx.z)
    int atomic_out;       // 1: add into out with L2 reductions (split K); 0: one writer per element
    int add_residual;     // with atomic_out == 0: out += tile, else out = tile
    float *out;           // [M][H] fp32
    int *ctl;
};

template <int BN>
struct DownShape {
    static constexpr int kA = BM * 128, kB = BN * 128;
    static constexpr int kStage = kA + kB;
    static constexpr int kStages = (kSmemBudget / kStage) > 6 ? 6 : (kSmemBudget / kStage);
    static constexpr size_t kSmem = (size_t)kStages * kStage + 1024 + 256;
    static_assert(kStage % 1024 == 0, "stages keep the 1024-byte alignment of the swizzle atoms");
    static_assert(BN <= (int)kTmemCols, "the accumulator fits the TMEM allocation");
};

// One 128-token x BN-column tile of Y = h W_down over one split of the K range.
// Grid: (ceil(H / BN), ceil(M / 128), splits).
template <int BN>
__global__ void __launch_bounds__(kThreads, 1)
    down_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB, const DownParams p)
{
    using Sh = DownShape<BN>;
    extern __shared__ uint8_t smem_raw[];
    uint8_t *ring = align1024(smem_raw);
    uint64_t *full = reinterpret_cast<uint64_t *>(ring + (size_t)Sh::kStages * Sh::kStage);
    uint64_t *empty = full + Sh::kStages;
    uint64_t *acc_full = empty + Sh::kStages;
    uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(acc_full + 1);
    __shared__ int abort_flag, issued_s, consumed_s;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int m0 = blockIdx.y * BM, h0 = blockIdx.x * BN;
    const int KB = (p.N + BK - 1) / BK;
    const int kb0 = blockIdx.z * p.kb_per_split;
    const int kb1 = min(KB, kb0 + p.kb_per_split);

    if (threadIdx.x == 0) {
        for (int s = 0; s < Sh::kStages; ++s) {
            mbar_init(&full[s], 1);
            mbar_init(&empty[s], 1);
        }
        mbar_init(acc_full, 1);
        abort_flag = 0;
        issued_s = 0;
        consumed_s = 0;
        mbar_init_fence();
    }
    if (warp == 1) tmem_alloc(tmem_slot, kTmemCols);
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_slot;

    if (warp == 0 && lane == 0) {
        int i = 0;
        for (uint32_t s = 0, ph = 0; kb0 + i < kb1; ++i) {
            if (!mbar_wait(&empty[s], ph ^ 1u, &abort_flag)) {
                abort_flag = 1;
                atomicOr(p.ctl + kCtlStatus, kStatusTimeout);
                break;
            }
            uint8_t *st = ring + (size_t)s * Sh::kStage;
            mbar_arrive_expect_tx(&full[s], (uint32_t)Sh::kStage);
            tma_load(st, &tmA, (kb0 + i) * BK, m0, &full[s]);
            tma_load(st + Sh::kA, &tmB, (kb0 + i) * BK, h0, &full[s]);
            if (++s == (uint32_t)Sh::kStages) { s = 0; ph ^= 1u; }
        }
        issued_s = i;
    } else if (warp == 1 && lane == 0) {
        constexpr uint32_t idesc = instr_desc(BM, BN);
        int i = 0;
        for (uint32_t s = 0, ph = 0; kb0 + i < kb1; ++i) {
            if (!mbar_wait(&full[s], ph, &abort_flag)) {
                abort_flag = 1;
                atomicOr(p.ctl + kCtlStatus, kStatusTimeout);
                break;
            }
            tc_fence_after();
            const uint32_t st = smem_addr(ring + (size_t)s * Sh::kStage);
#pragma unroll
            for (int kk = 0; kk < BK / 16; ++kk)
                mma_bf16(tmem, smem_desc(st + kk * 32), smem_desc(st + Sh::kA + kk * 32), idesc,
                         (i | kk) ? 1u : 0u);
            mma_commit(&empty[s]);
            if (++s == (uint32_t)Sh::kStages) { s = 0; ph ^= 1u; }
        }
        consumed_s = i;
        mma_commit(acc_full);
    } else if (warp >= 2) {
        const bool ok = mbar_wait(acc_full, 0u, &abort_flag) && kb1 > kb0;
        tc_fence_after();
        const int lb = 32 * (warp & 3);
        const int m = m0 + lb + lane;
        const bool row_ok = ok && m < p.M;
        for (int c0 = 0; c0 < BN; c0 += 16) {
            float v[16];
            tmem_ld16(tmem + ((uint32_t)lb << 16) + (uint32_t)c0, v);
            tmem_ld_wait();
            const int h = h0 + c0;
            if (!row_ok || h >= p.H) continue;
            float *dst = p.out + (size_t)m * p.H + h;
            const bool vec = h + 16 <= p.H;   // H is a multiple of 8: dst is 16-byte aligned
            if (p.atomic_out) {
                if (vec) {
#pragma unroll
                    for (int q = 0; q < 4; ++q) red_add_v4(dst + 4 * q, v[4 * q], v[4 * q + 1], v[4 * q + 2], v[4 * q + 3]);
                } else {
#pragma unroll
                    for (int e = 0; e < 16; ++e)
                        if (h + e < p.H) atomicAdd(dst + e, v[e]);
                }
            } else if (vec) {
                float4 *d4 = reinterpret_cast<float4 *>(dst);
#pragma unroll
                for (int q = 0; q < 4; ++q) {
                    float4 o = p.add_residual ? d4[q] : make_float4(0.f, 0.f, 0.f, 0.f);
                    o.x += v[4 * q];
                    o.y += v[4 * q + 1];
                    o.z += v[4 * q + 2];
                    o.w += v[4 * q + 3];
                    d4[q] = o;
                }
            } else {
#pragma unroll
                for (int e = 0; e < 16; ++e)
                    if (h + e < p.H) dst[e] = p.add_residual ? dst[e] + v[e] : v[e];
            }
        }
        tc_fence_before();
    }
    __syncthreads();
    if (abort_flag && threadIdx.x == 0) drain_after_abort(full, Sh::kStages, issued_s, consumed_s, acc_full);
    __syncthreads();
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc(tmem, kTmemCols);
    }
}

// ---------------------------------------------------------------------- kept lists
// Token m's ascending kept list from its keep bytes (one CTA per token).
__global__ void __launch_bounds__(512) keep_list_kernel(const uint8_t *__restrict__ keep, int stride, int N,
                                                        int32_t *__restrict__ idx, int32_t *__restrict__ cnt)
{
    const int m = blockIdx.x;
    const uint8_t *k = keep + (size_t)m * stride;
    __shared__ int warp_sums[16];
    __shared__ int base_s;
    if (threadIdx.x == 0) base_s = 0;
    __syncthreads();
    for (int c0 = 0; c0 < N; c0 += 512) {
        const int n = c0 + threadIdx.x;
        const int f = (n < N && k[n]) ? 1 : 0;
        const uint32_t bal = __ballot_sync(0xffffffffu, f);
        const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
        if (lane == 0) warp_sums[w] = __popc(bal);
        __syncthreads();
        int before = base_s;
        for (int i = 0; i < w; ++i) before += warp_sums[i];
        if (f) idx[(size_t)m * N + before + __popc(bal & ((1u << lane) - 1u))] = n;
        __syncthreads();
        if (threadIdx.x == 0) {
            int tot = 0;
            for (int i = 0; i < 16; ++i) tot += warp_sums[i];
            base_s += tot;
        }
        __syncthreads();
    }
    if (threadIdx.x == 0 && cnt) cnt[m] = base_s;
}

// ---------------------------------------------------------------------- host
PFN_cuTensorMapEncodeTiled_v12000 encode_fn()
{
    static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
    static std::once_flag once;
    std::call_once(once, [] {
        void *ptr = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(ptr);
    });
    return fn;
}

// bf16 matrix [rows][cols] with the given row stride, read in boxes of
// box_rows x 64 with 128-byte swizzle.
bool make_map(CUtensorMap *map, const void *base, uint64_t rows, uint64_t cols, uint64_t row_stride_bytes,
              uint32_t box_rows)
{
    auto fn = encode_fn();
    if (!fn) return false;
    const cuuint64_t dims[2] = {cols, rows};
    const cuuint64_t strides[1] = {row_stride_bytes};
    const cuuint32_t box[2] = {(cuuint32_t)BK, box_rows};
    const cuuint32_t es[2] = {1, 1};
    return fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void *>(base), dims, strides, box, es,
              CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
              CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// Raises the kernel's dynamic shared-memory limit once per device; `configured`
// is the caller's flag word, one per kernel instantiation.
template <typename K>
cudaError_t set_smem(K kernel, size_t bytes, std::atomic<unsigned long long> &configured)
{
    int dev = 0;
    cudaGetDevice(&dev);
    const unsigned long long bit = 1ull << (dev & 63);
    if (configured.load() & bit) return cudaSuccess;
    const cudaError_t e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)bytes);
    if (e == cudaSuccess) configured.fetch_or(bit);
    return e;
}

template <int BN, bool SPLIT>
cudaError_t launch_gu_t(const CUtensorMap &a, const CUtensorMap &a2, const CUtensorMap &g, const CUtensorMap &u,
                        const GuParams &p, cudaStream_t stream)
{
    using Sh = GuShape<BN, SPLIT>;
    static std::atomic<unsigned long long> configured{0};
    cudaError_t e = set_smem(gu_kernel<BN, SPLIT>, Sh::kSmem, configured);
    if (e != cudaSuccess) return e;
    const dim3 grid((p.N + BN - 1) / BN, (p.M + BM - 1) / BM);
    gu_kernel<BN, SPLIT><<<grid, kThreads, Sh::kSmem, stream>>>(a, a2, g, u, p);
    return cudaGetLastError();
}

template <int BN>
cudaError_t launch_down_t(const CUtensorMap &a, const CUtensorMap &b, const DownParams &p, int splits,
                          cudaStream_t stream)
{
    using Sh = DownShape<BN>;
    static std::atomic<unsigned long long> configured{0};
    cudaError_t e = set_smem(down_kernel<BN>, Sh::kSmem, configured);
    if (e != cudaSuccess) return e;
    const dim3 grid((p.H + BN - 1) / BN, (p.M + BM - 1) / BM, splits);
    down_kernel<BN><<<grid, kThreads, Sh::kSmem, stream>>>(a, b, p);
    return cudaGetLastError();
}

}  // namespace
}  // namespace tc

namespace {
struct TcLayout {
    size_t xhi, xlo, hact, keep, total;
};

TcLayout tc_layout(int H, int N, int B)
{
    auto al = [](size_t v) { return (v + 255) & ~(size_t)255; };
    const size_t ldn = ((size_t)N + 7) & ~(size_t)7;
    TcLayout L{};
    size_t off = 0;
    L.xhi = off;
    off += al((size_t)B * H * 2);
    L.xlo = off;
    off += al((size_t)B * H * 2);
    L.hact = off;
    off += al((size_t)B * ldn * 2);
    L.keep = off;
    off += al((size_t)B * (((size_t)N + 15) & ~(size_t)15));
    L.total = off;
    return L;
}
}  // namespace

bool use_tc_path(int H, int B) { return B > fused_tokens_per_pass(H); }

size_t tc_workspace_bytes(int H, int N, int B) { return tc_layout(H, N, B).total; }

// The thresholded MLP for a batch of B tokens on the tensor cores.
//   x: bf16 [B][H] (x_mode kXBf16) or fp32 [B][H] (kXF32 / kXResidNorm, then
//   split into bf16 hi + lo, after RMSNorm with norm_w for kXResidNorm).
//   out: y [B][H] (kOutY) or the residual (kOutResid, += y).
cudaError_t run_tc_layer(const sats_layer *layer, int x_mode, const void *x, int B, float t_l, const float *norm_w,
                         float eps, const uint8_t *dense_flags, int out_mode, float *out, int32_t *active_idx,
                         int32_t *active_cnt, uint8_t *keep_trace, void *tc_ws, int *ctl, cudaStream_t stream)
{
    using namespace tc;
    const int H = layer->H, N = layer->N, ldn = layer->ldn;
    const TcLayout W = tc_layout(H, N, B);
    uint8_t *base = static_cast<uint8_t *>(tc_ws);
    uint16_t *xhi = reinterpret_cast<uint16_t *>(base + W.xhi);
    uint16_t *xlo = reinterpret_cast<uint16_t *>(base + W.xlo);
    uint16_t *hact = reinterpret_cast<uint16_t *>(base + W.hact);
    uint8_t *keep = base + W.keep;
    const int kstride = (N + 15) & ~15;

    const bool split = x_mode != kXBf16;
    const uint16_t *a_ptr = split ? xhi : static_cast<const uint16_t *>(x);
    cudaError_t e;
    if (split) {
        split_kernel<<<B, 256, 0, stream>>>(static_cast<const float *>(x), H,
                                            x_mode == kXResidNorm ? norm_w : nullptr, eps, xhi, xlo);
        if ((e = cudaGetLastError()) != cudaSuccess) return e;
    }
    // 96-neuron tiles give ~150 CTAs for N = 14336 at one token tile
    const int bn = B <= BM ? 96 : 128;
    CUtensorMap mA, mA2, mG, mU, mH, mD;
    if (!make_map(&mA, a_ptr, B, H, (uint64_t)H * 2, BM) ||
        !make_map(&mA2, split ? xlo : a_ptr, B, H, (uint64_t)H * 2, BM) ||
        !make_map(&mG, layer->wg_t, N, H, (uint64_t)H * 2, bn) ||
        !make_map(&mU, layer->w_ud, N, H, (uint64_t)H * 4, bn))
        return cudaErrorInvalidValue;
    GuParams gp{};
    gp.M = B;
    gp.N = N;
    gp.H = H;
    gp.t_l = t_l;
    gp.dense_flags = dense_flags;
    gp.hact = hact;
    gp.ldh = ldn;
    gp.keep = active_idx ? keep : nullptr;
    gp.keep_stride = kstride;
    gp.keep_trace = keep_trace;
    gp.ctl = ctl;
    if (bn == 96)
        e = split ? launch_gu_t<96, true>(mA, mA2, mG, mU, gp, stream)
                  : launch_gu_t<96, false>(mA, mA2, mG, mU, gp, stream);
    else
        e = split ? launch_gu_t<128, true>(mA, mA2, mG, mU, gp, stream)
                  : launch_gu_t<128, false>(mA, mA2, mG, mU, gp, stream);
    if (e != cudaSuccess) return e;

    // down projection; split K (neurons) when the tile grid alone leaves SMs idle
    const int dbn = B <= BM ? 128 : 256;
    const int tiles = ((H + dbn - 1) / dbn) * ((B + BM - 1) / BM);
    const int KB = (N + BK - 1) / BK;
    int sms = 0, dev = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    int splits = tiles >= sms ? 1 : (sms + tiles - 1) / tiles;
    if (splits > KB) splits = KB;
    const int kbps = (KB + splits - 1) / splits;
    splits = (KB + kbps - 1) / kbps;
    if (!make_map(&mH, hact, B, N, (uint64_t)ldn * 2, BM) || !make_map(&mD, layer->wd_t, H, N, (uint64_t)ldn * 2, dbn))
        return cudaErrorInvalidValue;
    DownParams dp{};
    dp.M = B;
    dp.N = N;
    dp.H = H;
    dp.kb_per_split = kbps;
    dp.atomic_out = splits > 1 ? 1 : 0;
    dp.add_residual = out_mode == kOutResid ? 1 : 0;
    dp.out = out;
    dp.ctl = ctl;
    if (splits > 1 && out_mode == kOutY) {
        if ((e = cudaMemsetAsync(out, 0, (size_t)B * H * sizeof(float), stream)) != cudaSuccess) return e;
    }
    e = dbn == 128 ? launch_down_t<128>(mH, mD, dp, splits, stream) : launch_down_t<256>(mH, mD, dp, splits, stream);
    if (e != cudaSuccess) return e;
    if (active_idx) {
        keep_list_kernel<<<B, 512, 0, stream>>>(keep, kstride, N, active_idx, active_cnt);
        if ((e = cudaGetLastError()) != cudaSuccess) return e;
    }
    return cudaSuccess;
}

}  // namespace sats
