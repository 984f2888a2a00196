// tc_common.cuh -- helpers shared by the tensor-core kernels (gemm_tc.cu,
// union_mlp.cu): tcgen05 descriptors and instructions, TMEM access, TMA tile
// loads, and the host side of tensor maps, shared-memory limits and launches
// with programmatic dependent launch.  Included once per translation unit;
// everything is in an unnamed namespace.
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <cudaTypedefs.h>

#include <atomic>
#include <cmath>
#include <mutex>
#include <utility>

#include "common.cuh"
#include "internal.h"

namespace sats {
namespace tc {
namespace {

constexpr int BM = 128;              // MMA M: rows of the A operand
constexpr int BK = 64;               // K per TMA box: one 128-byte swizzle row of bf16
constexpr int kThreads = 192;
// Epilogue groups of four warps in the prefill kernels: the last tile's epilogue of the
// persistent gate/up kernel, and every tile's of the down projection, follow their MMAs.
constexpr int kWideGuGroups = 4;     // at most: 128-neuron tiles, two 16-neuron blocks each
constexpr int kWideDownGroups = 4;   // 256 columns: four 16-column blocks each
constexpr int kWideMaxThreads = 64 + 128 * 4;
constexpr int kSkinnyMaxGroups = 6;                             // epilogue groups of four warps
constexpr int kSkinnyMaxThreads = 64 + 128 * kSkinnyMaxGroups;  // of the batched-decode gate/up kernel
constexpr int kSmemBudget = 196608;  // stage ring (one CTA per SM)
constexpr int kSmemWide = 225280;    // stage ring of the persistent prefill kernels, at most
constexpr int kMaxStages = 8;
constexpr int kMaxSkinny = 256;      // largest batch on the skinny orientation (MMA N <= 256)
// with fp32 activations (bf16 high and low parts), larger batches run faster on the prefill
// kernels: at hidden 4096 / intermediate 14336, 256 tokens took 135 us skinny and 129 us wide
// (224 tokens: 125 and 126 us); with bf16 activations the skinny kernels stay ahead up to 256
constexpr int kMaxSkinnySplit = 224;
constexpr int kMaxUnion = 8;         // largest batch on the union path (sparse-path tokens only)
constexpr int kTileBytes = BK * 2;   // bytes of one tile row
// The prefill kernels bring their weight stages into L2 this many stages ahead of
// the loads: every weight stage is read by the CTAs of all token tiles at about
// the same time, and a ring of four or five stages does not cover a miss to HBM.
constexpr int kWidePrefetch = 16;

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

// Starts bringing one TMA box (inner coordinate c0, row c1) of the tensor into L2;
// no completion to wait for.
__device__ __forceinline__ void tma_prefetch_l2(const CUtensorMap *map, int c0, int c1)
{
    asm volatile("cp.async.bulk.prefetch.tensor.2d.L2.global.tile [%0, {%1, %2}];" ::"l"(map), "r"(c0), "r"(c1)
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


__device__ __forceinline__ void set_timeout(int *ctl, volatile int *abort_flag)
{
    *abort_flag = 1;
    atomicOr(ctl + kCtlStatus, kStatusTimeout);
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

// bf16 matrix [rows][cols] with the given row stride (a multiple of 16 bytes),
// read in boxes of box_rows x 64 with 128-byte swizzle.
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

// The device's opt-in limit of shared memory per CTA.
int smem_optin()
{
    static int by_dev[64] = {0};
    int dev = 0;
    cudaGetDevice(&dev);
    int &n = by_dev[dev & 63];
    if (n == 0) cudaDeviceGetAttribute(&n, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev);
    return n;
}

// Raises the kernel's dynamic shared-memory limit on the current device to at
// least `bytes`; `configured` is the caller's per-device record for this kernel.
template <typename K>
cudaError_t set_smem(K kernel, size_t bytes, std::atomic<int> (&configured)[64])
{
    int dev = 0;
    cudaGetDevice(&dev);
    std::atomic<int> &have = configured[dev & 63];
    if ((int)bytes <= have.load()) return cudaSuccess;
    const cudaError_t e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)bytes);
    if (e == cudaSuccess) have.store((int)bytes);
    return e;
}

// Launch with programmatic dependent launch: the kernel may start while the
// preceding kernel in the stream finishes; it calls griddepcontrol.wait before
// touching anything that kernel produces.
template <typename... KArgs, typename... Args>
cudaError_t launch_pdl(void (*kernel)(KArgs...), dim3 grid, size_t smem, cudaStream_t stream, Args &&...args)
{
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = dim3(kThreads);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, kernel, std::forward<Args>(args)...);
}

// As launch_pdl, for the small kernels (no dynamic shared memory, `threads` per CTA).
template <typename... KArgs, typename... Args>
cudaError_t launch_pdl_threads(void (*kernel)(KArgs...), dim3 grid, int threads, cudaStream_t stream, Args &&...args)
{
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = dim3(threads);
    cfg.dynamicSmemBytes = 0;
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, kernel, std::forward<Args>(args)...);
}

// As launch_pdl, with `threads` per CTA and `smem` bytes of dynamic shared memory.
template <typename... KArgs, typename... Args>
cudaError_t launch_pdl_cfg(void (*kernel)(KArgs...), dim3 grid, int threads, size_t smem, cudaStream_t stream,
                           Args &&...args)
{
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = dim3(threads);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, kernel, std::forward<Args>(args)...);
}

// Dynamic shared memory of a launch: the stage ring, 1 KB of alignment slack and the barriers.
size_t smem_for(int stages, int stage_bytes) { return (size_t)stages * stage_bytes + 1024 + 256; }

// Ring budget of the prefill kernels: kSmemWide, or less if the device allows
// less (the opt-in limit covers the kernel's static shared memory as well).
int wide_budget()
{
    const int lim = smem_optin() - 1024 - 256 - 64;
    return lim < kSmemWide ? lim : kSmemWide;
}

int stages_for(int stage_bytes, int budget = kSmemBudget)
{
    const int s = budget / stage_bytes;
    return s > kMaxStages ? kMaxStages : s;
}

uint32_t tmem_cols_for(int cols)
{
    uint32_t c = 32;
    while ((int)c < cols) c <<= 1;
    return c;
}

int sm_count()
{
    static int by_dev[64] = {0};
    int dev = 0;
    cudaGetDevice(&dev);
    int &n = by_dev[dev & 63];
    if (n == 0) cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev);
    return n > 0 ? n : 1;
}

// Neurons per tile: the multiple of 16 (<= 128) that minimises waves x rows,
// so that the neuron tiles cover the SMs in about one wave.
int choose_rows(int N, int sms)
{
    int best = 16;
    long long best_cost = -1;
    for (int R = 16; R <= BM; R += 16) {
        const long long tiles = (N + R - 1) / R;
        const long long cost = ((tiles + sms - 1) / sms) * R;
        if (best_cost < 0 || cost <= best_cost) {
            best_cost = cost;
            best = R;
        }
    }
    return best;
}

// Neurons per tile of the prefill gate/up kernel: the multiple of 16 (<= 128,
// spanning at most two of the packed R-neuron tiles) that minimises waves x
// shared-memory bytes per K step.  Each operand byte is
// written to shared memory once by the copy engine and read once by the MMA; that
// traffic (the x tile, twice for split activations, plus 2 Rw weight rows) paces
// the MMA loop, while the tile's work grows with Rw.
int wide_rows(int N, int R, int mtiles, int sms, bool split)
{
    int best = 16;
    long long best_cost = -1;
    for (int Rw = 16; Rw <= BM; Rw += 16) {
        int g = Rw, r = R;   // gcd(Rw, R): a wide tile then spans at most two tiles of R neurons
        while (r) {
            const int t = g % r;
            g = r;
            r = t;
        }
        if (Rw - g > R) continue;
        const long long tiles = (long long)mtiles * ((N + Rw - 1) / Rw);
        const long long cost = ((tiles + sms - 1) / sms) * (BM * (split ? 2 : 1) + 2 * Rw);
        if (best_cost < 0 || cost <= best_cost) {
            best_cost = cost;
            best = Rw;
        }
    }
    return best;
}

// Splits of the neuron range in the prefill down projection: the count (<= 8,
// none empty) that minimises waves x (K blocks per unit + 4), the 4 standing for
// a unit's fixed cost (its accumulator's reductions into the output).
int wide_down_splits(int tiles, int KBn, int sms)
{
    int best = 1;
    long long best_cost = -1;
    for (int s = 1; s <= 8 && s <= KBn; ++s) {
        const int kps = (KBn + s - 1) / s;
        if ((KBn + kps - 1) / kps != s) continue;
        const long long units = (long long)tiles * s;
        const long long cost = ((units + sms - 1) / sms) * (kps + 4);
        if (best_cost < 0 || cost < best_cost) {
            best_cost = cost;
            best = s;
        }
    }
    return best;
}

}  // namespace
}  // namespace tc
}  // namespace sats
