// common.cuh -- device helpers shared by the library's kernels (sm_103a).
//
// Inline-PTX wrappers for the Blackwell features the kernels use: mbarrier
// phases with transaction counts, the bulk (non-tensor) asynchronous copy
// global -> shared (cp.async.bulk, completes on an mbarrier), L2 eviction
// policies, named barriers and the global nanosecond timer used to bound every
// device-side wait.
#pragma once

#include <cstdint>
#include <cuda_runtime.h>

namespace sats {

// Bits of the device status word (workspace control block or caller's word).
constexpr int kStatusBadToken = 1;   // a token id outside [0, V)
constexpr int kStatusTimeout = 2;    // a bounded wait gave up
constexpr int kStatusInternal = 4;   // an index-list position out of range (a kernel defect; the store is skipped)

// Upper bound of every device-side wait before it reports kStatusTimeout.
constexpr unsigned long long kWaitLimitNs = 2000000000ull;   // 2 s

__device__ __forceinline__ uint32_t smem_addr(const void *p)
{
    return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ unsigned long long global_ns()
{
    unsigned long long t;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
    return t;
}

__device__ __forceinline__ void mbar_init(uint64_t *bar, uint32_t count)
{
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_addr(bar)), "r"(count) : "memory");
}

// Make mbarrier initialisation visible to the other threads and to the async proxy.
__device__ __forceinline__ void mbar_init_fence()
{
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

__device__ __forceinline__ void mbar_arrive(uint64_t *bar)
{
    asm volatile("mbarrier.arrive.release.cta.shared::cta.b64 _, [%0];" ::"r"(smem_addr(bar)) : "memory");
}

__device__ __forceinline__ void mbar_arrive_expect_tx(uint64_t *bar, uint32_t bytes)
{
    asm volatile("mbarrier.arrive.expect_tx.release.cta.shared::cta.b64 _, [%0], %1;"
                 ::"r"(smem_addr(bar)), "r"(bytes) : "memory");
}

// Tests the phase; if it is not complete the thread is suspended (not spinning)
// until it completes or about kSuspendHintNs elapse.
constexpr uint32_t kSuspendHintNs = 100000;

__device__ __forceinline__ bool mbar_try_wait(uint64_t *bar, uint32_t parity)
{
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.acquire.cta.shared::cta.b64 p, [%1], %2, %3;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(smem_addr(bar)), "r"(parity), "r"(kSuspendHintNs)
        : "memory");
    return ok != 0;
}

// Waits for the phase with the given parity to complete.  Gives up after
// kWaitLimitNs or as soon as *abort becomes non-zero; returns false then.
__device__ __forceinline__ bool mbar_wait(uint64_t *bar, uint32_t parity, volatile int *abort)
{
    if (mbar_try_wait(bar, parity)) return true;
    const unsigned long long t0 = global_ns();
    for (;;) {
        if (mbar_try_wait(bar, parity)) return true;
        if (*abort) return false;
        if (global_ns() - t0 > kWaitLimitNs) return false;
    }
}

// L2 policy for data read exactly once (weights streamed per call).
__device__ __forceinline__ uint64_t l2_policy_evict_first()
{
    uint64_t p;
    asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(p));
    return p;
}

// One bulk copy global -> shared; completes `bytes` transaction bytes on `bar`.
// dst, src 16-byte aligned; bytes a multiple of 16.
__device__ __forceinline__ void bulk_load(void *dst, const void *src, uint32_t bytes, uint64_t *bar,
                                          uint64_t policy)
{
    asm volatile(
        "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint"
        " [%0], [%1], %2, [%3], %4;"
        ::"r"(smem_addr(dst)), "l"(src), "r"(bytes), "r"(smem_addr(bar)), "l"(policy)
        : "memory");
}

// As bulk_load, with the default L2 policy (data that other CTAs read too).
__device__ __forceinline__ void bulk_load_shared(void *dst, const void *src, uint32_t bytes, uint64_t *bar)
{
    asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];"
                 ::"r"(smem_addr(dst)), "l"(src), "r"(bytes), "r"(smem_addr(bar))
                 : "memory");
}

// Starts bringing `bytes` (a multiple of 16) at a 16-byte aligned global
// address into L2; no completion to wait for.
__device__ __forceinline__ void bulk_prefetch_l2(const void *src, uint32_t bytes)
{
    asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(src), "r"(bytes) : "memory");
}

// Barrier among `count` threads (a multiple of 32) on hardware barrier `id`.
__device__ __forceinline__ void named_barrier(int id, int count)
{
    asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(count) : "memory");
}

// Programmatic dependent launch: wait until the preceding grid in the stream
// has completed and its memory is visible / allow the next grid to launch.
__device__ __forceinline__ void grid_dependency_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void grid_launch_dependents() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }

// y[0..3] += v (one vector reduction in L2, no return value).
__device__ __forceinline__ void red_add_v4(float *addr, float a, float b, float c, float d)
{
    asm volatile("red.global.add.v4.f32 [%0], {%1, %2, %3, %4};" ::"l"(addr), "f"(a), "f"(b), "f"(c), "f"(d)
                 : "memory");
}

__device__ __forceinline__ int atom_add_acq_rel_gpu(int *p, int v)
{
    int old;
    asm volatile("atom.acq_rel.gpu.global.add.s32 %0, [%1], %2;" : "=r"(old) : "l"(p), "r"(v) : "memory");
    return old;
}

__device__ __forceinline__ int ld_acquire_gpu(const int *p)
{
    int v;
    asm volatile("ld.acquire.gpu.global.b32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
    return v;
}

// Relaxed (no ordering) 64-bit accesses at GPU scope, for words that carry
// their whole payload.
__device__ __forceinline__ uint64_t ld_relaxed_gpu_u64(const uint64_t *p)
{
    uint64_t v;
    asm volatile("ld.relaxed.gpu.global.b64 %0, [%1];" : "=l"(v) : "l"(p) : "memory");
    return v;
}

__device__ __forceinline__ void st_relaxed_gpu_u64(uint64_t *p, uint64_t v)
{
    asm volatile("st.relaxed.gpu.global.b64 [%0], %1;" ::"l"(p), "l"(v) : "memory");
}

__device__ __forceinline__ void st_release_gpu(int *p, int v)
{
    asm volatile("st.release.gpu.global.b32 [%0], %1;" ::"l"(p), "r"(v) : "memory");
}

// bf16 pair (one 32-bit word, element 2i in the low half) -> two floats.
__device__ __forceinline__ float bf16_lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf16_hi(uint32_t w) { return __uint_as_float(w & 0xffff0000u); }

__device__ __forceinline__ void unpack8(const uint4 &v, float (&f)[8])
{
    f[0] = bf16_lo(v.x); f[1] = bf16_hi(v.x);
    f[2] = bf16_lo(v.y); f[3] = bf16_hi(v.y);
    f[4] = bf16_lo(v.z); f[5] = bf16_hi(v.z);
    f[6] = bf16_lo(v.w); f[7] = bf16_hi(v.w);
}

// Packed pair of floats in one 64-bit register (low half = even element), the
// operand type of the sm_100-family paired FP32 instructions.
typedef unsigned long long f32x2;

__device__ __forceinline__ f32x2 pack2(float lo, float hi)
{
    f32x2 r;
    asm("mov.b64 %0, {%1, %2};" : "=l"(r) : "f"(lo), "f"(hi));
    return r;
}

__device__ __forceinline__ float2 unpack2(f32x2 v)
{
    float lo, hi;
    asm("mov.b64 {%0, %1}, %2;" : "=f"(lo), "=f"(hi) : "l"(v));
    return make_float2(lo, hi);
}

// d = a * b + c on both halves, each rounded once (fma.rn per element).
__device__ __forceinline__ f32x2 ffma2(f32x2 a, f32x2 b, f32x2 c)
{
    f32x2 d;
    asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(d) : "l"(a), "l"(b), "l"(c));
    return d;
}

// One 32-bit word holding two bf16 (element 2i low) -> their exact float pair.
__device__ __forceinline__ f32x2 bf16x2_to_f32x2(uint32_t w)
{
    return pack2(__uint_as_float(w << 16), __uint_as_float(w & 0xffff0000u));
}

// acc += w[0..7] * x[0..7] on pairs (w: 8 bf16 in a uint4, x: 4 float pairs).
__device__ __forceinline__ f32x2 dot8_acc(const uint4 &w, const f32x2 (&x)[4], f32x2 acc)
{
    acc = ffma2(bf16x2_to_f32x2(w.x), x[0], acc);
    acc = ffma2(bf16x2_to_f32x2(w.y), x[1], acc);
    acc = ffma2(bf16x2_to_f32x2(w.z), x[2], acc);
    acc = ffma2(bf16x2_to_f32x2(w.w), x[3], acc);
    return acc;
}

// y[0..7] += h * w[0..7] on pairs.
__device__ __forceinline__ void axpy8(const uint4 &w, f32x2 hh, f32x2 (&y)[4])
{
    y[0] = ffma2(bf16x2_to_f32x2(w.x), hh, y[0]);
    y[1] = ffma2(bf16x2_to_f32x2(w.y), hh, y[1]);
    y[2] = ffma2(bf16x2_to_f32x2(w.z), hh, y[2]);
    y[3] = ffma2(bf16x2_to_f32x2(w.w), hh, y[3]);
}

__device__ __forceinline__ float hsum2(f32x2 v)
{
    const float2 f = unpack2(v);
    return f.x + f.y;
}

// Sums four per-lane values p[0..3] over the warp with 6 shuffles: on return,
// lane L holds the warp total of p[(L >> 3) & 3] (lanes 0, 8, 16, 24 hold
// rows 0, 1, 2, 3).
__device__ __forceinline__ float warp_sum4_transposed(float p0, float p1, float p2, float p3, int lane)
{
    const bool up = (lane & 16) != 0;
    float a0 = up ? p2 : p0, a1 = up ? p3 : p1;
    const float s0 = up ? p0 : p2, s1 = up ? p1 : p3;
    a0 += __shfl_xor_sync(0xffffffffu, s0, 16);
    a1 += __shfl_xor_sync(0xffffffffu, s1, 16);
    const bool b3 = (lane & 8) != 0;
    float b = b3 ? a1 : a0;
    const float s = b3 ? a0 : a1;
    b += __shfl_xor_sync(0xffffffffu, s, 8);
    b += __shfl_xor_sync(0xffffffffu, b, 4);
    b += __shfl_xor_sync(0xffffffffu, b, 2);
    b += __shfl_xor_sync(0xffffffffu, b, 1);
    return b;
}

// Same for two values: lanes 0-15 hold the total of p0, lanes 16-31 of p1.
__device__ __forceinline__ float warp_sum2_transposed(float p0, float p1, int lane)
{
    const bool up = (lane & 16) != 0;
    float a = up ? p1 : p0;
    const float s = up ? p0 : p1;
    a += __shfl_xor_sync(0xffffffffu, s, 16);
    a += __shfl_xor_sync(0xffffffffu, a, 8);
    a += __shfl_xor_sync(0xffffffffu, a, 4);
    a += __shfl_xor_sync(0xffffffffu, a, 2);
    a += __shfl_xor_sync(0xffffffffu, a, 1);
    return a;
}

__device__ __forceinline__ float warp_sum(float v)
{
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}

}  // namespace sats
