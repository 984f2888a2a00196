// small_mlp.cu -- the CATS-thresholded gated MLP (Sec. 2, Eqs. 1-5 of
// arXiv 2607.08991) for small layers (hidden <= 1024 and a few thousand
// neurons): one thread-block cluster per call, no global synchronisation.
//
// For a layer this small a call is a few round trips to memory, and the
// persistent decode kernel's machinery (a grid-wide prologue count, the slice
// look-back of the index lists, the end-of-call election of 152 CTAs) would be
// most of its time.  Here one cluster of C CTAs (16 where the GPU offers
// clusters that large, else 8) takes the call; CTA c owns the neurons
// [c R, (c + 1) R), each of its NW warps RW <= MR consecutive ones (R = NW RW):
//   1. before the dependency wait of programmatic dependent launch (weights do
//      not depend on the previous call) the CTA's gate rows, one contiguous
//      block of Wg_t, land in shared memory by bulk copies;
//   2. every warp loads the activations (RMSNorm for a stack) and computes its
//      rows' gate dot products from shared memory (paired FP32 FMAs, all its
//      rows in one transposed warp reduction), SiLU (Eq. 2) and the mask
//      |a| >= t per token (Eqs. 4-5);
//   3. each warp reads the W_ud rows of its kept neurons only (a skipped
//      neuron costs no bytes beyond its gate row) straight into registers,
//      each lane the 16-byte vectors it multiplies, two rows' loads in flight
//      at a time; then up dot product, h = a u, and the down projection
//      h W_down[j, :] into its y columns;
//   4. as soon as the masks are known, the CTA's kept count per token goes into
//      the shared memory of the CTAs after it (distributed shared memory), the
//      CTA clears its slice of y (a plain output), and its threads arrive on
//      the cluster barrier - every CTA has then read its activations (the
//      output may alias them), cleared its slice and sent its counts;
//   5. after step 3 the threads wait on that barrier (long complete by then),
//      write the CTA's entries of the ascending index lists at the offset the
//      earlier CTAs' counts give, sum the warps' y partials through shared
//      memory and add the CTA's partial y into the output with vector
//      reductions in L2.  Nothing touches another CTA's shared memory after
//      the barrier.
// The only wait is the bounded one on the gate rows' bulk copies; the cluster
// barrier is a hardware barrier of co-scheduled CTAs.
#include <cmath>

#include "common.cuh"
#include "internal.h"

namespace sats {
namespace {

constexpr int kSmMaxH = 1024;
constexpr size_t kSmMaxRowBytes = 192 * 1024;     // a CTA's gate rows in shared memory
constexpr size_t kSmMaxSmem = kSmMaxRowBytes + 9216;
constexpr uint32_t kSmCopyBytes = 32768;          // bytes per bulk copy of gate rows

// 16-byte load of read-once data (the W_ud rows): not kept in L1.
__device__ __forceinline__ uint4 ld_stream_v4(const uint4 *p)
{
    uint4 v;
    asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0, %1, %2, %3}, [%4];"
                 : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
                 : "l"(p));
    return v;
}

__device__ __forceinline__ uint32_t cluster_ctarank()
{
    uint32_t r;
    asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
    return r;
}

// Address of `p` (this CTA's shared memory) in the shared memory of cluster CTA `rank`.
__device__ __forceinline__ uint32_t dsmem_addr(const void *p, uint32_t rank)
{
    uint32_t r;
    asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(smem_addr(p)), "r"(rank));
    return r;
}

__device__ __forceinline__ void st_dsmem_s32(uint32_t addr, int v)
{
    asm volatile("st.shared::cluster.s32 [%0], %1;" ::"r"(addr), "r"(v) : "memory");
}

// Sums eight per-lane values p[0..7] over the warp with 9 shuffles: on return,
// lane L holds the warp total of p[(L >> 2) & 7] (lanes 0, 4, ..., 28 hold rows 0 .. 7).
__device__ __forceinline__ float warp_sum8_transposed(const float (&p)[8], int lane)
{
    const bool b4 = (lane & 16) != 0, b3 = (lane & 8) != 0, b2 = (lane & 4) != 0;
    float a[4], c[2];
#pragma unroll
    for (int k = 0; k < 4; ++k) {
        const float keep = b4 ? p[4 + k] : p[k], send = b4 ? p[k] : p[4 + k];
        a[k] = keep + __shfl_xor_sync(0xffffffffu, send, 16);
    }
#pragma unroll
    for (int k = 0; k < 2; ++k) {
        const float keep = b3 ? a[2 + k] : a[k], send = b3 ? a[k] : a[2 + k];
        c[k] = keep + __shfl_xor_sync(0xffffffffu, send, 8);
    }
    float d = (b2 ? c[1] : c[0]) + __shfl_xor_sync(0xffffffffu, b2 ? c[0] : c[1], 4);
    d += __shfl_xor_sync(0xffffffffu, d, 2);
    d += __shfl_xor_sync(0xffffffffu, d, 1);
    return d;
}

// Layout of the dynamic shared memory: the CTA's R gate rows of 2H bytes; the
// region then holds the warps' y partials, [NW][BT][H] floats, once every warp
// is past the gate rows.
struct SmallLayout {
    size_t rows, total;
    int per;   // float4 column groups of y per CTA slice (cleared by that CTA)
};

__host__ __device__ inline SmallLayout small_layout(int H, int R, int NW, int BT, int C)
{
    SmallLayout L{};
    const size_t row_bytes = (size_t)R * H * 2;
    const size_t red_bytes = (size_t)NW * BT * H * 4;
    L.per = ((H >> 2) + C - 1) / C;
    L.rows = 0;
    L.total = ((row_bytes > red_bytes ? row_bytes : red_bytes) + 127) & ~(size_t)127;
    return L;
}

template <int BT, int NW>
struct SmallState {
    uint64_t gfull;               // the gate rows have landed
    uint32_t keepw[BT][32];       // the CTA's keep words per token (bit j of word i = neuron 32 i + j of the CTA)
    int wpre[BT][32];             // kept neurons of the CTA in the words before word i
    int cnt_recv[BT][16];         // kept counts of the CTAs before this one (stored by them)
    int warp_any[32];             // warp w has a y partial
    int ok;
};

template <int MR>
__device__ __forceinline__ float warp_sum_rows_transposed(const float (&p)[MR], int lane);

template <>
__device__ __forceinline__ float warp_sum_rows_transposed<4>(const float (&p)[4], int lane)
{
    return warp_sum4_transposed(p[0], p[1], p[2], p[3], lane);   // lane 8 r owns row r
}

template <>
__device__ __forceinline__ float warp_sum_rows_transposed<8>(const float (&p)[8], int lane)
{
    return warp_sum8_transposed(p, lane);                        // lane 4 r owns row r
}

template <int BT, int VPL, int NW, int MR>
__global__ void __launch_bounds__(NW * 32, 1) small_mlp_kernel(const FusedParams p, int R, int RW)
{
    extern __shared__ __align__(128) uint8_t smem[];
    __shared__ SmallState<BT, NW> S;
    constexpr int kThreads = NW * 32;
    constexpr int kLead = 32 / MR;                 // lane stride of the row owners after the reduction
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int H = p.H, N = p.N, HV = H >> 3, H4 = H >> 2;
    const uint32_t C = gridDim.x;                  // the grid is one cluster
    const uint32_t rank = cluster_ctarank();
    const int c0 = (int)rank * R;                  // the CTA's first neuron
    const int cn = max(0, min(N - c0, R));         // neurons of this CTA
    const SmallLayout Ls = small_layout(H, R, NW, BT, (int)C);
    uint8_t *rows_s = smem + Ls.rows;              // gate rows [R][2H bytes]
    float *red_s = reinterpret_cast<float *>(smem + Ls.rows);    // [NW][BT][H], last
    const int per = Ls.per;

    // 1. the CTA's gate rows (contiguous in Wg_t) into shared memory, before the dependency wait
    if (tid == 0) {
        mbar_init(&S.gfull, 1);
        mbar_init_fence();
    }
    for (int i = tid; i < BT * 32; i += kThreads) S.keepw[i / 32][i % 32] = 0u;
    if (tid < 32) S.warp_any[tid] = 0;
    if (tid == 0) S.ok = 1;
    __syncthreads();
    const uint64_t pol = l2_policy_evict_first();
    if (tid == 0) {
        const uint32_t bytes = (uint32_t)cn * (uint32_t)H * 2u;
        mbar_arrive_expect_tx(&S.gfull, bytes);
        const char *src = reinterpret_cast<const char *>(p.wg_t + (size_t)c0 * H);
        for (uint32_t off = 0; off < bytes; off += kSmCopyBytes)
            bulk_load(rows_s + off, src + off, min(kSmCopyBytes, bytes - off), &S.gfull, pol);
    }
    grid_launch_dependents();   // the next call may start loading its weights
    grid_dependency_wait();     // x, the output and the status word belong to the previous call until it ends

    // 2. activations as float pairs (lane owns vectors lane + 32 i); RMSNorm per warp (each warp holds all of x)
    f32x2 xp[BT][VPL][4];
#pragma unroll
    for (int b = 0; b < BT; ++b) {
        float xv[VPL][8];
#pragma unroll
        for (int i = 0; i < VPL; ++i) {
            const int v = lane + 32 * i;
#pragma unroll
            for (int e = 0; e < 8; ++e) xv[i][e] = 0.f;
            if (v < HV && b < p.nb) {
                if (p.x_mode == kXBf16) {
                    unpack8(reinterpret_cast<const uint4 *>(static_cast<const uint16_t *>(p.x) + (size_t)b * H)[v],
                            xv[i]);
                } else {
                    const float4 *src = reinterpret_cast<const float4 *>(static_cast<const float *>(p.x) + (size_t)b * H);
                    const float4 lo = src[2 * v], hi = src[2 * v + 1];
                    xv[i][0] = lo.x; xv[i][1] = lo.y; xv[i][2] = lo.z; xv[i][3] = lo.w;
                    xv[i][4] = hi.x; xv[i][5] = hi.y; xv[i][6] = hi.z; xv[i][7] = hi.w;
                }
            }
        }
        if (p.x_mode == kXResidNorm) {
            float s = 0.f;
#pragma unroll
            for (int i = 0; i < VPL; ++i)
#pragma unroll
                for (int e = 0; e < 8; ++e) s = fmaf(xv[i][e], xv[i][e], s);
            const float inv = 1.0f / sqrtf(warp_sum(s) / (float)H + p.eps);
#pragma unroll
            for (int i = 0; i < VPL; ++i) {
                const int v = lane + 32 * i;
                if (v < HV) {
                    const float4 *gw4 = reinterpret_cast<const float4 *>(p.norm_w);
                    const float4 lo = gw4[2 * v], hi = gw4[2 * v + 1];
                    const float g8[8] = {lo.x, lo.y, lo.z, lo.w, hi.x, hi.y, hi.z, hi.w};
#pragma unroll
                    for (int e = 0; e < 8; ++e) xv[i][e] = xv[i][e] * inv * g8[e];
                }
            }
        }
#pragma unroll
        for (int i = 0; i < VPL; ++i)
#pragma unroll
            for (int e = 0; e < 4; ++e) xp[b][i][e] = pack2(xv[i][2 * e], xv[i][2 * e + 1]);
    }
    float thr[BT];
#pragma unroll
    for (int b = 0; b < BT; ++b)
        thr[b] = b < p.nb ? ((p.dense_flags && p.dense_flags[b]) ? 0.f : p.t_l) : INFINITY;

    // gate rows landed (bounded wait); on a timeout the call reports it and writes no output
    int never = 0;
    if (!mbar_wait(&S.gfull, 0u, &never)) {
        if (lane == 0) {
            S.ok = 0;
            atomicOr(p.ctl + kCtlStatus, kStatusTimeout);
        }
        (void)mbar_wait(&S.gfull, 0u, &never);   // once more, bounded: copies still in flight land first
    }

    // gate dot products of the warp's rows w0 .. w0 + RW - 1 (CTA-local) in one transposed reduction;
    // lane kLead r owns row w0 + r afterwards
    const int w0 = warp * RW;
    const int myr = lane / kLead;
    const bool leader = (lane % kLead) == 0 && myr < RW && w0 + myr < cn;
    float am[BT];          // keep ? a : 0 of the leader lane's row
    uint32_t kept = 0;     // bit r: row w0 + r kept by some token
    {
        f32x2 a2[MR][BT];
#pragma unroll
        for (int r = 0; r < MR; ++r)
#pragma unroll
            for (int b = 0; b < BT; ++b) a2[r][b] = 0ull;
#pragma unroll
        for (int i = 0; i < VPL; ++i) {
            const int v = lane + 32 * i;
            if (v < HV) {
#pragma unroll
                for (int r = 0; r < MR; ++r) {
                    const int row = w0 + r;   // rows past the warp's or the CTA's read zeros and are never kept
                    const uint4 w = (r < RW && row < cn)
                                        ? reinterpret_cast<const uint4 *>(rows_s + (size_t)row * H * 2)[v]
                                        : make_uint4(0u, 0u, 0u, 0u);
#pragma unroll
                    for (int b = 0; b < BT; ++b) a2[r][b] = dot8_acc(w, xp[b][i], a2[r][b]);
                }
            }
        }
#pragma unroll
        for (int b = 0; b < BT; ++b) {
            float part[MR];
#pragma unroll
            for (int r = 0; r < MR; ++r) part[r] = hsum2(a2[r][b]);
            const float g = warp_sum_rows_transposed<MR>(part, lane);
            const float a = g / (1.0f + expf(-g));                        // SiLU, Eq. 2
            const bool keep = leader && b < p.nb && fabsf(a) >= thr[b];   // Eqs. 4-5
            am[b] = keep ? a : 0.f;
            const uint32_t bal = __ballot_sync(0xffffffffu, keep);
            uint32_t rk = 0;
#pragma unroll
            for (int r = 0; r < MR; ++r) rk |= ((bal >> (kLead * r)) & 1u) << r;
            kept |= rk;
            if (leader && b < p.nb && p.keep_trace) p.keep_trace[(size_t)b * N + c0 + w0 + myr] = keep ? 1 : 0;
            if (keep) atomicOr(&S.keepw[b][(w0 + myr) >> 5], 1u << ((w0 + myr) & 31));
        }
    }
    __syncthreads();   // every warp is past the gate rows: the region may hold the y partials from here on
    if (!S.ok) kept = 0u;

    // 4. the CTA's kept counts to the CTAs after it, its slice of y cleared, then the arrival
    if (warp == 0) {
        const int nwords = (R + 31) >> 5;
#pragma unroll
        for (int b = 0; b < BT; ++b) {
            const int c = lane < nwords ? __popc(S.keepw[b][lane]) : 0;
            int incl = c;
#pragma unroll
            for (int o = 1; o < 32; o <<= 1) {
                const int t = __shfl_up_sync(0xffffffffu, incl, o);
                if (lane >= o) incl += t;
            }
            S.wpre[b][lane] = incl - c;
            const int tot = __shfl_sync(0xffffffffu, incl, 31);
            if (lane > (int)rank && lane < (int)C) st_dsmem_s32(dsmem_addr(&S.cnt_recv[b][rank], (uint32_t)lane), tot);
        }
    }
    if (p.out_mode == kOutY) {
        const int k0 = (int)rank * per, nk = max(0, min(H4, k0 + per) - k0);
        for (int q = tid; q < p.nb * nk; q += kThreads)
            reinterpret_cast<float4 *>(p.out + (size_t)(q / nk) * H)[k0 + q % nk] = make_float4(0.f, 0.f, 0.f, 0.f);
    }
    asm volatile("barrier.cluster.arrive.release.aligned;" ::: "memory");

    // 3. the warp's kept W_ud rows, read straight into registers: lane takes the 16-byte vectors
    //    lane + 32 i of each kept row's up half and down half, two rows' loads in flight at a time.
    //    (One bulk copy per 2H-byte row had queued on the SM's copy engine: with about fifty rows
    //    per CTA the last warp's rows landed 2.3 us after the first's.)
    f32x2 yp[BT][VPL][4];
#pragma unroll
    for (int b = 0; b < BT; ++b)
#pragma unroll
        for (int i = 0; i < VPL; ++i)
#pragma unroll
            for (int e = 0; e < 4; ++e) yp[b][i][e] = 0ull;
    for (uint32_t todo = kept; todo;) {
        int rr[2];
        uint4 wu[2][VPL], wd[2][VPL];
#pragma unroll
        for (int k = 0; k < 2; ++k) {
            rr[k] = todo ? __ffs(todo) - 1 : -1;
            if (todo) todo &= todo - 1u;
            const uint4 *row = rr[k] >= 0 ? reinterpret_cast<const uint4 *>(p.w_ud + (size_t)(c0 + w0 + rr[k]) * 2 * H)
                                          : nullptr;
#pragma unroll
            for (int i = 0; i < VPL; ++i) {
                const int v = lane + 32 * i;
                const bool in = row != nullptr && v < HV;
                wu[k][i] = in ? ld_stream_v4(row + v) : make_uint4(0u, 0u, 0u, 0u);
                wd[k][i] = in ? ld_stream_v4(row + HV + v) : make_uint4(0u, 0u, 0u, 0u);
            }
        }
#pragma unroll
        for (int k = 0; k < 2; ++k) {
            if (rr[k] < 0) break;
#pragma unroll
            for (int b = 0; b < BT; ++b) {
                f32x2 u2 = 0ull;
#pragma unroll
                for (int i = 0; i < VPL; ++i) u2 = dot8_acc(wu[k][i], xp[b][i], u2);
                const float u = warp_sum(hsum2(u2));
                const float h = __shfl_sync(0xffffffffu, am[b], kLead * rr[k]) * u;   // CATS_t(a) (x W_up), Eqs. 1, 5
                const f32x2 hh = pack2(h, h);
#pragma unroll
                for (int i = 0; i < VPL; ++i) axpy8(wd[k][i], hh, yp[b][i]);
            }
        }
    }

    // 5. every CTA has sent its counts, cleared its slice of y and read its activations
    asm volatile("barrier.cluster.wait.acquire.aligned;" ::: "memory");
    if (p.active_idx) {
        for (int b = 0; b < p.nb; ++b) {
            int before = 0;
            for (uint32_t r = 0; r < rank; ++r) before += S.cnt_recv[b][r];
            for (int row = tid; row < cn; row += kThreads) {
                const uint32_t w = S.keepw[b][row >> 5];
                const uint32_t bit = 1u << (row & 31);
                if (!(w & bit)) continue;
                const int pos = before + S.wpre[b][row >> 5] + __popc(w & (bit - 1u));
                if (pos < N) p.active_idx[(size_t)b * N + pos] = c0 + row;
                else atomicOr(p.ctl + kCtlStatus, kStatusInternal);
            }
            if (rank == C - 1 && tid == 0 && p.active_cnt) {
                int own = 0;
                for (int i = 0; i < 32; ++i) own += __popc(S.keepw[b][i]);
                p.active_cnt[b] = before + own;
            }
        }
    }
    // the CTA's partial y: each warp with kept rows writes its partial, the columns are summed over
    // the warps and added into the output (a cleared y, or the residual stream)
    if (kept) {
        if (lane == 0) S.warp_any[warp] = 1;
#pragma unroll
        for (int b = 0; b < BT; ++b)
#pragma unroll
            for (int i = 0; i < VPL; ++i) {
                const int v = lane + 32 * i;
                if (v < HV) {
                    float4 *dst = reinterpret_cast<float4 *>(red_s + ((size_t)warp * BT + b) * H + 8 * v);
                    const float2 y0 = unpack2(yp[b][i][0]), y1 = unpack2(yp[b][i][1]);
                    const float2 y2 = unpack2(yp[b][i][2]), y3 = unpack2(yp[b][i][3]);
                    dst[0] = make_float4(y0.x, y0.y, y1.x, y1.y);
                    dst[1] = make_float4(y2.x, y2.y, y3.x, y3.y);
                }
            }
    }
    __syncthreads();
    if (!S.ok) return;
    for (int q = tid; q < p.nb * H4; q += kThreads) {
        const int b = q / H4, k = q % H4;
        float4 s = make_float4(0.f, 0.f, 0.f, 0.f);
        bool any = false;
        for (int w = 0; w < NW; ++w) {
            if (!S.warp_any[w]) continue;
            const float4 v = reinterpret_cast<const float4 *>(red_s + ((size_t)w * BT + b) * H)[k];
            s.x += v.x; s.y += v.y; s.z += v.z; s.w += v.w;
            any = true;
        }
        if (any) red_add_v4(p.out + (size_t)b * H + 4 * k, s.x, s.y, s.z, s.w);
    }
}

// The kernel's shapes: threads per CTA (NW warps) and rows per warp (MR) by tokens and vectors
// per lane.  One token on H <= 512: 24 warps of at most four rows (85 registers a thread); two
// tokens: 16 warps of at most eight; H <= 1024: 8 warps of at most eight.
template <int BT, int VPL>
struct SmallShape {
    static constexpr int NW = VPL <= 2 ? (BT == 1 ? 24 : 16) : 8;
    static constexpr int MR = (VPL <= 2 && BT == 1) ? 4 : 8;
};

// Cluster size available for a kernel on the current device: 16 if the GPU
// co-schedules clusters that large with this shared memory, else 8, else 0.
template <int BT, int VPL>
int cluster_size_for()
{
    using Sh = SmallShape<BT, VPL>;
    static int cached[64] = {0};   // per device: C + 1 (0 = not yet asked)
    int dev = 0;
    cudaGetDevice(&dev);
    int &slot = cached[dev & 63];
    if (slot) return slot - 1;
    auto kern = small_mlp_kernel<BT, VPL, Sh::NW, Sh::MR>;
    int C = 0;
    if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kSmMaxSmem) == cudaSuccess &&
        cudaFuncSetAttribute(kern, cudaFuncAttributeNonPortableClusterSizeAllowed, 1) == cudaSuccess) {
        for (int c : {16, 8}) {
            cudaLaunchConfig_t cfg = {};
            cfg.gridDim = dim3(c);
            cfg.blockDim = dim3(Sh::NW * 32);
            cfg.dynamicSmemBytes = kSmMaxSmem;
            cudaLaunchAttribute attr[1];
            attr[0].id = cudaLaunchAttributeClusterDimension;
            attr[0].val.clusterDim.x = c;
            attr[0].val.clusterDim.y = 1;
            attr[0].val.clusterDim.z = 1;
            cfg.attrs = attr;
            cfg.numAttrs = 1;
            int n = 0;
            if (cudaOccupancyMaxActiveClusters(&n, kern, &cfg) == cudaSuccess && n >= 1) {
                C = c;
                break;
            }
        }
    }
    cudaGetLastError();   // a refused size is not an error of the caller
    slot = C + 1;
    return C;
}

struct SmallPlan {
    int C = 0, R = 0, RW = 0;
    size_t smem = 0;
};

template <int BT, int VPL>
SmallPlan plan_small(int H, int N)
{
    using Sh = SmallShape<BT, VPL>;
    SmallPlan pl;
    const int C = cluster_size_for<BT, VPL>();
    if (C == 0) return pl;
    const int RW = (N + C * Sh::NW - 1) / (C * Sh::NW);
    if (RW > Sh::MR) return pl;
    const int R = RW * Sh::NW;
    const SmallLayout L = small_layout(H, R, Sh::NW, BT, C);
    if ((size_t)R * H * 2 > kSmMaxRowBytes || L.total > kSmMaxSmem || R > 32 * 32) return pl;
    pl.C = C;
    pl.R = R;
    pl.RW = RW;
    pl.smem = L.total;
    return pl;
}

template <int BT, int VPL>
cudaError_t launch_small_t(const FusedParams &p, cudaStream_t stream)
{
    using Sh = SmallShape<BT, VPL>;
    const SmallPlan pl = plan_small<BT, VPL>(p.H, p.N);
    if (pl.C == 0) return cudaErrorNotSupported;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(pl.C);
    cfg.blockDim = dim3(Sh::NW * 32);
    cfg.dynamicSmemBytes = pl.smem;
    cfg.stream = stream;
    cudaLaunchAttribute attr[2];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = pl.C;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[1].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 2;
    return cudaLaunchKernelEx(&cfg, small_mlp_kernel<BT, VPL, Sh::NW, Sh::MR>, p, pl.R, pl.RW);
}

int vectors_per_lane(int H) { return H <= 256 ? 1 : (H <= 512 ? 2 : 4); }

}  // namespace

bool use_small_path(int H, int N, int nb)
{
    if (H > kSmMaxH || nb < 1 || nb > 2) return false;
    const int vpl = vectors_per_lane(H);
    SmallPlan pl;
    if (nb == 1)
        pl = vpl == 1 ? plan_small<1, 1>(H, N) : (vpl == 2 ? plan_small<1, 2>(H, N) : plan_small<1, 4>(H, N));
    else
        pl = vpl == 1 ? plan_small<2, 1>(H, N) : (vpl == 2 ? plan_small<2, 2>(H, N) : plan_small<2, 4>(H, N));
    return pl.C != 0;
}

cudaError_t launch_small(const FusedParams &p, cudaStream_t stream)
{
    if (p.nb < 1 || p.nb > 2 || p.H > kSmMaxH || p.lora_blk) return cudaErrorInvalidValue;
    const int vpl = vectors_per_lane(p.H);
    if (p.nb == 1) {
        if (vpl == 1) return launch_small_t<1, 1>(p, stream);
        if (vpl == 2) return launch_small_t<1, 2>(p, stream);
        return launch_small_t<1, 4>(p, stream);
    }
    if (vpl == 1) return launch_small_t<2, 1>(p, stream);
    if (vpl == 2) return launch_small_t<2, 2>(p, stream);
    return launch_small_t<2, 4>(p, stream);
}

}  // namespace sats
