// union_mlp.cu -- batched decode on the union of the tokens' kept neurons.
//
// For a small batch of sparse-path tokens (Sec. 2, Eqs. 1-5 per token, one
// threshold t_l), the gate is dense but the up and down projections are needed
// only for neurons that some token keeps: U = {j : exists m, |a_mj| >= t_l}.
// After the gate-only tensor-core GEMM (gemm_tc.cu) has written
// a_keep[m][j] = keep_mj ? a_mj : 0 and one union flag per neuron:
//   union_list_kernel     U as an ascending list (one CTA, one pass);
//   union_up_rows_kernel  u[m][p] = x_m . W_up[:, U_p]
//   union_down_rows_kernel y_m += sum_p (a_keep[m][U_p] u[m][p]) W_down[U_p, :]
// Each CTA takes a contiguous range of union positions.  The rows of a union
// neuron are read whole (its up half, then its down half: 2H contiguous bytes
// each, one bulk copy per row) into a ring of shared-memory stages, since the
// copies must be a few KB each to stream at the memory's rate; gathering 128-
// byte row pieces for tensor-core tiles is limited by the per-copy cost, and
// at a handful of tokens the CUDA cores keep up (2 FLOP per weight per token).
// Thread t covers hidden units 8t..8t+7: x (up) or y (down) for every token
// stays in its registers as float pairs, products use paired FMAs.  Only W_gate
// and the union's W_ud rows are read.  Every wait is bounded and sets the
// status word when it gives up.
#include "tc_common.cuh"

namespace sats {
namespace tc {
namespace {

constexpr int kRowThreads = 512;     // 16 warps; thread t covers hidden units 8t..8t+7 (H <= 4096)
constexpr int kRowWarps = kRowThreads / 32;
constexpr int kRowsPerStage = 4;
constexpr int kRowStages = 6;        // ring: 6 stages of 4 rows (192 KB at H = 4096)

// ---------------------------------------------------------------------- union list
// U from the flags in one pass: thread t counts the flags of neurons 16t..16t+15
// of each 16384-neuron block, a block scan places them.
__global__ void __launch_bounds__(1024) union_list_kernel(const uint8_t *__restrict__ uflag, int N,
                                                          int32_t *__restrict__ ulist, int32_t *__restrict__ ucount)
{
    grid_dependency_wait();   // the flags are written by the gate kernel
    grid_launch_dependents();
    __shared__ int warp_sums[32];
    __shared__ int base_s;
    const int t = threadIdx.x, lane = t & 31, w = t >> 5;
    if (t == 0) base_s = 0;
    __syncthreads();
    for (int b0 = 0; b0 < N; b0 += 16 * 1024) {
        const int n0 = b0 + 16 * t;
        uint32_t bits = 0;   // bit i: neuron n0 + i is in the union
        if (n0 < N) {
            const uint4 v = *reinterpret_cast<const uint4 *>(uflag + n0);   // the flag array is padded to 16
            const uint32_t wv[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
            for (int q = 0; q < 16; ++q)
                if (((wv[q >> 2] >> (8 * (q & 3))) & 0xffu) && n0 + q < N) bits |= 1u << q;
        }
        const int cnt = __popc(bits);
        int incl = cnt;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int v = __shfl_up_sync(0xffffffffu, incl, o);
            if (lane >= o) incl += v;
        }
        if (lane == 31) warp_sums[w] = incl;
        __syncthreads();
        int before = base_s, total = 0;
        for (int i = 0; i < 32; ++i) {
            if (i < w) before += warp_sums[i];
            total += warp_sums[i];
        }
        int pos = before + incl - cnt;
        for (uint32_t m = bits; m; m &= m - 1u) ulist[pos++] = n0 + __ffs(m) - 1;
        __syncthreads();
        if (t == 0) base_s += total;
        __syncthreads();
    }
    if (t == 0) *ucount = base_s;
}

// ---------------------------------------------------------------------- union rows
struct UnionRowParams {
    const uint16_t *w_ud;         // [N][2H] bf16: up half of row j, then its down half
    const int32_t *ulist;
    const int32_t *ucount;
    const uint16_t *xa, *xlo;     // [M][H] bf16: x, or its high and low parts (xlo nullptr for bf16 x)
    const float *a_keep;          // [M][lda]
    int lda;
    float *u;                     // [M][ldu]: written by the up kernel, read by the down kernel
    int ldu;
    float *out;                   // [M][H], added to
    int M, H;
    int *ctl;
};

// The sums over the warp of MB per-lane values p[0..MB): on return lane L holds
// the total of p[v(L)], v(L) = the bits of L above bit log2(32 / MB) ... taken
// from the top: for MB = 8, v = 4 [L & 16] + 2 [L & 8] + [L & 4].
template <int MB>
__device__ __forceinline__ float warp_sum_transposed(float (&p)[MB], int lane)
{
#pragma unroll
    for (int half = MB / 2, o = 16; half >= 1; half >>= 1, o >>= 1) {
        const bool up = (lane & o) != 0;
#pragma unroll
        for (int i = 0; i < half; ++i) {
            const float keep = up ? p[i + half] : p[i];
            const float send = up ? p[i] : p[i + half];
            p[i] = keep + __shfl_xor_sync(0xffffffffu, send, o);
        }
    }
    float v = p[0];
#pragma unroll
    for (int o = 16 / MB; o >= 1; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}

template <int MB>
__device__ __forceinline__ int transposed_index(int lane)
{
    int v = 0;
#pragma unroll
    for (int half = MB / 2, o = 16; half >= 1; half >>= 1, o >>= 1)
        if (lane & o) v += half;
    return v;
}

// Per-CTA state of a row stream: union positions [p0, p1), their neurons in
// stages of kRowsPerStage rows, one bulk copy of `half` (0: up, 1: down) per row.
struct RowStream {
    uint8_t *ring;
    uint64_t *full;
    int *rows;                    // [kRowStages][kRowsPerStage]
    int p0, p1, H;
    const uint16_t *w_ud;
    const int32_t *ulist;
    int half;

    __device__ int stages() const { return (p1 - p0 + kRowsPerStage - 1) / kRowsPerStage; }
    __device__ int rows_in(int j) const { return min(kRowsPerStage, p1 - (p0 + j * kRowsPerStage)); }
    // thread 0, error path: wait (bounded) for the stages issued but not consumed
    // (j0 .. j0 + kRowStages - 1), so that no copy lands after the CTA has exited
    __device__ void drain(int j0) const
    {
        int never = 0;
        for (int j = j0; j < stages() && j < j0 + kRowStages; ++j)
            mbar_wait(&full[j % kRowStages], (uint32_t)((j / kRowStages) & 1), &never);
    }
    // thread 0: stage j's rows into its slot
    __device__ void issue(int j) const
    {
        const int slot = j % kRowStages, nr = rows_in(j);
        const uint32_t bytes = (uint32_t)H * 2u;
        int *r = rows + slot * kRowsPerStage;
        mbar_arrive_expect_tx(&full[slot], bytes * (uint32_t)nr);
        const uint64_t pol = l2_policy_evict_first();
        for (int i = 0; i < nr; ++i) {
            const int n = ulist[p0 + j * kRowsPerStage + i];
            r[i] = n;
            bulk_load(ring + ((size_t)slot * kRowsPerStage + i) * bytes, w_ud + (size_t)n * 2 * H + (size_t)half * H,
                      bytes, &full[slot], pol);
        }
    }
};

// u[m][p] = x_m . W_up[:, U_p] for this CTA's union positions.
template <int MB>
__global__ void __launch_bounds__(kRowThreads, 1) union_up_rows_kernel(const UnionRowParams p)
{
    extern __shared__ __align__(128) uint8_t ring[];
    __shared__ uint64_t full[kRowStages];
    __shared__ int rows[kRowStages * kRowsPerStage];
    __shared__ float red[kRowsPerStage][kRowWarps][MB];
    __shared__ int abort_flag;
    const int t = threadIdx.x, lane = t & 31, warp = t >> 5;
    grid_launch_dependents();
    grid_dependency_wait();   // the union list and x come from the preceding kernels
    const int count = *p.ucount;
    RowStream rs{ring, full, rows, (int)(((long long)count * blockIdx.x) / gridDim.x),
                 (int)(((long long)count * (blockIdx.x + 1)) / gridDim.x), p.H, p.w_ud, p.ulist, 0};
    const int nst = rs.stages();
    if (t == 0) {
        for (int s = 0; s < kRowStages; ++s) mbar_init(&full[s], 1);
        abort_flag = 0;
        mbar_init_fence();
        for (int j = 0; j < nst && j < kRowStages; ++j) rs.issue(j);
    }
    // x for hidden units 8t..8t+7 of every token, as float pairs
    const bool in = 8 * t < p.H;
    f32x2 xr[MB][4];
#pragma unroll
    for (int m = 0; m < MB; ++m) {
        uint4 hi = make_uint4(0u, 0u, 0u, 0u), lo = make_uint4(0u, 0u, 0u, 0u);
        if (in && m < p.M) {
            hi = *reinterpret_cast<const uint4 *>(p.xa + (size_t)m * p.H + 8 * t);
            if (p.xlo) lo = *reinterpret_cast<const uint4 *>(p.xlo + (size_t)m * p.H + 8 * t);
        }
        const uint32_t hw[4] = {hi.x, hi.y, hi.z, hi.w}, lw[4] = {lo.x, lo.y, lo.z, lo.w};
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            const float2 a = unpack2(bf16x2_to_f32x2(hw[i])), b = unpack2(bf16x2_to_f32x2(lw[i]));
            xr[m][i] = pack2(a.x + b.x, a.y + b.y);   // hi + lo: exact in fp32
        }
    }
    __syncthreads();
    const int vi = transposed_index<MB>(lane);
    int failed_at = -1;
    for (int j = 0; j < nst; ++j) {
        const int slot = j % kRowStages, nr = rs.rows_in(j);
        const bool bad = !mbar_wait(&full[slot], (uint32_t)((j / kRowStages) & 1), &abort_flag);
        if (__syncthreads_or(bad)) {   // every thread leaves together
            failed_at = j;
            break;
        }
        for (int r = 0; r < nr; ++r) {
            float part[MB];
            const uint4 w = in ? *reinterpret_cast<const uint4 *>(
                                     ring + ((size_t)slot * kRowsPerStage + r) * p.H * 2 + 16 * t)
                               : make_uint4(0u, 0u, 0u, 0u);
            const f32x2 wf[4] = {bf16x2_to_f32x2(w.x), bf16x2_to_f32x2(w.y), bf16x2_to_f32x2(w.z),
                                 bf16x2_to_f32x2(w.w)};
#pragma unroll
            for (int m = 0; m < MB; ++m) {
                f32x2 acc = ffma2(wf[0], xr[m][0], 0ull);
                acc = ffma2(wf[1], xr[m][1], acc);
                acc = ffma2(wf[2], xr[m][2], acc);
                acc = ffma2(wf[3], xr[m][3], acc);
                part[m] = hsum2(acc);
            }
            const float v = warp_sum_transposed<MB>(part, lane);
            if ((lane & (32 / MB - 1)) == 0) red[r][warp][vi] = v;
        }
        __syncthreads();
        if (t < nr * MB) {
            const int r = t / MB, m = t % MB;
            float sum = 0.f;
#pragma unroll
            for (int w = 0; w < kRowWarps; ++w) sum += red[r][w][m];
            if (m < p.M) p.u[(size_t)m * p.ldu + rs.p0 + j * kRowsPerStage + r] = sum;
        }
        __syncthreads();   // the slot and red are free again
        if (t == 0 && j + kRowStages < nst) rs.issue(j + kRowStages);
    }
    if (failed_at >= 0 && t == 0) {
        atomicOr(p.ctl + kCtlStatus, kStatusTimeout);
        rs.drain(failed_at);
    }
}

// y_m += sum over this CTA's union positions of (a_keep[m][n] u[m][p]) W_down[n, :].
template <int MB>
__global__ void __launch_bounds__(kRowThreads, 1) union_down_rows_kernel(const UnionRowParams p)
{
    extern __shared__ __align__(128) uint8_t ring[];
    __shared__ uint64_t full[kRowStages];
    __shared__ int rows[kRowStages * kRowsPerStage];
    __shared__ __align__(16) float hs[kRowStages][kRowsPerStage][MB];
    __shared__ int abort_flag;
    const int t = threadIdx.x;
    grid_launch_dependents();
    grid_dependency_wait();   // u comes from the up kernel
    const int count = *p.ucount;
    RowStream rs{ring, full, rows, (int)(((long long)count * blockIdx.x) / gridDim.x),
                 (int)(((long long)count * (blockIdx.x + 1)) / gridDim.x), p.H, p.w_ud, p.ulist, 1};
    const int nst = rs.stages();
    if (t == 0) {
        for (int s = 0; s < kRowStages; ++s) mbar_init(&full[s], 1);
        abort_flag = 0;
        mbar_init_fence();
        for (int j = 0; j < nst && j < kRowStages; ++j) rs.issue(j);
    }
    __syncthreads();
    const bool in = 8 * t < p.H;
    f32x2 yr[MB][4];
#pragma unroll
    for (int m = 0; m < MB; ++m)
#pragma unroll
        for (int i = 0; i < 4; ++i) yr[m][i] = 0ull;
    int failed_at = -1;
    for (int j = 0; j < nst; ++j) {
        const int slot = j % kRowStages, nr = rs.rows_in(j);
        if (t < nr * MB) {   // h of the stage's rows (rows[] was written by thread 0 before the last barrier)
            const int r = t / MB, m = t % MB;
            float h = 0.f;
            if (m < p.M)
                h = p.a_keep[(size_t)m * p.lda + rows[slot * kRowsPerStage + r]] *
                    p.u[(size_t)m * p.ldu + rs.p0 + j * kRowsPerStage + r];
            hs[slot][r][m] = h;
        }
        const bool bad = !mbar_wait(&full[slot], (uint32_t)((j / kRowStages) & 1), &abort_flag);
        if (__syncthreads_or(bad)) {   // also publishes hs; every thread leaves together
            failed_at = j;
            break;
        }
        if (in) {
            for (int r = 0; r < nr; ++r) {
                const uint4 w = *reinterpret_cast<const uint4 *>(
                    ring + ((size_t)slot * kRowsPerStage + r) * p.H * 2 + 16 * t);
                const f32x2 wf[4] = {bf16x2_to_f32x2(w.x), bf16x2_to_f32x2(w.y), bf16x2_to_f32x2(w.z),
                                     bf16x2_to_f32x2(w.w)};
#pragma unroll
                for (int m = 0; m < MB; ++m) {
                    const float h = hs[slot][r][m];
                    const f32x2 hh = pack2(h, h);
#pragma unroll
                    for (int i = 0; i < 4; ++i) yr[m][i] = ffma2(wf[i], hh, yr[m][i]);
                }
            }
        }
        __syncthreads();   // the slot is free again
        if (t == 0 && j + kRowStages < nst) rs.issue(j + kRowStages);
    }
    if (failed_at >= 0) {
        if (t == 0) {
            atomicOr(p.ctl + kCtlStatus, kStatusTimeout);
            rs.drain(failed_at);
        }
        return;
    }
    if (in && nst > 0) {
#pragma unroll
        for (int m = 0; m < MB; ++m) {
            if (m < p.M) {
                float *dst = p.out + (size_t)m * p.H + 8 * t;
                const float2 a = unpack2(yr[m][0]), b = unpack2(yr[m][1]);
                const float2 c = unpack2(yr[m][2]), d = unpack2(yr[m][3]);
                red_add_v4(dst, a.x, a.y, b.x, b.y);
                red_add_v4(dst + 4, c.x, c.y, d.x, d.y);
            }
        }
    }
}

}  // namespace
}  // namespace tc

bool union_path_ok(int H, int B) { return B <= tc::kMaxUnion && H <= 8 * tc::kRowThreads; }

// Launches the union list and the union up and down projections after the
// gate-only kernel (see gemm_tc.cu).
cudaError_t launch_union_tail(const sats_layer *layer, int B, const uint16_t *xa, const uint16_t *xlo,
                              const uint8_t *uflag, int32_t *ulist, int32_t *ucount, const float *a_keep, int lda,
                              float *u, int ldu, float *out, int *ctl, cudaStream_t stream)
{
    using namespace tc;
    const int H = layer->H, N = layer->N;
    cudaError_t e = launch_pdl_threads(union_list_kernel, dim3(1), 1024, stream, uflag, N, ulist, ucount);
    if (e != cudaSuccess) return e;
    UnionRowParams rp{};
    rp.w_ud = layer->w_ud;
    rp.ulist = ulist;
    rp.ucount = ucount;
    rp.xa = xa;
    rp.xlo = xlo;
    rp.a_keep = a_keep;
    rp.lda = lda;
    rp.u = u;
    rp.ldu = ldu;
    rp.out = out;
    rp.M = B;
    rp.H = H;
    rp.ctl = ctl;
    const size_t ring = (size_t)kRowStages * kRowsPerStage * H * 2;
    const dim3 grid(sm_count());
    static std::atomic<int> cfg_u4[64], cfg_u8[64], cfg_d4[64], cfg_d8[64];
    if (B <= 4) {
        if ((e = set_smem(union_up_rows_kernel<4>, ring, cfg_u4)) != cudaSuccess) return e;
        if ((e = set_smem(union_down_rows_kernel<4>, ring, cfg_d4)) != cudaSuccess) return e;
        e = launch_pdl_cfg(union_up_rows_kernel<4>, grid, kRowThreads, ring, stream, rp);
        if (e == cudaSuccess) e = launch_pdl_cfg(union_down_rows_kernel<4>, grid, kRowThreads, ring, stream, rp);
        return e;
    }
    if ((e = set_smem(union_up_rows_kernel<8>, ring, cfg_u8)) != cudaSuccess) return e;
    if ((e = set_smem(union_down_rows_kernel<8>, ring, cfg_d8)) != cudaSuccess) return e;
    e = launch_pdl_cfg(union_up_rows_kernel<8>, grid, kRowThreads, ring, stream, rp);
    if (e == cudaSuccess) e = launch_pdl_cfg(union_down_rows_kernel<8>, grid, kRowThreads, ring, stream, rp);
    return e;
}

}  // namespace sats
