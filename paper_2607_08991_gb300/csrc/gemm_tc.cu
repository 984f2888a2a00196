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
// the same accumulator, so that the gate values keep ~fp32 accuracy.  h goes
// to the second GEMM the same way, as a bf16 high part and a bf16 low part
// (about 16 significant bits), so that errors do not build up along a stack.
// (Rounding h, or x for the up projection, to bf16 alone was measured to put a
// Llama-shaped layer's output 2.9e-2 off the fp64 result in the worst element,
// beyond the 2e-2 output tolerance, so both GEMMs keep both parts.)
//
// Routing (Sec. 3.2, Fig. 2): with the routing kernel's permutation (base-path
// tokens first, n_dense of them, read on the device, so no host round trip),
// row i of the packed activations is token perm[i], rows below n_dense take
// threshold 0, and outputs, keep traces and kept lists go back to token perm[i].
//
// Two orientations:
//  - skinny (M <= 256 tokens, 224 with fp32 activations; bandwidth-bound): the
//    weights are the MMA's A operand (128 rows: neurons, or hidden units for the
//    down projection) and the tokens its N dimension, so no MMA row is spent on
//    absent tokens.  The
//    down projection splits its 64-neuron K blocks evenly over one CTA per SM
//    and adds partial sums into y with L2 reductions.
//  - wide (prefill): tokens are the A operand in tiles of 128, the weights the
//    B operand (up to 128 neurons' gate and up rows, gathered from the packed
//    tiles); both kernels are persistent, and CTAs that run together share
//    weight tiles through L2.  The down projection splits the neuron range so
//    that its units even out over the SMs, and adds every unit into the output.
// The weights are read from tile-contiguous copies made at layer creation
// (gu_blk, wd_blk), so that every TMA box is one contiguous DRAM read.
//
// Kernel layout (64 + 128 G threads): warp 0 lane 0 issues the TMA loads, warp 1
// owns the TMEM allocation and lane 0 issues the MMAs, warps 2 .. 4 G + 1 run the
// epilogue in G groups of four (warp w reads TMEM lanes 32 (w mod 4) .. 32 (w mod
// 4) + 31; the groups split the accumulator's columns; G = 1 in the down kernel of
// batched decode, up to six in its gate/up kernel, four in the prefill kernels).
// Every wait is bounded in time and sets the status word when it gives up.
#include "tc_common.cuh"

namespace sats {
namespace tc {
namespace {

// ---------------------------------------------------------------------- activations
// Row m of X = row perm[m] of x (row m without a permutation), fp32, optionally
// RMS-normalised with gain w -> bf16 hi + lo.  Thread t holds the float4 vectors
// t, t + 256, ... of the row in registers (H <= 8 * 4 * 256); the gains, a layer
// constant, are read before the dependency wait.
constexpr int kSplitVec = kMaxH / (4 * 256);

__global__ void __launch_bounds__(256) split_kernel(const float *__restrict__ x, int H, const float *__restrict__ w,
                                                    float eps, uint16_t *__restrict__ hi, uint16_t *__restrict__ lo,
                                                    const int32_t *__restrict__ perm)
{
    const int H4 = H >> 2, t = threadIdx.x;
    float4 wv[kSplitVec];
#pragma unroll
    for (int k = 0; k < kSplitVec; ++k) {
        const int i = t + 256 * k;
        wv[k] = (w && i < H4) ? reinterpret_cast<const float4 *>(w)[i] : make_float4(1.f, 1.f, 1.f, 1.f);
    }
    grid_dependency_wait();   // x may be the residual written by the preceding kernel
    grid_launch_dependents();
    const int m = blockIdx.x;
    const float4 *xr = reinterpret_cast<const float4 *>(x + (size_t)(perm ? perm[m] : m) * H);
    float4 xv[kSplitVec];
    float s = 0.f;
#pragma unroll
    for (int k = 0; k < kSplitVec; ++k) {
        const int i = t + 256 * k;
        xv[k] = i < H4 ? xr[i] : make_float4(0.f, 0.f, 0.f, 0.f);
        s = fmaf(xv[k].x, xv[k].x, fmaf(xv[k].y, xv[k].y, fmaf(xv[k].z, xv[k].z, fmaf(xv[k].w, xv[k].w, s))));
    }
    float inv = 1.0f;
    if (w) {
        __shared__ float red[8];
        s = warp_sum(s);
        if ((t & 31) == 0) red[t >> 5] = s;
        __syncthreads();
        float tot = 0.f;
        for (int i = 0; i < 8; ++i) tot += red[i];
        inv = 1.0f / sqrtf(tot / (float)H + eps);
    }
#pragma unroll
    for (int k = 0; k < kSplitVec; ++k) {
        const int i = t + 256 * k;
        if (i >= H4) break;
        const float v[4] = {xv[k].x * inv * wv[k].x, xv[k].y * inv * wv[k].y, xv[k].z * inv * wv[k].z,
                            xv[k].w * inv * wv[k].w};
        uint16_t hb[4], lb[4];
#pragma unroll
        for (int e = 0; e < 4; ++e) {
            hb[e] = bf16_bits(v[e]);
            lb[e] = bf16_bits(v[e] - __uint_as_float((uint32_t)hb[e] << 16));
        }
        reinterpret_cast<uint2 *>(hi + (size_t)m * H)[i] =
            make_uint2((uint32_t)hb[0] | ((uint32_t)hb[1] << 16), (uint32_t)hb[2] | ((uint32_t)hb[3] << 16));
        reinterpret_cast<uint2 *>(lo + (size_t)m * H)[i] =
            make_uint2((uint32_t)lb[0] | ((uint32_t)lb[1] << 16), (uint32_t)lb[2] | ((uint32_t)lb[3] << 16));
    }
}

// ---------------------------------------------------------------------- weight tiles
// Tiles are stored exactly as the MMA reads them from shared memory: rows of
// 128 bytes whose 16-byte chunks are permuted by the 128-byte swizzle (chunk c
// of row r at position c ^ (r mod 8)), so that one bulk copy of a whole tile to
// a 1024-byte aligned address yields a valid SWIZZLE_128B K-major operand.
__device__ __forceinline__ size_t swizzled_chunk(size_t row_elem_base, int r, int chunk)
{
    return row_elem_base + (size_t)((chunk ^ (r & 7)) * 8);
}

// gu_blk[t][kb][g][r][.] holds (g ? W_up : W_gate)[k][n] for n = t R + r and
// k = kb 64 + c at chunk c / 8 (swizzled), read from wg_t [N][H] and the W_up
// half of w_ud [N][2H].  One thread per 16-byte chunk (H is a multiple of 8).
__global__ void pack_gu_kernel(const uint16_t *__restrict__ wg_t, const uint16_t *__restrict__ w_ud, int H, int N,
                               int R, int KBh, size_t total8, uint16_t *__restrict__ dst)
{
    for (size_t i = blockIdx.x * (size_t)blockDim.x + threadIdx.x; i < total8; i += (size_t)gridDim.x * blockDim.x) {
        const int chunk = (int)(i % 8), c = chunk * 8;
        size_t rest = i / 8;
        const int r = (int)(rest % R);
        rest /= R;
        const int g = (int)(rest % 2);
        rest /= 2;
        const int kb = (int)(rest % KBh);
        const int t = (int)(rest / KBh);
        const int n = t * R + r, k = kb * BK + c;
        uint4 v = make_uint4(0u, 0u, 0u, 0u);
        if (n < N && k < H)
            v = *reinterpret_cast<const uint4 *>(g ? w_ud + (size_t)n * 2 * H + k : wg_t + (size_t)n * H + k);
        // row g R + r of the tile; R is a multiple of 16, so its swizzle phase is r mod 8
        *reinterpret_cast<uint4 *>(dst + swizzled_chunk((i / 8) * BK, r, chunk)) = v;
    }
}

// wd_blk[d][kb][r][.] holds W_down[n][h] for n = kb 64 + c, h = d 128 + r at
// chunk c / 8 (swizzled); W_down row n is the second half of w_ud row n.  One
// CTA per (kb, d) tile, through shared memory so that both sides are read and
// written in rows.
__global__ void __launch_bounds__(256) pack_wd_kernel(const uint16_t *__restrict__ w_ud, int H, int N, int KBn,
                                                      uint16_t *__restrict__ dst)
{
    __shared__ uint16_t tile[BK][BM + 2];
    const int kb = blockIdx.x, d = blockIdx.y;
    for (int i = threadIdx.x; i < BK * BM; i += 256) {
        const int c = i / BM, r = i % BM;
        const int n = kb * BK + c, h = d * BM + r;
        tile[c][r] = (n < N && h < H) ? w_ud[(size_t)n * 2 * H + H + h] : (uint16_t)0;
    }
    __syncthreads();
    uint16_t *out = dst + ((size_t)d * KBn + kb) * BM * BK;
    for (int i = threadIdx.x; i < BM * BK; i += 256) {
        const int r = i / BK, c = i % BK;
        out[swizzled_chunk((size_t)r * BK, r, c / 8) + (c % 8)] = tile[c][r];
    }
}

// ---------------------------------------------------------------------- skinny gate + up
struct SkinnyGuParams {
    const uint16_t *w;            // gu_blk
    int M, N, R, KBh, NT;
    int split;                    // 1: two B operands (bf16 hi and lo parts of fp32 x)
    int merge;                    // split and NT <= 128: one MMA of N = 2 NT over both parts
    float t_l;                    // threshold of sparse-path tokens
    const uint8_t *dense_flags;   // [M] (1 = base path, threshold 0) or nullptr
    const int32_t *perm;          // routed order: row j is token perm[j], rows j < *n_dense on the base path; or nullptr
    const int32_t *n_dense;
    uint16_t *hact;               // [M][ldh] bf16: h rounded to bf16
    uint16_t *hact_lo;            // [M][ldh] bf16: h minus that rounding
    int ldh;
    uint8_t *keep;                // [M][keep_stride] or nullptr
    int keep_stride;
    uint8_t *keep_trace;          // [M][N] or nullptr
    int *ctl;
    float *zero;                  // y [M][H] to clear for the down projection's additions, or nullptr
    int zero_count;               // M H (a multiple of 8)
    // gate-only mode (the union path): no up tile; the epilogue writes a_keep and the union flags
    int gate_only;
    float *a_keep;                // [M][ldh] fp32: keep ? SiLU(g) : 0
    uint8_t *uflag;               // [N]: 1 if any token keeps the neuron
    int stages, stage_bytes, a_bytes, x_bytes;
    int ring_bytes;               // stages * stage_bytes + room for the last up tile's 128-row read
    uint32_t tmem_cols;
};

// One tile of R neurons (gate and up) against all M tokens: D[r][j] in TMEM
// lane r, column j (gate) and NT + j (up).  Grid: tc_T CTAs.  In gate-only mode
// only the gate rows are read and multiplied.  The epilogue runs once all MMAs
// are done, on G groups of four warps (blockDim 64 + 128 G): group g takes the
// 16-token column blocks g, g + G, ... of every row (G = 1 in gate-only mode).
__global__ void __launch_bounds__(kSkinnyMaxThreads, 1)
    gu_skinny_kernel(const __grid_constant__ CUtensorMap tmX, const __grid_constant__ CUtensorMap tmX2,
                     const SkinnyGuParams p)
{
    extern __shared__ uint8_t smem_raw[];
    uint8_t *ring = align1024(smem_raw);
    uint64_t *full = reinterpret_cast<uint64_t *>(ring + p.ring_bytes);
    uint64_t *empty = full + kMaxStages;
    uint64_t *acc_full = empty + kMaxStages;
    uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(acc_full + 1);
    __shared__ int abort_flag, issued_s, consumed_s;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int t = blockIdx.x, R = p.R, NT = p.NT, S = p.stages;
    const int NX = p.merge ? 2 * NT : NT;   // accumulator columns per matrix: tokens, or their high then low parts

    if (threadIdx.x == 0) {
        for (int s = 0; s < S; ++s) {
            mbar_init(&full[s], 1);
            mbar_init(&empty[s], 1);
        }
        mbar_init(acc_full, 1);
        abort_flag = 0;
        issued_s = 0;
        consumed_s = 0;
        mbar_init_fence();
    }
    if (warp == 1) tmem_alloc(tmem_slot, p.tmem_cols);
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_slot;
    grid_launch_dependents();   // the down projection may start prefetching its weights

    if (warp == 0 && lane == 0) {
        const uint32_t w_bytes = (uint32_t)((p.gate_only ? 1 : 2) * R * kTileBytes);
        const uint32_t load_bytes = w_bytes + (uint32_t)(p.x_bytes * (p.split ? 2 : 1));
        const uint64_t policy = l2_policy_evict_first();   // each weight tile is read by this CTA only
        // the weight tiles do not depend on the preceding kernel: start them before waiting for it
        const int npre = p.KBh < S ? p.KBh : S;
        for (int i = 0; i < npre; ++i) {
            mbar_arrive_expect_tx(&full[i], load_bytes);
            bulk_load(ring + (size_t)i * p.stage_bytes, p.w + (size_t)(t * p.KBh + i) * 2 * R * BK, w_bytes, &full[i],
                      policy);
        }
        grid_dependency_wait();   // x (and this call's buffers) may belong to the preceding kernel
        int kb = 0;
        for (int s = 0, ph = 0; kb < p.KBh; ++kb) {
            uint8_t *st = ring + (size_t)s * p.stage_bytes;
            if (kb >= npre) {
                if (!mbar_wait(&empty[s], (uint32_t)ph ^ 1u, &abort_flag)) { set_timeout(p.ctl, &abort_flag); break; }
                mbar_arrive_expect_tx(&full[s], load_bytes);
                bulk_load(st, p.w + (size_t)(t * p.KBh + kb) * 2 * R * BK, w_bytes, &full[s], policy);
            }
            tma_load(st + p.a_bytes, &tmX, kb * BK, 0, &full[s]);
            if (p.split) tma_load(st + p.a_bytes + p.x_bytes, &tmX2, kb * BK, 0, &full[s]);
            if (++s == S) { s = 0; ph ^= 1; }
        }
        issued_s = kb;   // a break happens only before stage kb's loads are issued (kb >= npre)
    } else if (warp == 1 && lane == 0) {
        // x's high and low parts sit back to back in the stage (one 2 NT-row tile): merged,
        // one MMA of N = 2 NT covers both, its two column halves summed in the epilogue;
        // otherwise (N would pass 256) a second MMA adds the low part into the same columns
        const uint32_t idesc = instr_desc(BM, NX);
        int kb = 0;
        for (int s = 0, ph = 0; kb < p.KBh; ++kb) {
            if (!mbar_wait(&full[s], (uint32_t)ph, &abort_flag)) { set_timeout(p.ctl, &abort_flag); break; }
            tc_fence_after();
            const uint32_t st = smem_addr(ring + (size_t)s * p.stage_bytes);
            const uint32_t xa = st + p.a_bytes;
#pragma unroll
            for (int kk = 0; kk < BK / 16; ++kk) {
                const uint32_t acc = (kb | kk) ? 1u : 0u;
                const uint64_t ag = smem_desc(st + kk * 32);
                const uint64_t au = smem_desc(st + R * kTileBytes + kk * 32);
                const uint64_t b = smem_desc(xa + kk * 32);
                mma_bf16(tmem, ag, b, idesc, acc);
                if (!p.gate_only) mma_bf16(tmem + NX, au, b, idesc, acc);
                if (p.split && !p.merge) {
                    const uint64_t b2 = smem_desc(xa + p.x_bytes + kk * 32);
                    mma_bf16(tmem, ag, b2, idesc, 1u);
                    if (!p.gate_only) mma_bf16(tmem + NX, au, b2, idesc, 1u);
                }
            }
            mma_commit(&empty[s]);
            if (++s == S) { s = 0; ph ^= 1; }
        }
        consumed_s = kb;
        mma_commit(acc_full);
    } else if (warp >= 2) {
        grid_dependency_wait();   // y, h and the keep bytes may still be in use by the preceding kernel
        if (p.zero) {
            // this CTA's share of y, cleared for the down projection's additions
            const int per = (((p.zero_count + (int)gridDim.x - 1) / (int)gridDim.x) + 7) & ~7;
            const int z0 = (int)blockIdx.x * per, z1 = min(p.zero_count, z0 + per);
            float4 *z = reinterpret_cast<float4 *>(p.zero);
            for (int i = z0 / 4 + (int)threadIdx.x - 64; i < z1 / 4; i += (int)blockDim.x - 64)
                z[i] = make_float4(0.f, 0.f, 0.f, 0.f);
        }
        // epilogue: thread = neuron r of the tile, columns = tokens (the base-path count is read
        // while the MMAs run)
        const int nd = p.perm ? *p.n_dense : 0;
        const bool ok = mbar_wait(acc_full, 0u, &abort_flag);
        tc_fence_after();
        const int lb = 32 * (warp & 3);
        const int G = ((int)blockDim.x - 64) / 128, grp = (warp - 2) >> 2;
        const int r = lb + lane, n = t * R + r;
        const bool row_ok = ok && r < R && n < p.N;
        bool any = false;   // gate-only mode: some token keeps neuron n
        for (int c0 = 16 * grp; c0 < NT; c0 += 16 * G) {
            float g[16], u[16], lo[16];
            tmem_ld16(tmem + ((uint32_t)lb << 16) + (uint32_t)c0, g);
            if (p.merge) {
                tmem_ld16(tmem + ((uint32_t)lb << 16) + (uint32_t)(NT + c0), lo);
                tmem_ld_wait();
#pragma unroll
                for (int e = 0; e < 16; ++e) g[e] += lo[e];
            }
            if (p.gate_only) {
                tmem_ld_wait();
                if (!row_ok) continue;
#pragma unroll
                for (int e = 0; e < 16; ++e) {
                    const int j = c0 + e;
                    if (j < p.M) {
                        const float a = g[e] / (1.0f + expf(-g[e]));   // SiLU, Eq. 2
                        const bool keep = fabsf(a) >= p.t_l;            // Eqs. 4-5
                        any = any || keep;
                        p.a_keep[(size_t)j * p.ldh + n] = keep ? a : 0.f;
                        if (p.keep) p.keep[(size_t)j * p.keep_stride + n] = keep ? 1 : 0;
                        if (p.keep_trace) p.keep_trace[(size_t)j * p.N + n] = keep ? 1 : 0;
                    }
                }
                continue;
            }
            tmem_ld16(tmem + ((uint32_t)lb << 16) + (uint32_t)(NX + c0), u);
            if (p.merge) {
                tmem_ld16(tmem + ((uint32_t)lb << 16) + (uint32_t)(NX + NT + c0), lo);
                tmem_ld_wait();
#pragma unroll
                for (int e = 0; e < 16; ++e) u[e] += lo[e];
            }
            tmem_ld_wait();
            if (!row_ok) continue;
#pragma unroll
            for (int e = 0; e < 16; ++e) {
                const int j = c0 + e;
                if (j < p.M) {
                    const bool base = p.perm ? j < nd : (p.dense_flags && p.dense_flags[j]);
                    const float thr = base ? 0.f : p.t_l;
                    const float a = g[e] / (1.0f + expf(-g[e]));   // SiLU, Eq. 2
                    const bool keep = fabsf(a) >= thr;             // Eqs. 4-5
                    const float h = keep ? a * u[e] : 0.f;
                    const uint16_t hb = bf16_bits(h);
                    p.hact[(size_t)j * p.ldh + n] = hb;
                    p.hact_lo[(size_t)j * p.ldh + n] = bf16_bits(h - __uint_as_float((uint32_t)hb << 16));
                    if (p.keep) p.keep[(size_t)j * p.keep_stride + n] = keep ? 1 : 0;
                    if (p.keep_trace) p.keep_trace[(size_t)(p.perm ? p.perm[j] : j) * p.N + n] = keep ? 1 : 0;
                }
            }
        }
        if (p.gate_only && row_ok) p.uflag[n] = any ? 1 : 0;
        tc_fence_before();
    }
    __syncthreads();
    if (abort_flag && threadIdx.x == 0) drain_after_abort(full, S, issued_s, consumed_s, acc_full);
    __syncthreads();
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc(tmem, p.tmem_cols);
    }
}

// ---------------------------------------------------------------------- skinny down
struct SkinnyDownParams {
    const uint16_t *w;            // wd_blk
    int M, H, NT, KBn, units;     // units = tc_dt * KBn (hidden tile, neuron block) pairs
    float *out;                   // [M][H] fp32, added to with L2 reductions
    const int32_t *perm;          // routed order: column j of h is token perm[j]; or nullptr
    int *ctl;
    int stages, stage_bytes, a_bytes;
    int merge;                    // NT <= 128: one MMA of N = 2 NT over h's high and low parts
    uint32_t tmem_cols;           // two accumulators of NX columns (NX = 2 NT merged, else NT)
};

// CTA c handles units [c U / G, (c+1) U / G) in order; consecutive units of one
// hidden tile form a segment accumulated in TMEM (two buffers, so that the
// epilogue of one segment overlaps the MMAs of the next) and added into y.
// Unit u's weight tile is tile u of wd_blk; h arrives as its high and low bf16
// parts, one tile of 2 NT rows: merged, one MMA per step whose column halves the
// epilogue sums; otherwise two MMAs into the same accumulator.
__global__ void __launch_bounds__(kThreads, 1)
    down_skinny_kernel(const __grid_constant__ CUtensorMap tmH, const __grid_constant__ CUtensorMap tmH2,
                       const SkinnyDownParams p)
{
    extern __shared__ uint8_t smem_raw[];
    uint8_t *ring = align1024(smem_raw);
    uint64_t *full = reinterpret_cast<uint64_t *>(ring + (size_t)p.stages * p.stage_bytes);
    uint64_t *empty = full + kMaxStages;
    uint64_t *acc_full = empty + kMaxStages;   // [2]
    uint64_t *acc_empty = acc_full + 2;        // [2]
    uint64_t *mma_done = acc_empty + 2;        // every MMA of this CTA has completed
    uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(mma_done + 1);
    __shared__ int abort_flag, issued_s, consumed_s;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int S = p.stages, NT = p.NT, KBn = p.KBn;
    const int NX = p.merge ? 2 * NT : NT;
    const int u0 = (int)((long long)blockIdx.x * p.units / gridDim.x);
    const int u1 = (int)((long long)(blockIdx.x + 1) * p.units / gridDim.x);
    const int nu = u1 - u0;

    if (threadIdx.x == 0) {
        for (int s = 0; s < S; ++s) {
            mbar_init(&full[s], 1);
            mbar_init(&empty[s], 1);
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(&acc_full[b], 1);
            mbar_init(&acc_empty[b], 128);
        }
        mbar_init(mma_done, 1);
        abort_flag = 0;
        issued_s = 0;
        consumed_s = 0;
        mbar_init_fence();
    }
    if (warp == 1) tmem_alloc(tmem_slot, p.tmem_cols);
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_slot;
    grid_launch_dependents();   // the next call's kernels may start their prologue as SMs free up

    if (warp == 0 && lane == 0) {
        const uint32_t w_bytes = (uint32_t)(BM * kTileBytes);
        const uint32_t load_bytes = w_bytes + (uint32_t)(2 * NT * kTileBytes);
        const uint64_t policy = l2_policy_evict_first();
        // the weight tiles do not depend on the preceding kernel: start them first
        const int npre = nu < S ? nu : S;
        for (int i = 0; i < npre; ++i) {
            mbar_arrive_expect_tx(&full[i], load_bytes);
            bulk_load(ring + (size_t)i * p.stage_bytes, p.w + (size_t)(u0 + i) * BM * BK, w_bytes, &full[i], policy);
        }
        grid_dependency_wait();   // h is written by the preceding gate/up kernel
        int i = 0;
        for (int s = 0, ph = 0; i < nu; ++i) {
            const int u = u0 + i;
            uint8_t *st = ring + (size_t)s * p.stage_bytes;
            if (i >= npre) {
                if (!mbar_wait(&empty[s], (uint32_t)ph ^ 1u, &abort_flag)) { set_timeout(p.ctl, &abort_flag); break; }
                mbar_arrive_expect_tx(&full[s], load_bytes);
                bulk_load(st, p.w + (size_t)u * BM * BK, w_bytes, &full[s], policy);
            }
            tma_load(st + p.a_bytes, &tmH, (u % KBn) * BK, 0, &full[s]);
            tma_load(st + p.a_bytes + NT * kTileBytes, &tmH2, (u % KBn) * BK, 0, &full[s]);
            if (++s == S) { s = 0; ph ^= 1; }
        }
        issued_s = i;   // a break happens only before stage i's loads are issued (i >= npre)
    } else if (warp == 1 && lane == 0) {
        const uint32_t idesc = instr_desc(BM, NX);
        int i = 0, q = 0;
        int s = 0, ph = 0;
        for (int u = u0; u < u1 && !abort_flag;) {
            const int seg_end = min(u1, (u / KBn + 1) * KBn);
            const int buf = q & 1;
            if (!mbar_wait(&acc_empty[buf], (uint32_t)((q >> 1) & 1) ^ 1u, &abort_flag)) {
                set_timeout(p.ctl, &abort_flag);
                break;
            }
            tc_fence_after();
            bool first = true;
            for (; u < seg_end; ++u, ++i) {
                if (!mbar_wait(&full[s], (uint32_t)ph, &abort_flag)) { set_timeout(p.ctl, &abort_flag); break; }
                tc_fence_after();
                const uint32_t st = smem_addr(ring + (size_t)s * p.stage_bytes);
#pragma unroll
                for (int kk = 0; kk < BK / 16; ++kk) {
                    const uint64_t w = smem_desc(st + kk * 32);
                    mma_bf16(tmem + (uint32_t)(buf * NX), w, smem_desc(st + p.a_bytes + kk * 32), idesc,
                             (first && kk == 0) ? 0u : 1u);
                    if (!p.merge)
                        mma_bf16(tmem + (uint32_t)(buf * NX), w, smem_desc(st + p.a_bytes + NT * kTileBytes + kk * 32),
                                 idesc, 1u);
                }
                first = false;
                mma_commit(&empty[s]);
                if (++s == S) { s = 0; ph ^= 1; }
            }
            mma_commit(&acc_full[buf]);
            ++q;
        }
        consumed_s = i;
        mma_commit(mma_done);
    } else if (warp >= 2) {
        // a warp's 32 rows x 16 tokens go through shared memory, so that each lane adds four
        // vectors of four consecutive hidden units of one token (vector reductions in L2)
        __shared__ float tr[4][16][33];
        __shared__ int tok_s[kMaxSkinny];   // output row of each column (the routing permutation, read early)
        float(*T)[33] = tr[warp & 3];
        grid_dependency_wait();   // (the permutation is older than the preceding kernel; its MMAs run meanwhile)
        for (int j = (int)threadIdx.x - 64; j < NT; j += (int)blockDim.x - 64)
            tok_s[j] = j < p.M ? (p.perm ? p.perm[j] : j) : 0;
        named_barrier(1, (int)blockDim.x - 64);   // the epilogue warps only
        const int lb = 32 * (warp & 3);
        const int te = lane >> 1, r0 = (lane & 1) * 16;   // this lane's token in the block, first row
        int q = 0;
        for (int u = u0; u < u1; ++q) {
            const int d = u / KBn;
            const int seg_end = min(u1, (d + 1) * KBn);
            const int buf = q & 1;
            const bool ok = mbar_wait(&acc_full[buf], (uint32_t)((q >> 1) & 1), &abort_flag);
            tc_fence_after();
            const int h0 = d * BM + lb + r0;
            for (int c0 = 0; c0 < NT; c0 += 16) {
                float v[16], lo[16];
                tmem_ld16(tmem + ((uint32_t)lb << 16) + (uint32_t)(buf * NX + c0), v);
                if (p.merge) {
                    tmem_ld16(tmem + ((uint32_t)lb << 16) + (uint32_t)(buf * NX + NT + c0), lo);
                    tmem_ld_wait();
#pragma unroll
                    for (int e = 0; e < 16; ++e) v[e] += lo[e];
                }
                tmem_ld_wait();
#pragma unroll
                for (int e = 0; e < 16; ++e) T[e][lane] = v[e];
                __syncwarp();
                const int j = c0 + te;
                if (ok && j < p.M) {
                    float *dst = p.out + (size_t)tok_s[j] * p.H + h0;
#pragma unroll
                    for (int k = 0; k < 4; ++k)   // H is a multiple of 8: a vector is in range or not at all
                        if (h0 + 4 * k < p.H)
                            red_add_v4(dst + 4 * k, T[te][r0 + 4 * k], T[te][r0 + 4 * k + 1], T[te][r0 + 4 * k + 2],
                                       T[te][r0 + 4 * k + 3]);
                }
                __syncwarp();
            }
            tc_fence_before();
            mbar_arrive(&acc_empty[buf]);
            if (!ok) break;
            u = seg_end;
        }
    }
    __syncthreads();
    if (threadIdx.x == 0) {
        // the arrival on mma_done must land before this CTA's shared memory is released
        int never = 0;
        if (abort_flag)
            for (int k = consumed_s; k < issued_s; ++k) mbar_wait(&full[k % S], (uint32_t)((k / S) & 1), &never);
        mbar_wait(mma_done, 0u, &never);
    }
    __syncthreads();
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc(tmem, p.tmem_cols);
    }
}

// ---------------------------------------------------------------------- wide gate + up
struct WideGuParams {
    const uint16_t *w;            // gu_blk: tiles of R neurons
    int M, N, R, KBh, T;          // T: tiles of gu_blk
    int Rw;                       // neurons per wide tile (a multiple of 16, <= 128): MMA N = 2 Rw
    int mtiles, tiles;            // token tiles; tiles = mtiles * ceil(N / Rw)
    int split;
    float t_l;
    const uint8_t *dense_flags;
    const int32_t *perm;          // routed order (see the file comment) or nullptr
    const int32_t *n_dense;
    uint16_t *hact, *hact_lo;     // h as bf16 high and low parts
    int ldh;
    uint8_t *keep;
    int keep_stride;              // a multiple of 16
    uint8_t *keep_trace;
    int *ctl;
    float *zero;                  // y [M][H] to clear for the down projection's additions, or nullptr
    long long zero_count;         // M H (a multiple of 8; M H can exceed 2^31 at prefill sizes)
    int stages, stage_bytes;
    uint32_t tmem_cols;           // two accumulator buffers of 2 Rw columns
};

// Persistent: CTA c takes tiles c, c + G, c + 2G, ... of 128 tokens x Rw
// neurons; tile q covers token tile q mod mtiles of neuron tile q / mtiles, so
// the CTAs running together share few weight tiles and read them through L2.
// A stage holds the x tile(s), then the tile's Rw gate rows and Rw up rows,
// gathered from gu_blk's tiles of R neurons: every operand byte passes through
// shared memory twice (written by the copy engine, read by the MMA), and that
// traffic rather than the MMA rate paces the loop, so a wider weight tile (up
// to 128 neurons, MMA N = 256) puts more work on each byte.
// Per tile, D[m][c] accumulates in TMEM lane m, column b 2Rw + c (gate) and
// b 2Rw + Rw + c (up), b alternating between tiles so that one tile's epilogue
// overlaps the next tile's MMAs; the load ring runs across tile boundaries.
__global__ void __launch_bounds__(kWideMaxThreads, 1)
    gu_wide_kernel(const __grid_constant__ CUtensorMap tmX, const __grid_constant__ CUtensorMap tmX2,
                   const WideGuParams p)
{
    constexpr int kA = BM * kTileBytes;
    extern __shared__ uint8_t smem_raw[];
    uint8_t *ring = align1024(smem_raw);
    uint64_t *full = reinterpret_cast<uint64_t *>(ring + (size_t)p.stages * p.stage_bytes);
    uint64_t *empty = full + kMaxStages;
    uint64_t *acc_full = empty + kMaxStages;   // [2]
    uint64_t *acc_empty = acc_full + 2;        // [2]
    uint64_t *mma_done = acc_empty + 2;
    uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(mma_done + 1);
    __shared__ int abort_flag, issued_s, consumed_s;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int R = p.R, Rw = p.Rw, S = p.stages, KBh = p.KBh;
    const int wofs = kA * (p.split ? 2 : 1);

    if (threadIdx.x == 0) {
        for (int s = 0; s < S; ++s) {
            mbar_init(&full[s], 1);
            mbar_init(&empty[s], 1);
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(&acc_full[b], 1);
            mbar_init(&acc_empty[b], blockDim.x - 64);   // every epilogue thread
        }
        mbar_init(mma_done, 1);
        abort_flag = 0;
        issued_s = 0;
        consumed_s = 0;
        mbar_init_fence();
    }
    if (warp == 1) tmem_alloc(tmem_slot, p.tmem_cols);
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_slot;

    if (warp == 0 && lane == 0) {
        // a wide tile's gate (and up) rows lie in at most two tiles of gu_blk: la rows from row r0
        // of tile t0, then lb rows from the start of tile t0 + 1 (the host keeps Rw - gcd(Rw, R)
        // <= R).  R and Rw are multiples of 16, so each piece keeps its rows' swizzle phase.  Rows
        // past the last packed tile are not loaded: their columns of D belong to neurons >= N,
        // which the epilogue skips.  Offsets in rows of BK elements at K block 0, worked out
        // once per tile: this one thread's per-stage work must stay well below a stage's MMAs.
        struct Pieces {
            size_t a, b;
            int la, lb;
        };
        auto pieces_of = [&](int tw) {
            const int n0 = tw * Rw, rows = min(Rw, p.T * R - n0);
            const int t0 = n0 / R, r0 = n0 - t0 * R;
            Pieces w;
            w.la = min(R - r0, rows);
            w.lb = rows - w.la;
            w.a = (size_t)t0 * KBh * 2 * R + r0;
            w.b = (size_t)(t0 + 1) * KBh * 2 * R;
            return w;
        };
        const size_t kb_rows = (size_t)2 * R;   // rows of a gu_blk tile per K block
        // L2 prefetch of the weight stage kWidePrefetch loads ahead (this CTA's own sequence of
        // tiles); of the CTAs that share a weight tile, one asks for each stage, in turn (the CTA
        // of token tile m takes the K blocks kb with (m + kb) mod mtiles = 0), so that the
        // prefetches add the same work to every CTA's load thread
        int pq = blockIdx.x, pkb = 0, prot = 0;
        Pieces pf{};
        auto prefetch_tile = [&]() {
            if (pq >= p.tiles) return;
            prot = pq % p.mtiles;
            pf = pieces_of(pq / p.mtiles);
        };
        prefetch_tile();
        auto prefetch_ahead = [&]() {
            if (pq >= p.tiles) return;
            const bool go = prot == 0;
            if (++prot == p.mtiles) prot = 0;
            if (go) {
                const size_t o = (size_t)pkb * kb_rows;
                for (int g = 0; g < 2; ++g) {
                    bulk_prefetch_l2(p.w + (pf.a + o + g * R) * BK, (uint32_t)(pf.la * kTileBytes));
                    if (pf.lb) bulk_prefetch_l2(p.w + (pf.b + o + g * R) * BK, (uint32_t)(pf.lb * kTileBytes));
                }
            }
            if (++pkb == KBh) {
                pkb = 0;
                pq += gridDim.x;
                prefetch_tile();
            }
        };
        for (int j = 0; j < kWidePrefetch; ++j) prefetch_ahead();
        int i = 0, s = 0, ph = 0;
        bool stop = false;
        for (int q = blockIdx.x; q < p.tiles && !stop; q += gridDim.x) {
            const int m0 = (q % p.mtiles) * BM;
            const Pieces pc = pieces_of(q / p.mtiles);
            const uint32_t load_bytes = (uint32_t)(wofs + 2 * (pc.la + pc.lb) * kTileBytes);
            for (int kb = 0; kb < KBh; ++kb, ++i) {
                if (!mbar_wait(&empty[s], (uint32_t)ph ^ 1u, &abort_flag)) {
                    set_timeout(p.ctl, &abort_flag);
                    stop = true;
                    break;
                }
                uint8_t *st = ring + (size_t)s * p.stage_bytes;
                mbar_arrive_expect_tx(&full[s], load_bytes);
                tma_load(st, &tmX, kb * BK, m0, &full[s]);
                if (p.split) tma_load(st + kA, &tmX2, kb * BK, m0, &full[s]);
                const size_t o = (size_t)kb * kb_rows;
                for (int g = 0; g < 2; ++g) {
                    uint8_t *dst = st + wofs + g * Rw * kTileBytes;
                    bulk_load_shared(dst, p.w + (pc.a + o + g * R) * BK, (uint32_t)(pc.la * kTileBytes), &full[s]);
                    if (pc.lb)
                        bulk_load_shared(dst + pc.la * kTileBytes, p.w + (pc.b + o + g * R) * BK,
                                         (uint32_t)(pc.lb * kTileBytes), &full[s]);
                }
                prefetch_ahead();
                if (++s == S) { s = 0; ph ^= 1; }
            }
        }
        issued_s = i;
    } else if (warp == 1 && lane == 0) {
        // gate rows and up rows are adjacent in the stage: one MMA with N = 2Rw writes the gate
        // accumulator to columns [0, Rw) and the up accumulator to [Rw, 2Rw)
        const uint32_t idesc = instr_desc(BM, 2 * Rw);
        int i = 0, s = 0, ph = 0, it = 0;
        bool stop = false;
        for (int q = blockIdx.x; q < p.tiles && !stop; q += gridDim.x, ++it) {
            const int buf = it & 1;
            if (!mbar_wait(&acc_empty[buf], (uint32_t)((it >> 1) & 1) ^ 1u, &abort_flag)) {
                set_timeout(p.ctl, &abort_flag);
                break;
            }
            tc_fence_after();
            const uint32_t d = tmem + (uint32_t)(buf * 2 * Rw);
            for (int kb = 0; kb < KBh; ++kb, ++i) {
                if (!mbar_wait(&full[s], (uint32_t)ph, &abort_flag)) {
                    set_timeout(p.ctl, &abort_flag);
                    stop = true;
                    break;
                }
                tc_fence_after();
                const uint32_t st = smem_addr(ring + (size_t)s * p.stage_bytes);
                const uint32_t wa = st + wofs;
#pragma unroll
                for (int kk = 0; kk < BK / 16; ++kk) {
                    const uint64_t w = smem_desc(wa + kk * 32);
                    mma_bf16(d, smem_desc(st + kk * 32), w, idesc, (kb | kk) ? 1u : 0u);
                    if (p.split) mma_bf16(d, smem_desc(st + kA + kk * 32), w, idesc, 1u);
                }
                mma_commit(&empty[s]);
                if (++s == S) { s = 0; ph ^= 1; }
            }
            mma_commit(&acc_full[buf]);
        }
        consumed_s = i;
        mma_commit(mma_done);
    } else if (warp >= 2) {
        if (p.zero) {
            // this CTA's share of y, cleared for the down projection's additions while the first
            // tile's MMAs run
            const long long per = ((p.zero_count + gridDim.x - 1) / gridDim.x + 7) & ~7LL;
            const long long z0 = (long long)blockIdx.x * per, z1 = min(p.zero_count, z0 + per);
            float4 *z = reinterpret_cast<float4 *>(p.zero);
            for (long long i = z0 / 4 + (int)threadIdx.x - 64; i < z1 / 4; i += (int)blockDim.x - 64)
                z[i] = make_float4(0.f, 0.f, 0.f, 0.f);
        }
        // epilogue: thread = token row of the tile, 16 neurons at a time; group g of four warps
        // takes the 16-neuron column blocks g, g + G, ...
        const int lb = 32 * (warp & 3);
        const int G = ((int)blockDim.x - 64) / 128, grp = (warp - 2) >> 2;
        const int nd = p.perm ? *p.n_dense : 0;   // the base-path count (routed order), read once
        int it = 0;
        for (int q = blockIdx.x; q < p.tiles; q += gridDim.x, ++it) {
            const int buf = it & 1;
            const int m = (q % p.mtiles) * BM + lb + lane, t = q / p.mtiles;
            const bool ok = mbar_wait(&acc_full[buf], (uint32_t)((it >> 1) & 1), &abort_flag);
            tc_fence_after();
            const bool row_ok = ok && m < p.M;
            float thr = INFINITY;
            if (row_ok) thr = (p.perm ? m < nd : (p.dense_flags && p.dense_flags[m])) ? 0.f : p.t_l;
            const uint32_t dg = tmem + ((uint32_t)lb << 16) + (uint32_t)(buf * 2 * Rw);
            for (int c0 = 16 * grp; c0 < Rw; c0 += 16 * G) {
                float g[16], u[16];
                tmem_ld16(dg + (uint32_t)c0, g);
                tmem_ld16(dg + (uint32_t)(Rw + c0), u);
                tmem_ld_wait();
                const int n = t * Rw + c0;
                if (!row_ok || n >= p.N) continue;
                uint32_t hw[8], lw[8], kw[4] = {0u, 0u, 0u, 0u};
#pragma unroll
                for (int e = 0; e < 16; e += 2) {
                    const float a0 = g[e] / (1.0f + expf(-g[e]));             // SiLU, Eq. 2
                    const float a1 = g[e + 1] / (1.0f + expf(-g[e + 1]));
                    const bool k0 = fabsf(a0) >= thr, k1 = fabsf(a1) >= thr;   // Eqs. 4-5
                    const float h0 = k0 ? a0 * u[e] : 0.f, h1 = k1 ? a1 * u[e + 1] : 0.f;
                    const uint16_t b0 = bf16_bits(h0), b1 = bf16_bits(h1);
                    hw[e / 2] = (uint32_t)b0 | ((uint32_t)b1 << 16);
                    lw[e / 2] = (uint32_t)bf16_bits(h0 - __uint_as_float((uint32_t)b0 << 16)) |
                                ((uint32_t)bf16_bits(h1 - __uint_as_float((uint32_t)b1 << 16)) << 16);
                    kw[e / 4] |= ((k0 ? 1u : 0u) << (8 * (e % 4))) | ((k1 ? 1u : 0u) << (8 * (e % 4) + 8));
                }
                uint16_t *hrow = p.hact + (size_t)m * p.ldh + n;
                uint16_t *lrow = p.hact_lo + (size_t)m * p.ldh + n;
                uint8_t *krow = p.keep ? p.keep + (size_t)m * p.keep_stride + n : nullptr;
                if (n + 16 <= p.N) {   // n is a multiple of 16: 32-byte aligned h, 16-byte aligned keep
                    reinterpret_cast<uint4 *>(hrow)[0] = make_uint4(hw[0], hw[1], hw[2], hw[3]);
                    reinterpret_cast<uint4 *>(hrow)[1] = make_uint4(hw[4], hw[5], hw[6], hw[7]);
                    reinterpret_cast<uint4 *>(lrow)[0] = make_uint4(lw[0], lw[1], lw[2], lw[3]);
                    reinterpret_cast<uint4 *>(lrow)[1] = make_uint4(lw[4], lw[5], lw[6], lw[7]);
                    if (krow) *reinterpret_cast<uint4 *>(krow) = make_uint4(kw[0], kw[1], kw[2], kw[3]);
                } else {
#pragma unroll
                    for (int e = 0; e < 16; ++e) {
                        if (n + e < p.N) {
                            hrow[e] = (uint16_t)(hw[e / 2] >> (16 * (e & 1)));
                            lrow[e] = (uint16_t)(lw[e / 2] >> (16 * (e & 1)));
                            if (krow) krow[e] = (uint8_t)(kw[e / 4] >> (8 * (e & 3)));
                        }
                    }
                }
                if (p.keep_trace) {
                    uint8_t *trow = p.keep_trace + (size_t)(p.perm ? p.perm[m] : m) * p.N + n;
#pragma unroll
                    for (int e = 0; e < 16; ++e)
                        if (n + e < p.N) trow[e] = (uint8_t)(kw[e / 4] >> (8 * (e & 3)));
                }
            }
            tc_fence_before();
            mbar_arrive(&acc_empty[buf]);
            if (!ok) break;
        }
    }
    __syncthreads();
    if (threadIdx.x == 0) {
        // the arrival on mma_done must land before this CTA's shared memory is released
        int never = 0;
        if (abort_flag)
            for (int k = consumed_s; k < issued_s; ++k) mbar_wait(&full[k % S], (uint32_t)((k / S) & 1), &never);
        mbar_wait(mma_done, 0u, &never);
    }
    __syncthreads();
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc(tmem, p.tmem_cols);
    }
}
// ---------------------------------------------------------------------- wide down
struct WideDownParams {
    const uint16_t *w;    // wd_blk
    int M, H, KBn;
    int dtiles;           // 128-row hidden tiles per unit (1 or 2: MMA N = 128 dtiles)
    int mtiles, dcols;    // token tiles; unit columns (tc_dt / dtiles)
    int kb_per_split;     // K blocks of 64 neurons per unit
    int units;            // mtiles * dcols * splits
    float *out;           // [M][H] fp32: every unit adds its partial tile with L2 reductions
    const int32_t *perm;  // routed order: row m of h is token perm[m]; or nullptr
    int *ctl;
    int stages, stage_bytes;
    uint32_t tmem_cols;   // two accumulator buffers of 128 dtiles columns
};

// Persistent: CTA c takes units c, c + G, c + 2G, ...; unit u is the 128-token
// x (128 dtiles)-column tile (u mod mtiles, (u / mtiles) mod dcols) of
// Y = h W_down over the neuron split u / (mtiles dcols).  The splits even out the
// units per CTA (the tile count alone can leave most SMs idle in a last wave),
// and the units that run together share one split's h and weight tiles through
// L2.  h arrives as its high and low bf16 parts (two A tiles); the accumulator
// alternates between two TMEM buffers, so that one unit's epilogue (L2
// reductions into the output rows) overlaps the next unit's MMAs.
__global__ void __launch_bounds__(kWideMaxThreads, 1)
    down_wide_kernel(const __grid_constant__ CUtensorMap tmH, const __grid_constant__ CUtensorMap tmH2,
                     const WideDownParams p)
{
    constexpr int kA = BM * kTileBytes;
    extern __shared__ uint8_t smem_raw[];
    uint8_t *ring = align1024(smem_raw);
    uint64_t *full = reinterpret_cast<uint64_t *>(ring + (size_t)p.stages * p.stage_bytes);
    uint64_t *empty = full + kMaxStages;
    uint64_t *acc_full = empty + kMaxStages;   // [2]
    uint64_t *acc_empty = acc_full + 2;        // [2]
    uint64_t *mma_done = acc_empty + 2;
    uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(mma_done + 1);
    __shared__ int abort_flag, issued_s, consumed_s;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int S = p.stages, BN = BM * p.dtiles, KBn = p.KBn;
    const int per_split = p.mtiles * p.dcols;
    // unit u -> its token tile's first row, first hidden tile and K-block range
    auto unit = [&](int u, int &m0, int &d0, int &kb0, int &kb1) {
        const int z = u / per_split, rem = u - z * per_split;
        m0 = (rem % p.mtiles) * BM;
        d0 = (rem / p.mtiles) * p.dtiles;
        kb0 = z * p.kb_per_split;
        kb1 = min(KBn, kb0 + p.kb_per_split);
    };

    if (threadIdx.x == 0) {
        for (int s = 0; s < S; ++s) {
            mbar_init(&full[s], 1);
            mbar_init(&empty[s], 1);
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(&acc_full[b], 1);
            mbar_init(&acc_empty[b], blockDim.x - 64);   // every epilogue thread
        }
        mbar_init(mma_done, 1);
        abort_flag = 0;
        issued_s = 0;
        consumed_s = 0;
        mbar_init_fence();
    }
    if (warp == 1) tmem_alloc(tmem_slot, p.tmem_cols);
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_slot;

    if (warp == 0 && lane == 0) {
        const uint32_t load_bytes = (uint32_t)(2 * kA + BN * kTileBytes);
        // L2 prefetch kWidePrefetch stages ahead (this CTA's own sequence of units): the weight
        // tiles by the CTAs of the first two token tiles, the h tiles by every fourth unit column;
        // the cursor's unit is decoded once per unit
        int pu = blockIdx.x, pkb = 0, pkb1 = 0, pm0 = 0, pd0 = 0;
        bool pf_w = false, pf_h = false;
        auto prefetch_unit = [&]() {
            if (pu >= p.units) return;
            unit(pu, pm0, pd0, pkb, pkb1);
            pf_w = pm0 < 2 * BM;
            pf_h = (pd0 / p.dtiles) % 4 == 0;
        };
        prefetch_unit();
        auto prefetch_ahead = [&]() {
            if (pu >= p.units) return;
            if (pf_w)
                for (int q = 0; q < p.dtiles; ++q)
                    bulk_prefetch_l2(p.w + ((size_t)(pd0 + q) * KBn + pkb) * BM * BK, (uint32_t)kA);
            if (pf_h) {
                tma_prefetch_l2(&tmH, pkb * BK, pm0);
                tma_prefetch_l2(&tmH2, pkb * BK, pm0);
            }
            if (++pkb == pkb1) {
                pu += gridDim.x;
                prefetch_unit();
            }
        };
        for (int j = 0; j < kWidePrefetch; ++j) prefetch_ahead();
        int i = 0, s = 0, ph = 0;
        bool stop = false;
        for (int u = blockIdx.x; u < p.units && !stop; u += gridDim.x) {
            int m0, d0, kb0, kb1;
            unit(u, m0, d0, kb0, kb1);
            for (int kb = kb0; kb < kb1; ++kb, ++i) {
                if (!mbar_wait(&empty[s], (uint32_t)ph ^ 1u, &abort_flag)) {
                    set_timeout(p.ctl, &abort_flag);
                    stop = true;
                    break;
                }
                uint8_t *st = ring + (size_t)s * p.stage_bytes;
                mbar_arrive_expect_tx(&full[s], load_bytes);
                tma_load(st, &tmH, kb * BK, m0, &full[s]);
                tma_load(st + kA, &tmH2, kb * BK, m0, &full[s]);
                for (int q = 0; q < p.dtiles; ++q)
                    bulk_load_shared(st + 2 * kA + q * kA, p.w + ((size_t)(d0 + q) * KBn + kb) * BM * BK,
                                     (uint32_t)kA, &full[s]);
                prefetch_ahead();
                if (++s == S) { s = 0; ph ^= 1; }
            }
        }
        issued_s = i;
    } else if (warp == 1 && lane == 0) {
        const uint32_t idesc = instr_desc(BM, BN);
        int i = 0, s = 0, ph = 0, it = 0;
        bool stop = false;
        for (int u = blockIdx.x; u < p.units && !stop; u += gridDim.x, ++it) {
            int m0, d0, kb0, kb1;
            unit(u, m0, d0, kb0, kb1);
            const int buf = it & 1;
            if (!mbar_wait(&acc_empty[buf], (uint32_t)((it >> 1) & 1) ^ 1u, &abort_flag)) {
                set_timeout(p.ctl, &abort_flag);
                break;
            }
            tc_fence_after();
            const uint32_t d = tmem + (uint32_t)(buf * BN);
            for (int kb = kb0; kb < kb1; ++kb, ++i) {
                if (!mbar_wait(&full[s], (uint32_t)ph, &abort_flag)) {
                    set_timeout(p.ctl, &abort_flag);
                    stop = true;
                    break;
                }
                tc_fence_after();
                const uint32_t st = smem_addr(ring + (size_t)s * p.stage_bytes);
#pragma unroll
                for (int kk = 0; kk < BK / 16; ++kk) {
                    const uint64_t w = smem_desc(st + 2 * kA + kk * 32);
                    mma_bf16(d, smem_desc(st + kk * 32), w, idesc, (kb > kb0 || kk) ? 1u : 0u);
                    mma_bf16(d, smem_desc(st + kA + kk * 32), w, idesc, 1u);
                }
                mma_commit(&empty[s]);
                if (++s == S) { s = 0; ph ^= 1; }
            }
            mma_commit(&acc_full[buf]);
        }
        consumed_s = i;
        mma_commit(mma_done);
    } else if (warp >= 2) {
        // thread = token row of the unit's tile; group g of four warps takes the 16-column blocks
        // g, g + G, ...
        const int lb = 32 * (warp & 3);
        const int G = ((int)blockDim.x - 64) / 128, grp = (warp - 2) >> 2;
        int it = 0;
        for (int u = blockIdx.x; u < p.units; u += gridDim.x, ++it) {
            int m0, d0, kb0, kb1;
            unit(u, m0, d0, kb0, kb1);
            const int buf = it & 1;
            const int m = m0 + lb + lane;
            const int out_row = (p.perm && m < p.M) ? p.perm[m] : m;   // read before the wait
            const bool ok = mbar_wait(&acc_full[buf], (uint32_t)((it >> 1) & 1), &abort_flag);
            tc_fence_after();
            const bool row_ok = ok && m < p.M;
            for (int c0 = 16 * grp; c0 < BN; c0 += 16 * G) {
                float v[16];
                tmem_ld16(tmem + ((uint32_t)lb << 16) + (uint32_t)(buf * BN + c0), v);
                tmem_ld_wait();
                const int h = d0 * BM + c0;
                if (!row_ok || h >= p.H) continue;
                float *dst = p.out + (size_t)out_row * p.H + h;
                if (h + 16 <= p.H) {   // H is a multiple of 8: dst is 16-byte aligned
#pragma unroll
                    for (int q = 0; q < 4; ++q) red_add_v4(dst + 4 * q, v[4 * q], v[4 * q + 1], v[4 * q + 2], v[4 * q + 3]);
                } else {
#pragma unroll
                    for (int e = 0; e < 16; ++e)
                        if (h + e < p.H) atomicAdd(dst + e, v[e]);
                }
            }
            tc_fence_before();
            mbar_arrive(&acc_empty[buf]);
            if (!ok) break;
        }
    }
    __syncthreads();
    if (threadIdx.x == 0) {
        // the arrival on mma_done must land before this CTA's shared memory is released
        int never = 0;
        if (abort_flag)
            for (int k = consumed_s; k < issued_s; ++k) mbar_wait(&full[k % S], (uint32_t)((k / S) & 1), &never);
        mbar_wait(mma_done, 0u, &never);
    }
    __syncthreads();
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc(tmem, p.tmem_cols);
    }
}

// ---------------------------------------------------------------------- kept lists
// Row m's ascending kept list from its keep bytes (one CTA per row), written as
// the list of token perm[m] (token m without a permutation).  Thread t takes the
// 16-byte vectors [t per, (t + 1) per) of the row: it counts their kept bytes, a
// block scan gives its first position, and it writes its entries in order.  Two
// passes over the row in all (the second from L1/L2), one block scan.
__global__ void __launch_bounds__(512) keep_list_kernel(const uint8_t *__restrict__ keep, int stride, int N,
                                                        int32_t *__restrict__ idx, int32_t *__restrict__ cnt,
                                                        const int32_t *__restrict__ perm)
{
    grid_dependency_wait();   // the keep bytes are written by the preceding kernel
    grid_launch_dependents();
    const int m = blockIdx.x;
    const int tok = perm ? perm[m] : m;
    const uint4 *k = reinterpret_cast<const uint4 *>(keep + (size_t)m * stride);   // stride: a multiple of 16
    const int t = threadIdx.x, lane = t & 31, w = t >> 5;
    const int nv = (N + 15) >> 4;
    const int per = (nv + 511) >> 9;
    const int v0 = t * per, v1 = min(nv, v0 + per);
    // the kept bytes (0 or 1) of vector v as a 16-bit mask; bytes at or past N are not counted
    auto mask16 = [&](int v) {
        const uint4 q = k[v];
        const uint32_t wq[4] = {q.x, q.y, q.z, q.w};
        uint32_t bits = 0;
#pragma unroll
        for (int i = 0; i < 4; ++i)
            bits |= ((wq[i] & 1u) | ((wq[i] >> 7) & 2u) | ((wq[i] >> 14) & 4u) | ((wq[i] >> 21) & 8u)) << (4 * i);
        const int rest = N - 16 * v;
        return rest >= 16 ? bits : bits & ((1u << rest) - 1u);
    };
    int c = 0;
    for (int v = v0; v < v1; ++v) c += __popc(mask16(v));
    __shared__ int warp_sums[16];
    int incl = c;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const int x = __shfl_up_sync(0xffffffffu, incl, o);
        if (lane >= o) incl += x;
    }
    if (lane == 31) warp_sums[w] = incl;
    __syncthreads();
    int pos = incl - c, total = 0;
#pragma unroll
    for (int i = 0; i < 16; ++i) {
        if (i < w) pos += warp_sums[i];
        total += warp_sums[i];
    }
    int32_t *out = idx + (size_t)tok * N;
    for (int v = v0; v < v1; ++v)
        for (uint32_t bits = mask16(v); bits; bits &= bits - 1u) out[pos++] = 16 * v + __ffs(bits) - 1;
    if (t == 0 && cnt) cnt[tok] = total;
}


}  // namespace
}  // namespace tc

cudaError_t tc_pack_layer(sats_layer *l, cudaStream_t stream)
{
    using namespace tc;
    const int H = l->H, N = l->N;
    l->tc_R = choose_rows(N, sm_count());
    l->tc_T = (N + l->tc_R - 1) / l->tc_R;
    l->tc_kbh = (H + BK - 1) / BK;
    l->tc_dt = (H + BM - 1) / BM;
    l->tc_kbn = (N + BK - 1) / BK;
    l->ldn = (N + 7) & ~7;
    const size_t gu_elems = (size_t)l->tc_T * l->tc_kbh * 2 * l->tc_R * BK;
    const size_t wd_elems = (size_t)l->tc_dt * l->tc_kbn * BM * BK;
    cudaError_t e = cudaMalloc(&l->gu_blk, gu_elems * 2);
    if (e == cudaSuccess) e = cudaMalloc(&l->wd_blk, wd_elems * 2);
    if (e != cudaSuccess) return e;
    const size_t total8 = gu_elems / 8;
    const size_t blocks = (total8 + 255) / 256;
    pack_gu_kernel<<<(unsigned)(blocks < 8192 ? blocks : 8192), 256, 0, stream>>>(l->wg_t, l->w_ud, H, N, l->tc_R,
                                                                                 l->tc_kbh, total8, l->gu_blk);
    pack_wd_kernel<<<dim3(l->tc_kbn, l->tc_dt), 256, 0, stream>>>(l->w_ud, H, N, l->tc_kbn, l->wd_blk);
    return cudaGetLastError();
}

cudaError_t tc_free_layer(sats_layer *l)
{
    const cudaError_t e1 = cudaFree(l->gu_blk);
    const cudaError_t e2 = cudaFree(l->wd_blk);
    l->gu_blk = l->wd_blk = nullptr;
    return e1 != cudaSuccess ? e1 : e2;
}

namespace {
// The dynamic shared-memory limit set for gu_skinny_kernel on each device (both
// of its modes raise it through this one record, so neither lowers it under the other).
std::atomic<int> cfg_gu_skinny[64];

struct TcLayout {
    size_t xhi, xlo, hact, hact_lo, keep;
    size_t a_keep, u, uflag, ulist, ucount;   // the union path (batches up to kMaxUnion)
    size_t total;
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
    L.hact_lo = off;
    off += al((size_t)B * ldn * 2);
    L.keep = off;
    off += al((size_t)B * (((size_t)N + 15) & ~(size_t)15));
    if (B <= tc::kMaxUnion) {
        L.a_keep = off;
        off += al((size_t)B * ldn * 4);
        L.u = off;
        off += al((size_t)B * ldn * 4);
        L.uflag = off;   // padded to 16 bytes (read as 16-byte vectors)
        off += al(((size_t)N + 15) & ~(size_t)15);
        L.ulist = off;
        off += al((size_t)N * 4);
        L.ucount = off;
        off += al(4);
    }
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
//   perm, n_dense: the routing kernel's permutation and base-path count (device), or
//   nullptr (then dense_flags, or no token on the base path).  With a permutation x
//   must be fp32 (it is gathered into the split parts).
cudaError_t run_tc_layer(const sats_layer *layer, int x_mode, const void *x, int B, float t_l, const float *norm_w,
                         float eps, const uint8_t *dense_flags, const int32_t *perm, const int32_t *n_dense,
                         int out_mode, float *out, int32_t *active_idx, int32_t *active_cnt, uint8_t *keep_trace,
                         void *tc_ws, int *ctl, cudaStream_t stream, bool union_path)
{
    using namespace tc;
    auto fail = [](cudaError_t err, const char *where) {
        cuda_fail(err, where);
        return err;
    };
    const int H = layer->H, N = layer->N, ldn = layer->ldn, R = layer->tc_R;
    const TcLayout W = tc_layout(H, N, B);
    uint8_t *base = static_cast<uint8_t *>(tc_ws);
    uint16_t *xhi = reinterpret_cast<uint16_t *>(base + W.xhi);
    uint16_t *xlo = reinterpret_cast<uint16_t *>(base + W.xlo);
    uint16_t *hact = reinterpret_cast<uint16_t *>(base + W.hact);
    uint16_t *hact_lo = reinterpret_cast<uint16_t *>(base + W.hact_lo);
    uint8_t *keep = base + W.keep;
    const int kstride = (N + 15) & ~15;
    const int sms = sm_count();
    const bool split = x_mode != kXBf16;
    if (perm && (!split || !n_dense || union_path)) return fail(cudaErrorInvalidValue, "routed batch arguments");
    const uint16_t *xa = split ? xhi : static_cast<const uint16_t *>(x);
    cudaError_t e;

    if (split) {
        e = launch_pdl_threads(split_kernel, dim3(B), 256, stream, static_cast<const float *>(x), H,
                               x_mode == kXResidNorm ? norm_w : nullptr, eps, xhi, xlo, perm);
        if (e != cudaSuccess) return fail(e, "split kernel launch");
    }

    if (union_path) {   // the caller has checked union_path_ok(H, B) and that no token is on the base path
        // union path: gate on the tensor cores, then up and down for the union of the kept neurons
        const int NT = (B + 15) & ~15;
        CUtensorMap mX, mX2;
        if (!make_map(&mX, xa, B, H, (uint64_t)H * 2, NT) || !make_map(&mX2, split ? xlo : xa, B, H, (uint64_t)H * 2, NT))
            return fail(cudaErrorInvalidValue, "tensor map encoding");
        float *a_keep = reinterpret_cast<float *>(base + W.a_keep);
        float *u = reinterpret_cast<float *>(base + W.u);
        uint8_t *uflag = base + W.uflag;
        int32_t *ulist = reinterpret_cast<int32_t *>(base + W.ulist);
        int32_t *ucount = reinterpret_cast<int32_t *>(base + W.ucount);
        SkinnyGuParams gp{};
        gp.w = layer->gu_blk;
        gp.M = B;
        gp.N = N;
        gp.R = R;
        gp.KBh = layer->tc_kbh;
        gp.NT = NT;
        gp.split = split ? 1 : 0;
        gp.t_l = t_l;
        gp.ldh = ldn;
        gp.keep = active_idx ? keep : nullptr;
        gp.keep_stride = kstride;
        gp.keep_trace = keep_trace;
        gp.ctl = ctl;
        gp.zero = out_mode == kOutY ? out : nullptr;   // the down projection adds into y
        gp.zero_count = B * H;
        gp.gate_only = 1;
        gp.a_keep = a_keep;
        gp.uflag = uflag;
        // stage: the gate rows, then the token tile(s); the gate MMA reads 128 rows from the
        // stage start (rows R..127 of D are not used), so the ring ends with room for that read
        gp.a_bytes = R * kTileBytes;
        gp.x_bytes = NT * kTileBytes;
        gp.stage_bytes = gp.a_bytes + gp.x_bytes * (split ? 2 : 1);
        const int over = BM * kTileBytes - gp.stage_bytes;
        const int slack = over > 0 ? ((over + 1023) & ~1023) : 0;
        gp.stages = stages_for(gp.stage_bytes, kSmemBudget - slack);
        gp.ring_bytes = gp.stages * gp.stage_bytes + slack;
        gp.merge = split && NT <= 128 ? 1 : 0;
        gp.tmem_cols = tmem_cols_for(gp.merge ? 2 * NT : NT);
        if ((e = set_smem(gu_skinny_kernel, smem_for(1, gp.ring_bytes), cfg_gu_skinny)) != cudaSuccess)
            return fail(e, "shared-memory attribute");
        e = launch_pdl_cfg(gu_skinny_kernel, dim3(layer->tc_T), 64 + 128, smem_for(1, gp.ring_bytes), stream, mX, mX2,
                           gp);
        if (e != cudaSuccess) return fail(e, "gate kernel launch");
        e = launch_union_tail(layer, B, xa, split ? xlo : nullptr, uflag, ulist, ucount, a_keep, ldn, u, ldn, out, ctl,
                              stream);
        if (e != cudaSuccess) return fail(e, "union kernels launch");
    } else if (B <= (split ? kMaxSkinnySplit : kMaxSkinny)) {
        const int NT = (B + 15) & ~15;
        CUtensorMap mX, mX2, mH, mH2;
        if (!make_map(&mX, xa, B, H, (uint64_t)H * 2, NT) || !make_map(&mX2, split ? xlo : xa, B, H, (uint64_t)H * 2, NT) ||
            !make_map(&mH, hact, B, N, (uint64_t)ldn * 2, NT) || !make_map(&mH2, hact_lo, B, N, (uint64_t)ldn * 2, NT))
            return fail(cudaErrorInvalidValue, "tensor map encoding");
        SkinnyGuParams gp{};
        gp.w = layer->gu_blk;
        gp.M = B;
        gp.N = N;
        gp.R = R;
        gp.KBh = layer->tc_kbh;
        gp.NT = NT;
        gp.split = split ? 1 : 0;
        gp.t_l = t_l;
        gp.dense_flags = dense_flags;
        gp.perm = perm;
        gp.n_dense = n_dense;
        gp.hact = hact;
        gp.hact_lo = hact_lo;
        gp.ldh = ldn;
        gp.keep = active_idx ? keep : nullptr;
        gp.keep_stride = kstride;
        gp.keep_trace = keep_trace;
        gp.ctl = ctl;
        gp.zero = out_mode == kOutY ? out : nullptr;   // the down projection adds into y
        gp.zero_count = B * H;
        // stage: gate + up rows, then the token tile(s).  The up tile's MMA reads 128 rows from
        // row R; past 2R they are other data of the ring (rows R..127 of D are not used), and the
        // ring ends with enough room for the last stage's read.
        gp.a_bytes = 2 * R * kTileBytes;
        gp.x_bytes = NT * kTileBytes;
        gp.stage_bytes = gp.a_bytes + gp.x_bytes * (split ? 2 : 1);
        const int over = (R + BM) * kTileBytes - gp.stage_bytes;
        const int slack = over > 0 ? ((over + 1023) & ~1023) : 0;
        gp.stages = stages_for(gp.stage_bytes, kSmemBudget - slack);
        gp.ring_bytes = gp.stages * gp.stage_bytes + slack;
        gp.merge = split && NT <= 128 ? 1 : 0;
        gp.tmem_cols = tmem_cols_for((gp.merge ? 4 : 2) * NT);
        if ((e = set_smem(gu_skinny_kernel, smem_for(1, gp.ring_bytes), cfg_gu_skinny)) != cudaSuccess)
            return fail(e, "shared-memory attribute");
        // epilogue groups: one per 16-token column block, at most kSkinnyMaxGroups (the epilogue
        // runs after the last MMA, so its time adds to the call's)
        const int groups = NT / 16 < kSkinnyMaxGroups ? NT / 16 : kSkinnyMaxGroups;
        e = launch_pdl_cfg(gu_skinny_kernel, dim3(layer->tc_T), 64 + 128 * groups, smem_for(1, gp.ring_bytes), stream,
                           mX, mX2, gp);
        if (e != cudaSuccess) return fail(e, "gate/up kernel launch");

        SkinnyDownParams dp{};
        dp.w = layer->wd_blk;
        dp.M = B;
        dp.H = H;
        dp.NT = NT;
        dp.KBn = layer->tc_kbn;
        dp.units = layer->tc_dt * layer->tc_kbn;
        dp.out = out;
        dp.perm = perm;
        dp.ctl = ctl;
        dp.a_bytes = BM * kTileBytes;
        dp.stage_bytes = dp.a_bytes + 2 * NT * kTileBytes;
        dp.stages = stages_for(dp.stage_bytes);
        dp.merge = NT <= 128 ? 1 : 0;
        dp.tmem_cols = tmem_cols_for((dp.merge ? 4 : 2) * NT);
        static std::atomic<int> cfg_dn[64];
        if ((e = set_smem(down_skinny_kernel, smem_for(dp.stages, dp.stage_bytes), cfg_dn)) != cudaSuccess)
            return fail(e, "shared-memory attribute");
        e = launch_pdl(down_skinny_kernel, dim3(dp.units < sms ? dp.units : sms), smem_for(dp.stages, dp.stage_bytes),
                       stream, mH, mH2, dp);
        if (e != cudaSuccess) return fail(e, "down kernel launch");
    } else {
        CUtensorMap mX, mX2, mH, mH2;
        if (!make_map(&mX, xa, B, H, (uint64_t)H * 2, BM) ||
            !make_map(&mX2, split ? xlo : xa, B, H, (uint64_t)H * 2, BM) ||
            !make_map(&mH, hact, B, N, (uint64_t)ldn * 2, BM) || !make_map(&mH2, hact_lo, B, N, (uint64_t)ldn * 2, BM))
            return fail(cudaErrorInvalidValue, "tensor map encoding");
        const int mtiles = (B + BM - 1) / BM;

        WideGuParams gp{};
        gp.w = layer->gu_blk;
        gp.M = B;
        gp.N = N;
        gp.R = R;
        gp.KBh = layer->tc_kbh;
        gp.T = layer->tc_T;
        gp.Rw = wide_rows(N, R, mtiles, sms, split);
        gp.mtiles = mtiles;
        gp.tiles = mtiles * ((N + gp.Rw - 1) / gp.Rw);
        gp.tmem_cols = tmem_cols_for(4 * gp.Rw);
        gp.split = split ? 1 : 0;
        gp.t_l = t_l;
        gp.dense_flags = dense_flags;
        gp.perm = perm;
        gp.n_dense = n_dense;
        gp.hact = hact;
        gp.hact_lo = hact_lo;
        gp.ldh = ldn;
        gp.keep = active_idx ? keep : nullptr;
        gp.keep_stride = kstride;
        gp.keep_trace = keep_trace;
        gp.ctl = ctl;
        gp.zero = out_mode == kOutY ? out : nullptr;   // the down projection adds into y
        gp.zero_count = (long long)B * H;
        gp.stage_bytes = BM * kTileBytes * (split ? 2 : 1) + 2 * gp.Rw * kTileBytes;
        gp.stages = stages_for(gp.stage_bytes, wide_budget());
        // epilogue groups: the tile's 16-neuron column blocks split evenly over at most kWideGuGroups
        const int blocks16 = gp.Rw / 16, per_group = (blocks16 + kWideGuGroups - 1) / kWideGuGroups;
        const int gu_groups = (blocks16 + per_group - 1) / per_group;
        static std::atomic<int> cfg_gu[64];
        if ((e = set_smem(gu_wide_kernel, smem_for(gp.stages, gp.stage_bytes), cfg_gu)) != cudaSuccess)
            return fail(e, "shared-memory attribute");
        gu_wide_kernel<<<dim3(gp.tiles < sms ? gp.tiles : sms), 64 + 128 * gu_groups, smem_for(gp.stages, gp.stage_bytes),
                         stream>>>(mX, mX2, gp);
        if ((e = cudaGetLastError()) != cudaSuccess) return fail(e, "gate/up kernel launch");

        // down projection: 256 output columns per unit when the hidden tiles pair up; the neuron
        // range split so that the persistent CTAs' units come out even; every unit adds into the
        // output (y cleared by the gate/up kernel, or the residual stream)
        WideDownParams dp{};
        dp.w = layer->wd_blk;
        dp.M = B;
        dp.H = H;
        dp.KBn = layer->tc_kbn;
        dp.dtiles = (layer->tc_dt % 2 == 0) ? 2 : 1;
        dp.mtiles = mtiles;
        dp.dcols = layer->tc_dt / dp.dtiles;
        const int splits = wide_down_splits(mtiles * dp.dcols, dp.KBn, sms);
        dp.kb_per_split = (dp.KBn + splits - 1) / splits;
        dp.units = mtiles * dp.dcols * splits;
        dp.out = out;
        dp.perm = perm;
        dp.ctl = ctl;
        dp.stage_bytes = BM * kTileBytes * (2 + dp.dtiles);
        dp.stages = stages_for(dp.stage_bytes, wide_budget());
        dp.tmem_cols = tmem_cols_for(2 * BM * dp.dtiles);
        static std::atomic<int> cfg_dn[64];
        if ((e = set_smem(down_wide_kernel, smem_for(dp.stages, dp.stage_bytes), cfg_dn)) != cudaSuccess)
            return fail(e, "shared-memory attribute");
        down_wide_kernel<<<dim3(dp.units < sms ? dp.units : sms), 64 + 128 * kWideDownGroups,
                           smem_for(dp.stages, dp.stage_bytes), stream>>>(mH, mH2, dp);
        if ((e = cudaGetLastError()) != cudaSuccess) return fail(e, "down kernel launch");
    }
    if (active_idx) {
        e = launch_pdl_threads(keep_list_kernel, dim3(B), 512, stream, static_cast<const uint8_t *>(keep), kstride, N,
                               active_idx, active_cnt, perm);
        if (e != cudaSuccess) return fail(e, "kept-list kernel launch");
    }
    return cudaSuccess;
}

}  // namespace sats
