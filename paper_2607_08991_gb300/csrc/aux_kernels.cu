// aux_kernels.cu -- weight repacking, token routing (Sec. 3.2, Eq. 13),
// the calibration gate activation (Sec. 2, Eqs. 1-2) and the percentile
// threshold selection (Sec. 2, Eq. 3) for sm_103a.
#include <cmath>

#include "common.cuh"
#include "internal.h"

namespace sats {
namespace {

// ------------------------------------------------------------------ repacking
// Wg [H][N] -> wg_t [N][H];  Wu [H][N] -> w_ud[:, 0:H] (transposed);
// Wd [N][H] -> w_ud[:, H:2H] (row copy).  32x32 tiles through shared memory.
constexpr int kTile = 32;

__global__ void transpose_kernel(const uint16_t *__restrict__ src, int rows, int cols,
                                 uint16_t *__restrict__ dst, int dst_stride)
{
    // src [rows][cols] -> dst[c * dst_stride + r]
    __shared__ uint16_t tile[kTile][kTile + 2];
    const int c0 = blockIdx.x * kTile, r0 = blockIdx.y * kTile;
    for (int dy = threadIdx.y; dy < kTile; dy += blockDim.y) {
        const int r = r0 + dy, c = c0 + threadIdx.x;
        if (r < rows && c < cols) tile[dy][threadIdx.x] = src[(size_t)r * cols + c];
    }
    __syncthreads();
    for (int dy = threadIdx.y; dy < kTile; dy += blockDim.y) {
        const int c = c0 + dy, r = r0 + threadIdx.x;
        if (r < rows && c < cols) dst[(size_t)c * dst_stride + r] = tile[threadIdx.x][dy];
    }
}

__global__ void copy_rows_kernel(const uint16_t *__restrict__ src, int rows, int cols,
                                 uint16_t *__restrict__ dst, int dst_stride)
{
    const size_t total = (size_t)rows * cols;
    for (size_t i = blockIdx.x * (size_t)blockDim.x + threadIdx.x; i < total; i += (size_t)gridDim.x * blockDim.x) {
        const size_t r = i / cols, c = i - r * cols;
        dst[r * dst_stride + c] = src[i];
    }
}

// ------------------------------------------------------------------ routing
// One CTA of 1024 threads.  Pass 1 counts base-path tokens; pass 2 walks the
// batch in tiles of 1024 with a block-wide exclusive scan, placing each token
// at its rank within its group: a stable partition, identical on every run.
constexpr int kRouteThreads = 1024;

__device__ __forceinline__ int route_flag(const int32_t *ids, int b, const uint8_t *lut, int V, int32_t *status)
{
    const int id = ids[b];
    if (id < 0 || id >= V) {
        if (status) atomicOr(status, kStatusBadToken);
        return 1;   // unknown ids take the base path
    }
    return lut[id] ? 1 : 0;
}

__device__ int block_excl_scan(int v, int *warp_tot, int *total)
{
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    int incl = v;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const int t = __shfl_up_sync(0xffffffffu, incl, o);
        if (lane >= o) incl += t;
    }
    if (lane == 31) warp_tot[warp] = incl;
    __syncthreads();
    if (warp == 0) {
        int w = lane < (int)(blockDim.x >> 5) ? warp_tot[lane] : 0;
        int wi = w;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int t = __shfl_up_sync(0xffffffffu, wi, o);
            if (lane >= o) wi += t;
        }
        warp_tot[lane] = wi - w;   // exclusive prefix of warp totals
        if (lane == 31) *total = wi;
    }
    __syncthreads();
    const int r = warp_tot[warp] + incl - v;
    __syncthreads();
    return r;
}

__global__ void __launch_bounds__(kRouteThreads) route_kernel(const int32_t *ids, int B, const uint8_t *lut, int V,
                                                              int32_t *perm, int32_t *n_dense, uint8_t *flags,
                                                              int32_t *status)
{
    __shared__ int warp_tot[32];
    __shared__ int total;
    int cnt = 0;
    for (int b = threadIdx.x; b < B; b += kRouteThreads) cnt += route_flag(ids, b, lut, V, nullptr);
    (void)block_excl_scan(cnt, warp_tot, &total);
    const int nd = total;
    __syncthreads();
    int dense_before = 0;
    for (int base = 0; base < B; base += kRouteThreads) {
        const int b = base + threadIdx.x;
        const int f = b < B ? route_flag(ids, b, lut, V, status) : 0;
        const int excl = block_excl_scan(f, warp_tot, &total);
        if (b < B) {
            const int d = dense_before + excl;                 // base-path tokens before b
            perm[f ? d : nd + (b - d)] = b;
            if (flags) flags[b] = (uint8_t)f;
        }
        dense_before += total;
        __syncthreads();
    }
    if (threadIdx.x == 0) *n_dense = nd;
}

// ------------------------------------------------------------------ calibration
// 8 consecutive activations of token row xr starting at element 8 v, as floats.
__device__ __forceinline__ void load_x8(const uint16_t *xr, int v, float (&xf)[8])
{
    unpack8(reinterpret_cast<const uint4 *>(xr)[v], xf);
}
__device__ __forceinline__ void load_x8(const float *xr, int v, float (&xf)[8])
{
    const float4 p = reinterpret_cast<const float4 *>(xr)[2 * v], q = reinterpret_cast<const float4 *>(xr)[2 * v + 1];
    xf[0] = p.x; xf[1] = p.y; xf[2] = p.z; xf[3] = p.w;
    xf[4] = q.x; xf[5] = q.y; xf[6] = q.z; xf[7] = q.w;
}

// a[b][j] = SiLU(x_b . W_gate[:, j]), one warp per neuron row of wg_t, tokens
// in groups of 8 (weights re-read from L2 per group; calibration only).
// X is uint16_t (bf16 activations) or float.
template <typename X>
__global__ void gate_act_kernel(const uint16_t *__restrict__ wg_t, int H, int N, const X *__restrict__ x,
                                int B, float *__restrict__ a)
{
    const int warp = (blockIdx.x * blockDim.x + threadIdx.x) >> 5;
    const int lane = threadIdx.x & 31;
    if (warp >= N) return;
    const uint4 *row = reinterpret_cast<const uint4 *>(wg_t + (size_t)warp * H);
    const int HV = H >> 3;
    for (int b0 = 0; b0 < B; b0 += 8) {
        float acc[8];
#pragma unroll
        for (int t = 0; t < 8; ++t) acc[t] = 0.f;
        for (int v = lane; v < HV; v += 32) {
            float w[8];
            unpack8(row[v], w);
#pragma unroll
            for (int t = 0; t < 8; ++t) {
                if (b0 + t < B) {
                    float xf[8];
                    load_x8(x + (size_t)(b0 + t) * H, v, xf);
#pragma unroll
                    for (int e = 0; e < 8; ++e) acc[t] = fmaf(w[e], xf[e], acc[t]);
                }
            }
        }
#pragma unroll
        for (int t = 0; t < 8; ++t) {
            const float g = warp_sum(acc[t]);
            if (lane == 0 && b0 + t < B) a[(size_t)(b0 + t) * N + warp] = g / (1.0f + expf(-g));
        }
    }
}

// ------------------------------------------------------------------ selection
// The m-th smallest |a_i| by a two-level radix select on the IEEE bit pattern
// of |a_i| (non-negative floats order as their unsigned bit patterns):
// histogram of the high 16 bits, locate the bin holding rank m, histogram of
// the low 16 bits inside that bin, locate again.
constexpr int kBins = 65536;

__global__ void hist_kernel(const float *__restrict__ a, int64_t n, int level, const int *__restrict__ sel,
                            unsigned *__restrict__ hist)
{
    const int hi_bin = level ? sel[0] : 0;
    for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x) {
        const uint32_t bits = __float_as_uint(a[i]) & 0x7fffffffu;
        if (level == 0) atomicAdd(&hist[bits >> 16], 1u);
        else if ((int)(bits >> 16) == hi_bin) atomicAdd(&hist[bits & 0xffffu], 1u);
    }
}

// sel[2*level] <- bin holding rank r (1-based), sel[2*level+1] <- rank inside it.
// rank r comes from sel[1] for level 1, from `m` for level 0.
__global__ void __launch_bounds__(1024) find_bin_kernel(const unsigned *__restrict__ hist, int64_t m, int level,
                                                        int *__restrict__ sel, float *__restrict__ t_out)
{
    __shared__ unsigned long long warp_tot[32];
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const long long r = level ? (long long)sel[1] : (long long)m;
    constexpr int kPer = kBins / 1024;
    unsigned long long s = 0;
    for (int i = 0; i < kPer; ++i) s += hist[tid * kPer + i];
    unsigned long long incl = s;
    for (int o = 1; o < 32; o <<= 1) {
        const unsigned long long t = __shfl_up_sync(0xffffffffu, incl, o);
        if (lane >= o) incl += t;
    }
    if (lane == 31) warp_tot[warp] = incl;
    __syncthreads();
    unsigned long long before = 0;
    for (int w = 0; w < warp; ++w) before += warp_tot[w];
    const unsigned long long lo = before + incl - s;     // count of values in bins below this thread's range
    if ((long long)lo < r && (long long)(lo + s) >= r) {
        unsigned long long run = lo;
        for (int i = 0; i < kPer; ++i) {
            const unsigned c = hist[tid * kPer + i];
            if ((long long)(run + c) >= r) {
                const int bin = tid * kPer + i;
                if (level == 0) {
                    sel[0] = bin;
                    sel[1] = (int)(r - (long long)run);
                } else {
                    const uint32_t bits = ((uint32_t)sel[0] << 16) | (uint32_t)bin;
                    *t_out = __uint_as_float(bits);
                }
                break;
            }
            run += c;
        }
    }
}

}  // namespace

cudaError_t launch_pack(const uint16_t *Wg, const uint16_t *Wu, const uint16_t *Wd, int H, int N,
                        uint16_t *wg_t, uint16_t *w_ud, cudaStream_t stream)
{
    const dim3 block(kTile, 8);
    const dim3 grid((N + kTile - 1) / kTile, (H + kTile - 1) / kTile);
    transpose_kernel<<<grid, block, 0, stream>>>(Wg, H, N, wg_t, H);
    transpose_kernel<<<grid, block, 0, stream>>>(Wu, H, N, w_ud, 2 * H);
    copy_rows_kernel<<<1024, 256, 0, stream>>>(Wd, N, H, w_ud + H, 2 * H);
    return cudaGetLastError();
}

// LoRA adapter layout of the fused kernel (one element per thread, grid-stride):
//   blk [ceil(N/8)][8][3r]: neuron j = 8c + i holds B_gate[:, j], B_up[:, j], A_down[j, :]
//   (neurons past N are zero); agu [H][2r]: A_gate[h, :], A_up[h, :]; bd = B_down [r][H].
__global__ void pack_lora_kernel(const uint16_t *__restrict__ Ag, const uint16_t *__restrict__ Bg,
                                 const uint16_t *__restrict__ Au, const uint16_t *__restrict__ Bu,
                                 const uint16_t *__restrict__ Ad, const uint16_t *__restrict__ Bd, int H, int N, int r,
                                 uint16_t *__restrict__ blk, uint16_t *__restrict__ agu, uint16_t *__restrict__ bd)
{
    const size_t nblk = (size_t)((N + 7) / 8) * 8 * 3 * r, nagu = (size_t)H * 2 * r, nbd = (size_t)r * H;
    for (size_t i = blockIdx.x * (size_t)blockDim.x + threadIdx.x; i < nblk + nagu + nbd;
         i += (size_t)gridDim.x * blockDim.x) {
        if (i < nblk) {
            const int j = (int)(i / (3 * r)), e = (int)(i % (3 * r));
            const int part = e / r, q = e % r;
            uint16_t v = 0;
            if (j < N) v = part == 0 ? Bg[(size_t)q * N + j] : (part == 1 ? Bu[(size_t)q * N + j] : Ad[(size_t)j * r + q]);
            blk[i] = v;
        } else if (i < nblk + nagu) {
            const size_t k = i - nblk;
            const int h = (int)(k / (2 * r)), e = (int)(k % (2 * r));
            agu[k] = e < r ? Ag[(size_t)h * r + e] : Au[(size_t)h * r + (e - r)];
        } else {
            const size_t k = i - nblk - nagu;
            bd[k] = Bd[k];
        }
    }
}

cudaError_t launch_pack_lora(const uint16_t *Ag, const uint16_t *Bg, const uint16_t *Au, const uint16_t *Bu,
                             const uint16_t *Ad, const uint16_t *Bd, int H, int N, int r, sats_lora *l,
                             cudaStream_t stream)
{
    pack_lora_kernel<<<1024, 256, 0, stream>>>(Ag, Bg, Au, Bu, Ad, Bd, H, N, r, l->blk, l->agu, l->bd);
    return cudaGetLastError();
}

cudaError_t launch_route(const int32_t *ids, int B, const uint8_t *lut, int V, int32_t *perm, int32_t *n_dense,
                         uint8_t *flags, int32_t *status, cudaStream_t stream)
{
    route_kernel<<<1, kRouteThreads, 0, stream>>>(ids, B, lut, V, perm, n_dense, flags, status);
    return cudaGetLastError();
}

// The library's bounded waits, made to run out: an mbarrier phase that no thread
// completes (the wait every ring of the MLP kernels uses) and a counter in the
// workspace that no CTA raises (the form of the fused kernel's prologue wait).
// Each gives up after kWaitLimitNs and records a timeout in the status word.
__global__ void wait_timeout_kernel(int *ctl)
{
    __shared__ uint64_t bar;
    __shared__ int never;
    if (threadIdx.x == 0) {
        mbar_init(&bar, 1);
        never = 0;
        mbar_init_fence();
    }
    __syncthreads();
    if (threadIdx.x != 0) return;
    if (!mbar_wait(&bar, 0u, &never)) atomicOr(ctl + kCtlStatus, kStatusTimeout);
    const unsigned long long t0 = global_ns();
    while (ld_acquire_gpu(ctl + kCtlSelftest) == 0) {
        if (global_ns() - t0 > kWaitLimitNs) {
            atomicOr(ctl + kCtlStatus, kStatusTimeout);
            break;
        }
        __nanosleep(256);
    }
}

cudaError_t launch_wait_timeout(int *ctl, cudaStream_t stream)
{
    wait_timeout_kernel<<<1, 32, 0, stream>>>(ctl);
    return cudaGetLastError();
}

cudaError_t launch_gate_act(const sats_layer *layer, const uint16_t *x, int B, float *a, cudaStream_t stream)
{
    const int threads = 256;
    const int blocks = (layer->N * 32 + threads - 1) / threads;
    gate_act_kernel<uint16_t><<<blocks, threads, 0, stream>>>(layer->wg_t, layer->H, layer->N, x, B, a);
    return cudaGetLastError();
}

cudaError_t launch_gate_act_f32(const sats_layer *layer, const float *x, int B, float *a, cudaStream_t stream)
{
    const int threads = 256;
    const int blocks = (layer->N * 32 + threads - 1) / threads;
    gate_act_kernel<float><<<blocks, threads, 0, stream>>>(layer->wg_t, layer->H, layer->N, x, B, a);
    return cudaGetLastError();
}

size_t select_ws_bytes() { return (size_t)kBins * sizeof(unsigned) + 256; }

cudaError_t launch_select(const float *a, int64_t n, int64_t m, void *ws, float *t_dev, cudaStream_t stream)
{
    unsigned *hist = static_cast<unsigned *>(ws);
    int *sel = reinterpret_cast<int *>(static_cast<char *>(ws) + (size_t)kBins * sizeof(unsigned));
    const int blocks = 1024;
    cudaError_t e = cudaMemsetAsync(hist, 0, (size_t)kBins * sizeof(unsigned), stream);
    if (e != cudaSuccess) return e;
    hist_kernel<<<blocks, 256, 0, stream>>>(a, n, 0, sel, hist);
    find_bin_kernel<<<1, 1024, 0, stream>>>(hist, m, 0, sel, t_dev);
    e = cudaMemsetAsync(hist, 0, (size_t)kBins * sizeof(unsigned), stream);
    if (e != cudaSuccess) return e;
    hist_kernel<<<blocks, 256, 0, stream>>>(a, n, 1, sel, hist);
    find_bin_kernel<<<1, 1024, 0, stream>>>(hist, m, 1, sel, t_dev);
    return cudaGetLastError();
}

}  // namespace sats
