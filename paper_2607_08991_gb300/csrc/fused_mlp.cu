// fused_mlp.cu -- the CATS-thresholded gated MLP (Sec. 2, Eqs. 1-5 of
// arXiv 2607.08991) as one persistent, warp-specialised kernel for sm_103a.
//
// Per call, for nb <= 4 tokens with per-token threshold t_b:
//   a_j = SiLU(x . W_gate[:, j]);  keep_bj = |a_bj| >= t_b
//   y_b = sum_j keep_bj * a_bj * (x_b . W_up[:, j]) * W_down[j, :]
//
// Layout (made by the packer): Wg_t [N][H] and W_ud [N][2H], so that the gate
// row of neuron j is 2H contiguous bytes and its up column + down row are 4H
// contiguous bytes.  A neuron no token keeps costs no HBM traffic beyond its
// gate row.
//
// One CTA per SM (288 threads, ~205 KB shared memory):
//   * producer warp, one thread: claims chunks of 16 neurons from a global
//     counter and streams, through a ring of 6 x 32 KB shared-memory stages,
//     first the chunk's gate rows, then -- once the consumers have published
//     which neurons of the previous chunk are kept -- that chunk's W_ud rows.
//     Every copy is one cp.async.bulk that completes on the stage's mbarrier.
//   * 8 consumer warps: thread t owns 16-byte vectors t, t + 256, ... of every
//     row, holds the matching x values and y accumulators in registers, forms
//     dot-product partials, reduces them per warp and across warps through
//     shared memory, applies SiLU and the mask, compacts the kept neurons with
//     warp ballots, and accumulates h_j * W_down[j, :] into its y registers.
//   * after the stream: each CTA writes its y partial, a bounded grid barrier,
//     then every CTA reduces a slice of y across the partials in a fixed order
//     (deterministic), and the per-chunk index lists are compacted into the
//     ascending per-token active-index list.
// Every wait is bounded in time; a wait that gives up sets the status word.
#include <cmath>
#include <cstdio>

#include "common.cuh"
#include "internal.h"

namespace sats {
namespace {

constexpr int kConsumerWarps = 8;
constexpr int kConsumers = kConsumerWarps * 32;   // 256
constexpr int kThreads = kConsumers + 32;         // + producer warp
constexpr int kStageBytes = 32768;
constexpr int kStages = 6;

enum StageKind { kGate = 0, kUpDown = 1, kEnd = 2 };

template <int BT>
struct StageDesc {
    int kind, nrows, chunk_pos, last, buf, chunk, pad0, pad1;
    int neuron[kChunk];
    float am[kChunk][BT];   // keep ? a : 0, per row and token
};

template <int BT>
struct Shared {
    uint64_t full[kStages];
    uint64_t empty[kStages];
    uint64_t listready[2];
    uint64_t csync;                                  // consumer-wide barrier
    StageDesc<BT> desc[kStages];
    float gpart[2][kChunk][BT][kConsumerWarps];      // gate partials per chunk buffer
    float upart[2][kChunk][BT][kConsumerWarps];      // up partials per UD stage parity
    int ulist[2][kChunk];                            // kept-by-any-token rows of a chunk
    float uam[2][kChunk][BT];
    int ucnt[2];
    int issued[kStages];                             // producer: parity+1 of last fill
    float thr[BT];
    float red[kConsumerWarps][BT];
    int warp_sums[kThreads / 32];
    int abort;
};

template <int BT>
constexpr size_t smem_bytes() { return (size_t)kStages * kStageBytes + sizeof(Shared<BT>); }

__device__ __forceinline__ void flag_status(int *ctl, int bits) { atomicOr(ctl + kCtlStatus, bits); }

// Consumer-wide barrier on an mbarrier (one arrival per consumer warp), bounded in time.
struct ConsumerSync {
    uint64_t *bar;
    uint32_t parity;
    __device__ bool operator()(int lane, volatile int *abort)
    {
        __syncwarp();
        if (lane == 0) mbar_arrive(bar);
        const bool ok = mbar_wait(bar, parity, abort);
        parity ^= 1u;
        return ok;
    }
};

// ------------------------------------------------------------------ producer
template <int BT>
__device__ void producer(const FusedParams &p, Shared<BT> &S, uint8_t *stages)
{
    const uint64_t pol = l2_policy_evict_first();
    const int H = p.H, N = p.N;
    const uint32_t gate_row_bytes = (uint32_t)H * 2u;
    const uint32_t ud_row_bytes = (uint32_t)H * 4u;
    const int rows_per_gate_stage = min(kChunk, kStageBytes / (int)gate_row_bytes);
    const int rows_per_ud_stage = min(kChunk, kStageBytes / (int)ud_row_bytes);
    int *counter = p.ctl + kCtlChunk;

    uint32_t stage = 0, phase = 0;
    uint32_t lr_uses[2] = {0u, 0u};
    int seq = 0, prev = -1, prev_buf = 0;
    bool ok = true;
    int next = atomicAdd(counter, 1);

    auto advance = [&]() {
        if (++stage == kStages) { stage = 0; phase ^= 1u; }
    };

    for (;;) {
        const int c = next;
        const bool have = c < p.nchunks;
        const int buf = seq & 1;
        if (have) {
            next = atomicAdd(counter, 1);
            const int n0 = c * kChunk;
            const int rows = min(kChunk, N - n0);
            for (int r0 = 0; r0 < rows; r0 += rows_per_gate_stage) {
                const int nr = min(rows_per_gate_stage, rows - r0);
                if (!mbar_wait(&S.empty[stage], phase ^ 1u, &S.abort)) { ok = false; break; }
                StageDesc<BT> &d = S.desc[stage];
                d.kind = kGate;
                d.nrows = nr;
                d.chunk_pos = r0;
                d.last = (r0 + nr >= rows) ? 1 : 0;
                d.buf = buf;
                d.chunk = c;
                S.issued[stage] = (int)phase + 1;
                mbar_arrive_expect_tx(&S.full[stage], (uint32_t)nr * gate_row_bytes);
                bulk_load(stages + (size_t)stage * kStageBytes, p.wg_t + (size_t)(n0 + r0) * H,
                          (uint32_t)nr * gate_row_bytes, &S.full[stage], pol);
                advance();
            }
            if (!ok) break;
        }
        if (prev >= 0) {
            if (!mbar_wait(&S.listready[prev_buf], lr_uses[prev_buf] & 1u, &S.abort)) { ok = false; break; }
            ++lr_uses[prev_buf];
            const int cnt = S.ucnt[prev_buf];
            const int n0 = prev * kChunk;
            for (int k0 = 0; k0 < cnt; k0 += rows_per_ud_stage) {
                const int nr = min(rows_per_ud_stage, cnt - k0);
                if (!mbar_wait(&S.empty[stage], phase ^ 1u, &S.abort)) { ok = false; break; }
                StageDesc<BT> &d = S.desc[stage];
                d.kind = kUpDown;
                d.nrows = nr;
                for (int k = 0; k < nr; ++k) {
                    d.neuron[k] = n0 + S.ulist[prev_buf][k0 + k];
#pragma unroll
                    for (int b = 0; b < BT; ++b) d.am[k][b] = S.uam[prev_buf][k0 + k][b];
                }
                S.issued[stage] = (int)phase + 1;
                mbar_arrive_expect_tx(&S.full[stage], (uint32_t)nr * ud_row_bytes);
                uint8_t *dst = stages + (size_t)stage * kStageBytes;
                for (int k = 0; k < nr; ++k)
                    bulk_load(dst + (size_t)k * ud_row_bytes, p.w_ud + (size_t)d.neuron[k] * 2 * H, ud_row_bytes,
                              &S.full[stage], pol);
                advance();
            }
            if (!ok) break;
        }
        if (!have) break;
        prev = c;
        prev_buf = buf;
        ++seq;
    }
    if (ok && mbar_wait(&S.empty[stage], phase ^ 1u, &S.abort)) {
        S.desc[stage].kind = kEnd;
        mbar_arrive(&S.full[stage]);
    } else {
        S.abort = 1;
        flag_status(p.ctl, kStatusTimeout);
    }
}

// Bounded wait for every bulk copy still in flight (only on the error path).
template <int BT>
__device__ void drain_copies(Shared<BT> &S)
{
    int never = 0;
    for (int s = 0; s < kStages; ++s)
        if (S.issued[s] > 0) (void)mbar_wait(&S.full[s], (uint32_t)(S.issued[s] - 1), &never);
}

// ------------------------------------------------------------------ consumers
template <int BT, int VPT>
__device__ void chunk_lists(const FusedParams &p, Shared<BT> &S, int buf, int chunk, int lane)
{
    const int n0 = chunk * kChunk;
    const int rows = min(kChunk, p.N - n0);
    const int r = lane;
    const bool in = r < rows;
    float a[BT];
    uint32_t bal[BT];
    uint32_t uni = 0;
#pragma unroll
    for (int b = 0; b < BT; ++b) {
        float g = 0.f;
        if (in) {
#pragma unroll
            for (int w = 0; w < kConsumerWarps; ++w) g += S.gpart[buf][r][b][w];
        }
        a[b] = g / (1.0f + expf(-g));                 // SiLU, Eq. 2
        const bool keep = in && b < p.nb && fabsf(a[b]) >= S.thr[b];   // Eqs. 4-5
        bal[b] = __ballot_sync(0xffffffffu, keep);
        uni |= bal[b];
    }
    const uint32_t lt = (1u << lane) - 1u;
    if ((uni >> lane) & 1u) {
        const int pos = __popc(uni & lt);
        S.ulist[buf][pos] = r;
#pragma unroll
        for (int b = 0; b < BT; ++b) S.uam[buf][pos][b] = ((bal[b] >> lane) & 1u) ? a[b] : 0.f;
    }
    if (lane == 0) S.ucnt[buf] = __popc(uni);
    if (p.active_idx) {
        const int stride = p.nchunks * kChunk;
#pragma unroll
        for (int b = 0; b < BT; ++b) {
            if (b >= p.nb) break;
            if ((bal[b] >> lane) & 1u) p.idx_tmp[b * stride + n0 + __popc(bal[b] & lt)] = n0 + r;
            if (lane == 0) p.chunk_cnt[chunk * kMaxTokensPerPass + b] = __popc(bal[b]);
        }
    }
    if (p.keep_trace && in) {
#pragma unroll
        for (int b = 0; b < BT; ++b)
            if (b < p.nb) p.keep_trace[(size_t)b * p.N + n0 + r] = (uint8_t)((bal[b] >> lane) & 1u);
    }
    __syncwarp();
    if (lane == 0) mbar_arrive(&S.listready[buf]);
}

template <int BT, int VPT>
__device__ void consumer(const FusedParams &p, Shared<BT> &S, const uint8_t *stages, float (&yv)[BT][VPT][8])
{
    const int tid = threadIdx.x;
    const int warp = tid >> 5, lane = tid & 31;
    const int H = p.H, HV = H >> 3;
    const size_t gate_row_bytes = (size_t)H * 2, ud_row_bytes = (size_t)H * 4;
    ConsumerSync csync{&S.csync, 0u};

    // ---- activations of this pass, in registers
    float xv[BT][VPT][8];
#pragma unroll
    for (int b = 0; b < BT; ++b)
#pragma unroll
        for (int i = 0; i < VPT; ++i) {
            const int v = tid + i * kConsumers;
#pragma unroll
            for (int e = 0; e < 8; ++e) { xv[b][i][e] = 0.f; yv[b][i][e] = 0.f; }
            if (v < HV && b < p.nb) {
                if (p.x_mode == kXBf16) {
                    const uint4 w = reinterpret_cast<const uint4 *>(static_cast<const uint16_t *>(p.x) + (size_t)b * H)[v];
                    unpack8(w, xv[b][i]);
                } else {
                    const float4 *src = reinterpret_cast<const float4 *>(static_cast<const float *>(p.x) + (size_t)b * H);
                    const float4 lo = src[2 * v], hi = src[2 * v + 1];
                    xv[b][i][0] = lo.x; xv[b][i][1] = lo.y; xv[b][i][2] = lo.z; xv[b][i][3] = lo.w;
                    xv[b][i][4] = hi.x; xv[b][i][5] = hi.y; xv[b][i][6] = hi.z; xv[b][i][7] = hi.w;
                }
            }
        }
    if (p.x_mode == kXResidNorm) {
        // RMSNorm of the residual stream: x / sqrt(mean(x^2) + eps) * w
        float ss[BT];
#pragma unroll
        for (int b = 0; b < BT; ++b) {
            float s = 0.f;
#pragma unroll
            for (int i = 0; i < VPT; ++i)
#pragma unroll
                for (int e = 0; e < 8; ++e) s = fmaf(xv[b][i][e], xv[b][i][e], s);
            ss[b] = warp_sum(s);
        }
        if (lane == 0) {
#pragma unroll
            for (int b = 0; b < BT; ++b) S.red[warp][b] = ss[b];
        }
        if (!csync(lane, &S.abort)) { S.abort = 1; flag_status(p.ctl, kStatusTimeout); return; }
#pragma unroll
        for (int b = 0; b < BT; ++b) {
            float tot = 0.f;
            for (int w = 0; w < kConsumerWarps; ++w) tot += S.red[w][b];
            const float inv = 1.0f / sqrtf(tot / (float)H + p.eps);
#pragma unroll
            for (int i = 0; i < VPT; ++i) {
                const int v = tid + i * kConsumers;
                if (v < HV) {
                    const float4 *gw = reinterpret_cast<const float4 *>(p.norm_w);
                    const float4 lo = gw[2 * v], hi = gw[2 * v + 1];
                    const float g8[8] = {lo.x, lo.y, lo.z, lo.w, hi.x, hi.y, hi.z, hi.w};
#pragma unroll
                    for (int e = 0; e < 8; ++e) xv[b][i][e] = xv[b][i][e] * inv * g8[e];
                }
            }
        }
    }

    uint32_t stage = 0, phase = 0;
    int ud_seq = 0;
    for (;;) {
        if (!mbar_wait(&S.full[stage], phase, &S.abort)) {
            S.abort = 1;
            flag_status(p.ctl, kStatusTimeout);
            return;
        }
        const StageDesc<BT> &d = S.desc[stage];
        const int kind = d.kind;
        if (kind == kEnd) break;
        const uint8_t *sbase = stages + (size_t)stage * kStageBytes;
        const int nr = d.nrows;
        if (kind == kGate) {
            const int r0 = d.chunk_pos, buf = d.buf, last = d.last, chunk = d.chunk;
#pragma unroll 4
            for (int r = 0; r < nr; ++r) {
                const uint4 *row = reinterpret_cast<const uint4 *>(sbase + (size_t)r * gate_row_bytes);
                float acc[BT];
#pragma unroll
                for (int b = 0; b < BT; ++b) acc[b] = 0.f;
#pragma unroll
                for (int i = 0; i < VPT; ++i) {
                    const int v = tid + i * kConsumers;
                    if (v < HV) {
                        float f[8];
                        unpack8(row[v], f);
#pragma unroll
                        for (int b = 0; b < BT; ++b)
#pragma unroll
                            for (int e = 0; e < 8; ++e) acc[b] = fmaf(f[e], xv[b][i][e], acc[b]);
                    }
                }
#pragma unroll
                for (int b = 0; b < BT; ++b) acc[b] = warp_sum(acc[b]);
                if (lane == 0) {
#pragma unroll
                    for (int b = 0; b < BT; ++b) S.gpart[buf][r0 + r][b][warp] = acc[b];
                }
            }
            __syncwarp();
            if (lane == 0) mbar_arrive(&S.empty[stage]);
            if (last) {
                if (!csync(lane, &S.abort)) { S.abort = 1; flag_status(p.ctl, kStatusTimeout); return; }
                if (warp == 0) chunk_lists<BT, VPT>(p, S, buf, chunk, lane);
            }
        } else {
            const int ub = ud_seq & 1;
#pragma unroll 2
            for (int k = 0; k < nr; ++k) {
                const uint4 *up = reinterpret_cast<const uint4 *>(sbase + (size_t)k * ud_row_bytes);
                float acc[BT];
#pragma unroll
                for (int b = 0; b < BT; ++b) acc[b] = 0.f;
#pragma unroll
                for (int i = 0; i < VPT; ++i) {
                    const int v = tid + i * kConsumers;
                    if (v < HV) {
                        float f[8];
                        unpack8(up[v], f);
#pragma unroll
                        for (int b = 0; b < BT; ++b)
#pragma unroll
                            for (int e = 0; e < 8; ++e) acc[b] = fmaf(f[e], xv[b][i][e], acc[b]);
                    }
                }
#pragma unroll
                for (int b = 0; b < BT; ++b) acc[b] = warp_sum(acc[b]);
                if (lane == 0) {
#pragma unroll
                    for (int b = 0; b < BT; ++b) S.upart[ub][k][b][warp] = acc[b];
                }
            }
            if (!csync(lane, &S.abort)) { S.abort = 1; flag_status(p.ctl, kStatusTimeout); return; }
            for (int k = 0; k < nr; ++k) {
                float h[BT];
#pragma unroll
                for (int b = 0; b < BT; ++b) {
                    float u = S.upart[ub][k][b][lane & (kConsumerWarps - 1)];
                    u += __shfl_xor_sync(0xffffffffu, u, 4);
                    u += __shfl_xor_sync(0xffffffffu, u, 2);
                    u += __shfl_xor_sync(0xffffffffu, u, 1);
                    h[b] = d.am[k][b] * u;     // CATS_t(a) * (x W_up), Eqs. 1 and 5
                }
                const uint4 *down = reinterpret_cast<const uint4 *>(sbase + (size_t)k * ud_row_bytes + (size_t)H * 2);
#pragma unroll
                for (int i = 0; i < VPT; ++i) {
                    const int v = tid + i * kConsumers;
                    if (v < HV) {
                        float f[8];
                        unpack8(down[v], f);
#pragma unroll
                        for (int b = 0; b < BT; ++b)
#pragma unroll
                            for (int e = 0; e < 8; ++e) yv[b][i][e] = fmaf(h[b], f[e], yv[b][i][e]);
                    }
                }
            }
            __syncwarp();
            if (lane == 0) mbar_arrive(&S.empty[stage]);
            ++ud_seq;
        }
        if (++stage == kStages) { stage = 0; phase ^= 1u; }
    }
}

// ------------------------------------------------------------------ grid-wide tail
__device__ bool grid_barrier(int *ctl)
{
    __shared__ int ok_s;
    __syncthreads();
    if (threadIdx.x == 0) {
        int ok = 1;
        __threadfence();
        const int gen = ld_acquire_gpu(ctl + kCtlBarGen);
        const int arrived = atomicAdd(ctl + kCtlBarCount, 1);
        if (arrived == (int)gridDim.x - 1) {
            atomicExch(ctl + kCtlBarCount, 0);
            atomicExch(ctl + kCtlChunk, 0);
            __threadfence();
            st_release_gpu(ctl + kCtlBarGen, gen + 1);
        } else {
            const unsigned long long t0 = global_ns();
            while (ld_acquire_gpu(ctl + kCtlBarGen) == gen) {
                if (global_ns() - t0 > kWaitLimitNs) {
                    flag_status(ctl, kStatusTimeout);
                    ok = 0;
                    break;
                }
                __nanosleep(64);
            }
        }
        __threadfence();
        ok_s = ok;
    }
    __syncthreads();
    return ok_s != 0;
}

template <int BT>
__device__ void reduce_partials(const FusedParams &p)
{
    const int H4 = p.H >> 2;
    const int total = p.nb * H4;                       // float4 elements of y for this pass
    const int G = gridDim.x;
    const int per = (total + G - 1) / G;
    const int q0 = blockIdx.x * per;
    const int q1 = min(total, q0 + per);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int nwarps = kThreads / 32;
    const float4 *part = reinterpret_cast<const float4 *>(p.partials);
    for (int q = q0 + warp; q < q1; q += nwarps) {
        const int b = q / H4, c4 = q - b * H4;
        float4 s = make_float4(0.f, 0.f, 0.f, 0.f);
        for (int g = lane; g < G; g += 32) {
            const float4 v = __ldcg(part + ((size_t)g * kMaxTokensPerPass + b) * H4 + c4);
            s.x += v.x; s.y += v.y; s.z += v.z; s.w += v.w;
        }
        s.x = warp_sum(s.x); s.y = warp_sum(s.y); s.z = warp_sum(s.z); s.w = warp_sum(s.w);
        if (lane == 0) {
            float4 *dst = reinterpret_cast<float4 *>(p.out) + (size_t)b * H4 + c4;
            if (p.out_mode == kOutResid) {
                const float4 r = __ldcg(dst);
                s.x += r.x; s.y += r.y; s.z += r.z; s.w += r.w;
            }
            *dst = s;
        }
    }
}

template <int BT>
__device__ void compact_indices(const FusedParams &p, Shared<BT> &S, int *prefix)
{
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int nw = kThreads / 32;
    const int nc = p.nchunks;
    const int stride = nc * kChunk;
    const int per = (nc + kThreads - 1) / kThreads;
    for (int b = 0; b < p.nb; ++b) {
        // exclusive scan of the per-chunk counts of token b
        const int c0 = min(nc, tid * per), c1 = min(nc, c0 + per);
        int local = 0;
        for (int c = c0; c < c1; ++c) local += __ldcg(p.chunk_cnt + c * kMaxTokensPerPass + b);
        int incl = local;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int v = __shfl_up_sync(0xffffffffu, incl, o);
            if (lane >= o) incl += v;
        }
        if (lane == 31) S.warp_sums[warp] = incl;
        __syncthreads();
        int base = 0;
        for (int w = 0; w < warp; ++w) base += S.warp_sums[w];
        int run = base + incl - local;
        for (int c = c0; c < c1; ++c) {
            prefix[c] = run;
            run += __ldcg(p.chunk_cnt + c * kMaxTokensPerPass + b);
        }
        if (blockIdx.x == 0 && tid == kThreads - 1) {
            int tot = 0;
            for (int w = 0; w < nw; ++w) tot += S.warp_sums[w];
            if (p.active_cnt) p.active_cnt[b] = tot;
        }
        __syncthreads();
        // copy this CTA's chunks (c = blockIdx.x + k * gridDim.x), 16 entries each
        const int slots = kThreads / kChunk;   // chunks per sweep
        for (int s0 = 0;; s0 += slots) {
            const int ci = s0 + tid / kChunk;
            const int c = blockIdx.x + ci * gridDim.x;
            if (blockIdx.x + s0 * gridDim.x >= nc) break;
            const int k = tid % kChunk;
            if (c < nc && tid < slots * kChunk) {
                const int cnt = __ldcg(p.chunk_cnt + c * kMaxTokensPerPass + b);
                if (k < cnt)
                    p.active_idx[(size_t)b * p.N + prefix[c] + k] = __ldcg(p.idx_tmp + b * stride + c * kChunk + k);
            }
        }
        __syncthreads();
    }
}

template <int BT, int VPT>
__global__ void __launch_bounds__(kThreads, 1) fused_mlp_kernel(const FusedParams p)
{
    extern __shared__ __align__(128) uint8_t smem[];
    uint8_t *stages = smem;
    Shared<BT> &S = *reinterpret_cast<Shared<BT> *>(smem + (size_t)kStages * kStageBytes);
    const int tid = threadIdx.x;
    const int warp = tid >> 5, lane = tid & 31;

    if (tid == 0) {
        for (int s = 0; s < kStages; ++s) {
            mbar_init(&S.full[s], 1);
            mbar_init(&S.empty[s], kConsumerWarps);
            S.issued[s] = 0;
        }
        mbar_init(&S.listready[0], 1);
        mbar_init(&S.listready[1], 1);
        mbar_init(&S.csync, kConsumerWarps);
        S.abort = 0;
        mbar_init_fence();
    }
    if (tid < BT) {
        float t = INFINITY;
        if (tid < p.nb) t = (p.dense_flags && p.dense_flags[tid]) ? 0.f : p.t_l;
        S.thr[tid] = t;
    }
    __syncthreads();

    float yv[BT][VPT][8];
    if (warp == kConsumerWarps) {
        if (lane == 0) {
            producer<BT>(p, S, stages);
            if (S.abort) drain_copies<BT>(S);
        }
        __syncwarp();
    } else {
        consumer<BT, VPT>(p, S, stages, yv);
        // y partial of this CTA: partials[blockIdx.x][b][:]
        const int HV = p.H >> 3;
#pragma unroll
        for (int b = 0; b < BT; ++b) {
            if (b >= p.nb) break;
#pragma unroll
            for (int i = 0; i < VPT; ++i) {
                const int v = tid + i * kConsumers;
                if (v < HV) {
                    float4 *dst = reinterpret_cast<float4 *>(
                        p.partials + ((size_t)blockIdx.x * kMaxTokensPerPass + b) * p.H + (size_t)v * 8);
                    dst[0] = make_float4(yv[b][i][0], yv[b][i][1], yv[b][i][2], yv[b][i][3]);
                    dst[1] = make_float4(yv[b][i][4], yv[b][i][5], yv[b][i][6], yv[b][i][7]);
                }
            }
        }
    }
    if (!grid_barrier(p.ctl)) return;
    reduce_partials<BT>(p);
    if (p.active_idx && !S.abort) compact_indices<BT>(p, S, reinterpret_cast<int *>(stages));
}

template <int BT, int VPT>
cudaError_t launch_t(const FusedParams &p, int grid, cudaStream_t stream)
{
    static unsigned long long configured = 0;   // one bit per device ordinal
    const size_t smem = smem_bytes<BT>();
    int dev = 0;
    cudaGetDevice(&dev);
    const unsigned long long bit = 1ull << (dev & 63);
    if (!(configured & bit)) {
        cudaError_t e = cudaFuncSetAttribute(fused_mlp_kernel<BT, VPT>,
                                             cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        if (e != cudaSuccess) return e;
        configured |= bit;
    }
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(grid);
    cfg.blockDim = dim3(kThreads);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeCooperative;
    attr[0].val.cooperative = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, fused_mlp_kernel<BT, VPT>, p);
}

}  // namespace

int fused_grid(int nchunks)
{
    int dev = 0, sms = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    int g = sms < kMaxGrid ? sms : kMaxGrid;
    if (nchunks < g) g = nchunks;
    return g < 1 ? 1 : g;
}

cudaError_t launch_fused(const FusedParams &p, cudaStream_t stream)
{
    const int grid = fused_grid(p.nchunks);
    // vectors of 8 bf16 per consumer thread and row: VPT = ceil(H / 8 / 256)
    const int vpt = p.H <= 2048 ? 1 : (p.H <= 4096 ? 2 : 4);
    if (vpt == 1) {
        if (p.nb <= 1) return launch_t<1, 1>(p, grid, stream);
        if (p.nb <= 2) return launch_t<2, 1>(p, grid, stream);
        return launch_t<4, 1>(p, grid, stream);
    }
    if (vpt == 2) {
        if (p.nb <= 1) return launch_t<1, 2>(p, grid, stream);
        if (p.nb <= 2) return launch_t<2, 2>(p, grid, stream);
        return launch_t<4, 2>(p, grid, stream);
    }
    if (p.nb <= 1) return launch_t<1, 4>(p, grid, stream);
    if (p.nb <= 2) return launch_t<2, 4>(p, grid, stream);
    return cudaErrorInvalidValue;   // callers split H > 4096 into passes of <= 2 tokens
}

}  // namespace sats
