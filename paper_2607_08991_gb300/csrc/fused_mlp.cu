// fused_mlp.cu -- the CATS-thresholded gated MLP (Sec. 2, Eqs. 1-5 of
// arXiv 2607.08991) as one persistent, warp-specialised kernel for sm_103a.
//
// Per call, for nb tokens with per-token threshold t_b:
//   a_j = SiLU(x . W_gate[:, j]);  keep_bj = |a_bj| >= t_b
//   y_b = sum_j keep_bj * a_bj * (x_b . W_up[:, j]) * W_down[j, :]
//
// Layout (made by the packer): Wg_t [N][H] and W_ud [N][2H], so that the gate
// row of neuron j is 2H contiguous bytes and its up column + down row are 4H
// contiguous bytes.  A neuron no token keeps costs no HBM traffic beyond its
// gate row.
//
// One CTA per SM (544 threads, ~210 KB shared memory):
//   * producer warp: claims chunks of 8 neurons from a global counter and
//     streams them through a ring of 6 x 32 KB shared-memory stages with
//     cp.async.bulk copies that complete on per-stage mbarriers.  Stream
//     order: gate rows of chunks c0 .. cD (D = gate lookahead), then W_ud rows
//     of the kept neurons of c0, gate rows of c(D+1), W_ud rows of c1, ...
//     Once the consumers' gate partials of a chunk are in, the producer warp
//     forms its kept list itself (lane = row: SiLU, mask, ballots) and issues
//     the W_ud rows; the D chunks of gate rows in between keep the ring full
//     meanwhile.
//   * 16 consumer warps: thread t owns the 16-byte vectors t, t + 512 of
//     every row, keeps the matching activations and its y accumulators in
//     registers as float pairs, and computes with paired FP32 FMAs
//     (fma.rn.f32x2).  Gate rows are reduced four at a time with a transposed
//     warp reduction, then across warps through shared memory, and each warp
//     arrives on the chunk's barrier without waiting.  For a W_ud stage
//     the up dot products are reduced across warps through a split barrier:
//     each warp arrives, performs the down projection of the previous W_ud
//     stage (h_j * W_down[j, :] into its y columns), then waits.
//   * after the stream: each CTA writes its y partial; a bounded grid barrier;
//     every CTA sums a slice of y over the partials in a fixed order; the
//     per-chunk index lists are compacted into the ascending per-token list.
// Every wait is bounded in time; a wait that gives up sets the status word.
#include <cmath>

#include "common.cuh"
#include "internal.h"

namespace sats {
namespace {

constexpr int kConsumerWarps = 16;
constexpr int kConsumers = kConsumerWarps * 32;   // 512
constexpr int kThreads = kConsumers + 32;         // + producer warp
constexpr int kStageBytes = 32768;
constexpr int kStages = 6;
constexpr int kMaxLook = 4;                       // gate lookahead, chunks
constexpr int kBufs = kMaxLook + 1;
constexpr int kMaxRowsPerStage = 16;

enum StageKind { kGate = 0, kUpDown = 1, kEnd = 2 };

template <int BT>
struct StageDesc {
    int kind, nrows, chunk_pos, last, buf, chunk, pad0, pad1;
    int neuron[kMaxRowsPerStage];
    float am[kMaxRowsPerStage][BT];   // keep ? a : 0, per row and token
};

template <int BT>
struct Shared {
    uint64_t full[kStages];
    uint64_t empty[kStages];
    uint64_t csync;                                     // consumer-wide barrier (prologue, W_ud stages)
    uint64_t gsync[kBufs];                              // per chunk buffer: gate partials written
    StageDesc<BT> desc[kStages];
    float gpart[kBufs][kChunk][BT][kConsumerWarps];     // gate partials per chunk buffer
    float upart[3][kMaxRowsPerStage][BT][kConsumerWarps];   // by W_ud stage, mod 3
    int bufchunk[kBufs];
    int issued[kStages];                                // producer: parity+1 of last fill
    float thr[BT];
    float red[kConsumerWarps][BT];
    int warp_sums[kThreads / 32];
    int abort;
};

template <int BT>
constexpr size_t smem_bytes() { return (size_t)kStages * kStageBytes + sizeof(Shared<BT>); }

__device__ __forceinline__ void flag_status(int *ctl, int bits) { atomicOr(ctl + kCtlStatus, bits); }

// Consumer-wide barrier on an mbarrier (one arrival per consumer warp), bounded
// in time; arrive() and wait() may be separated by independent work.
struct ConsumerSync {
    uint64_t *bar;
    uint32_t parity;
    __device__ void arrive(int lane)
    {
        __syncwarp();
        if (lane == 0) mbar_arrive(bar);
    }
    __device__ bool wait(volatile int *abort)
    {
        const bool ok = mbar_wait(bar, parity, abort);
        parity ^= 1u;
        return ok;
    }
    __device__ bool operator()(int lane, volatile int *abort)
    {
        arrive(lane);
        return wait(abort);
    }
};

// ------------------------------------------------------------------ producer
// The kept list of one chunk, formed by the producer warp (lane r = row r):
// sums the consumers' gate partials across warps, applies SiLU (Eq. 2) and the
// CATS mask (Eqs. 4-5) per token, writes the optional index outputs, and
// returns the union of the rows kept by any token (a ballot mask) together
// with each lane's a values and keep bits.
template <int BT>
__device__ uint32_t chunk_keep(const FusedParams &p, Shared<BT> &S, int buf, int chunk, int lane, float (&a)[BT],
                               uint32_t (&bal)[BT])
{
    const int n0 = chunk * kChunk;
    const int rows = min(kChunk, p.N - n0);
    const bool in = lane < rows;
    uint32_t uni = 0;
#pragma unroll
    for (int b = 0; b < BT; ++b) {
        float g = 0.f;
        if (in) {
#pragma unroll
            for (int w = 0; w < kConsumerWarps; ++w) g += S.gpart[buf][lane][b][w];
        }
        a[b] = g / (1.0f + expf(-g));                                   // SiLU, Eq. 2
        const bool keep = in && b < p.nb && fabsf(a[b]) >= S.thr[b];    // Eqs. 4-5
        bal[b] = __ballot_sync(0xffffffffu, keep);
        uni |= bal[b];
    }
    const uint32_t lt = (1u << lane) - 1u;
    if (p.active_idx) {
        const int stride = p.nchunks * kChunk;
#pragma unroll
        for (int b = 0; b < BT; ++b) {
            if (b >= p.nb) break;
            if ((bal[b] >> lane) & 1u) p.idx_tmp[b * stride + n0 + __popc(bal[b] & lt)] = n0 + lane;
            if (lane == 0) p.chunk_cnt[chunk * kMaxTokensPerPass + b] = __popc(bal[b]);
        }
    }
    if (p.keep_trace && in) {
#pragma unroll
        for (int b = 0; b < BT; ++b)
            if (b < p.nb) p.keep_trace[(size_t)b * p.N + n0 + lane] = (uint8_t)((bal[b] >> lane) & 1u);
    }
    return uni;
}

// Runs on the whole producer warp with uniform control flow; lane 0 claims
// chunks and posts gate stages, every lane whose row is kept issues that row's
// W_ud copy.
template <int BT>
__device__ void producer(const FusedParams &p, Shared<BT> &S, uint8_t *stages, int look, int lane)
{
    const uint64_t pol = l2_policy_evict_first();
    const int H = p.H, N = p.N;
    const uint32_t gate_row_bytes = (uint32_t)H * 2u;
    const uint32_t ud_row_bytes = (uint32_t)H * 4u;
    const int rows_per_gate_stage = min(kChunk, kStageBytes / (int)gate_row_bytes);
    const int rows_per_ud_stage = min(kMaxRowsPerStage, kStageBytes / (int)ud_row_bytes);
    const int nbufs = look + 1;
    int *counter = p.ctl + kCtlChunk;
    const uint32_t lt = (1u << lane) - 1u;

    uint32_t stage = 0, phase = 0;
    int seq_gate = 0, seq_ud = 0;     // chunks whose gate / W_ud rows have been issued
    bool more = true, ok = true;
    int next = 0;
    if (lane == 0) next = atomicAdd(counter, 1);
    next = __shfl_sync(0xffffffffu, next, 0);

    for (;;) {
        // gate rows, up to `look` chunks ahead of the W_ud rows
        while (ok && more && seq_gate - seq_ud <= look) {
            const int c = next;
            if (c >= p.nchunks) { more = false; break; }
            if (lane == 0) next = atomicAdd(counter, 1);
            next = __shfl_sync(0xffffffffu, next, 0);
            const int buf = seq_gate % nbufs;
            const int n0 = c * kChunk;
            const int rows = min(kChunk, N - n0);
            for (int r0 = 0; r0 < rows; r0 += rows_per_gate_stage) {
                const int nr = min(rows_per_gate_stage, rows - r0);
                if (!mbar_wait(&S.empty[stage], phase ^ 1u, &S.abort)) { ok = false; break; }
                if (lane == 0) {
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
                }
                __syncwarp();
                if (++stage == kStages) { stage = 0; phase ^= 1u; }
            }
            if (lane == 0) S.bufchunk[buf] = c;
            ++seq_gate;
        }
        if (!ok || seq_ud == seq_gate) break;
        // kept list of the oldest chunk whose gate rows were issued, then its W_ud rows
        const int buf = seq_ud % nbufs;
        if (!mbar_wait(&S.gsync[buf], (uint32_t)(seq_ud / nbufs) & 1u, &S.abort)) { ok = false; break; }
        __syncwarp();
        const int chunk = S.bufchunk[buf];
        float a[BT];
        uint32_t bal[BT];
        const uint32_t uni = chunk_keep<BT>(p, S, buf, chunk, lane, a, bal);
        const int cnt = __popc(uni);
        const int pos = __popc(uni & lt);
        const bool mine = (uni >> lane) & 1u;
        const int nid = chunk * kChunk + lane;
        for (int k0 = 0; k0 < cnt; k0 += rows_per_ud_stage) {
            const int nr = min(rows_per_ud_stage, cnt - k0);
            if (!mbar_wait(&S.empty[stage], phase ^ 1u, &S.abort)) { ok = false; break; }
            StageDesc<BT> &d = S.desc[stage];
            const bool in_stage = mine && pos >= k0 && pos < k0 + nr;
            if (in_stage) {
                const int k = pos - k0;
                d.neuron[k] = nid;
#pragma unroll
                for (int b = 0; b < BT; ++b) d.am[k][b] = ((bal[b] >> lane) & 1u) ? a[b] : 0.f;
            }
            __syncwarp();     // descriptor entries written before lane 0's release below
            if (lane == 0) {
                d.kind = kUpDown;
                d.nrows = nr;
                S.issued[stage] = (int)phase + 1;
                mbar_arrive_expect_tx(&S.full[stage], (uint32_t)nr * ud_row_bytes);
            }
            __syncwarp();
            if (in_stage)
                bulk_load(stages + (size_t)stage * kStageBytes + (size_t)(pos - k0) * ud_row_bytes,
                          p.w_ud + (size_t)nid * 2 * H, ud_row_bytes, &S.full[stage], pol);
            __syncwarp();
            if (++stage == kStages) { stage = 0; phase ^= 1u; }
        }
        ++seq_ud;
    }
    if (ok && mbar_wait(&S.empty[stage], phase ^ 1u, &S.abort)) {
        if (lane == 0) {
            S.desc[stage].kind = kEnd;
            mbar_arrive(&S.full[stage]);
        }
    } else if (lane == 0) {
        S.abort = 1;
        flag_status(p.ctl, kStatusTimeout);
    }
    __syncwarp();
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
__device__ void load_activations(const FusedParams &p, Shared<BT> &S, ConsumerSync &csync, int tid,
                                 f32x2 (&xp)[BT][VPT][4], bool &ok)
{
    const int lane = tid & 31, warp = tid >> 5;
    const int H = p.H, HV = H >> 3;
    float xv[BT][VPT][8];
#pragma unroll
    for (int b = 0; b < BT; ++b)
#pragma unroll
        for (int i = 0; i < VPT; ++i) {
            const int v = tid + i * kConsumers;
#pragma unroll
            for (int e = 0; e < 8; ++e) xv[b][i][e] = 0.f;
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
        if (!csync(lane, &S.abort)) { ok = false; return; }
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
#pragma unroll
    for (int b = 0; b < BT; ++b)
#pragma unroll
        for (int i = 0; i < VPT; ++i)
#pragma unroll
            for (int e = 0; e < 4; ++e) xp[b][i][e] = pack2(xv[b][i][2 * e], xv[b][i][2 * e + 1]);
}

// Down projection of one W_ud stage: y[cols] += h_j * W_down[j, cols] for the
// stage's rows, with h_j = am_j * u_j and u_j the cross-warp sum of the stage's
// up partials.  Then releases the stage to the producer.
template <int BT, int VPT>
__device__ __forceinline__ void down_stage(const FusedParams &p, Shared<BT> &S, const uint8_t *sbase,
                                           const StageDesc<BT> &d, int nr, int ub, uint32_t stage, int tid, int lane,
                                           f32x2 (&yp)[BT][VPT][4])
{
    const int H = p.H, HV = H >> 3;
    const size_t ud_row_bytes = (size_t)H * 4;
    for (int k = 0; k < nr; ++k) {
        f32x2 hh[BT];
#pragma unroll
        for (int b = 0; b < BT; ++b) {
            float u = S.upart[ub][k][b][lane & (kConsumerWarps - 1)];
#pragma unroll
            for (int o = kConsumerWarps / 2; o > 0; o >>= 1) u += __shfl_xor_sync(0xffffffffu, u, o);
            const float h = d.am[k][b] * u;     // CATS_t(a) * (x W_up), Eqs. 1 and 5
            hh[b] = pack2(h, h);
        }
        const uint4 *down = reinterpret_cast<const uint4 *>(sbase + (size_t)k * ud_row_bytes + (size_t)H * 2);
#pragma unroll
        for (int i = 0; i < VPT; ++i) {
            const int v = tid + i * kConsumers;
            if (v < HV) {
                const uint4 w = down[v];
#pragma unroll
                for (int b = 0; b < BT; ++b) axpy8(w, hh[b], yp[b][i]);
            }
        }
    }
    __syncwarp();
    if (lane == 0) mbar_arrive(&S.empty[stage]);
}

template <int BT, int VPT>
__device__ void consumer(const FusedParams &p, Shared<BT> &S, const uint8_t *stages, f32x2 (&yp)[BT][VPT][4])
{
    const int tid = threadIdx.x;
    const int warp = tid >> 5, lane = tid & 31;
    const int H = p.H, HV = H >> 3;
    const size_t gate_row_bytes = (size_t)H * 2, ud_row_bytes = (size_t)H * 4;
    ConsumerSync csync{&S.csync, 0u};
    const uint4 zero4 = make_uint4(0u, 0u, 0u, 0u);

#pragma unroll
    for (int b = 0; b < BT; ++b)
#pragma unroll
        for (int i = 0; i < VPT; ++i)
#pragma unroll
            for (int e = 0; e < 4; ++e) yp[b][i][e] = 0ull;

    f32x2 xp[BT][VPT][4];
    bool ok = true;
    load_activations<BT, VPT>(p, S, csync, tid, xp, ok);
    if (!ok) { S.abort = 1; flag_status(p.ctl, kStatusTimeout); return; }

    uint32_t stage = 0, phase = 0;
    int ud_seq = 0;
    // a W_ud stage whose up sums are complete but whose down projection is
    // still to do (it is done while waiting on the next W_ud stage's barrier)
    int pend_stage = -1, pend_nr = 0, pend_ub = 0;
    for (;;) {
        if (!mbar_wait(&S.full[stage], phase, &S.abort)) {
            S.abort = 1;
            flag_status(p.ctl, kStatusTimeout);
            return;
        }
        const StageDesc<BT> &d = S.desc[stage];
        const int kind = d.kind;
        if (kind != kUpDown && pend_stage >= 0) {
            down_stage<BT, VPT>(p, S, stages + (size_t)pend_stage * kStageBytes, S.desc[pend_stage], pend_nr,
                                pend_ub, (uint32_t)pend_stage, tid, lane, yp);
            pend_stage = -1;
        }
        if (kind == kEnd) break;
        const uint8_t *sbase = stages + (size_t)stage * kStageBytes;
        const int nr = d.nrows;
        if (kind == kGate) {
            const int r0 = d.chunk_pos, buf = d.buf, last = d.last;
            for (int q = 0; q < nr; q += 4) {
                // four rows at once: independent FMA chains, one transposed reduction
                f32x2 acc[4][BT];
#pragma unroll
                for (int r = 0; r < 4; ++r)
#pragma unroll
                    for (int b = 0; b < BT; ++b) acc[r][b] = 0ull;
#pragma unroll
                for (int i = 0; i < VPT; ++i) {
                    const int v = tid + i * kConsumers;
                    if (v < HV) {
                        uint4 w[4];
#pragma unroll
                        for (int r = 0; r < 4; ++r)
                            w[r] = (q + r < nr)
                                       ? reinterpret_cast<const uint4 *>(sbase + (size_t)(q + r) * gate_row_bytes)[v]
                                       : zero4;
#pragma unroll
                        for (int r = 0; r < 4; ++r)
#pragma unroll
                            for (int b = 0; b < BT; ++b) acc[r][b] = dot8_acc(w[r], xp[b][i], acc[r][b]);
                    }
                }
#pragma unroll
                for (int b = 0; b < BT; ++b) {
                    const float tot = warp_sum4_transposed(hsum2(acc[0][b]), hsum2(acc[1][b]), hsum2(acc[2][b]),
                                                           hsum2(acc[3][b]), lane);
                    const int r = (lane >> 3) & 3;
                    if ((lane & 7) == 0 && q + r < nr) S.gpart[buf][r0 + q + r][b][warp] = tot;
                }
            }
            __syncwarp();
            if (lane == 0) {
                mbar_arrive(&S.empty[stage]);
                if (last) mbar_arrive(&S.gsync[buf]);   // this warp's partials of the chunk are written
            }
        } else {
            const int ub = ud_seq % 3;
            // up dot products, two rows at a time
            for (int q = 0; q < nr; q += 2) {
                f32x2 acc[2][BT];
#pragma unroll
                for (int r = 0; r < 2; ++r)
#pragma unroll
                    for (int b = 0; b < BT; ++b) acc[r][b] = 0ull;
#pragma unroll
                for (int i = 0; i < VPT; ++i) {
                    const int v = tid + i * kConsumers;
                    if (v < HV) {
                        uint4 w[2];
#pragma unroll
                        for (int r = 0; r < 2; ++r)
                            w[r] = (q + r < nr) ? reinterpret_cast<const uint4 *>(sbase + (size_t)(q + r) * ud_row_bytes)[v]
                                                : zero4;
#pragma unroll
                        for (int r = 0; r < 2; ++r)
#pragma unroll
                            for (int b = 0; b < BT; ++b) acc[r][b] = dot8_acc(w[r], xp[b][i], acc[r][b]);
                    }
                }
#pragma unroll
                for (int b = 0; b < BT; ++b) {
                    const float tot = warp_sum2_transposed(hsum2(acc[0][b]), hsum2(acc[1][b]), lane);
                    const int r = lane >> 4;
                    if ((lane & 15) == 0 && q + r < nr) S.upart[ub][q + r][b][warp] = tot;
                }
            }
            csync.arrive(lane);
            if (pend_stage >= 0) {
                down_stage<BT, VPT>(p, S, stages + (size_t)pend_stage * kStageBytes, S.desc[pend_stage], pend_nr,
                                    pend_ub, (uint32_t)pend_stage, tid, lane, yp);
            }
            if (!csync.wait(&S.abort)) { S.abort = 1; flag_status(p.ctl, kStatusTimeout); return; }
            pend_stage = (int)stage;
            pend_nr = nr;
            pend_ub = ub;
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
                __nanosleep(32);
            }
        }
        __threadfence();
        ok_s = ok;
    }
    __syncthreads();
    return ok_s != 0;
}

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
        // copy this CTA's chunks (c = blockIdx.x + k * gridDim.x)
        const int slots = kThreads / kChunk;   // chunks per sweep
        for (int s0 = 0;; s0 += slots) {
            if (blockIdx.x + s0 * gridDim.x >= nc) break;
            const int c = blockIdx.x + (s0 + tid / kChunk) * gridDim.x;
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
__global__ void __launch_bounds__(kThreads, 1) fused_mlp_kernel(const FusedParams p, int look)
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
        for (int b = 0; b < kBufs; ++b) mbar_init(&S.gsync[b], kConsumerWarps);
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

    f32x2 yp[BT][VPT][4];
    if (warp == kConsumerWarps) {
        producer<BT>(p, S, stages, look, lane);
        if (lane == 0 && S.abort) drain_copies<BT>(S);
        __syncwarp();
    } else {
        consumer<BT, VPT>(p, S, stages, yp);
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
                    const float2 y0 = unpack2(yp[b][i][0]), y1 = unpack2(yp[b][i][1]);
                    const float2 y2 = unpack2(yp[b][i][2]), y3 = unpack2(yp[b][i][3]);
                    dst[0] = make_float4(y0.x, y0.y, y1.x, y1.y);
                    dst[1] = make_float4(y2.x, y2.y, y3.x, y3.y);
                }
            }
        }
    }
    if (!grid_barrier(p.ctl)) return;
    reduce_partials(p);
    if (p.active_idx && !S.abort) compact_indices<BT>(p, S, reinterpret_cast<int *>(stages));
}

template <int BT, int VPT>
cudaError_t launch_t(const FusedParams &p, int grid, int look, cudaStream_t stream)
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
    return cudaLaunchKernelEx(&cfg, fused_mlp_kernel<BT, VPT>, p, look);
}

}  // namespace

int fused_grid(int nchunks)
{
    static int sms_by_dev[64] = {0};
    int dev = 0;
    cudaGetDevice(&dev);
    int &sms = sms_by_dev[dev & 63];
    if (sms == 0) cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    int g = sms < kMaxGrid ? sms : kMaxGrid;
    if (nchunks < g) g = nchunks;
    return g < 1 ? 1 : g;
}

// 16-byte vectors per consumer thread and row: ceil(H / 8 / 512).
static int fused_vectors_per_thread(int H) { return H <= 4096 ? 1 : 2; }

int fused_tokens_per_pass(int H) { return fused_vectors_per_thread(H) == 1 ? 2 : 1; }

cudaError_t launch_fused(const FusedParams &p, cudaStream_t stream)
{
    const int grid = fused_grid(p.nchunks);
    // chunks of gate rows kept in flight ahead of the W_ud rows: about 128 KB
    int look = (128 * 1024) / (kChunk * 2 * p.H);
    look = look < 1 ? 1 : (look > kMaxLook ? kMaxLook : look);
    const int vpt = fused_vectors_per_thread(p.H);
    if (p.nb < 1 || p.nb > fused_tokens_per_pass(p.H)) return cudaErrorInvalidValue;
    if (vpt == 1) {
        if (p.nb <= 1) return launch_t<1, 1>(p, grid, look, stream);
        return launch_t<2, 1>(p, grid, look, stream);
    }
    return launch_t<1, 2>(p, grid, look, stream);
}

}  // namespace sats
