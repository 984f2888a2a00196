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
// One CTA per SM, 608 threads in five roles, two shared-memory rings fed by
// cp.async.bulk copies that complete on per-stage mbarriers:
//   * gate producer (one thread): works through chunks of 8 neurons: first the
//     CTA's fixed chunks c, c + G, ... (four, three with a LoRA adapter; it
//     streams the first and brings the others into L2 before the previous call
//     has finished), then chunks claimed in increasing order from one counter,
//     so that faster SMs take more of them (over the last chunks, only while its
//     W_ud rows keep up); a chunk is started only when one of four list buffers
//     is free.  Streams gate rows into the gate ring (5 x 16 KB).
//   * 8 gate warps: thread t owns the 16-byte vectors t, t + 256, ... of every
//     gate row and keeps the matching activations in registers as float pairs;
//     dot products use paired FP32 FMAs (fma.rn.f32x2), four rows per
//     transposed warp reduction (stages of one or two rows taken in pairs);
//     per-warp partials go to the chunk's list buffer, then each warp arrives on
//     the buffer's barrier.
//   * list producer (one warp, lane = row): sums the partials of a chunk,
//     applies SiLU (Eq. 2) and the mask (Eqs. 4-5) per token, publishes the
//     chunk's kept counts, frees the buffer, and streams the W_ud rows of the
//     kept neurons into the W_ud ring (4 slots of 32 KB).
//   * index warp: waits until every CTA has cleared its chunk words (the words
//     are then this call's) and tells the gate warps.  Once their stream has
//     ended, the gate warps turn the kept rows of the CTA's slice of consecutive
//     chunks into their entries of the ascending index lists: a chunk's place in
//     the list is the number of neurons kept in all earlier chunks, summed
//     directly from those chunks' published words (256 threads, one round of
//     loads once the words are there), so no CTA waits on another's sums.
//   * 8 up/down warps: thread t owns vectors t, t + 256, ... of the up and
//     down halves of each W_ud row and keeps its y columns in registers.  The
//     up dot products of a stage are reduced across these warps through a
//     split barrier: each warp arrives, performs the down projection of the
//     previous stage (h_j * W_down[j, :] into its y columns), then waits.
// The two groups run concurrently, so neither kind of row waits behind the
// other.  After its stream each CTA adds its y partial into the output with
// vector reductions in L2 (red.global.add.v4.f32); a counter guarantees that
// every CTA has read its activations (the residual stream, which the output
// may alias), zeroed its slice of y and cleared its slice of the chunk flags
// before any CTA adds or touches a flag.  The last CTA to finish resets the
// counters.
// Every wait is bounded in time; a wait that gives up sets the status word.
#include <cmath>

#include "common.cuh"
#include "internal.h"

namespace sats {
namespace {

constexpr int kGateWarps = 8;
constexpr int kUdWarps = 8;
constexpr int kGateThreads = kGateWarps * 32;        // 256
constexpr int kUdThreads = kUdWarps * 32;            // 256
constexpr int kGateProducerWarp = kGateWarps + kUdWarps;   // 16
constexpr int kListWarp = kGateProducerWarp + 1;           // 17
constexpr int kIndexWarp = kListWarp + 1;                  // 18
constexpr int kThreads = (kIndexWarp + 1) * 32;            // 608
constexpr int kGateStageBytes = 16384;
constexpr int kGateStages = 5;
constexpr int kUdRingBytes = 131072;
constexpr int kUdSlots = 4;
constexpr int kUdSlotBytes = kUdRingBytes / kUdSlots;      // 32 KB
constexpr int kBufs = 4;                                   // list buffers (gate lookahead, chunks)
// Fixed chunks per CTA before the claimed ones, and the gate bytes of the fixed chunks past
// the first brought into L2 before the previous call ends.  With a LoRA adapter the first
// mask waits for every CTA's share of x A, and the deeper prefetch measured slower there.
template <bool LORA> constexpr int kStaticChunks = LORA ? 3 : 4;
template <bool LORA> constexpr uint32_t kL2PrefetchBytes = (LORA ? 128u : 192u) * 1024u;
constexpr int kTailChunks = 4;                             // the last kTailChunks * G chunks are claimed ...
constexpr int kTailLag = 2;                                // ... only kTailLag chunks ahead of the W_ud rows
constexpr int kPendingChunks = 16;                        // chunk words held back until every CTA has cleared its flags
constexpr int kMaxUdRows = 8;                              // W_ud rows per stage (small H)
constexpr int kSliceWords = 64;                            // a slice's chunk words kept in shared memory

// Index-list words (the flags region: one word per chunk; CTA c's slice of the
// lists is chunks [c per, (c + 1) per), per = ceil(nchunks / G)).  Chunk word:
// [63:62] status (0: not yet published this call, kChunkKept: published),
// [8b + 7:8b] the rows of the chunk kept for token b.  Every CTA clears the words
// of its slice before it passes its prologue, and the words are written and read
// only after every CTA has passed it.  A word holds its whole payload and moves
// only from 0 to its final value, so the accesses are relaxed.
constexpr uint64_t kChunkKept = 1ull << 62;

__device__ __forceinline__ uint32_t flag_state(uint64_t f) { return (uint32_t)(f >> 62); }
__device__ __forceinline__ uint32_t chunk_rows(uint64_t f, int b) { return (uint32_t)(f >> (8 * b)) & 0xFFu; }

enum StageKind { kRows = 0, kEnd = 1 };

struct GateDesc {
    int kind, nrows, chunk_pos, last, buf, pad0, pad1, pad2;
};

template <int BT>
struct UdDesc {
    int kind, nrows, pad0, pad1;
    float am[kMaxUdRows][BT];   // keep ? a : 0, per row and token
};

template <int BT>
struct Shared {
    uint64_t gfull[kGateStages], gempty[kGateStages];
    uint64_t ufull[kUdSlots], uempty[kUdSlots];
    uint64_t gsync[kBufs];      // gate partials of a buffer written (one arrival per gate warp)
    uint64_t bfree[kBufs];      // buffer's list formed (one arrival by the list producer)
    uint64_t xloaded;           // every consumer warp holds its activations
    uint64_t gbar;              // gate-warp barrier
    uint64_t ubar;              // up/down-warp barrier
    GateDesc gdesc[kGateStages];
    UdDesc<BT> udesc[kUdSlots];
    float gpart[kBufs][kChunk][BT][kGateWarps];
    float upart[3][kMaxUdRows][BT][kUdWarps];   // by W_ud stage, mod 3
    int chunkq[kBufs];          // first neuron of the chunk in a buffer (-1: no more work)
    int chunkrows[kBufs];
    int gissued[kGateStages], uissued[kUdSlots];
    float thr[BT];              // per-token threshold, written and read by the list producer
    float red[kGateWarps + kUdWarps][BT];
    uint64_t pend_word[kPendingChunks];   // chunk words not yet published (list producer)
    int pend_chunk[kPendingChunks];
    int abort;
    int seen;                   // the list producer has seen every CTA past its prologue
    int flags_ready;            // index warp: 1 once every CTA has cleared its chunk words, -1 if that wait gave up
    uint32_t ired[kGateWarps][2];   // per-warp kept counts of the chunks before this CTA's slice
    uint64_t sword[kSliceWords];    // the chunk words of this CTA's slice (slices of up to kSliceWords chunks)
    int quiet;                  // roles past their last use of the counters (list producer, index warp)
    int ldone;                  // chunks whose W_ud rows the list producer has issued (read by the gate producer)
};

// Extra shared state of the LoRA variant (Sec. 4, fine-tuned sparse path), placed
// after Shared<BT>, 128-byte aligned.
template <int BT>
struct LoraShared {
    uint16_t blk[kBufs][kChunk * 3 * kMaxLoraRank];        // the chunk's B_gate, B_up columns, A_down rows (pitch 3r)
    float z[BT][2 * kMaxLoraRank];                         // x A_gate, x A_up summed over every CTA
    float lu[kUdSlots][kMaxUdRows][BT];                    // scale (x A_up) B_up[:, j] of each W_ud row
    uint32_t ad[kUdSlots][kMaxUdRows][kMaxLoraRank / 2];   // A_down[j, :] of each W_ud row, bf16 pairs
    float w[BT][kMaxLoraRank];                             // this CTA's sum of h_j A_down[j, :]
    float zred[kUdWarps][BT][2 * kMaxLoraRank];            // per-warp partials of this CTA's slice of x A
    uint64_t zdone;                                        // this CTA's slice of x A has been added
};

template <int BT, bool LORA>
constexpr size_t smem_bytes()
{
    return (size_t)kGateStages * kGateStageBytes + kUdRingBytes + sizeof(Shared<BT>) +
           (LORA ? sizeof(LoraShared<BT>) + 128 : 0);
}

template <int BT>
__device__ __forceinline__ LoraShared<BT> &lora_of(Shared<BT> &S)
{
    const uintptr_t a = (reinterpret_cast<uintptr_t>(&S) + sizeof(Shared<BT>) + 127) & ~(uintptr_t)127;
    return *reinterpret_cast<LoraShared<BT> *>(a);
}

__device__ __forceinline__ void flag_status(int *ctl, int bits) { atomicOr(ctl + kCtlStatus, bits); }

// Geometry of the W_ud ring for a hidden size: rows per stage and slots per stage.
struct UdGeometry {
    int rows, slots, stages;
    size_t stage_bytes;
    __device__ explicit UdGeometry(int H)
    {
        const int row_bytes = 4 * H;
        rows = max(1, min(kMaxUdRows, kUdSlotBytes / row_bytes));
        slots = (rows * row_bytes + kUdSlotBytes - 1) / kUdSlotBytes;
        stages = kUdSlots / slots;
        stage_bytes = (size_t)slots * kUdSlotBytes;
    }
};

// Barrier over one warp group on an mbarrier (one arrival per warp), bounded in
// time; arrive() and wait() may be separated by independent work.
struct GroupSync {
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

// The RMSNorm gains of thread `t`'s vectors t + nthreads * i (a layer constant:
// loaded before the dependency wait, so that the normalisation does not wait for them).
template <int VPT>
__device__ __forceinline__ void load_norm_gains(const FusedParams &p, int t, int nthreads, float (&gw)[VPT][8])
{
    const int HV = p.H >> 3;
#pragma unroll
    for (int i = 0; i < VPT; ++i) {
        const int v = t + i * nthreads;
        float4 lo = make_float4(0.f, 0.f, 0.f, 0.f), hi = lo;
        if (p.x_mode == kXResidNorm && v < HV) {
            const float4 *gw4 = reinterpret_cast<const float4 *>(p.norm_w);
            lo = gw4[2 * v];
            hi = gw4[2 * v + 1];
        }
        gw[i][0] = lo.x; gw[i][1] = lo.y; gw[i][2] = lo.z; gw[i][3] = lo.w;
        gw[i][4] = hi.x; gw[i][5] = hi.y; gw[i][6] = hi.z; gw[i][7] = hi.w;
    }
}

// Activations of this pass for one warp group: thread `t` of `nthreads` owns
// the vectors t + nthreads * i (i < VPT).  RMSNorm (kXResidNorm) reduces over
// the group through `gs`, using red[red0 + warp-in-group], and scales by the
// gains `gain` (load_norm_gains).
template <int BT, int VPT>
__device__ bool load_activations(const FusedParams &p, Shared<BT> &S, GroupSync &gs, int t, int nthreads,
                                 int red0, const float (&gain)[VPT][8], f32x2 (&xp)[BT][VPT][4])
{
    const int lane = t & 31, gw = t >> 5, nw = nthreads >> 5;
    const int H = p.H, HV = H >> 3;
    float xv[BT][VPT][8];
#pragma unroll
    for (int b = 0; b < BT; ++b)
#pragma unroll
        for (int i = 0; i < VPT; ++i) {
            const int v = t + i * nthreads;
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
            for (int b = 0; b < BT; ++b) S.red[red0 + gw][b] = ss[b];
        }
        if (!gs(lane, &S.abort)) return false;
#pragma unroll
        for (int b = 0; b < BT; ++b) {
            float tot = 0.f;
            for (int w = 0; w < nw; ++w) tot += S.red[red0 + w][b];
            const float inv = 1.0f / sqrtf(tot / (float)H + p.eps);
#pragma unroll
            for (int i = 0; i < VPT; ++i) {
                const int v = t + i * nthreads;
                if (v < HV) {
#pragma unroll
                    for (int e = 0; e < 8; ++e) xv[b][i][e] = xv[b][i][e] * inv * gain[i][e];
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
    return true;
}

// ------------------------------------------------------------------ gate producer
template <int BT, bool LORA>
__device__ void gate_producer(const FusedParams &p, Shared<BT> &S, uint8_t *gring)
{
    const uint64_t pol = l2_policy_evict_first();
    const int H = p.H, N = p.N, G = gridDim.x, nch = p.nchunks;
    const uint32_t row_bytes = (uint32_t)H * 2u;
    const int rows_per_stage = min(kChunk, kGateStageBytes / (int)row_bytes);
    // chunk k holds neurons [8k, 8k + 8); chunks c + s G (s < kStaticChunks) are this
    // CTA's; the others, from kStaticChunks * G on, are claimed in increasing order
    constexpr int kStatic = kStaticChunks<LORA>;
    const int nstatic = kStatic * G;
    auto static_chunk = [&](int s) { return (int)blockIdx.x + s * G; };
    auto prefetch_fixed = [&]() {
        // The weights do not depend on the previous call: while it finishes (its tail
        // leaves HBM mostly idle), start moving this CTA's fixed chunks past the first
        // (which the gate ring takes) into L2.
        size_t left = kL2PrefetchBytes<LORA>;
        for (int s = 1; s < kStatic && left > 0; ++s) {
            const int k = static_chunk(s);
            if (k >= nch) break;
            const int n0 = k * kChunk;
            const char *src = reinterpret_cast<const char *>(p.wg_t + (size_t)n0 * H);
            size_t bytes = min(left, (size_t)min(kChunk, N - n0) * row_bytes);
            left -= bytes;
            for (size_t off = 0; bytes > 0;) {
                const uint32_t nbytes = (uint32_t)min(bytes, (size_t)65536);
                bulk_prefetch_l2(src + off, nbytes);
                off += nbytes;
                bytes -= nbytes;
            }
        }
    };
    int next_k = -1;       // a claimed chunk not yet started
    bool waited = false;   // the claim counter belongs to the previous call until that call has ended
    auto claim = [&]() {
        if (!waited) {
            grid_dependency_wait();
            waited = true;
        }
        return nstatic + atomicAdd(p.ctl + kCtlChunk, 1);
    };
    uint32_t stage = 0, phase = 0;
    bool ok = true;
    for (int seq = 0;; ++seq) {
        const int buf = seq % kBufs;
        // the buffer's previous list has been formed (first kBufs uses pass)
        if (!mbar_wait(&S.bfree[buf], ((uint32_t)(seq / kBufs) & 1u) ^ 1u, &S.abort)) { ok = false; break; }
        const bool fixed = seq < kStatic && static_chunk(seq) < nch;
        int k;
        if (fixed) {
            k = static_chunk(seq);
        } else {
            k = next_k >= 0 ? next_k : claim();
            next_k = -1;
        }
        const int n0 = k < nch ? k * kChunk : -1;
        if (n0 < 0) {
            S.chunkq[buf] = -1;                                   // end of work for the list producer
            for (int w = 0; w < kGateWarps; ++w) mbar_arrive(&S.gsync[buf]);
            break;
        }
        const int rows = min(kChunk, N - n0);
        S.chunkq[buf] = n0;
        S.chunkrows[buf] = rows;
        for (int r0 = 0; r0 < rows; r0 += rows_per_stage) {
            const int nr = min(rows_per_stage, rows - r0);
            if (!mbar_wait(&S.gempty[stage], phase ^ 1u, &S.abort)) { ok = false; break; }
            GateDesc &d = S.gdesc[stage];
            d.kind = kRows;
            d.nrows = nr;
            d.chunk_pos = r0;
            d.last = (r0 + nr >= rows) ? 1 : 0;
            d.buf = buf;
            S.gissued[stage] = (int)phase + 1;
            uint32_t extra = 0;   // the LoRA variant: the chunk's adapter block rides on its first stage
            if constexpr (LORA)
                if (r0 == 0) extra = (uint32_t)rows * 6u * (uint32_t)p.lora_r;
            mbar_arrive_expect_tx(&S.gfull[stage], (uint32_t)nr * row_bytes + extra);
            bulk_load(gring + (size_t)stage * kGateStageBytes, p.wg_t + (size_t)(n0 + r0) * H, (uint32_t)nr * row_bytes,
                      &S.gfull[stage], pol);
            if constexpr (LORA)
                if (extra)
                    bulk_load(lora_of(S).blk[buf], p.lora_blk + (size_t)n0 * 3 * p.lora_r, extra, &S.gfull[stage], pol);
            if (++stage == kGateStages) { stage = 0; phase ^= 1u; }
        }
        if (!ok) break;
        if (seq == 0) {
            // Only once the first chunk's rows have landed: issued together, every CTA's
            // prefetch of later chunks queued ahead of other CTAs' first rows in HBM, and the
            // first chunk's mask came 1.3 us after the dependency was released (instrumented).
            // (each ring slot on the latest phase this loop issued: only this thread re-arms a slot)
            for (int s2 = 0; s2 < kGateStages && ok; ++s2)
                if (S.gissued[s2] > 0) ok = mbar_wait(&S.gfull[s2], (uint32_t)(S.gissued[s2] - 1), &S.abort);
            if (!ok) break;
            prefetch_fixed();
        }
        // the next chunk is a claimed one: claim it while this chunk's rows stream.  Near the
        // end of the chunks, first let the list producer catch up (its W_ud rows issued up to
        // kTailLag chunks behind this one): a CTA whose kept rows pile up takes no more chunks,
        // so that the CTAs run out of W_ud rows at about the same time
        const bool next_fixed = seq + 1 < kStatic && static_chunk(seq + 1) < nch;
        if (!next_fixed) {
            if (k >= nch - kTailChunks * G) {
                const unsigned long long t0 = global_ns();
                while (*(volatile int *)&S.ldone < seq + 1 - kTailLag) {
                    if (global_ns() - t0 > kWaitLimitNs || *(volatile int *)&S.abort) { ok = false; break; }
                    __nanosleep(32);
                }
                if (!ok) break;
            }
            next_k = claim();
        }
    }
    if (ok && mbar_wait(&S.gempty[stage], phase ^ 1u, &S.abort)) {
        S.gdesc[stage].kind = kEnd;
        mbar_arrive(&S.gfull[stage]);
    } else {
        S.abort = 1;
        flag_status(p.ctl, kStatusTimeout);
    }
}

// ------------------------------------------------------------------ index lists
// The chunks [k0, k1) whose index-list entries CTA c writes.
__device__ __forceinline__ void list_slice(int nch, int &k0, int &k1)
{
    const int per = (nch + gridDim.x - 1) / gridDim.x;
    k0 = min(nch, (int)blockIdx.x * per);
    k1 = min(nch, k0 + per);
}

// Waits (bounded, with backoff) until chunk word k is published; returns it, or 0
// if the wait gave up.
template <int BT>
__device__ uint64_t await_word(const FusedParams &p, Shared<BT> &S, int k, unsigned long long t0)
{
    uint64_t w;
    uint32_t ns = 64;
    while (flag_state(w = ld_relaxed_gpu_u64(p.flags + k)) == 0u) {
        if (global_ns() - t0 > kWaitLimitNs || *(volatile int *)&S.abort) return 0ull;
        __nanosleep(ns);
        ns = min(ns * 2u, 512u);
    }
    return w;
}

// The gate warps, after their stream: the entries of this CTA's slice of the
// ascending index lists.  The entries of chunk k start at the number of neurons
// kept in chunks [0, k):
//   1. every thread reads its chunk words up to the slice's end (words t,
//      t + 256, ...; eight loads in flight; an unpublished word is awaited,
//      and taken as the wait read it), sums the kept rows of those before the slice
//      and leaves the slice's own words in shared memory; the sums are reduced
//      over the gate warps;
//   2. the first gate warp writes the slice's entries from a warp scan of its
//      chunks' counts, 32 chunks at a time, and the last slice the counts.
// Chunks are taken in increasing order, so the words before a slice are mostly
// published by the time this CTA's stream ends; the slices need no word but the
// chunks', and no CTA waits for another CTA's sums.
template <int BT>
__device__ void slice_index_lists(const FusedParams &p, Shared<BT> &S, GroupSync &gs, int t, int lane, int warp)
{
    static_assert(BT <= 2, "chunk words carry two tokens' rows");
    const int N = p.N, nch = p.nchunks;
    int k0, k1;
    list_slice(nch, k0, k1);
    if (k0 >= k1) return;
    const unsigned long long t0 = global_ns();
    int ready;
    while ((ready = *(volatile int *)&S.flags_ready) == 0) {
        if (global_ns() - t0 > kWaitLimitNs || *(volatile int *)&S.abort) {
            ready = -1;
            break;
        }
        __nanosleep(64);
    }
    bool ok = ready > 0;
    // 1.
    const bool own_in_smem = k1 - k0 <= kSliceWords;
    const int kend = own_in_smem ? k1 : k0;
    uint32_t pre0 = 0, pre1 = 0;
    for (int k = t; ok && k < kend; k += kGateThreads * 8) {
        uint64_t w[8];
#pragma unroll
        for (int i = 0; i < 8; ++i) {
            const int kk = k + kGateThreads * i;
            w[i] = kk < kend ? ld_relaxed_gpu_u64(p.flags + kk) : kChunkKept;
        }
        // every published word is taken now; an unpublished one is awaited and then taken
        // as the wait read it (no second load)
#pragma unroll
        for (int i = 0; i < 8; ++i) {
            const int kk = k + kGateThreads * i;
            if (kk >= kend || !ok) continue;
            if (flag_state(w[i]) == 0u) {
                w[i] = await_word<BT>(p, S, kk, t0);
                if (w[i] == 0ull) {
                    ok = false;
                    continue;
                }
            }
            if (kk < k0) {
                pre0 += (uint32_t)__popc(chunk_rows(w[i], 0));
                if (BT > 1) pre1 += (uint32_t)__popc(chunk_rows(w[i], 1));
            } else {
                S.sword[kk - k0] = w[i];
            }
        }
    }
    pre0 = (uint32_t)__reduce_add_sync(0xffffffffu, pre0);
    pre1 = (uint32_t)__reduce_add_sync(0xffffffffu, pre1);
    if (lane == 0) {
        S.ired[warp][0] = pre0;
        S.ired[warp][1] = pre1;
    }
    if (!__all_sync(0xffffffffu, ok) && lane == 0) {
        S.abort = 1;
        flag_status(p.ctl, kStatusTimeout);
    }
    if (!gs(lane, &S.abort) || warp != 0) return;
    // 2.
    uint32_t run[2] = {0u, 0u};
#pragma unroll
    for (int w = 0; w < kGateWarps; ++w) {
        run[0] += S.ired[w][0];
        run[1] += S.ired[w][1];
    }
    for (int base = k0; base < k1; base += 32) {
        const int k = base + lane;
        uint64_t f = 0ull;
        bool good = true;
        if (k < k1 && own_in_smem) {
            f = S.sword[k - k0];
        } else if (k < k1) {
            f = ld_relaxed_gpu_u64(p.flags + k);
            if (flag_state(f) == 0u) good = (f = await_word<BT>(p, S, k, t0)) != 0ull;
        }
        if (!__all_sync(0xffffffffu, good)) {
            if (lane == 0) {
                S.abort = 1;
                flag_status(p.ctl, kStatusTimeout);
            }
            return;
        }
#pragma unroll
        for (int b = 0; b < BT; ++b) {
            uint32_t m = k < k1 ? chunk_rows(f, b) : 0u;
            const uint32_t cnt = (uint32_t)__popc(m);
            uint32_t pre = cnt;
#pragma unroll
            for (int o = 1; o < 32; o <<= 1) {
                const uint32_t v = __shfl_up_sync(0xffffffffu, pre, o);
                if (lane >= o) pre += v;
            }
            uint32_t pos = run[b] + pre - cnt;
            for (; m; m &= m - 1u, ++pos) {
                if (pos < (uint32_t)N) p.active_idx[(size_t)b * N + pos] = k * kChunk + __ffs(m) - 1;
                else flag_status(p.ctl, kStatusInternal);
            }
            run[b] += __shfl_sync(0xffffffffu, pre, 31);
        }
    }
    if (k1 == nch && lane == 0 && p.active_cnt) {
#pragma unroll
        for (int b = 0; b < BT; ++b)
            if (b < p.nb) p.active_cnt[b] = (int)run[b];
    }
}

// ------------------------------------------------------------------ gate warps
template <int BT, int VPT>
__device__ void gate_warps(const FusedParams &p, Shared<BT> &S, const uint8_t *gring)
{
    const int t = threadIdx.x, lane = t & 31, warp = t >> 5;
    const int H = p.H, HV = H >> 3;
    const size_t row_bytes = (size_t)H * 2;
    const uint4 zero4 = make_uint4(0u, 0u, 0u, 0u);
    GroupSync gs{&S.gbar, 0u};
    f32x2 xp[BT][VPT][4];
    float gw[VPT][8];
    load_norm_gains<VPT>(p, t, kGateThreads, gw);
    grid_dependency_wait();   // x may be the previous launch's output
    const bool loaded = load_activations<BT, VPT>(p, S, gs, t, kGateThreads, 0, gw, xp);
    __syncwarp();
    if (lane == 0) mbar_arrive(&S.xloaded);
    if (!loaded) {
        S.abort = 1;
        flag_status(p.ctl, kStatusTimeout);
        return;
    }
    uint32_t stage = 0, phase = 0;
    for (;;) {
        if (!mbar_wait(&S.gfull[stage], phase, &S.abort)) {
            S.abort = 1;
            flag_status(p.ctl, kStatusTimeout);
            return;
        }
        const GateDesc &d0 = S.gdesc[stage];
        if (d0.kind == kEnd) break;
        const int nr0 = d0.nrows, r0 = d0.chunk_pos, buf = d0.buf;
        int last = d0.last;
        const uint8_t *sb0 = gring + (size_t)stage * kGateStageBytes;
        // Four rows share one transposed warp reduction (its shuffle chain bounds these
        // warps).  Stages of four rows or more are taken alone; stages of one or two rows
        // (H >= 4096) in pairs of one chunk, each stage released once its rows are in registers.
        int adv = 1;
        if (nr0 > 2) {
            for (int q = 0; q < nr0; q += 4) {
                f32x2 acc[4][BT];
#pragma unroll
                for (int r = 0; r < 4; ++r)
#pragma unroll
                    for (int b = 0; b < BT; ++b) acc[r][b] = 0ull;
#pragma unroll
                for (int i = 0; i < VPT; ++i) {
                    const int v = t + i * kGateThreads;
                    if (v < HV) {
                        uint4 w[4];
#pragma unroll
                        for (int r = 0; r < 4; ++r)
                            w[r] = q + r < nr0 ? reinterpret_cast<const uint4 *>(sb0 + (size_t)(q + r) * row_bytes)[v] : zero4;
#pragma unroll
                        for (int r = 0; r < 4; ++r)
#pragma unroll
                            for (int b = 0; b < BT; ++b) acc[r][b] = dot8_acc(w[r], xp[b][i], acc[r][b]);
                    }
                }
                if (q + 4 >= nr0) {   // every row of the stage is in registers: the producer may refill it
                    __syncwarp();
                    if (lane == 0) mbar_arrive(&S.gempty[stage]);
                }
#pragma unroll
                for (int b = 0; b < BT; ++b) {
                    const float tot = warp_sum4_transposed(hsum2(acc[0][b]), hsum2(acc[1][b]), hsum2(acc[2][b]),
                                                           hsum2(acc[3][b]), lane);
                    const int r = (lane >> 3) & 3;
                    if ((lane & 7) == 0 && q + r < nr0) S.gpart[buf][r0 + q + r][b][warp] = tot;
                }
            }
        } else {
            // acc[0..1]: this stage's rows; acc[2..3]: the next stage's, when the chunk goes on
            f32x2 acc[4][BT];
#pragma unroll
            for (int r = 0; r < 4; ++r)
#pragma unroll
                for (int b = 0; b < BT; ++b) acc[r][b] = 0ull;
            auto rows2 = [&](const uint8_t *sb, int n, int o) {
#pragma unroll
                for (int i = 0; i < VPT; ++i) {
                    const int v = t + i * kGateThreads;
                    if (v < HV) {
                        const uint4 w0 = reinterpret_cast<const uint4 *>(sb)[v];
                        const uint4 w1 = n > 1 ? reinterpret_cast<const uint4 *>(sb + row_bytes)[v] : zero4;
#pragma unroll
                        for (int b = 0; b < BT; ++b) {
                            acc[o][b] = dot8_acc(w0, xp[b][i], acc[o][b]);
                            acc[o + 1][b] = dot8_acc(w1, xp[b][i], acc[o + 1][b]);
                        }
                    }
                }
            };
            rows2(sb0, nr0, 0);
            __syncwarp();
            if (lane == 0) mbar_arrive(&S.gempty[stage]);
            int nr1 = 0;
            if (!last) {
                const uint32_t stage1 = stage + 1 == kGateStages ? 0u : stage + 1;
                const uint32_t phase1 = stage + 1 == kGateStages ? phase ^ 1u : phase;
                if (!mbar_wait(&S.gfull[stage1], phase1, &S.abort)) {
                    S.abort = 1;
                    flag_status(p.ctl, kStatusTimeout);
                    return;
                }
                const GateDesc &d1 = S.gdesc[stage1];
                nr1 = d1.nrows;
                last = d1.last;
                rows2(gring + (size_t)stage1 * kGateStageBytes, nr1, 2);
                __syncwarp();
                if (lane == 0) mbar_arrive(&S.gempty[stage1]);
                adv = 2;
            }
#pragma unroll
            for (int b = 0; b < BT; ++b) {
                const float tot = warp_sum4_transposed(hsum2(acc[0][b]), hsum2(acc[1][b]), hsum2(acc[2][b]),
                                                       hsum2(acc[3][b]), lane);
                const int j = (lane >> 3) & 3;   // rows j < 2 of this stage, j - 2 of the next
                const bool valid = j < 2 ? j < nr0 : j - 2 < nr1;
                if ((lane & 7) == 0 && valid) S.gpart[buf][r0 + (j < 2 ? j : nr0 + j - 2)][b][warp] = tot;
            }
        }
        __syncwarp();
        if (lane == 0 && last) mbar_arrive(&S.gsync[buf]);   // this warp's partials of the chunk are written
        for (int k = 0; k < adv; ++k)
            if (++stage == kGateStages) { stage = 0; phase ^= 1u; }
    }
    if (p.active_idx) slice_index_lists<BT>(p, S, gs, t, lane, warp);
}

// Waits (bounded) until every CTA has passed its prologue.
__device__ bool wait_prologues(int *ctl)
{
    const unsigned long long t0 = global_ns();
    while (ld_acquire_gpu(ctl + kCtlPrologue) < (int)gridDim.x) {
        if (global_ns() - t0 > kWaitLimitNs) {
            flag_status(ctl, kStatusTimeout);
            return false;
        }
        __nanosleep(64);
    }
    return true;
}

// Called once by the list producer and once by the index warp (one thread
// each), when each has made its last use of the control counters (the gate
// producer's claims precede the list producer's end).  The second call counts
// the CTA done; the last CTA counted resets the counters for the next call,
// which uses them only after this grid has ended.
template <int BT, bool LORA>
__device__ void counters_released(const FusedParams &p, Shared<BT> &S)
{
    uint32_t prior;
    asm volatile("atom.acq_rel.cta.shared.add.u32 %0, [%1], 1;" : "=r"(prior) : "r"(smem_addr(&S.quiet)) : "memory");
    if (prior != 1u) return;
    if (atom_add_acq_rel_gpu(p.ctl + kCtlDone, 1) == (int)gridDim.x - 1) {
        atomicExch(p.ctl + kCtlPrologue, 0);
        atomicExch(p.ctl + kCtlChunk, 0);
        atomicExch(p.ctl + kCtlDone, 0);
        if constexpr (LORA) {   // every CTA has read x A: clear the sums this call used, for the next call
            const int r2 = 2 * p.lora_r;
            for (int k = 0; k < kLoraZCopies; ++k)
                for (int b = 0; b < p.nb; ++b)
                    for (int c = 0; c < r2; c += 4)
                        *reinterpret_cast<float4 *>(p.lora_z + (k * kMaxTokensPerPass + b) * 2 * kMaxLoraRank + c) =
                            make_float4(0.f, 0.f, 0.f, 0.f);
        }
    }
}

// ------------------------------------------------------------------ list producer
// Lane r = row r of the chunk: sums the gate partials across the gate warps,
// SiLU (Eq. 2), CATS mask (Eqs. 4-5) per token, keep trace.  Returns the
// union of rows kept by any token, with each lane's a values and the kept rows
// per token.
template <int BT, bool LORA>
__device__ uint32_t chunk_keep(const FusedParams &p, Shared<BT> &S, int buf, int n0, int rows, int lane,
                               float (&a)[BT], uint32_t (&bal)[BT], float (&lu)[BT],
                               uint32_t (&adr)[kMaxLoraRank / 2])
{
    const bool in = lane < rows;
    uint32_t uni = 0;
    const uint16_t *lb = nullptr;   // LoRA: this row's B_gate column, B_up column, A_down row
    if constexpr (LORA) {
        lb = lora_of(S).blk[buf] + lane * 3 * p.lora_r;
#pragma unroll
        for (int q2 = 0; q2 < kMaxLoraRank / 2; ++q2)
            adr[q2] = (in && 2 * q2 < p.lora_r) ? reinterpret_cast<const uint32_t *>(lb + 2 * p.lora_r)[q2] : 0u;
    }
#pragma unroll
    for (int b = 0; b < BT; ++b) {
        float g = 0.f;
        if (in) {
#pragma unroll
            for (int w = 0; w < kGateWarps; ++w) g += S.gpart[buf][lane][b][w];
        }
        if constexpr (LORA) {
            // g += scale (x A_gate) B_gate[:, j];  the up term scale (x A_up) B_up[:, j] for the W_ud stage
            float lg = 0.f, lv = 0.f;
            if (in) {
                const float *z = lora_of(S).z[b];
                for (int q = 0; q < p.lora_r; ++q) {
                    lg = fmaf(z[q], __uint_as_float((uint32_t)lb[q] << 16), lg);
                    lv = fmaf(z[p.lora_r + q], __uint_as_float((uint32_t)lb[p.lora_r + q] << 16), lv);
                }
            }
            g = fmaf(p.lora_scale, lg, g);
            lu[b] = p.lora_scale * lv;
        }
        a[b] = g / (1.0f + expf(-g));                                   // SiLU, Eq. 2
        const bool keep = in && b < p.nb && fabsf(a[b]) >= S.thr[b];    // Eqs. 4-5
        bal[b] = __ballot_sync(0xffffffffu, keep);
        uni |= bal[b];
    }
    if (in) {
#pragma unroll
        for (int b = 0; b < BT; ++b) {
            if (b >= p.nb) break;
            if (p.keep_trace) p.keep_trace[(size_t)b * p.N + n0 + lane] = (uint8_t)((bal[b] >> lane) & 1u);
        }
    }
    return uni;
}

template <int BT, bool LORA>
__device__ void list_producer(const FusedParams &p, Shared<BT> &S, uint8_t *uring, int lane)
{
    const uint64_t pol = l2_policy_evict_first();
    const int H = p.H;
    const uint32_t ud_row_bytes = (uint32_t)H * 4u;
    const UdGeometry geo(H);
    const uint32_t lt = (1u << lane) - 1u;
    uint32_t stage = 0, phase = 0;
    grid_dependency_wait();   // the workspace and y belong to the previous launch until it ends
    if (lane < BT) {
        // per-token threshold (0: the token takes the dense path); only this warp reads it
        float t = INFINITY;
        if (lane < p.nb) t = (p.dense_flags && p.dense_flags[lane]) ? 0.f : p.t_l;
        S.thr[lane] = t;
    }
    __syncwarp();
    if (p.out_mode == kOutY) {
        // zero this CTA's slice of y; every CTA adds into y only after all
        // CTAs have passed their prologue (kCtlPrologue)
        const int total4 = p.nb * (p.H >> 2);
        const int per = (total4 + gridDim.x - 1) / gridDim.x;
        const int q1 = min(total4, (int)(blockIdx.x + 1) * per);
        for (int q = blockIdx.x * per + lane; q < q1; q += 32)
            reinterpret_cast<float4 *>(p.out)[q] = make_float4(0.f, 0.f, 0.f, 0.f);
    }
    if (p.active_idx) {
        // clear the chunk words of this CTA's slice (read and written only after every prologue)
        int j0, j1;
        list_slice(p.nchunks, j0, j1);
        for (int j = j0 + lane; j < j1; j += 32) p.flags[j] = 0ull;
    }
    __threadfence();
    bool ok = mbar_wait(&S.xloaded, 0u, &S.abort);
    if constexpr (LORA) ok = ok && mbar_wait(&lora_of(S).zdone, 0u, &S.abort);   // this CTA's slice of x A is added
    __syncwarp();
    if (ok && lane == 0) {
        // this CTA has read its activations, zeroed its slice of y and cleared its flags
        __threadfence();
        atomicAdd(p.ctl + kCtlPrologue, 1);
    }
    __syncwarp();
    // Lane 0 publishes each chunk's word once every CTA has cleared its words;
    // words of chunks finished before that wait in shared memory (and the warp
    // waits for the prologues once kPendingChunks of them are held).
    bool flags_open = false;
    int npend = 0;
    auto publish = [&](int k, uint64_t w, bool must) -> bool {
        if (!flags_open) flags_open = ld_acquire_gpu(p.ctl + kCtlPrologue) >= (int)gridDim.x;
        if (!flags_open && (must || npend == kPendingChunks)) {
            flags_open = wait_prologues(p.ctl);
            if (!flags_open) return false;
        }
        if (!flags_open) {
            S.pend_chunk[npend] = k;
            S.pend_word[npend] = w;
            ++npend;
            return true;
        }
        for (int i = 0; i < npend; ++i) st_relaxed_gpu_u64(p.flags + S.pend_chunk[i], S.pend_word[i]);
        npend = 0;
        if (k >= 0) st_relaxed_gpu_u64(p.flags + k, w);
        return true;
    };
    for (int seq = 0; ok; ++seq) {
        const int buf = seq % kBufs;
        if (!mbar_wait(&S.gsync[buf], (uint32_t)(seq / kBufs) & 1u, &S.abort)) { ok = false; break; }
        __syncwarp();
        const int n0 = S.chunkq[buf];
        if (n0 < 0) break;
        const int rows = S.chunkrows[buf];
        if constexpr (LORA) {
            if (seq == 0) {
                // x A (summed by every CTA before its prologue) is complete once every CTA is past it
                int open = 1;
                if (lane == 0 && !flags_open) open = (flags_open = wait_prologues(p.ctl)) ? 1 : 0;
                if (!__shfl_sync(0xffffffffu, open, 0)) { ok = false; break; }
                const int r2 = 2 * p.lora_r;
                for (int i = lane; i < BT * r2; i += 32) {
                    const int b = i / r2, c = i % r2;
                    float v[kLoraZCopies];
#pragma unroll
                    for (int k = 0; k < kLoraZCopies; ++k)
                        v[k] = b < p.nb ? __ldcg(p.lora_z + (k * kMaxTokensPerPass + b) * 2 * kMaxLoraRank + c) : 0.f;
                    float z = 0.f;
#pragma unroll
                    for (int k = 0; k < kLoraZCopies; ++k) z += v[k];
                    lora_of(S).z[b][c] = z;
                }
                __syncwarp();
            }
        }
        float a[BT], lu[BT];
        uint32_t bal[BT], adr[kMaxLoraRank / 2];
        const uint32_t uni = chunk_keep<BT, LORA>(p, S, buf, n0, rows, lane, a, bal, lu, adr);
        __syncwarp();
        if (lane == 0) mbar_arrive(&S.bfree[buf]);   // partials read: the gate producer may refill the buffer
        if (!p.active_idx) {
            if (lane == 0 && !flags_open) flags_open = ld_acquire_gpu(p.ctl + kCtlPrologue) >= (int)gridDim.x;
        } else {
            int good = 1;
            if (lane == 0) {
                uint64_t w = kChunkKept;
#pragma unroll
                for (int b = 0; b < BT; ++b)
                    if (b < p.nb) w |= (uint64_t)(bal[b] & 0xFFu) << (8 * b);
                good = publish(n0 / kChunk, w, false) ? 1 : 0;
            }
            if (!__shfl_sync(0xffffffffu, good, 0)) { ok = false; break; }
        }
        const int cnt = __popc(uni);
        const int pos = __popc(uni & lt);
        const bool mine = (uni >> lane) & 1u;
        const int nid = n0 + lane;
        for (int k0 = 0; k0 < cnt; k0 += geo.rows) {
            const int nr = min(geo.rows, cnt - k0);
            if (!mbar_wait(&S.uempty[stage], phase ^ 1u, &S.abort)) { ok = false; break; }
            UdDesc<BT> &d = S.udesc[stage];
            const bool in_stage = mine && pos >= k0 && pos < k0 + nr;
            if (in_stage) {
#pragma unroll
                for (int b = 0; b < BT; ++b) d.am[pos - k0][b] = ((bal[b] >> lane) & 1u) ? a[b] : 0.f;
                if constexpr (LORA) {
                    LoraShared<BT> &L = lora_of(S);
#pragma unroll
                    for (int b = 0; b < BT; ++b) L.lu[stage][pos - k0][b] = lu[b];
#pragma unroll
                    for (int q2 = 0; q2 < kMaxLoraRank / 2; ++q2) L.ad[stage][pos - k0][q2] = adr[q2];
                }
            }
            __syncwarp();     // descriptor entries written before lane 0's release below
            if (lane == 0) {
                d.kind = kRows;
                d.nrows = nr;
                S.uissued[stage] = (int)phase + 1;
                mbar_arrive_expect_tx(&S.ufull[stage], (uint32_t)nr * ud_row_bytes);
            }
            __syncwarp();
            if (in_stage)
                bulk_load(uring + (size_t)stage * geo.stage_bytes + (size_t)(pos - k0) * ud_row_bytes,
                          p.w_ud + (size_t)nid * 2 * H, ud_row_bytes, &S.ufull[stage], pol);
            __syncwarp();
            if (++stage == (uint32_t)geo.stages) { stage = 0; phase ^= 1u; }
        }
        if (!ok) break;
        if (lane == 0) *(volatile int *)&S.ldone = seq + 1;   // the gate producer may claim further
    }
    if (ok && p.active_idx) {
        int good = 1;
        if (lane == 0 && npend > 0) good = publish(-1, 0ull, true) ? 1 : 0;
        ok = __shfl_sync(0xffffffffu, good, 0) != 0;
    }
    if (lane == 0) {
        // the CTA adds into y only after every CTA has read its activations; the up/down
        // warps read this with the end marker below
        if (!flags_open && !*(volatile int *)&S.abort) flags_open = wait_prologues(p.ctl);
        S.seen = flags_open ? 1 : 0;
    }
    __syncwarp();
    if (ok && mbar_wait(&S.uempty[stage], phase ^ 1u, &S.abort)) {
        if (lane == 0) {
            S.udesc[stage].kind = kEnd;
            mbar_arrive(&S.ufull[stage]);
        }
    } else if (lane == 0) {
        S.abort = 1;
        flag_status(p.ctl, kStatusTimeout);
    }
    if (lane == 0) counters_released<BT, LORA>(p, S);
    __syncwarp();
}

// ------------------------------------------------------------------ index warp
// Index warp: its only use of the counters is to wait (bounded) until every CTA
// has cleared its chunk words; it then tells the gate warps (S.flags_ready) and
// releases the counters.
template <int BT, bool LORA>
__device__ void index_warp(const FusedParams &p, Shared<BT> &S, int lane)
{
    int k0, k1;
    list_slice(p.nchunks, k0, k1);
    // the control words and index words belong to the previous call until it has ended
    grid_dependency_wait();
    if (lane == 0) {
        int ready = 1;
        if (p.active_idx && k0 < k1) ready = wait_prologues(p.ctl) ? 1 : -1;
        *(volatile int *)&S.flags_ready = ready;
        counters_released<BT, LORA>(p, S);
    }
}

// ------------------------------------------------------------------ up/down warps
// Down projection of one W_ud stage: y[cols] += h_j * W_down[j, cols], with
// h_j = am_j * u_j and u_j the cross-warp sum of the stage's up partials; then
// releases the stage to the list producer.
template <int BT, int VPT, bool LORA>
__device__ __forceinline__ void down_stage(const FusedParams &p, Shared<BT> &S, const uint8_t *sbase, int nr,
                                           int ub, int st, int t, int lane, f32x2 (&yp)[BT][VPT][4],
                                           float (&wacc)[BT])
{
    const int H = p.H, HV = H >> 3;
    const size_t ud_row_bytes = (size_t)H * 4;
    for (int k = 0; k < nr; ++k) {
        f32x2 hh[BT];
#pragma unroll
        for (int b = 0; b < BT; ++b) {
            float u = S.upart[ub][k][b][lane & (kUdWarps - 1)];
#pragma unroll
            for (int o = kUdWarps / 2; o > 0; o >>= 1) u += __shfl_xor_sync(0xffffffffu, u, o);
            if constexpr (LORA) u += lora_of(S).lu[st][k][b];   // + scale (x A_up) B_up[:, j]
            const float h = S.udesc[st].am[k][b] * u;     // CATS_t(a) * (x W_up), Eqs. 1 and 5
            hh[b] = pack2(h, h);
            if constexpr (LORA) {
                // the first up/down warp sums h_j A_down[j, :], lane q holding column q
                if (t < 32 && lane < p.lora_r) {
                    const uint32_t wd = lora_of(S).ad[st][k][lane >> 1];
                    wacc[b] = fmaf(h, __uint_as_float((lane & 1) ? (wd & 0xffff0000u) : (wd << 16)), wacc[b]);
                }
            }
        }
        const uint4 *down = reinterpret_cast<const uint4 *>(sbase + (size_t)k * ud_row_bytes + (size_t)H * 2);
#pragma unroll
        for (int i = 0; i < VPT; ++i) {
            const int v = t + i * kUdThreads;
            if (v < HV) {
                const uint4 w = down[v];
#pragma unroll
                for (int b = 0; b < BT; ++b) axpy8(w, hh[b], yp[b][i]);
            }
        }
    }
    __syncwarp();
    if (lane == 0) mbar_arrive(&S.uempty[st]);
}

// Returns true once the end marker has been taken and this thread's y columns are final.
template <int BT, int VPT, bool LORA>
__device__ bool updown_warps(const FusedParams &p, Shared<BT> &S, const uint8_t *uring, f32x2 (&yp)[BT][VPT][4])
{
    float wacc[BT];   // LoRA: this lane's column of sum_j h_j A_down[j, :] (first warp only)
#pragma unroll
    for (int b = 0; b < BT; ++b) wacc[b] = 0.f;
    const int t = threadIdx.x - kGateThreads;
    const int lane = t & 31, uw = t >> 5;
    const int H = p.H, HV = H >> 3;
    const size_t ud_row_bytes = (size_t)H * 4;
    const UdGeometry geo(H);
    const uint4 zero4 = make_uint4(0u, 0u, 0u, 0u);
    GroupSync us{&S.ubar, 0u};

#pragma unroll
    for (int b = 0; b < BT; ++b)
#pragma unroll
        for (int i = 0; i < VPT; ++i)
#pragma unroll
            for (int e = 0; e < 4; ++e) yp[b][i][e] = 0ull;
    f32x2 xp[BT][VPT][4];
    float gw[VPT][8];
    load_norm_gains<VPT>(p, t, kUdThreads, gw);
    grid_dependency_wait();
    const bool loaded = load_activations<BT, VPT>(p, S, us, t, kUdThreads, kGateWarps, gw, xp);
    __syncwarp();
    if (lane == 0) mbar_arrive(&S.xloaded);
    if (!loaded) {
        S.abort = 1;
        flag_status(p.ctl, kStatusTimeout);
        return false;
    }
    if constexpr (LORA) {
        // While no W_ud row can arrive yet (the first one follows the first chunk's mask, which
        // needs x A_gate from every CTA): this CTA's share of x A_gate, x A_up over hidden rows
        // [h0, h1).  Thread t takes row h0 + 32 pass + t / 8 and columns (t % 8) cw .. + cw - 1;
        // the partials are summed over the rows in the warp (shuffles), then over the warps
        // (shared memory), and added into one of kLoraZCopies copies of the sums.
        LoraShared<BT> &L = lora_of(S);
        const int r2 = 2 * p.lora_r, cw = r2 / 8;   // 2, 4, 6 or 8 columns per thread
        const int h0 = (int)(((long long)H * blockIdx.x) / gridDim.x);
        const int h1 = (int)(((long long)H * (blockIdx.x + 1)) / gridDim.x);
        const int cg = t & 7;
        float zp[BT][8];
#pragma unroll
        for (int b = 0; b < BT; ++b)
#pragma unroll
            for (int c = 0; c < 8; ++c) zp[b][c] = 0.f;
        for (int h = h0 + (t >> 3); h < h1; h += kUdThreads / 8) {
            float xv[BT];
#pragma unroll
            for (int b = 0; b < BT; ++b)
                xv[b] = b >= p.nb ? 0.f
                        : p.x_mode == kXBf16
                            ? __uint_as_float((uint32_t)static_cast<const uint16_t *>(p.x)[(size_t)b * H + h] << 16)
                            : static_cast<const float *>(p.x)[(size_t)b * H + h];
            const uint16_t *arow = p.lora_agu + (size_t)h * r2 + cg * cw;
#pragma unroll
            for (int c = 0; c < 8; ++c) {
                if (c < cw) {
                    const float av = __uint_as_float((uint32_t)arow[c] << 16);
#pragma unroll
                    for (int b = 0; b < BT; ++b) zp[b][c] = fmaf(xv[b], av, zp[b][c]);
                }
            }
        }
        // lanes l, l ^ 8, l ^ 16, l ^ 24 hold the same columns for four rows
#pragma unroll
        for (int b = 0; b < BT; ++b)
#pragma unroll
            for (int c = 0; c < 8; ++c) {
                zp[b][c] += __shfl_xor_sync(0xffffffffu, zp[b][c], 8);
                zp[b][c] += __shfl_xor_sync(0xffffffffu, zp[b][c], 16);
            }
        if (lane < 8) {
#pragma unroll
            for (int b = 0; b < BT; ++b)
#pragma unroll
                for (int c = 0; c < 8; ++c)
                    if (c < cw) L.zred[uw][b][cg * cw + c] = zp[b][c];
        }
        if (!us(lane, &S.abort)) {
            S.abort = 1;
            flag_status(p.ctl, kStatusTimeout);
            return false;
        }
        if (t < BT * r2) {
            const int b = t / r2, c = t % r2;
            float z = 0.f;
#pragma unroll
            for (int w = 0; w < kUdWarps; ++w) z += L.zred[w][b][c];
            if (b < p.nb && h1 > h0)   // one of kLoraZCopies copies: few additions per address
                atomicAdd(p.lora_z + ((blockIdx.x % kLoraZCopies) * kMaxTokensPerPass + b) * 2 * kMaxLoraRank + c, z);
        }
        __threadfence();
        if (!us(lane, &S.abort)) {
            S.abort = 1;
            flag_status(p.ctl, kStatusTimeout);
            return false;
        }
        if (t == 0) mbar_arrive(&L.zdone);
    }
    uint32_t stage = 0, phase = 0;
    int ud_seq = 0;
    // a W_ud stage whose up sums are complete but whose down projection is
    // still to do (done while waiting on the next stage's barrier)
    int pend_stage = -1, pend_nr = 0, pend_ub = 0;
    for (;;) {
        if (!mbar_wait(&S.ufull[stage], phase, &S.abort)) {
            S.abort = 1;
            flag_status(p.ctl, kStatusTimeout);
            return false;
        }
        const UdDesc<BT> &d = S.udesc[stage];
        if (d.kind == kEnd) {
            if (pend_stage >= 0)
                down_stage<BT, VPT, LORA>(p, S, uring + (size_t)pend_stage * geo.stage_bytes, pend_nr, pend_ub,
                                          pend_stage, t, lane, yp, wacc);
            break;
        }
        const int nr = d.nrows;
        const int ub = ud_seq % 3;
        const uint8_t *sbase = uring + (size_t)stage * geo.stage_bytes;
        // up dot products, two rows per transposed reduction
        for (int q = 0; q < nr; q += 2) {
            f32x2 acc[2][BT];
#pragma unroll
            for (int r = 0; r < 2; ++r)
#pragma unroll
                for (int b = 0; b < BT; ++b) acc[r][b] = 0ull;
#pragma unroll
            for (int i = 0; i < VPT; ++i) {
                const int v = t + i * kUdThreads;
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
                if ((lane & 15) == 0 && q + r < nr) S.upart[ub][q + r][b][uw] = tot;
            }
        }
        us.arrive(lane);
        if (pend_stage >= 0)
            down_stage<BT, VPT, LORA>(p, S, uring + (size_t)pend_stage * geo.stage_bytes, pend_nr, pend_ub, pend_stage,
                                      t, lane, yp, wacc);
        if (!us.wait(&S.abort)) {
            S.abort = 1;
            flag_status(p.ctl, kStatusTimeout);
            return false;
        }
        pend_stage = (int)stage;
        pend_nr = nr;
        pend_ub = ub;
        ++ud_seq;
        if (++stage == (uint32_t)geo.stages) { stage = 0; phase ^= 1u; }
    }
    if constexpr (LORA) {
        // y += scale (sum_j h_j A_down[j, :]) B_down over this CTA's rows, before the L2 reduction
        LoraShared<BT> &L = lora_of(S);
        if (t < 32 && lane < p.lora_r) {
#pragma unroll
            for (int b = 0; b < BT; ++b) L.w[b][lane] = wacc[b];
        }
        if (!us(lane, &S.abort)) {
            S.abort = 1;
            flag_status(p.ctl, kStatusTimeout);
            return false;
        }
        // four rank columns at a time, their B_down loads issued together (the rank is a multiple of 8)
        for (int q0 = 0; q0 < p.lora_r; q0 += 4) {
            uint4 wv[4][VPT];
#pragma unroll
            for (int j = 0; j < 4; ++j)
#pragma unroll
                for (int i = 0; i < VPT; ++i) {
                    const int v = t + i * kUdThreads;
                    wv[j][i] = v < HV ? __ldg(reinterpret_cast<const uint4 *>(p.lora_bd + (size_t)(q0 + j) * H) + v)
                                      : make_uint4(0u, 0u, 0u, 0u);
                }
#pragma unroll
            for (int j = 0; j < 4; ++j) {
                f32x2 wq[BT];
#pragma unroll
                for (int b = 0; b < BT; ++b) {
                    const float v = p.lora_scale * L.w[b][q0 + j];
                    wq[b] = pack2(v, v);
                }
#pragma unroll
                for (int i = 0; i < VPT; ++i)
#pragma unroll
                    for (int b = 0; b < BT; ++b) axpy8(wv[j][i], wq[b], yp[b][i]);
            }
        }
    }
    return true;
}

// Bounded wait for every bulk copy still in flight (only on the error path).
template <int BT>
__device__ void drain_copies(Shared<BT> &S)
{
    int never = 0;
    for (int s = 0; s < kGateStages; ++s)
        if (S.gissued[s] > 0) (void)mbar_wait(&S.gfull[s], (uint32_t)(S.gissued[s] - 1), &never);
    for (int s = 0; s < kUdSlots; ++s)
        if (S.uissued[s] > 0) (void)mbar_wait(&S.ufull[s], (uint32_t)(S.uissued[s] - 1), &never);
}


// Adds up/down thread t's y columns into the output with L2 vector reductions.  Only
// once every CTA has passed its prologue (has read its activations, which the output
// may alias, and zeroed its slice of y).
template <int BT, int VPT>
__device__ __forceinline__ void add_partial_y(const FusedParams &p, const f32x2 (&yp)[BT][VPT][4], int t)
{
    const int HV = p.H >> 3;
#pragma unroll
    for (int b = 0; b < BT; ++b) {
        if (b >= p.nb) break;
#pragma unroll
        for (int i = 0; i < VPT; ++i) {
            const int v = t + i * kUdThreads;
            if (v < HV) {
                float *dst = p.out + (size_t)b * p.H + (size_t)v * 8;
                const float2 y0 = unpack2(yp[b][i][0]), y1 = unpack2(yp[b][i][1]);
                const float2 y2 = unpack2(yp[b][i][2]), y3 = unpack2(yp[b][i][3]);
                red_add_v4(dst, y0.x, y0.y, y1.x, y1.y);
                red_add_v4(dst + 4, y2.x, y2.y, y3.x, y3.y);
            }
        }
    }
}

template <int BT, int VPT, bool LORA>
__global__ void __launch_bounds__(kThreads, 1) fused_mlp_kernel(const FusedParams p)
{
    extern __shared__ __align__(128) uint8_t smem[];
    uint8_t *gring = smem;
    uint8_t *uring = smem + (size_t)kGateStages * kGateStageBytes;
    Shared<BT> &S = *reinterpret_cast<Shared<BT> *>(uring + kUdRingBytes);
    const int tid = threadIdx.x;
    const int warp = tid >> 5, lane = tid & 31;

    if (tid == 0) {
        for (int s = 0; s < kGateStages; ++s) {
            mbar_init(&S.gfull[s], 1);
            mbar_init(&S.gempty[s], kGateWarps);
            S.gissued[s] = 0;
        }
        for (int s = 0; s < kUdSlots; ++s) {
            mbar_init(&S.ufull[s], 1);
            mbar_init(&S.uempty[s], kUdWarps);
            S.uissued[s] = 0;
        }
        for (int b = 0; b < kBufs; ++b) {
            mbar_init(&S.gsync[b], kGateWarps);
            mbar_init(&S.bfree[b], 1);
        }
        mbar_init(&S.xloaded, kGateWarps + kUdWarps);
        if constexpr (LORA) mbar_init(&lora_of(S).zdone, 1);
        mbar_init(&S.gbar, kGateWarps);
        mbar_init(&S.ubar, kUdWarps);
        S.abort = 0;
        S.seen = 0;
        S.flags_ready = 0;
        S.quiet = 0;
        S.ldone = 0;
        mbar_init_fence();
    }
    __syncthreads();
    // the next launch in the stream may start its weight stream on SMs this
    // grid frees; it waits for this grid's end before touching x, y or the workspace
    grid_launch_dependents();

    f32x2 yp[BT][VPT][4];
    bool y_added = false;
    if (warp < kGateWarps) {
        gate_warps<BT, VPT>(p, S, gring);
    } else if (warp < kGateProducerWarp) {
        // the CTA's partial y goes out as soon as its last stage is done, while the gate warps
        // may still be writing the CTA's slice of the index lists
        if (updown_warps<BT, VPT, LORA>(p, S, uring, yp) && S.seen) {
            add_partial_y<BT, VPT>(p, yp, tid - kGateThreads);
            y_added = true;
        }
    } else if (warp == kGateProducerWarp) {
        if (lane == 0) gate_producer<BT, LORA>(p, S, gring);
        __syncwarp();
    } else if (warp == kListWarp) {
        list_producer<BT, LORA>(p, S, uring, lane);
    } else {
        index_warp<BT, LORA>(p, S, lane);
    }
    __syncthreads();
    if (tid == 0 && S.abort) drain_copies<BT>(S);

    // otherwise (a role gave up early) the partial y is added here, if the list producer has
    // seen every CTA past its prologue
    if (!y_added && S.seen && warp >= kGateWarps && warp < kGateProducerWarp)
        add_partial_y<BT, VPT>(p, yp, tid - kGateThreads);
}

template <int BT, int VPT, bool LORA>
cudaError_t launch_t(const FusedParams &p, int grid, cudaStream_t stream)
{
    static unsigned long long configured = 0;   // one bit per device ordinal
    const size_t smem = smem_bytes<BT, LORA>();
    int dev = 0;
    cudaGetDevice(&dev);
    const unsigned long long bit = 1ull << (dev & 63);
    if (!(configured & bit)) {
        cudaError_t e = cudaFuncSetAttribute(fused_mlp_kernel<BT, VPT, LORA>,
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
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, fused_mlp_kernel<BT, VPT, LORA>, p);
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

// 16-byte vectors per gate or up/down thread and row: ceil(H / 8 / 256).
static int fused_vectors_per_thread(int H) { return H <= 2048 ? 1 : (H <= 4096 ? 2 : 4); }

int fused_tokens_per_pass(int H) { return fused_vectors_per_thread(H) == 4 ? 1 : 2; }

cudaError_t launch_fused(const FusedParams &p, cudaStream_t stream)
{
    const int grid = fused_grid(p.nchunks);
    const int vpt = fused_vectors_per_thread(p.H);
    if (p.nb < 1 || p.nb > fused_tokens_per_pass(p.H)) return cudaErrorInvalidValue;
    if (p.lora_blk) {   // the LoRA variant
        if (p.lora_r < 8 || p.lora_r > kMaxLoraRank || (p.lora_r % 8) || p.x_mode == kXResidNorm)
            return cudaErrorInvalidValue;
        if (vpt == 1) return p.nb <= 1 ? launch_t<1, 1, true>(p, grid, stream) : launch_t<2, 1, true>(p, grid, stream);
        if (vpt == 2) return p.nb <= 1 ? launch_t<1, 2, true>(p, grid, stream) : launch_t<2, 2, true>(p, grid, stream);
        return launch_t<1, 4, true>(p, grid, stream);
    }
    if (vpt == 1) {
        if (p.nb <= 1) return launch_t<1, 1, false>(p, grid, stream);
        return launch_t<2, 1, false>(p, grid, stream);
    }
    if (vpt == 2) {
        if (p.nb <= 1) return launch_t<1, 2, false>(p, grid, stream);
        return launch_t<2, 2, false>(p, grid, stream);
    }
    return launch_t<1, 4, false>(p, grid, stream);
}

}  // namespace sats
