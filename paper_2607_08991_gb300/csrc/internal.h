// internal.h -- declarations shared by the library's translation units.
#pragma once

#include <cstddef>
#include <cstdint>
#include <cuda_runtime.h>

#include "sats.h"

struct sats_layer {
    int H = 0;
    int N = 0;
    int device = 0;
    uint16_t *wg_t = nullptr;   // [N][H]: row j = column j of W_gate
    uint16_t *w_ud = nullptr;   // [N][2H]: row j = column j of W_up, then row j of W_down
    // Tensor-core path: the same weights cut into tiles of 64 K-elements whose
    // rows (128 bytes each) are contiguous, so that one TMA box is one
    // contiguous read.  Padding rows and columns are zero.
    uint16_t *gu_blk = nullptr;   // [tc_T][tc_kbh][2][tc_R][64]: W_gate then W_up columns of neuron tile t
    uint16_t *wd_blk = nullptr;   // [tc_dt][tc_kbn][128][64]: W_down columns of hidden tile d, neuron block kb
    int tc_R = 0;                 // neurons per tile (a multiple of 16, at most 128)
    int tc_T = 0;                 // neuron tiles, ceil(N / tc_R)
    int tc_kbh = 0;               // ceil(H / 64)
    int tc_dt = 0;                // hidden tiles, ceil(H / 128)
    int tc_kbn = 0;               // ceil(N / 64)
    int ldn = 0;                  // row stride of h (N rounded up to a multiple of 8)
};

// A LoRA adapter of one MLP block for the sparse path of a fine-tuned model
// (Sec. 4): W + scale A B for gate, up and down, packed for the fused kernel.
struct sats_lora {
    int H = 0, N = 0, r = 0, device = 0;
    float scale = 0.f;
    uint16_t *blk = nullptr;      // [ceil(N / 8)][8][3 r]: neuron j's B_gate[:, j], B_up[:, j], A_down[j, :]
    uint16_t *agu = nullptr;      // [H][2 r]: A_gate[h, :], A_up[h, :]
    uint16_t *bd = nullptr;       // [r][H]: B_down
};

namespace sats {

constexpr int kChunk = 8;               // neurons per scheduling unit of the fused kernel
constexpr int kMaxTokensPerPass = 4;    // tokens one fused launch carries
constexpr int kMaxGrid = 256;           // upper bound of the fused grid
constexpr int kMaxH = 8192;
constexpr int kMaxN = 1 << 20;
constexpr int kMaxLoraRank = 32;        // LoRA rank of the fused kernel, a multiple of 8
constexpr int kLoraZCopies = 16;        // copies of the x A sums, CTA c adding into copy c mod 16

// Control block at the start of the workspace (ints).
enum {
    kCtlChunk = 0,      // next dynamically claimed chunk of the fused kernel (reset by the last CTA)
    kCtlBarCount = 1,   // reserved
    kCtlBarGen = 2,     // reserved
    kCtlStatus = 3,     // device status word (kStatus* bits)
    kCtlNDense = 4,     // route output of the stack driver
    kCtlPrologue = 5,   // CTAs that have read their activations (reset by the last CTA)
    kCtlDone = 6,       // CTAs past their last use of the counters (reset by the last CTA)
    kCtlSelftest = 7,   // stays 0: the wait self-test polls it until its time limit
    kCtlInts = 64
};

// Workspace regions.  flags: the fused kernel's index-list words, one 64-bit
// word per chunk of kChunk neurons (its kept rows) and one per CTA (its slice's
// kept counts and prefix), cleared by the kernel itself at the start of each call.
struct WsLayout {
    size_t ctl, lora_z, flags, route_perm, route_flags, tc, total;
};

// Zeroes the control words of a workspace (the fused kernel's counters and status).
cudaError_t clear_fused_state(void *ws, int H, int N, int B, cudaStream_t stream);
WsLayout ws_layout(int H, int N, int B);

enum XMode { kXBf16 = 0, kXF32 = 1, kXResidNorm = 2 };
enum OutMode { kOutY = 0, kOutResid = 1 };

struct FusedParams {
    const uint16_t *wg_t;
    const uint16_t *w_ud;
    int H, N, nchunks;
    int nb;                       // tokens in this pass, 1..kMaxTokensPerPass
    int x_mode;
    const void *x;                // first token of this pass ([nb][H])
    const float *norm_w;          // kXResidNorm: RMSNorm gain [H]
    float eps;
    float t_l;                    // threshold of sparse-path tokens
    const uint8_t *dense_flags;   // [nb] (1 = base path, threshold 0) or nullptr
    int out_mode;
    float *out;                   // kOutY: y [nb][H]; kOutResid: residual [nb][H] (+=)
    int *ctl;                     // workspace control block
    uint64_t *flags;              // [nchunks]: index-list words (index output only)
    int32_t *active_idx;          // [nb][N] or nullptr
    int32_t *active_cnt;          // [nb] or nullptr
    uint8_t *keep_trace;          // [nb][N] or nullptr
    const sats_lora *lora;        // host view of the adapter, or nullptr (the kernel reads the fields below)
    const uint16_t *lora_blk, *lora_agu, *lora_bd;
    int lora_r;
    float lora_scale;
    float *lora_z;                // [kLoraZCopies][kMaxTokensPerPass][2 kMaxLoraRank]: partial sums of x A_gate, x A_up
};

// Records the CUDA error behind a SATS_ECUDA result (per host thread), with a
// static description of the step that failed; returns SATS_ECUDA.
sats_status cuda_fail(cudaError_t e, const char *where);

// Number of CTAs the fused kernel runs with on `device` (all co-resident).
int fused_grid(int nchunks);
int fused_tokens_per_pass(int H);
cudaError_t launch_fused(const FusedParams &p, cudaStream_t stream);
// small_mlp.cu: a pass of nb <= 2 tokens on a small layer (hidden <= 1024, a few thousand
// neurons; use_small_path says which) runs as one thread-block cluster with no workspace use
// beyond the status word.
bool use_small_path(int H, int N, int nb);
cudaError_t launch_small(const FusedParams &p, cudaStream_t stream);

cudaError_t launch_pack(const uint16_t *Wg, const uint16_t *Wu, const uint16_t *Wd, int H, int N,
                        uint16_t *wg_t, uint16_t *w_ud, cudaStream_t stream);
cudaError_t launch_pack_lora(const uint16_t *Ag, const uint16_t *Bg, const uint16_t *Au, const uint16_t *Bu,
                             const uint16_t *Ad, const uint16_t *Bd, int H, int N, int r, sats_lora *l,
                             cudaStream_t stream);

// Tensor-core path (gemm_tc.cu) for batches larger than one fused pass.
// tc_pack_layer allocates and fills gu_blk / wd_blk from wg_t and w_ud;
// tc_free_layer releases them.
cudaError_t tc_pack_layer(sats_layer *layer, cudaStream_t stream);
cudaError_t tc_free_layer(sats_layer *layer);
bool use_tc_path(int H, int B);
size_t tc_workspace_bytes(int H, int N, int B);
// union_mlp.cu: whether a batch may take the union path (B <= 8 sparse-path
// tokens, H <= 4096), and its list, up and down kernels after the gate-only kernel.
bool union_path_ok(int H, int B);
cudaError_t launch_union_tail(const sats_layer *layer, int B, const uint16_t *xa, const uint16_t *xlo,
                              const uint8_t *uflag, int32_t *ulist, int32_t *ucount, const float *a_keep, int lda,
                              float *u, int ldu, float *out, int *ctl, cudaStream_t stream);
cudaError_t run_tc_layer(const sats_layer *layer, int x_mode, const void *x, int B, float t_l, const float *norm_w,
                         float eps, const uint8_t *dense_flags, const int32_t *perm, const int32_t *n_dense,
                         int out_mode, float *out, int32_t *active_idx, int32_t *active_cnt, uint8_t *keep_trace,
                         void *tc_ws, int *ctl, cudaStream_t stream, bool union_path = false);
cudaError_t launch_wait_timeout(int *ctl, cudaStream_t stream);
cudaError_t launch_route(const int32_t *ids, int B, const uint8_t *lut, int V, int32_t *perm,
                         int32_t *n_dense, uint8_t *flags, int32_t *status, cudaStream_t stream);
cudaError_t launch_gate_act(const sats_layer *layer, const uint16_t *x, int B, float *a,
                            cudaStream_t stream);
cudaError_t launch_gate_act_f32(const sats_layer *layer, const float *x, int B, float *a, cudaStream_t stream);

// One block over B tokens (fused kernel or tensor cores), as the C ABI calls run it
// (api.cu).  ws: a workspace of ws_layout(H, N, B).total bytes with zeroed control words.
// dense_flags (per token, original order) serve the fused passes; perm / n_dense (the
// routing kernel's output) serve the tensor-core path, which then works in routed order.
sats_status run_layer(const sats_layer *layer, int x_mode, const void *x, int B, const float *t_l,
                      const float *norm_w, float eps, const uint8_t *dense_flags, int out_mode, float *out,
                      int32_t *active_idx, int32_t *active_cnt, uint8_t *keep_trace, void *ws, cudaStream_t stream,
                      const sats_lora *lora = nullptr, const int32_t *perm = nullptr,
                      const int32_t *n_dense = nullptr);
size_t select_ws_bytes();
cudaError_t launch_select(const float *a, int64_t n, int64_t m, void *ws, float *t_dev,
                          cudaStream_t stream);

}  // namespace sats
