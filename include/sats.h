/*
 * sats.h -- C ABI of the GB300 (sm_103a) library for the runtime path of
 * "Sensitivity-Aware Thresholding and Token Routing for Activation
 * Sparsification in Large Language Models" (arXiv 2607.08991).
 *
 * The path: the CATS-thresholded gated MLP (Sec. 2, Eqs. 1-5; SATS, Sec. 3.1,
 * keeps this runtime mask and only chooses the per-layer threshold t_l), run
 * under per-token routing between the base (dense) and sparse MLP through a
 * vocabulary lookup table (Sec. 3.2, Eq. 13 and Fig. 2), chained over a
 * stack of decoder MLP blocks with RMSNorm and a residual add.
 *
 * Conventions for every call
 *   - Matrices follow the paper's row-vector convention y = x W: W_gate and
 *     W_up are [H][N] (hidden x intermediate), W_down is [N][H]; activations
 *     are [B][H].  All arrays are row-major and contiguous.
 *   - bf16 data is passed as its 16-bit patterns (const void*, 2 bytes each).
 *   - Pointers marked "device" are CUDA device pointers on the current device;
 *     "host" pointers are ordinary host memory.  The caller owns every buffer
 *     it passes; the library keeps no pointer to caller memory after a call
 *     returns, except that work it enqueued on `stream` reads/writes them.
 *   - `stream` is a cudaStream_t (NULL = legacy default stream).  Every call
 *     that takes a stream only enqueues work on it and returns without
 *     synchronising, unless stated otherwise.
 *   - Argument errors are detected on the host and returned before anything is
 *     enqueued.  Errors found by a kernel (a token id outside the vocabulary, a
 *     wait that ran out of time) are recorded in a status word in the
 *     workspace (or in the caller's status word for sats_route) and returned by
 *     sats_get_error.  No call aborts, throws, or traps on the device.
 *   - Calls never allocate device memory, except sats_layer_create.
 *   - Requirements: H a multiple of 8 and 8 <= H <= 8192; N >= 1; B >= 0.
 *   - SM occupancy: the single-token / two-token decode kernel (the small-batch
 *     path of sats_sparse_mlp and the calls built on it) runs one CTA on every
 *     SM (about 216 KB of shared memory each) and its CTAs wait, bounded, for
 *     one another's prologue.  It needs every SM to become free while it runs:
 *     a kernel on another stream that holds SMs for longer than 2 s (a
 *     persistent kernel, or one spinning on a flag) makes the call give up with
 *     SATS_ETIMEOUT from sats_get_error, and y and the index lists are then
 *     incomplete.  Ordinary kernels on other streams only delay the call.  The
 *     kernel is not launched cooperatively: that guarantees co-residency but
 *     stops the next call from starting on SMs this call frees, which measured
 *     8 us slower per call on the Llama-shaped layer.
 */
#ifndef SATS_H
#define SATS_H

#include <stddef.h>
#include <stdint.h>

#if defined(__GNUC__)
#define SATS_API __attribute__((visibility("default")))
#else
#define SATS_API
#endif

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
    SATS_OK = 0,
    SATS_EINVAL = 1,    /* null pointer, negative size, NaN or negative threshold, bad k */
    SATS_ESHAPE = 2,    /* H not a multiple of 8, H or N out of range */
    SATS_ECUDA = 3,     /* a CUDA runtime call failed (launch, copy, allocation) */
    SATS_EDEVICE = 4,   /* a kernel reported bad input (token id outside [0, V)) or an internal fault */
    SATS_ETIMEOUT = 5,  /* a bounded device-side wait gave up */
    SATS_ENOSPACE = 6   /* workspace smaller than sats_workspace_bytes() */
} sats_status;

/* Opaque handle of one MLP block; owns its repacked device weights. */
typedef struct sats_layer sats_layer;
typedef struct sats_lora sats_lora;

/* Library version, (major << 16) | minor. */
SATS_API int sats_version(void);

/* Human-readable name of a status code (static string, never NULL). */
SATS_API const char *sats_status_string(sats_status s);

/*
 * sats_layer_create -- repack one gated-MLP block (Sec. 2, Eq. 1) for the
 * runtime path.
 *   W_gate, W_up : device bf16 [H][N];  W_down : device bf16 [N][H].
 * The handle stores two device arrays that it allocates (the only allocation
 * in this library): Wg_t [N][H] (row j = column j of W_gate) and
 * W_ud [N][2H] (row j = column j of W_up followed by row j of W_down), so that
 * the weights a kept neuron needs are one contiguous 4H-byte row and a
 * skipped neuron costs no memory traffic.  The repacking runs on `stream`;
 * the call synchronises `stream` before returning, after which the caller may
 * free the three source arrays.  *out receives the handle.
 */
SATS_API sats_status sats_layer_create(const void *W_gate, const void *W_up, const void *W_down,
                              int H, int N, void *stream, sats_layer **out);

/* Frees the handle's device arrays (synchronises the device first). */
SATS_API sats_status sats_layer_destroy(sats_layer *layer);

/* Reads back H and N of a layer (host outputs, may be NULL). */
SATS_API sats_status sats_layer_shape(const sats_layer *layer, int *H, int *N);

/*
 * Workspace.  Every compute call takes a device workspace `ws` of at least
 * sats_workspace_bytes(H, N, B) bytes (B = the largest batch the caller will
 * pass).  It holds scheduling counters, the device status word, the LoRA
 * path's partial sums (16 KB), one 64-bit word per 8 neurons (kept counts and
 * prefixes for the index outputs) and the routing scratch of sats_mlp_stack:
 * N bytes plus B * 5 plus about 19 KB.  A batch that runs on the
 * tensor cores (sats_uses_tensor_cores) also needs, per token, bf16 copies of
 * its activations and of h (two parts each) plus one keep byte per neuron:
 * about B * (4 H + 5 N) bytes more.  It must be
 * zero-filled once before first use (sats_workspace_init does that on
 * `stream`); every call leaves its counters at zero for the next call.  Calls
 * that share one workspace must not overlap on the GPU.
 */
SATS_API size_t sats_workspace_bytes(int H, int N, int B);
SATS_API sats_status sats_workspace_init(void *ws, size_t ws_bytes, void *stream);

/*
 * sats_sparse_mlp -- the CATS-thresholded gated MLP (Sec. 2, Eqs. 1-5):
 *   a = SiLU(x W_gate);  keep_j = |a_j| >= t_l;  y = ((keep * a) * (x W_up)) W_down
 * for each of B tokens, bf16 weights with fp32 accumulation.
 *
 * Two execution paths, chosen by batch size (sats_uses_tensor_cores):
 *  - small batches (B <= 2 for H <= 4096, B = 1 above) stream W_gate once per
 *    call and read only the W_up columns and W_down rows of kept neurons;
 *  - larger batches run as two tensor-core GEMMs over all neurons,
 *    [x W_gate | x W_up] and then h W_down, with the mask applied to
 *    h = CATS(SiLU(x W_gate)) * (x W_up) between them; h, and fp32
 *    activations, are carried as a bf16 high part plus a bf16 low part
 *    (about 16 significant bits) with fp32 accumulation.
 *   x          : device bf16 [B][H]
 *   t_l        : threshold, >= 0 (0 keeps every neuron: the dense MLP;
 *                +inf keeps none and gives y = 0).  NaN or < 0 -> SATS_EINVAL.
 *   y          : device fp32 [B][H], written.
 *   active_idx : device int32 [B][N] or NULL.  Row b receives the kept neuron
 *                indices of token b in increasing order (entries past the
 *                count are unspecified).
 *   active_cnt : device int32 [B] or NULL; the number of kept neurons per token.
 * active_idx and active_cnt must both be NULL or both be given.
 */
SATS_API sats_status sats_sparse_mlp(const sats_layer *layer, const void *x, int B, float t_l,
                            float *y, int32_t *active_idx, int32_t *active_cnt,
                            void *ws, size_t ws_bytes, void *stream);

/*
 * sats_sparse_mlp_fixed_scratch -- sats_sparse_mlp with no workspace argument,
 * for callers that cannot allocate device memory.  The paper has no
 * counterpart to this call.  Such callers include plug-ins whose host
 * application owns every device allocation through its own allocator, code
 * that runs where cudaMalloc is not permitted or would stall (it synchronises
 * the device), and plain C callers that link only this library and have no
 * device allocator at all.
 *
 * Arguments, results and errors are those of sats_sparse_mlp.  Instead of a
 * workspace the call uses one 256 KiB array in the library's device memory;
 * every GPU that loads the library holds this array until the process exits.
 * A call whose workspace would exceed the array, i.e. with
 * sats_workspace_bytes(H, N, B) > 256 KiB, is rejected with SATS_ENOSPACE
 * before anything is enqueued.  On the fused small-batch kernel (B <= 2 for
 * H <= 4096, B = 1 above) the workspace is one 64-bit word per 8 neurons plus
 * about 17 KB, which admits N up to about 245,000; a batch on the tensor-core
 * path (sats_uses_tensor_cores) also needs its staging (activations, h and
 * keep bytes per token, and padding to whole tiles), so only small layers fit
 * there: for example N <= 5504 at H = 8192, B = 2, and N <= 1008 at H = 4096,
 * B = 8.  The call allocates nothing: before its kernels it clears the
 * array's control words with cudaMemsetAsync on `stream`.
 *
 *   dev_status : device int32 [1] or NULL.  If given, it receives this call's
 *                device status word after the kernels, in stream order (0 when
 *                every bounded device wait completed); sats_get_status_word
 *                reads it back and returns SATS_OK, SATS_ETIMEOUT or
 *                SATS_EDEVICE.  Without it, device-side errors of this call (a
 *                bounded wait that gave up, leaving y and the index lists
 *                incomplete) are not reported.
 *
 * Each call looks up the array's device address on the current device
 * (cudaGetSymbolAddress, which neither allocates nor synchronises), so the
 * address is always that of the current device and context.  All calls share
 * the one array, so calls that can overlap on the GPU (on different streams,
 * or from several host threads without ordering) race and must be serialised
 * by the caller.
 */
SATS_API sats_status sats_sparse_mlp_fixed_scratch(const sats_layer *layer, const void *x, int B, float t_l,
                                                   float *y, int32_t *active_idx, int32_t *active_cnt,
                                                   int32_t *dev_status, void *stream);

/*
 * sats_uses_tensor_cores -- 1 if a call with batch B on a layer of hidden size
 * H runs on the tensor-core path described under sats_sparse_mlp (also for
 * sats_dense_mlp and for each block of sats_mlp_stack), 0 if it runs on the
 * fused small-batch kernel.  Pure host function.
 */
SATS_API int sats_uses_tensor_cores(int H, int B);

/*
 * sats_last_cuda_error -- text of the CUDA error behind the most recent
 * SATS_ECUDA returned on the calling host thread, with the step that failed
 * (a static or thread-local string, valid until the thread's next call).
 */
SATS_API const char *sats_last_cuda_error(void);

/* As sats_sparse_mlp, with fp32 activations x: device fp32 [B][H]. */
SATS_API sats_status sats_sparse_mlp_f32(const sats_layer *layer, const float *x, int B, float t_l,
                                float *y, int32_t *active_idx, int32_t *active_cnt,
                                void *ws, size_t ws_bytes, void *stream);

/*
 * sats_sparse_mlp_union, sats_sparse_mlp_union_f32 -- sats_sparse_mlp for a
 * batch of 3 to 8 tokens (H <= 4096), computed over the union of the tokens'
 * kept neurons: the gate runs over all neurons on the tensor cores; then only
 * neurons some token keeps have their W_up column and W_down row read, once for
 * the whole batch (Sec. 2, Eqs. 1-5 per token: each token still keeps exactly
 * its own neurons, so the result equals sats_sparse_mlp's).  This reads
 * 2HN (1 + 2 |U| / N) bytes instead of 6HN, |U| the union size, which pays
 * when the tokens' kept sets overlap strongly; for independent kept sets at
 * these batch sizes the default path of sats_sparse_mlp is faster.
 * Arguments, results and errors are those of sats_sparse_mlp (x bf16) and
 * sats_sparse_mlp_f32 (x fp32, carried as bf16 high and low parts), with a
 * workspace of sats_workspace_bytes(H, N, B); B outside [3, 8] or H > 4096
 * returns SATS_ESHAPE.
 */
SATS_API sats_status sats_sparse_mlp_union(const sats_layer *layer, const void *x, int B, float t_l, float *y,
                                           int32_t *active_idx, int32_t *active_cnt, void *ws, size_t ws_bytes,
                                           void *stream);
SATS_API sats_status sats_sparse_mlp_union_f32(const sats_layer *layer, const float *x, int B, float t_l,
                                               float *y, int32_t *active_idx, int32_t *active_cnt, void *ws,
                                               size_t ws_bytes, void *stream);

/*
 * LoRA-aware sparse path (Sec. 4, fine-tuned models: the sparse path of a routed
 * fine-tuned model runs the thresholded MLP on its adapted weights, with the
 * low-rank updates folded into the sparse kernel).  An adapter of rank r holds,
 * for each projection W of the block, factors A, B with W' = W + scale A B:
 *   A_gate, A_up [H][r], B_gate, B_up [r][N], A_down [N][r], B_down [r][H]
 * (device bf16, row-major; the adapter keeps its own packed copies, so the
 * caller may free them after sats_lora_create returns).  r is 8, 16, 24 or 32
 * (else SATS_ESHAPE); scale finite (else SATS_EINVAL).
 *
 * sats_sparse_mlp_lora computes, for each of B tokens,
 *   g = x W_gate + scale (x A_gate) B_gate,  a = SiLU(g),  keep = |a| >= t_l
 *   u = x W_up + scale (x A_up) B_up,        h = keep ? a u : 0
 *   y = h W_down + scale (h A_down) B_down
 * in the decode kernel: the gate's low-rank term for every neuron, the up and
 * down terms only for kept neurons; batches run as passes of that kernel.
 * Arguments, index outputs, workspace and errors are those of sats_sparse_mlp
 * (x bf16) and sats_sparse_mlp_f32 (x fp32); the adapter must match the
 * layer's H and N (else SATS_ESHAPE).
 */
SATS_API sats_status sats_lora_create(const sats_layer *layer, const void *A_gate, const void *B_gate,
                                      const void *A_up, const void *B_up, const void *A_down, const void *B_down,
                                      int r, float scale, void *stream, sats_lora **out);
SATS_API sats_status sats_lora_destroy(sats_lora *lora);
SATS_API sats_status sats_sparse_mlp_lora(const sats_layer *layer, const sats_lora *lora, const void *x, int B,
                                          float t_l, float *y, int32_t *active_idx, int32_t *active_cnt, void *ws,
                                          size_t ws_bytes, void *stream);
SATS_API sats_status sats_sparse_mlp_lora_f32(const sats_layer *layer, const sats_lora *lora, const float *x, int B,
                                              float t_l, float *y, int32_t *active_idx, int32_t *active_cnt,
                                              void *ws, size_t ws_bytes, void *stream);

/*
 * sats_dense_mlp -- the base gated MLP of Sec. 2, Eq. 1 (every neuron kept):
 *   x : device bf16 [B][H];  y : device fp32 [B][H].
 */
SATS_API sats_status sats_dense_mlp(const sats_layer *layer, const void *x, int B, float *y,
                           void *ws, size_t ws_bytes, void *stream);

/*
 * sats_route -- token routing by lookup table (Sec. 3.2, Eq. 13; Fig. 2).
 *   token_ids : device int32 [B]
 *   lut       : device uint8 [V]; lut[v] != 0 sends token id v to the base
 *               (dense) path, 0 to the sparse path.
 *   perm      : device int32 [B], written: the positions b of base-path tokens
 *               in increasing order, then those of sparse-path tokens in
 *               increasing order (a stable partition, bit-exact).
 *   n_dense   : device int32 [1], written: the number of base-path tokens.
 *   dev_status: device int32 [1] or NULL.  If a token id lies outside [0, V)
 *               the kernel ORs 1 into *dev_status and routes that token to the
 *               base path; sats_get_status_word reads it back.
 */
SATS_API sats_status sats_route(const int32_t *token_ids, int B, const uint8_t *lut, int V,
                       int32_t *perm, int32_t *n_dense, int32_t *dev_status, void *stream);

/*
 * sats_mlp_stack -- L decoder MLP blocks on a residual stream:
 *   for l in 0..L-1:  x <- x + MLP_l( RMSNorm(x) * norm_w[l] )
 * with RMSNorm(x) = x / sqrt(mean(x^2) + eps).  Routing (Sec. 3.2) is decided
 * once per token from its id and holds in every block: a base-path token uses
 * the dense MLP (Eq. 1), a sparse-path token the CATS mask with threshold t[l]
 * (Eq. 5).  token_ids == NULL sends every token to the sparse path.
 *   layers    : host array of L layer handles (all with the same H, N)
 *   norm_w    : host array of L device fp32 [H] RMSNorm gains
 *   t         : host fp32 [L], per-layer thresholds (>= 0, not NaN)
 *   token_ids : device int32 [B] or NULL;  lut : device uint8 [V] (V >= 1 when ids given)
 *   x         : device fp32 [B][H], read and overwritten in place.
 *   keep_trace: device uint8 [L][B][N] or NULL; receives each block's keep mask
 *               per token (1 = neuron used), for verification.
 * A token id outside [0, V) is routed to the base path and sets the
 * workspace status word (SATS_EDEVICE from sats_get_error).
 */
SATS_API sats_status sats_mlp_stack(const sats_layer *const *layers, const float *const *norm_w,
                           const float *t, int L, float eps,
                           const int32_t *token_ids, const uint8_t *lut, int V,
                           float *x, int B, uint8_t *keep_trace,
                           void *ws, size_t ws_bytes, void *stream);

/*
 * sats_gate_act -- calibration helper: a = SiLU(x W_gate) (Sec. 2, Eqs. 1-2)
 * for B tokens, the post-gate activations from which thresholds are chosen
 * (Eq. 3 for CATS; candidate set T_l for SATS, Sec. 3.1).
 *   x : device bf16 [B][H];  a : device fp32 [B][N], written.
 */
SATS_API sats_status sats_gate_act(const sats_layer *layer, const void *x, int B, float *a,
                          void *ws, size_t ws_bytes, void *stream);

/*
 * sats_percentile_threshold -- Eq. 3: t = min{t' : F(t') >= k}, F the empirical
 * CDF of |a_i| over n values, i.e. the m-th smallest |a_i| with m = ceil(k n)
 * (k read as a decimal fraction; k*n is taken down by a relative 2^-50 before
 * the ceiling).  k <= 0 gives 0, k > 1 gives +inf.
 *   a      : device fp32 [n] (NaN not allowed)
 *   t_out  : host fp32 [1], written.
 *   ws     : device workspace of at least sats_select_workspace_bytes() bytes.
 * Synchronises `stream` (the result is returned on the host).
 */
SATS_API size_t sats_select_workspace_bytes(void);
SATS_API sats_status sats_percentile_threshold(const float *a, int64_t n, double k, float *t_out,
                                      void *ws, size_t ws_bytes, void *stream);

/*
 * SATS calibration (Sec. 3.1): choose each block's threshold by its local
 * distortion instead of a percentile.
 *
 * sats_rmsnorm -- out[b] = x[b] / sqrt(mean_i x[b][i]^2 + eps) * w, the
 *   pre-MLP normalisation of a decoder block.  x, out: device fp32 [B][H];
 *   w: device fp32 [H].
 *
 * sats_gate_act_f32 -- sats_gate_act for fp32 activations x [B][H].
 *
 * sats_layer_err -- Eq. 6 for K candidate thresholds t (host fp32 [K], each
 *   >= 0) on C calibration inputs x (device fp32 [C][H], the block's MLP
 *   inputs):
 *     err[k] = (1/C) sum_c ||y(x_c) - y~_{t_k}(x_c)||_2 / (||y(x_c)||_2 + eps)
 *     sp[k]  = (1/C) sum_c (neurons with |a| < t_k) / N
 *   y is the dense output (Eq. 1), y~_t the thresholded one (Eqs. 4-5), both
 *   computed by the library's MLP kernels.  err, sp: host double [K].  ws:
 *   device workspace of sats_layer_err_workspace_bytes(H, N, C, K) bytes,
 *   256-byte aligned (no initialisation needed).  Synchronises `stream`.
 *
 * sats_sats_select -- Eqs. 7-10 on the host over a candidate table t, err,
 *   sp (host double [L][K]; every block also has the candidate t = 0 with
 *   error 0 and sparsity 0):
 *     t*_l(b) = max{t in T_l : Err_l(t) <= b}             (Eq. 7)
 *     S(b) = (1/L) sum_l sp_l(t*_l(b))                     (Eqs. 8-9)
 *     b* = argmin_b |S(b) - s_tar|                         (Eq. 10)
 *   over b in {0} and every error in the table, ties to the smaller b.  Block
 *   `guard` (-1 for none) keeps guard_t (sparsity guard_sp) and takes no part
 *   in Eq. 7.  Writes b*, t_out[L] = T*(b*) and S(b*).
 *
 * sats_sats_calibrate -- the whole calibration of an L-block stack, in the
 *   paper's order: (1) the dense stack on the calibration inputs x_cal
 *   (device fp32 [C][H]) gives each block's MLP inputs RMSNorm(x_l) w_l;
 *   (2) coarse candidates: Eq. 3 percentiles of |SiLU(n_l W_gate)| at k/K0,
 *   k = 1..K0-1; (3) Eq. 6 for each; (4) Eqs. 7-10; (5) K1 fine candidates
 *   evenly spaced strictly between the coarse candidates that neighbour each
 *   block's choice (0 below the first, the largest |a| above the last); (6)
 *   Eqs. 6-10 over coarse and fine candidates together.  With guardrail != 0
 *   the last block keeps the CATS threshold (the Eq. 3 percentile at s_tar),
 *   as Sec. 4 does.  Writes t_out (host fp32 [L]), b* and S(b*), and, if all
 *   three are given, the candidate table (host double [L][K0 - 1 + K1]).
 *   ws: sats_sats_workspace_bytes(H, N, C, L, K0, K1) bytes, 256-byte aligned.
 *   Synchronises `stream`.
 */
SATS_API sats_status sats_rmsnorm(const float *x, int B, int H, const float *w, float eps, float *out,
                                  void *stream);
SATS_API sats_status sats_gate_act_f32(const sats_layer *layer, const float *x, int B, float *a, void *stream);
SATS_API size_t sats_layer_err_workspace_bytes(int H, int N, int C, int K);
SATS_API sats_status sats_layer_err(const sats_layer *layer, const float *x, int C, const float *t, int K,
                                    float eps, double *err, double *sp, void *ws, size_t ws_bytes, void *stream);
SATS_API sats_status sats_sats_select(const double *t, const double *err, const double *sp, int L, int K,
                                      double s_tar, int guard, double guard_t, double guard_sp, double *b_out,
                                      double *t_out, double *S_out);
SATS_API size_t sats_sats_workspace_bytes(int H, int N, int C, int L, int K0, int K1);
SATS_API sats_status sats_sats_calibrate(const sats_layer *const *layers, const float *const *norm_w, int L,
                                         float eps, const float *x_cal, int C, double s_tar, int K0, int K1,
                                         int guardrail, float err_eps, float *t_out, double *b_out, double *S_out,
                                         double *table_t, double *table_err, double *table_sp, void *ws,
                                         size_t ws_bytes, void *stream);

/*
 * Routing calibration (Sec. 3.2).
 *
 * sats_token_scores -- Eqs. 11-12: for n corpus occurrences (ids: device
 *   int32 [n]; l_base, l_sparse: device fp32 [n], the next-token losses of
 *   the base and sparse paths), d_i = max(0, l_sparse_i - l_base_i) and
 *   score[v] = mean of d_i over the occurrences of v (device fp32 [V]); a
 *   token that never occurs gets +inf (it keeps the base path).  An id
 *   outside [0, V) returns SATS_EDEVICE.  ws: sats_route_calib_workspace_bytes(V)
 *   bytes, 256-byte aligned.  Synchronises `stream`.
 *
 * sats_route_calibrate -- Eq. 14: tau* = argmin_tau |R(tau) - r_tar|, where
 *   R(tau) is the fraction of the m held-out occurrences (heldout_ids: device
 *   int32 [m]) whose score is < tau (routed to the sparse path, Eq. 13); the
 *   candidates are 0, every score of a token occurring in the held-out split,
 *   and +inf, and a tie goes to the smaller tau.  Writes tau* and R(tau*)
 *   (host), and, if lut is given, the routing table lut[v] = score[v] >= tau*
 *   (device uint8 [V]; 1 = base path), as sats_route and sats_mlp_stack take
 *   it.  Synchronises `stream`.
 */
SATS_API size_t sats_route_calib_workspace_bytes(int V);
SATS_API sats_status sats_token_scores(const int32_t *ids, const float *l_base, const float *l_sparse, int64_t n,
                                       int V, float *score, void *ws, size_t ws_bytes, void *stream);
SATS_API sats_status sats_route_calibrate(const float *score, int V, const int32_t *heldout_ids, int64_t m,
                                          double r_tar, float *tau_out, double *R_out, uint8_t *lut, void *ws,
                                          size_t ws_bytes, void *stream);

/*
 * sats_selftest_wait_timeout -- exercises the failure path of the device-side
 * waits without a fault: one small kernel runs the library's bounded waits on
 * conditions nothing satisfies (an mbarrier phase no thread completes, a
 * workspace counter no CTA raises).  Each gives up after its time limit (2 s)
 * and records a timeout in the workspace status word, so a following
 * sats_get_error returns SATS_ETIMEOUT (and clears it).  Takes about 4 s;
 * the workspace and the device stay usable.  ws: a workspace of any layer
 * shape (at least 256 bytes), not in use by another call.
 */
SATS_API sats_status sats_selftest_wait_timeout(void *ws, size_t ws_bytes, void *stream);

/*
 * sats_get_error -- synchronises `stream`, reads the status word in the
 * workspace, clears it, and returns SATS_OK, SATS_EDEVICE (bad token id) or
 * SATS_ETIMEOUT (a device wait gave up).
 */
SATS_API sats_status sats_get_error(void *ws, size_t ws_bytes, void *stream);

/* Same for a caller-owned status word (as passed to sats_route). */
SATS_API sats_status sats_get_status_word(int32_t *dev_status, void *stream);

#ifdef __cplusplus
}
#endif

#endif /* SATS_H */
