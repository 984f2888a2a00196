// api.cu -- the C ABI declared in include/sats.h: argument checks, the
// workspace layout, and the host-side drivers that split a batch into passes
// of the fused kernel and chain the blocks of a stack.
#include <cmath>
#include <cstdio>
#include <cstring>
#include <new>

#include "common.cuh"
#include "internal.h"

namespace sats {

static size_t align256(size_t v) { return (v + 255) & ~(size_t)255; }

static int nchunks_of(int N) { return (N + kChunk - 1) / kChunk; }

WsLayout ws_layout(int H, int N, int B)
{
    WsLayout L{};
    size_t off = 0;
    L.ctl = off;
    off += align256(kCtlInts * sizeof(int));
    L.lora_z = off;   // cleared with the control words; the fused kernel's last CTA clears it after a LoRA call
    off += align256((size_t)kLoraZCopies * kMaxTokensPerPass * 2 * kMaxLoraRank * sizeof(float));
    L.flags = off;   // one 64-bit word per chunk of kChunk neurons (the fused kernel's index-list words)
    off += align256((size_t)nchunks_of(N) * sizeof(uint64_t));
    L.route_perm = off;
    off += align256((size_t)(B > 0 ? B : 1) * sizeof(int32_t));
    L.route_flags = off;
    off += align256((size_t)(B > 0 ? B : 1));
    L.tc = off;   // bf16 activations, h and keep bytes of the tensor-core path (batches only)
    if (use_tc_path(H, B)) off += tc_workspace_bytes(H, N, B);
    L.total = off;
    return L;
}

static bool aligned16(const void *p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

cudaError_t clear_fused_state(void *ws, int H, int N, int B, cudaStream_t stream)
{
    // the fused kernel clears the chunk flags itself; its counters (and the LoRA sums) must start at zero
    return cudaMemsetAsync(ws, 0, ws_layout(H, N, B).flags, stream);
}

static thread_local cudaError_t g_last_cuda = cudaSuccess;
static thread_local const char *g_last_where = nullptr;
static thread_local char g_last_text[256];

sats_status cuda_fail(cudaError_t e, const char *where)
{
    g_last_cuda = e;
    g_last_where = where;
    return SATS_ECUDA;
}

static sats_status from_cuda(cudaError_t e, const char *where = "CUDA call")
{
    return e == cudaSuccess ? SATS_OK : cuda_fail(e, where);
}

static bool bad_threshold(float t) { return std::isnan(t) || t < 0.0f; }

// Runs one block over B tokens: on the tensor cores when the batch is larger
// than one pass of the fused kernel, else in passes of fused_tokens_per_pass(H)
// tokens of the fused kernel (of the small-layer kernel for small layers).
sats_status run_layer(const sats_layer *layer, int x_mode, const void *x, int B, const float *t_per_pass_l,
                      const float *norm_w, float eps, const uint8_t *dense_flags, int out_mode, float *out,
                      int32_t *active_idx, int32_t *active_cnt, uint8_t *keep_trace, void *ws, cudaStream_t stream,
                      const sats_lora *lora, const int32_t *perm, const int32_t *n_dense)
{
    const int H = layer->H, N = layer->N;
    const WsLayout L = ws_layout(H, N, B);
    char *base = static_cast<char *>(ws);
    if (!lora && use_tc_path(H, B)) {   // the LoRA variant runs in passes of the fused kernel at any batch
        const cudaError_t e = run_tc_layer(layer, x_mode, x, B, *t_per_pass_l, norm_w, eps, perm ? nullptr : dense_flags,
                                           perm, n_dense, out_mode,
                                           out, active_idx, active_cnt, keep_trace, base + L.tc,
                                           reinterpret_cast<int *>(base + L.ctl), stream);
        return e == cudaSuccess ? SATS_OK : SATS_ECUDA;   // run_tc_layer recorded the failing step
    }
    const int per_pass = fused_tokens_per_pass(H);
    const size_t x_elem = (x_mode == kXBf16) ? 2 : 4;
    for (int b0 = 0; b0 < B; b0 += per_pass) {
        FusedParams p{};
        p.wg_t = layer->wg_t;
        p.w_ud = layer->w_ud;
        p.H = H;
        p.N = N;
        p.nchunks = nchunks_of(N);
        p.nb = B - b0 < per_pass ? B - b0 : per_pass;
        p.x_mode = x_mode;
        p.x = static_cast<const char *>(x) + (size_t)b0 * H * x_elem;
        p.norm_w = norm_w;
        p.eps = eps;
        p.t_l = *t_per_pass_l;
        p.dense_flags = dense_flags ? dense_flags + b0 : nullptr;
        p.out_mode = out_mode;
        p.out = out + (size_t)b0 * H;
        p.ctl = reinterpret_cast<int *>(base + L.ctl);
        p.flags = reinterpret_cast<uint64_t *>(base + L.flags);
        p.active_idx = active_idx ? active_idx + (size_t)b0 * N : nullptr;
        p.active_cnt = active_cnt ? active_cnt + b0 : nullptr;
        p.keep_trace = keep_trace ? keep_trace + (size_t)b0 * N : nullptr;
        if (lora) {
            p.lora = lora;
            p.lora_blk = lora->blk;
            p.lora_agu = lora->agu;
            p.lora_bd = lora->bd;
            p.lora_r = lora->r;
            p.lora_scale = lora->scale;
            p.lora_z = reinterpret_cast<float *>(base + L.lora_z);
        }
        if (!lora && use_small_path(H, N, p.nb)) {
            const cudaError_t e = launch_small(p, stream);
            if (e != cudaSuccess) return cuda_fail(e, "small-layer kernel launch");
            continue;
        }
        const cudaError_t e = launch_fused(p, stream);
        if (e != cudaSuccess) return cuda_fail(e, "fused kernel launch");
    }
    return SATS_OK;
}

static sats_status check_layer(const sats_layer *layer, void *ws, size_t ws_bytes, int B)
{
    if (!layer || !ws) return SATS_EINVAL;
    if (B < 0) return SATS_EINVAL;
    if (!aligned16(ws)) return SATS_EINVAL;
    if (ws_bytes < ws_layout(layer->H, layer->N, B).total) return SATS_ENOSPACE;
    return SATS_OK;
}

static sats_status sparse_common(const sats_layer *layer, int x_mode, const void *x, int B, float t_l, float *y,
                                 int32_t *active_idx, int32_t *active_cnt, void *ws, size_t ws_bytes, void *stream)
{
    sats_status s = check_layer(layer, ws, ws_bytes, B);
    if (s != SATS_OK) return s;
    if (bad_threshold(t_l)) return SATS_EINVAL;
    if ((active_idx == nullptr) != (active_cnt == nullptr)) return SATS_EINVAL;
    if (B == 0) return SATS_OK;
    if (!x || !y || !aligned16(x) || !aligned16(y)) return SATS_EINVAL;
    return run_layer(layer, x_mode, x, B, &t_l, nullptr, 0.f, nullptr, kOutY, y, active_idx, active_cnt, nullptr,
                     ws, static_cast<cudaStream_t>(stream));
}

// ---------------------------------------------------------------------------
// Fixed scratch for sats_sparse_mlp_fixed_scratch: one array in this file's
// device memory, present on every GPU that loads the library until the
// process exits.  Host code cannot use the symbol itself as a device address;
// the address is looked up with cudaGetSymbolAddress on every call (it
// allocates nothing and does not synchronise), so it always belongs to the
// current device and context, also after a cudaDeviceReset reloaded the module.
constexpr size_t kFixedScratchBytes = (size_t)1 << 18;   // 256 KiB
static __device__ __align__(256) unsigned char g_fixed_scratch[kFixedScratchBytes];

// Device address of g_fixed_scratch on the current device, or nullptr (with the
// CUDA error in *err) on failure.
static void *fixed_scratch_current_device(cudaError_t *err)
{
    void *ptr = nullptr;
    *err = cudaGetSymbolAddress(&ptr, g_fixed_scratch);
    if (*err == cudaSuccess && !ptr) *err = cudaErrorInvalidSymbol;
    return *err == cudaSuccess ? ptr : nullptr;
}

}  // namespace sats

using namespace sats;

extern "C" {

int sats_version(void) { return (1 << 16) | 0; }

const char *sats_status_string(sats_status s)
{
    switch (s) {
    case SATS_OK: return "ok";
    case SATS_EINVAL: return "invalid argument";
    case SATS_ESHAPE: return "unsupported shape";
    case SATS_ECUDA: return "CUDA runtime error";
    case SATS_EDEVICE: return "bad input detected on the device (token id outside the vocabulary)";
    case SATS_ETIMEOUT: return "a bounded device-side wait gave up";
    case SATS_ENOSPACE: return "workspace too small";
    }
    return "unknown status";
}

sats_status sats_layer_create(const void *W_gate, const void *W_up, const void *W_down, int H, int N, void *stream,
                              sats_layer **out)
{
    if (!out) return SATS_EINVAL;
    *out = nullptr;
    if (!W_gate || !W_up || !W_down) return SATS_EINVAL;
    if (H < 8 || H > kMaxH || (H % 8) != 0 || N < 1 || N > kMaxN) return SATS_ESHAPE;
    sats_layer *l = new (std::nothrow) sats_layer();
    if (!l) return cuda_fail(cudaErrorMemoryAllocation, "host allocation");
    l->H = H;
    l->N = N;
    cudaGetDevice(&l->device);
    const size_t row_elems = (size_t)N * H;
    cudaError_t e = cudaMalloc(&l->wg_t, row_elems * 2);
    if (e == cudaSuccess) e = cudaMalloc(&l->w_ud, row_elems * 4);
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    if (e == cudaSuccess)
        e = launch_pack(static_cast<const uint16_t *>(W_gate), static_cast<const uint16_t *>(W_up),
                        static_cast<const uint16_t *>(W_down), H, N, l->wg_t, l->w_ud, s);
    if (e == cudaSuccess) e = tc_pack_layer(l, s);
    if (e == cudaSuccess) e = cudaStreamSynchronize(s);
    if (e != cudaSuccess) {
        cudaFree(l->wg_t);
        cudaFree(l->w_ud);
        tc_free_layer(l);
        delete l;
        return cuda_fail(e, "layer allocation or repacking");
    }
    *out = l;
    return SATS_OK;
}

sats_status sats_layer_destroy(sats_layer *layer)
{
    if (!layer) return SATS_EINVAL;
    cudaDeviceSynchronize();
    const cudaError_t e1 = cudaFree(layer->wg_t);
    const cudaError_t e2 = cudaFree(layer->w_ud);
    const cudaError_t e3 = tc_free_layer(layer);
    delete layer;
    if (e1 != cudaSuccess) return cuda_fail(e1, "cudaFree");
    if (e2 != cudaSuccess) return cuda_fail(e2, "cudaFree");
    return from_cuda(e3, "cudaFree");
}

sats_status sats_lora_create(const sats_layer *layer, const void *A_gate, const void *B_gate, const void *A_up,
                             const void *B_up, const void *A_down, const void *B_down, int r, float scale,
                             void *stream, sats_lora **out)
{
    if (!out) return SATS_EINVAL;
    *out = nullptr;
    if (!layer || !A_gate || !B_gate || !A_up || !B_up || !A_down || !B_down || !std::isfinite(scale))
        return SATS_EINVAL;
    if (r < 8 || r > kMaxLoraRank || (r % 8) != 0) return SATS_ESHAPE;
    sats_lora *l = new (std::nothrow) sats_lora();
    if (!l) return cuda_fail(cudaErrorMemoryAllocation, "host allocation");
    l->H = layer->H;
    l->N = layer->N;
    l->r = r;
    l->scale = scale;
    cudaGetDevice(&l->device);
    const size_t nblk = (size_t)nchunks_of(l->N) * kChunk * 3 * r;
    cudaError_t e = cudaMalloc(&l->blk, nblk * 2);
    if (e == cudaSuccess) e = cudaMalloc(&l->agu, (size_t)l->H * 2 * r * 2);
    if (e == cudaSuccess) e = cudaMalloc(&l->bd, (size_t)r * l->H * 2);
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    if (e == cudaSuccess)
        e = launch_pack_lora(static_cast<const uint16_t *>(A_gate), static_cast<const uint16_t *>(B_gate),
                             static_cast<const uint16_t *>(A_up), static_cast<const uint16_t *>(B_up),
                             static_cast<const uint16_t *>(A_down), static_cast<const uint16_t *>(B_down), l->H, l->N,
                             r, l, st);
    if (e == cudaSuccess) e = cudaStreamSynchronize(st);
    if (e != cudaSuccess) {
        cudaFree(l->blk);
        cudaFree(l->agu);
        cudaFree(l->bd);
        delete l;
        return cuda_fail(e, "adapter allocation or repacking");
    }
    *out = l;
    return SATS_OK;
}

sats_status sats_lora_destroy(sats_lora *lora)
{
    if (!lora) return SATS_EINVAL;
    cudaDeviceSynchronize();
    const cudaError_t e1 = cudaFree(lora->blk);
    const cudaError_t e2 = cudaFree(lora->agu);
    const cudaError_t e3 = cudaFree(lora->bd);
    delete lora;
    if (e1 != cudaSuccess) return cuda_fail(e1, "cudaFree");
    if (e2 != cudaSuccess) return cuda_fail(e2, "cudaFree");
    return from_cuda(e3, "cudaFree");
}

static sats_status lora_common(const sats_layer *layer, const sats_lora *lora, int x_mode, const void *x, int B,
                               float t_l, float *y, int32_t *active_idx, int32_t *active_cnt, void *ws,
                               size_t ws_bytes, void *stream)
{
    sats_status s = check_layer(layer, ws, ws_bytes, B);
    if (s != SATS_OK) return s;
    if (!lora) return SATS_EINVAL;
    if (lora->H != layer->H || lora->N != layer->N) return SATS_ESHAPE;
    if (bad_threshold(t_l)) return SATS_EINVAL;
    if ((active_idx == nullptr) != (active_cnt == nullptr)) return SATS_EINVAL;
    if (B == 0) return SATS_OK;
    if (!x || !y || !aligned16(x) || !aligned16(y)) return SATS_EINVAL;
    return run_layer(layer, x_mode, x, B, &t_l, nullptr, 0.f, nullptr, kOutY, y, active_idx, active_cnt, nullptr, ws,
                     static_cast<cudaStream_t>(stream), lora);
}

sats_status sats_sparse_mlp_lora(const sats_layer *layer, const sats_lora *lora, const void *x, int B, float t_l,
                                 float *y, int32_t *active_idx, int32_t *active_cnt, void *ws, size_t ws_bytes,
                                 void *stream)
{
    return lora_common(layer, lora, kXBf16, x, B, t_l, y, active_idx, active_cnt, ws, ws_bytes, stream);
}

sats_status sats_sparse_mlp_lora_f32(const sats_layer *layer, const sats_lora *lora, const float *x, int B,
                                     float t_l, float *y, int32_t *active_idx, int32_t *active_cnt, void *ws,
                                     size_t ws_bytes, void *stream)
{
    return lora_common(layer, lora, kXF32, x, B, t_l, y, active_idx, active_cnt, ws, ws_bytes, stream);
}

sats_status sats_layer_shape(const sats_layer *layer, int *H, int *N)
{
    if (!layer) return SATS_EINVAL;
    if (H) *H = layer->H;
    if (N) *N = layer->N;
    return SATS_OK;
}

size_t sats_workspace_bytes(int H, int N, int B)
{
    if (H < 8 || H > kMaxH || (H % 8) != 0 || N < 1 || N > kMaxN || B < 0) return 0;
    return ws_layout(H, N, B).total;
}

sats_status sats_workspace_init(void *ws, size_t ws_bytes, void *stream)
{
    if (!ws) return SATS_EINVAL;
    return from_cuda(cudaMemsetAsync(ws, 0, ws_bytes, static_cast<cudaStream_t>(stream)));
}

sats_status sats_sparse_mlp(const sats_layer *layer, const void *x, int B, float t_l, float *y, int32_t *active_idx,
                            int32_t *active_cnt, void *ws, size_t ws_bytes, void *stream)
{
    return sparse_common(layer, kXBf16, x, B, t_l, y, active_idx, active_cnt, ws, ws_bytes, stream);
}

sats_status sats_sparse_mlp_fixed_scratch(const sats_layer *layer, const void *x, int B, float t_l, float *y,
                                          int32_t *active_idx, int32_t *active_cnt, int32_t *dev_status,
                                          void *stream)
{
    if (!layer || B < 0) return SATS_EINVAL;
    if (ws_layout(layer->H, layer->N, B).total > kFixedScratchBytes) return SATS_ENOSPACE;
    if (bad_threshold(t_l)) return SATS_EINVAL;
    if ((active_idx == nullptr) != (active_cnt == nullptr)) return SATS_EINVAL;
    if (dev_status && (reinterpret_cast<uintptr_t>(dev_status) & 3u)) return SATS_EINVAL;
    if (B == 0) return SATS_OK;
    if (!x || !y || !aligned16(x) || !aligned16(y)) return SATS_EINVAL;
    cudaError_t el = cudaSuccess;
    void *ws = fixed_scratch_current_device(&el);
    if (!ws) return cuda_fail(el, "fixed scratch lookup");
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    // the array keeps the previous call's contents: the control words
    // (scheduling counters, status) must start at zero
    const cudaError_t ez = clear_fused_state(ws, layer->H, layer->N, B, st);
    if (ez != cudaSuccess) return cuda_fail(ez, "fixed scratch clear");
    const sats_status s = sparse_common(layer, kXBf16, x, B, t_l, y, active_idx, active_cnt, ws,
                                        kFixedScratchBytes, stream);
    if (s != SATS_OK || !dev_status) return s;
    // this call's device status word (cleared above, so it holds this call's errors only)
    const int32_t *word = static_cast<const int32_t *>(ws) + kCtlStatus;   // the control block starts the scratch
    return from_cuda(cudaMemcpyAsync(dev_status, word, sizeof(int32_t), cudaMemcpyDeviceToDevice, st),
                     "fixed scratch status copy");
}

int sats_uses_tensor_cores(int H, int B) { return use_tc_path(H, B) ? 1 : 0; }

const char *sats_last_cuda_error(void)
{
    if (g_last_cuda == cudaSuccess) return "no CUDA error recorded";
    snprintf(g_last_text, sizeof g_last_text, "%s: %s (%s)", g_last_where ? g_last_where : "CUDA call",
             cudaGetErrorString(g_last_cuda), cudaGetErrorName(g_last_cuda));
    return g_last_text;
}

sats_status sats_sparse_mlp_f32(const sats_layer *layer, const float *x, int B, float t_l, float *y,
                                int32_t *active_idx, int32_t *active_cnt, void *ws, size_t ws_bytes, void *stream)
{
    return sparse_common(layer, kXF32, x, B, t_l, y, active_idx, active_cnt, ws, ws_bytes, stream);
}

static sats_status union_common(const sats_layer *layer, int x_mode, const void *x, int B, float t_l, float *y,
                                int32_t *active_idx, int32_t *active_cnt, void *ws, size_t ws_bytes, void *stream)
{
    sats_status s = check_layer(layer, ws, ws_bytes, B);
    if (s != SATS_OK) return s;
    if (bad_threshold(t_l)) return SATS_EINVAL;
    if ((active_idx == nullptr) != (active_cnt == nullptr)) return SATS_EINVAL;
    if (B < 3 || !union_path_ok(layer->H, B)) return SATS_ESHAPE;
    if (!x || !y || !aligned16(x) || !aligned16(y)) return SATS_EINVAL;
    const WsLayout L = ws_layout(layer->H, layer->N, B);
    char *base = static_cast<char *>(ws);
    const cudaError_t e = run_tc_layer(layer, x_mode, x, B, t_l, nullptr, 0.f, nullptr, nullptr, nullptr, kOutY, y, active_idx,
                                       active_cnt, nullptr, base + L.tc, reinterpret_cast<int *>(base + L.ctl),
                                       static_cast<cudaStream_t>(stream), true);
    return e == cudaSuccess ? SATS_OK : SATS_ECUDA;   // run_tc_layer recorded the failing step
}

sats_status sats_sparse_mlp_union(const sats_layer *layer, const void *x, int B, float t_l, float *y,
                                  int32_t *active_idx, int32_t *active_cnt, void *ws, size_t ws_bytes, void *stream)
{
    return union_common(layer, kXBf16, x, B, t_l, y, active_idx, active_cnt, ws, ws_bytes, stream);
}

sats_status sats_sparse_mlp_union_f32(const sats_layer *layer, const float *x, int B, float t_l, float *y,
                                      int32_t *active_idx, int32_t *active_cnt, void *ws, size_t ws_bytes,
                                      void *stream)
{
    return union_common(layer, kXF32, x, B, t_l, y, active_idx, active_cnt, ws, ws_bytes, stream);
}

sats_status sats_dense_mlp(const sats_layer *layer, const void *x, int B, float *y, void *ws, size_t ws_bytes,
                           void *stream)
{
    return sparse_common(layer, kXBf16, x, B, 0.0f, y, nullptr, nullptr, ws, ws_bytes, stream);
}

sats_status sats_route(const int32_t *token_ids, int B, const uint8_t *lut, int V, int32_t *perm, int32_t *n_dense,
                       int32_t *dev_status, void *stream)
{
    if (B < 0 || V < 1 || !lut || !n_dense) return SATS_EINVAL;
    if (B > 0 && (!token_ids || !perm)) return SATS_EINVAL;
    return from_cuda(launch_route(token_ids, B, lut, V, perm, n_dense, nullptr, dev_status,
                                  static_cast<cudaStream_t>(stream)));
}

sats_status sats_mlp_stack(const sats_layer *const *layers, const float *const *norm_w, const float *t, int L,
                           float eps, const int32_t *token_ids, const uint8_t *lut, int V, float *x, int B,
                           uint8_t *keep_trace, void *ws, size_t ws_bytes, void *stream)
{
    if (!layers || !norm_w || !t || L < 0 || B < 0 || !ws) return SATS_EINVAL;
    if (std::isnan(eps) || eps < 0.0f) return SATS_EINVAL;
    if (L == 0 || B == 0) return SATS_OK;
    if (!x || !aligned16(x)) return SATS_EINVAL;
    if (token_ids && (!lut || V < 1)) return SATS_EINVAL;
    const int H = layers[0] ? layers[0]->H : 0, N = layers[0] ? layers[0]->N : 0;
    for (int l = 0; l < L; ++l) {
        if (!layers[l] || layers[l]->H != H || layers[l]->N != N) return SATS_EINVAL;
        if (!norm_w[l] || !aligned16(norm_w[l])) return SATS_EINVAL;
        if (bad_threshold(t[l])) return SATS_EINVAL;
    }
    sats_status s = check_layer(layers[0], ws, ws_bytes, B);
    if (s != SATS_OK) return s;
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    const WsLayout W = ws_layout(H, N, B);
    char *base = static_cast<char *>(ws);
    int *ctl = reinterpret_cast<int *>(base + W.ctl);
    // Routing once for every block (Eq. 13 through the table): the per-token flags serve the
    // fused passes (B <= 2), the permutation (base-path tokens first) and its count the
    // tensor-core path, which gathers the tokens in that order and scatters the results back.
    uint8_t *flags = nullptr;
    int32_t *perm = nullptr;
    const int32_t *n_dense = nullptr;
    if (token_ids) {
        flags = reinterpret_cast<uint8_t *>(base + W.route_flags);
        perm = reinterpret_cast<int32_t *>(base + W.route_perm);
        n_dense = ctl + kCtlNDense;
        cudaError_t e = launch_route(token_ids, B, lut, V, perm, ctl + kCtlNDense, flags, ctl + kCtlStatus, st);
        if (e != cudaSuccess) return cuda_fail(e, "route kernel launch");
    }
    for (int l = 0; l < L; ++l) {
        s = run_layer(layers[l], kXResidNorm, x, B, &t[l], norm_w[l], eps, flags, kOutResid, x, nullptr, nullptr,
                      keep_trace ? keep_trace + (size_t)l * B * N : nullptr, ws, st, nullptr, perm, n_dense);
        if (s != SATS_OK) return s;
    }
    return SATS_OK;
}

sats_status sats_gate_act(const sats_layer *layer, const void *x, int B, float *a, void *ws, size_t ws_bytes,
                          void *stream)
{
    (void)ws;
    (void)ws_bytes;
    if (!layer || B < 0) return SATS_EINVAL;
    if (B == 0) return SATS_OK;
    if (!x || !a || !aligned16(x)) return SATS_EINVAL;
    return from_cuda(launch_gate_act(layer, static_cast<const uint16_t *>(x), B, a, static_cast<cudaStream_t>(stream)));
}

size_t sats_select_workspace_bytes(void) { return select_ws_bytes(); }

sats_status sats_percentile_threshold(const float *a, int64_t n, double k, float *t_out, void *ws, size_t ws_bytes,
                                      void *stream)
{
    if (!t_out || n < 0 || std::isnan(k)) return SATS_EINVAL;
    if (n == 0 || !(k > 0.0)) { *t_out = 0.0f; return SATS_OK; }
    if (k > 1.0) { *t_out = INFINITY; return SATS_OK; }
    if (!a || !ws || ws_bytes < select_ws_bytes() || !aligned16(ws)) return SATS_EINVAL;
    // m = ceil(k n), with k read as the decimal fraction it stands for
    int64_t m = (int64_t)std::ceil((k * (double)n) * (1.0 - std::ldexp(1.0, -50)));
    if (m < 1) m = 1;
    if (m > n) m = n;
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    float *t_dev = reinterpret_cast<float *>(static_cast<char *>(ws) + select_ws_bytes() - 128);
    cudaError_t e = launch_select(a, n, m, ws, t_dev, st);
    if (e == cudaSuccess) e = cudaMemcpyAsync(t_out, t_dev, sizeof(float), cudaMemcpyDeviceToHost, st);
    if (e == cudaSuccess) e = cudaStreamSynchronize(st);
    return from_cuda(e);
}

static sats_status read_status(int32_t *word, cudaStream_t st)
{
    int32_t v = 0;
    cudaError_t e = cudaStreamSynchronize(st);
    if (e == cudaSuccess) e = cudaMemcpy(&v, word, sizeof v, cudaMemcpyDeviceToHost);
    if (e == cudaSuccess && v != 0) e = cudaMemset(word, 0, sizeof v);
    if (e != cudaSuccess) return cuda_fail(e, "status read");
    if (v & kStatusTimeout) return SATS_ETIMEOUT;
    if (v & (kStatusBadToken | kStatusInternal)) return SATS_EDEVICE;
    return SATS_OK;
}

sats_status sats_selftest_wait_timeout(void *ws, size_t ws_bytes, void *stream)
{
    if (!ws || ws_bytes < (size_t)kCtlInts * sizeof(int)) return SATS_EINVAL;
    return from_cuda(launch_wait_timeout(static_cast<int *>(ws), static_cast<cudaStream_t>(stream)));
}

sats_status sats_get_error(void *ws, size_t ws_bytes, void *stream)
{
    if (!ws || ws_bytes < (size_t)kCtlInts * sizeof(int)) return SATS_EINVAL;
    return read_status(static_cast<int32_t *>(ws) + kCtlStatus, static_cast<cudaStream_t>(stream));
}

sats_status sats_get_status_word(int32_t *dev_status, void *stream)
{
    if (!dev_status) return SATS_EINVAL;
    return read_status(dev_status, static_cast<cudaStream_t>(stream));
}

}  // extern "C"
