// calib.cu -- SATS threshold calibration (Sec. 3.1, Eqs. 6-10; Sec. 4 guardrail)
// on the GPU, with the same kernels that run the thresholded MLP.
//
// Eq. 6, Err_l(t) = E_x[ ||y(x) - y~_t(x)|| / (||y(x)|| + eps) ], is evaluated for
// many candidate thresholds at once per block: the dense output once, then one
// thresholded pass per candidate (the fused kernel or the tensor-core path,
// whichever the batch of calibration inputs takes), each followed by a small
// reduction kernel that adds the per-token relative distortion and realised
// sparsity into device accumulators.  Eqs. 7-10 (budget selection) run on the
// host; the coarse-to-fine driver chains everything for a whole stack.
#include <algorithm>
#include <cmath>
#include <vector>

#include "common.cuh"
#include "internal.h"

namespace sats {
namespace {

size_t al256(size_t v) { return (v + 255) & ~(size_t)255; }

// out[b] = x[b] / sqrt(mean_i x[b][i]^2 + eps) * w  (one CTA per row).
__global__ void __launch_bounds__(256) rmsnorm_kernel(const float *__restrict__ x, int H, const float *__restrict__ w,
                                                      float eps, float *__restrict__ out)
{
    const float *xr = x + (size_t)blockIdx.x * H;
    float *o = out + (size_t)blockIdx.x * H;
    __shared__ float red[8];
    float s = 0.f;
    for (int i = threadIdx.x; i < H; i += 256) s = fmaf(xr[i], xr[i], s);
    s = warp_sum(s);
    if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = s;
    __syncthreads();
    float tot = 0.f;
    for (int i = 0; i < 8; ++i) tot += red[i];
    const float inv = 1.0f / sqrtf(tot / (float)H + eps);
    for (int i = threadIdx.x; i < H; i += 256) o[i] = xr[i] * inv * w[i];
}

// Token c: acc[0] += ||yd_c - yk_c|| / (||yd_c|| + eps), acc[1] += (N - kept_c) / N.
__global__ void __launch_bounds__(256) err_accum_kernel(const float *__restrict__ yd, const float *__restrict__ yk,
                                                        int H, const int32_t *__restrict__ cnt, int N, float eps,
                                                        double *__restrict__ acc)
{
    const int c = blockIdx.x;
    const float *a = yd + (size_t)c * H, *b = yk + (size_t)c * H;
    double dd = 0.0, yy = 0.0;
    for (int i = threadIdx.x; i < H; i += 256) {
        const double d = (double)a[i] - (double)b[i];
        dd += d * d;
        yy += (double)a[i] * (double)a[i];
    }
    __shared__ double r0[8], r1[8];
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        dd += __shfl_xor_sync(0xffffffffu, dd, o);
        yy += __shfl_xor_sync(0xffffffffu, yy, o);
    }
    if ((threadIdx.x & 31) == 0) {
        r0[threadIdx.x >> 5] = dd;
        r1[threadIdx.x >> 5] = yy;
    }
    __syncthreads();
    if (threadIdx.x == 0) {
        double d = 0.0, y = 0.0;
        for (int i = 0; i < 8; ++i) {
            d += r0[i];
            y += r1[i];
        }
        atomicAdd(acc, sqrt(d) / (sqrt(y) + (double)eps));
        atomicAdd(acc + 1, (double)(N - cnt[c]) / (double)N);
    }
}

struct ErrLayout {
    size_t mlp, yd, yk, idx, cnt, acc, total;
};

ErrLayout err_layout(int H, int N, int C, int K)
{
    ErrLayout L{};
    size_t off = 0;
    L.mlp = off;
    off += al256(ws_layout(H, N, C).total);
    L.yd = off;
    off += al256((size_t)C * H * sizeof(float));
    L.yk = off;
    off += al256((size_t)C * H * sizeof(float));
    L.idx = off;
    off += al256((size_t)C * N * sizeof(int32_t));
    L.cnt = off;
    off += al256((size_t)C * sizeof(int32_t));
    L.acc = off;
    off += al256((size_t)2 * (K > 0 ? K : 1) * sizeof(double));
    L.total = off;
    return L;
}

struct SatsLayout {
    size_t x, n, a, sel, err, total;
};

SatsLayout sats_layout(int H, int N, int C, int L, int K)
{
    SatsLayout S{};
    size_t off = 0;
    S.x = off;
    off += al256((size_t)C * H * sizeof(float));
    S.n = off;
    off += al256((size_t)L * C * H * sizeof(float));
    S.a = off;
    off += al256((size_t)C * N * sizeof(float));
    S.sel = off;
    off += al256(select_ws_bytes());
    S.err = off;
    off += err_layout(H, N, C, K).total;
    S.total = off;
    return S;
}

bool bad_t(double t) { return std::isnan(t) || t < 0.0; }

}  // namespace
}  // namespace sats

using namespace sats;

extern "C" {

sats_status sats_rmsnorm(const float *x, int B, int H, const float *w, float eps, float *out, void *stream)
{
    if (B < 0 || H < 1 || std::isnan(eps) || eps < 0.0f) return SATS_EINVAL;
    if (B == 0) return SATS_OK;
    if (!x || !w || !out) return SATS_EINVAL;
    rmsnorm_kernel<<<B, 256, 0, static_cast<cudaStream_t>(stream)>>>(x, H, w, eps, out);
    const cudaError_t e = cudaGetLastError();
    return e == cudaSuccess ? SATS_OK : cuda_fail(e, "rmsnorm kernel launch");
}

sats_status sats_gate_act_f32(const sats_layer *layer, const float *x, int B, float *a, void *stream)
{
    if (!layer || B < 0) return SATS_EINVAL;
    if (B == 0) return SATS_OK;
    if (!x || !a || (reinterpret_cast<uintptr_t>(x) & 15u)) return SATS_EINVAL;
    const cudaError_t e = launch_gate_act_f32(layer, x, B, a, static_cast<cudaStream_t>(stream));
    return e == cudaSuccess ? SATS_OK : cuda_fail(e, "gate activation kernel launch");
}

size_t sats_layer_err_workspace_bytes(int H, int N, int C, int K)
{
    if (H < 8 || H > kMaxH || (H % 8) != 0 || N < 1 || N > kMaxN || C < 1 || K < 0) return 0;
    return err_layout(H, N, C, K).total;
}

sats_status sats_layer_err(const sats_layer *layer, const float *x, int C, const float *t, int K, float eps,
                           double *err, double *sp, void *ws, size_t ws_bytes, void *stream)
{
    if (!layer || !x || C < 1 || K < 0 || !ws || (reinterpret_cast<uintptr_t>(x) & 15u) ||
        (reinterpret_cast<uintptr_t>(ws) & 255u))
        return SATS_EINVAL;
    if (K > 0 && (!t || !err || !sp)) return SATS_EINVAL;
    if (std::isnan(eps) || eps < 0.0f) return SATS_EINVAL;
    for (int k = 0; k < K; ++k)
        if (bad_t(t[k])) return SATS_EINVAL;
    const int H = layer->H, N = layer->N;
    const ErrLayout W = err_layout(H, N, C, K);
    if (ws_bytes < W.total) return SATS_ENOSPACE;
    if (K == 0) return SATS_OK;
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    char *base = static_cast<char *>(ws);
    void *mlp = base + W.mlp;
    float *yd = reinterpret_cast<float *>(base + W.yd), *yk = reinterpret_cast<float *>(base + W.yk);
    int32_t *idx = reinterpret_cast<int32_t *>(base + W.idx), *cnt = reinterpret_cast<int32_t *>(base + W.cnt);
    double *acc = reinterpret_cast<double *>(base + W.acc);
    cudaError_t e = clear_fused_state(mlp, H, N, C, st);
    if (e == cudaSuccess) e = cudaMemsetAsync(acc, 0, (size_t)2 * K * sizeof(double), st);
    if (e != cudaSuccess) return cuda_fail(e, "layer error workspace clear");
    const float zero = 0.0f;
    sats_status s = run_layer(layer, kXF32, x, C, &zero, nullptr, 0.f, nullptr, kOutY, yd, nullptr, nullptr,
                              nullptr, mlp, st);
    for (int k = 0; k < K && s == SATS_OK; ++k) {
        s = run_layer(layer, kXF32, x, C, &t[k], nullptr, 0.f, nullptr, kOutY, yk, idx, cnt, nullptr, mlp, st);
        if (s != SATS_OK) break;
        err_accum_kernel<<<C, 256, 0, st>>>(yd, yk, H, cnt, N, eps, acc + 2 * k);
        if ((e = cudaGetLastError()) != cudaSuccess) return cuda_fail(e, "error reduction kernel launch");
    }
    if (s != SATS_OK) return s;
    std::vector<double> h((size_t)2 * K);
    e = cudaMemcpyAsync(h.data(), acc, h.size() * sizeof(double), cudaMemcpyDeviceToHost, st);
    if (e == cudaSuccess) e = cudaStreamSynchronize(st);
    if (e != cudaSuccess) return cuda_fail(e, "layer error read-back");
    s = sats_get_error(mlp, ws_layout(H, N, C).total, stream);
    if (s != SATS_OK) return s;
    for (int k = 0; k < K; ++k) {
        err[k] = h[2 * (size_t)k] / C;
        sp[k] = h[2 * (size_t)k + 1] / C;
    }
    return SATS_OK;
}

sats_status sats_sats_select(const double *t, const double *err, const double *sp, int L, int K, double s_tar,
                             int guard, double guard_t, double guard_sp, double *b_out, double *t_out,
                             double *S_out)
{
    if (L < 1 || K < 0 || !t_out || !b_out || !S_out || std::isnan(s_tar)) return SATS_EINVAL;
    if (K > 0 && (!t || !err || !sp)) return SATS_EINVAL;
    if (guard >= L) return SATS_EINVAL;
    // per block, candidate indices by decreasing threshold (stable: the first listed wins a tie)
    std::vector<std::vector<int>> order((size_t)L);
    std::vector<double> budgets(1, 0.0);
    for (int l = 0; l < L; ++l) {
        std::vector<int> &o = order[(size_t)l];
        for (int k = 0; k < K; ++k) {
            const size_t i = (size_t)l * K + k;
            if (std::isnan(t[i]) || std::isnan(err[i]) || std::isnan(sp[i])) return SATS_EINVAL;
            o.push_back(k);
            budgets.push_back(err[i]);
        }
        std::stable_sort(o.begin(), o.end(), [&](int p, int q) { return t[(size_t)l * K + p] > t[(size_t)l * K + q]; });
    }
    std::sort(budgets.begin(), budgets.end());
    budgets.erase(std::unique(budgets.begin(), budgets.end()), budgets.end());
    // Eq. 7 for one block at budget b: the largest admissible threshold (index, or -1 for t = 0)
    auto pick = [&](int l, double b) {
        for (int k : order[(size_t)l]) {
            const size_t i = (size_t)l * K + k;
            if (t[i] <= 0.0) break;
            if (err[i] <= b) return k;
        }
        return -1;
    };
    double best_gap = INFINITY, best_b = 0.0, best_S = 0.0;
    for (double b : budgets) {   // Eqs. 8-10; increasing b, so a tie keeps the smaller budget
        double S = 0.0;
        for (int l = 0; l < L; ++l) {
            if (l == guard) {
                S += guard_sp;
                continue;
            }
            const int k = pick(l, b);
            S += k < 0 ? 0.0 : sp[(size_t)l * K + k];
        }
        S /= L;
        const double gap = std::fabs(S - s_tar);
        if (gap < best_gap) {
            best_gap = gap;
            best_b = b;
            best_S = S;
        }
    }
    for (int l = 0; l < L; ++l) {
        if (l == guard) {
            t_out[l] = guard_t;
            continue;
        }
        const int k = pick(l, best_b);
        t_out[l] = k < 0 ? 0.0 : t[(size_t)l * K + k];
    }
    *b_out = best_b;
    *S_out = best_S;
    return SATS_OK;
}

size_t sats_sats_workspace_bytes(int H, int N, int C, int L, int K0, int K1)
{
    if (H < 8 || H > kMaxH || (H % 8) != 0 || N < 1 || N > kMaxN || C < 1 || L < 1 || K0 < 2 || K1 < 0) return 0;
    const int K = std::max(std::max(K0 - 1, K1), 1);
    return sats_layout(H, N, C, L, K).total;
}

sats_status sats_sats_calibrate(const sats_layer *const *layers, const float *const *norm_w, int L, float eps,
                                const float *x_cal, int C, double s_tar, int K0, int K1, int guardrail, float err_eps,
                                float *t_out, double *b_out, double *S_out, double *table_t, double *table_err,
                                double *table_sp, void *ws, size_t ws_bytes, void *stream)
{
    if (!layers || !norm_w || L < 1 || !x_cal || C < 1 || K0 < 2 || K1 < 0 || !t_out || !ws) return SATS_EINVAL;
    if (std::isnan(eps) || eps < 0.0f || std::isnan(err_eps) || err_eps < 0.0f || !(s_tar >= 0.0 && s_tar <= 1.0))
        return SATS_EINVAL;
    if ((reinterpret_cast<uintptr_t>(x_cal) & 15u) || (reinterpret_cast<uintptr_t>(ws) & 255u)) return SATS_EINVAL;
    const int H = layers[0] ? layers[0]->H : 0, N = layers[0] ? layers[0]->N : 0;
    for (int l = 0; l < L; ++l)
        if (!layers[l] || layers[l]->H != H || layers[l]->N != N || !norm_w[l]) return SATS_EINVAL;
    const int Kc = K0 - 1, Kmax = std::max(std::max(Kc, K1), 1), Kt = Kc + K1;
    const SatsLayout W = sats_layout(H, N, C, L, Kmax);
    if (ws_bytes < W.total) return SATS_ENOSPACE;
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    char *base = static_cast<char *>(ws);
    float *x = reinterpret_cast<float *>(base + W.x);
    float *nall = reinterpret_cast<float *>(base + W.n);
    float *a = reinterpret_cast<float *>(base + W.a);
    void *sel = base + W.sel;
    void *ews = base + W.err;
    const size_t ews_bytes = W.total - W.err;
    void *mlp = base + W.err + err_layout(H, N, C, Kmax).mlp;
    auto n_of = [&](int l) { return nall + (size_t)l * C * H; };
    const int guard = guardrail ? L - 1 : -1;

    // 1-2: the dense stack gives each block's MLP inputs; coarse candidates from |SiLU(n W_gate)|
    cudaError_t e = cudaMemcpyAsync(x, x_cal, (size_t)C * H * sizeof(float), cudaMemcpyDeviceToDevice, st);
    if (e == cudaSuccess) e = clear_fused_state(mlp, H, N, C, st);
    if (e != cudaSuccess) return cuda_fail(e, "calibration set-up");
    std::vector<double> tc((size_t)L * Kc), amax((size_t)L), errc((size_t)L * Kc), spc((size_t)L * Kc);
    double g_t = 0.0, g_sp = 0.0;
    const float zero = 0.0f;
    sats_status s;
    for (int l = 0; l < L; ++l) {
        if ((s = sats_rmsnorm(x, C, H, norm_w[l], eps, n_of(l), stream)) != SATS_OK) return s;
        if ((s = sats_gate_act_f32(layers[l], n_of(l), C, a, stream)) != SATS_OK) return s;
        const int64_t n = (int64_t)C * N;
        for (int k = 1; k <= Kc; ++k) {   // Eq. 3 at k / K0
            float tv = 0.f;
            if ((s = sats_percentile_threshold(a, n, (double)k / K0, &tv, sel, select_ws_bytes(), stream)) != SATS_OK)
                return s;
            tc[(size_t)l * Kc + k - 1] = tv;
        }
        float mx = 0.f;
        if ((s = sats_percentile_threshold(a, n, 1.0, &mx, sel, select_ws_bytes(), stream)) != SATS_OK) return s;
        amax[(size_t)l] = mx;
        if (l == guard) {
            float gt = 0.f;
            if ((s = sats_percentile_threshold(a, n, s_tar, &gt, sel, select_ws_bytes(), stream)) != SATS_OK)
                return s;
            g_t = gt;
        }
        // x <- x + MLP_l(n_l) with every neuron kept
        if ((s = run_layer(layers[l], kXF32, n_of(l), C, &zero, nullptr, 0.f, nullptr, kOutResid, x, nullptr,
                           nullptr, nullptr, mlp, st)) != SATS_OK)
            return s;
    }
    // 3: Eq. 6 for every coarse candidate (and the guardrail's CATS threshold)
    std::vector<float> tf((size_t)Kmax);
    std::vector<double> eb((size_t)Kmax), sb((size_t)Kmax);
    for (int l = 0; l < L; ++l) {
        for (int k = 0; k < Kc; ++k) tf[(size_t)k] = (float)tc[(size_t)l * Kc + k];
        if ((s = sats_layer_err(layers[l], n_of(l), C, tf.data(), Kc, err_eps, eb.data(), sb.data(), ews, ews_bytes,
                                stream)) != SATS_OK)
            return s;
        for (int k = 0; k < Kc; ++k) {
            errc[(size_t)l * Kc + k] = eb[(size_t)k];
            spc[(size_t)l * Kc + k] = sb[(size_t)k];
        }
        if (l == guard) {
            const float gt = (float)g_t;
            double ge = 0.0;
            if ((s = sats_layer_err(layers[l], n_of(l), C, &gt, 1, err_eps, &ge, &g_sp, ews, ews_bytes, stream)) !=
                SATS_OK)
                return s;
        }
    }
    // 4: Eqs. 7-10 over the coarse candidates
    double b0 = 0.0, S0 = 0.0;
    std::vector<double> t0((size_t)L);
    if ((s = sats_sats_select(tc.data(), errc.data(), spc.data(), L, Kc, s_tar, guard, g_t, g_sp, &b0, t0.data(),
                              &S0)) != SATS_OK)
        return s;
    // 5-6: K1 candidates strictly between the coarse neighbours of each block's choice, then
    // Eqs. 6-10 over coarse and fine candidates together
    std::vector<double> ta((size_t)L * Kt), ea((size_t)L * Kt), sa((size_t)L * Kt);
    for (int l = 0; l < L; ++l) {
        double lo = 0.0, hi = amax[(size_t)l];
        bool above = false;
        for (int k = 0; k < Kc; ++k) {
            const double v = tc[(size_t)l * Kc + k];
            if (v < t0[(size_t)l]) lo = std::max(lo, v);
            if (v > t0[(size_t)l]) {
                hi = above ? std::min(hi, v) : v;
                above = true;
            }
        }
        for (int k = 0; k < Kc; ++k) {
            ta[(size_t)l * Kt + k] = tc[(size_t)l * Kc + k];
            ea[(size_t)l * Kt + k] = errc[(size_t)l * Kc + k];
            sa[(size_t)l * Kt + k] = spc[(size_t)l * Kc + k];
        }
        for (int k = 0; k < K1; ++k) tf[(size_t)k] = (float)(lo + (hi - lo) * (k + 1) / (K1 + 1));
        if (K1 > 0 && (s = sats_layer_err(layers[l], n_of(l), C, tf.data(), K1, err_eps, eb.data(), sb.data(), ews,
                                          ews_bytes, stream)) != SATS_OK)
            return s;
        for (int k = 0; k < K1; ++k) {
            ta[(size_t)l * Kt + Kc + k] = tf[(size_t)k];
            ea[(size_t)l * Kt + Kc + k] = eb[(size_t)k];
            sa[(size_t)l * Kt + Kc + k] = sb[(size_t)k];
        }
    }
    double b = 0.0, S = 0.0;
    std::vector<double> tt((size_t)L);
    if ((s = sats_sats_select(ta.data(), ea.data(), sa.data(), L, Kt, s_tar, guard, g_t, g_sp, &b, tt.data(), &S)) !=
        SATS_OK)
        return s;
    for (int l = 0; l < L; ++l) t_out[l] = (float)tt[(size_t)l];
    if (b_out) *b_out = b;
    if (S_out) *S_out = S;
    if (table_t && table_err && table_sp) {
        std::copy(ta.begin(), ta.end(), table_t);
        std::copy(ea.begin(), ea.end(), table_err);
        std::copy(sa.begin(), sa.end(), table_sp);
    }
    return SATS_OK;
}

}  // extern "C"

// ---------------------------------------------------------------------- routing calibration (Sec. 3.2)
namespace sats {
namespace {

// Eqs. 11-12, the sums: for every occurrence, d = max(0, l_sparse - l_base) into the token's total.
__global__ void score_accum_kernel(const int32_t *__restrict__ ids, const float *__restrict__ lb,
                                   const float *__restrict__ ls, int64_t n, int V, double *__restrict__ total,
                                   unsigned *__restrict__ count, int32_t *__restrict__ status)
{
    for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x) {
        const int id = ids[i];
        if (id < 0 || id >= V) {
            atomicOr(status, kStatusBadToken);
            continue;
        }
        atomicAdd(total + id, (double)fmaxf(0.0f, ls[i] - lb[i]));
        atomicAdd(count + id, 1u);
    }
}

// Eq. 12, the means; +inf for a token that never occurs (it keeps the base path).
__global__ void score_final_kernel(const double *__restrict__ total, const unsigned *__restrict__ count, int V,
                                   float *__restrict__ score)
{
    const int v = blockIdx.x * blockDim.x + threadIdx.x;
    if (v < V) score[v] = count[v] ? (float)(total[v] / count[v]) : INFINITY;
}

__global__ void freq_kernel(const int32_t *__restrict__ ids, int64_t m, int V, unsigned *__restrict__ freq,
                            int32_t *__restrict__ status)
{
    for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < m; i += (int64_t)gridDim.x * blockDim.x) {
        const int id = ids[i];
        if (id < 0 || id >= V) {
            atomicOr(status, kStatusBadToken);
            continue;
        }
        atomicAdd(freq + id, 1u);
    }
}

// Eq. 13 as a table: 1 (base path) where score >= tau, 0 (sparse path) where score < tau.
__global__ void lut_kernel(const float *__restrict__ score, int V, float tau, uint8_t *__restrict__ lut)
{
    const int v = blockIdx.x * blockDim.x + threadIdx.x;
    if (v < V) lut[v] = score[v] < tau ? 0 : 1;
}

struct ScoreLayout {
    size_t status, total, count, total_bytes;
};

ScoreLayout score_layout(int V)
{
    ScoreLayout S{};
    size_t off = 0;
    S.status = off;
    off += 256;
    S.total = off;
    off += al256((size_t)V * sizeof(double));
    S.count = off;
    off += al256((size_t)V * sizeof(unsigned));
    S.total_bytes = off;
    return S;
}

sats_status read_status_word(int32_t *word, cudaStream_t st)
{
    int32_t v = 0;
    cudaError_t e = cudaMemcpyAsync(&v, word, sizeof v, cudaMemcpyDeviceToHost, st);
    if (e == cudaSuccess) e = cudaStreamSynchronize(st);
    if (e != cudaSuccess) return cuda_fail(e, "status read");
    return (v & kStatusBadToken) ? SATS_EDEVICE : SATS_OK;
}

int grid_for(int64_t n)
{
    const int64_t g = (n + 255) / 256;
    return (int)(g < 4096 ? (g > 0 ? g : 1) : 4096);
}

}  // namespace
}  // namespace sats

extern "C" {

size_t sats_route_calib_workspace_bytes(int V)
{
    if (V < 1) return 0;
    return score_layout(V).total_bytes;
}

sats_status sats_token_scores(const int32_t *ids, const float *l_base, const float *l_sparse, int64_t n, int V,
                              float *score, void *ws, size_t ws_bytes, void *stream)
{
    if (V < 1 || n < 0 || !score || !ws || (n > 0 && (!ids || !l_base || !l_sparse))) return SATS_EINVAL;
    const ScoreLayout S = score_layout(V);
    if (ws_bytes < S.total_bytes || (reinterpret_cast<uintptr_t>(ws) & 255u)) return ws_bytes < S.total_bytes ? SATS_ENOSPACE : SATS_EINVAL;
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    char *base = static_cast<char *>(ws);
    int32_t *status = reinterpret_cast<int32_t *>(base + S.status);
    double *total = reinterpret_cast<double *>(base + S.total);
    unsigned *count = reinterpret_cast<unsigned *>(base + S.count);
    cudaError_t e = cudaMemsetAsync(ws, 0, S.total_bytes, st);
    if (e != cudaSuccess) return cuda_fail(e, "score workspace clear");
    if (n > 0) score_accum_kernel<<<grid_for(n), 256, 0, st>>>(ids, l_base, l_sparse, n, V, total, count, status);
    score_final_kernel<<<(V + 255) / 256, 256, 0, st>>>(total, count, V, score);
    if ((e = cudaGetLastError()) != cudaSuccess) return cuda_fail(e, "score kernel launch");
    return read_status_word(status, st);
}

sats_status sats_route_calibrate(const float *score, int V, const int32_t *heldout_ids, int64_t m, double r_tar,
                                 float *tau_out, double *R_out, uint8_t *lut, void *ws, size_t ws_bytes, void *stream)
{
    if (V < 1 || m < 0 || !score || !tau_out || !ws || std::isnan(r_tar) || (m > 0 && !heldout_ids)) return SATS_EINVAL;
    const ScoreLayout S = score_layout(V);
    if (ws_bytes < S.total_bytes || (reinterpret_cast<uintptr_t>(ws) & 255u)) return ws_bytes < S.total_bytes ? SATS_ENOSPACE : SATS_EINVAL;
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    char *base = static_cast<char *>(ws);
    int32_t *status = reinterpret_cast<int32_t *>(base + S.status);
    unsigned *freq = reinterpret_cast<unsigned *>(base + S.count);
    cudaError_t e = cudaMemsetAsync(status, 0, 256, st);
    if (e == cudaSuccess) e = cudaMemsetAsync(freq, 0, (size_t)V * sizeof(unsigned), st);
    if (e != cudaSuccess) return cuda_fail(e, "held-out count clear");
    if (m > 0) freq_kernel<<<grid_for(m), 256, 0, st>>>(heldout_ids, m, V, freq, status);
    if ((e = cudaGetLastError()) != cudaSuccess) return cuda_fail(e, "held-out count kernel launch");
    sats_status s = read_status_word(status, st);
    if (s != SATS_OK) return s;
    // Eq. 14 on the host over the V scores: R(tau) = (held-out occurrences with score < tau) / m
    std::vector<float> sc((size_t)V);
    std::vector<unsigned> fr((size_t)V);
    e = cudaMemcpyAsync(sc.data(), score, sc.size() * sizeof(float), cudaMemcpyDeviceToHost, st);
    if (e == cudaSuccess) e = cudaMemcpyAsync(fr.data(), freq, fr.size() * sizeof(unsigned), cudaMemcpyDeviceToHost, st);
    if (e == cudaSuccess) e = cudaStreamSynchronize(st);
    if (e != cudaSuccess) return cuda_fail(e, "score read-back");
    std::vector<std::pair<float, unsigned>> occ;
    for (int v = 0; v < V; ++v)
        if (fr[(size_t)v]) occ.emplace_back(sc[(size_t)v], fr[(size_t)v]);
    std::sort(occ.begin(), occ.end());
    // candidates in increasing order: 0, each distinct finite held-out score, +inf; below(tau) is the
    // number of held-out occurrences whose score is < tau
    const double M = m > 0 ? (double)m : 1.0;
    double best_gap = INFINITY, best_R = 0.0;
    float best_tau = 0.0f;
    auto consider = [&](float tau, uint64_t below) {
        const double R = (double)below / M;
        const double gap = std::fabs(R - r_tar);
        if (gap < best_gap) {
            best_gap = gap;
            best_tau = tau;
            best_R = R;
        }
    };
    uint64_t below = 0;
    size_t i = 0;
    while (i < occ.size() && occ[i].first < 0.0f) below += occ[i++].second;   // (scores are >= 0)
    consider(0.0f, below);
    while (i < occ.size() && std::isfinite(occ[i].first)) {
        const float v = occ[i].first;
        if (v > 0.0f) consider(v, below);   // R(v) counts the scores strictly below v
        while (i < occ.size() && occ[i].first == v) below += occ[i++].second;
    }
    consider(INFINITY, below);
    *tau_out = best_tau;
    if (R_out) *R_out = best_R;
    if (lut) {
        lut_kernel<<<(V + 255) / 256, 256, 0, st>>>(score, V, best_tau, lut);
        if ((e = cudaGetLastError()) != cudaSuccess) return cuda_fail(e, "table kernel launch");
    }
    return SATS_OK;
}

}  // extern "C"
