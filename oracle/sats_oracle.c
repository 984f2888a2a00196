/*
 * sats_oracle.c -- CPU oracle for the thresholded gated MLP and token routing.
 *
 * TEST INFRASTRUCTURE ONLY.  Only tests/, __graft_entry__.smoke() and the
 * cpu_baseline / reference legs of bench.py may load this library.  It shares
 * no code, header, table or helper with the CUDA library under
 * paper_2607_08991_gb300/; neither side includes or links the other.
 *
 * Every routine is a plain, slow, literal statement of one equation of
 * "Sensitivity-Aware Thresholding and Token Routing for Activation
 * Sparsification in Large Language Models" (arXiv 2607.08991), computed in
 * IEEE double precision on the exact values of the bf16 inputs:
 *
 *   oracle_silu               Sec. 2, Eq. 2    SiLU(z) = z / (1 + e^-z)
 *   oracle_gate_act           Sec. 2, Eqs. 1-2 a = SiLU(x W_gate)
 *   oracle_up_proj            Sec. 2, Eq. 1    u = x W_up
 *   oracle_cats_mask          Sec. 2, Eqs. 4-5 keep_j = |a_j| >= t
 *   oracle_masked_mlp         Sec. 2, Eqs. 1,5 y = (CATS_t(a) * u) W_down
 *   oracle_sparse_mlp         Sec. 2, Eqs. 1-5 composition of the above
 *   oracle_dense_mlp          Sec. 2, Eq. 1    the base (unthresholded) MLP
 *   oracle_percentile_threshold  Sec. 2, Eq. 3 t = min{t' : F(t') >= k}
 *   oracle_route              Sec. 3.2, Eq. 13 LUT lookup, dense group first
 *   oracle_rmsnorm            pre-MLP RMSNorm of a Llama/Qwen decoder block
 *   oracle_mlp_stack          Sec. 3.2: a token routed to the sparse path uses
 *                             the thresholded MLP in every block, a base token
 *                             uses the dense MLP in every block.
 *   oracle_layer_err          Sec. 3.1, Eq. 6  Err_l(t) and the sparsity sp_l(t)
 *                             of one block at candidate thresholds
 *   oracle_sats_select        Sec. 3.1, Eqs. 7-10 t*_l(b), T*(b), S(b), b*
 *   oracle_sparse_mlp_lora    Sec. 4 (fine-tuned routing): the sparse path on
 *                             LoRA-adapted weights W + scale A B, the low-rank
 *                             terms applied without forming W + scale A B
 *
 * Layouts follow the paper's row-vector convention x W: W_gate and W_up are
 * [H][N] (hidden x intermediate), W_down is [N][H], all row-major bf16 bit
 * patterns (uint16).  Activations are double [B][H].
 *
 * Ties at the threshold.  The mask is discontinuous at |a| = t: a neuron whose
 * |a| lies within a relative distance band_rel of t may be decided either way
 * by any finite-precision evaluation.  When a caller passes keep_hint and
 * band_rel > 0, the oracle takes the hint's decision for such in-band neurons
 * only (both decisions are admissible results of Eq. 5); every other decision
 * is the oracle's own.  With keep_hint == NULL the routines are exactly Eq. 5.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

/* bf16 bit pattern -> its exact value (bf16 is the top half of a binary32). */
static double bf16_value(uint16_t bits)
{
    uint32_t u = ((uint32_t)bits) << 16;
    float f;
    memcpy(&f, &u, sizeof f);
    return (double)f;
}

void oracle_bf16_to_f64(int64_t n, const uint16_t *src, double *dst)
{
    for (int64_t i = 0; i < n; ++i) dst[i] = bf16_value(src[i]);
}

/* Sec. 2, Eq. 2. */
double oracle_silu(double z)
{
    return z / (1.0 + exp(-z));
}

/* Sec. 2, Eqs. 1-2: a[b][j] = SiLU(sum_k x[b][k] * W_gate[k][j]). */
void oracle_gate_act(int B, int H, int N, const double *x, const uint16_t *Wg, double *a)
{
    double *g = (double *)malloc(sizeof(double) * (size_t)N);
    for (int b = 0; b < B; ++b) {
        for (int j = 0; j < N; ++j) g[j] = 0.0;
        for (int k = 0; k < H; ++k) {
            const double xk = x[(size_t)b * H + k];
            const uint16_t *row = Wg + (size_t)k * N;
            for (int j = 0; j < N; ++j) g[j] += xk * bf16_value(row[j]);
        }
        for (int j = 0; j < N; ++j) a[(size_t)b * N + j] = oracle_silu(g[j]);
    }
    free(g);
}

/* Sec. 2, Eq. 1: u[b][j] = sum_k x[b][k] * W_up[k][j]. */
void oracle_up_proj(int B, int H, int N, const double *x, const uint16_t *Wu, double *u)
{
    for (int b = 0; b < B; ++b) {
        double *ub = u + (size_t)b * N;
        for (int j = 0; j < N; ++j) ub[j] = 0.0;
        for (int k = 0; k < H; ++k) {
            const double xk = x[(size_t)b * H + k];
            const uint16_t *row = Wu + (size_t)k * N;
            for (int j = 0; j < N; ++j) ub[j] += xk * bf16_value(row[j]);
        }
    }
}

/* Sec. 2, Eqs. 4-5: keep a_j iff |a_j| >= t (t per token).  Returns the number
 * of in-band neurons (| |a|-t | <= band_rel * t) for which keep_hint decided. */
int64_t oracle_cats_mask(int B, int N, const double *a, const double *t,
                         const uint8_t *keep_hint, double band_rel, uint8_t *keep)
{
    int64_t in_band = 0;
    for (int b = 0; b < B; ++b) {
        for (int j = 0; j < N; ++j) {
            const size_t i = (size_t)b * N + j;
            const double mag = fabs(a[i]);
            uint8_t k = (uint8_t)(mag >= t[b]);
            if (keep_hint && band_rel > 0.0 && isfinite(t[b]) &&
                fabs(mag - t[b]) <= band_rel * t[b]) {
                k = keep_hint[i] ? 1 : 0;
                ++in_band;
            }
            keep[i] = k;
        }
    }
    return in_band;
}

/* Sec. 2, Eqs. 1 and 5 with the mask given:
 * y[b][i] = sum_j (keep[b][j] ? a[b][j] : 0) * u[b][j] * W_down[j][i]. */
void oracle_masked_mlp(int B, int H, int N, const double *x, const uint16_t *Wg,
                       const uint16_t *Wu, const uint16_t *Wd, const uint8_t *keep, double *y)
{
    double *a = (double *)malloc(sizeof(double) * (size_t)B * N);
    double *u = (double *)malloc(sizeof(double) * (size_t)B * N);
    oracle_gate_act(B, H, N, x, Wg, a);
    oracle_up_proj(B, H, N, x, Wu, u);
    for (int b = 0; b < B; ++b) {
        double *yb = y + (size_t)b * H;
        for (int i = 0; i < H; ++i) yb[i] = 0.0;
        for (int j = 0; j < N; ++j) {
            const size_t bj = (size_t)b * N + j;
            const double cats = keep[bj] ? a[bj] : 0.0;   /* CATS_t(SiLU(x W_gate)) */
            const double h = cats * u[bj];
            const uint16_t *row = Wd + (size_t)j * H;
            for (int i = 0; i < H; ++i) yb[i] += h * bf16_value(row[i]);
        }
    }
    free(a);
    free(u);
}

/* Sec. 2, Eqs. 1-5: the thresholded gated MLP for per-token thresholds t[b].
 * a_out ([B][N]) and keep_out ([B][N]) are optional.  Returns the in-band count. */
int64_t oracle_sparse_mlp(int B, int H, int N, const double *x, const uint16_t *Wg,
                          const uint16_t *Wu, const uint16_t *Wd, const double *t,
                          const uint8_t *keep_hint, double band_rel,
                          double *y, double *a_out, uint8_t *keep_out)
{
    double *a = (double *)malloc(sizeof(double) * (size_t)B * N);
    uint8_t *keep = (uint8_t *)malloc((size_t)B * N);
    oracle_gate_act(B, H, N, x, Wg, a);
    const int64_t in_band = oracle_cats_mask(B, N, a, t, keep_hint, band_rel, keep);
    oracle_masked_mlp(B, H, N, x, Wg, Wu, Wd, keep, y);
    if (a_out) memcpy(a_out, a, sizeof(double) * (size_t)B * N);
    if (keep_out) memcpy(keep_out, keep, (size_t)B * N);
    free(a);
    free(keep);
    return in_band;
}

/* Sec. 4, fine-tuned models: the sparse path runs the thresholded MLP of Sec. 2
 * (Eqs. 1-5) on LoRA-adapted projections W + scale A B (A: [in][r], B: [r][out]),
 * with the low-rank products taken factor by factor:
 *   g = x W_gate + scale (x A_g) B_g,   a = SiLU(g),   keep = |a| >= t  (Eqs. 1-5)
 *   u = x W_up   + scale (x A_u) B_u,   h = keep ? a u : 0
 *   y = h W_down + scale (h A_d) B_d
 * A_g, A_u [H][r]; B_g, B_u [r][N]; A_d [N][r]; B_d [r][H]; bf16 bit patterns.
 * keep_hint / band_rel as for oracle_sparse_mlp.  Returns the in-band count. */
int64_t oracle_sparse_mlp_lora(int B, int H, int N, int r, const double *x, const uint16_t *Wg,
                               const uint16_t *Wu, const uint16_t *Wd, const uint16_t *Ag,
                               const uint16_t *Bg, const uint16_t *Au, const uint16_t *Bu,
                               const uint16_t *Ad, const uint16_t *Bd, double scale, const double *t,
                               const uint8_t *keep_hint, double band_rel,
                               double *y, double *a_out, uint8_t *keep_out)
{
    double *a = (double *)malloc(sizeof(double) * (size_t)B * N);
    double *u = (double *)malloc(sizeof(double) * (size_t)B * N);
    uint8_t *keep = (uint8_t *)malloc((size_t)B * N);
    double *zg = (double *)malloc(sizeof(double) * (size_t)r);
    double *zu = (double *)malloc(sizeof(double) * (size_t)r);
    double *w = (double *)malloc(sizeof(double) * (size_t)r);
    for (int b = 0; b < B; ++b) {
        const double *xb = x + (size_t)b * H;
        for (int q = 0; q < r; ++q) {   /* x A_g, x A_u */
            zg[q] = 0.0;
            zu[q] = 0.0;
            for (int k = 0; k < H; ++k) {
                zg[q] += xb[k] * bf16_value(Ag[(size_t)k * r + q]);
                zu[q] += xb[k] * bf16_value(Au[(size_t)k * r + q]);
            }
        }
        for (int j = 0; j < N; ++j) {
            double g = 0.0, v = 0.0, lg = 0.0, lu = 0.0;
            for (int k = 0; k < H; ++k) {
                g += xb[k] * bf16_value(Wg[(size_t)k * N + j]);
                v += xb[k] * bf16_value(Wu[(size_t)k * N + j]);
            }
            for (int q = 0; q < r; ++q) {
                lg += zg[q] * bf16_value(Bg[(size_t)q * N + j]);
                lu += zu[q] * bf16_value(Bu[(size_t)q * N + j]);
            }
            a[(size_t)b * N + j] = oracle_silu(g + scale * lg);
            u[(size_t)b * N + j] = v + scale * lu;
        }
    }
    const int64_t in_band = oracle_cats_mask(B, N, a, t, keep_hint, band_rel, keep);
    for (int b = 0; b < B; ++b) {
        double *yb = y + (size_t)b * H;
        for (int i = 0; i < H; ++i) yb[i] = 0.0;
        for (int q = 0; q < r; ++q) w[q] = 0.0;
        for (int j = 0; j < N; ++j) {
            const size_t bj = (size_t)b * N + j;
            const double h = keep[bj] ? a[bj] * u[bj] : 0.0;
            for (int i = 0; i < H; ++i) yb[i] += h * bf16_value(Wd[(size_t)j * H + i]);
            for (int q = 0; q < r; ++q) w[q] += h * bf16_value(Ad[(size_t)j * r + q]);   /* h A_d */
        }
        for (int q = 0; q < r; ++q)
            for (int i = 0; i < H; ++i) yb[i] += scale * w[q] * bf16_value(Bd[(size_t)q * H + i]);
    }
    if (a_out) memcpy(a_out, a, sizeof(double) * (size_t)B * N);
    if (keep_out) memcpy(keep_out, keep, (size_t)B * N);
    free(a);
    free(u);
    free(keep);
    free(zg);
    free(zu);
    free(w);
    return in_band;
}

/* Sec. 2, Eq. 1 written out on its own (no mask anywhere):
 * y = (SiLU(x W_gate) * (x W_up)) W_down. */
void oracle_dense_mlp(int B, int H, int N, const double *x, const uint16_t *Wg,
                      const uint16_t *Wu, const uint16_t *Wd, double *y)
{
    double *h = (double *)malloc(sizeof(double) * (size_t)N);
    for (int b = 0; b < B; ++b) {
        const double *xb = x + (size_t)b * H;
        for (int j = 0; j < N; ++j) {
            double g = 0.0, u = 0.0;
            for (int k = 0; k < H; ++k) {
                g += xb[k] * bf16_value(Wg[(size_t)k * N + j]);
                u += xb[k] * bf16_value(Wu[(size_t)k * N + j]);
            }
            h[j] = oracle_silu(g) * u;
        }
        for (int i = 0; i < H; ++i) {
            double s = 0.0;
            for (int j = 0; j < N; ++j) s += h[j] * bf16_value(Wd[(size_t)j * H + i]);
            y[(size_t)b * H + i] = s;
        }
    }
    free(h);
}

static int cmp_double(const void *p, const void *q)
{
    const double a = *(const double *)p, b = *(const double *)q;
    return (a > b) - (a < b);
}

/* Sec. 2, Eq. 3 with the empirical CDF F of the magnitudes |v_i| (i < n):
 * t = min{t' : F(t') >= k} = the m-th smallest |v_i|, m = ceil(k n).
 * k is read as the decimal fraction it stands for (0.1 means one tenth): the
 * product k*n is taken down by a relative 2^-50 before the ceiling, which
 * absorbs the binary representation error of k and of the product, so that
 * 0.1 * 100 gives m = 10, not 11.  k <= 0 gives t = 0 (every value kept);
 * k > 1 gives +inf (none kept). */
double oracle_percentile_threshold(const double *v, int64_t n, double k)
{
    if (n <= 0 || !(k > 0.0)) return 0.0;
    if (k > 1.0) return INFINITY;
    const double prod = k * (double)n;
    int64_t m = (int64_t)ceil(prod * (1.0 - ldexp(1.0, -50)));
    if (m < 1) m = 1;
    if (m > n) m = n;
    double *s = (double *)malloc(sizeof(double) * (size_t)n);
    for (int64_t i = 0; i < n; ++i) s[i] = fabs(v[i]);
    qsort(s, (size_t)n, sizeof(double), cmp_double);
    const double t = s[m - 1];
    free(s);
    return t;
}

/* Sec. 3.2, Eq. 13 as a lookup table: lut[v] != 0 marks a token id v routed
 * to the base (dense) path, lut[v] == 0 the sparse path.  perm lists the
 * base-path positions in increasing order, then the sparse-path positions in
 * increasing order; *n_dense is the number of base-path tokens.
 * Returns 0, or -1 if any id lies outside [0, V) (perm is then unspecified). */
int oracle_route(int B, const int32_t *ids, int V, const uint8_t *lut,
                 int32_t *perm, int32_t *n_dense)
{
    for (int b = 0; b < B; ++b)
        if (ids[b] < 0 || ids[b] >= V) return -1;
    int n = 0;
    for (int b = 0; b < B; ++b)
        if (lut[ids[b]]) perm[n++] = b;
    *n_dense = n;
    for (int b = 0; b < B; ++b)
        if (!lut[ids[b]]) perm[n++] = b;
    return 0;
}

/* RMSNorm: out[b][i] = x[b][i] / sqrt(mean_i x[b][i]^2 + eps) * w[i]. */
void oracle_rmsnorm(int B, int H, const double *x, const float *w, double eps, double *out)
{
    for (int b = 0; b < B; ++b) {
        double ss = 0.0;
        for (int i = 0; i < H; ++i) ss += x[(size_t)b * H + i] * x[(size_t)b * H + i];
        const double inv = 1.0 / sqrt(ss / H + eps);
        for (int i = 0; i < H; ++i)
            out[(size_t)b * H + i] = x[(size_t)b * H + i] * inv * (double)w[i];
    }
}

/* A stack of L gated-MLP blocks with RMSNorm and a residual add:
 *   x <- x + MLP_l(RMSNorm(x) * w_l),  l = 0..L-1.
 * Routing (Sec. 3.2) is decided once per token from its id: a base-path token
 * runs oracle_dense_mlp in every block, a sparse-path token the CATS-masked
 * MLP with the block's threshold t[l].  ids == NULL routes every token to the
 * sparse path.  x is [B][H] in/out.  keep_out ([L][B][N], optional) receives
 * the per-layer masks (all ones for base-path tokens).  keep_hint/band_rel
 * decide in-band neurons as in oracle_cats_mask (layout [L][B][N]).
 * Returns the total in-band count, or -1 for an id outside [0, V). */
int64_t oracle_mlp_stack(int L, int B, int H, int N,
                         const uint16_t *const *Wg, const uint16_t *const *Wu,
                         const uint16_t *const *Wd, const float *const *norm_w,
                         const double *t, double eps,
                         const int32_t *ids, const uint8_t *lut, int V,
                         double *x, const uint8_t *keep_hint, double band_rel,
                         uint8_t *keep_out)
{
    uint8_t *dense = (uint8_t *)calloc((size_t)(B > 0 ? B : 1), 1);
    if (ids) {
        for (int b = 0; b < B; ++b) {
            if (ids[b] < 0 || ids[b] >= V) { free(dense); return -1; }
            dense[b] = lut[ids[b]] ? 1 : 0;
        }
    }
    double *xn = (double *)malloc(sizeof(double) * (size_t)H);
    double *y = (double *)malloc(sizeof(double) * (size_t)H);
    uint8_t *keep = (uint8_t *)malloc((size_t)N);
    int64_t in_band = 0;
    for (int l = 0; l < L; ++l) {
        for (int b = 0; b < B; ++b) {
            double *xb = x + (size_t)b * H;
            oracle_rmsnorm(1, H, xb, norm_w[l], eps, xn);
            const size_t off = ((size_t)l * B + b) * N;
            if (dense[b]) {
                oracle_dense_mlp(1, H, N, xn, Wg[l], Wu[l], Wd[l], y);
                memset(keep, 1, (size_t)N);
            } else {
                const double tb = t[l];
                in_band += oracle_sparse_mlp(1, H, N, xn, Wg[l], Wu[l], Wd[l], &tb,
                                             keep_hint ? keep_hint + off : NULL, band_rel,
                                             y, NULL, keep);
            }
            if (keep_out) memcpy(keep_out + off, keep, (size_t)N);
            for (int i = 0; i < H; ++i) xb[i] += y[i];
        }
    }
    free(dense);
    free(xn);
    free(y);
    free(keep);
    return in_band;
}

/* Sec. 3.1, Eq. 6: the local thresholding error of one block at each of K
 * candidate thresholds t[k], over C calibration inputs x [C][H] (the block's
 * MLP inputs):
 *   err[k] = (1/C) sum_c ||y(x_c) - y~_{t_k}(x_c)||_2 / (||y(x_c)||_2 + eps)
 * with y the dense output (Eq. 1) and y~_t the thresholded output (Eqs. 4-5).
 * sp[k] = (1/C) sum_c (number of neurons with |a_j| < t_k) / N, the realised
 * sparsity of the block under t_k that Eq. 9 averages. */
void oracle_layer_err(int C, int H, int N, const double *x, const uint16_t *Wg, const uint16_t *Wu,
                      const uint16_t *Wd, int K, const double *t, double eps, double *err, double *sp)
{
    double *y = (double *)malloc(sizeof(double) * (size_t)C * H);
    double *yt = (double *)malloc(sizeof(double) * (size_t)C * H);
    uint8_t *keep = (uint8_t *)malloc((size_t)C * N);
    double *tt = (double *)malloc(sizeof(double) * (size_t)(C > 0 ? C : 1));
    oracle_dense_mlp(C, H, N, x, Wg, Wu, Wd, y);
    for (int k = 0; k < K; ++k) {
        for (int c = 0; c < C; ++c) tt[c] = t[k];
        oracle_sparse_mlp(C, H, N, x, Wg, Wu, Wd, tt, NULL, 0.0, yt, NULL, keep);
        double e = 0.0, z = 0.0;
        for (int c = 0; c < C; ++c) {
            double dd = 0.0, yy = 0.0;
            for (int i = 0; i < H; ++i) {
                const double d = y[(size_t)c * H + i] - yt[(size_t)c * H + i];
                dd += d * d;
                yy += y[(size_t)c * H + i] * y[(size_t)c * H + i];
            }
            e += sqrt(dd) / (sqrt(yy) + eps);
            int64_t off = 0;
            for (int j = 0; j < N; ++j) off += keep[(size_t)c * N + j] ? 0 : 1;
            z += (double)off / (double)N;
        }
        err[k] = C > 0 ? e / C : 0.0;
        sp[k] = C > 0 ? z / C : 0.0;
    }
    free(y);
    free(yt);
    free(keep);
    free(tt);
}

/* Sec. 3.1, Eqs. 7-10 over a table of candidates: t, err, sp are [L][K]
 * (candidate k of block l with its Eq. 6 error and its sparsity).  Every block
 * also has the candidate t = 0 (nothing removed: error 0, sparsity 0).
 *   Eq. 7:  t*_l(b) = max{t in T_l : Err_l(t) <= b}
 *   Eq. 8:  T*(b) = [t*_1(b), ..., t*_L(b)]
 *   Eq. 9:  S(b) = (1/L) sum_l sp_l(t*_l(b))
 *   Eq. 10: b* = argmin_b |S(b) - s_tar|
 * b ranges over 0 and every error value in the table (S changes only there),
 * in increasing order; a tie in Eq. 10 goes to the smaller budget.  Block
 * `guard` (if >= 0) keeps the fixed threshold guard_t with sparsity guard_sp
 * and takes no part in Eq. 7 (the final-block guardrail of Sec. 4).
 * Writes b*, T*(b*) and S(b*). */
void oracle_sats_select(int L, int K, const double *t, const double *err, const double *sp, double s_tar,
                        int guard, double guard_t, double guard_sp, double *b_out, double *t_out, double *S_out)
{
    const int nb = 1 + L * K;
    double *budgets = (double *)malloc(sizeof(double) * (size_t)nb);
    budgets[0] = 0.0;
    for (int i = 0; i < L * K; ++i) budgets[1 + i] = err[i];
    qsort(budgets, (size_t)nb, sizeof(double), cmp_double);
    double best_gap = INFINITY, best_b = 0.0, best_S = 0.0;
    for (int q = 0; q < nb; ++q) {
        const double b = budgets[q];
        if (q > 0 && b == budgets[q - 1]) continue;
        double S = 0.0;
        for (int l = 0; l < L; ++l) {
            if (l == guard) { S += guard_sp; continue; }
            double tl = 0.0, sl = 0.0;            /* the t = 0 candidate */
            for (int k = 0; k < K; ++k) {
                const int i = l * K + k;
                if (err[i] <= b && t[i] > tl) { tl = t[i]; sl = sp[i]; }
            }
            S += sl;
        }
        S /= L;
        const double gap = fabs(S - s_tar);
        if (gap < best_gap) { best_gap = gap; best_b = b; best_S = S; }
    }
    for (int l = 0; l < L; ++l) {
        if (l == guard) { t_out[l] = guard_t; continue; }
        double tl = 0.0;
        for (int k = 0; k < K; ++k) {
            const int i = l * K + k;
            if (err[i] <= best_b && t[i] > tl) tl = t[i];
        }
        t_out[l] = tl;
    }
    *b_out = best_b;
    *S_out = best_S;
    free(budgets);
}
