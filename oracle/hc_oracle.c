/*
 * CPU oracle for the sparse contact operators of "ECO: Efficient Human-Contact
 * Representation for Human-Scene Interaction".
 *
 * TEST INFRASTRUCTURE ONLY. This file is the plain, slow reference that the
 * CUDA path is checked against. Only the tests, the smoke check and the
 * benchmark's CPU-baseline leg may load it; the product path never does.
 * It shares no code, header, table or helper with the CUDA library.
 *
 * Arithmetic: every sum is accumulated in fp64 in the order the definition
 * reads (spiral slot, then input channel). bf16 inputs are widened exactly;
 * outputs are rounded once, from fp64, to the storage type (fp32, or bf16
 * round-to-nearest-even). The fp64 value before that rounding is also
 * returned so tests can apply tolerances against it.
 *
 * Functions (each cites the passage it follows):
 *   hco_mask_compact        decomposition into (C', S') coordinates, Eq. 2,
 *                           plus the inverse map idx() of Eq. 4
 *   hco_conv_rulebook       the indexing matrix of Eq. 4 (tap -> input row)
 *   hco_sparse_spiral_conv  sparse convolution, Eqs. 4-5, with the spiral
 *                           neighbourhood of the POSA spiral blocks (Fig. 2)
 *                           and the activation of Eq. 10
 *   hco_dense_spiral_conv   the same layer on every vertex, no mask (the dense
 *                           operator the sparse one replaces, Sec. 3.2)
 *   hco_sparse_linear       linear layer on compact rows, Eq. 6
 *   hco_sparse_group_norm   group normalisation over each frame's active rows,
 *                           Eqs. 7-9 (G = 1: layer normalisation)
 *   hco_scatter_dense       inverse of the decomposition: compact rows back
 *                           into a dense [B, V, C] tensor
 *   hco_mask_score          the mask-score update of Eq. 3 (Gram matrices of
 *                           the per-mask outputs, Frobenius norms)
 *   hco_select_topk         the kappa masks with the highest score kept at
 *                           inference (Sec. 3.1, "Sparse Mask Selection")
 *   hco_kappa_masks         the kept masks applied to every sample: kappa
 *                           frames per sample (Eq. 1 per kept mask)
 *   hco_gather_rows         the feature matrix S' of Eq. 2: the input rows
 *                           at the active coordinates
 *   hco_sparse_conv_bwd     gradients of the sparse convolution (Eqs. 4-5,
 *                           6, 10) with respect to its input rows, weight
 *                           and bias, through the Eq. 4 indexing matrix
 *   hco_bf16_round          fp64 -> bf16 rounding (storage format)
 *
 * Parity status: compaction, conv, dense conv, linear, group norm, scatter,
 * the mask score, top-kappa selection, kappa masks and the row gather are
 * pinned by tests against library routines (numpy.nonzero, numpy matmul,
 * numpy argsort), closed forms, invariances, hand-worked cases and brute
 * force (tests/test_oracle_pins.py). The paper prints no numeric worked
 * example for any operator.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#define HCO_F32 0
#define HCO_BF16 1
#define HCO_ACT_NONE 0
#define HCO_ACT_ELU 1
#define HCO_ACT_RELU 2
#define HCO_LAYOUT_DENSE 0
#define HCO_LAYOUT_COMPACT 1

/* ---------------------------------------------------------------- dtypes */

/* bf16 is the upper half of an IEEE binary32 pattern: widening is exact. */
static double bf16_to_double(uint16_t h) {
    uint32_t u = (uint32_t)h << 16;
    float f;
    memcpy(&f, &u, sizeof f);
    return (double)f;
}

/* fp64 -> bf16, round to nearest, ties to even, from the format's
 * definition: bf16 has 8 significant bits for normal numbers (exponent
 * range of binary32) and a fixed quantum of 2^-133 below 2^-126. The value
 * is scaled by its quantum (exact: a power of two), rounded to an integer
 * with nearbyint (default mode: nearest-even), and scaled back; the result
 * is a bf16 number, so converting it to binary32 is exact and its upper
 * 16 bits are the answer. Overflow gives infinity; NaN stays NaN. */
uint16_t hco_bf16_round(double x) {
    float f;
    uint32_t u;
    if (isnan(x)) return (uint16_t)0x7FC0;
    if (x == 0.0 || isinf(x)) {
        f = (float)x;
        memcpy(&u, &f, sizeof u);
        return (uint16_t)(u >> 16);
    }
    int e;
    frexp(x, &e); /* |x| in [2^(e-1), 2^e) */
    int qexp = e - 8;       /* quantum for 8 significant bits */
    if (qexp < -133) qexp = -133; /* subnormal range: fixed quantum */
    double n = nearbyint(ldexp(x, -qexp));
    double r = ldexp(n, qexp);
    f = (float)r; /* exact, or +-inf past the largest bf16 */
    memcpy(&u, &f, sizeof u);
    return (uint16_t)(u >> 16);
}

static double load_elem(const void* p, int dtype, int64_t i) {
    if (dtype == HCO_F32) return (double)((const float*)p)[i];
    return bf16_to_double(((const uint16_t*)p)[i]);
}

static void store_elem(void* p, int dtype, int64_t i, double v) {
    if (dtype == HCO_F32)
        ((float*)p)[i] = (float)v;
    else
        ((uint16_t*)p)[i] = hco_bf16_round(v);
}

/* Activation of Eq. 10; ELU with alpha = 1. */
static double activate(double z, int act) {
    if (act == HCO_ACT_ELU) return z > 0.0 ? z : expm1(z);
    if (act == HCO_ACT_RELU) return z > 0.0 ? z : 0.0;
    return z;
}

/* ----------------------------------------------------------- compaction */

/* Eq. 2: drop the zero rows of the masked tensor. Row (b, v) is kept iff
 * mask[b, v] != 0; kept rows are listed in ascending (b, v) order as the
 * coordinate matrix C' (frame index b, vertex index v). row_of[b, v] is the
 * position of (b, v) in C' or -1: this is idx() of Eq. 4. offsets[b] counts
 * the kept rows of frames before b, so rows of frame b are
 * [offsets[b], offsets[b+1]) (the "i : C[i][0] = b" ranges of Eqs. 7-8).
 * Returns N', the number of kept rows. */
int64_t hco_mask_compact(const uint8_t* mask, int64_t B, int64_t V,
                         int32_t* coords, int32_t* row_of, int32_t* offsets) {
    int64_t n = 0;
    for (int64_t b = 0; b < B; ++b) {
        offsets[b] = (int32_t)n;
        for (int64_t v = 0; v < V; ++v) {
            if (mask[b * V + v] != 0) {
                coords[2 * n + 0] = (int32_t)b;
                coords[2 * n + 1] = (int32_t)v;
                row_of[b * V + v] = (int32_t)n;
                ++n;
            } else {
                row_of[b * V + v] = -1;
            }
        }
    }
    offsets[B] = (int32_t)n;
    return n;
}

/* ------------------------------------------------------------- mapping */

/* Eq. 4, materialised for the spiral neighbourhood: the indexing matrix that
 * pairs every kernel tap of an output coordinate with the input row it reads.
 * For output row n (coordinate (b, v) = C'[n]) and spiral slot l:
 *     rulebook[l*stride + n] = idx(b, spiral[v][l])   if that tap is present,
 *                            = -1                     otherwise,
 * where the tap is present iff spiral[v][l] >= 0 and (b, spiral[v][l]) is an
 * active row. idx() is the row of the input: b*V + u for a dense input, the
 * compact position row_of[b, u] for a compact one. */
void hco_conv_rulebook(const int32_t* coords, const int32_t* row_of, int64_t n_rows,
                       const int32_t* spiral, int64_t V, int L, int x_layout, int64_t stride,
                       int32_t* rulebook) {
    for (int64_t n = 0; n < n_rows; ++n) {
        int64_t b = coords[2 * n + 0], v = coords[2 * n + 1];
        for (int l = 0; l < L; ++l) {
            int64_t u = spiral[v * L + l];
            int32_t e = -1;
            if (u >= 0) {
                int64_t j = row_of[b * V + u];
                if (j >= 0) e = (int32_t)(x_layout == HCO_LAYOUT_DENSE ? b * V + u : j);
            }
            rulebook[(int64_t)l * stride + n] = e;
        }
    }
}

/* --------------------------------------------------- sparse spiral conv */

/* Eqs. 4-5 on the spiral neighbourhood. For the output row at coordinate
 * (b, v) = C'[r]:
 *     acc[o] = sum_{l < L} sum_{c < C_in} S[idx(b, spiral[v][l])][c] * W[l*C_in + c][o]
 * where a term is present only if spiral[v][l] >= 0 and the neighbour
 * (b, spiral[v][l]) is an active row (Eq. 4 keeps only kernel taps whose
 * coordinate is found in C). Slot 0 of the spiral is the vertex itself, the
 * centre tap of Eq. 4. Then y = act(acc + bias) (Eqs. 6 and 10), and the
 * output coordinate is the centre coordinate (Eq. 5, first line).
 *
 * x_layout DENSE: S row of (b, u) is x[(b*V + u)*C_in ...] (read only when
 * (b, u) is active); COMPACT: it is x[row_of[b*V + u]*C_in ...].
 * rows: the output rows to compute (indices into coords), or NULL for
 * 0..n_rows-1. Output i goes to y_pre[i*C_out ...] (fp64, before rounding)
 * and y[i*C_out ...] (storage dtype); either may be NULL. */
void hco_sparse_spiral_conv(const void* x, int x_layout, int dtype,
                            const int32_t* coords, const int32_t* row_of,
                            const int64_t* rows, int64_t n_rows,
                            const int32_t* spiral, int64_t B, int64_t V, int L,
                            int C_in, int C_out, const void* W, const float* bias,
                            int act, double* y_pre, void* y, int n_threads) {
    (void)B;
#pragma omp parallel for schedule(dynamic, 8) num_threads(n_threads > 0 ? n_threads : 1)
    for (int64_t i = 0; i < n_rows; ++i) {
        int64_t r = rows ? rows[i] : i;
        int64_t b = coords[2 * r + 0];
        int64_t v = coords[2 * r + 1];
        double* acc = (double*)calloc((size_t)C_out, sizeof(double));
        for (int l = 0; l < L; ++l) {
            int64_t u = spiral[v * L + l];
            if (u < 0) continue; /* no neighbour in this slot */
            int64_t j = row_of[b * V + u];
            if (j < 0) continue; /* neighbour not in C: tap absent */
            int64_t src = (x_layout == HCO_LAYOUT_DENSE) ? (b * V + u) : j;
            for (int c = 0; c < C_in; ++c) {
                double xv = load_elem(x, dtype, src * C_in + c);
                for (int o = 0; o < C_out; ++o)
                    acc[o] += xv * load_elem(W, dtype, ((int64_t)l * C_in + c) * C_out + o);
            }
        }
        for (int o = 0; o < C_out; ++o) {
            double z = acc[o] + (bias ? (double)bias[o] : 0.0);
            double a = activate(z, act);
            if (y_pre) y_pre[i * C_out + o] = a;
            if (y) store_elem(y, dtype, i * C_out + o, a);
        }
        free(acc);
    }
}

/* ---------------------------------------------------- dense spiral conv */

/* The dense layer the sparse one replaces: every (b, v) of the [B, V] grid
 * is an output row (row index r = b*V + v), every neighbour slot with
 * spiral[v][l] >= 0 contributes, no mask is consulted.
 *     acc[o] = sum_{l < L} sum_{c < C_in} x[b, spiral[v][l], c] * W[l*C_in + c][o]
 * Written as its own loop so that "sparse == dense on the masked input"
 * compares two independent codings of the definition. */
void hco_dense_spiral_conv(const void* x, int dtype, const int64_t* rows, int64_t n_rows,
                           const int32_t* spiral, int64_t B, int64_t V, int L, int C_in,
                           int C_out, const void* W, const float* bias, int act,
                           double* y_pre, void* y, int n_threads) {
    (void)B;
#pragma omp parallel for schedule(dynamic, 8) num_threads(n_threads > 0 ? n_threads : 1)
    for (int64_t i = 0; i < n_rows; ++i) {
        int64_t r = rows ? rows[i] : i;
        int64_t b = r / V, v = r % V;
        double* acc = (double*)calloc((size_t)C_out, sizeof(double));
        for (int l = 0; l < L; ++l) {
            int64_t u = spiral[v * L + l];
            if (u < 0) continue;
            for (int c = 0; c < C_in; ++c) {
                double xv = load_elem(x, dtype, (b * V + u) * C_in + c);
                for (int o = 0; o < C_out; ++o)
                    acc[o] += xv * load_elem(W, dtype, ((int64_t)l * C_in + c) * C_out + o);
            }
        }
        for (int o = 0; o < C_out; ++o) {
            double a = activate(acc[o] + (bias ? (double)bias[o] : 0.0), act);
            if (y_pre) y_pre[i * C_out + o] = a;
            if (y) store_elem(y, dtype, i * C_out + o, a);
        }
        free(acc);
    }
}

/* -------------------------------------------------------- sparse linear */

/* Eq. 6, row-wise: y_i = act(s_i^T W_l + b) for every compact row i; the
 * coordinates are unchanged. W_l is [C_in, C_out] row-major. */
void hco_sparse_linear(const void* x, int dtype, const int64_t* rows, int64_t n_rows,
                       int C_in, int C_out, const void* W, const float* bias, int act,
                       double* y_pre, void* y, int n_threads) {
#pragma omp parallel for schedule(dynamic, 8) num_threads(n_threads > 0 ? n_threads : 1)
    for (int64_t i = 0; i < n_rows; ++i) {
        int64_t r = rows ? rows[i] : i;
        for (int o = 0; o < C_out; ++o) {
            double acc = 0.0;
            for (int c = 0; c < C_in; ++c)
                acc += load_elem(x, dtype, r * C_in + c) * load_elem(W, dtype, (int64_t)c * C_out + o);
            double a = activate(acc + (bias ? (double)bias[o] : 0.0), act);
            if (y_pre) y_pre[i * C_out + o] = a;
            if (y) store_elem(y, dtype, i * C_out + o, a);
        }
    }
}

/* ---------------------------------------------------------- group norm */

/* Eqs. 7-9: group normalisation over the active rows of each frame. Frame b
 * owns the compact rows [offsets[b], offsets[b+1]) (the rows i with
 * C'[i][0] = b); the C channels split into G groups of C/G consecutive
 * channels. For every (b, g), with n = (rows of frame b) * (C/G) values:
 *     mu     = (1/n) * sum of the group's values over the frame's rows   (Eq. 7)
 *     sigma2 = (1/n) * sum of (value - mu)^2                             (Eq. 8)
 *     out    = (value - mu) / sqrt(sigma2 + eps)                         (Eq. 9)
 * then, per channel, out * gamma[c] + beta[c] when gamma/beta are given, and
 * the activation of Eq. 10. Two passes in fp64. Frames without active rows
 * produce nothing. */
void hco_sparse_group_norm(const void* x, int dtype, const int32_t* offsets, int64_t B, int C,
                           int G, double eps, const float* gamma, const float* beta, int act,
                           double* y_pre, void* y) {
    int cpg = C / G;
    for (int64_t b = 0; b < B; ++b) {
        int64_t r0 = offsets[b], r1 = offsets[b + 1];
        if (r1 <= r0) continue;
        for (int g = 0; g < G; ++g) {
            double n = (double)(r1 - r0) * cpg;
            double sum = 0.0;
            for (int64_t i = r0; i < r1; ++i)
                for (int c = g * cpg; c < (g + 1) * cpg; ++c) sum += load_elem(x, dtype, i * C + c);
            double mu = sum / n;
            double ss = 0.0;
            for (int64_t i = r0; i < r1; ++i)
                for (int c = g * cpg; c < (g + 1) * cpg; ++c) {
                    double d = load_elem(x, dtype, i * C + c) - mu;
                    ss += d * d;
                }
            double inv = 1.0 / sqrt(ss / n + eps);
            for (int64_t i = r0; i < r1; ++i)
                for (int c = g * cpg; c < (g + 1) * cpg; ++c) {
                    double v = (load_elem(x, dtype, i * C + c) - mu) * inv;
                    if (gamma) v *= (double)gamma[c];
                    if (beta) v += (double)beta[c];
                    v = activate(v, act);
                    if (y_pre) y_pre[i * C + c] = v;
                    if (y) store_elem(y, dtype, i * C + c, v);
                }
        }
    }
}

/* ------------------------------------------------------------- scatter */

/* Inverse of the decomposition (Eq. 2): compact row n goes back to dense
 * position coords[n] = (b, v). With zero_fill, every dense row first
 * becomes zero, so inactive rows read 0 (the masked tensor of Eq. 1);
 * without it they are left as they were. Elements are copied bit for bit. */
void hco_scatter_dense(const void* y, int elem_bytes, const int32_t* coords, int64_t count,
                       int64_t B, int64_t V, int C, int zero_fill, void* out) {
    const unsigned char* src = (const unsigned char*)y;
    unsigned char* dst = (unsigned char*)out;
    int64_t row_bytes = (int64_t)C * elem_bytes;
    if (zero_fill) memset(dst, 0, (size_t)(B * V * row_bytes));
    for (int64_t n = 0; n < count; ++n) {
        int64_t b = coords[2 * n + 0], v = coords[2 * n + 1];
        memcpy(dst + (b * V + v) * row_bytes, src + n * row_bytes, (size_t)row_bytes);
    }
}

/* ---------------------------------------------------------- mask score */

/* Eq. 3: with O_k the [N, D] output for mask k (row-major, masks stacked
 * as [K, N, D]), and ||.||_F the Frobenius norm,
 *     S[i][k]   = || O_i^T O_k ||_F^2            (D x D Gram of the pair)
 *     sim[i][k] = S[i][k] / (|| O_k^T O_k ||_F || O_i^T O_i ||_F)
 *               = S[i][k] / sqrt(S[i][i] * S[k][k])
 *     alpha_out[k] = alpha_in[k] + 1/(K-1) * sum over i != k of (1 - sim[i][k])
 * Every Gram entry is a plain fp64 sum over the N rows, squared and summed
 * over the D x D entries. Readings where the equation is silent: a mask
 * whose output is all zero has no defined similarity, and its terms count
 * as 1 - 0 (it shares nothing); with K = 1 the sum is empty and alpha is
 * unchanged. S and sim are [K, K] (either may be NULL). */
void hco_mask_score(const void* O, int dtype, int64_t K, int64_t N, int64_t D,
                    const double* alpha_in, double* alpha_out, double* sim_out, double* S_out,
                    int n_threads) {
    double* S = (double*)calloc((size_t)(K * K), sizeof(double));
    int64_t n_pairs = K * (K + 1) / 2;
    #pragma omp parallel for schedule(dynamic) num_threads(n_threads)
    for (int64_t p = 0; p < n_pairs; ++p) {
        /* pair p -> (i, k), i <= k */
        int64_t i = 0, rem = p;
        while (rem >= K - i) {
            rem -= K - i;
            ++i;
        }
        int64_t k = i + rem;
        double acc = 0.0;
        for (int64_t d = 0; d < D; ++d)
            for (int64_t e = 0; e < D; ++e) {
                double g = 0.0;
                for (int64_t n = 0; n < N; ++n)
                    g += load_elem(O, dtype, (i * N + n) * D + d) *
                         load_elem(O, dtype, (k * N + n) * D + e);
                acc += g * g;
            }
        S[i * K + k] = acc;
        S[k * K + i] = acc;
    }
    for (int64_t k = 0; k < K; ++k) {
        double sum = 0.0;
        for (int64_t i = 0; i < K; ++i) {
            double den = sqrt(S[i * K + i]) * sqrt(S[k * K + k]);
            double sim = den > 0.0 ? S[i * K + k] / den : 0.0;
            if (sim_out) sim_out[i * K + k] = sim;
            if (i != k) sum += 1.0 - sim;
        }
        alpha_out[k] = K > 1 ? alpha_in[k] + sum / (double)(K - 1) : alpha_in[k];
    }
    if (S_out) memcpy(S_out, S, sizeof(double) * (size_t)(K * K));
    free(S);
}

/* Sec. 3.1, Sparse Mask Selection: at inference only the kappa masks with
 * the highest score are kept. Selected in order of decreasing score; equal
 * scores are taken lowest index first. The scores are fp32 (as stored). The
 * paper does not consider undefined scores: a NaN ranks below every number
 * (NaNs among themselves by index). */
static int score_above(float a, float b) {
    if (isnan(a)) return 0;
    return isnan(b) || a > b;
}

void hco_select_topk(const float* alpha, int64_t K, int64_t kappa, int32_t* selected) {
    unsigned char* taken = (unsigned char*)calloc((size_t)K, 1);
    for (int64_t j = 0; j < kappa; ++j) {
        int64_t best = -1;
        for (int64_t k = 0; k < K; ++k) {
            if (taken[k]) continue;
            if (best < 0 || score_above(alpha[k], alpha[best])) best = k;
        }
        taken[best] = 1;
        selected[j] = (int32_t)best;
    }
    free(taken);
}

/* Eq. 1 with every kept mask applied to every sample independently
 * (Sec. 3.1): frame f = b * kappa + j is sample b under kept mask
 * selected[j], so out[f][v] = masks[selected[j]][v]. masks is [K, V]. */
void hco_kappa_masks(const uint8_t* masks, int64_t V, const int32_t* selected, int64_t kappa,
                     int64_t B, uint8_t* out) {
    for (int64_t b = 0; b < B; ++b)
        for (int64_t j = 0; j < kappa; ++j)
            memcpy(out + (b * kappa + j) * V, masks + (int64_t)selected[j] * V, (size_t)V);
}

/* Eq. 2, the feature matrix S': row n holds the input features at the n-th
 * active coordinate (f, v). The input is the dense [B_in, V, C] tensor of
 * samples; frame f reads sample f / frames_per_sample (frames_per_sample =
 * kappa when every sample was masked by kappa kept masks, else 1). Rows are
 * copied bit for bit. */
void hco_gather_rows(const void* x, int elem_bytes, int64_t V, int C, const int32_t* coords,
                     int64_t count, int64_t frames_per_sample, void* y) {
    const unsigned char* src = (const unsigned char*)x;
    unsigned char* dst = (unsigned char*)y;
    int64_t row_bytes = (int64_t)C * elem_bytes;
    for (int64_t n = 0; n < count; ++n) {
        int64_t f = coords[2 * n + 0], v = coords[2 * n + 1];
        memcpy(dst + n * row_bytes, src + ((f / frames_per_sample) * V + v) * row_bytes,
               (size_t)row_bytes);
    }
}

/* ------------------------------------------------------ sparse conv bwd */

/* Gradients of the sparse spiral convolution (the paper gives the forward
 * only; these follow from it by the chain rule). With the indexing matrix
 * of Eq. 4, rulebook[l*stride + n] = the input row j read by tap l of
 * output row n (or -1), the forward is
 *     z[n][o] = bias[o] + sum_l sum_c x[j(n,l)][c] * W[l*C_in + c][o],
 *     y = act(z)                                                (Eq. 10)
 * and, for an upstream gradient dy = dL/dy over the n_rows output rows,
 *     dz[n][o]   = dy[n][o] * act'(z[n][o])
 *     dbias[o]   = sum_n dz[n][o]
 *     dW[l*C_in + c][o] = sum_n x[j(n,l)][c] * dz[n][o]   (present taps only)
 *     dx[j][c]   = sum over (n, l) with j(n,l) = j of sum_o dz[n][o] * W[l*C_in + c][o]
 * act' is read off the stored output y: ELU (alpha = 1) has derivative 1
 * for z > 0 and e^z = y + 1 otherwise; ReLU 1 for z > 0 else 0; none 1.
 * dx ([x_rows, C_in]), dW ([L*C_in, C_out]) and dbias ([C_out]) are fp64
 * and overwritten (rows of dx no tap reads are 0); any may be NULL. */
static double act_grad_from_output(double y, int act) {
    if (act == HCO_ACT_ELU) return y > 0.0 ? 1.0 : y + 1.0;
    if (act == HCO_ACT_RELU) return y > 0.0 ? 1.0 : 0.0;
    return 1.0;
}

void hco_sparse_conv_bwd(const void* x, int dtype, int64_t x_rows, const int32_t* rulebook,
                         int64_t n_rows, int64_t stride, int L, int C_in, int C_out, const void* W,
                         const void* y, const void* dy, int act, double* dx, double* dW,
                         double* dbias) {
    if (dx) memset(dx, 0, sizeof(double) * (size_t)(x_rows * C_in));
    if (dW) memset(dW, 0, sizeof(double) * (size_t)((int64_t)L * C_in * C_out));
    if (dbias) memset(dbias, 0, sizeof(double) * (size_t)C_out);
    double* dz = (double*)malloc(sizeof(double) * (size_t)C_out);
    for (int64_t n = 0; n < n_rows; ++n) {
        for (int o = 0; o < C_out; ++o)
            dz[o] = load_elem(dy, dtype, n * C_out + o) *
                    act_grad_from_output(load_elem(y, dtype, n * C_out + o), act);
        if (dbias)
            for (int o = 0; o < C_out; ++o) dbias[o] += dz[o];
        for (int l = 0; l < L; ++l) {
            int64_t j = rulebook[(int64_t)l * stride + n];
            if (j < 0) continue; /* absent tap: no term, no gradient */
            for (int c = 0; c < C_in; ++c) {
                int64_t k = (int64_t)l * C_in + c;
                if (dW) {
                    double xv = load_elem(x, dtype, j * C_in + c);
                    for (int o = 0; o < C_out; ++o) dW[k * C_out + o] += xv * dz[o];
                }
                if (dx) {
                    double g = 0.0;
                    for (int o = 0; o < C_out; ++o) g += dz[o] * load_elem(W, dtype, k * C_out + o);
                    dx[j * C_in + c] += g;
                }
            }
        }
    }
    free(dz);
}
