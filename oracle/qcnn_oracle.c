/*
 * qcnn_oracle.c -- float64 CPU oracle for the test-phase response of
 * product-quantized (PQ) fully-connected and convolutional layers
 * (Wu et al., "Quantized Convolutional Neural Networks for Mobile Devices",
 * arXiv 1512.06473).
 *
 * TEST INFRASTRUCTURE ONLY.  Only the test suite, the smoke check and the
 * CPU-baseline leg of the benchmark may load this code.  It shares nothing
 * with the CUDA library: no headers, no tables, no helpers.  It is written
 * to be read against the paper, not to be fast: every loop below is one
 * symbol of an equation, in the paper's order.
 *
 * Notation (Sec. 2, Sec. 3.1, Sec. 3.2):
 *   S        layer input; FC: a C_s vector, conv: C_s maps of H x W
 *   C'_s     sub-space dimension (Csp); M = C_s / C'_s sub-spaces
 *   D^(m)    sub-codebook m: K sub-codewords of C'_s values,
 *            stored D[m][k][j]  (the k-th column of D^(m) in the paper)
 *   k_m(c_t) / k_m(c_t, p_k)   index of the sub-codeword that quantizes
 *            the m-th sub-vector of weight vector c_t (at kernel offset p_k)
 *            FC codes stored codes[m][c_t]; conv codes stored
 *            codes[c_t][p_k][m] with p_k = ky * kw + kx.
 *
 * Readings where the paper is silent (each is also listed in the design
 * notes of the repository):
 *   - sub-space m holds the contiguous channels [m*C'_s, (m+1)*C'_s);
 *   - convolution is cross-correlation, p_s = p_t * stride - pad + p_k,
 *     with zero padding (a padded position contributes nothing);
 *   - a bias, absent from Eq. 1-7, is added after the sum when given;
 *   - an optional ReLU is applied last.
 *
 * All arithmetic is IEEE double; build with -ffp-contract=off so that the
 * result does not depend on whether the host fuses multiply-adds.
 *
 * Reduced-precision tables: with lut_bf16 = 1 every table entry is rounded
 * to bfloat16 (8 significant bits, round to nearest, ties to even) before
 * it is summed; the sums stay exact in double.  The paper builds its tables
 * in full precision; this models the reduced-precision table variant of
 * the library.  The entry is rounded from its exact value.
 *
 * Every function returns 0 on success and a negative value on an invalid
 * argument (non-positive size, C_s not a multiple of C'_s, K outside
 * [1, 256], a code >= K) or an allocation failure.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>

#define QO_OK 0
#define QO_EINVAL (-1)
#define QO_ENOMEM (-2)
#define QO_ECODE (-3)

typedef long long i64;

/*
 * Round v to the nearest bfloat16 value, ties to even.  bfloat16 keeps the
 * 8-bit exponent of binary32 and 8 significant bits (7 stored): write
 * v = f * 2^e with 0.5 <= |f| < 1, scale f to an integer significand
 * f * 2^8 in [128, 256), round that to an integer (nearbyint rounds to
 * nearest, ties to even, in the default rounding mode) and scale back.
 * Values below the binary32 normal range are not handled (the tests keep
 * far from them).
 */
double qo_round_bf16(double v)
{
    if (v == 0.0 || !isfinite(v)) return v;
    int e;
    const double f = frexp(v, &e);
    return ldexp(nearbyint(ldexp(f, 8)), e - 8);
}

/* ------------------------------------------------------------------ */
/* Look-up table of one input vector (Sec. 3.1, the paragraph after    */
/* Eq. 5): for every sub-space m and every sub-codeword k,             */
/*     LUT[m][k] = < S^(m), D^(m)_k > = sum_j S[m*C'_s + j] * D[m][k][j] */
/* ------------------------------------------------------------------ */
static void lut_of_vector(const double *s, i64 s_stride, int M, int Csp,
                          int K, const double *D, int lut_bf16,
                          double *lut /* [M][K] */)
{
    for (int m = 0; m < M; ++m) {
        for (int k = 0; k < K; ++k) {
            const double *dk = D + ((i64)m * K + k) * Csp;
            double acc = 0.0;
            for (int j = 0; j < Csp; ++j)
                acc += s[(i64)(m * Csp + j) * s_stride] * dk[j];
            lut[(i64)m * K + k] = lut_bf16 ? qo_round_bf16(acc) : acc;
        }
    }
}

static int check_pq(int Cs, int Csp, int K)
{
    if (Cs <= 0 || Csp <= 0 || K < 1 || K > 256) return QO_EINVAL;
    if (Cs % Csp != 0) return QO_EINVAL;
    return QO_OK;
}

static int check_codes(const uint8_t *codes, i64 n, int K)
{
    for (i64 i = 0; i < n; ++i)
        if ((int)codes[i] >= K) return QO_ECODE;
    return QO_OK;
}

/*
 * FC look-up tables for a batch:  lut[n][m][k] = < x_n^(m), D^(m)_k >.
 * x: [N][Cs]; D: [M][K][Csp]; lut: [N][M][K].
 */
int qo_fc_lut(const double *x, int N, int Cs, const double *D, int Csp, int K,
              int lut_bf16, double *lut)
{
    int rc = check_pq(Cs, Csp, K);
    if (rc || N <= 0) return QO_EINVAL;
    const int M = Cs / Csp;
    for (int n = 0; n < N; ++n)
        lut_of_vector(x + (i64)n * Cs, 1, M, Csp, K, D, lut_bf16,
                      lut + (i64)n * M * K);
    return QO_OK;
}

/*
 * FC layer response, Eq. 5:
 *     T(c_t) ~= sum_m < D^(m)_{k_m(c_t)}, S^(m) > = sum_m LUT[m][k_m(c_t)]
 * computed by first filling the table and then doing M additions per
 * output, as the text after Eq. 5 describes.
 * x: [N][Cs]; codes: [M][Ct]; bias: [Ct] or NULL; y: [N][Ct].
 */
int qo_fc_forward(const double *x, int N, int Cs, int Ct, const double *D,
                  int Csp, int K, const uint8_t *codes, const double *bias,
                  int relu, int lut_bf16, double *y)
{
    int rc = check_pq(Cs, Csp, K);
    if (rc || N <= 0 || Ct <= 0) return QO_EINVAL;
    const int M = Cs / Csp;
    if (check_codes(codes, (i64)M * Ct, K)) return QO_ECODE;
    double *lut = (double *)malloc(sizeof(double) * (size_t)M * K);
    if (!lut) return QO_ENOMEM;
    for (int n = 0; n < N; ++n) {
        lut_of_vector(x + (i64)n * Cs, 1, M, Csp, K, D, lut_bf16, lut);
        for (int ct = 0; ct < Ct; ++ct) {
            double t = 0.0;
            for (int m = 0; m < M; ++m)
                t += lut[(i64)m * K + codes[(i64)m * Ct + ct]];
            if (bias) t += bias[ct];
            if (relu && t < 0.0) t = 0.0;
            y[(i64)n * Ct + ct] = t;
        }
    }
    free(lut);
    return QO_OK;
}

/*
 * Conv look-up tables (Sec. 3.2, the paragraph after Eq. 7): one table per
 * input position p_s = (iy, ix):
 *     lut[n][m][iy*W + ix][k] = < S_{n,p_s}^(m), D^(m)_k >
 * x: [N][Cs][H][W] (NCHW); lut: [N][M][H*W][K].
 */
int qo_conv_lut(const double *x, int N, int Cs, int H, int W, const double *D,
                int Csp, int K, int lut_bf16, double *lut)
{
    int rc = check_pq(Cs, Csp, K);
    if (rc || N <= 0 || H <= 0 || W <= 0) return QO_EINVAL;
    const int M = Cs / Csp;
    const i64 P = (i64)H * W;
    double *row = (double *)malloc(sizeof(double) * (size_t)M * K);
    if (!row) return QO_ENOMEM;
    for (int n = 0; n < N; ++n) {
        const double *xn = x + (i64)n * Cs * P;
        for (i64 p = 0; p < P; ++p) {
            lut_of_vector(xn + p, P, M, Csp, K, D, lut_bf16, row);
            for (int m = 0; m < M; ++m)
                for (int k = 0; k < K; ++k)
                    lut[(((i64)n * M + m) * P + p) * K + k] = row[(i64)m * K + k];
        }
    }
    free(row);
    return QO_OK;
}

/*
 * Conv layer response, Eq. 7:
 *     T_{p_t}(c_t) ~= sum_{(p_k, p_s)} sum_m LUT_{p_s}[m][k_m(c_t, p_k)]
 * where (p_k, p_s) runs over the receptive field of p_t:
 *     iy = oy*stride - pad + ky,  ix = ox*stride - pad + kx,
 * and a (p_k, p_s) pair whose p_s falls outside the map contributes 0
 * (zero padding).  Output size Ho = floor((H + 2 pad - kh) / stride) + 1.
 * x: [N][Cs][H][W]; codes: [Ct][kh*kw][M]; bias: [Ct] or NULL;
 * y: [N][Ct][Ho][Wo].
 */
int qo_conv_forward(const double *x, int N, int Cs, int H, int W, int Ct,
                    int kh, int kw, int stride, int pad, const double *D,
                    int Csp, int K, const uint8_t *codes, const double *bias,
                    int relu, int lut_bf16, double *y)
{
    int rc = check_pq(Cs, Csp, K);
    if (rc || N <= 0 || H <= 0 || W <= 0 || Ct <= 0 || kh <= 0 || kw <= 0 ||
        stride <= 0 || pad < 0)
        return QO_EINVAL;
    const int M = Cs / Csp;
    const int Ho = (H + 2 * pad - kh) / stride + 1;
    const int Wo = (W + 2 * pad - kw) / stride + 1;
    if (H + 2 * pad < kh || W + 2 * pad < kw || Ho <= 0 || Wo <= 0)
        return QO_EINVAL;
    const int KK = kh * kw;
    if (check_codes(codes, (i64)Ct * KK * M, K)) return QO_ECODE;
    const i64 P = (i64)H * W;
    /* lut[m][p][k] for one image */
    double *lut = (double *)malloc(sizeof(double) * (size_t)M * P * K);
    if (!lut) return QO_ENOMEM;
    for (int n = 0; n < N; ++n) {
        rc = qo_conv_lut(x + (i64)n * Cs * P, 1, Cs, H, W, D, Csp, K, lut_bf16,
                         lut);
        if (rc) { free(lut); return rc; }
        for (int ct = 0; ct < Ct; ++ct) {
            for (int oy = 0; oy < Ho; ++oy) {
                for (int ox = 0; ox < Wo; ++ox) {
                    double t = 0.0;
                    for (int ky = 0; ky < kh; ++ky) {
                        const int iy = oy * stride - pad + ky;
                        if (iy < 0 || iy >= H) continue;
                        for (int kx = 0; kx < kw; ++kx) {
                            const int ix = ox * stride - pad + kx;
                            if (ix < 0 || ix >= W) continue;
                            const int pk = ky * kw + kx;
                            const i64 ps = (i64)iy * W + ix;
                            for (int m = 0; m < M; ++m) {
                                const int k = codes[((i64)ct * KK + pk) * M + m];
                                t += lut[((i64)m * P + ps) * K + k];
                            }
                        }
                    }
                    if (bias) t += bias[ct];
                    if (relu && t < 0.0) t = 0.0;
                    y[(((i64)n * Ct + ct) * Ho + oy) * Wo + ox] = t;
                }
            }
        }
    }
    free(lut);
    return QO_OK;
}

/*
 * Max-pooling used between the layers of the whole-network experiments
 * (Sec. 4.2.3, AlexNet-style k x k window, stride s, no padding, floor
 * output size).  x: [N][C][H][W]; y: [N][C][Ho][Wo].
 */
int qo_maxpool(const double *x, int N, int C, int H, int W, int k, int s,
               double *y)
{
    if (N <= 0 || C <= 0 || H < k || W < k || k <= 0 || s <= 0) return QO_EINVAL;
    const int Ho = (H - k) / s + 1;
    const int Wo = (W - k) / s + 1;
    for (i64 nc = 0; nc < (i64)N * C; ++nc) {
        const double *xp = x + nc * H * W;
        for (int oy = 0; oy < Ho; ++oy)
            for (int ox = 0; ox < Wo; ++ox) {
                double v = xp[(i64)(oy * s) * W + ox * s];
                for (int dy = 0; dy < k; ++dy)
                    for (int dx = 0; dx < k; ++dx) {
                        const double u = xp[(i64)(oy * s + dy) * W + ox * s + dx];
                        if (u > v) v = u;
                    }
                y[(nc * Ho + oy) * Wo + ox] = v;
            }
    }
    return QO_OK;
}

/* ------------------------------------------------------------------ */
/* Quantizer: k-means in every sub-space (Sec. 3.1, Eq. 4; Sec. 3.2,   */
/* Eq. 6).  For sub-space m, the points are the m-th sub-vectors of    */
/* all weight vectors (FC: one per c_t; conv: one per (c_t, p_k)); the */
/* K centroids become D^(m) and the index of each point's centroid its */
/* code, minimising sum ||D^(m) B^(m) - W^(m)||_F^2 (Lloyd's           */
/* algorithm: alternate the assignment and the centroid update).       */
/*                                                                     */
/* Readings (the paper only says "k-means clustering"):                */
/*   - the initial centroids are an input (the caller's seeded draw);  */
/*   - `iters` rounds of (assign, update), then a final assignment     */
/*     against the final centroids gives the codes;                    */
/*   - squared distances are evaluated in binary32, term by term in    */
/*     j order: d = sum_j (x_j - c_j)^2 with each subtraction,         */
/*     product and sum rounded to binary32, because the assignment is  */
/*     an integer decided by floating point and the GPU kernels decide */
/*     it in that precision; ties go to the smallest index;            */
/*   - a centroid is the mean of its points: the sum in double over    */
/*     the points in index order, divided by the count, rounded to     */
/*     binary32; a centroid with no points keeps its value.            */
/* ------------------------------------------------------------------ */
static int kmeans_assign(const float *pts, i64 P, int d, int K, const float *cen,
                         uint8_t *assign)
{
    for (i64 p = 0; p < P; ++p) {
        const float *x = pts + p * d;
        int best = 0;
        float best_d = 0.0f;
        for (int k = 0; k < K; ++k) {
            const float *c = cen + (i64)k * d;
            float dist = 0.0f;
            for (int j = 0; j < d; ++j) {
                const float diff = x[j] - c[j];
                const float sq = diff * diff;
                dist = dist + sq;
            }
            if (k == 0 || dist < best_d) {
                best = k;
                best_d = dist;
            }
        }
        assign[p] = (uint8_t)best;
    }
    return QO_OK;
}

static int kmeans_update(const float *pts, i64 P, int d, int K, const uint8_t *assign,
                         float *cen)
{
    double *sum = (double *)calloc((size_t)K * d, sizeof(double));
    i64 *cnt = (i64 *)calloc((size_t)K, sizeof(i64));
    if (!sum || !cnt) { free(sum); free(cnt); return QO_ENOMEM; }
    for (i64 p = 0; p < P; ++p) {
        const int k = assign[p];
        cnt[k] += 1;
        for (int j = 0; j < d; ++j) sum[(i64)k * d + j] += (double)pts[p * d + j];
    }
    for (int k = 0; k < K; ++k)
        if (cnt[k] > 0)
            for (int j = 0; j < d; ++j)
                cen[(i64)k * d + j] = (float)(sum[(i64)k * d + j] / (double)cnt[k]);
    free(sum);
    free(cnt);
    return QO_OK;
}

/*
 * k-means on the points of one sub-space.
 * pts: [P][d] binary32; init: [K][d]; cen (out): [K][d]; assign (out): [P].
 */
int qo_kmeans(const float *pts, i64 P, int d, int K, const float *init, int iters,
              float *cen, uint8_t *assign)
{
    if (P <= 0 || d <= 0 || K < 1 || K > 256 || iters < 0) return QO_EINVAL;
    for (i64 e = 0; e < (i64)K * d; ++e) cen[e] = init[e];
    for (int it = 0; it < iters; ++it) {
        kmeans_assign(pts, P, d, K, cen, assign);
        int rc = kmeans_update(pts, P, d, K, assign, cen);
        if (rc) return rc;
    }
    return kmeans_assign(pts, P, d, K, cen, assign);
}

/*
 * PQ quantization of an FC weight matrix (Eq. 4).  The paper's W is
 * C_s x C_t with weight vectors as columns; here W is stored [Ct][Cs]
 * (one weight vector per row).  init: [M][K][Csp].
 * D (out): [M][K][Csp]; codes (out): [M][Ct].
 */
int qo_pq_quantize_fc(const float *W, int Ct, int Cs, int Csp, int K, const float *init,
                      int iters, float *D, uint8_t *codes)
{
    if (check_pq(Cs, Csp, K) || Ct <= 0) return QO_EINVAL;
    const int M = Cs / Csp;
    float *pts = (float *)malloc(sizeof(float) * (size_t)Ct * Csp);
    if (!pts) return QO_ENOMEM;
    int rc = QO_OK;
    for (int m = 0; m < M && rc == QO_OK; ++m) {
        for (int ct = 0; ct < Ct; ++ct)
            for (int j = 0; j < Csp; ++j)
                pts[(i64)ct * Csp + j] = W[(i64)ct * Cs + m * Csp + j];
        rc = qo_kmeans(pts, Ct, Csp, K, init + (i64)m * K * Csp, iters,
                       D + (i64)m * K * Csp, codes + (i64)m * Ct);
    }
    free(pts);
    return rc;
}

/*
 * PQ quantization of conv kernels (Eq. 6): sub-space m pools the m-th
 * sub-vectors of every kernel at every offset, point index
 * p = c_t * (kh*kw) + p_k.  W: [Ct][Cs][kh][kw]; init: [M][K][Csp].
 * D (out): [M][K][Csp]; codes (out): [Ct][kh*kw][M].
 */
int qo_pq_quantize_conv(const float *W, int Ct, int Cs, int kh, int kw, int Csp, int K,
                        const float *init, int iters, float *D, uint8_t *codes)
{
    if (check_pq(Cs, Csp, K) || Ct <= 0 || kh <= 0 || kw <= 0) return QO_EINVAL;
    const int M = Cs / Csp, KK = kh * kw;
    const i64 P = (i64)Ct * KK;
    float *pts = (float *)malloc(sizeof(float) * (size_t)P * Csp);
    uint8_t *a = (uint8_t *)malloc((size_t)P);
    if (!pts || !a) { free(pts); free(a); return QO_ENOMEM; }
    int rc = QO_OK;
    for (int m = 0; m < M && rc == QO_OK; ++m) {
        for (int ct = 0; ct < Ct; ++ct)
            for (int pk = 0; pk < KK; ++pk)
                for (int j = 0; j < Csp; ++j)
                    pts[((i64)ct * KK + pk) * Csp + j] =
                        W[((i64)ct * Cs + m * Csp + j) * KK + pk];
        rc = qo_kmeans(pts, P, Csp, K, init + (i64)m * K * Csp, iters,
                       D + (i64)m * K * Csp, a);
        for (i64 p = 0; p < P; ++p) codes[p * M + m] = a[p];
    }
    free(pts);
    free(a);
    return rc;
}
