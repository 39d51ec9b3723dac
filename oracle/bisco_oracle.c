/*
 * bisco_oracle.c -- plain, slow, fp64 CPU oracle for the BiSCo-LLM inference
 * hot path (binary spherical coding of LLM weights, arxiv 2607.08643).
 *
 * TEST INFRASTRUCTURE ONLY.  Nothing in the product path may link, load or
 * call this file: only the tests, the smoke check and the benchmark's CPU
 * baseline leg use it.  It shares no code, header or constant with the CUDA
 * library; the two agree only through the paper and the storage format.
 *
 * What it computes (all arithmetic in IEEE binary64, no FMA contraction --
 * build with -ffp-contract=off -- and no reordering of sums):
 *
 *   encode   Sec. III-E Eq. 8 (protected input channels, TopK of g_j*||W_:,j||_2),
 *            Sec. III-E Eq. 10 (8-bit quantiser on the protected slices),
 *            Sec. III-C Eq. 3 (unit-sphere normalisation and sign binarisation,
 *            q = sign(u)/sqrt(b)) with the identity encoder (b = d) and the
 *            decoder read as "rescale the unit code by the chunk's stored
 *            fp16 L2 norm", and Sec. III-D Eq. 5-7 (residual stages
 *            r(s) = r(s-1) - rhat(s)).
 *   decode   Sec. III-G Eq. 12 (stages decoded independently and summed)
 *            with the Eq. 10 scatter of the protected columns.
 *   matmul   y[b][i] = sum_j What[i][j] * x[b][j]  (plain definition).
 *   rows     output-row protection and the coupled MLP channel score of
 *            Sec. III-E Eq. 9 (gate/up rows and down columns share one
 *            protected set), with Eq. 10's 8-bit quantiser on the rows.
 *   fp8      the FP8 (E4M3, E5M2) and BF16 protected-payload formats of the
 *            paper's protected-format ablation, as variants of Eq. 10's
 *            quantiser.
 *   decoder  the decoder step of Eq. 1 as per-stage tables over the 256
 *            code bytes: a linear decoder A q, or an odd (sign-symmetric)
 *            tanh perceptron with an optional residual block, the table
 *            form of the paper's decoder ablation; decode with the tables
 *            follows Eq. 12.
 *   lora     y[b][n] + scale * sum_r Bm[n][r] * (sum_k A[r][k] * x[b][k]),
 *            the optional low-rank compensation of Sec. III-F (plain
 *            definition, the adapter's down projection first).
 *
 * Storage format produced by encode (identical bytes are required from the
 * GPU encoder):
 *   codes [S][N][K/8] uint8  one byte per 8-element chunk; bit k = element k
 *                            of the chunk, 1 = negative, 0 = positive (the
 *                            sign of +0.0, -0.0 and exact zeros is positive)
 *   norms [S][N][K/8] uint16 IEEE binary16 bits of the stage target's chunk
 *                            L2 norm, rounded to nearest-even
 *   q8    [N][p_pad]  int8   p_pad = p rounded up to a multiple of 16, zero pad
 *   scale [p]         uint16 binary16 bits of max_i |W_ij| / 127
 *   idx   [p]         int32  protected input columns, ascending
 *
 * Readings of the paper taken here (the paper is silent on them):
 *   - no learned encoder/decoder: b = d = 8, the decoder is n16 * q;
 *   - protected entries are masked to zero before every stage (Eq. 10's
 *     complement realised by masking, not compaction);
 *   - sign(0) = +1;  g = NULL means g_j = 1;  ties in TopK go to the lower
 *     column index;  p is given by the caller (= ceil(rho * K)).
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#define OR_OK 0
#define OR_ERR_INVALID_ARG 1
#define OR_ERR_RANGE 3

/* ---------------------------------------------------------------- numbers */

/* bf16 -> binary64: bf16 is the upper half of a binary32, so widening is
 * exact for every bit pattern. */
double or_bf16_to_double(uint16_t b)
{
    uint32_t u = (uint32_t)b << 16;
    float f;
    memcpy(&f, &u, sizeof f);
    return (double)f;
}

/* binary16 bits -> binary64 (exact). */
double or_fp16_to_double(uint16_t h)
{
    int sign = (h >> 15) & 1;
    int e = (h >> 10) & 0x1f;
    int m = h & 0x3ff;
    double v;
    if (e == 0)
        v = ldexp((double)m, -24);                 /* zero or subnormal */
    else if (e == 31)
        v = m ? NAN : INFINITY;
    else
        v = ldexp((double)(1024 + m), e - 25);     /* 1.m * 2^(e-15) */
    return sign ? -v : v;
}

/* binary64 -> binary16 bits, round to nearest, ties to even, gradual
 * underflow, overflow to infinity.  The significand is scaled by a power of
 * two (exact in binary64) so that the 11 kept bits form the integer part,
 * and rounded once with nearbyint() in the default rounding mode. */
uint16_t or_double_to_fp16(double x)
{
    uint16_t sign = signbit(x) ? 0x8000 : 0;
    double a = fabs(x);
    if (isnan(x))
        return (uint16_t)(sign | 0x7e00);
    if (a < ldexp(1.0, -14)) {
        /* subnormal range: units of 2^-24; 1024 units is the least normal */
        double m = nearbyint(a * ldexp(1.0, 24));
        return (uint16_t)(sign | (uint16_t)m);
    }
    if (isinf(a))
        return (uint16_t)(sign | 0x7c00);
    int ex;
    frexp(a, &ex);                 /* a = f * 2^ex, f in [0.5, 1) */
    int E = ex - 1;                /* a in [2^E, 2^(E+1)) */
    if (E > 15)
        return (uint16_t)(sign | 0x7c00);
    double m = nearbyint(ldexp(a, 10 - E));   /* in [1024, 2048] */
    if (m == 2048.0) {
        m = 1024.0;
        E += 1;
        if (E > 15)
            return (uint16_t)(sign | 0x7c00);
    }
    return (uint16_t)(sign | (uint16_t)((E + 15) << 10) | (uint16_t)(m - 1024.0));
}

/* 1/sqrt(d) for d = 8, the spherical code's per-element magnitude (Eq. 3). */
static double or_inv_sqrt8(void) { return 1.0 / sqrt(8.0); }

int32_t or_pad16(int32_t p) { return (p + 15) / 16 * 16; }

/* Byte sizes of the five buffers of one encoded layer (Eq. 2 real-size
 * terms: S_code = codes, S_meta = norms + scales + indices, S_8bit = q8). */
int or_encoded_sizes(int32_t N, int32_t K, int32_t S, int32_t p, int64_t out[5])
{
    if (N <= 0 || K <= 0 || K % 8 != 0 || S < 1 || p < 0 || p > K)
        return OR_ERR_INVALID_ARG;
    int64_t C = K / 8;
    out[0] = (int64_t)S * N * C;                 /* codes  */
    out[1] = (int64_t)S * N * C * 2;             /* norms  */
    out[2] = (int64_t)N * or_pad16(p);           /* q8     */
    out[3] = (int64_t)p * 2;                     /* scales */
    out[4] = (int64_t)p * 4;                     /* idx    */
    return OR_OK;
}

/* ------------------------------------------------ Eq. 8: protected columns */

typedef struct { double score; int32_t j; } or_scored;

static int or_cmp_scored(const void *a, const void *b)
{
    const or_scored *x = (const or_scored *)a, *y = (const or_scored *)b;
    if (x->score > y->score) return -1;        /* larger score first */
    if (x->score < y->score) return 1;
    return (x->j < y->j) ? -1 : (x->j > y->j); /* tie: lower index first */
}

static int or_cmp_i32(const void *a, const void *b)
{
    int32_t x = *(const int32_t *)a, y = *(const int32_t *)b;
    return (x > y) - (x < y);
}

/* score_j = g_j * sqrt(sum_{i=0..N-1} W_ij^2), the sum taken in ascending i;
 * P = the p columns of largest score, returned ascending.  Also writes the
 * scores when scores_out != NULL. */
int or_select_protected(const uint16_t *W, const float *g, int32_t N, int32_t K,
                        int32_t p, int32_t *idx_out, double *scores_out)
{
    if (p < 0 || p > K) return OR_ERR_INVALID_ARG;
    or_scored *sc = (or_scored *)malloc(sizeof(or_scored) * (size_t)K);
    if (!sc) return OR_ERR_INVALID_ARG;
    for (int32_t j = 0; j < K; ++j) {
        double sum = 0.0;
        for (int32_t i = 0; i < N; ++i) {
            double w = or_bf16_to_double(W[(int64_t)i * K + j]);
            sum = sum + w * w;
        }
        double s = sqrt(sum);
        if (g) s = (double)g[j] * s;
        sc[j].score = s;
        sc[j].j = j;
        if (scores_out) scores_out[j] = s;
    }
    qsort(sc, (size_t)K, sizeof(or_scored), or_cmp_scored);
    for (int32_t t = 0; t < p; ++t) idx_out[t] = sc[t].j;
    qsort(idx_out, (size_t)p, sizeof(int32_t), or_cmp_i32);
    free(sc);
    return OR_OK;
}

/* ----------------------------------------- Eq. 10: 8-bit protected slices */

/* Per protected column j (a per-channel 8-bit quantiser):
 *   scale_j = fp16(max_i |W_ij| / 127)
 *   q8_ij   = clamp(rint(W_ij / scale_j), -127, 127), or 0 if scale_j == 0. */
int or_quantize_protected(const uint16_t *W, int32_t N, int32_t K,
                          const int32_t *idx, int32_t p,
                          int8_t *q8_out, uint16_t *scale_out)
{
    int32_t pp = or_pad16(p);
    memset(q8_out, 0, (size_t)N * (size_t)pp);
    for (int32_t t = 0; t < p; ++t) {
        int32_t j = idx[t];
        double m = 0.0;
        for (int32_t i = 0; i < N; ++i) {
            double a = fabs(or_bf16_to_double(W[(int64_t)i * K + j]));
            if (a > m) m = a;
        }
        uint16_t s16 = or_double_to_fp16(m / 127.0);
        if ((s16 & 0x7c00) == 0x7c00) return OR_ERR_RANGE;
        scale_out[t] = s16;
        double s = or_fp16_to_double(s16);
        for (int32_t i = 0; i < N; ++i) {
            double q = 0.0;
            if (s != 0.0) {
                q = nearbyint(or_bf16_to_double(W[(int64_t)i * K + j]) / s);
                if (q > 127.0) q = 127.0;
                if (q < -127.0) q = -127.0;
            }
            q8_out[(int64_t)i * pp + t] = (int8_t)q;
        }
    }
    return OR_OK;
}

/* --------------------------------- Eq. 3 + Eq. 5-7: spherical sign stages */

/* For every row i and chunk c (8 contiguous input columns), with
 * r(0) = the chunk of W with protected entries set to zero, for s = 1..S:
 *   n      = sqrt(((((((v0^2+v1^2)+v2^2)+v3^2)+v4^2)+v5^2)+v6^2)+v7^2)
 *   n16    = fp16(n)                       (stored norm; overflow -> RANGE)
 *   bit_k  = (v_k < 0)                     (stored sign pattern, Eq. 3)
 *   rhat_k = (bit_k ? -1 : +1) * n16 / sqrt(8)
 *   r(s)_k = r(s-1)_k - rhat_k, then 0 at protected entries   (Eq. 5-7)  */
int or_encode_stages(const uint16_t *W, int32_t N, int32_t K, int32_t S,
                     const int32_t *idx, int32_t p,
                     uint8_t *codes_out, uint16_t *norms_out)
{
    int32_t C = K / 8;
    double inv_sqrt8 = or_inv_sqrt8();
    unsigned char *prot = (unsigned char *)calloc((size_t)K, 1);
    if (!prot) return OR_ERR_INVALID_ARG;
    for (int32_t t = 0; t < p; ++t) prot[idx[t]] = 1;
    int rc = OR_OK;
    for (int32_t i = 0; i < N && rc == OR_OK; ++i) {
        for (int32_t c = 0; c < C; ++c) {
            double v[8];
            for (int k = 0; k < 8; ++k) {
                int32_t j = 8 * c + k;
                v[k] = prot[j] ? 0.0 : or_bf16_to_double(W[(int64_t)i * K + j]);
            }
            for (int32_t s = 0; s < S; ++s) {
                double sum = v[0] * v[0];
                for (int k = 1; k < 8; ++k) sum = sum + v[k] * v[k];
                double n = sqrt(sum);
                uint16_t n16 = or_double_to_fp16(n);
                if ((n16 & 0x7c00) == 0x7c00) { rc = OR_ERR_RANGE; break; }
                uint8_t bits = 0;
                for (int k = 0; k < 8; ++k)
                    if (v[k] < 0.0) bits |= (uint8_t)(1u << k);
                double t = or_fp16_to_double(n16) * inv_sqrt8;
                for (int k = 0; k < 8; ++k) {
                    double rhat = ((bits >> k) & 1) ? -t : t;
                    v[k] = v[k] - rhat;
                    if (prot[8 * c + k]) v[k] = 0.0;
                }
                int64_t o = ((int64_t)s * N + i) * C + c;
                codes_out[o] = bits;
                norms_out[o] = n16;
            }
            if (rc != OR_OK) break;
        }
    }
    free(prot);
    return rc;
}

/* Whole offline encoder: non-finite weights are rejected with RANGE. */
int or_encode(const uint16_t *W, const float *g, int32_t N, int32_t K,
              int32_t S, int32_t p, uint8_t *codes, uint16_t *norms,
              int8_t *q8, uint16_t *scale, int32_t *idx)
{
    if (N <= 0 || K <= 0 || K % 8 != 0 || S < 1 || S > 3 || p < 0 || p > K)
        return OR_ERR_INVALID_ARG;
    for (int64_t e = 0; e < (int64_t)N * K; ++e)
        if (!isfinite(or_bf16_to_double(W[e]))) return OR_ERR_RANGE;
    int rc = or_select_protected(W, g, N, K, p, idx, NULL);
    if (rc) return rc;
    rc = or_quantize_protected(W, N, K, idx, p, q8, scale);
    if (rc) return rc;
    return or_encode_stages(W, N, K, S, idx, p, codes, norms);
}

/* ------------------------------------------------ Eq. 12 + Eq. 10: decode */

/* Dense reconstruction of rows [row0, row0+nrows):
 *   What_ij = sum_{s=1..S} (bit ? -1 : +1) * n16_{s,i,c} / sqrt(8)   j not in P
 *   What_ij = scale_j * q8_ij                                         j in P   */
void or_decode_rows(const uint8_t *codes, const uint16_t *norms,
                    const int8_t *q8, const uint16_t *scale, const int32_t *idx,
                    int32_t N, int32_t K, int32_t S, int32_t p,
                    int32_t row0, int32_t nrows, double *out)
{
    int32_t C = K / 8, pp = or_pad16(p);
    double inv_sqrt8 = or_inv_sqrt8();
    for (int32_t r = 0; r < nrows; ++r) {
        int32_t i = row0 + r;
        double *o = out + (int64_t)r * K;
        for (int32_t j = 0; j < K; ++j) {
            int32_t c = j / 8, k = j % 8;
            double acc = 0.0;
            for (int32_t s = 0; s < S; ++s) {
                int64_t e = ((int64_t)s * N + i) * C + c;
                double t = or_fp16_to_double(norms[e]) * inv_sqrt8;
                acc = acc + (((codes[e] >> k) & 1) ? -t : t);
            }
            o[j] = acc;
        }
        for (int32_t t = 0; t < p; ++t)
            o[idx[t]] = or_fp16_to_double(scale[t]) * (double)q8[(int64_t)i * pp + t];
    }
}

/* y[b][r] = sum_j What[r][j] * x[b][j], ascending j, for a block of rows. */
void or_matmul(const double *What, int32_t nrows, int32_t K,
               const uint16_t *X, int32_t B, double *Y)
{
    for (int32_t b = 0; b < B; ++b)
        for (int32_t r = 0; r < nrows; ++r) {
            double acc = 0.0;
            for (int32_t j = 0; j < K; ++j)
                acc = acc + What[(int64_t)r * K + j] *
                            or_bf16_to_double(X[(int64_t)b * K + j]);
            Y[(int64_t)b * nrows + r] = acc;
        }
}

/* Y[b][t] = (x_b . What[rows[t], :]) for a list of rows, decoding one row at
 * a time (used to check full-size layers on sampled outputs). */
int or_apply_rows(const uint8_t *codes, const uint16_t *norms,
                  const int8_t *q8, const uint16_t *scale, const int32_t *idx,
                  int32_t N, int32_t K, int32_t S, int32_t p,
                  const int32_t *rows, int32_t nrows,
                  const uint16_t *X, int32_t B, double *Y)
{
    double *w = (double *)malloc(sizeof(double) * (size_t)K);
    double *y = (double *)malloc(sizeof(double) * (size_t)B);
    if (!w || !y) { free(w); free(y); return OR_ERR_INVALID_ARG; }
    for (int32_t t = 0; t < nrows; ++t) {
        or_decode_rows(codes, norms, q8, scale, idx, N, K, S, p, rows[t], 1, w);
        or_matmul(w, 1, K, X, B, y);
        for (int32_t b = 0; b < B; ++b) Y[(int64_t)b * nrows + t] = y[b];
    }
    free(w);
    free(y);
    return OR_OK;
}

/* Low-rank compensation added to a layer output (Sec. III-F: LoRA adapters
 * trained with the codes fixed).  A [rank][K], Bm [N][rank] and X [B][K] are
 * bf16 bits, Y0 [B][N] the output before compensation.  First
 * t[b][r] = sum_k A[r][k] x[b][k] (ascending k), then
 * Y[b][n] = Y0[b][n] + scale * sum_r Bm[n][r] t[b][r] (ascending r). */
int or_lora_apply(const uint16_t *A, const uint16_t *Bm, int32_t rank, int32_t N, int32_t K,
                  double scale, const uint16_t *X, int32_t B, const double *Y0, double *Y)
{
    if (rank < 1 || N < 1 || K < 1 || B < 1) return OR_ERR_INVALID_ARG;
    double *t = (double *)malloc(sizeof(double) * (size_t)rank);
    if (!t) return OR_ERR_INVALID_ARG;
    for (int32_t b = 0; b < B; ++b) {
        for (int32_t r = 0; r < rank; ++r) {
            double acc = 0.0;
            for (int32_t k = 0; k < K; ++k)
                acc = acc + or_bf16_to_double(A[(int64_t)r * K + k]) *
                            or_bf16_to_double(X[(int64_t)b * K + k]);
            t[r] = acc;
        }
        for (int32_t n = 0; n < N; ++n) {
            double acc = 0.0;
            for (int32_t r = 0; r < rank; ++r)
                acc = acc + or_bf16_to_double(Bm[(int64_t)n * rank + r]) * t[r];
            Y[(int64_t)b * N + n] = Y0[(int64_t)b * N + n] + scale * acc;
        }
    }
    free(t);
    return OR_OK;
}

/* ------------------------------- output-row protection (Eq. 9, Eq. 10) */

/* score_i = g_i * sqrt(sum_k W_ik^2) (ascending k) for output row i; P = the
 * p rows of largest score, ties to the lower index, returned ascending. */
int or_select_rows(const uint16_t *W, const float *g, int32_t N, int32_t K, int32_t p,
                   int32_t *idx_out, double *scores_out)
{
    if (p < 0 || p > N) return OR_ERR_INVALID_ARG;
    or_scored *sc = (or_scored *)malloc(sizeof(or_scored) * (size_t)N);
    if (!sc) return OR_ERR_INVALID_ARG;
    for (int32_t i = 0; i < N; ++i) {
        double sum = 0.0;
        for (int32_t k = 0; k < K; ++k) {
            double w = or_bf16_to_double(W[(int64_t)i * K + k]);
            sum = sum + w * w;
        }
        double s = sqrt(sum);
        if (g) s = (double)g[i] * s;
        sc[i].score = s;
        sc[i].j = i;
        if (scores_out) scores_out[i] = s;
    }
    qsort(sc, (size_t)N, sizeof(or_scored), or_cmp_scored);
    for (int32_t t = 0; t < p; ++t) idx_out[t] = sc[t].j;
    qsort(idx_out, (size_t)p, sizeof(int32_t), or_cmp_i32);
    free(sc);
    return OR_OK;
}

/* Eq. 9, the coupled score of intermediate channel j of a gated MLP:
 *   S_j = gg_j ||Wg[j,:]||_2 + gu_j ||Wu[j,:]||_2 + gd_j ||Wd[:,j]||_2
 * with Wg, Wu [F][H] (gate/up rows) and Wd [H][F] (down columns); each norm
 * is the square root of a sum in ascending index, and the three terms are
 * added in that order.  A NULL g means 1.  P = TopK_j, ties to the lower j,
 * returned ascending. */
int or_select_coupled(const uint16_t *Wg, const uint16_t *Wu, const uint16_t *Wd,
                      const float *gg, const float *gu, const float *gd,
                      int32_t F, int32_t H, int32_t p, int32_t *idx_out, double *scores_out)
{
    if (F <= 0 || H <= 0 || p < 0 || p > F) return OR_ERR_INVALID_ARG;
    or_scored *sc = (or_scored *)malloc(sizeof(or_scored) * (size_t)F);
    if (!sc) return OR_ERR_INVALID_ARG;
    for (int32_t j = 0; j < F; ++j) {
        double sg = 0.0, su = 0.0, sd = 0.0;
        for (int32_t h = 0; h < H; ++h) {
            double a = or_bf16_to_double(Wg[(int64_t)j * H + h]);
            double b = or_bf16_to_double(Wu[(int64_t)j * H + h]);
            sg = sg + a * a;
            su = su + b * b;
        }
        for (int32_t h = 0; h < H; ++h) {
            double c = or_bf16_to_double(Wd[(int64_t)h * F + j]);
            sd = sd + c * c;
        }
        double tg = sqrt(sg), tu = sqrt(su), td = sqrt(sd);
        if (gg) tg = (double)gg[j] * tg;
        if (gu) tu = (double)gu[j] * tu;
        if (gd) td = (double)gd[j] * td;
        double s = (tg + tu) + td;
        sc[j].score = s;
        sc[j].j = j;
        if (scores_out) scores_out[j] = s;
    }
    qsort(sc, (size_t)F, sizeof(or_scored), or_cmp_scored);
    for (int32_t t = 0; t < p; ++t) idx_out[t] = sc[t].j;
    qsort(idx_out, (size_t)p, sizeof(int32_t), or_cmp_i32);
    free(sc);
    return OR_OK;
}

/* Eq. 10 on protected rows, one scale per row (the protected channel):
 *   scale_t = fp16(max_k |W_{i_t,k}| / 127)
 *   q8[t][k] = clamp(rint(W_{i_t,k} / scale_t), -127, 127), or 0 if scale_t == 0
 * q8 is [p][kp], kp = K rounded up to a multiple of 16, zero padding. */
int or_quantize_protected_rows(const uint16_t *W, int32_t N, int32_t K,
                               const int32_t *idx, int32_t p,
                               int8_t *q8_out, uint16_t *scale_out)
{
    int32_t kp = or_pad16(K);
    memset(q8_out, 0, (size_t)(p > 0 ? p : 0) * (size_t)kp);
    for (int32_t t = 0; t < p; ++t) {
        int32_t i = idx[t];
        if (i < 0 || i >= N) return OR_ERR_INVALID_ARG;
        double m = 0.0;
        for (int32_t k = 0; k < K; ++k) {
            double a = fabs(or_bf16_to_double(W[(int64_t)i * K + k]));
            if (a > m) m = a;
        }
        uint16_t s16 = or_double_to_fp16(m / 127.0);
        if ((s16 & 0x7c00) == 0x7c00) return OR_ERR_RANGE;
        scale_out[t] = s16;
        double s = or_fp16_to_double(s16);
        for (int32_t k = 0; k < K; ++k) {
            double q = 0.0;
            if (s != 0.0) {
                q = nearbyint(or_bf16_to_double(W[(int64_t)i * K + k]) / s);
                if (q > 127.0) q = 127.0;
                if (q < -127.0) q = -127.0;
            }
            q8_out[(int64_t)t * kp + k] = (int8_t)q;
        }
    }
    return OR_OK;
}

/* Whole encoder with output-row protection.  P is selected by
 * or_select_rows when idx_in is NULL, else taken from idx_in (ascending,
 * e.g. the coupled MLP set of or_select_coupled).  The protected rows are
 * zero in the BSQ target (masking, as for columns), so each of their chunks
 * stores norm 0 and sign byte 0; the stages are or_encode_stages on that
 * masked matrix with no protected columns. */
int or_encode_rows(const uint16_t *W, const float *g, int32_t N, int32_t K, int32_t S,
                   int32_t p, const int32_t *idx_in, uint8_t *codes, uint16_t *norms,
                   int8_t *q8, uint16_t *scale, int32_t *idx)
{
    if (N <= 0 || K <= 0 || K % 8 != 0 || S < 1 || S > 3 || p < 0 || p > N)
        return OR_ERR_INVALID_ARG;
    for (int64_t e = 0; e < (int64_t)N * K; ++e)
        if (!isfinite(or_bf16_to_double(W[e]))) return OR_ERR_RANGE;
    int rc = OR_OK;
    if (idx_in) {
        for (int32_t t = 0; t < p; ++t) {
            if (idx_in[t] < 0 || idx_in[t] >= N || (t > 0 && idx_in[t] <= idx_in[t - 1]))
                return OR_ERR_INVALID_ARG;
            idx[t] = idx_in[t];
        }
    } else {
        rc = or_select_rows(W, g, N, K, p, idx, NULL);
        if (rc) return rc;
    }
    rc = or_quantize_protected_rows(W, N, K, idx, p, q8, scale);
    if (rc) return rc;
    uint16_t *Wm = (uint16_t *)malloc(sizeof(uint16_t) * (size_t)N * (size_t)K);
    if (!Wm) return OR_ERR_INVALID_ARG;
    memcpy(Wm, W, sizeof(uint16_t) * (size_t)N * (size_t)K);
    for (int32_t t = 0; t < p; ++t)
        memset(Wm + (int64_t)idx[t] * K, 0, sizeof(uint16_t) * (size_t)K);
    rc = or_encode_stages(Wm, N, K, S, NULL, 0, codes, norms);
    free(Wm);
    return rc;
}

/* Dense rows [row0, row0+nrows) of a row-protected layer:
 *   What[i][:] = scale_t * q8[t][:]                  i = idx[t]
 *   What[i][:] = the BSQ rows of Eq. 12              otherwise */
void or_decode_rows_axis1(const uint8_t *codes, const uint16_t *norms,
                          const int8_t *q8, const uint16_t *scale, const int32_t *idx,
                          int32_t N, int32_t K, int32_t S, int32_t p,
                          int32_t row0, int32_t nrows, double *out)
{
    int32_t kp = or_pad16(K);
    or_decode_rows(codes, norms, NULL, NULL, NULL, N, K, S, 0, row0, nrows, out);
    for (int32_t t = 0; t < p; ++t) {
        int32_t i = idx[t];
        if (i < row0 || i >= row0 + nrows) continue;
        double s = or_fp16_to_double(scale[t]);
        for (int32_t k = 0; k < K; ++k)
            out[(int64_t)(i - row0) * K + k] = s * (double)q8[(int64_t)t * kp + k];
    }
}

/* ------------------------------- FP8 and BF16 protected payloads (Eq. 10) */

/* Formats of the protected payload: 0 = INT8 (or_quantize_protected),
 * 1 = FP8 E4M3 (bias 7, largest finite 448, S.1111.111 is NaN, no
 * infinities), 2 = FP8 E5M2 (bias 15, largest finite 57344, IEEE-style
 * infinities and NaNs), 3 = BF16 (the weight itself). */
#define OR_FMT_INT8 0
#define OR_FMT_E4M3 1
#define OR_FMT_E5M2 2
#define OR_FMT_BF16 3

static int or_fp8_params(int fmt, int *mbits, int *bias, double *maxf, uint8_t *maxcode)
{
    if (fmt == OR_FMT_E4M3) { *mbits = 3; *bias = 7; *maxf = 448.0; *maxcode = 0x7e; return 1; }
    if (fmt == OR_FMT_E5M2) { *mbits = 2; *bias = 15; *maxf = 57344.0; *maxcode = 0x7b; return 1; }
    return 0;
}

/* binary64 -> FP8 bits: round to nearest, ties to even, gradual underflow;
 * a finite value that rounds above the largest finite one gives the largest
 * finite one (saturation), +-inf too; NaN gives the format's NaN.  Same
 * method as or_double_to_fp16: scale the significand by a power of two so
 * that the kept bits are the integer part, and round once with nearbyint(). */
uint8_t or_double_to_fp8(double x, int fmt)
{
    int mb, bias;
    double maxf;
    uint8_t maxcode;
    if (!or_fp8_params(fmt, &mb, &bias, &maxf, &maxcode)) return 0;
    uint8_t sign = signbit(x) ? 0x80 : 0;
    if (isnan(x)) return (uint8_t)(sign | (fmt == OR_FMT_E4M3 ? 0x7f : 0x7e));
    double a = fabs(x);
    if (isinf(a)) return (uint8_t)(sign | maxcode);
    if (a < ldexp(1.0, 1 - bias)) {
        /* subnormal range: units of 2^(1 - bias - mb); 2^mb units is the
         * least normal, whose code is the same integer */
        double m = nearbyint(ldexp(a, bias - 1 + mb));
        return (uint8_t)(sign | (uint8_t)m);
    }
    int ex;
    frexp(a, &ex);                  /* a = f * 2^ex, f in [0.5, 1) */
    int E = ex - 1;                 /* a in [2^E, 2^(E+1)) */
    double m = nearbyint(ldexp(a, mb - E));   /* in [2^mb, 2^(mb+1)] */
    if (m == ldexp(1.0, mb + 1)) {
        m = ldexp(1.0, mb);
        E += 1;
    }
    double v = ldexp(m, E - mb);
    if (v > maxf) return (uint8_t)(sign | maxcode);
    return (uint8_t)(sign | (uint8_t)((E + bias) << mb) | (uint8_t)(m - ldexp(1.0, mb)));
}

/* FP8 bits -> binary64 (exact). */
double or_fp8_to_double(uint8_t v, int fmt)
{
    int mb, bias;
    double maxf;
    uint8_t maxcode;
    if (!or_fp8_params(fmt, &mb, &bias, &maxf, &maxcode)) return NAN;
    int sign = v >> 7;
    int emax = (1 << (7 - mb)) - 1;
    int e = (v >> mb) & emax;
    int mant = v & ((1 << mb) - 1);
    double r;
    if (fmt == OR_FMT_E4M3 && e == emax && mant == (1 << mb) - 1)
        r = NAN;
    else if (fmt == OR_FMT_E5M2 && e == emax)
        r = mant ? NAN : INFINITY;
    else if (e == 0)
        r = ldexp((double)mant, 1 - bias - mb);
    else
        r = ldexp((double)((1 << mb) + mant), e - bias - mb);
    return sign ? -r : r;
}

/* Eq. 10 with an FP8 payload, per protected column j:
 *   scale_j = fp16(max_i |W_ij| / largest finite FP8 value)
 *   q_ij    = fp8(W_ij / scale_j), or +0 if scale_j == 0
 * With BF16 the payload is the weight's own bits and the scale is 1.0.
 * q is [N][p_pad] bytes (FP8) or [N][p_pad] bf16 (BF16), zero padding. */
int or_quantize_protected_fmt(const uint16_t *W, int32_t N, int32_t K,
                              const int32_t *idx, int32_t p, int fmt,
                              void *q_out, uint16_t *scale_out)
{
    int32_t pp = or_pad16(p);
    int mb, bias;
    double maxf;
    uint8_t maxcode;
    if (fmt == OR_FMT_BF16) {
        uint16_t *q = (uint16_t *)q_out;
        memset(q, 0, sizeof(uint16_t) * (size_t)N * (size_t)pp);
        for (int32_t t = 0; t < p; ++t) {
            scale_out[t] = 0x3c00;   /* 1.0 */
            for (int32_t i = 0; i < N; ++i) q[(int64_t)i * pp + t] = W[(int64_t)i * K + idx[t]];
        }
        return OR_OK;
    }
    if (!or_fp8_params(fmt, &mb, &bias, &maxf, &maxcode)) return OR_ERR_INVALID_ARG;
    uint8_t *q = (uint8_t *)q_out;
    memset(q, 0, (size_t)N * (size_t)pp);
    for (int32_t t = 0; t < p; ++t) {
        int32_t j = idx[t];
        double m = 0.0;
        for (int32_t i = 0; i < N; ++i) {
            double a = fabs(or_bf16_to_double(W[(int64_t)i * K + j]));
            if (a > m) m = a;
        }
        uint16_t s16 = or_double_to_fp16(m / maxf);
        if ((s16 & 0x7c00) == 0x7c00) return OR_ERR_RANGE;
        scale_out[t] = s16;
        double s = or_fp16_to_double(s16);
        for (int32_t i = 0; i < N; ++i)
            q[(int64_t)i * pp + t] =
                s != 0.0 ? or_double_to_fp8(or_bf16_to_double(W[(int64_t)i * K + j]) / s, fmt) : 0;
    }
    return OR_OK;
}

/* The decoded protected value of column t in row i: scale_t * value(q). */
double or_protected_value_fmt(const void *q, const uint16_t *scale, int32_t p,
                              int fmt, int32_t i, int32_t t)
{
    int32_t pp = or_pad16(p);
    double s = or_fp16_to_double(scale[t]);
    if (fmt == OR_FMT_BF16) return s * or_bf16_to_double(((const uint16_t *)q)[(int64_t)i * pp + t]);
    if (fmt == OR_FMT_INT8) return s * (double)((const int8_t *)q)[(int64_t)i * pp + t];
    return s * or_fp8_to_double(((const uint8_t *)q)[(int64_t)i * pp + t], fmt);
}


/* ------------------------------------- learned decoder step (Eq. 1, Eq. 12) */

/* The decoder D of Eq. 1 maps a stage's code q in {-1/sqrt(8), +1/sqrt(8)}^8
 * (Eq. 3 with b = d = 8) to a chunk.  With the stored norm kept, a chunk of
 * stage s decodes to n16 * D_s(q).  Since q takes only 256 values, D_s is
 * fully described by its table T_s[v][k] = D_s(q(v))_k, v the code byte
 * (bit k of v set <=> q_k = -1/sqrt(8)).  The identity decoder q -> q is the
 * norm-rescale decoder of the rest of this file. */

/* q(v)_k = (bit k of v ? -1 : +1) / sqrt(8) */
static double or_code_elem(int v, int k)
{
    double t = or_inv_sqrt8();
    return ((v >> k) & 1) ? -t : t;
}

/* Linear decoder D(q) = A q, A [8][8] row-major (output k, code position j):
 * T[v][k] = sum_j A[k][j] * q(v)_j, ascending j. */
void or_decoder_table_linear(const double *A, double *T)
{
    for (int v = 0; v < 256; ++v)
        for (int k = 0; k < 8; ++k) {
            double acc = 0.0;
            for (int j = 0; j < 8; ++j) acc = acc + A[k * 8 + j] * or_code_elem(v, j);
            T[v * 8 + k] = acc;
        }
}

/* Symmetric (odd) nonlinear decoder, D(-q) = -D(q): a bias-free perceptron
 * with the odd activation tanh,
 *   h   = tanh(W1 q)                 W1 [hdim][8]
 *   h   = h + tanh(Wr h)             Wr [hdim][hdim], only if Wr != NULL
 *                                    (the residual block)
 *   out = W2 h                       W2 [8][hdim]
 * every product summed in ascending index order. */
int or_decoder_table_mlp(const double *W1, int32_t hdim, const double *Wr,
                         const double *W2, double *T)
{
    if (hdim <= 0) return OR_ERR_INVALID_ARG;
    double *h = (double *)malloc(sizeof(double) * (size_t)hdim);
    double *g = (double *)malloc(sizeof(double) * (size_t)hdim);
    if (!h || !g) { free(h); free(g); return OR_ERR_INVALID_ARG; }
    for (int v = 0; v < 256; ++v) {
        for (int32_t a = 0; a < hdim; ++a) {
            double acc = 0.0;
            for (int j = 0; j < 8; ++j) acc = acc + W1[(int64_t)a * 8 + j] * or_code_elem(v, j);
            h[a] = tanh(acc);
        }
        if (Wr) {
            for (int32_t a = 0; a < hdim; ++a) {
                double acc = 0.0;
                for (int32_t c = 0; c < hdim; ++c) acc = acc + Wr[(int64_t)a * hdim + c] * h[c];
                g[a] = tanh(acc);
            }
            for (int32_t a = 0; a < hdim; ++a) h[a] = h[a] + g[a];
        }
        for (int k = 0; k < 8; ++k) {
            double acc = 0.0;
            for (int32_t a = 0; a < hdim; ++a) acc = acc + W2[(int64_t)k * hdim + a] * h[a];
            T[v * 8 + k] = acc;
        }
    }
    free(h);
    free(g);
    return OR_OK;
}

/* Dense reconstruction with per-stage decoder tables (Eq. 12 with Eq. 1):
 *   What_ij = sum_{s=1..S} n16_{s,i,c} * T_s[code_{s,i,c}][j % 8]   j not in P
 *   What_ij = scale_j * q8_ij                                       j in P
 * tables [S][256][8] are binary16 bits: the evaluated decoder as a kernel
 * would hold it. */
void or_decode_rows_table(const uint8_t *codes, const uint16_t *norms, const uint16_t *tables,
                          const int8_t *q8, const uint16_t *scale, const int32_t *idx,
                          int32_t N, int32_t K, int32_t S, int32_t p,
                          int32_t row0, int32_t nrows, double *out)
{
    int32_t C = K / 8, pp = or_pad16(p);
    for (int32_t r = 0; r < nrows; ++r) {
        int32_t i = row0 + r;
        double *o = out + (int64_t)r * K;
        for (int32_t j = 0; j < K; ++j) {
            int32_t c = j / 8, k = j % 8;
            double acc = 0.0;
            for (int32_t s = 0; s < S; ++s) {
                int64_t e = ((int64_t)s * N + i) * C + c;
                double t = or_fp16_to_double(tables[((int64_t)s * 256 + codes[e]) * 8 + k]);
                acc = acc + or_fp16_to_double(norms[e]) * t;
            }
            o[j] = acc;
        }
        for (int32_t t = 0; t < p; ++t)
            o[idx[t]] = or_fp16_to_double(scale[t]) * (double)q8[(int64_t)i * pp + t];
    }
}
