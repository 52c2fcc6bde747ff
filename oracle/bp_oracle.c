/*
 * Plain CPU oracle for block-based / block-punched pruned-layer inference
 * (arXiv 2111.11581).  TEST INFRASTRUCTURE ONLY: this file is compiled into
 * liboracle.so, which only the tests, the smoke check and the benchmark's CPU
 * baseline load.  The product library never links or calls it, and it shares
 * no code, header or table with the CUDA path.
 *
 * Everything here is written as slow, obvious loops in fp64, following the
 * paper's definitions:
 *   - weight notation and block partition:   Sec. 4.2 (W_i in R^{P x Q x Kh x Kw},
 *     J equal blocks of p x q (x Kh x Kw));
 *   - block-based pruning (FC / GEMM view):  Sec. 4.1.1 (prune whole columns
 *     inside each block, per-block rate may differ);
 *   - block-punched pruning (CONV):          Sec. 4.1.2 (prune the same kernel
 *     positions in every kernel of a filters x channels block);
 *   - column score ||[W_ij]_{:,n}||_F^2:     Eq. (column), Sec. 4.2;
 *   - position score ||[W_ij]_{:,:,m,n}||^2:  Eq. (punched), Sec. 4.2;
 *   - one-shot magnitude pruning at a rate:  Sec. 5.1;
 *   - compact per-row-block storage (BCS):   Sec. 4.3;
 *   - inference with only kept weights:      Sec. 4.3 (pruned weights do not
 *     take part in the computation).
 * Readings of points the paper leaves open (fp64 scores in a fixed order,
 * tie-breaking, non-integer per-block keep counts, partial edge blocks,
 * output rounding) are listed in the design notes; each is restated at the
 * function that implements it.
 *
 * Tensors of 16-bit floats are passed as their raw uint16 bit patterns.
 * dtype 0 = IEEE binary16 (fp16), dtype 1 = bfloat16.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#define OR_OK 0
#define OR_ERR_ARG 1
#define OR_ERR_NONFINITE 3

/* ------------------------------------------------------------------------ */
/* 16-bit float <-> double, written from the IEEE 754 / bfloat16 encodings.  */
/* ------------------------------------------------------------------------ */

double oracle_half_to_double(uint16_t h, int dtype)
{
    int sign = (h >> 15) & 1;
    double v;
    if (dtype == 1) { /* bfloat16: 1 sign, 8 exponent (bias 127), 7 fraction bits */
        int e = (h >> 7) & 0xff;
        int f = h & 0x7f;
        if (e == 0xff) v = f ? NAN : INFINITY;
        else if (e == 0) v = ldexp((double)f, -133);           /* f * 2^-126 * 2^-7 */
        else v = ldexp((double)(128 + f), e - 127 - 7);
    } else {          /* binary16: 1 sign, 5 exponent (bias 15), 10 fraction bits */
        int e = (h >> 10) & 0x1f;
        int f = h & 0x3ff;
        if (e == 0x1f) v = f ? NAN : INFINITY;
        else if (e == 0) v = ldexp((double)f, -24);            /* f * 2^-14 * 2^-10 */
        else v = ldexp((double)(1024 + f), e - 15 - 10);
    }
    return sign ? -v : v;
}

/* Round a double to the nearest representable 16-bit float, ties to even,
 * directly from the double (one rounding).  Overflow goes to infinity. */
uint16_t oracle_double_to_half(double x, int dtype)
{
    const int fbits = dtype == 1 ? 7 : 10;       /* stored fraction bits     */
    const int emin = dtype == 1 ? -126 : -14;    /* smallest normal exponent */
    const int emax = dtype == 1 ? 127 : 15;      /* largest normal exponent  */
    const int bias = dtype == 1 ? 127 : 15;
    const int ebits = dtype == 1 ? 8 : 5;
    uint16_t sign = signbit(x) ? (uint16_t)(1u << 15) : 0;
    if (isnan(x)) return (uint16_t)(dtype == 1 ? 0x7fc0 : 0x7e00);
    double a = fabs(x);
    uint16_t inf = (uint16_t)(sign | (((1u << ebits) - 1u) << fbits));
    if (isinf(a)) return inf;
    if (a == 0.0) return sign;
    int ex;
    frexp(a, &ex);              /* a = f * 2^ex, f in [0.5, 1) */
    int E = ex - 1;             /* a in [2^E, 2^(E+1)) */
    int Eq = E < emin ? emin : E;
    /* quantum of the target format in the binade of a (subnormal quantum below emin) */
    double n = ldexp(a, -(Eq - fbits));
    double r = ldexp(nearbyint(n), Eq - fbits);  /* default rounding: nearest, ties to even */
    if (r == 0.0) return sign;
    if (r >= ldexp(1.0, emax + 1)) return inf;
    frexp(r, &ex);
    E = ex - 1;
    if (E < emin) {             /* subnormal result */
        uint32_t mant = (uint32_t)ldexp(r, -(emin - fbits));
        return (uint16_t)(sign | mant);
    }
    uint32_t mant = (uint32_t)ldexp(r, -(E - fbits)) - (1u << fbits);
    return (uint16_t)(sign | ((uint32_t)(E + bias) << fbits) | mant);
}

void oracle_to_double(const uint16_t *src, double *dst, int64_t n, int dtype)
{
    for (int64_t i = 0; i < n; ++i) dst[i] = oracle_half_to_double(src[i], dtype);
}

void oracle_from_double(const double *src, uint16_t *dst, int64_t n, int dtype)
{
    for (int64_t i = 0; i < n; ++i) dst[i] = oracle_double_to_half(src[i], dtype);
}

/* ------------------------------------------------------------------------ */
/* Block partition (Sec. 4.2).                                               */
/*   scheme 0 = block-based (Sec. 4.1.1): W is the M x K GEMM view; rows are  */
/*     split into row-blocks of bm, columns into column-blocks of bk; the    */
/*     units of a block are its columns.                                     */
/*   scheme 1 = block-punched (Sec. 4.1.2): W is F x C x kh x kw (OIHW), so   */
/*     M = F and K = C*kh*kw; filters split by bm, channels by bk; the units */
/*     of a block are the kh*kw kernel positions.                            */
/* The last row-/column-block may be partial; it keeps its real size.        */
/* Units are numbered g = (rb*CB + cb)*Pmax + u, i.e. row-block major, then  */
/* column-block, then unit, which is also the tie-breaking order.            */
/* ------------------------------------------------------------------------ */

typedef struct {
    int scheme;
    int64_t M, K;
    int64_t kh, kw, KK, C;     /* KK = kh*kw, C = K / KK */
    int64_t bm, bk;
    int64_t RB, CB;            /* number of row-blocks, column-blocks */
    int64_t Pmax;              /* units per full block */
    int64_t U;                 /* total units RB*CB*Pmax (block-based: RB*K) */
} part_t;

static int make_part(part_t *p, int scheme, int64_t M, int64_t K, int64_t kh, int64_t kw,
                     int64_t bm, int64_t bk)
{
    if (M < 1 || K < 1 || bm < 1 || bk < 1 || kh < 1 || kw < 1) return OR_ERR_ARG;
    if (scheme != 0 && scheme != 1) return OR_ERR_ARG;
    p->scheme = scheme; p->M = M; p->K = K; p->kh = kh; p->kw = kw; p->bm = bm; p->bk = bk;
    p->KK = kh * kw;
    if (K % p->KK) return OR_ERR_ARG;
    p->C = K / p->KK;
    p->RB = (M + bm - 1) / bm;
    if (scheme == 0) {
        p->CB = (K + bk - 1) / bk;
        p->Pmax = bk;
        p->U = p->RB * K;
    } else {
        p->CB = (p->C + bk - 1) / bk;
        p->Pmax = p->KK;
        p->U = p->RB * p->CB * p->KK;
    }
    return OR_OK;
}

/* number of units in block (rb, cb) */
static int64_t block_units(const part_t *p, int64_t cb)
{
    if (p->scheme == 1) return p->KK;
    int64_t w = p->K - cb * p->bk;
    return w < p->bk ? w : p->bk;
}

/* linear unit index of unit u of block (rb, cb) */
static int64_t unit_index(const part_t *p, int64_t rb, int64_t cb, int64_t u)
{
    if (p->scheme == 0) return rb * p->K + cb * p->bk + u;   /* = rb*K + column */
    return (rb * p->CB + cb) * p->KK + u;
}

int64_t oracle_num_units(int scheme, int64_t M, int64_t K, int64_t kh, int64_t kw,
                         int64_t bm, int64_t bk)
{
    part_t p;
    if (make_part(&p, scheme, M, K, kh, kw, bm, bk)) return -1;
    return p.U;
}

/* Scores, Eq. (column) and Eq. (punched): the squared Frobenius norm of each
 * unit, accumulated in fp64.  Block-based: s = sum over the row-block's rows,
 * ascending, of W[r,j]^2.  Block-punched: s = sum over filters f ascending,
 * then channels c ascending, of W[f,c,pos]^2.  (A product of two 16-bit
 * floats is exact in fp64, so only the additions round, in this order.) */
int oracle_scores(int scheme, int dtype, int64_t M, int64_t K, int64_t kh, int64_t kw,
                  int64_t bm, int64_t bk, const uint16_t *W, double *scores)
{
    part_t p;
    int st = make_part(&p, scheme, M, K, kh, kw, bm, bk);
    if (st) return st;
    for (int64_t i = 0; i < M * K; ++i)
        if (!isfinite(oracle_half_to_double(W[i], dtype))) return OR_ERR_NONFINITE;
#pragma omp parallel for schedule(static)
    for (int64_t rb = 0; rb < p.RB; ++rb) {
        int64_t r0 = rb * p.bm, r1 = r0 + p.bm < M ? r0 + p.bm : M;
        for (int64_t cb = 0; cb < p.CB; ++cb) {
            int64_t P = block_units(&p, cb);
            for (int64_t u = 0; u < P; ++u) {
                double s = 0.0;
                if (p.scheme == 0) {
                    int64_t j = cb * p.bk + u;
                    for (int64_t r = r0; r < r1; ++r) {
                        double w = oracle_half_to_double(W[r * K + j], dtype);
                        s += w * w;
                    }
                } else {
                    int64_t c0 = cb * p.bk, c1 = c0 + p.bk < p.C ? c0 + p.bk : p.C;
                    for (int64_t f = r0; f < r1; ++f)
                        for (int64_t c = c0; c < c1; ++c) {
                            double w = oracle_half_to_double(W[f * K + c * p.KK + u], dtype);
                            s += w * w;
                        }
                }
                scores[unit_index(&p, rb, cb, u)] = s;
            }
        }
    }
    return OR_OK;
}

/* Reweighted group-Lasso regulariser of one layer (Eq. prob_block with
 * Eq. column for block-based and Eq. punched for block-punched blocks) and
 * its gradient with respect to W, the reweighting factors held fixed:
 *   s_u     = ||W_u||_F^2 over the unit's weights (as oracle_scores),
 *   alpha_u = 1 / (s_u + eps)                        (the reweighting rule),
 *   R       = lambda * sum_u ||alpha_u o W_u||_F^2 = lambda * sum_u alpha_u^2 s_u,
 *   dR/dW   = 2 lambda alpha_u^2 W  for every weight of unit u.
 * Reading: alpha_u is a scalar per unit, so "alpha o W_u" scales the unit and
 * its squared norm picks up alpha_u^2.  R is summed in unit order.  */
int oracle_reweighted_penalty(int scheme, int dtype, int64_t M, int64_t K, int64_t kh,
                              int64_t kw, int64_t bm, int64_t bk, const uint16_t *W, double eps,
                              double lambda, double *alpha, double *R, double *grad)
{
    part_t p;
    int st = make_part(&p, scheme, M, K, kh, kw, bm, bk);
    if (st) return st;
    if (!(eps > 0.0)) return OR_ERR_ARG;
    st = oracle_scores(scheme, dtype, M, K, kh, kw, bm, bk, W, alpha);
    if (st) return st;
    double r = 0.0;
    for (int64_t u = 0; u < p.U; ++u) {
        double s = alpha[u];
        alpha[u] = 1.0 / (s + eps);
        r += alpha[u] * alpha[u] * s;
    }
    *R = lambda * r;
#pragma omp parallel for schedule(static)
    for (int64_t f = 0; f < M; ++f) {
        int64_t rb = f / p.bm;
        for (int64_t k = 0; k < K; ++k) {
            int64_t u;
            if (p.scheme == 0) {
                u = rb * K + k;                                   /* (row-block, column) */
            } else {
                int64_t c = k / p.KK, pos = k % p.KK;               /* OIHW: k = c*KK + pos */
                u = unit_index(&p, rb, c / p.bk, pos);
            }
            double a = alpha[u];
            grad[f * K + k] = 2.0 * lambda * a * a * oracle_half_to_double(W[f * K + k], dtype);
        }
    }
    return OR_OK;
}

/* The same regulariser with the row groups of block-based pruning (Sec. 4.2,
 * Eq. row): the units are the rows of each bm x bk block, i.e. unit
 * u = r * CB + cb holds W[r, cb*bk .. min(cb*bk + bk, K) - 1], summed with k
 * ascending; alpha_u = 1 / (s_u + eps), R = lambda * sum_u alpha_u^2 s_u and
 * grad = 2 lambda alpha_u^2 W.  bm does not enter (a block's rows are its
 * groups); block-punched layouts have no row groups here (OR_ERR_ARG). */
int oracle_reweighted_penalty_rows(int dtype, int64_t M, int64_t K, int64_t bk,
                                   const uint16_t *W, double eps, double lambda, double *alpha,
                                   double *R, double *grad)
{
    if (M < 1 || K < 1 || bk < 1 || !(eps > 0.0)) return OR_ERR_ARG;
    const int64_t CB = (K + bk - 1) / bk;
    for (int64_t r = 0; r < M; ++r)
        for (int64_t cb = 0; cb < CB; ++cb) {
            double s = 0.0;
            for (int64_t k = cb * bk; k < K && k < cb * bk + bk; ++k) {
                double w = oracle_half_to_double(W[r * K + k], dtype);
                s += w * w;
            }
            alpha[r * CB + cb] = s;        /* the score; the factor below */
        }
    double sum = 0.0;
    for (int64_t u = 0; u < M * CB; ++u) {
        double s = alpha[u];
        alpha[u] = 1.0 / (s + eps);
        sum += alpha[u] * alpha[u] * s;
    }
    *R = lambda * sum;
    for (int64_t r = 0; r < M; ++r)
        for (int64_t k = 0; k < K; ++k) {
            double a = alpha[r * CB + k / bk];
            grad[r * K + k] = 2.0 * lambda * a * a * oracle_half_to_double(W[r * K + k], dtype);
        }
    return OR_OK;
}

/* Keep counts for a rate r >= 1 (Sec. 5.1 one-shot pruning at a set rate;
 * the rate is the parameter-reduction factor).  A block of P units keeps at
 * least base = floor(P / r); the layer keeps T = floor(sum P / r + 0.5) units
 * in total, and the E = T - sum(base) units left over go to the best
 * remaining units of the whole layer, so that the per-block rate may differ
 * (Sec. 4.1.1) while the layer's rate is the requested one. */
int oracle_counts(int scheme, int64_t M, int64_t K, int64_t kh, int64_t kw, int64_t bm,
                  int64_t bk, double rate, int64_t *sum_base, int64_t *total_keep,
                  int64_t *extras)
{
    part_t p;
    int st = make_part(&p, scheme, M, K, kh, kw, bm, bk);
    if (st) return st;
    if (!(rate >= 1.0) || !isfinite(rate)) return OR_ERR_ARG;
    int64_t sb = 0, sp = 0;
    for (int64_t rb = 0; rb < p.RB; ++rb)
        for (int64_t cb = 0; cb < p.CB; ++cb) {
            int64_t P = block_units(&p, cb);
            sb += (int64_t)floor((double)P / rate);
            sp += P;
        }
    int64_t T = (int64_t)floor((double)sp / rate + 0.5);
    *sum_base = sb; *total_keep = T; *extras = T - sb;
    return OR_OK;
}

typedef struct { double s; int64_t g; } cand_t;

/* higher score first; equal scores: lower unit index first */
static int cand_cmp(const void *a, const void *b)
{
    const cand_t *x = (const cand_t *)a, *y = (const cand_t *)b;
    if (x->s > y->s) return -1;
    if (x->s < y->s) return 1;
    return (x->g > y->g) - (x->g < y->g);
}

/* One-shot magnitude pruning by block (Sec. 4.1, Sec. 5.1): the units with the
 * largest squared norms survive.  Step 1: every block keeps its base
 * highest-scoring units.  Step 2: the E extra units are the highest-scoring
 * of all units not kept in step 1.  Ties go to the lower unit index.
 * Output: keep[g] in {0,1} per unit and the element mask M x K. */
int oracle_prune(int scheme, int dtype, int64_t M, int64_t K, int64_t kh, int64_t kw,
                 int64_t bm, int64_t bk, double rate, const uint16_t *W, uint8_t *keep,
                 uint8_t *mask)
{
    part_t p;
    int st = make_part(&p, scheme, M, K, kh, kw, bm, bk);
    if (st) return st;
    int64_t sb, T, E;
    st = oracle_counts(scheme, M, K, kh, kw, bm, bk, rate, &sb, &T, &E);
    if (st) return st;
    double *s = (double *)malloc((size_t)p.U * sizeof(double));
    cand_t *blk = (cand_t *)malloc((size_t)p.Pmax * sizeof(cand_t));
    cand_t *rest = (cand_t *)malloc((size_t)p.U * sizeof(cand_t));
    uint8_t *kp = keep ? keep : (uint8_t *)malloc((size_t)p.U);
    st = oracle_scores(scheme, dtype, M, K, kh, kw, bm, bk, W, s);
    if (st) goto done;
    memset(kp, 0, (size_t)p.U);
    int64_t nrest = 0;
    for (int64_t rb = 0; rb < p.RB; ++rb)
        for (int64_t cb = 0; cb < p.CB; ++cb) {
            int64_t P = block_units(&p, cb);
            int64_t base = (int64_t)floor((double)P / rate);
            for (int64_t u = 0; u < P; ++u) {
                int64_t g = unit_index(&p, rb, cb, u);
                blk[u].s = s[g]; blk[u].g = g;
            }
            qsort(blk, (size_t)P, sizeof(cand_t), cand_cmp);
            for (int64_t i = 0; i < P; ++i) {
                if (i < base) kp[blk[i].g] = 1;
                else rest[nrest++] = blk[i];
            }
        }
    qsort(rest, (size_t)nrest, sizeof(cand_t), cand_cmp);
    for (int64_t i = 0; i < E && i < nrest; ++i) kp[rest[i].g] = 1;
    /* element mask */
    if (mask) {
        for (int64_t r = 0; r < M; ++r) {
            int64_t rb = r / p.bm;
            for (int64_t k = 0; k < K; ++k) {
                int64_t g;
                if (p.scheme == 0) g = rb * K + k;
                else {
                    int64_t c = k / p.KK, pos = k % p.KK, cb = c / p.bk;
                    g = (rb * p.CB + cb) * p.KK + pos;
                }
                mask[r * K + k] = kp[g];
            }
        }
    }
done:
    free(s); free(blk); free(rest);
    if (!keep) free(kp);
    return st;
}

/* Row pruning of block-based layers (Sec. 4.1.1: rows and columns of each
 * block are pruned independently; Eq. row names the row groups).  The units
 * of block (rb, cb) are its rows r, i.e. the segments
 * W[r, cb*bk .. min(cb*bk + bk, K) - 1], scored by their squared norm in
 * fp64 with k ascending.  Counts as for column units: a block of P rows keeps
 * floor(P / rate) units, the layer keeps T = floor(M*CB / rate + 0.5) units,
 * and the T - sum(floor(P / rate)) extras go to the best remaining units of
 * the whole layer.  Units are numbered block-major and then by row,
 * g = rb*bm*CB + cb*rows_rb + (r - rb*bm) (rows_rb = real rows of rb), which is
 * also the tie order.  The row keep is ANDed into mask: an element survives
 * when its row unit survives and mask already held it (for example the column
 * mask of oracle_prune).  keep (optional, M*CB) receives the row-unit flags. */
int oracle_prune_rows(int dtype, int64_t M, int64_t K, int64_t bm, int64_t bk, double rate,
                      const uint16_t *W, uint8_t *keep, uint8_t *mask)
{
    if (M < 1 || K < 1 || bm < 1 || bk < 1) return OR_ERR_ARG;
    if (!(rate >= 1.0) || !isfinite(rate)) return OR_ERR_ARG;
    const int64_t RB = (M + bm - 1) / bm, CB = (K + bk - 1) / bk, U = M * CB;
    double *s = (double *)malloc((size_t)U * sizeof(double));
    cand_t *blk = (cand_t *)malloc((size_t)bm * sizeof(cand_t));
    cand_t *rest = (cand_t *)malloc((size_t)U * sizeof(cand_t));
    uint8_t *kp = keep ? keep : (uint8_t *)malloc((size_t)U);
    int st = OR_OK;
    memset(kp, 0, (size_t)U);
    int64_t nrest = 0, sum_base = 0;
    for (int64_t rb = 0; rb < RB; ++rb) {
        const int64_t r0 = rb * bm, rows = (r0 + bm <= M) ? bm : M - r0;
        for (int64_t cb = 0; cb < CB; ++cb) {
            const int64_t first = r0 * CB + cb * rows;
            for (int64_t i = 0; i < rows; ++i) {
                double acc = 0.0;
                for (int64_t k = cb * bk; k < K && k < cb * bk + bk; ++k) {
                    double w = oracle_half_to_double(W[(r0 + i) * K + k], dtype);
                    if (!isfinite(w)) { st = OR_ERR_NONFINITE; goto done; }
                    acc += w * w;
                }
                s[first + i] = acc;
                blk[i].s = acc; blk[i].g = first + i;
            }
            const int64_t base = (int64_t)floor((double)rows / rate);
            sum_base += base;
            qsort(blk, (size_t)rows, sizeof(cand_t), cand_cmp);
            for (int64_t i = 0; i < rows; ++i) {
                if (i < base) kp[blk[i].g] = 1;
                else rest[nrest++] = blk[i];
            }
        }
    }
    {
        const int64_t T = (int64_t)floor((double)U / rate + 0.5);
        const int64_t E = T - sum_base;
        qsort(rest, (size_t)nrest, sizeof(cand_t), cand_cmp);
        for (int64_t i = 0; i < E && i < nrest; ++i) kp[rest[i].g] = 1;
    }
    if (mask) {
        for (int64_t r = 0; r < M; ++r) {
            const int64_t rb = r / bm, r0 = rb * bm, rows = (r0 + bm <= M) ? bm : M - r0;
            for (int64_t k = 0; k < K; ++k) {
                const int64_t cb = k / bk;
                const int64_t g = r0 * CB + cb * rows + (r - r0);
                mask[r * K + k] = (uint8_t)(mask[r * K + k] && kp[g]);
            }
        }
    }
done:
    free(s); free(blk); free(rest);
    if (!keep) free(kp);
    return st;
}

/* Pattern-based pruning of 3x3 CONV layers (Sec. 2, pattern-based pruning:
 * kernel pattern pruning plus connectivity pruning), on the OIHW weight
 * (F filters, C channels, positions pos = 3i + j):
 *  - kernel pattern pruning: kernel (f, c) keeps the 4 positions of the
 *    pattern, among the npat given 9-bit masks (each with 4 bits set), whose
 *    kept squared norm (fp64, positions ascending) is largest; ties go to the
 *    lower pattern index;
 *  - connectivity pruning: of the F*C kernels, the T = floor(9 F C / (4 rate)
 *    + 0.5) with the largest kept norm survive (ties to the lower kernel index
 *    f*C + c), the others are removed whole; rate >= 9/4 is the
 *    parameter-reduction factor (9/4 keeps every kernel).
 * mask (F x 9C uint8) receives the element mask, pattern (optional, F*C) the
 * chosen pattern index of each kernel. */
int oracle_prune_pattern(int dtype, int64_t F, int64_t C, const uint16_t *patterns, int npat,
                         double rate, const uint16_t *W, uint8_t *pattern, uint8_t *mask)
{
    if (F < 1 || C < 1 || npat < 1 || npat > 255 || !(rate >= 2.25) || !isfinite(rate))
        return OR_ERR_ARG;
    for (int q = 0; q < npat; ++q) {
        int bits = 0;
        for (int b = 0; b < 9; ++b) bits += (patterns[q] >> b) & 1;
        if (bits != 4 || (patterns[q] >> 9)) return OR_ERR_ARG;
    }
    const int64_t U = F * C, K = 9 * C;
    cand_t *all = (cand_t *)malloc((size_t)U * sizeof(cand_t));
    uint8_t *pat = pattern ? pattern : (uint8_t *)malloc((size_t)U);
    int st = OR_OK;
    for (int64_t f = 0; f < F; ++f)
        for (int64_t c = 0; c < C; ++c) {
            double sq[9];
            for (int pos = 0; pos < 9; ++pos) {
                double w = oracle_half_to_double(W[f * K + c * 9 + pos], dtype);
                if (!isfinite(w)) { st = OR_ERR_NONFINITE; goto done; }
                sq[pos] = w * w;
            }
            double best = -1.0;
            int bq = 0;
            for (int q = 0; q < npat; ++q) {
                double e = 0.0;
                for (int pos = 0; pos < 9; ++pos)
                    if ((patterns[q] >> pos) & 1) e += sq[pos];
                if (e > best) { best = e; bq = q; }
            }
            pat[f * C + c] = (uint8_t)bq;
            all[f * C + c].s = best;
            all[f * C + c].g = f * C + c;
        }
    {
        const int64_t T = (int64_t)floor(9.0 * (double)U / (4.0 * rate) + 0.5);
        qsort(all, (size_t)U, sizeof(cand_t), cand_cmp);
        memset(mask, 0, (size_t)(F * K));
        for (int64_t i = 0; i < T && i < U; ++i) {
            const int64_t g = all[i].g, f = g / C, c = g % C;
            const uint16_t m = patterns[pat[g]];
            for (int pos = 0; pos < 9; ++pos)
                if ((m >> pos) & 1) mask[f * K + c * 9 + pos] = 1;
        }
    }
done:
    free(all);
    if (!pattern) free(pat);
    return st;
}

/* Compact storage (BCS, Sec. 4.3).  Because every row of a row-block keeps
 * the same columns, one column list serves the whole row-block (the
 * "occurrence" rows rb*bm .. rb*bm+bm_rb-1):
 *   rb_ptr[rb]      start of row-block rb's list in col_idx (RB+1 entries);
 *   col_idx[...]    kept column indices, ascending within a row-block;
 *   values[...]     row-block major, each row-block bm_rb x K'_rb row-major,
 *                   row-block rb starting at bm*rb_ptr[rb].
 * Returns OR_ERR_ARG if some row disagrees with the first row of its
 * row-block.  Pass NULL outputs to only count. */
int oracle_pack(int dtype, int64_t M, int64_t K, int64_t bm, const uint16_t *W,
                const uint8_t *mask, int64_t *rb_ptr, int32_t *col_idx, uint16_t *values,
                int64_t *nnz_cols, int64_t *nnz_vals)
{
    (void)dtype;
    if (M < 1 || K < 1 || bm < 1) return OR_ERR_ARG;
    int64_t RB = (M + bm - 1) / bm;
    int64_t nc = 0, nv = 0;
    for (int64_t rb = 0; rb < RB; ++rb) {
        int64_t r0 = rb * bm, r1 = r0 + bm < M ? r0 + bm : M;
        for (int64_t r = r0 + 1; r < r1; ++r)
            for (int64_t k = 0; k < K; ++k)
                if ((mask[r * K + k] != 0) != (mask[r0 * K + k] != 0)) return OR_ERR_ARG;
        if (rb_ptr) rb_ptr[rb] = nc;
        int64_t kp = 0;
        for (int64_t k = 0; k < K; ++k)
            if (mask[r0 * K + k]) {
                if (col_idx) col_idx[nc + kp] = (int32_t)k;
                ++kp;
            }
        if (values)
            for (int64_t r = r0; r < r1; ++r) {
                int64_t i = 0;
                for (int64_t k = 0; k < K; ++k)
                    if (mask[r0 * K + k])
                        values[bm * nc + (r - r0) * kp + (i++)] = W[r * K + k];
            }
        nc += kp;
        nv += (r1 - r0) * kp;
    }
    if (rb_ptr) rb_ptr[RB] = nc;
    if (nnz_cols) *nnz_cols = nc;
    if (nnz_vals) *nnz_vals = nv;
    return OR_OK;
}

/* Inverse of oracle_pack: rebuild the dense masked weight and the mask. */
int oracle_unpack(int64_t M, int64_t K, int64_t bm, const int64_t *rb_ptr,
                  const int32_t *col_idx, const uint16_t *values, uint16_t *W, uint8_t *mask)
{
    int64_t RB = (M + bm - 1) / bm;
    memset(W, 0, (size_t)(M * K) * sizeof(uint16_t));
    memset(mask, 0, (size_t)(M * K));
    for (int64_t rb = 0; rb < RB; ++rb) {
        int64_t r0 = rb * bm, r1 = r0 + bm < M ? r0 + bm : M;
        int64_t kp = rb_ptr[rb + 1] - rb_ptr[rb];
        for (int64_t r = r0; r < r1; ++r)
            for (int64_t i = 0; i < kp; ++i) {
                int64_t k = col_idx[rb_ptr[rb] + i];
                if (k < 0 || k >= K) return OR_ERR_ARG;
                W[r * K + k] = values[bm * rb_ptr[rb] + (r - r0) * kp + i];
                mask[r * K + k] = 1;
            }
    }
    return OR_OK;
}

/* Block-sparse layer output = dense product with the masked weight (pruned
 * weights contribute nothing, Sec. 4.3):
 *   acc[m,n] = sum over k ascending with mask[m,k]=1 of W[m,k]*X[k,n]  (fp64),
 *   y = acc + bias[m] (if bias), ReLU (if relu), rounded once to dtype.
 * X is K x N row-major with leading dimension ldx; Y is M x N with ldy.
 * acc_out (optional) receives the fp64 pre-rounding values, M x N dense. */
int oracle_masked_gemm(int dtype, int64_t M, int64_t K, int64_t N, const uint16_t *W,
                       const uint8_t *mask, const uint16_t *X, int64_t ldx, const float *bias,
                       int relu, uint16_t *Y, int64_t ldy, double *acc_out)
{
    if (M < 0 || K < 0 || N < 0 || ldx < N || ldy < N) return OR_ERR_ARG;
#pragma omp parallel
    {
        double *acc = (double *)malloc((size_t)(N > 0 ? N : 1) * sizeof(double));
#pragma omp for schedule(dynamic, 1)
        for (int64_t m = 0; m < M; ++m) {
            for (int64_t n = 0; n < N; ++n) acc[n] = 0.0;
            for (int64_t k = 0; k < K; ++k) {
                if (!mask[m * K + k]) continue;
                double w = oracle_half_to_double(W[m * K + k], dtype);
                const uint16_t *xr = X + k * ldx;
                for (int64_t n = 0; n < N; ++n) acc[n] += w * oracle_half_to_double(xr[n], dtype);
            }
            for (int64_t n = 0; n < N; ++n) {
                double v = acc[n];
                if (bias) v += (double)bias[m];
                if (relu && v < 0.0) v = 0.0;
                if (acc_out) acc_out[m * N + n] = v;
                if (Y) Y[m * ldy + n] = oracle_double_to_half(v, dtype);
            }
        }
        free(acc);
    }
    return OR_OK;
}

/* Masked direct convolution, NCHW input / OIHW weight / NCHW output, zero
 * padding, given stride (the CONV layer of Sec. 4.2 with its weight seen as
 * the F x (C*kh*kw) matrix whose column k = c*kh*kw + i*kw + j):
 *   acc[b,f,oh,ow] = sum over c, i, j ascending with mask[f,k]=1 of
 *                    W[f,c,i,j] * in[b,c,oh*sh+i-ph, ow*sw+j-pw]  (0 outside),
 *   then + bias[f], ReLU, one rounding to dtype. */
int oracle_masked_conv2d(int dtype, int64_t F, int64_t C, int64_t kh, int64_t kw,
                         const uint16_t *W, const uint8_t *mask, const uint16_t *in,
                         int64_t Nb, int64_t H, int64_t Wd, int64_t ph, int64_t pw, int64_t sh,
                         int64_t sw, const float *bias, int relu, uint16_t *out,
                         double *acc_out)
{
    if (F < 1 || C < 1 || kh < 1 || kw < 1 || Nb < 0 || sh < 1 || sw < 1 || ph < 0 || pw < 0)
        return OR_ERR_ARG;
    int64_t Ho = (H + 2 * ph - kh) / sh + 1, Wo = (Wd + 2 * pw - kw) / sw + 1;
    if (H + 2 * ph < kh || Wd + 2 * pw < kw) return OR_ERR_ARG;
    int64_t K = C * kh * kw;
#pragma omp parallel
    {
        double *acc = (double *)malloc((size_t)(Ho * Wo) * sizeof(double));
#pragma omp for schedule(dynamic, 1) collapse(2)
        for (int64_t b = 0; b < Nb; ++b)
            for (int64_t f = 0; f < F; ++f) {
                for (int64_t q = 0; q < Ho * Wo; ++q) acc[q] = 0.0;
                for (int64_t c = 0; c < C; ++c)
                    for (int64_t i = 0; i < kh; ++i)
                        for (int64_t j = 0; j < kw; ++j) {
                            int64_t k = c * kh * kw + i * kw + j;
                            if (!mask[f * K + k]) continue;
                            double w = oracle_half_to_double(W[f * K + k], dtype);
                            const uint16_t *plane = in + (b * C + c) * H * Wd;
                            for (int64_t oh = 0; oh < Ho; ++oh) {
                                int64_t ih = oh * sh + i - ph;
                                if (ih < 0 || ih >= H) continue;
                                for (int64_t ow = 0; ow < Wo; ++ow) {
                                    int64_t iw = ow * sw + j - pw;
                                    if (iw < 0 || iw >= Wd) continue;
                                    acc[oh * Wo + ow] +=
                                        w * oracle_half_to_double(plane[ih * Wd + iw], dtype);
                                }
                            }
                        }
                for (int64_t q = 0; q < Ho * Wo; ++q) {
                    double v = acc[q];
                    if (bias) v += (double)bias[f];
                    if (relu && v < 0.0) v = 0.0;
                    int64_t o = ((b * F + f) * Ho) * Wo + q;
                    if (acc_out) acc_out[o] = v;
                    if (out) out[o] = oracle_double_to_half(v, dtype);
                }
            }
        free(acc);
    }
    return OR_OK;
}

int oracle_max_threads(void)
{
#ifdef _OPENMP
    extern int omp_get_max_threads(void);
    return omp_get_max_threads();
#else
    return 1;
#endif
}

/* Threads of the parallel loops from now on (timing only: every loop's
 * result is the same for any thread count, each output element being
 * computed by one thread in a fixed order). */
void oracle_set_threads(int n)
{
#ifdef _OPENMP
    extern void omp_set_num_threads(int);
    if (n >= 1) omp_set_num_threads(n);
#else
    (void)n;
#endif
}
