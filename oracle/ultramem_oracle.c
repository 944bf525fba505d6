/*
 * ultramem_oracle.c -- the CPU oracle of the UltraMem memory-layer forward.
 *
 * TEST INFRASTRUCTURE ONLY (tests, smoke check, CPU-baseline leg of the
 * benchmark).  Plain loops in fp64 that follow the paper's steps in its
 * order and notation; no blocking, fusion or reordering.  Shares no code with
 * the CUDA library.  See ultramem_oracle.h for the equation map.
 *
 * Readings of points the paper leaves open (each one is listed with its
 * justification in the design notes of the repository):
 *  - keys per axis K = sqrt(E) * n (Sec. 3.2 IVE: "the key size is expanded
 *    by sqrt(E) times"), physical rows N = n * n, virtual grid K*K = E*N;
 *  - the final top-m runs over the k*k surviving candidates only (Eq. 10);
 *  - ties in any top-k / top-m go to the smaller index (key index per axis,
 *    virtual address v = i*K + j for the grid);
 *  - heads are summed: all H*m weighted rows are pooled into one output;
 *  - virtual block p = v' div N, physical row = v' mod N where v' is the
 *    shuffled address (blocks concatenated in order, Eq. 13-14);
 *  - the shuffle is the seeded affine bijection documented at uo_shuffle;
 *  - Trick 4's convolution feeds the query linear directly (no activation);
 *    tap j multiplies the input j tokens back, within the token's sequence
 *    or from the state before it;
 *  - Trick 2's query LayerNorm runs over each head's D_k query entries
 *    (population variance, epsilon inside the square root), after the
 *    projection and before the key scores; a separate column query has its
 *    own gain and bias;
 *  - precision of the discrete decisions: every score is computed in fp64,
 *    but each top-k / top-m orders the scores rounded to fp32 (the `key` of
 *    `scored` below), with the value itself kept in fp64 for the weights.
 *    The paper fixes no precision for these decisions; fp32 is the
 *    precision the GPU kernels decide in, so a pair of scores that are
 *    equal in fp32 is ordered by the tie rule on both sides instead of by a
 *    difference below fp32 resolution that only the oracle sees.  Scores
 *    closer than 1e-5 relative are treated as near-ties by the parity
 *    tests, so this choice moves no test outcome outside that band.
 */
#include "ultramem_oracle.h"

#include <math.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

/* ---- reading stored tensors ------------------------------------------- */

/* Widen element i of a stored tensor to double.  bf16 is the top half of an
 * IEEE binary32, so the widening is exact. */
static double load(const void *p, int32_t dtype, int64_t i)
{
    if (dtype == UO_BF16) {
        uint32_t bits = (uint32_t)((const uint16_t *)p)[i] << 16;
        float f;
        memcpy(&f, &bits, sizeof f);
        return (double)f;
    }
    return (double)((const float *)p)[i];
}

static int64_t keys_per_axis(const uo_config *cfg)
{
    int64_t s = (int64_t)llround(sqrt((double)cfg->expand_e));
    return s * (int64_t)cfg->n;
}

static int check_config(const uo_config *cfg)
{
    if (!cfg) return UO_EINVAL;
    if (cfg->d_in <= 0 || cfg->d_k <= 0 || cfg->heads <= 0 || cfg->rank <= 0)
        return UO_EINVAL;
    if (cfg->d_k % cfg->rank != 0) return UO_EINVAL;
    if (cfg->n <= 0 || cfg->expand_e <= 0 || cfg->d_v <= 0) return UO_EINVAL;
    int64_t s = (int64_t)llround(sqrt((double)cfg->expand_e));
    if (s * s != cfg->expand_e) return UO_EINVAL;
    int64_t K = keys_per_axis(cfg);
    if (cfg->topk <= 0 || cfg->topk > K) return UO_EINVAL;
    if (cfg->topm <= 0 || (int64_t)cfg->topm > (int64_t)cfg->topk * cfg->topk)
        return UO_EINVAL;
    if (!cfg->has_proj && cfg->expand_e != 1) return UO_EINVAL;
    if (!cfg->has_proj && cfg->d_out != cfg->d_v) return UO_EINVAL;
    if (cfg->has_proj && cfg->d_out <= 0) return UO_EINVAL;
    if (cfg->dtype != UO_F32 && cfg->dtype != UO_BF16) return UO_EINVAL;
    if (cfg->act != UO_ACT_NONE && cfg->act != UO_ACT_SOFTMAX) return UO_EINVAL;
    if (cfg->cores < 0 || cfg->cores > 8) return UO_EINVAL;
    if (cfg->cores > 1 && (cfg->d_v % cfg->cores != 0 || cfg->act != UO_ACT_NONE))
        return UO_EINVAL;
    if (cfg->conv_k < 0 || cfg->conv_k > 64) return UO_EINVAL;
    if (cfg->query_ln != 0 && cfg->query_ln != 1) return UO_EINVAL;
    if (cfg->query_ln && !(cfg->ln_eps >= 0.0)) return UO_EINVAL;
    if (cfg->score_mode != UO_SCORE_TUCKER && cfg->score_mode != UO_SCORE_PKM) return UO_EINVAL;
    if (cfg->score_mode == UO_SCORE_PKM && (cfg->rank != 1 || cfg->cores > 1)) return UO_EINVAL;
    return UO_OK;
}

/* tokens per sequence of a batch of B (Trick 4) */
static int64_t seq_len_of(const uo_tensors *x, int64_t B) { return x->seq_len > 0 ? x->seq_len : B; }

/* h, the number of component cores of each head (Sec. 3.2, MCS) */
static int32_t cores_of(const uo_config *cfg) { return cfg->cores > 1 ? cfg->cores : 1; }

/* ---- Eq. 7 / Eq. 11: leading singular triplet of the Tucker core -------- */

/* Eigen-decomposition of a symmetric r x r matrix by cyclic Jacobi
 * rotations (Jacobi 1846; any numerical-analysis text).  a is destroyed;
 * column j of vec holds the eigenvector of eigenvalue a[j][j]. */
static void jacobi_eigen(double *a, int32_t r, double *vec)
{
    for (int32_t i = 0; i < r; ++i)
        for (int32_t j = 0; j < r; ++j) vec[i * r + j] = (i == j) ? 1.0 : 0.0;
    for (int sweep = 0; sweep < 100; ++sweep) {
        double off = 0.0, diag = 0.0;
        for (int32_t p = 0; p < r; ++p) {
            diag += a[p * r + p] * a[p * r + p];
            for (int32_t q = p + 1; q < r; ++q) off += a[p * r + q] * a[p * r + q];
        }
        if (off <= 1e-32 * diag || off == 0.0) break;
        for (int32_t p = 0; p < r; ++p) {
            for (int32_t q = p + 1; q < r; ++q) {
                double apq = a[p * r + q];
                if (apq == 0.0) continue;
                /* rotation angle that zeroes a[p][q]: tan = t */
                double theta = (a[q * r + q] - a[p * r + p]) / (2.0 * apq);
                double t = (theta >= 0.0 ? 1.0 : -1.0) /
                           (fabs(theta) + sqrt(theta * theta + 1.0));
                double c = 1.0 / sqrt(t * t + 1.0), s = t * c;
                for (int32_t k = 0; k < r; ++k) { /* columns p, q of a */
                    double akp = a[k * r + p], akq = a[k * r + q];
                    a[k * r + p] = c * akp - s * akq;
                    a[k * r + q] = s * akp + c * akq;
                }
                for (int32_t k = 0; k < r; ++k) { /* rows p, q of a */
                    double apk = a[p * r + k], aqk = a[q * r + k];
                    a[p * r + k] = c * apk - s * aqk;
                    a[q * r + k] = s * apk + c * aqk;
                }
                for (int32_t k = 0; k < r; ++k) { /* accumulate eigenvectors */
                    double vkp = vec[k * r + p], vkq = vec[k * r + q];
                    vec[k * r + p] = c * vkp - s * vkq;
                    vec[k * r + q] = s * vkp + c * vkq;
                }
            }
        }
    }
}

int uo_rank1(const double *c, int32_t r, double *u, double *t, double *sigma)
{
    if (!c || !u || !t || r <= 0) return UO_EINVAL;
    double *ctc = malloc(sizeof(double) * r * r);
    double *vec = malloc(sizeof(double) * r * r);
    if (!ctc || !vec) { free(ctc); free(vec); return UO_ENOMEM; }
    /* C^T C = T Lambda^2 T^T: its top eigenvector is the right singular
     * vector t, its eigenvalue sigma^2. */
    for (int32_t i = 0; i < r; ++i)
        for (int32_t j = 0; j < r; ++j) {
            double acc = 0.0;
            for (int32_t k = 0; k < r; ++k) acc += c[k * r + i] * c[k * r + j];
            ctc[i * r + j] = acc;
        }
    jacobi_eigen(ctc, r, vec);
    int32_t best = 0;
    for (int32_t j = 1; j < r; ++j)
        if (ctc[j * r + j] > ctc[best * r + best]) best = j;
    double lam = ctc[best * r + best];
    double sig = sqrt(lam > 0.0 ? lam : 0.0);
    if (!(sig > 0.0)) { free(ctc); free(vec); return UO_EINVAL; }
    for (int32_t j = 0; j < r; ++j) t[j] = vec[j * r + best];
    for (int32_t i = 0; i < r; ++i) { /* u = C t / sigma */
        double acc = 0.0;
        for (int32_t j = 0; j < r; ++j) acc += c[i * r + j] * t[j];
        u[i] = acc / sig;
    }
    /* sign rule: sum(u) > 0, else the first non-zero entry of u > 0 */
    double su = 0.0;
    for (int32_t i = 0; i < r; ++i) su += u[i];
    int flip = su < 0.0;
    if (su == 0.0) {
        for (int32_t i = 0; i < r; ++i)
            if (u[i] != 0.0) { flip = u[i] < 0.0; break; }
    }
    if (flip)
        for (int32_t i = 0; i < r; ++i) u[i] = -u[i];
    for (int32_t j = 0; j < r; ++j) { /* t = C^T u / sigma */
        double acc = 0.0;
        for (int32_t i = 0; i < r; ++i) acc += c[i * r + j] * u[i];
        t[j] = acc / sig;
    }
    *sigma = sig;
    free(ctc);
    free(vec);
    return UO_OK;
}

/* ---- Eq. 14: shuffle of virtual addresses ------------------------------- */

/* SplitMix64 output function (Steele, Lea and Flood, "Fast splittable
 * pseudorandom number generators", OOPSLA 2014). */
static uint64_t splitmix64(uint64_t state)
{
    uint64_t z = state + 0x9E3779B97F4A7C15ull;
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
    z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
    return z ^ (z >> 31);
}

uint64_t uo_splitmix64(uint64_t state) { return splitmix64(state); }

static uint64_t gcd_u64(uint64_t a, uint64_t b)
{
    while (b) { uint64_t r = a % b; a = b; b = r; }
    return a;
}

/* The paper shuffles the E*N virtual addresses at random (Eq. 14) and fixes
 * nothing more about the permutation.  Reading: pi(v) = (a*v + c) mod M with M = E*N, where
 * o1, o2 are the first two outputs of SplitMix64 seeded with `seed`:
 *   a = 1 + o1 mod (M-1), stepped up by one until gcd(a, M) = 1 (wrapping
 *       from M back to 1), which makes pi a bijection,
 *   c = o2 mod M;
 * seed 0 is the identity (a = 1, c = 0). */
void uo_shuffle_params(uint64_t seed, uint64_t m, uint64_t *a, uint64_t *c)
{
    if (seed == 0 || m <= 1) { *a = 1; *c = 0; return; }
    uint64_t aa = 1 + splitmix64(seed) % (m - 1);
    while (gcd_u64(aa, m) != 1) {
        aa += 1;
        if (aa >= m) aa = 1;
    }
    *a = aa;
    *c = splitmix64(seed + 0x9E3779B97F4A7C15ull) % m; /* second output */
}

int64_t uo_shuffle(const uo_config *cfg, const int64_t *perm, int64_t v)
{
    uint64_t m = (uint64_t)cfg->expand_e * (uint64_t)cfg->n * (uint64_t)cfg->n;
    if (perm) return perm[v];
    uint64_t a, c;
    uo_shuffle_params(cfg->shuffle_seed, m, &a, &c);
    /* M < 2^32 is required by the configuration check, so a*v < 2^64 */
    return (int64_t)(((uint64_t)a * (uint64_t)v + c) % m);
}

/* ---- top-k with the fp32 decision and the smaller-index tie rule ------- */

typedef struct { float key; int64_t index; double value; } scored;

static int by_score_desc_index_asc(const void *pa, const void *pb)
{
    const scored *a = pa, *b = pb;
    if (a->key > b->key) return -1;
    if (a->key < b->key) return 1;
    return (a->index < b->index) ? -1 : (a->index > b->index);
}

/* ---- Eq. 4: row and column scores of one head -------------------------- */

static void row_col_scores(const uo_config *cfg, const uo_tensors *x, int32_t h,
                           const double *q_row, const double *q_col,
                           double *s_row, double *s_col)
{
    const int64_t K = keys_per_axis(cfg);
    const int32_t r = cfg->rank, dk = cfg->d_k / cfg->rank, D = cfg->d_k;
    /* K_row, K_col in R^{r x n x (D_k/r)}: rank chunk alpha is columns
     * [alpha*D_k/r, (alpha+1)*D_k/r) of each stored key row. */
    for (int32_t al = 0; al < r; ++al)
        for (int64_t i = 0; i < K; ++i) {
            double sr = 0.0, sc = 0.0;
            int64_t base = ((int64_t)h * K + i) * D + (int64_t)al * dk;
            for (int32_t c = 0; c < dk; ++c) {
                sr += load(x->k_row, cfg->dtype, base + c) * q_row[al * dk + c];
                sc += load(x->k_col, cfg->dtype, base + c) * q_col[al * dk + c];
            }
            s_row[(int64_t)al * K + i] = sr;
            s_col[(int64_t)al * K + i] = sc;
        }
}

/* Input d of the token j positions before token b (j >= 0) of a batch of B:
 * from the same sequence, else from the state before it (zero without one). */
static double input_back(const uo_config *cfg, const uo_tensors *x, int64_t B, int64_t b,
                         int64_t j, int32_t d)
{
    const int64_t L = seq_len_of(x, B), s = b / L, pos = b - s * L - j;
    if (pos >= 0) return load(x->x, cfg->dtype, (b - j) * cfg->d_in + d);
    if (!x->conv_state) return 0.0;
    /* the state holds the conv_k - 1 inputs before position 0, oldest first */
    const int64_t row = (cfg->conv_k - 1) + pos;
    return load(x->conv_state, cfg->dtype, (s * (cfg->conv_k - 1) + row) * cfg->d_in + d);
}

/* The query's input row: x itself, or (Trick 4) its causal depthwise
 * convolution  x~[d] = b[d] + sum_j w[j][d] x[t - j][d]. */
static void query_input(const uo_config *cfg, const uo_tensors *x, int64_t B, int64_t b,
                        double *xin)
{
    for (int32_t d = 0; d < cfg->d_in; ++d) {
        if (cfg->conv_k == 0) {
            xin[d] = load(x->x, cfg->dtype, b * cfg->d_in + d);
            continue;
        }
        double acc = x->conv_b ? (double)x->conv_b[d] : 0.0;
        for (int32_t j = 0; j < cfg->conv_k; ++j)
            acc += (double)x->conv_w[(int64_t)j * cfg->d_in + d] * input_back(cfg, x, B, b, j, d);
        xin[d] = acc;
    }
}

/* q = W_q x for all heads; q has H*D_k entries.  With Trick 2, each head's
 * D_k entries are then layer-normalised with gain g and bias bb. */
static void query(const uo_config *cfg, const void *w, const double *xin, const float *g,
                  const float *bb, double *q)
{
    const int64_t rows = (int64_t)cfg->heads * cfg->d_k;
    for (int64_t o = 0; o < rows; ++o) {
        double acc = 0.0;
        for (int32_t d = 0; d < cfg->d_in; ++d)
            acc += load(w, cfg->dtype, o * cfg->d_in + d) * xin[d];
        q[o] = acc;
    }
    if (!cfg->query_ln) return;
    for (int32_t h = 0; h < cfg->heads; ++h) {
        double *qh = q + (int64_t)h * cfg->d_k;
        double mean = 0.0, var = 0.0;
        for (int32_t c = 0; c < cfg->d_k; ++c) mean += qh[c];
        mean /= cfg->d_k;
        for (int32_t c = 0; c < cfg->d_k; ++c) var += (qh[c] - mean) * (qh[c] - mean);
        var /= cfg->d_k;
        const double inv = 1.0 / sqrt(var + cfg->ln_eps);
        for (int32_t c = 0; c < cfg->d_k; ++c) {
            const int64_t o = (int64_t)h * cfg->d_k + c;
            qh[c] = (qh[c] - mean) * inv * (double)g[o] + (bb ? (double)bb[o] : 0.0);
        }
    }
}

/* Both queries of token b (Trick 5: the column keys share the row query). */
static void queries(const uo_config *cfg, const uo_tensors *x, int64_t B, int64_t b,
                    double *xin, double *q)
{
    const int64_t HD = (int64_t)cfg->heads * cfg->d_k;
    query_input(cfg, x, B, b, xin);
    query(cfg, x->w_q, xin, x->ln_g, x->ln_b, q);
    if (cfg->share_query) memcpy(q + HD, q, sizeof(double) * HD);
    else query(cfg, x->w_q_col, xin, x->ln_g ? x->ln_g + HD : NULL,
               x->ln_b ? x->ln_b + HD : NULL, q + HD);
}

/* Checks the query-side tensors a forward of B tokens reads. */
static int check_query_extras(const uo_config *cfg, const uo_tensors *x, int64_t B)
{
    if (cfg->conv_k > 0) {
        if (!x->conv_w || x->seq_len < 0) return UO_EINVAL;
        if (x->seq_len > 0 && B % x->seq_len != 0) return UO_EINVAL;
    }
    if (cfg->query_ln && !x->ln_g) return UO_EINVAL;
    return UO_OK;
}

int uo_conv_state(const uo_config *cfg, const uo_tensors *x, int64_t B, double *state_out)
{
    if (check_config(cfg) != UO_OK || !x || !x->x || !state_out || B <= 0) return UO_EINVAL;
    if (cfg->conv_k <= 0 || check_query_extras(cfg, x, B) != UO_OK) return UO_EINVAL;
    const int64_t L = seq_len_of(x, B), S = B / L, kk = cfg->conv_k - 1;
    for (int64_t s = 0; s < S; ++s)
        for (int64_t i = 0; i < kk; ++i)   /* row i holds input L - kk + i of sequence s */
            for (int32_t d = 0; d < cfg->d_in; ++d)
                state_out[(s * kk + i) * cfg->d_in + d] =
                    input_back(cfg, x, B, s * L + L - 1, kk - 1 - i, d);
    return UO_OK;
}

int uo_key_ln(const void *keys, int32_t dtype, int64_t n_rows, int32_t d, const float *g,
              const float *b, double eps, double *out)
{
    if (!keys || !g || !out || n_rows < 0 || d <= 0 || !(eps >= 0.0)) return UO_EINVAL;
    if (dtype != UO_F32 && dtype != UO_BF16) return UO_EINVAL;
    for (int64_t i = 0; i < n_rows; ++i) {
        double mean = 0.0, var = 0.0;
        for (int32_t c = 0; c < d; ++c) mean += load(keys, dtype, i * d + c);
        mean /= d;
        for (int32_t c = 0; c < d; ++c) {
            const double e = load(keys, dtype, i * d + c) - mean;
            var += e * e;
        }
        var /= d;
        const double inv = 1.0 / sqrt(var + eps);
        for (int32_t c = 0; c < d; ++c)
            out[i * d + c] = (load(keys, dtype, i * d + c) - mean) * inv * (double)g[c] +
                             (b ? (double)b[c] : 0.0);
    }
    return UO_OK;
}

int uo_row_col_scores(const uo_config *cfg, const uo_tensors *x, int64_t B, int64_t b,
                      int32_t h, double *s_row, double *s_col)
{
    if (check_config(cfg) != UO_OK || check_query_extras(cfg, x, B) != UO_OK) return UO_EINVAL;
    if (b < 0 || b >= B) return UO_EINVAL;
    const int64_t HD = (int64_t)cfg->heads * cfg->d_k;
    double *q = malloc(sizeof(double) * HD * 2);
    double *xin = malloc(sizeof(double) * cfg->d_in);
    if (!q || !xin) { free(q); free(xin); return UO_ENOMEM; }
    queries(cfg, x, B, b, xin, q);
    row_col_scores(cfg, x, h, q + (int64_t)h * cfg->d_k,
                   q + HD + (int64_t)h * cfg->d_k, s_row, s_col);
    free(q);
    free(xin);
    return UO_OK;
}

/* ---- Eq. 14-15: shuffled lookup, pooling per virtual block, projection -- */

/* acc[E][d_v] += w * V[row] for each selected slot; then out = sum_p W_p^T
 * acc[p] (or acc[0] when there is no projector). */
static void pool_and_project(const uo_config *cfg, const uo_tensors *x,
                             const int64_t *idx, const double *w, double *acc,
                             double *out)
{
    const int64_t N = (int64_t)cfg->n * cfg->n;
    const int32_t E = cfg->expand_e, Dv = cfg->d_v, Do = cfg->d_out;
    const int64_t hm = (int64_t)cfg->heads * cfg->topm;
    const int32_t nc = cores_of(cfg), slice = Dv / nc;
    memset(acc, 0, sizeof(double) * E * Dv);
    for (int64_t e = 0; e < hm; ++e) {
        int64_t vs = uo_shuffle(cfg, x->perm, idx[e]);
        int64_t p = vs / N, row = vs % N;
        /* MCS: element c of the row lies in slice c / (D_v/h), weighted by
         * that core's score (one slice, the plain weight, without MCS) */
        for (int32_t c = 0; c < Dv; ++c)
            acc[p * Dv + c] += w[e * nc + c / slice] * load(x->values, cfg->dtype, row * Dv + c);
    }
    if (!cfg->has_proj) {
        for (int32_t c = 0; c < Dv; ++c) out[c] = acc[c];
        return;
    }
    for (int32_t o = 0; o < Do; ++o) {
        double s = 0.0;
        for (int32_t p = 0; p < E; ++p)
            for (int32_t c = 0; c < Dv; ++c)
                s += load(x->w_proj, cfg->dtype, ((int64_t)p * Dv + c) * Do + o) *
                     acc[p * Dv + c];
        out[o] = s;
    }
}

int uo_lookup_reduce(const uo_config *cfg, const uo_tensors *x, int64_t n_tokens,
                     const int64_t *idx, const double *w, double *out,
                     int32_t n_threads)
{
    if (check_config(cfg) != UO_OK || !x || !idx || !w || !out) return UO_EINVAL;
    if (cfg->has_proj && !x->w_proj) return UO_EINVAL;
    const int64_t hm = (int64_t)cfg->heads * cfg->topm;
    const int64_t M = (int64_t)cfg->expand_e * cfg->n * cfg->n;
    for (int64_t e = 0; e < n_tokens * hm; ++e)
        if (idx[e] < 0 || idx[e] >= M) return UO_EINVAL;
    int status = UO_OK;
#ifdef _OPENMP
    if (n_threads > 0) omp_set_num_threads(n_threads);
#else
    (void)n_threads;
#endif
#pragma omp parallel
    {
        double *acc = malloc(sizeof(double) * cfg->expand_e * cfg->d_v);
        if (!acc) {
#pragma omp atomic write
            status = UO_ENOMEM;
        } else {
#pragma omp for schedule(dynamic, 1)
            for (int64_t b = 0; b < n_tokens; ++b)
                pool_and_project(cfg, x, idx + b * hm, w + b * hm * cores_of(cfg), acc,
                                 out + b * cfg->d_out);
        }
        free(acc);
    }
    return status;
}

/* ---- grid scores --------------------------------------------------------- */

/* The score of slot (i, j): Eq. 5's S_row[:,i]^T C S_col[:,j] (TDQKR), or
 * Eq. 2's s_row[i] + s_col[j] (product keys, rank 1). */
static double grid_score(const uo_config *cfg, const double *s_row, const double *s_col,
                         const double *C, int64_t K, int64_t i, int64_t j)
{
    if (cfg->score_mode == UO_SCORE_PKM) return s_row[i] + s_col[j];
    const int32_t r = cfg->rank;
    double g = 0.0;
    for (int32_t al = 0; al < r; ++al)
        for (int32_t be = 0; be < r; ++be)
            g += s_row[(int64_t)al * K + i] * C[al * r + be] * s_col[(int64_t)be * K + j];
    return g;
}

/* Each head's Tucker core, the sum of its component cores (MCS), in C. */
static void head_core(const uo_config *cfg, const uo_tensors *x, int32_t h, double *C)
{
    const int32_t r = cfg->rank, nc = cores_of(cfg);
    for (int32_t e = 0; e < r * r; ++e) {
        C[e] = 0.0;
        if (cfg->score_mode == UO_SCORE_PKM) continue;
        for (int32_t i = 0; i < nc; ++i) C[e] += (double)x->core[((int64_t)h * nc + i) * r * r + e];
    }
}

/* ---- backward of Eq. 14-15 (App. D's fused lookup-reduce) -------------- */

int uo_lookup_reduce_backward(const uo_config *cfg, const uo_tensors *x, int64_t n_tokens,
                              const int64_t *idx, const double *w, const void *g, double *dv,
                              double *dw, double *dwp)
{
    if (check_config(cfg) != UO_OK || !x || !x->values || !idx || !w || !g || n_tokens < 0)
        return UO_EINVAL;
    if (cfg->has_proj && !x->w_proj) return UO_EINVAL;
    const int32_t E = cfg->expand_e, Dv = cfg->d_v, Do = cfg->d_out, nc = cores_of(cfg);
    const int32_t slice = Dv / nc;
    const int64_t N = (int64_t)cfg->n * cfg->n, M = (int64_t)E * N;
    const int64_t hm = (int64_t)cfg->heads * cfg->topm;
    for (int64_t e = 0; e < n_tokens * hm; ++e)
        if (idx[e] < 0 || idx[e] >= M) return UO_EINVAL;
    double *acc = malloc(sizeof(double) * E * Dv), *dacc = malloc(sizeof(double) * E * Dv);
    if (!acc || !dacc) { free(acc); free(dacc); return UO_ENOMEM; }
    if (dwp) memset(dwp, 0, sizeof(double) * E * Dv * Do);
    for (int64_t b = 0; b < n_tokens; ++b) {
        /* dL/dacc_p = W_p dL/do (the output is acc_0 itself without a projector) */
        for (int32_t p = 0; p < E; ++p)
            for (int32_t c = 0; c < Dv; ++c) {
                double s = 0.0;
                if (!cfg->has_proj) s = load(g, cfg->dtype, b * Do + c);
                else
                    for (int32_t o = 0; o < Do; ++o)
                        s += load(x->w_proj, cfg->dtype, ((int64_t)p * Dv + c) * Do + o) *
                             load(g, cfg->dtype, b * Do + o);
                dacc[p * Dv + c] = s;
                acc[p * Dv + c] = 0.0;
            }
        for (int64_t e = 0; e < hm; ++e) {
            const int64_t slot = b * hm + e;
            const int64_t vs = uo_shuffle(cfg, x->perm, idx[slot]);
            const int64_t p = vs / N, row = vs % N;
            if (dw)
                for (int32_t i = 0; i < nc; ++i) dw[slot * nc + i] = 0.0;
            for (int32_t c = 0; c < Dv; ++c) {
                const int32_t sl = c / slice;
                const double we = w[slot * nc + sl], V = load(x->values, cfg->dtype, row * Dv + c);
                if (dv) dv[row * Dv + c] += we * dacc[p * Dv + c];
                if (dw) dw[slot * nc + sl] += dacc[p * Dv + c] * V;
                acc[p * Dv + c] += we * V;
            }
        }
        /* dL/dW_p[c][o] = sum over tokens of acc_p[c] dL/do[o] */
        if (dwp && cfg->has_proj)
            for (int32_t p = 0; p < E; ++p)
                for (int32_t c = 0; c < Dv; ++c)
                    for (int32_t o = 0; o < Do; ++o)
                        dwp[((int64_t)p * Dv + c) * Do + o] +=
                            acc[p * Dv + c] * load(g, cfg->dtype, b * Do + o);
    }
    free(acc);
    free(dacc);
    return UO_OK;
}

/* ---- the whole layer for one token ------------------------------------- */

typedef struct {
    double *q, *xin, *s_row, *s_col, *a, *bcol, *acc, *sel_w, *pool_w, *core;
    scored *axis, *cand;
    int64_t *sel_i, *sel_j, *sel_v;
} scratch;

static void token_forward(const uo_config *cfg, const uo_tensors *x, int64_t B, int64_t b,
                          const double *u_all, const double *t_all, scratch *sc,
                          double *out, int64_t *idx_out, double *w_out)
{
    const int64_t K = keys_per_axis(cfg);
    const int32_t H = cfg->heads, r = cfg->rank, k = cfg->topk, m = cfg->topm;
    const int64_t HD = (int64_t)H * cfg->d_k;

    /* query projection (Sec. 3.1; Trick 5 shares it between the key sets,
     * Trick 4 convolves its input, Trick 2 normalises it) */
    queries(cfg, x, B, b, sc->xin, sc->q);

    const int32_t nc = cores_of(cfg);
    for (int32_t h = 0; h < H; ++h) {
        const double *u = u_all + (int64_t)h * r, *t = t_all + (int64_t)h * r;
        /* the Tucker core is the sum of the head's component cores (MCS) */
        const float *Ci = x->core ? x->core + (int64_t)h * nc * r * r : NULL;
        double *C = sc->core;
        head_core(cfg, x, h, C);

        /* Eq. 4: S_row, S_col in R^{r x K} */
        row_col_scores(cfg, x, h, sc->q + (int64_t)h * cfg->d_k,
                       sc->q + HD + (int64_t)h * cfg->d_k, sc->s_row, sc->s_col);

        /* Eq. 6-7: rank-1 scores u^T S_row and t^T S_col */
        for (int64_t i = 0; i < K; ++i) {
            double ai = 0.0, bi = 0.0;
            for (int32_t al = 0; al < r; ++al) {
                ai += u[al] * sc->s_row[(int64_t)al * K + i];
                bi += t[al] * sc->s_col[(int64_t)al * K + i];
            }
            sc->a[i] = ai;
            sc->bcol[i] = bi;
        }

        /* Eq. 8-9: keep the top-k of each axis */
        for (int64_t i = 0; i < K; ++i) {
            sc->axis[i].key = (float)sc->a[i];
            sc->axis[i].index = i;
            sc->axis[i].value = sc->a[i];
        }
        qsort(sc->axis, (size_t)K, sizeof(scored), by_score_desc_index_asc);
        for (int32_t e = 0; e < k; ++e) sc->sel_i[e] = sc->axis[e].index;
        for (int64_t j = 0; j < K; ++j) {
            sc->axis[j].key = (float)sc->bcol[j];
            sc->axis[j].index = j;
            sc->axis[j].value = sc->bcol[j];
        }
        qsort(sc->axis, (size_t)K, sizeof(scored), by_score_desc_index_asc);
        for (int32_t e = 0; e < k; ++e) sc->sel_j[e] = sc->axis[e].index;

        /* Eq. 10: exact Tucker score S_row^T C S_col on the k*k survivors
         * (with product keys, Eq. 2's sum s_row + s_col) */
        int64_t ncand = 0;
        for (int32_t ei = 0; ei < k; ++ei)
            for (int32_t ej = 0; ej < k; ++ej) {
                int64_t i = sc->sel_i[ei], j = sc->sel_j[ej];
                const double g = grid_score(cfg, sc->s_row, sc->s_col, C, K, i, j);
                sc->cand[ncand].key = (float)g;
                sc->cand[ncand].index = i * K + j; /* virtual address v */
                sc->cand[ncand].value = g;
                ++ncand;
            }
        qsort(sc->cand, (size_t)ncand, sizeof(scored), by_score_desc_index_asc);

        /* Trick 1 uses the selected scores as weights; PKM softmaxes them
         * over the m selected slots (Eq. 3). */
        if (cfg->act == UO_ACT_SOFTMAX) {
            double mx = sc->cand[0].value, z = 0.0;
            for (int32_t e = 1; e < m; ++e)
                if (sc->cand[e].value > mx) mx = sc->cand[e].value;
            for (int32_t e = 0; e < m; ++e) z += exp(sc->cand[e].value - mx);
            for (int32_t e = 0; e < m; ++e)
                sc->sel_w[e] = exp(sc->cand[e].value - mx) / z;
        } else if (nc == 1) {
            for (int32_t e = 0; e < m; ++e) sc->sel_w[e] = sc->cand[e].value;
        } else {
            /* MCS: each selected slot's individual scores S_row^T C^(i) S_col */
            for (int32_t e = 0; e < m; ++e) {
                const int64_t i = sc->cand[e].index / K, j = sc->cand[e].index % K;
                for (int32_t ci = 0; ci < nc; ++ci) {
                    const float *Cc = Ci + (int64_t)ci * r * r;
                    double g = 0.0;
                    for (int32_t al = 0; al < r; ++al)
                        for (int32_t be = 0; be < r; ++be)
                            g += sc->s_row[(int64_t)al * K + i] * (double)Cc[al * r + be] *
                                 sc->s_col[(int64_t)be * K + j];
                    sc->sel_w[(int64_t)e * nc + ci] = g;
                }
            }
        }
        for (int32_t e = 0; e < m; ++e) {
            sc->sel_v[(int64_t)h * m + e] = sc->cand[e].index;
            if (idx_out) idx_out[(int64_t)h * m + e] = sc->cand[e].index;
            for (int32_t ci = 0; ci < nc; ++ci)
                if (w_out) w_out[((int64_t)h * m + e) * nc + ci] = sc->sel_w[(int64_t)e * nc + ci];
        }
        /* keep this head's weights next to its addresses for pooling */
        memcpy(sc->pool_w + (int64_t)h * m * nc, sc->sel_w, sizeof(double) * m * nc);
    }
    /* Eq. 14-15 over all heads' slots together (heads are summed) */
    pool_and_project(cfg, x, sc->sel_v, sc->pool_w, sc->acc, out);
}

int uo_forward(const uo_config *cfg, const uo_tensors *x, int64_t B,
               const int64_t *tokens, int64_t n_tokens, double *out,
               int64_t *idx, double *w, int32_t n_threads)
{
    if (check_config(cfg) != UO_OK || !x || !out || B < 0) return UO_EINVAL;
    if (!x->x || !x->w_q || !x->k_row || !x->k_col || !x->values) return UO_EINVAL;
    if (!x->core && cfg->score_mode != UO_SCORE_PKM) return UO_EINVAL;
    if (!cfg->share_query && !x->w_q_col) return UO_EINVAL;
    if (cfg->has_proj && !x->w_proj) return UO_EINVAL;
    if ((x->u == NULL) != (x->t == NULL)) return UO_EINVAL;
    if (check_query_extras(cfg, x, B) != UO_OK) return UO_EINVAL;
    uint64_t M = (uint64_t)cfg->expand_e * (uint64_t)cfg->n * (uint64_t)cfg->n;
    if (M >= (1ull << 32)) return UO_EINVAL;
    if (!tokens) n_tokens = B;
    for (int64_t e = 0; tokens && e < n_tokens; ++e)
        if (tokens[e] < 0 || tokens[e] >= B) return UO_EINVAL;

    const int32_t H = cfg->heads, r = cfg->rank;
    const int64_t K = keys_per_axis(cfg);
    const int64_t hm = (int64_t)H * cfg->topm;

    /* Eq. 7: (u, t) per head, given by the caller or from the SVD of C_h */
    double *u_all = malloc(sizeof(double) * H * r);
    double *t_all = malloc(sizeof(double) * H * r);
    double *cd = malloc(sizeof(double) * r * r);
    if (!u_all || !t_all || !cd) { free(u_all); free(t_all); free(cd); return UO_ENOMEM; }
    for (int32_t h = 0; h < H; ++h) {
        if (cfg->score_mode == UO_SCORE_PKM) {   /* r = 1: the axis scores themselves */
            u_all[h] = 1.0;
            t_all[h] = 1.0;
        } else if (x->u) {
            for (int32_t al = 0; al < r; ++al) {
                u_all[h * r + al] = x->u[h * r + al];
                t_all[h * r + al] = x->t[h * r + al];
            }
        } else {
            double sigma;
            head_core(cfg, x, h, cd);   /* the aggregate core (MCS) */
            if (uo_rank1(cd, r, u_all + h * r, t_all + h * r, &sigma) != UO_OK) {
                free(u_all); free(t_all); free(cd);
                return UO_EINVAL;
            }
        }
    }
    free(cd);

    int status = UO_OK;
#ifdef _OPENMP
    if (n_threads > 0) omp_set_num_threads(n_threads);
#else
    (void)n_threads;
#endif
#pragma omp parallel
    {
        scratch sc;
        int64_t kk = (int64_t)cfg->topk * cfg->topk;
        sc.q = malloc(sizeof(double) * 2 * H * cfg->d_k);
        sc.xin = malloc(sizeof(double) * cfg->d_in);
        sc.s_row = malloc(sizeof(double) * r * K);
        sc.s_col = malloc(sizeof(double) * r * K);
        sc.a = malloc(sizeof(double) * K);
        sc.pool_w = malloc(sizeof(double) * hm * cores_of(cfg));
        sc.core = malloc(sizeof(double) * r * r);
        sc.bcol = malloc(sizeof(double) * K);
        sc.acc = malloc(sizeof(double) * cfg->expand_e * cfg->d_v);
        sc.sel_w = malloc(sizeof(double) * cfg->topm * cores_of(cfg));
        sc.axis = malloc(sizeof(scored) * K);
        sc.cand = malloc(sizeof(scored) * kk);
        sc.sel_i = malloc(sizeof(int64_t) * cfg->topk);
        sc.sel_j = malloc(sizeof(int64_t) * cfg->topk);
        sc.sel_v = malloc(sizeof(int64_t) * hm);
        int ok = sc.q && sc.xin && sc.s_row && sc.s_col && sc.a && sc.bcol && sc.acc &&
                 sc.sel_w && sc.pool_w && sc.core && sc.axis && sc.cand && sc.sel_i &&
                 sc.sel_j && sc.sel_v;
        if (!ok) {
#pragma omp atomic write
            status = UO_ENOMEM;
        } else {
#pragma omp for schedule(dynamic, 1)
            for (int64_t e = 0; e < n_tokens; ++e) {
                int64_t b = tokens ? tokens[e] : e;
                token_forward(cfg, x, B, b, u_all, t_all, &sc, out + e * cfg->d_out,
                              idx ? idx + e * hm : NULL, w ? w + e * hm * cores_of(cfg) : NULL);
            }
        }
        free(sc.q); free(sc.xin); free(sc.s_row); free(sc.s_col); free(sc.a); free(sc.bcol);
        free(sc.acc); free(sc.sel_w); free(sc.pool_w); free(sc.core); free(sc.axis);
        free(sc.cand);
        free(sc.sel_i); free(sc.sel_j); free(sc.sel_v);
    }
    free(u_all);
    free(t_all);
    return status;
}

/* ---- Eq. 5 by brute force: the exact top-m of the whole grid ------------ */

/* a ranks before b: score (fp32 key) descending, then index ascending */
static int better(const scored *a, const scored *b)
{
    return a->key > b->key || (a->key == b->key && a->index < b->index);
}

/* Min-heap of the m best so far (the root is the worst kept). */
static void heap_sift_down(scored *hp, int32_t n, int32_t i)
{
    for (;;) {
        int32_t l = 2 * i + 1, r = l + 1, w = i;
        if (l < n && better(&hp[w], &hp[l])) w = l;
        if (r < n && better(&hp[w], &hp[r])) w = r;
        if (w == i) return;
        scored t = hp[i]; hp[i] = hp[w]; hp[w] = t;
        i = w;
    }
}

static void heap_push(scored *hp, int32_t *n, int32_t cap, scored c)
{
    if (*n < cap) {   /* sift up */
        int32_t i = (*n)++;
        hp[i] = c;
        while (i > 0) {
            int32_t p = (i - 1) / 2;
            if (!better(&hp[p], &hp[i])) break;
            scored t = hp[i]; hp[i] = hp[p]; hp[p] = t;
            i = p;
        }
    } else if (better(&c, &hp[0])) {
        hp[0] = c;
        heap_sift_down(hp, *n, 0);
    }
}

int uo_exact_topm(const uo_config *cfg, const uo_tensors *x, int64_t B, const int64_t *tokens,
                  int64_t n_tokens, int64_t *idx, double *w, int32_t n_threads)
{
    if (check_config(cfg) != UO_OK || !x || B < 0) return UO_EINVAL;
    if (!x->x || !x->w_q || !x->k_row || !x->k_col) return UO_EINVAL;
    if (!x->core && cfg->score_mode != UO_SCORE_PKM) return UO_EINVAL;
    if (!cfg->share_query && !x->w_q_col) return UO_EINVAL;
    if (check_query_extras(cfg, x, B) != UO_OK) return UO_EINVAL;
    if (!tokens) n_tokens = B;
    for (int64_t e = 0; tokens && e < n_tokens; ++e)
        if (tokens[e] < 0 || tokens[e] >= B) return UO_EINVAL;
    const int32_t H = cfg->heads, r = cfg->rank, m = cfg->topm;
    const int64_t K = keys_per_axis(cfg), HD = (int64_t)H * cfg->d_k;
    int status = UO_OK;
#ifdef _OPENMP
    if (n_threads > 0) omp_set_num_threads(n_threads);
#else
    (void)n_threads;
#endif
#pragma omp parallel
    {
        double *q = malloc(sizeof(double) * 2 * HD), *xin = malloc(sizeof(double) * cfg->d_in);
        double *s_row = malloc(sizeof(double) * r * K), *s_col = malloc(sizeof(double) * r * K);
        double *C = malloc(sizeof(double) * r * r);
        scored *hp = malloc(sizeof(scored) * m);
        if (!q || !xin || !s_row || !s_col || !C || !hp) {
#pragma omp atomic write
            status = UO_ENOMEM;
        } else {
#pragma omp for schedule(dynamic, 1)
            for (int64_t e = 0; e < n_tokens; ++e) {
                const int64_t b = tokens ? tokens[e] : e;
                queries(cfg, x, B, b, xin, q);
                for (int32_t h = 0; h < H; ++h) {
                    head_core(cfg, x, h, C);
                    row_col_scores(cfg, x, h, q + (int64_t)h * cfg->d_k,
                                   q + HD + (int64_t)h * cfg->d_k, s_row, s_col);
                    int32_t n = 0;
                    for (int64_t i = 0; i < K; ++i)
                        for (int64_t j = 0; j < K; ++j) {
                            scored c;
                            c.value = grid_score(cfg, s_row, s_col, C, K, i, j);
                            c.key = (float)c.value;
                            c.index = i * K + j;
                            heap_push(hp, &n, m, c);
                        }
                    qsort(hp, (size_t)n, sizeof(scored), by_score_desc_index_asc);
                    for (int32_t t = 0; t < m; ++t) {
                        const int64_t o = (e * H + h) * m + t;
                        if (idx) idx[o] = hp[t].index;
                        if (w) w[o] = hp[t].value;
                    }
                }
            }
        }
        free(q); free(xin); free(s_row); free(s_col); free(C); free(hp);
    }
    return status;
}
