/*
 * ultramem_oracle.h -- the CPU oracle of the UltraMem memory-layer forward.
 *
 * TEST INFRASTRUCTURE ONLY.  This is a plain, slow, fp64 statement of what the
 * layer computes, written from "Ultra-Sparse Memory Network" (Huang et al.,
 * ICLR 2025, arXiv 2411.12364).  Only the tests, the smoke check and the
 * benchmark's CPU-baseline leg may load it.  It shares no code, header, table
 * or helper with the CUDA library; neither includes or links the other.
 *
 * Every tensor is read in the precision it is stored in (fp32, or bf16 given
 * as raw uint16 bit patterns) and widened exactly to double.  All arithmetic
 * is fp64.  Where a floating-point score decides an index (the per-axis top-k
 * and the final top-m), the decision is taken on the score rounded to fp32,
 * the precision the GPU kernels decide in; ties go to the smaller index.
 *
 * Paper sections and equations cited below use the paper's own numbering:
 *   Eq. 1   generic memory layer          s = sigma(K q),  o = V^T s
 *   Eq. 2-3 product keys (PKM)            two-phase top-m, softmax pooling
 *           (score_mode UO_SCORE_PKM: additive grid score, exact two-phase)
 *   Eq. 4   row/column scores             S_row = K_row q_row, S_col = K_col q_col
 *   Eq. 5   Tucker grid score             S_grid = TopM(S_row^T C S_col)
 *   Eq. 6-7 rank-1 approximation          C ~ u t^T (leading singular pair)
 *   Eq. 8-9 per-axis pruning              I_TopM(u^T S_row), I_TopM(t^T S_col)
 *   Eq. 10  exact score on the survivors  TopM(S~_row^T C S~_col)
 *   Eq. 13  virtual blocks                V~_p = V W_p
 *   Eq. 14  shuffle of virtual addresses  s^ = Shuffle(vec(S_grid))
 *   Eq. 15  implicit value expansion      o = sum_p W_p^T (V^T s^_p)
 *   Eq. 16-17 Multi-Core Scoring (MCS)    C = sum_i C^(i); top-m on the
 *           aggregate S_row^T C S_col; physical value slice i (D_v/h wide)
 *           weighted by the individual score S_row^T C^(i) S_col
 *   Sec. 3.1 Trick 4  causal depthwise convolution of the input before the
 *           query linear: x~[t] = b + sum_j w_j (.) x[t - j], per channel
 *   Sec. 3.1 Trick 2  LayerNorm of each head's query (and of the keys, which
 *           at inference is a fixed transform of the key table: uo_key_ln)
 */
#ifndef ULTRAMEM_ORACLE_H
#define ULTRAMEM_ORACLE_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

enum { UO_F32 = 0, UO_BF16 = 1 };          /* storage type of the big tensors */
enum { UO_ACT_NONE = 0, UO_ACT_SOFTMAX = 1 }; /* Trick 1 removes the softmax   */
enum { UO_SCORE_TUCKER = 0, UO_SCORE_PKM = 1 }; /* grid score: Eq. 5 or Eq. 2   */

typedef struct {
    int32_t d_in;        /* D_i: width of the input hidden x                    */
    int32_t d_k;         /* D_k: query/key width of one head, D_k % r == 0      */
    int32_t heads;       /* H: key sets sharing one value table (Sec. 3.1)      */
    int32_t rank;        /* r: Tucker rank (Eq. 5)                              */
    int32_t n;           /* physical grid side; the table holds N = n*n rows    */
    int32_t expand_e;    /* E: virtual expansion, a perfect square (Eq. 13)     */
    int32_t d_v;         /* D_v: physical value width                           */
    int32_t d_out;       /* D'_v: virtual value width = output width            */
    int32_t topk;        /* k: survivors per axis (Eq. 8-9)                     */
    int32_t topm;        /* m: values read per head (Eq. 10)                    */
    int32_t has_proj;    /* 1: IVE projectors W_p present; 0 needs E == 1       */
    int32_t share_query; /* 1: one query for both key sets (Trick 5)            */
    int32_t act;         /* UO_ACT_NONE (Trick 1) or UO_ACT_SOFTMAX (PKM)       */
    int32_t dtype;       /* UO_F32 or UO_BF16 for x, W_q, keys, V, W_p          */
    int32_t cores;       /* h: component cores per head (MCS); 0 or 1 = one core.
                            h > 1 needs D_v % h == 0 and UO_ACT_NONE            */
    int32_t conv_k;      /* taps of the causal depthwise conv on x (Trick 4);
                            0 = no convolution                                  */
    int32_t query_ln;    /* 1: LayerNorm over each head's D_k query (Trick 2)   */
    int32_t score_mode;  /* UO_SCORE_TUCKER: S_row^T C S_col (TDQKR, Eq. 5, 10);
                            UO_SCORE_PKM: s_row[i] + s_col[j] (product keys,
                            Eq. 2-3), needs rank 1 and one core; no core read  */
    uint64_t shuffle_seed; /* 0: identity shuffle; else the seeded bijection   */
    double ln_eps;       /* LayerNorm epsilon (inside the square root)          */
} uo_config;

typedef struct {
    const void *x;        /* [B][d_in]                                           */
    const void *w_q;      /* [H*d_k][d_in]  q = W_q x, head h = rows h*d_k..     */
    const void *w_q_col;  /* [H*d_k][d_in] column query when share_query == 0   */
    const void *k_row;    /* [H][K][d_k], K = sqrt(E)*n keys per axis            */
    const void *k_col;    /* [H][K][d_k]                                         */
    const float *core;    /* [H][h][r][r] component cores C_h^(i), always fp32;
                             the Tucker core of head h is their sum            */
    const float *u;       /* [H][r] or NULL: leading left singular vectors       */
    const float *t;       /* [H][r] or NULL: leading right singular vectors      */
    const void *values;   /* [N][d_v] physical table V                           */
    const void *w_proj;   /* [E][d_v][d_out] projectors W_p, or NULL             */
    const int64_t *perm;  /* [E*N] explicit shuffle, or NULL for the seeded one  */
    /* query-side extras (read only when conv_k > 0 / query_ln == 1) */
    const float *conv_w;  /* [conv_k][d_in]: tap j multiplies x[t - j]            */
    const float *conv_b;  /* [d_in] or NULL                                       */
    const void *conv_state; /* [B/seq_len][conv_k-1][d_in], storage type: the
                             inputs before each sequence, oldest first; NULL =
                             zeros (every sequence starts fresh)                */
    int64_t seq_len;      /* tokens per sequence, the batch being B/seq_len
                             sequences back to back; 0 = one sequence of B      */
    const float *ln_g;    /* [A][H*d_k] query LayerNorm gain (A = 1 shared
                             query, 2 with a column query)                      */
    const float *ln_b;    /* [A][H*d_k] or NULL                                 */
} uo_tensors;

/* Status codes. */
enum { UO_OK = 0, UO_EINVAL = -1, UO_ENOMEM = -2 };

/* Full forward (Sec. 3.2, Eq. 4-10 then Eq. 13-15) for the tokens listed in
 * `tokens` (n_tokens entries, each in [0, B)); tokens == NULL means all B in
 * order.  Outputs are indexed by position in that list:
 *   out [n_tokens][d_out]   layer output o
 *   idx [n_tokens][H][m]    virtual address v = i*K + j of each selected slot,
 *                           ordered by (score desc, v asc); may be NULL
 *   w   [n_tokens][H][m][h] the weights applied to that slot, one per core
 *                           (slice of the value row); may be NULL
 * n_threads <= 0 uses the OpenMP default. */
int uo_forward(const uo_config *cfg, const uo_tensors *x, int64_t B,
               const int64_t *tokens, int64_t n_tokens,
               double *out, int64_t *idx, double *w, int32_t n_threads);

/* Eq. 5 (or Eq. 2 with PKM scoring) without the two-phase search: the top-m
 * of the whole K x K grid of each head, by brute force, in the order and tie
 * rule of uo_forward.  idx [n_tokens][H][m], w [n_tokens][H][m] (the grid
 * scores of the summed core, raw), either may be NULL.  Used to measure the
 * recall of the approximate search of Eq. 6-10. */
int uo_exact_topm(const uo_config *cfg, const uo_tensors *x, int64_t B, const int64_t *tokens,
                  int64_t n_tokens, int64_t *idx, double *w, int32_t n_threads);

/* Eq. 14-15 alone: pool the given (virtual address, weights) and project.
 * idx is [n_tokens][H][m], w [n_tokens][H][m][h]; only values, w_proj and
 * perm of `x` are read. */
int uo_lookup_reduce(const uo_config *cfg, const uo_tensors *x, int64_t n_tokens,
                     const int64_t *idx, const double *w, double *out,
                     int32_t n_threads);

/* The backward of Eq. 14-15 (the fused lookup-reduce of App. D), by the chain
 * rule on its definition.  For slots idx [n_tokens][H][m] with weights w
 * [n_tokens][H][m][h] and the gradient g = dL/do [n_tokens][d_out] (stored in
 * the config's type), with acc_p = sum_e w_e V[row_e] (block p) and
 * o = sum_p W_p^T acc_p:
 *   dacc_p = W_p g                       (g itself without a projector)
 *   dv[row][c]   += w_e^(slice c) dacc_{p_e}[c]        accumulated, [N][d_v]
 *   dw[e][i]      = sum_{c in slice i} dacc_{p_e}[c] V[row_e][c]   [n][H][m][h]
 *   dwp[p][c][o]  = sum_tokens acc_p[c] g[o]                       [E][d_v][d_out]
 * Any output may be NULL.  An address outside [0, E*N) is an error. */
int uo_lookup_reduce_backward(const uo_config *cfg, const uo_tensors *x, int64_t n_tokens,
                              const int64_t *idx, const double *w, const void *g, double *dv,
                              double *dw, double *dwp);

/* Eq. 4 for one (token b of a batch of B, head h): s_row[r][K], s_col[r][K]. */
int uo_row_col_scores(const uo_config *cfg, const uo_tensors *x, int64_t B, int64_t b,
                      int32_t h, double *s_row, double *s_col);

/* Leading singular triplet of an r x r matrix (row-major), Eq. 7 / Eq. 11.
 * Sign rule: sum(u) > 0, or if that sum is exactly 0 the first non-zero
 * entry of u is positive; t = C^T u / sigma.  Returns UO_OK. */
int uo_rank1(const double *c, int32_t r, double *u, double *t, double *sigma);

/* Trick 4: the conv state after the batch, [B/seq_len][conv_k-1][d_in] in
 * double: the last conv_k - 1 inputs of each sequence, oldest first (from the
 * previous state when a sequence is shorter than conv_k - 1). */
int uo_conv_state(const uo_config *cfg, const uo_tensors *x, int64_t B, double *state_out);

/* Trick 2 for keys: LayerNorm of each of n_rows rows of width d (stored in
 * `dtype`), gain g [d], bias b [d] or NULL, epsilon eps; out [n_rows][d]. */
int uo_key_ln(const void *keys, int32_t dtype, int64_t n_rows, int32_t d, const float *g,
              const float *b, double eps, double *out);

/* Eq. 14: the shuffled virtual address pi(v) for v in [0, E*N). */
int64_t uo_shuffle(const uo_config *cfg, const int64_t *perm, int64_t v);

/* The first output of a SplitMix64 generator whose state is `state`. */
uint64_t uo_splitmix64(uint64_t state);

/* The multiplier and offset of the seeded bijection pi(v) = (a v + c) mod M. */
void uo_shuffle_params(uint64_t seed, uint64_t m, uint64_t *a, uint64_t *c);

#ifdef __cplusplus
}
#endif
#endif
