/*
 * ultramem.h -- C ABI of the UltraMem memory-layer forward for GB300 (sm_103a).
 *
 * The layer is the one of "Ultra-Sparse Memory Network" (Huang et al., ICLR
 * 2025, arXiv 2411.12364), Sec. 3.2, inference forward only:
 *
 *   S1  q = W_q x                                  query projection, shared by the
 *                                                  row and column key sets (Trick 5)
 *   S2  S_row = K_row q, S_col = K_col q           Eq. 4, keys reshaped r x K x (D_k/r)
 *   S3  a = u^T S_row, b = t^T S_col               Eq. 6-7, (u, t) leading singular
 *                                                  pair of the Tucker core C
 *   S4  I = top-k(a), J = top-k(b)                 Eq. 8-9
 *   S5  g(i,j) = S_row[:,i]^T C S_col[:,j]         Eq. 10, only on I x J
 *   S6  top-m of g; weights = the raw scores       Eq. 10, Trick 1 (softmax removed)
 *   S7  v' = Shuffle(v), p = v' / N, row = v' % N  Eq. 14, v = i*K + j
 *   S8  acc[p] += w * V[row]                       Eq. 15, pooled per virtual block
 *   S9  o = sum_p W_p^T acc[p]                     Eq. 13/15 (IVE) + Trick 6 output
 *
 * Query-side extras (Sec. 3.1): with cfg.conv_k > 0 (Trick 4) the query input
 * is the causal depthwise convolution x~[t] = conv_b + sum_j conv_w[j] (.) x[t-j]
 * over the tokens of each sequence (the conv state supplies the inputs before
 * a sequence); with cfg.query_ln = 1 (Trick 2) each head's D_k-wide query is
 * layer-normalised (gain ln_g, bias ln_b, epsilon ln_eps) before S2.  The key
 * LayerNorm of Trick 2 is a fixed transform of the key table at inference:
 * ultramem_key_ln applies it once to stored keys.
 *
 * Multi-Core Scoring (Sec. 3.2, Eq. 16-17), when cfg.cores = h > 1: each head's
 * Tucker core is the sum of h component cores, C = sum_i C^(i).  S3-S6 run on
 * that sum; each selected slot then carries h weights, the individual scores
 * g_i(i,j) = S_row[:,i]^T C^(i) S_col[:,j], and weight i scales slice i (columns
 * i*D_v/h .. (i+1)*D_v/h - 1) of the physical value row in S8 (with IVE the
 * physical table is split, so Eq. 15 still holds per block).
 *
 * Shapes (all row-major and contiguous):
 *   K = sqrt(E) * n keys per axis (IVE grows each axis' key count by a factor
 *   sqrt(E), Sec. 3.2); N = n*n physical value rows; the virtual grid has
 *   K*K = E*N slots.  Heads share the value table and their pooled rows are summed.
 *
 * Conventions for every entry point:
 *   - Tensor pointers are DEVICE pointers unless a comment says HOST.  The
 *     layer borrows the caller's weights for its whole lifetime and never
 *     copies the value table; the caller keeps them alive and unchanged.
 *   - `stream` is a cudaStream_t passed as void* (NULL = legacy default
 *     stream).  Calls that take a stream are asynchronous on it.
 *   - Errors are returned as ultramem_status; nothing aborts, traps or throws.
 *     ULTRAMEM_EINVAL means the call was rejected before anything launched.
 *   - One layer handle must not be used by two calls at once (its workspace
 *     is shared); different handles are independent.
 */
#ifndef ULTRAMEM_H
#define ULTRAMEM_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum ultramem_status {
    ULTRAMEM_OK = 0,
    ULTRAMEM_EINVAL = -1,   /* invalid config, size or pointer; nothing launched    */
    ULTRAMEM_ENOMEM = -2,   /* a device or host allocation failed                    */
    ULTRAMEM_ECUDA = -3,    /* a CUDA runtime call or kernel launch failed           */
    ULTRAMEM_ETIMEOUT = -4, /* a bounded device-side wait gave up                    */
    ULTRAMEM_EDEVICE = -5,  /* a kernel's own check recorded an error (bad index)    */
    ULTRAMEM_ENODEV = -6    /* no CUDA device of compute capability 10.3             */
} ultramem_status;

enum { ULTRAMEM_F32 = 0, ULTRAMEM_BF16 = 1 };          /* storage of x, W_q, keys, V, W_p, out */
enum { ULTRAMEM_ACT_NONE = 0, ULTRAMEM_ACT_SOFTMAX = 1 }; /* Trick 1 vs PKM's softmax (Eq. 3)  */
enum { ULTRAMEM_SCORE_TUCKER = 0, ULTRAMEM_SCORE_PKM = 1 };   /* grid score: Eq. 5 or Eq. 2 */

/* Hyper-parameters of one layer, in the paper's notation. */
typedef struct ultramem_config {
    int32_t d_in;        /* D_i, width of x, <= 2^20                                 */
    int32_t d_k;         /* D_k, query/key width of one head; d_k % rank == 0, <= 4096 */
    int32_t heads;       /* H, key sets that read the shared table (Sec. 3.1), 1..64  */
    int32_t rank;        /* r, Tucker rank (Eq. 5), 1..8                              */
    int32_t n;           /* physical grid side, N = n*n rows; K = sqrt(E)*n <= 20480  */
    int32_t expand_e;    /* E, virtual expansion, a perfect square 1..16 (Eq. 13)    */
    int32_t d_v;         /* D_v, physical value width, multiple of 8                  */
    int32_t d_out;       /* D'_v, output width; == d_v when has_proj == 0             */
    int32_t topk;        /* k, survivors per axis (Eq. 8-9), 1..min(K, 128)           */
    int32_t topm;        /* m, slots read per head (Eq. 10), 1..min(k*k, 1024)        */
    int32_t has_proj;    /* 1: projectors W_p present; 0 requires E == 1              */
    int32_t share_query; /* 1: one query for both key sets (Trick 5); 0: W_q_col too  */
    int32_t act;         /* ULTRAMEM_ACT_NONE or ULTRAMEM_ACT_SOFTMAX                 */
    int32_t dtype;       /* ULTRAMEM_F32 or ULTRAMEM_BF16                              */
    int32_t max_tokens;  /* largest B any later call may pass; sizes the workspace    */
    int32_t cores;       /* h, component cores per head (MCS, Eq. 16-17): 0 or 1 = one
                            core; 2..8 needs act == ULTRAMEM_ACT_NONE and
                            (d_v / h) % 8 == 0                                        */
    int32_t conv_k;      /* taps of the causal depthwise query convolution (Trick 4),
                            0..64; 0 = none                                           */
    int32_t query_ln;    /* 1: LayerNorm of each head's query (Trick 2); d_k <= 256  */
    int32_t score_mode;  /* ULTRAMEM_SCORE_TUCKER: g(i,j) = S_row[:,i]^T C S_col[:,j]
                            (TDQKR, Eq. 5, 10); ULTRAMEM_SCORE_PKM: the product-key
                            memory's g(i,j) = s_row[i] + s_col[j] (Eq. 2-3), exact
                            two-phase search; needs rank 1 and one core, no core read */
    uint64_t shuffle_seed; /* Eq. 14 shuffle: 0 = identity, otherwise the seeded
                              bijection pi(v) = (a v + c) mod E*N whose a and c come
                              from the first two SplitMix64 outputs of the seed
                              (a = 1 + o1 mod (E*N - 1) stepped up to gcd(a, E*N) = 1,
                              c = o2 mod E*N); E*N must be < 2^32                     */
    float ln_eps;        /* query LayerNorm epsilon, >= 0 (inside the square root)   */
    int64_t shard_rows;  /* 0: `values` holds all N rows.  > 0: number-wise partition
                            of the table (App. D): `values` holds this rank's shard of
                            shard_rows (<= N) consecutive rows; the calls that read the
                            whole table (forward, lookup_reduce and its backward)
                            return ULTRAMEM_EINVAL, and the ultramem_shard_* calls
                            below serve the lookup                                   */
} ultramem_config;

/* The layer's parameters.  Device tensors are in the storage type cfg.dtype
 * (fp32, or bf16 as 16-bit words) unless noted. */
typedef struct ultramem_weights {
    const void *w_q;       /* [H*D_k][D_i]; head h owns rows h*D_k..h*D_k+D_k-1       */
    const void *w_q_col;   /* [H*D_k][D_i] column query when share_query == 0, else NULL */
    const void *k_row;     /* [H][K][D_k]; rank chunk alpha = columns alpha*D_k/r..    */
    const void *k_col;     /* [H][K][D_k]                                              */
    const float *core;     /* HOST fp32 [H][h][r][r] (h = max(1, cores)): component
                              cores C_h^(i), copied at create; C_h is their sum.  NULL
                              with ULTRAMEM_SCORE_PKM                                   */
    const float *u;        /* HOST fp32 [H][r] or NULL: leading left singular vectors  */
    const float *t;        /* HOST fp32 [H][r] or NULL (both or neither); when NULL
                              they are computed at create from the SVD of C_h (the sum
                              of the head's component cores) with the
                              sign rule sum(u) > 0 (first non-zero entry if the sum is 0) */
    const void *values;    /* [N][D_v], physical table V; 16-byte aligned              */
    const void *w_proj;    /* [E][D_v][D'_v] projectors W_p, or NULL when has_proj == 0 */
    const uint32_t *perm;  /* [E*N] explicit shuffle v -> v', or NULL for the seeded one */
    const float *conv_w;   /* fp32 [conv_k][D_i] when conv_k > 0: tap j multiplies the
                              input j tokens back (j = 0: the token itself), else NULL */
    const float *conv_b;   /* fp32 [D_i] convolution bias, or NULL                     */
    const float *ln_g;     /* fp32 [A][H*D_k] query LayerNorm gain when query_ln == 1
                              (A = 1 with share_query, 2 with a column query), else NULL */
    const float *ln_b;     /* fp32 [A][H*D_k] LayerNorm bias, or NULL                   */
} ultramem_weights;

typedef struct ultramem_layer ultramem_layer;

/* Validates cfg and weights, computes (u, t) if not given, derives the shuffle,
 * allocates the workspace for cfg.max_tokens tokens on the current device and
 * writes a new handle to *out.  Returns ULTRAMEM_EINVAL for an invalid config
 * (including a core whose leading singular value is 0 when u, t are NULL),
 * ULTRAMEM_ENOMEM if the workspace cannot be allocated, ULTRAMEM_ENODEV if the
 * current device is not compute capability 10.3. */
ultramem_status ultramem_create(const ultramem_config *cfg, const ultramem_weights *w,
                                ultramem_layer **out);

/* Frees the workspace and the handle; borrowed weights are untouched.  NULL is
 * a no-op.  Waits for work still queued on the layer's workspace. */
void ultramem_destroy(ultramem_layer *layer);

/* S1-S9 for B tokens: x [B][D_i] -> out [B][D'_v] (both cfg.dtype).  With a
 * query convolution the B tokens are one sequence with nothing before it
 * (ultramem_forward_seq gives the general case).  Optional
 * outputs (NULL to skip): idx_out [B][H][m] int64 virtual addresses v = i*K + j,
 * w_out [B][H][m][h] fp32 weights (h = max(1, cores): the slot's score, or its h
 * individual scores under MCS), each head's m slots ordered by (aggregate score
 * desc, v asc).  0 <= B <= max_tokens (B == 0 launches nothing). */
ultramem_status ultramem_forward(ultramem_layer *layer, const void *x, int32_t B,
                                 void *out, int64_t *idx_out, float *w_out, void *stream);

/* The forward on n_seq sequences of seq_len tokens each, back to back in x
 * [n_seq*seq_len][D_i] (B = n_seq*seq_len <= max_tokens); out, idx_out and w_out
 * as in ultramem_forward.  The query convolution (Trick 4) reaches back only
 * within a sequence and, before its first token, into conv_state_in
 * [n_seq][conv_k-1][D_i] (cfg.dtype, the inputs before each sequence, oldest
 * first; NULL = zeros).  conv_state_out (same shape, may be NULL) receives the
 * last conv_k-1 inputs of each sequence, reaching into conv_state_in when
 * seq_len < conv_k-1; it must not overlap conv_state_in.  Decode is seq_len = 1
 * with the states of the previous step.  Without a convolution the sequence
 * layout changes nothing and the states are ignored. */
ultramem_status ultramem_forward_seq(ultramem_layer *layer, const void *x, int32_t n_seq,
                                     int32_t seq_len, const void *conv_state_in,
                                     void *conv_state_out, void *out, int64_t *idx_out,
                                     float *w_out, void *stream);

/* The same forward on HOST buffers: moves x to the device, runs the forward
 * and moves out back, all on `stream`, and returns after the stream has
 * finished.  Page-locked (pinned, mapped) buffers that are 16-byte aligned are
 * moved by a copy kernel that reads and writes them over the host link;
 * other host memory (pageable works) by the copy engines. */
ultramem_status ultramem_forward_host(ultramem_layer *layer, const void *x_host, int32_t B,
                                      void *out_host, void *stream);

/* S1-S6 only (retrieval, Eq. 4-10): idx_out [B][H][m] int64 and w_out
 * [B][H][m][h] fp32 as in ultramem_forward; both required. */
ultramem_status ultramem_retrieve(ultramem_layer *layer, const void *x, int32_t B,
                                  int64_t *idx_out, float *w_out, void *stream);

/* Eq. 5 (Eq. 2 with ULTRAMEM_SCORE_PKM) without the approximate search: S1
 * (with the query extras), then the top-m of each head's whole K x K grid by
 * brute force, for measuring the recall of the two-phase search of Eq. 6-10.
 * idx_out [B][H][m] int64 and w_out [B][H][m] fp32 (raw grid scores of the
 * summed core, no activation), ordered as in ultramem_forward; both required.
 * Much slower than ultramem_retrieve (every grid score is computed several
 * times).  ULTRAMEM_EINVAL when the layer's chunk scores do not fit one CTA's
 * shared memory (K r > about 25000). */
ultramem_status ultramem_retrieve_exact(ultramem_layer *layer, const void *x, int32_t B,
                                        int64_t *idx_out, float *w_out, void *stream);

/* S7-S9 only (the lookup-reduce of Eq. 14-15) on given slots: idx [B][H][m]
 * int64 virtual addresses in [0, E*N), w [B][H][m][h] fp32 (weight i scales value
 * slice i, as in ultramem_forward) -> out [B][D'_v].  An
 * address out of range is not read: the kernel records it and the next
 * ultramem_check returns ULTRAMEM_EDEVICE. */
ultramem_status ultramem_lookup_reduce(ultramem_layer *layer, const int64_t *idx,
                                       const float *w, int32_t B, void *out, void *stream);

/* The backward of the lookup-reduce (S7-S9; App. D's fused lookup-reduce
 * operator) for the slots idx [B][H][m] int64 and weights w [B][H][m][h] fp32
 * of a forward, given g = dL/dout [B][D'_v] (cfg.dtype), all DEVICE:
 *   dvalues [N][D_v] fp32: += sum over slots of w_e (.) dacc_{p_e} at row_e,
 *           dacc_p = W_p g (g itself without projectors); accumulated, so zero
 *           it first for a fresh gradient; repeated rows add (fp32 atomics:
 *           the summation order is not fixed)
 *   dw      [B][H][m][h] fp32: dacc_{p_e} . V[row_e] over each value slice
 *   dw_proj [E][D_v][D'_v] fp32: sum over tokens of acc_p g^T (written; ignored
 *           without projectors)
 * Any output may be NULL.  Out-of-range addresses are skipped (their dw is 0)
 * and reported by ultramem_check.  ULTRAMEM_EINVAL when a value row is wider
 * than 32 16-byte vectors.  Asynchronous on `stream`. */
ultramem_status ultramem_lookup_reduce_backward(ultramem_layer *layer, const int64_t *idx,
                                                const float *w, const void *g, int32_t B,
                                                float *dvalues, float *dw, float *dw_proj,
                                                void *stream);

/* The lookup-reduce of ultramem_lookup_reduce (S7-S9) without a layer handle
 * and without allocating anything.  The paper has no counterpart: this entry
 * point exists for callers that cannot call cudaMalloc or create a layer -- a
 * host that owns the device allocator, runs inside a fixed memory budget, or
 * must not risk an allocation blocking or failing at this point.  Its scratch
 * is one 8 MiB array of static device memory that every GPU loading the
 * library holds until the process exits; a batch whose scratch would exceed
 * it is rejected with ULTRAMEM_EINVAL.  cfg: d_k, rank, topk, max_tokens are
 * ignored; heads, topm, n, expand_e, d_v, d_out, has_proj, dtype, cores and
 * shuffle_seed are used as in ultramem_create.  values [N][D_v] and w_proj
 * [E][D_v][D'_v] as in ultramem_weights (w_proj may be NULL when has_proj is
 * 0), perm optional; idx [B][H][m] int64 and w [B][H][m][h] fp32 as in
 * ultramem_lookup_reduce; out [B][D'_v].  Out-of-range addresses are skipped
 * (weight 0).  Asynchronous on `stream`.  The first call on a device looks up
 * the array's device address and sets a kernel attribute; make that first
 * call before any stream capture.  Every call shares the one array, so calls
 * that overlap on the GPU (other streams, other host threads) race and must
 * be ordered by the caller. */
ultramem_status ultramem_lookup_reduce_noalloc(const ultramem_config *cfg, const void *values,
                                               const void *w_proj, const uint32_t *perm,
                                               const int64_t *idx, const float *w, int32_t B,
                                               void *out, void *stream);

/* Synchronises `stream`, then reads and clears the layer's device error word:
 * ULTRAMEM_EDEVICE if a kernel recorded a bad index (or, never expected, a
 * selection position outside its grid, whose slot it then skipped),
 * ULTRAMEM_ETIMEOUT if a bounded wait gave up, ULTRAMEM_ECUDA if the stream
 * reports an error. */
ultramem_status ultramem_check(ultramem_layer *layer, void *stream);

/* Trick 2 for keys: LayerNorm of each of n_rows rows of width d (DEVICE, dtype
 * ULTRAMEM_F32 or ULTRAMEM_BF16) with gain g [d] and bias b [d] (DEVICE fp32, b
 * may be NULL) and epsilon eps, computed in fp32 and written to out (same type
 * and shape; out == keys works in place).  At inference the key LayerNorm is a
 * fixed transform of the key table: apply it once and create the layer with
 * the result.  Asynchronous on `stream`. */
ultramem_status ultramem_key_ln(const void *keys, int32_t dtype, int64_t n_rows, int32_t d,
                                const float *g, const float *b, float eps, void *out,
                                void *stream);

/* Leading singular triplet of one r x r core (HOST, row-major fp32) with the
 * sign rule above (Eq. 7; the SVD of Eq. 11).  ULTRAMEM_EINVAL if sigma == 0. */
ultramem_status ultramem_rank1(const float *core, int32_t r, float *u, float *t,
                               float *sigma);

/* Per-stage timing for profiling: while enabled, every forward (also one
 * captured in a CUDA graph and replayed) has its kernels record the GPU's
 * global timer: per stage, the moment its first CTA passed its dependency
 * wait and the moment its last warp finished.  The forward runs unchanged,
 * as programmatic dependent launches.  ultramem_profile_read (the caller
 * synchronises first) fills ms[0..5) with each stage's device time (last
 * end minus first start, in ms; -1 for a stage that did not run) and, when
 * n >= 10, ms[5..10) with the hand-off before each stage (from the end of
 * the previous stage to this stage's start; 0 for the first); it returns
 * the number of values written.  ultramem_stage_name names stage i (0 query
 * with the convolution and LayerNorm, 1 score, 2 select, 3 gather, 4
 * projection).  The timer advances in 256 ns steps on GB300, so average
 * over many forwards.  Disabled by default. */
ultramem_status ultramem_profile_enable(ultramem_layer *layer, int32_t enable);
int32_t ultramem_profile_read(ultramem_layer *layer, float *ms, int32_t n);
const char *ultramem_stage_name(int32_t i);

/* Number of CUDA kernels the most recent successful ultramem_forward,
 * ultramem_forward_host, ultramem_retrieve or ultramem_lookup_reduce call on
 * this layer launched (a CUDA graph captured from a call launches the same
 * kernels on every replay); 0 before the first call or for a NULL layer. */
int32_t ultramem_last_launches(const ultramem_layer *layer);

/* Text of the last CUDA error behind an ULTRAMEM_ECUDA or ULTRAMEM_ENOMEM
 * returned on the calling thread ("" if none). */
const char *ultramem_last_error(void);

/* Human-readable name of a status code. */
const char *ultramem_status_string(ultramem_status s);

/* Number-wise partition of the value table over P ranks (App. D: indices
 * all-to-all to the rows' owners, lookup there, rows all-to-all back, then
 * the weighted sum pooling on the requester): rank q holds rows
 * [q R, min((q + 1) R, N)), R = rows_per_rank = ceil(N / P), and each rank
 * selects its own tokens' slots (S1-S6 with the keys replicated,
 * ultramem_retrieve).  Then:
 *   1. ultramem_shard_route: the S = n*H*m addresses idx [n][H][m] (int64,
 *      DEVICE) are shuffled (Eq. 14) to physical rows and grouped by owner
 *      q = row / R: counts [P] (int32, DEVICE) of requests per owner;
 *      send_rows [S] (int32, DEVICE) the owners' local row indices, owner by
 *      owner (owner q's block starts at the sum of counts[0..q)); slot_pos [S]
 *      (int32, DEVICE) the position of slot s in send_rows.  The order inside
 *      an owner's block is not fixed; every later step reads through slot_pos,
 *      so the result is.  An address outside [0, E N) is recorded in the error
 *      word and requested as row 0 of owner 0 (its slot is then skipped).
 *   2. (caller) all-to-all of counts, then of send_rows: each rank receives
 *      the local rows the others request from it.
 *   3. ultramem_shard_lookup: out_rows[i] = the layer's shard row rows[i]
 *      ([n_rows][D_v], the storage type, DEVICE), a row outside the shard
 *      recorded in the error word and returned as zeros.
 *   4. (caller) all-to-all of the looked-up rows back to the requesters, in
 *      the order of their send_rows (back_rows [S][D_v]).
 *   5. ultramem_shard_pool: the weighted sum pooling of Eq. 15 and the IVE
 *      projection on the returned rows: slot s reads back_rows[slot_pos[s]]
 *      with weight w[s] (w like ultramem_lookup_reduce's) into its block;
 *      out [n][D'_v] as ultramem_lookup_reduce writes it.
 * All three are asynchronous on `stream`, work on layers created with or
 * without shard_rows, and return ULTRAMEM_EINVAL for invalid sizes or null
 * pointers (P in 1..1024, rows_per_rank * P >= N, n <= max_tokens). */
ultramem_status ultramem_shard_route(ultramem_layer *layer, const int64_t *idx, int32_t n,
                                     int32_t P, int64_t rows_per_rank, int32_t *counts,
                                     int32_t *send_rows, int32_t *slot_pos, void *stream);
ultramem_status ultramem_shard_lookup(ultramem_layer *layer, const int32_t *rows,
                                      int64_t n_rows, void *out_rows, void *stream);
ultramem_status ultramem_shard_pool(ultramem_layer *layer, const int64_t *idx, const float *w,
                                    int32_t n, const int32_t *slot_pos, const void *back_rows,
                                    void *out, void *stream);

/* Failure-path hooks for tests; they inject failures on the host or behind
 * a bounded wait, never a device fault.
 *
 * ultramem_debug_wait_probe: arms the layer's next forward (tensor-core
 * path, bf16 storage; ULTRAMEM_EINVAL for other layers) so that its scoring
 * kernel, after its dependency wait and before it issues any copy or MMA or
 * takes tensor memory, waits on an mbarrier that nothing signals, with a
 * limit of a few thousand SM cycles instead of the usual ~1 s.  The wait
 * gives up, the kernel records ULTRAMEM_ETIMEOUT in the layer's error word
 * and returns; the rest of that forward runs on stale scores and its output
 * is meaningless.  ultramem_check then returns ULTRAMEM_ETIMEOUT once; the
 * hook disarms itself after one forward.
 *
 * ultramem_debug_fail_alloc: the nth device allocation (0-based, counted
 * from this call, over all layers of the process) that the library makes
 * fails as if the device were out of memory, without calling the allocator;
 * a negative n disarms.  ultramem_debug_live_allocations returns how many
 * device allocations the library holds (every live layer's workspace), so a
 * test can check that a failed create releases everything it took. */
ultramem_status ultramem_debug_wait_probe(ultramem_layer *layer);
void ultramem_debug_fail_alloc(int32_t nth);
int32_t ultramem_debug_live_allocations(void);

/* The scoring's two forms (tensor-core path), for tests and measurement.
 * Mode 0: the scoring writes every rank-1 key (Eq. 6-7) and the selection
 * takes each axis' top k from all of them (Eq. 8-9).  Mode 1: the scoring
 * runs twice: the first pass keeps the largest key of each group of 16 keys
 * of an axis, a bound kernel takes tau <= the k-th largest of those per
 * (token, head, axis) (k distinct groups reach tau, so the axis' top k is
 * >= tau), and the second pass writes only the keys >= tau, as per-axis
 * candidate lists, which the selection ranks instead.  Mode 2 (the
 * default): mode 1 on long grids (at least 3.5 of the list passes' tiles of
 * 128 tokens x 256 keys per SM), mode 0 below; a layer that cannot take the
 * lists always scores every key.  All forms rank the same keys in the same
 * order (score, then the smaller index), so the selection is the same.
 * Mode 1 needs the tensor-core path and k to 1024 groups of 16 keys an axis
 * (ULTRAMEM_ENODEV otherwise, and the layer keeps its mode);
 * ULTRAMEM_EINVAL for another mode. */
ultramem_status ultramem_debug_candidates(ultramem_layer *layer, int32_t mode);

/* ABI version, currently 2. */
int32_t ultramem_version(void);

#ifdef __cplusplus
}
#endif
#endif /* ULTRAMEM_H */
