// ultramem.cu -- the C ABI declared in include/ultramem.h: validation, the
// create-time SVD and shuffle parameters, workspace ownership, the launch
// sequence of one forward, per-stage profiling and the device error word.
#include <math.h>
#include <stdio.h>
#include <stdlib.h>
#include <string.h>

#include <atomic>
#include <new>

#include "um_internal.cuh"

using um::Dims;
using um::Ptrs;

namespace {

constexpr int kStages = 5;
const char *const kStageNames[kStages] = {"query", "score", "select", "gather", "project"};

struct Workspace {
    float *q_part = nullptr, *sel_w = nullptr, *acc = nullptr, *proj_part = nullptr;
    uint32_t *akey = nullptr;   // the rank-1 keys [B][H][2][K], or (Dims::cand) the
                                // candidate lists [B][H][2][16 G] u64 in the same space
    uint32_t *gstat = nullptr, *tau = nullptr;   // candidate lists: group maxima / counts, bounds
    int32_t *sel_row = nullptr, *sel_p = nullptr;
    float *core = nullptr, *u = nullptr, *t = nullptr;
    float *cores = nullptr;   // MCS component cores [H][h][r][r] (h > 1 only)
    int *err = nullptr;
    void *x_stage = nullptr, *out_stage = nullptr;
    void *xs = nullptr;   // the convolved query input (Trick 4)
    float *dacc = nullptr;   // backward: dL/dacc [B][E*D_v]
    __nv_bfloat16 *bwd_t = nullptr;   // backward (tensor cores): acc^T [E*D_v][2 B] (two
                                      // bf16 terms), g^T [D'_v][B]
    __nv_bfloat16 *qs = nullptr, *acc_bf = nullptr, *w_pt = nullptr;   // tensor path
    unsigned long long *stamps = nullptr;   // profiling: [kStampStages] begins, then ends
    int *shard_cursor = nullptr;            // ultramem_shard_route: [1024] per-owner cursors
};

}  // namespace

struct ultramem_layer {
    ultramem_config cfg;
    ultramem_weights w;
    int device;
    Dims base;           // every field but B, q_splits, p_splits
    Workspace ws;
    bool tc = false;     // bf16 tensor-core path (tcgen05) for S1, S2, S9
    um::TcMaps maps;     // weight descriptors of the tensor path
    bool profiling = false;
    bool profiled_once = false;
    int launches = 0;    // kernels launched by the most recent successful call
    bool exact_ok = false;   // the brute-force top-m fits this layer's grid
    bool backward_ok = false;   // the lookup-reduce backward fits this layer
    // ultramem_forward_host on mapped pinned buffers: one CUDA graph per
    // (batch, input, output) holding the two copy kernels and the forward,
    // captured on the first call and replayed after (a few, replaced in turn)
    struct HostGraph {
        int B = 0;
        const void *x = nullptr;
        void *o = nullptr;
        cudaGraphExec_t exec = nullptr;
        int launches = 0;
    };
    static constexpr int kHostGraphs = 16;
    HostGraph host_graphs[kHostGraphs];
    int host_graph_next = 0;
    cudaStream_t capture = nullptr;
    bool x_after_copy = false;   // x is written by the copy kernel just before the forward
    bool probe_armed = false;    // ultramem_debug_wait_probe: the next forward's score probes
    bool cand_ok = false;        // the candidate-list scoring fits this layer
    int cand_mode = 2;           // ultramem_debug_candidates: 0 every key, 1 candidate lists,
                                 // 2 (default) lists on long grids
    bool dacc_tc = false;        // the backward's dacc may run on the tensor cores
};

// A layer over a shard of the table (number-wise partition) serves only the
// calls that do not read the whole table.
static bool whole_table(const ultramem_layer *L) { return L->cfg.shard_rows == 0; }

namespace {

int64_t keys_per_axis(const ultramem_config &c) {
    int s = (int)lround(sqrt((double)c.expand_e));
    return (int64_t)s * c.n;
}

size_t elt_size(const ultramem_config &c) { return c.dtype == ULTRAMEM_BF16 ? 2 : 4; }

// Split counts of the two split-K contractions for a given batch: enough CTAs
// to cover the 152 SMs about twice, each split at least 64 deep.
int query_splits(const ultramem_config &c, int B) {
    int tiles = ((c.heads * c.d_k + 63) / 64) * ((B + 31) / 32) * (c.share_query ? 1 : 2);
    int s = (304 + tiles - 1) / tiles;
    int cap = c.d_in / 64 > 0 ? c.d_in / 64 : 1;
    if (s > 8) s = 8;
    if (s > cap) s = cap;
    return s < 1 ? 1 : s;
}

// Batches up to this many tokens run the query projection (S1) on CUDA
// cores (16 weight rows x 8 tokens per CTA, no split-K); larger ones, and
// the IVE projection at every batch, on tcgen05.  Measured on GB300: at 64
// tokens the CUDA-core query takes 3.3 us against 8.5 us for the split-K
// tensor-core one; above that (and for the projection, whose weight rows
// it re-reads once per 8 tokens) it is slower: 12.4 against 9.6 us at 96
// tokens of the 4M-slot layer (D_i 2048), 15.4 against 9.7 us at 128.
constexpr int kSmallQueryBatch = 64;

// Tensor path split-K plan: the N tile (tokens per tile) and the split count
// of a contraction of m_rows weight rows over B tokens and kdim.  About
// `target` CTAs stream the weight: with one tile of up to 256 tokens, at
// most one portable cluster (8) of whole K blocks per tile; when that grid
// is still short of the target, the token tile is halved (down to `nt_min`),
// so that a batch of 128 tokens over 4 weight tiles runs 128 CTAs instead
// of 32.
struct TcPlan {
    int n_tile, splits;
};
TcPlan tc_plan(int m_rows, int B, int kdim, int target, int max_splits, int nt_min) {
    const int m_tiles = (m_rows + 127) / 128;
    const int kb = (kdim + 63) / 64;
    int nt = um::tc_n_tile(B, 1);
    for (;;) {
        const int n_tiles = (B + nt - 1) / nt;
        int s = (target + m_tiles * n_tiles - 1) / (m_tiles * n_tiles);
        if (s > max_splits) s = max_splits;
        if (s > kb) s = kb;
        if (s < 1) s = 1;
        // a split tile's partial slices stay within shared memory: at most
        // 128 tokens when split
        if ((m_tiles * n_tiles * s >= target || nt <= nt_min) && (s == 1 || nt <= 128))
            return {nt, s};
        nt = (nt / 2 + 15) / 16 * 16;
    }
}
// Measured on GB300 (stage times of graph-replayed forwards; mid_4m at 128
// tokens, large_20m at 256): the query is fastest with about 128 CTAs, eight
// splits and token tiles down to 32 (11.1 against 16.6 us with one 128-token
// tile, 12.2 against 23.0 us at 256 tokens).  The IVE projection, whose B
// operand (two bf16 terms of the pooled rows) grows with the batch, keeps
// about 64 CTAs of up to eight splits up to 64 tokens; above, about 128 CTAs
// of at most four splits with token tiles down to 64 (6.9 against 9.5 us at
// 128 tokens, 9.6 against 15.4 us at 256).
TcPlan tc_query_plan(const ultramem_config &c, int B) {
    return tc_plan(c.heads * c.d_k, B, c.d_in, 128, 8, 32);
}
TcPlan tc_proj_plan(const ultramem_config &c, int B) {
    if (!c.has_proj) return {um::tc_n_tile(B, 1), 1};
    if (B <= 64) return tc_plan(c.d_out, B, c.expand_e * c.d_v, 64, 8, 256);
    return tc_plan(c.d_out, B, c.expand_e * c.d_v, 128, 4, 64);
}
int tc_query_splits(const ultramem_config &c, int B) { return tc_query_plan(c, B).splits; }
int tc_proj_splits(const ultramem_config &c, int B) { return tc_proj_plan(c, B).splits; }

// The tensor path needs bf16 storage and 16-byte rows for TMA (D_in, D_k and
// E*D_v multiples of 8 elements).
bool tc_eligible(const ultramem_config &c) {
    return c.dtype == ULTRAMEM_BF16 && c.d_in % 8 == 0 && (c.expand_e * c.d_v) % 8 == 0 &&
           c.d_k % 8 == 0;
}

int proj_splits(const ultramem_config &c, int B) {
    if (!c.has_proj) return 1;
    int tiles = ((c.d_out + 63) / 64) * ((B + 31) / 32);
    int s = (304 + tiles - 1) / tiles;
    int kd = c.expand_e * c.d_v;
    int cap = kd / 64 > 0 ? kd / 64 : 1;
    if (s > 8) s = 8;
    if (s > cap) s = cap;
    return s < 1 ? 1 : s;
}

ultramem_status validate(const ultramem_config *c, const ultramem_weights *w) {
    if (!c || !w) return ULTRAMEM_EINVAL;
    if (c->cores < 0 || c->cores > 8) return ULTRAMEM_EINVAL;
    if (c->cores > 1 && (c->act != ULTRAMEM_ACT_NONE || c->d_v % (8 * c->cores)))
        return ULTRAMEM_EINVAL;   // MCS: raw scores, value slices of whole 16-byte words
    if (c->conv_k < 0 || c->conv_k > 64 || (c->conv_k > 0 && !w->conv_w)) return ULTRAMEM_EINVAL;
    if (c->score_mode != ULTRAMEM_SCORE_TUCKER && c->score_mode != ULTRAMEM_SCORE_PKM)
        return ULTRAMEM_EINVAL;
    const bool pkm = c->score_mode == ULTRAMEM_SCORE_PKM;
    if (pkm && (c->rank != 1 || c->cores > 1)) return ULTRAMEM_EINVAL;
    if (c->query_ln != 0 && c->query_ln != 1) return ULTRAMEM_EINVAL;
    if (c->query_ln && (!w->ln_g || c->d_k > 256 || !(c->ln_eps >= 0.f) ||
                        !(c->ln_eps < INFINITY)))
        return ULTRAMEM_EINVAL;
    if (c->d_in <= 0 || c->d_k <= 0 || c->heads <= 0 || c->heads > 64 || c->rank < 1 ||
        c->rank > 8)
        return ULTRAMEM_EINVAL;
    if (c->d_k > 4096 || c->d_in > (1 << 20)) return ULTRAMEM_EINVAL;
    if (c->d_k % c->rank) return ULTRAMEM_EINVAL;
    if (c->n <= 0 || c->d_v <= 0 || c->d_v % 8) return ULTRAMEM_EINVAL;
    int s = (int)lround(sqrt((double)c->expand_e));
    if (c->expand_e < 1 || c->expand_e > 16 || s * s != c->expand_e) return ULTRAMEM_EINVAL;
    int64_t K = keys_per_axis(*c);
    if (K > 20480) return ULTRAMEM_EINVAL;
    uint64_t M = (uint64_t)c->expand_e * (uint64_t)c->n * (uint64_t)c->n;
    if (M >= (1ull << 32)) return ULTRAMEM_EINVAL;
    if (c->topk < 1 || c->topk > 128 || c->topk > K) return ULTRAMEM_EINVAL;
    if (c->topm < 1 || c->topm > 1024 || c->topm > c->topk * c->topk) return ULTRAMEM_EINVAL;
    if (c->has_proj != 0 && c->has_proj != 1) return ULTRAMEM_EINVAL;
    if (!c->has_proj && (c->expand_e != 1 || c->d_out != c->d_v)) return ULTRAMEM_EINVAL;
    if (c->has_proj && c->d_out <= 0) return ULTRAMEM_EINVAL;
    if (c->share_query != 0 && c->share_query != 1) return ULTRAMEM_EINVAL;
    if (c->act != ULTRAMEM_ACT_NONE && c->act != ULTRAMEM_ACT_SOFTMAX) return ULTRAMEM_EINVAL;
    if (c->dtype != ULTRAMEM_F32 && c->dtype != ULTRAMEM_BF16) return ULTRAMEM_EINVAL;
    if (c->max_tokens < 1 || c->max_tokens > (1 << 20)) return ULTRAMEM_EINVAL;
    if (!w->w_q || !w->k_row || !w->k_col || !w->values || (!w->core && !pkm))
        return ULTRAMEM_EINVAL;
    if (!c->share_query && !w->w_q_col) return ULTRAMEM_EINVAL;
    if (c->has_proj && !w->w_proj) return ULTRAMEM_EINVAL;
    if ((w->u == nullptr) != (w->t == nullptr)) return ULTRAMEM_EINVAL;
    if (((uintptr_t)w->values) % 16) return ULTRAMEM_EINVAL;
    if (c->shard_rows < 0 || c->shard_rows > (int64_t)c->n * c->n) return ULTRAMEM_EINVAL;
    return ULTRAMEM_OK;
}


// Leading singular triplet by one-sided (Hestenes) Jacobi on the columns of
// C: rotations orthogonalise the columns of U = C V; the column norms are the
// singular values and V holds the right singular vectors.
ultramem_status rank1_host(const double *c, int r, double *u, double *t, double *sigma) {
    double U[64], Vm[64];
    for (int i = 0; i < r * r; ++i) U[i] = c[i];
    for (int i = 0; i < r; ++i)
        for (int j = 0; j < r; ++j) Vm[i * r + j] = i == j ? 1.0 : 0.0;
    for (int sweep = 0; sweep < 60; ++sweep) {
        bool rotated = false;
        for (int p = 0; p < r; ++p)
            for (int q = p + 1; q < r; ++q) {
                double al = 0, be = 0, ga = 0;
                for (int i = 0; i < r; ++i) {
                    al += U[i * r + p] * U[i * r + p];
                    be += U[i * r + q] * U[i * r + q];
                    ga += U[i * r + p] * U[i * r + q];
                }
                if (fabs(ga) <= 1e-15 * sqrt(al * be) || ga == 0.0) continue;
                rotated = true;
                double zeta = (be - al) / (2.0 * ga);
                double tn = (zeta >= 0 ? 1.0 : -1.0) / (fabs(zeta) + sqrt(1.0 + zeta * zeta));
                double cs = 1.0 / sqrt(1.0 + tn * tn), sn = cs * tn;
                for (int i = 0; i < r; ++i) {
                    double x = U[i * r + p], y = U[i * r + q];
                    U[i * r + p] = cs * x - sn * y;
                    U[i * r + q] = sn * x + cs * y;
                    x = Vm[i * r + p];
                    y = Vm[i * r + q];
                    Vm[i * r + p] = cs * x - sn * y;
                    Vm[i * r + q] = sn * x + cs * y;
                }
            }
        if (!rotated) break;
    }
    int best = 0;
    double bestn = -1;
    for (int j = 0; j < r; ++j) {
        double nn = 0;
        for (int i = 0; i < r; ++i) nn += U[i * r + j] * U[i * r + j];
        if (nn > bestn) { bestn = nn; best = j; }
    }
    double sg = sqrt(bestn);
    if (!(sg > 0.0)) return ULTRAMEM_EINVAL;
    for (int i = 0; i < r; ++i) u[i] = U[i * r + best] / sg;
    double sum = 0;
    for (int i = 0; i < r; ++i) sum += u[i];
    bool flip = sum < 0;
    if (sum == 0)
        for (int i = 0; i < r; ++i)
            if (u[i] != 0) { flip = u[i] < 0; break; }
    if (flip)
        for (int i = 0; i < r; ++i) u[i] = -u[i];
    for (int j = 0; j < r; ++j) {   // t = C^T u / sigma
        double a = 0;
        for (int i = 0; i < r; ++i) a += c[i * r + j] * u[i];
        t[j] = a / sg;
    }
    *sigma = sg;
    return ULTRAMEM_OK;
}

uint64_t splitmix_out(uint64_t state) {   // SplitMix64 output function
    uint64_t z = state + 0x9E3779B97F4A7C15ull;
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
    z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
    return z ^ (z >> 31);
}

void shuffle_params(uint64_t seed, uint64_t M, uint64_t *a, uint64_t *c) {
    if (seed == 0 || M <= 1) { *a = 1; *c = 0; return; }
    uint64_t o1 = splitmix_out(seed), o2 = splitmix_out(seed + 0x9E3779B97F4A7C15ull);
    uint64_t x = 1 + o1 % (M - 1);
    for (;;) {
        uint64_t g = x, h = M;
        while (h) { uint64_t r = g % h; g = h; h = r; }
        if (g == 1) break;
        x = x + 1 >= M ? 1 : x + 1;
    }
    *a = x;
    *c = o2 % M;
}

// Every device allocation of the library goes through lib_malloc / lib_free:
// they count the live allocations and serve the allocation-failure hook of
// ultramem_debug_fail_alloc (countdown < 0: disarmed).
std::atomic<int> g_live_allocs{0};
std::atomic<int> g_fail_countdown{-1};

cudaError_t lib_malloc(void **p, size_t bytes) {
    *p = nullptr;
    int c = g_fail_countdown.load();
    while (c >= 0 && !g_fail_countdown.compare_exchange_weak(c, c - 1)) {
    }
    if (c == 0) return cudaErrorMemoryAllocation;   // the armed allocation fails
    const cudaError_t e = cudaMalloc(p, bytes);
    if (e == cudaSuccess) ++g_live_allocs;
    return e;
}

void lib_free(void *p) {
    if (p && cudaFree(p) == cudaSuccess) --g_live_allocs;
}

template <typename T> cudaError_t dalloc(T **p, size_t n) {
    if (n == 0) n = 1;
    void *v = nullptr;
    const cudaError_t e = lib_malloc(&v, n * sizeof(T));
    *p = static_cast<T *>(v);
    return e;
}

void free_workspace(Workspace &ws) {
    void *ptrs[] = {ws.q_part, ws.akey, ws.gstat, ws.tau, ws.sel_w,   ws.acc,       ws.proj_part,
                    ws.sel_row, ws.sel_p, ws.core,   ws.u,         ws.t,
                    ws.err,    ws.x_stage, ws.out_stage, ws.qs,     ws.acc_bf,
                    ws.w_pt,   ws.cores,   ws.xs,      ws.dacc,    ws.bwd_t,
                    ws.stamps, ws.shard_cursor};
    for (void *p : ptrs) lib_free(p);
    ws = Workspace();
}

Ptrs make_ptrs(ultramem_layer *L) {
    Ptrs p;
    memset(&p, 0, sizeof p);
    p.w_q = L->w.w_q;
    p.w_q_col = L->w.w_q_col;
    p.k_row = L->w.k_row;
    p.k_col = L->w.k_col;
    p.values = L->w.values;
    p.w_proj = L->w.w_proj;
    p.perm = L->w.perm;
    p.conv_w = L->w.conv_w;
    p.conv_b = L->w.conv_b;
    p.ln_g = L->w.ln_g;
    p.ln_b = L->w.ln_b;
    p.xs = L->ws.xs;
    p.core = L->ws.core;
    p.cores = L->ws.cores;
    p.u = L->ws.u;
    p.t = L->ws.t;
    p.q_part = L->ws.q_part;
    p.akey = L->ws.akey;
    p.gstat = L->ws.gstat;
    p.tau = L->ws.tau;
    p.cand = reinterpret_cast<unsigned long long *>(L->ws.akey);
    p.sel_w = L->ws.sel_w;
    p.acc = L->ws.acc;
    p.proj_part = L->ws.proj_part;
    p.sel_row = L->ws.sel_row;
    p.sel_p = L->ws.sel_p;
    p.err = L->ws.err;
    return p;
}

Dims dims_for(const ultramem_layer *L, int B) {
    Dims d = L->base;
    d.B = B;
    // Long grids (more than three selection CTAs per SM) with more than 4096
    // keys an axis: staging both axes' keys (8 K bytes) would leave room for
    // fewer than 4 selection CTAs per SM, so the selection reads them from L2
    // twice instead.  Measured at large_20m (K = 8960) with 256 tokens: select
    // 71.3 -> 56.4 us (2 -> 4 CTAs per SM); at K = 4096 staging is as fast.
    d.stream_keys = (int64_t)B * d.H > 3 * 152 && d.K > 4096 && d.K % 4 == 0;
    // Candidate lists (ScoreListOp): the tensor path scores twice and leaves
    // per-axis candidate lists, so the keys' round trip through memory goes
    // and the selection starts from about 2 % of them.  The passes pay off
    // once each SM has several of their tiles (128 tokens x 256 keys of one
    // head and axis) to pipeline: measured on GB300, lists against every key
    // at 3.5 or more tiles per SM (mid_4m with 1024 and 2048 tokens,
    // large_20m with 256, prefill_16k) 2-5 % shorter steps, below it (mid_4m
    // with 128-512 tokens, large_20m with 64 and 128, decode grids) 3-60 %
    // longer.  Mode 2 (the default) takes them from 3.5 tiles per SM on;
    // modes 0 and 1 force every key or the lists.
    const int64_t list_tiles = (int64_t)((d.K + 255) / 256) * ((B + 127) / 128) * 2 * d.H;
    const bool long_grid = 2 * list_tiles >= 7 * (int64_t)um::device_sm_count();
    d.cand = L->cand_ok && (L->cand_mode == 1 || (L->cand_mode == 2 && long_grid)) ? 1 : 0;
    if (d.cand) d.stream_keys = 0;
    d.seq_len = B;   // one sequence unless the caller says otherwise
    d.q_splits = L->tc ? tc_query_splits(L->cfg, B) : query_splits(L->cfg, B);
    d.p_splits = L->tc ? tc_proj_splits(L->cfg, B) : proj_splits(L->cfg, B);
    d.q_ntile = L->tc ? tc_query_plan(L->cfg, B).n_tile : 0;
    d.p_ntile = L->tc ? tc_proj_plan(L->cfg, B).n_tile : 0;
    return d;
}

thread_local char g_last_error[256] = "";

ultramem_status from_cuda(cudaError_t e) {
    if (e == cudaSuccess) return ULTRAMEM_OK;
    snprintf(g_last_error, sizeof g_last_error, "%s: %s", cudaGetErrorName(e),
             cudaGetErrorString(e));
    if (e == cudaErrorMemoryAllocation) return ULTRAMEM_ENOMEM;
    return ULTRAMEM_ECUDA;
}

// Profiling: the stage stamps are reset before the forward (begins to the
// largest value, ends to 0; memset nodes under stream capture) and each
// kernel gets the pair of its stage.
cudaError_t reset_stamps(ultramem_layer *L, cudaStream_t st) {
    if (!L->profiling) return cudaSuccess;
    unsigned long long *s = L->ws.stamps;
    cudaError_t e = cudaMemsetAsync(s, 0xff, sizeof(*s) * um::kStampStages, st);
    if (e == cudaSuccess)
        e = cudaMemsetAsync(s + um::kStampStages, 0, sizeof(*s) * um::kStampStages, st);
    return e;
}
Ptrs stage_ptrs(const ultramem_layer *L, const Ptrs &p, int stage) {
    Ptrs q = p;
    q.stamp = L->profiling ? L->ws.stamps + stage : nullptr;
    return q;
}

// What a call runs: the whole forward, S1..S6 (retrieval), or S1 and the
// brute-force exact top-m of the whole grid (recall measurement).
enum RunMode { kForward, kRetrieve, kExact };

// S1..S6 (retrieval) then S7..S9.
ultramem_status run_cuda_core(ultramem_layer *L, const Dims &d0, Ptrs p, cudaStream_t st,
                              RunMode mode, int *launches) {
    cudaError_t e;
    Dims d = d0;
    const int extras = (d.conv_k > 0) + d.query_ln;   // convolution, LayerNorm
    if ((e = reset_stamps(L, st)) != cudaSuccess) return from_cuda(e);
    const Ptrs p0 = stage_ptrs(L, p, 0);
    if (d.conv_k > 0 && (e = um::launch_query_conv(d, p0, false, st)) != cudaSuccess)
        return from_cuda(e);
    {
        Ptrs pq = p0;
        if (d.conv_k > 0) pq.x = p.xs;   // the fp32 convolved rows
        if ((e = um::launch_query(d, pq, d.conv_k > 0, st)) != cudaSuccess) return from_cuda(e);
    }
    if (d.query_ln) {
        if ((e = um::launch_query_ln(d, p0, nullptr, 0, st)) != cudaSuccess) return from_cuda(e);
        d.q_splits = 1;   // the normalised query is split 0
    }
    if (mode == kExact) {
        if ((e = um::launch_exact(d, p, p.idx_out, p.w_out, st)) != cudaSuccess)
            return from_cuda(e);
        *launches = 2 + extras;
        return ULTRAMEM_OK;
    }
    if ((e = um::launch_score(d, stage_ptrs(L, p, 1), st)) != cudaSuccess) return from_cuda(e);
    if ((e = um::launch_select(d, stage_ptrs(L, p, 2), st)) != cudaSuccess) return from_cuda(e);
    *launches = 3 + extras;
    if (mode == kRetrieve) return ULTRAMEM_OK;
    if ((e = um::launch_gather(d, stage_ptrs(L, p, 3), st)) != cudaSuccess) return from_cuda(e);
    if (d.has_proj && (e = um::launch_proj(d, stage_ptrs(L, p, 4), st)) != cudaSuccess)
        return from_cuda(e);
    *launches = 4 + (d.has_proj ? 2 : 0) + extras;   // the projection and its split-K reduce
    if (L->profiling) L->profiled_once = true;
    return ULTRAMEM_OK;
}

// The bf16 path: S1, S2 and S9 on tcgen05 tensor cores, S3-S8 as above.
ultramem_status run_tensor(ultramem_layer *L, const Dims &d, Ptrs p, cudaStream_t st,
                           RunMode mode, int *launches) {
    const ultramem_config &c = L->cfg;
    um::TcMaps mp = L->maps;
    const int Bmax = c.max_tokens;
    const int nt1 = um::tc_n_tile(d.B, 1);   // N tile of every contraction (one accumulator)
    const bool conv = d.conv_k > 0;
    if (!conv && !um::tc_encode(&mp.x, p.x, (uint64_t)c.d_in, (uint64_t)d.B, 1,
                                (uint32_t)d.q_ntile, 2))
        return ULTRAMEM_EINVAL;   // x must be 16-byte aligned
    if (conv && !um::tc_encode(&mp.xs, L->ws.xs, 3ull * c.d_in, (uint64_t)d.B, 1,
                               (uint32_t)d.q_ntile, 2))
        return ULTRAMEM_ECUDA;
    if (d.cand && !um::tc_encode(&mp.qs_t, L->ws.qs, 3ull * c.d_k, (uint64_t)Bmax, 2ull * d.H,
                                 128u, 3))
        return ULTRAMEM_ECUDA;
    if (!um::tc_encode(&mp.qs, L->ws.qs, 3ull * c.d_k, (uint64_t)Bmax, 2ull * d.H,
                       (uint32_t)nt1, 3) ||
        !um::tc_encode(&mp.acc, L->ws.acc_bf, 2ull * d.E * d.d_v, (uint64_t)Bmax, 1,
                       (uint32_t)d.p_ntile, 2))
        return ULTRAMEM_ECUDA;
    // the projection reads the pooled rows as two bf16 terms hi + lo
    p.acc_bf = c.has_proj ? L->ws.acc_bf : nullptr;
    p.acc_terms = 2;
    cudaError_t e;
    if ((e = reset_stamps(L, st)) != cudaSuccess) return from_cuda(e);
    // Every kernel after the first is a programmatic dependent launch of its
    // predecessor (also while profiling: the stamps are written by the
    // kernels themselves).  The first (the convolution, else the query
    // projection) waits for all earlier work on the stream.
    Dims dd = d;
    dd.pdl = 1;
    dd.probe_wait = L->probe_armed ? 1 : 0;
    L->probe_armed = false;   // one forward only
    // Trick 4: the convolution runs first and the query projection reads its
    // output (fp32 for the CUDA-core query, three bf16 terms for the tensor
    // cores); with Trick 2 the LayerNorm writes the scaled splits
    const bool small = d.B <= kSmallQueryBatch;
    const Ptrs p0 = stage_ptrs(L, p, 0);
    if (conv && (e = um::launch_query_conv(d, p0, !small, st)) != cudaSuccess) return from_cuda(e);
    const bool write_qs = !d.query_ln;
    // a dependent of the convolution, or of the copy kernel that brings x in
    const bool qpdl = (conv || L->x_after_copy) && dd.pdl;
    if ((e = small ? um::launch_query_small(d, p0, L->ws.qs, Bmax, conv, write_qs, qpdl, st)
                   : um::launch_query_tc(d, p0, mp, d.q_splits, L->ws.qs, Bmax, conv, write_qs,
                                         qpdl, st)) != cudaSuccess)
        return from_cuda(e);
    if (d.query_ln) {
        Dims dl = dd;
        dl.q_splits = 1;   // the projection left the summed query in split 0
        if ((e = um::launch_query_ln(dl, p0, L->ws.qs, Bmax, st)) != cudaSuccess)
            return from_cuda(e);
    }
    const int extras = conv + d.query_ln;
    if (mode == kExact) {
        Dims dx = dd;
        dx.q_splits = 1;   // the summed query is split 0
        if ((e = um::launch_exact(dx, p, p.idx_out, p.w_out, st)) != cudaSuccess)
            return from_cuda(e);
        *launches = d.A + 1 + extras;
        return ULTRAMEM_OK;
    }
    if ((e = um::launch_score_tc(dd, stage_ptrs(L, p, 1), mp, st)) != cudaSuccess)
        return from_cuda(e);
    Dims ds = dd;
    ds.q_splits = 1;   // the query projection wrote the summed query
    if ((e = um::launch_select(ds, stage_ptrs(L, p, 2), st)) != cudaSuccess) return from_cuda(e);
    // one query projection per query; the candidate-list scoring is three
    // launches (two passes and the bound)
    const int score = d.cand ? 3 : 1;
    *launches = d.A + 1 + score + extras;
    if (mode == kRetrieve) return ULTRAMEM_OK;
    if ((e = um::launch_gather(dd, stage_ptrs(L, p, 3), st)) != cudaSuccess) return from_cuda(e);
    if (d.has_proj && (e = um::launch_proj_tc(dd, stage_ptrs(L, p, 4), mp, st)) != cudaSuccess)
        return from_cuda(e);
    *launches = d.A + 2 + score + (d.has_proj ? 1 : 0) + extras;
    if (L->profiling) L->profiled_once = true;
    return ULTRAMEM_OK;
}

ultramem_status run(ultramem_layer *L, const Dims &d, Ptrs p, cudaStream_t st, RunMode mode) {
    cudaGetLastError();   // a stale error from unrelated work is not ours to report
    int n = 0;
    const ultramem_status s = L->tc ? run_tensor(L, d, p, st, mode, &n)
                                    : run_cuda_core(L, d, p, st, mode, &n);
    if (s == ULTRAMEM_OK) L->launches = n;
    return s;
}

}  // namespace

extern "C" {

int32_t ultramem_version(void) { return 2; }

const char *ultramem_last_error(void) { return g_last_error; }

const char *ultramem_status_string(ultramem_status s) {
    switch (s) {
    case ULTRAMEM_OK: return "ok";
    case ULTRAMEM_EINVAL: return "invalid argument";
    case ULTRAMEM_ENOMEM: return "out of memory";
    case ULTRAMEM_ECUDA: return "CUDA error";
    case ULTRAMEM_ETIMEOUT: return "device wait timed out";
    case ULTRAMEM_EDEVICE: return "device-side check failed";
    case ULTRAMEM_ENODEV: return "no compute capability 10.3 device";
    }
    return "unknown status";
}

const char *ultramem_stage_name(int32_t i) {
    return (i >= 0 && i < kStages) ? kStageNames[i] : nullptr;
}

ultramem_status ultramem_rank1(const float *core, int32_t r, float *u, float *t,
                               float *sigma) {
    if (!core || !u || !t || !sigma || r < 1 || r > 8) return ULTRAMEM_EINVAL;
    double c[64], uu[8], tt[8], sg;
    for (int i = 0; i < r * r; ++i) c[i] = core[i];
    ultramem_status s = rank1_host(c, r, uu, tt, &sg);
    if (s != ULTRAMEM_OK) return s;
    for (int i = 0; i < r; ++i) {
        u[i] = (float)uu[i];
        t[i] = (float)tt[i];
    }
    *sigma = (float)sg;
    return ULTRAMEM_OK;
}

ultramem_status ultramem_create(const ultramem_config *cfg, const ultramem_weights *w,
                                ultramem_layer **out) {
    if (!out) return ULTRAMEM_EINVAL;
    *out = nullptr;
    ultramem_status st = validate(cfg, w);
    if (st != ULTRAMEM_OK) return st;
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return ULTRAMEM_ENODEV;
    int major = 0, minor = 0;
    cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev);
    cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev);
    if (major != 10 || minor != 3) return ULTRAMEM_ENODEV;

    const int H = cfg->heads, r = cfg->rank, nc = cfg->cores > 1 ? cfg->cores : 1;
    // each head's Tucker core: the sum of its component cores (MCS, Eq. 16),
    // summed in fp64 and kept in fp32 for the Tucker combine
    float *hu = (float *)malloc(sizeof(float) * H * r);
    float *ht = (float *)malloc(sizeof(float) * H * r);
    float *hc = (float *)malloc(sizeof(float) * H * r * r);
    if (!hu || !ht || !hc) { free(hu); free(ht); free(hc); return ULTRAMEM_ENOMEM; }
    const bool pkm = cfg->score_mode == ULTRAMEM_SCORE_PKM;
    for (int h = 0; h < H; ++h) {
        double cd[64];
        if (pkm) {   // product keys (rank 1): the axis scores themselves, summed
            hc[h] = 1.f;
            hu[h] = 1.f;
            ht[h] = 1.f;
            continue;
        }
        for (int e = 0; e < r * r; ++e) {
            cd[e] = 0.0;
            for (int i = 0; i < nc; ++i) cd[e] += w->core[((size_t)h * nc + i) * r * r + e];
            hc[h * r * r + e] = (float)cd[e];
        }
        // (u, t): given, or the SVD of the summed core (Eq. 7)
        if (w->u) {
            memcpy(hu + h * r, w->u + h * r, sizeof(float) * r);
            memcpy(ht + h * r, w->t + h * r, sizeof(float) * r);
        } else {
            double uu[8], tt[8], sg;
            if (rank1_host(cd, r, uu, tt, &sg) != ULTRAMEM_OK) {
                free(hu); free(ht); free(hc);
                return ULTRAMEM_EINVAL;
            }
            for (int i = 0; i < r; ++i) {
                hu[h * r + i] = (float)uu[i];
                ht[h * r + i] = (float)tt[i];
            }
        }
    }

    ultramem_layer *L = new (std::nothrow) ultramem_layer();
    if (!L) { free(hu); free(ht); free(hc); return ULTRAMEM_ENOMEM; }
    L->cfg = *cfg;
    L->w = *w;
    L->device = dev;
    Dims &d = L->base;
    memset(&d, 0, sizeof d);
    d.d_in = cfg->d_in;
    d.d_k = cfg->d_k;
    d.H = H;
    d.r = r;
    d.dk = cfg->d_k / r;
    d.K = (int)keys_per_axis(*cfg);
    d.n_groups = (d.K + 15) / 16;
    d.N = (int64_t)cfg->n * cfg->n;
    d.M = (uint64_t)cfg->expand_e * (uint64_t)d.N;
    d.E = cfg->expand_e;
    d.d_v = cfg->d_v;
    d.d_out = cfg->d_out;
    d.k = cfg->topk;
    d.m = cfg->topm;
    d.nc = nc;
    d.conv_k = cfg->conv_k;
    d.query_ln = cfg->query_ln;
    d.pkm = pkm ? 1 : 0;
    d.ln_eps = cfg->ln_eps;
    d.A = cfg->share_query ? 1 : 2;
    d.act = cfg->act;
    d.dtype = cfg->dtype;
    d.has_proj = cfg->has_proj;
    shuffle_params(cfg->shuffle_seed, d.M, &d.shuf_a, &d.shuf_c);
    d.shuf_mu = um::barrett_mu(d.M);

    const size_t Bm = (size_t)cfg->max_tokens, HD = (size_t)H * cfg->d_k;
    size_t qmax = 0, pmax = 0;
    L->tc = tc_eligible(*cfg) && um::tc_init();
    // The split-K partial buffers hold splits(B) * B rows for every batch up
    // to Bm.  splits(B) only falls as B grows and changes only at multiples
    // of 16 tokens, so within a run of equal splits the product peaks at its
    // last batch: every batch up to 256, then every 16th, then Bm itself.
    auto visit = [&](size_t B) {
        size_t q = (size_t)query_splits(*cfg, (int)B) * B;
        size_t qt = (size_t)tc_query_splits(*cfg, (int)B) * B;
        size_t pp = (size_t)proj_splits(*cfg, (int)B) * B;
        size_t pt = (size_t)tc_proj_splits(*cfg, (int)B) * B;
        if (q > qmax) qmax = q;
        if (qt > qmax) qmax = qt;
        if (pp > pmax) pmax = pp;
        if (pt > pmax) pmax = pt;
    };
    for (size_t B = 1; B <= Bm && B <= 256; ++B) visit(B);
    for (size_t B = 272; B < Bm; B += 16) visit(B);
    if (Bm > 256) visit(Bm);
    Workspace &ws = L->ws;
    cudaError_t e = cudaSuccess;
    const size_t hm = Bm * H * cfg->topm;
    if (e == cudaSuccess) e = dalloc(&ws.q_part, qmax * d.A * HD);
    // the candidate-list scoring (long grids, tensor path) keeps its u64
    // lists (16 G entries an axis) where the keys would be
    L->cand_ok = L->tc && d.n_groups >= d.k && d.n_groups <= 1024;
    const size_t lists = Bm * H * 2;
    const size_t key_words = lists * (size_t)d.K;
    const size_t list_words = lists * 16 * (size_t)d.n_groups * 2;
    if (e == cudaSuccess)
        e = dalloc(&ws.akey, L->cand_ok && list_words > key_words ? list_words : key_words);
    if (e == cudaSuccess && L->cand_ok) e = dalloc(&ws.gstat, lists * (size_t)d.n_groups);
    if (e == cudaSuccess && L->cand_ok) e = dalloc(&ws.tau, lists);
    if (e == cudaSuccess) e = dalloc(&ws.sel_w, hm * nc);
    if (e == cudaSuccess) e = dalloc(&ws.sel_row, hm);
    if (e == cudaSuccess) e = dalloc(&ws.sel_p, hm);
    if (e == cudaSuccess) e = dalloc(&ws.acc, cfg->has_proj ? Bm * d.E * d.d_v : 1);
    if (e == cudaSuccess) e = dalloc(&ws.proj_part, cfg->has_proj ? pmax * d.d_out : 1);
    if (e == cudaSuccess) e = dalloc(&ws.core, (size_t)H * r * r);
    if (e == cudaSuccess && nc > 1) e = dalloc(&ws.cores, (size_t)H * nc * r * r);
    if (e == cudaSuccess) e = dalloc(&ws.u, (size_t)H * r);
    if (e == cudaSuccess) e = dalloc(&ws.t, (size_t)H * r);
    if (e == cudaSuccess) e = dalloc(&ws.err, 1);
    if (e == cudaSuccess) e = dalloc(&ws.stamps, 2 * um::kStampStages);
    if (e == cudaSuccess) e = dalloc(&ws.shard_cursor, 1024);
    if (e == cudaSuccess)
        e = lib_malloc(&ws.x_stage, Bm * cfg->d_in * elt_size(*cfg));
    if (e == cudaSuccess)
        e = lib_malloc(&ws.out_stage, Bm * cfg->d_out * elt_size(*cfg));
    // the convolved input: three bf16 terms (tensor path) or fp32, 6 B a value covers both
    if (e == cudaSuccess && cfg->conv_k > 0) e = lib_malloc(&ws.xs, Bm * cfg->d_in * 6);
    if (e == cudaSuccess)
        e = cudaMemcpy(ws.core, hc, sizeof(float) * H * r * r, cudaMemcpyHostToDevice);
    if (e == cudaSuccess && nc > 1)
        e = cudaMemcpy(ws.cores, w->core, sizeof(float) * H * nc * r * r,
                       cudaMemcpyHostToDevice);
    if (e == cudaSuccess) e = cudaMemcpy(ws.u, hu, sizeof(float) * H * r, cudaMemcpyHostToDevice);
    if (e == cudaSuccess) e = cudaMemcpy(ws.t, ht, sizeof(float) * H * r, cudaMemcpyHostToDevice);
    if (e == cudaSuccess) e = cudaMemset(ws.err, 0, sizeof(int));
    free(hu);
    free(ht);
    free(hc);
    const size_t kd = (size_t)d.E * d.d_v;
    if (e == cudaSuccess && L->tc) {
        // tensor path: split queries, bf16 acc, K-major copy of the projectors
        e = dalloc(&ws.qs, (size_t)2 * H * Bm * 3 * cfg->d_k);
        if (e == cudaSuccess) e = cudaMemset(ws.qs, 0, sizeof(__nv_bfloat16) * 2 * H * Bm * 3 * cfg->d_k);
        if (e == cudaSuccess) e = dalloc(&ws.acc_bf, 2 * Bm * kd);   // hi, lo terms
        if (e == cudaSuccess) e = cudaMemset(ws.acc_bf, 0, sizeof(__nv_bfloat16) * 2 * Bm * kd);
        if (e == cudaSuccess && cfg->has_proj) {
            e = dalloc(&ws.w_pt, kd * cfg->d_out);
            if (e == cudaSuccess) e = um::launch_transpose_bf16(w->w_proj, ws.w_pt, (int)kd, cfg->d_out, 0);
            if (e == cudaSuccess) e = cudaDeviceSynchronize();
        }
        if (e == cudaSuccess) e = um::configure_tc();
        if (e == cudaSuccess) e = um::configure_small();
        bool ok = e == cudaSuccess;
        const uint64_t HD = (uint64_t)H * cfg->d_k;
        ok = ok && um::tc_encode(&L->maps.w_q, w->w_q, cfg->d_in, HD, 1, 128, 2);
        ok = ok && um::tc_encode(&L->maps.w_q_col, cfg->share_query ? w->w_q : w->w_q_col,
                                 cfg->d_in, HD, 1, 128, 2);
        ok = ok && um::tc_encode(&L->maps.k_row, w->k_row, cfg->d_k, d.K, H, 128, 3);
        ok = ok && um::tc_encode(&L->maps.k_col, w->k_col, cfg->d_k, d.K, H, 128, 3);
        if (cfg->has_proj) {
            ok = ok && um::tc_encode(&L->maps.w_pt, ws.w_pt, kd, cfg->d_out, 1, 128, 2);
            // the projectors as stored, for the backward's dacc = W_p g (when
            // D'_v rows are whole 16-byte vectors; else the CUDA-core path)
            L->dacc_tc = um::tc_encode(&L->maps.w_p, w->w_proj, cfg->d_out, kd, 1, 128, 2);
        } else {
            L->maps.w_pt = L->maps.w_q;
        }
        if (e == cudaSuccess && !ok) {
            free_workspace(ws);
            delete L;
            return ULTRAMEM_EINVAL;   // a weight is not 16-byte aligned
        }
    }
    L->exact_ok = um::exact_fits(d);
    L->backward_ok = um::backward_fits(d);
    if (e == cudaSuccess && L->backward_ok) e = um::configure_backward(d);
    if (e == cudaSuccess && L->backward_ok && cfg->has_proj) e = dalloc(&ws.dacc, Bm * d.E * d.d_v);
    if (e == cudaSuccess && L->backward_ok && cfg->has_proj && L->tc)
        e = dalloc(&ws.bwd_t, Bm * (2 * (size_t)d.E * d.d_v + cfg->d_out));
    if (e == cudaSuccess && L->exact_ok) e = um::configure_exact(d);
    if (e == cudaSuccess) e = um::configure_select(d);
    if (e == cudaSuccess) e = um::configure_gather(d);
    if (e != cudaSuccess) {
        free_workspace(ws);
        delete L;
        cudaGetLastError();
        return from_cuda(e);
    }
    *out = L;
    return ULTRAMEM_OK;
}

void ultramem_destroy(ultramem_layer *L) {
    if (!L) return;
    cudaDeviceSynchronize();
    for (auto &g : L->host_graphs)
        if (g.exec) cudaGraphExecDestroy(g.exec);
    if (L->capture) cudaStreamDestroy(L->capture);
    free_workspace(L->ws);
    delete L;
}

ultramem_status ultramem_forward(ultramem_layer *L, const void *x, int32_t B, void *out,
                                 int64_t *idx_out, float *w_out, void *stream) {
    if (!L || B < 0 || B > L->cfg.max_tokens || !whole_table(L)) return ULTRAMEM_EINVAL;
    if (B == 0) return ULTRAMEM_OK;
    if (!x || !out) return ULTRAMEM_EINVAL;
    Dims d = dims_for(L, B);
    Ptrs p = make_ptrs(L);
    p.x = x;
    p.out = out;
    p.idx_out = idx_out;
    p.w_out = w_out;
    return run(L, d, p, (cudaStream_t)stream, kForward);
}

ultramem_status ultramem_forward_seq(ultramem_layer *L, const void *x, int32_t n_seq,
                                     int32_t seq_len, const void *conv_state_in,
                                     void *conv_state_out, void *out, int64_t *idx_out,
                                     float *w_out, void *stream) {
    if (!L || n_seq < 0 || seq_len < 1 || !whole_table(L)) return ULTRAMEM_EINVAL;
    if ((int64_t)n_seq * seq_len > L->cfg.max_tokens) return ULTRAMEM_EINVAL;
    const int B = n_seq * seq_len;
    if (B == 0) return ULTRAMEM_OK;
    if (!x || !out) return ULTRAMEM_EINVAL;
    Dims d = dims_for(L, B);
    d.seq_len = seq_len;
    Ptrs p = make_ptrs(L);
    p.x = x;
    p.out = out;
    p.idx_out = idx_out;
    p.w_out = w_out;
    if (L->cfg.conv_k > 1) {
        const size_t bytes = (size_t)n_seq * (L->cfg.conv_k - 1) * L->cfg.d_in * elt_size(L->cfg);
        const char *a = static_cast<const char *>(conv_state_in);
        const char *b = static_cast<const char *>(conv_state_out);
        if (a && b && a < b + bytes && b < a + bytes) return ULTRAMEM_EINVAL;   // overlap
        p.state_in = conv_state_in;
        p.state_out = conv_state_out;
    }
    return run(L, d, p, (cudaStream_t)stream, kForward);
}

ultramem_status ultramem_key_ln(const void *keys, int32_t dtype, int64_t n_rows, int32_t dd,
                                const float *g, const float *b, float eps, void *out,
                                void *stream) {
    if (!keys || !g || !out || n_rows < 0 || dd < 1 || !(eps >= 0.f) || !(eps < INFINITY))
        return ULTRAMEM_EINVAL;
    if (dtype != ULTRAMEM_F32 && dtype != ULTRAMEM_BF16) return ULTRAMEM_EINVAL;
    cudaGetLastError();
    return from_cuda(um::launch_key_ln(keys, dtype, n_rows, dd, g, b, eps, out,
                                       (cudaStream_t)stream));
}

ultramem_status ultramem_retrieve(ultramem_layer *L, const void *x, int32_t B,
                                  int64_t *idx_out, float *w_out, void *stream) {
    if (!L || B < 0 || B > L->cfg.max_tokens) return ULTRAMEM_EINVAL;
    if (B == 0) return ULTRAMEM_OK;
    if (!x || !idx_out || !w_out) return ULTRAMEM_EINVAL;
    Dims d = dims_for(L, B);
    Ptrs p = make_ptrs(L);
    p.x = x;
    p.idx_out = idx_out;
    p.w_out = w_out;
    return run(L, d, p, (cudaStream_t)stream, kRetrieve);
}

ultramem_status ultramem_retrieve_exact(ultramem_layer *L, const void *x, int32_t B,
                                        int64_t *idx_out, float *w_out, void *stream) {
    if (!L || B < 0 || B > L->cfg.max_tokens) return ULTRAMEM_EINVAL;
    if (B == 0) return ULTRAMEM_OK;
    if (!x || !idx_out || !w_out || !L->exact_ok) return ULTRAMEM_EINVAL;
    Dims d = dims_for(L, B);
    Ptrs p = make_ptrs(L);
    p.x = x;
    p.idx_out = idx_out;
    p.w_out = w_out;
    return run(L, d, p, (cudaStream_t)stream, kExact);
}

ultramem_status ultramem_lookup_reduce(ultramem_layer *L, const int64_t *idx, const float *w,
                                       int32_t B, void *out, void *stream) {
    if (!L || B < 0 || B > L->cfg.max_tokens || !whole_table(L)) return ULTRAMEM_EINVAL;
    if (B == 0) return ULTRAMEM_OK;
    if (!idx || !w || !out) return ULTRAMEM_EINVAL;
    Dims d = dims_for(L, B);
    Ptrs p = make_ptrs(L);
    p.idx_in = idx;
    p.w_in = w;
    p.out = out;
    cudaStream_t st = (cudaStream_t)stream;
    cudaError_t e;
    cudaGetLastError();
    if ((e = reset_stamps(L, st)) != cudaSuccess) return from_cuda(e);
    if ((e = um::launch_slots_from_addresses(d, p, st)) != cudaSuccess) return from_cuda(e);
    if ((e = um::launch_gather(d, stage_ptrs(L, p, 3), st)) != cudaSuccess) return from_cuda(e);
    if (d.has_proj && (e = um::launch_proj(d, stage_ptrs(L, p, 4), st)) != cudaSuccess)
        return from_cuda(e);
    L->launches = 2 + (d.has_proj ? 2 : 0);
    if (L->profiling) L->profiled_once = true;
    return ULTRAMEM_OK;
}

ultramem_status ultramem_lookup_reduce_backward(ultramem_layer *L, const int64_t *idx,
                                                const float *w, const void *g, int32_t B,
                                                float *dvalues, float *dw, float *dw_proj,
                                                void *stream) {
    if (!L || B < 0 || B > L->cfg.max_tokens || !whole_table(L)) return ULTRAMEM_EINVAL;
    if (B == 0) return ULTRAMEM_OK;
    if (!idx || !w || !g || !L->backward_ok) return ULTRAMEM_EINVAL;
    Dims d = dims_for(L, B);
    Ptrs p = make_ptrs(L);
    p.idx_in = idx;
    p.w_in = w;
    cudaStream_t st = (cudaStream_t)stream;
    cudaError_t e;
    cudaGetLastError();
    int n = 0;
    if (dw_proj && d.has_proj) {
        // dW_p needs the forward's pooled rows: the forward's slots and gather
        if ((e = um::launch_slots_from_addresses(d, p, st)) != cudaSuccess) return from_cuda(e);
        const int kd = d.E * d.d_v;
        // tensor cores from 256 tokens on (below, the transposes and extra
        // launches cost more than the CUDA-core contraction over few tokens,
        // measured: 65 against 51 us at 64 tokens, 112 against 143 us at 256):
        // the pooled rows as two bf16 terms (as the forward's projection reads
        // them), both operands transposed to put the tokens on K
        bool tc_dw = L->tc && L->ws.bwd_t && B >= 256 && B % 8 == 0 && L->cfg.d_out % 8 == 0;
        CUtensorMap am, gm;
        // acc_t2 [E D_v][2 B] (hi terms in columns [0, B), lo in [B, 2 B)), g_t [D'_v][B]
        __nv_bfloat16 *acc_t2 = L->ws.bwd_t, *g_t = L->ws.bwd_t + (size_t)2 * B * kd;
        tc_dw = tc_dw &&
                um::tc_encode(&am, acc_t2, 2ull * B, (uint64_t)kd, 1,
                              (uint32_t)um::tc_n_tile(kd, 1), 2) &&
                um::tc_encode(&gm, g_t, (uint64_t)B, (uint64_t)L->cfg.d_out, 1, 128, 2);
        Ptrs pg = p;
        if (tc_dw) {
            pg.acc_bf = L->ws.acc_bf;   // [B][2][E D_v]
            pg.acc_terms = 2;
        }
        if ((e = um::launch_gather(d, pg, st)) != cudaSuccess) return from_cuda(e);
        if (tc_dw) {
            for (int j = 0; j < 2; ++j)
                if ((e = um::launch_transpose_bf16(L->ws.acc_bf + (size_t)j * kd, acc_t2 + (size_t)j * B,
                                                   B, kd, st, 2 * kd, 2 * B)) != cudaSuccess)
                    return from_cuda(e);
            if ((e = um::launch_transpose_bf16(g, g_t, B, L->cfg.d_out, st)) != cudaSuccess ||
                (e = um::launch_dw_tc(d, gm, am, dw_proj, L->ws.err, st)) != cudaSuccess)
                return from_cuda(e);
            n += 6;
        } else {
            if ((e = um::launch_backward_proj(d, L->ws.acc, g, dw_proj, st)) != cudaSuccess)
                return from_cuda(e);
            n += 3;
        }
    }
    if (dvalues || dw) {
        // dacc = W_p g: on the tensor cores when the layer has its maps and g
        // is 16-byte aligned, else the CUDA-core contraction
        bool ready = false;
        if (d.has_proj && L->tc && L->dacc_tc) {
            um::TcMaps mp = L->maps;
            CUtensorMap gm;
            if (um::tc_encode(&gm, g, (uint64_t)d.d_out, (uint64_t)B, 1,
                              (uint32_t)um::tc_n_tile(B, 1), 2)) {
                if ((e = um::launch_dacc_tc(d, mp.w_p, gm, L->ws.dacc, L->ws.err, st)) !=
                    cudaSuccess)
                    return from_cuda(e);
                ready = true;
                ++n;
            }
        }
        if ((e = um::launch_backward_rows(d, p, g, L->ws.dacc, ready, dvalues, dw, st)) !=
            cudaSuccess)
            return from_cuda(e);
        n += (d.has_proj && !ready) ? 2 : 1;
    }
    L->launches = n;
    return ULTRAMEM_OK;
}

ultramem_status ultramem_forward_host(ultramem_layer *L, const void *x_host, int32_t B,
                                      void *out_host, void *stream) {
    if (!L || B < 0 || B > L->cfg.max_tokens || !whole_table(L)) return ULTRAMEM_EINVAL;
    if (B == 0) return ULTRAMEM_OK;
    if (!x_host || !out_host) return ULTRAMEM_EINVAL;
    cudaStream_t st = (cudaStream_t)stream;
    const size_t es = elt_size(L->cfg);
    const size_t in_bytes = (size_t)B * L->cfg.d_in * es, out_bytes = (size_t)B * L->cfg.d_out * es;
    cudaGetLastError();
    // Pinned (page-locked, mapped) host buffers are read by a copy kernel and
    // written by the forward's last kernel over the host link, inside a graph
    // replayed per (batch, buffers): at a decode batch graph copy nodes
    // measured 15 us and eager launches 10 us more.  Other host memory takes
    // the copy engines.
    const void *x_dev = um::mapped_host(x_host, in_bytes);
    void *o_dev = um::mapped_host(out_host, out_bytes);
    if (x_dev && o_dev && !L->profiling) {
        // replay (or capture once) the whole call as one graph: the launch
        // overhead of its kernels is paid once per batch shape and buffers
        ultramem_layer::HostGraph *hg = nullptr;
        for (auto &g : L->host_graphs)
            if (g.exec && g.B == B && g.x == x_dev && g.o == o_dev) hg = &g;
        if (!hg) {
            if (!L->capture && cudaStreamCreateWithFlags(&L->capture, cudaStreamNonBlocking) !=
                                   cudaSuccess)
                return from_cuda(cudaGetLastError());
            hg = &L->host_graphs[L->host_graph_next];
            L->host_graph_next = (L->host_graph_next + 1) % ultramem_layer::kHostGraphs;
            if (hg->exec) {
                cudaGraphExecDestroy(hg->exec);
                hg->exec = nullptr;
            }
            cudaStream_t cs = L->capture;
            cudaError_t e = cudaStreamBeginCapture(cs, cudaStreamCaptureModeThreadLocal);
            if (e != cudaSuccess) return from_cuda(e);
            // the last kernel writes the output straight into the mapped buffer
            e = um::launch_copy16(x_dev, L->ws.x_stage, in_bytes, cs);
            L->x_after_copy = true;   // the query may prefetch its weights meanwhile
            ultramem_status s = e == cudaSuccess
                                    ? ultramem_forward(L, L->ws.x_stage, B, o_dev, nullptr,
                                                       nullptr, cs)
                                    : ULTRAMEM_ECUDA;
            L->x_after_copy = false;
            cudaGraph_t graph = nullptr;
            const cudaError_t ee = cudaStreamEndCapture(cs, &graph);
            if (s == ULTRAMEM_OK && e == cudaSuccess && ee == cudaSuccess)
                e = cudaGraphInstantiate(&hg->exec, graph, 0);
            if (graph) cudaGraphDestroy(graph);
            if (s != ULTRAMEM_OK) return s;
            if (e != cudaSuccess || ee != cudaSuccess) {
                hg->exec = nullptr;
                return from_cuda(e != cudaSuccess ? e : ee);
            }
            hg->B = B;
            hg->x = x_dev;
            hg->o = o_dev;
            hg->launches = L->launches + 1;
        }
        cudaError_t e = cudaGraphLaunch(hg->exec, st);
        if (e != cudaSuccess) return from_cuda(e);
        L->launches = hg->launches;
        return from_cuda(cudaStreamSynchronize(st));
    }
    cudaError_t e = x_dev ? um::launch_copy16(x_dev, L->ws.x_stage, in_bytes, st)
                          : cudaMemcpyAsync(L->ws.x_stage, x_host, in_bytes,
                                            cudaMemcpyHostToDevice, st);
    if (e != cudaSuccess) return from_cuda(e);
    ultramem_status s = ultramem_forward(L, L->ws.x_stage, B, L->ws.out_stage, nullptr,
                                         nullptr, stream);
    if (s != ULTRAMEM_OK) return s;
    e = o_dev ? um::launch_copy16(L->ws.out_stage, o_dev, out_bytes, st)
              : cudaMemcpyAsync(out_host, L->ws.out_stage, out_bytes, cudaMemcpyDeviceToHost,
                                st);
    if (e != cudaSuccess) return from_cuda(e);
    return from_cuda(cudaStreamSynchronize(st));
}

ultramem_status ultramem_check(ultramem_layer *L, void *stream) {
    if (!L) return ULTRAMEM_EINVAL;
    cudaError_t e = cudaStreamSynchronize((cudaStream_t)stream);
    if (e != cudaSuccess) return ULTRAMEM_ECUDA;
    int flags = 0;
    if (cudaMemcpy(&flags, L->ws.err, sizeof(int), cudaMemcpyDeviceToHost) != cudaSuccess)
        return ULTRAMEM_ECUDA;
    if (flags && cudaMemset(L->ws.err, 0, sizeof(int)) != cudaSuccess) return ULTRAMEM_ECUDA;
    if (flags & um::kErrTimeout) return ULTRAMEM_ETIMEOUT;
    if (flags & (um::kErrBadIndex | um::kErrInternal)) return ULTRAMEM_EDEVICE;
    return ULTRAMEM_OK;
}

ultramem_status ultramem_shard_route(ultramem_layer *L, const int64_t *idx, int32_t n, int32_t P,
                                     int64_t rows_per_rank, int32_t *counts, int32_t *send_rows,
                                     int32_t *slot_pos, void *stream) {
    if (!L || n < 0 || n > L->cfg.max_tokens || P < 1 || P > 1024 || rows_per_rank < 1)
        return ULTRAMEM_EINVAL;
    const int64_t N = (int64_t)L->cfg.n * L->cfg.n;
    if (rows_per_rank * P < N) return ULTRAMEM_EINVAL;
    if (n == 0) return ULTRAMEM_OK;
    if (!idx || !counts || !send_rows || !slot_pos) return ULTRAMEM_EINVAL;
    Dims d = dims_for(L, n);
    Ptrs p = make_ptrs(L);
    p.idx_in = idx;
    cudaGetLastError();
    return from_cuda(um::launch_shard_route(d, p, P, rows_per_rank, counts, L->ws.shard_cursor,
                                            send_rows, slot_pos, (cudaStream_t)stream));
}

ultramem_status ultramem_shard_lookup(ultramem_layer *L, const int32_t *rows, int64_t n_rows,
                                      void *out_rows, void *stream) {
    if (!L || n_rows < 0) return ULTRAMEM_EINVAL;
    if (n_rows == 0) return ULTRAMEM_OK;
    if (!rows || !out_rows || ((uintptr_t)out_rows % 16)) return ULTRAMEM_EINVAL;
    const int64_t rows_held =
        L->cfg.shard_rows > 0 ? L->cfg.shard_rows : (int64_t)L->cfg.n * L->cfg.n;
    cudaGetLastError();
    return from_cuda(um::launch_shard_lookup(L->w.values, rows_held,
                                             L->cfg.d_v * (int)elt_size(L->cfg), rows, n_rows,
                                             out_rows, L->ws.err, (cudaStream_t)stream));
}

ultramem_status ultramem_shard_pool(ultramem_layer *L, const int64_t *idx, const float *w,
                                    int32_t n, const int32_t *slot_pos, const void *back_rows,
                                    void *out, void *stream) {
    if (!L || n < 0 || n > L->cfg.max_tokens) return ULTRAMEM_EINVAL;
    if (n == 0) return ULTRAMEM_OK;
    if (!idx || !w || !slot_pos || !back_rows || !out || ((uintptr_t)back_rows % 16))
        return ULTRAMEM_EINVAL;
    Dims d = dims_for(L, n);
    Ptrs p = make_ptrs(L);
    p.idx_in = idx;
    p.w_in = w;
    p.out = out;
    p.values = back_rows;   // slot s reads returned row slot_pos[s]
    cudaStream_t st = (cudaStream_t)stream;
    cudaError_t e;
    cudaGetLastError();
    if ((e = um::launch_shard_slots(d, p, slot_pos, st)) != cudaSuccess) return from_cuda(e);
    if ((e = um::launch_gather(d, p, st)) != cudaSuccess) return from_cuda(e);
    if (d.has_proj && (e = um::launch_proj(d, p, st)) != cudaSuccess) return from_cuda(e);
    L->launches = 2 + (d.has_proj ? 2 : 0);
    return ULTRAMEM_OK;
}

ultramem_status ultramem_debug_wait_probe(ultramem_layer *L) {
    if (!L || !L->tc) return ULTRAMEM_EINVAL;
    L->probe_armed = true;
    return ULTRAMEM_OK;
}

void ultramem_debug_fail_alloc(int32_t nth) { g_fail_countdown.store(nth < 0 ? -1 : nth); }

int32_t ultramem_debug_live_allocations(void) { return g_live_allocs.load(); }

ultramem_status ultramem_debug_candidates(ultramem_layer *L, int32_t mode) {
    if (!L || mode < 0 || mode > 2) return ULTRAMEM_EINVAL;
    if (mode == 1 && !L->cand_ok) return ULTRAMEM_ENODEV;
    if (mode != L->cand_mode) {
        // the host-buffer calls' cached graphs hold the launches of the
        // previous form: captured again on their next call
        for (auto &g : L->host_graphs) {
            if (g.exec) cudaGraphExecDestroy(g.exec);
            g.exec = nullptr;
        }
    }
    L->cand_mode = mode;
    return ULTRAMEM_OK;
}

ultramem_status ultramem_profile_enable(ultramem_layer *L, int32_t enable) {
    if (!L) return ULTRAMEM_EINVAL;
    L->profiling = enable != 0;
    L->profiled_once = false;
    return ULTRAMEM_OK;
}

int32_t ultramem_last_launches(const ultramem_layer *L) { return L ? L->launches : 0; }

int32_t ultramem_profile_read(ultramem_layer *L, float *ms, int32_t n) {
    if (!L || !ms || !L->profiled_once || n < 1) return 0;
    unsigned long long st[2 * um::kStampStages];
    if (cudaMemcpy(st, L->ws.stamps, sizeof st, cudaMemcpyDeviceToHost) != cudaSuccess) {
        cudaGetLastError();
        return 0;
    }
    const unsigned long long *bg = st, *en = st + um::kStampStages;
    auto ran = [&](int i) { return bg[i] != ~0ull && en[i] >= bg[i]; };
    const int cnt = n < kStages ? n : kStages;
    for (int i = 0; i < cnt; ++i) ms[i] = ran(i) ? (float)((en[i] - bg[i]) * 1e-6) : -1.f;
    // the hand-offs: from the end of the previous stage to this stage's first
    // CTA past its dependency wait
    for (int i = 0; i < kStages && kStages + i < n; ++i) {
        float g = 0.f;
        if (i > 0 && ran(i) && ran(i - 1))
            g = bg[i] > en[i - 1] ? (float)((bg[i] - en[i - 1]) * 1e-6) : 0.f;
        ms[kStages + i] = g;
    }
    return n < 2 * kStages ? cnt : 2 * kStages;
}

}  // extern "C"

namespace um {

namespace {
__global__ void copy16_kernel(const uint4 *__restrict__ src, uint4 *__restrict__ dst, size_t n) {
    pdl_trigger();   // a dependent may start its weight loads now
    for (size_t i = blockIdx.x * (size_t)blockDim.x + threadIdx.x; i < n;
         i += (size_t)gridDim.x * blockDim.x)
        dst[i] = src[i];
}
}  // namespace

// The device address of page-locked host memory that the device can read
// and write directly (mapped pinned memory), when [p, p + bytes) is such
// memory and 16-byte aligned; else null.
const void *mapped_host(const void *p, size_t bytes) {
    cudaPointerAttributes a;
    if (cudaPointerGetAttributes(&a, p) != cudaSuccess) {
        cudaGetLastError();
        return nullptr;
    }
    if (a.type != cudaMemoryTypeHost || !a.devicePointer) return nullptr;
    if (((uintptr_t)a.devicePointer | bytes) & 15) return nullptr;
    return a.devicePointer;
}
void *mapped_host(void *p, size_t bytes) {
    return const_cast<void *>(mapped_host(static_cast<const void *>(p), bytes));
}

// dst[0, bytes) = src[0, bytes), 16-byte aligned, bytes a multiple of 16.
cudaError_t launch_copy16(const void *src, void *dst, size_t bytes, cudaStream_t st) {
    const size_t n = bytes / 16;
    unsigned blocks = (unsigned)((n + 255) / 256);
    if (blocks > 1024) blocks = 1024;
    if (blocks < 1) blocks = 1;
    copy16_kernel<<<blocks, 256, 0, st>>>(static_cast<const uint4 *>(src), static_cast<uint4 *>(dst),
                                          n);
    return cudaGetLastError();
}

int device_sm_count() {
    static int n = 0;
    if (!n) {
        int dev = 0, v = 0;
        if (cudaGetDevice(&dev) != cudaSuccess ||
            cudaDeviceGetAttribute(&v, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || v < 1) {
            cudaGetLastError();
            v = 1;
        }
        n = v;
    }
    return n;
}

// The seeded shuffle's multiplier and offset, for entry points defined in
// other translation units.
void host_shuffle_params(uint64_t seed, uint64_t M, uint64_t *a, uint64_t *c) {
    shuffle_params(seed, M, a, c);
}
}  // namespace um
