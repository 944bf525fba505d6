// um_internal.cuh -- shared declarations of the UltraMem CUDA library.
//
// Every kernel receives the layer's dimensions (Dims) and the device pointers
// it touches (Ptrs) by value.  Workspace layouts (all fp32 unless noted):
//   q_part   [q_splits][A][B][H*D_k]   split-K partial sums of q = W_q x (the
//                                      tensor path leaves the sum in split 0)
//   akey     [B][H][2][K] uint32       order-preserving key of the rank-1 score
//                                      u^T S_row (axis 0) / t^T S_col (axis 1), Eq. 6
//   sel_row  [B][H][m] int32           physical row of each selected slot
//   sel_p    [B][H][m] int32           virtual block p of each selected slot
//   sel_w    [B][H][m][nc]             weights of each selected slot (nc > 1:
//                                      one per value slice, Multi-Core Scoring)
//   acc      [B][E*D_v]                per-block pooled rows, Eq. 15 inner sum
//   acc_bf   [B][T][E*D_v] bf16        the same as T bf16 terms (tensor path):
//                                      T = 2 for the projection, whose B operand
//                                      is then hi + lo (residual <= 2^-16 |acc|)
//   proj_part[p_splits][B][D'_v]       split-K partial sums of the projection
//   xs       the convolved query input x~ (Trick 4): bf16 [B][3][D_i], three
//            terms per value, for the tensor-core query; fp32 [B][D_i] for
//            the CUDA-core ones
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <type_traits>

#include "../../include/ultramem.h"

namespace um {

constexpr int kErrBadIndex = 1;   // an address outside [0, E*N) was given
constexpr int kErrTimeout = 2;    // a bounded wait gave up
constexpr int kErrInternal = 4;   // a selection produced an impossible position

struct Dims {
    int B;            // tokens in this call
    int d_in, d_k, H, r, dk;  // dk = D_k / r
    int K;            // keys per axis
    int64_t N;        // physical rows
    uint64_t M;       // virtual slots E*N
    int E, d_v, d_out, k, m;
    int nc;           // component cores per head (MCS, Eq. 16-17); 1 = one core
    int conv_k;       // taps of the causal depthwise query convolution; 0 = none
    int seq_len;      // tokens per sequence of this call (the convolution's scope)
    int query_ln;     // 1: LayerNorm of each head's query
    int pkm;          // 1: product-key grid score s_row[i] + s_col[j] (rank 1)
    float ln_eps;
    int A;            // 1 = shared query, 2 = separate column query
    int act, dtype, has_proj;
    uint64_t shuf_a, shuf_c;
    uint64_t shuf_mu;  // floor((2^64 - 1) / M), the Barrett constant of M
    int q_splits, p_splits;
    int q_ntile, p_ntile;   // tensor path: token tiles of the query and the projection
    int pdl;           // host side: launch as a programmatic dependent of the
                       // previous kernel on the stream
    int probe_wait;    // ultramem_debug_wait_probe: the scoring kernel's
                       // bounded wait on a barrier nothing signals
    int stream_keys;   // the selection reads its rank-1 keys from L2 twice
                       // instead of staging them in shared memory
    int cand;          // tensor path, long grids: the scoring leaves per-axis
                       // candidate lists instead of every key (see ScoreOp)
    int n_groups;      // candidate lists: groups of 16 keys an axis, ceil(K / 16)
};

struct Ptrs {
    const void *x, *w_q, *w_q_col, *k_row, *k_col, *values, *w_proj;
    const uint32_t *perm;
    const float *core, *u, *t;   // library copies: [H][r][r] (the summed core), [H][r], [H][r]
    const float *cores;          // [H][nc][r][r] component cores when nc > 1
    float *q_part, *sel_w, *acc, *proj_part;
    uint32_t *akey;
    // candidate lists (Dims::cand): per (token, head, axis) the largest key
    // of each group of 16 keys, then the group's count of candidates
    // [B][H][2][n_groups], the bound tau [B][H][2] and the list of
    // composites, a 16-entry segment per group [B][H][2][n_groups][16]
    uint32_t *gstat, *tau;
    unsigned long long *cand;
    int32_t *sel_row, *sel_p;
    void *out;
    int64_t *idx_out;
    float *w_out;
    __nv_bfloat16 *acc_bf;       // tensor path: acc as bf16 terms [B][acc_terms][E*D_v]
    int acc_terms;               // 2: hi + lo, the pooled value to 2^-16 relative (the
                                 // projection's operand); 1 (or 0): one rounding
    const int64_t *idx_in;       // lookup_reduce input addresses
    const float *w_in;           // lookup_reduce input weights [B][H][m][nc]
    const float *conv_w, *conv_b;   // [conv_k][D_i], [D_i] or null
    const float *ln_g, *ln_b;       // [A][H*D_k] each (ln_b may be null)
    const void *state_in;        // [B/seq_len][conv_k-1][D_i] storage type, or null
    void *state_out;             // same shape, or null
    void *xs;                    // the convolved input (layout above)
    int *err;                    // device error word (bit flags above)
    unsigned long long *stamp;   // profiling: this stage's [begin] (ends kStampStages later)
};

// TMA descriptors of the tensor-core path: weights (encoded at create) and
// the per-call operands (token batch x, split queries qs, pooled acc).
struct TcMaps {
    CUtensorMap w_q, w_q_col, k_row, k_col, w_pt;
    CUtensorMap x, qs, acc;
    CUtensorMap qs_t;    // the split queries with 128-token boxes (candidate lists)
    CUtensorMap xs;      // the convolved input's three bf16 terms [B][3 D_i]
    CUtensorMap w_p;     // the projectors as stored, [E D_v][D'_v] (backward's A)
};

bool tc_init();
bool tc_encode(CUtensorMap *map, const void *base, uint64_t inner, uint64_t mid, uint64_t outer,
               uint32_t box_rows, int rank);
int tc_n_tile(int B, int n_acc);
cudaError_t configure_tc();
cudaError_t launch_query_tc(const Dims &d, const Ptrs &p, const TcMaps &mp, int splits,
                            __nv_bfloat16 *qs, int Bmax, bool x_splits, bool write_qs,
                            bool pdl, cudaStream_t st);
cudaError_t launch_score_tc(const Dims &d, const Ptrs &p, const TcMaps &mp, cudaStream_t st);
// candidate lists: tau = the k-th largest group maximum per (token, head,
// axis)
cudaError_t launch_cand_bound(const Dims &d, const Ptrs &p, cudaStream_t st);
// small batches: S1 on CUDA cores, 16 weight rows x 8 tokens per CTA
cudaError_t configure_small();
// x_f32: the token rows are the fp32 convolved input (p.xs, [B][D_i])
// instead of x itself
cudaError_t launch_query_small(const Dims &d, const Ptrs &p, __nv_bfloat16 *qs, int Bmax,
                               bool x_f32, bool write_qs, bool pdl, cudaStream_t st);
cudaError_t launch_proj_tc(const Dims &d, const Ptrs &p, const TcMaps &mp, cudaStream_t st);
// the backward's dacc = W_p g on the tensor cores (g: map over [B][D'_v] bf16)
cudaError_t launch_dacc_tc(const Dims &d, const CUtensorMap &w_p, const CUtensorMap &g,
                           float *dacc, int *err, cudaStream_t st);
// the backward's dW_p = sum_tokens acc g^T on the tensor cores, from the
// transposed gradient rows [D'_v][B] and the transposed pooled rows as two
// bf16 terms [E D_v][2 B] (hi in columns [0, B), lo in [B, 2 B))
cudaError_t launch_dw_tc(const Dims &d, const CUtensorMap &g_t, const CUtensorMap &acc_t2,
                         float *dW, int *err, cudaStream_t st);
// dst[c][r] = src[r][c], rows x cols bf16; row strides ld_src / ld_dst in
// elements (0: cols / rows, contiguous)
cudaError_t launch_transpose_bf16(const void *src, void *dst, int rows, int cols,
                                  cudaStream_t st, int64_t ld_src = 0, int64_t ld_dst = 0);

// x_f32: the token rows p.x are fp32 (the convolved input) whatever the storage type
cudaError_t launch_query(const Dims &d, const Ptrs &p, bool x_f32, cudaStream_t st);
// Trick 4: the causal depthwise convolution of the call's tokens into p.xs
// (three bf16 terms when `splits`, else fp32) and the conv state after them
cudaError_t launch_query_conv(const Dims &d, const Ptrs &p, bool splits, cudaStream_t st);
// Trick 2: LayerNorm of each head's query in place (split 0 of q_part, the
// sum of d.q_splits partials), and its scaled splits when qs is not null
cudaError_t launch_query_ln(const Dims &d, const Ptrs &p, __nv_bfloat16 *qs, int Bmax,
                            cudaStream_t st);
// LayerNorm of n_rows stored rows of width dd (keys), result in the same type
cudaError_t launch_key_ln(const void *keys, int dtype, int64_t n_rows, int dd, const float *g,
                          const float *b, float eps, void *out, cudaStream_t st);
cudaError_t launch_score(const Dims &d, const Ptrs &p, cudaStream_t st);
cudaError_t launch_select(const Dims &d, const Ptrs &p, cudaStream_t st);
cudaError_t launch_slots_from_addresses(const Dims &d, const Ptrs &p, cudaStream_t st);
cudaError_t launch_gather(const Dims &d, const Ptrs &p, cudaStream_t st);
cudaError_t launch_proj(const Dims &d, const Ptrs &p, cudaStream_t st);

// The number-wise partitioned table (App. D): route slots to their rows'
// owners (counts and cursor: [P] scratch), look rows up in a shard, and the
// gather's per-slot inputs for the rows the owners returned.
cudaError_t launch_shard_route(const Dims &d, const Ptrs &p, int P, int64_t rows_per_rank,
                               int *counts, int *cursor, int32_t *send_rows, int32_t *slot_pos,
                               cudaStream_t st);
cudaError_t launch_shard_lookup(const void *values, int64_t shard_rows, int row_bytes,
                                const int32_t *rows, int64_t n, void *out, int *err,
                                cudaStream_t st);
cudaError_t launch_shard_slots(const Dims &d, const Ptrs &p, const int32_t *slot_pos,
                               cudaStream_t st);

// Eq. 5 by brute force (recall measurement): the exact top-m of every
// (token, head)'s whole grid into idx_out / w_out [B][H][m]
bool exact_fits(const Dims &d);
cudaError_t configure_exact(const Dims &d);
cudaError_t launch_exact(const Dims &d, const Ptrs &p, int64_t *idx_out, float *w_out,
                         cudaStream_t st);

// The backward of the lookup-reduce (App. D): dacc = W_p g, then dV (+=) and
// dw from the slots (p.idx_in, p.w_in); dW_p from the forward's pooled rows
bool backward_fits(const Dims &d);
cudaError_t configure_backward(const Dims &d);
// dacc_ready: dacc already holds W_p g (the tensor-core contraction ran)
cudaError_t launch_backward_rows(const Dims &d, const Ptrs &p, const void *g, float *dacc,
                                 bool dacc_ready, float *dV, float *dw, cudaStream_t st);
cudaError_t launch_backward_proj(const Dims &d, const float *acc, const void *g, float *dW,
                                 cudaStream_t st);

// kernel attributes for large dynamic shared memory, set at layer creation
cudaError_t configure_select(const Dims &d);
cudaError_t configure_gather(const Dims &d);
size_t select_smem_bytes(const Dims &d);
size_t gather_smem_bytes(const Dims &d);

// ---- programmatic dependent launch ----------------------------------------
// A kernel launched with programmatic stream serialization may start while
// the previous kernel on the stream still runs.  Every kernel of the library
// calls pdl_wait() before it touches memory that an earlier kernel writes or
// reads (the wait returns once the previous grid has completed and its
// memory is visible; since every kernel waits before it completes, that
// covers all earlier kernels), and pdl_trigger() once its own resources are
// held, to let the next kernel's CTAs be scheduled.  Both are no-ops for a
// kernel launched without the attribute.  Before the wait a kernel reads
// weights only.
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void pdl_trigger() {
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

// Launches kernel<<<grid, block, smem, st>>>(args...), as a programmatic
// dependent launch when `pdl`, in clusters of 1 x 1 x cluster_z CTAs when
// cluster_z > 1.
template <typename... KArgs, typename... Args>
cudaError_t launch_kernel(bool pdl, unsigned cluster_z, void (*kernel)(KArgs...), dim3 grid,
                          dim3 block, size_t smem, cudaStream_t st, Args &&...args) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = st;
    cudaLaunchAttribute attr[2];
    unsigned n = 0;
    if (pdl) {
        attr[n].id = cudaLaunchAttributeProgrammaticStreamSerialization;
        attr[n].val.programmaticStreamSerializationAllowed = 1;
        ++n;
    }
    if (cluster_z > 1) {
        attr[n].id = cudaLaunchAttributeClusterDimension;
        attr[n].val.clusterDim.x = 1;
        attr[n].val.clusterDim.y = 1;
        attr[n].val.clusterDim.z = cluster_z;
        ++n;
    }
    cfg.attrs = attr;
    cfg.numAttrs = n;
    return cudaLaunchKernelEx(&cfg, kernel, static_cast<Args &&>(args)...);
}

template <typename... KArgs, typename... Args>
cudaError_t launch_kernel(bool pdl, void (*kernel)(KArgs...), dim3 grid, dim3 block,
                          size_t smem, cudaStream_t st, Args &&...args) {
    return launch_kernel(pdl, 1u, kernel, grid, block, smem, st, static_cast<Args &&>(args)...);
}

// ---- CTA placement of dependent launches ----------------------------------
// The CTAs of a programmatic dependent launch are placed while the previous
// kernel still holds SMs, and the scheduler packs them onto whichever SMs have
// room at that moment.  Measured on GB300: the selection's 128 CTAs at decode
// ran 1.15x (decode_1m) to 1.5x (mid_4m) slower packed 2-3 per SM than spread
// one per SM.  A launch of `ctas` CTAs therefore asks for enough dynamic
// shared memory that at most ceil(ctas / SMs) of them fit on one SM.
constexpr size_t kSmemPerSM = 233472;     // 228 KB per SM
constexpr size_t kSmemPerCta = 232448;    // 227 KB at most per CTA
constexpr size_t kSmemReserved = 1024;    // the driver's reservation per CTA

int device_sm_count();

// Host buffers: the device address of mapped pinned memory (null otherwise),
// and a 16-byte copy kernel (host link or device memory).
const void *mapped_host(const void *p, size_t bytes);
void *mapped_host(void *p, size_t bytes);
cudaError_t launch_copy16(const void *src, void *dst, size_t bytes, cudaStream_t st);

// Dynamic shared memory for a launch of `ctas` CTAs that need `need` bytes
// each and have `static_bytes` of static shared memory.
inline size_t spread_smem(size_t need, size_t static_bytes, int64_t ctas) {
    const int sms = device_sm_count();
    const int64_t per_sm = (ctas + sms - 1) / sms;
    if (per_sm < 1 || per_sm >= 8) return need;
    // (per_sm + 1) CTAs must not fit: each takes more than this
    const size_t share = kSmemPerSM / (size_t)(per_sm + 1);
    if (share <= kSmemReserved + static_bytes) return need;
    const size_t pad = ((share - kSmemReserved - static_bytes + 1 + 127) / 128) * 128;
    if (pad + static_bytes > kSmemPerCta) return need;
    return pad > need ? pad : need;
}

// The static shared memory of kernel K (looked up once per kernel).
template <auto K> size_t static_smem_of() {
    static size_t bytes = [] {
        cudaFuncAttributes a;
        if (cudaFuncGetAttributes(&a, K) != cudaSuccess) {
            cudaGetLastError();
            return (size_t)0;
        }
        return (size_t)a.sharedSizeBytes;
    }();
    return bytes;
}

// ---- profiling stamps -----------------------------------------------------
// While a layer profiles, each kernel of a forward records, in nanoseconds
// of the GPU's global timer (it advances in 256 ns steps on GB300), the
// earliest moment one of its CTAs passed its dependency wait (atomicMin into stamp[0]) and
// the latest moment one of its warps finished (atomicMax into
// stamp[kStampStages]); the kernels of one stage share the pair.  The
// forward itself runs unchanged (programmatic dependent launches on), so the
// stage times are the kernels' own device times in the chain.
constexpr int kStampStages = 5;

__device__ __forceinline__ unsigned long long global_ns() {
    unsigned long long t;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
    return t;
}
__device__ __forceinline__ void stamp_begin(unsigned long long *s) {
    if (s && threadIdx.x == 0) atomicMin(s, global_ns());
}
__device__ __forceinline__ void stamp_end(unsigned long long *s) {
    if (s && (threadIdx.x & 31) == 0) atomicMax(s + kStampStages, global_ns());
}

// ---- small device helpers ------------------------------------------------

__device__ __forceinline__ float to_f(float v) { return v; }
__device__ __forceinline__ float to_f(__nv_bfloat16 v) { return __bfloat162float(v); }

template <typename T> __device__ __forceinline__ T from_f(float v);
template <> __device__ __forceinline__ float from_f<float>(float v) { return v; }
template <> __device__ __forceinline__ __nv_bfloat16 from_f<__nv_bfloat16>(float v) {
    return __float2bfloat16_rn(v);
}

// fp32 -> uint32 whose unsigned order is the float order (-0 folded into +0).
__device__ __forceinline__ uint32_t f2ord(float f) {
    uint32_t u = __float_as_uint(f + 0.0f);
    return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}
__device__ __forceinline__ float ord2f(uint32_t o) {
    uint32_t u = (o & 0x80000000u) ? (o & 0x7fffffffu) : ~o;
    return __uint_as_float(u);
}

// A selection candidate: (key, position) as one 64-bit value whose
// descending order is key descending, then position ascending.
__device__ __forceinline__ unsigned long long comp_of(uint32_t key, uint32_t pos) {
    return ((unsigned long long)key << 32) | (unsigned long long)(~pos);
}
__device__ __forceinline__ uint32_t key_of(unsigned long long c) { return (uint32_t)(c >> 32); }
__device__ __forceinline__ uint32_t pos_of(unsigned long long c) { return ~(uint32_t)c; }

// The scoring contraction's B operand for one query element: q[h][c] scaled
// by the rank-1 coefficient of its chunk (u for the row keys, t for the
// column keys), so that one dot product with a key row gives the folded
// score u^T S_row (Eq. 6-7 folded into Eq. 4), written as three bf16 terms
// q1 + q2 + q3 (each the rounding of what the previous ones leave; residual
// <= 2^-24 of the value).  qs is [2][H][Bmax][3][D_k], axis-major; `v` is
// the already scaled value.
__device__ __forceinline__ void put_split_query(__nv_bfloat16 *qs, int axis, int h, int c, int n,
                                                float v, int H, int Bmax, int d_k) {
    const __nv_bfloat16 q1 = __float2bfloat16_rn(v);
    const float r1 = v - __bfloat162float(q1);
    const __nv_bfloat16 q2 = __float2bfloat16_rn(r1);
    const float r2 = r1 - __bfloat162float(q2);
    const __nv_bfloat16 q3 = __float2bfloat16_rn(r2);
    __nv_bfloat16 *dst = qs + (((int64_t)(axis * H + h) * Bmax + n) * 3) * d_k + c;
    dst[0] = q1;
    dst[d_k] = q2;
    dst[2 * d_k] = q3;
}

// One pooled value acc[b][i] (i < E*D_v) into the buffer the next step
// reads: the tensor path's bf16 terms (hi = rn(v), lo = rn(v - hi), so that
// hi + lo equals v to 2^-16 relative), the fp32 acc of the CUDA-core
// projection, or, without a projector, the output row itself.
template <typename T>
__device__ __forceinline__ void store_pooled(const Dims &d, const Ptrs &p, int64_t b, int i,
                                             float v) {
    const int EDv = d.E * d.d_v;
    if (p.acc_bf) {
        const __nv_bfloat16 hi = __float2bfloat16_rn(v);
        __nv_bfloat16 *dst = p.acc_bf + b * (p.acc_terms > 1 ? 2 : 1) * EDv + i;
        dst[0] = hi;
        if (p.acc_terms > 1) dst[EDv] = __float2bfloat16_rn(v - __bfloat162float(hi));
    } else if (d.has_proj) {
        p.acc[b * EDv + i] = v;
    } else {
        static_cast<T *>(p.out)[b * d.d_v + i] = from_f<T>(v);
    }
}

// ---- fp32 storage: dot products to the working precision ---------------
// The fp32 mode promises outputs within 1e-4 of the exact result element by
// element (down to 1e-3 of a row's largest entry), which plain fp32
// accumulation over hundreds of terms does not reach.  Its CUDA-core
// contractions therefore accumulate with error-free transformations
// (Ogita, Rump and Oishi, "Accurate sum and dot product", SIAM J. Sci.
// Comput. 26(6), 2005, algorithm Dot2): TwoProduct by an FMA and Knuth's
// TwoSum, the rounding errors summed on the side, so that s + c is as
// accurate as a dot product computed in twice the working precision.  The
// intrinsics keep the compiler from contracting or reordering the steps.
struct Dot2 {
    float s, c;
    __device__ __forceinline__ Dot2() : s(0.f), c(0.f) {}
    // s + p = t + e exactly (TwoSum): s becomes t and e goes to c
    __device__ __forceinline__ void two_sum_into(float p) {
        const float t = __fadd_rn(s, p);
        const float z = __fsub_rn(t, s);
        const float e = __fadd_rn(__fsub_rn(s, __fsub_rn(t, z)), __fsub_rn(p, z));
        s = t;
        c = __fadd_rn(c, e);
    }
    __device__ __forceinline__ void add(float a, float b) {
        const float p = __fmul_rn(a, b);
        const float pe = __fmaf_rn(a, b, -p);   // a b = p + pe exactly
        two_sum_into(p);
        c = __fadd_rn(c, pe);
    }
    __device__ __forceinline__ void merge(const Dot2 &o) {   // add another partial sum
        two_sum_into(o.s);
        c = __fadd_rn(c, o.c);
    }
    __device__ __forceinline__ float value() const { return __fadd_rn(s, c); }
};

// Barrett's constant for reduction modulo M (P. Barrett, CRYPTO '86).
inline uint64_t barrett_mu(uint64_t M) { return M ? ~0ull / M : 0; }

// The Eq. 14 shuffle: explicit table or the seeded affine bijection
// (a v + c) mod M.  M < 2^32 and a, c, v < M, so a v + c < 2^64.  The
// remainder uses Barrett's reduction: with mu = floor((2^64 - 1) / M) the
// quotient estimate floor(x mu / 2^64) is at most 2 below floor(x / M), so
// at most two corrections make it exact.
__device__ __forceinline__ uint64_t shuffle_address(const Dims &d, const uint32_t *perm,
                                                    uint64_t v) {
    if (perm) return perm[v];
    const uint64_t x = d.shuf_a * v + d.shuf_c;
    uint64_t r = x - __umul64hi(x, d.shuf_mu) * d.M;
    if (r >= d.M) r -= d.M;
    if (r >= d.M) r -= d.M;
    return r;
}

}  // namespace um
