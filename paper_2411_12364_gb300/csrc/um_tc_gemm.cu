// um_tc_gemm.cu -- the three dense contractions of the layer on tcgen05
// tensor cores (bf16 storage mode):
//   S1  q_part = W_q x            M = H*D_k outputs, N = tokens, K = D_i (split-K)
//   S2  S_alpha = K_chunk q_chunk M = keys, N = tokens, K = D_k in r chunks (Eq. 4)
//   S9  out = W_p^T acc           M = D'_v outputs, N = tokens, K = E*D_v (Eq. 15)
// Weights fill the 128-row M side ("swap AB"), so a decode batch of B tokens
// is the N side of one MMA (N = B rounded up to 16).
//
// q is an fp32 result; the scores must be as exact as fp32 because they pick
// indices, so q enters S2 as three bf16 terms q = q1 + q2 + q3 (each the bf16
// rounding of what the previous terms leave, residual <= 2^-24 |q|) and each
// key tile is multiplied by all three, accumulating in fp32.  Keys are bf16
// and enter exactly.
//
// One CTA (8 warps) computes one 128 x N tile: warp 0 lane 0 issues the TMA
// loads of a 4-stage ring, warp 1 lane 0 issues the MMAs, and all eight warps
// then read TMEM for the epilogue (row i = lane i; warps w and w + 4 share a
// lane quarter and take alternate 32-column chunks).  Every mbarrier wait is
// bounded (~1 s); a timeout sets the layer's error word.
//
// Split-K (S1 and S9 at small batches, so that enough SMs stream the
// weights): the S CTAs of one tile form a thread-block cluster, used as a
// barrier that all of them are guaranteed to reach together.  Each writes
// its fp32 partial tile to a global (L2-resident) buffer; after the cluster
// barrier (release / acquire) each CTA adds a slice of the tile's columns
// over the S partials in split order (deterministic) and writes the result.
// (Reading the partials from the peers' shared memory instead measured
// several times slower on GB300.)
#include <cudaTypedefs.h>

#include "um_internal.cuh"
#include "um_tc.cuh"

namespace um {
namespace {

using namespace tc;

constexpr int kThreads = 256;
constexpr int kMaxStages = 4;
constexpr int kMaxAcc = 4;
constexpr int kMaxSplits = 8;                // split-K CTAs per tile: one portable cluster
constexpr size_t kSmemBudget = 225 * 1024;   // leaves room for static smem

struct Tile {
    int m0, n0;        // first A row, first B row of the tile
    int a_sel;         // which A map (0/1)
    int a_z, b_z;      // third coordinate of 3-D maps (-1: 2-D map)
    int kb0, nkb;      // K blocks [kb0, kb0 + nkb)
};

__host__ __device__ inline size_t stage_bytes_of(int nsplit, int n_tile) {
    return kTileABytes + (size_t)nsplit * n_tile * 128;
}

// As many ring stages as fit (at most 4, never more than the K blocks).
inline int stages_for(int nsplit, int n_tile, int nkb) {
    int s = (int)((kSmemBudget - 1024) / stage_bytes_of(nsplit, n_tile));
    if (s > kMaxStages) s = kMaxStages;
    if (s > nkb) s = nkb;
    return s < 1 ? 1 : s;
}

template <int NSPLIT, class Op>
__global__ void __launch_bounds__(kThreads, 1)
    tc_gemm_kernel(const __grid_constant__ CUtensorMap mapA0,
                   const __grid_constant__ CUtensorMap mapA1,
                   const __grid_constant__ CUtensorMap mapB, Op op) {
    extern __shared__ uint8_t smem_raw[];
    __shared__ __align__(8) uint64_t full[kMaxStages], empty[kMaxStages], accbar;
    __shared__ uint32_t tmem_slot;
    uint8_t *ring = reinterpret_cast<uint8_t *>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const Tile t = op.tile();
    const int n_tile = op.n_tile;
    const uint32_t b_bytes = (uint32_t)n_tile * 128;
    const uint32_t stage_bytes = kTileABytes + NSPLIT * b_bytes;
    // the epilogue reads 32 columns at a time: cover the last such read
    const uint32_t ncols =
        tmem_cols_for((uint32_t)((op.n_acc - 1) * n_tile + ((n_tile - 1) / 32) * 32 + 32));
    const CUtensorMap *mapA = t.a_sel ? &mapA1 : &mapA0;
    const int kStages = op.stages;

    if (threadIdx.x == 0) {
        for (int s = 0; s < kStages; ++s) {
            mbar_init(&full[s], 1);
            mbar_init(&empty[s], 1);
        }
        mbar_init(&accbar, 1);
        fence_mbar_init();
        prefetch_tensormap(mapA);
        prefetch_tensormap(&mapB);
    }
    __syncthreads();

    // The A operand is a weight: the first ring stages of it are requested
    // before the dependency wait, so that under programmatic dependent
    // launch they stream while the previous kernel finishes.  Each stage's
    // barrier expects its A and B bytes; B follows after the wait.
    const int pre = min(kStages, t.nkb);
    auto load_a = [&](int it) {
        const int s = it % kStages;
        uint8_t *sa = ring + (size_t)s * stage_bytes;
        mbar_arrive_expect_tx(&full[s], stage_bytes);
        const int kx = (t.kb0 + it) * kBlockK;
        if (t.a_z >= 0) tma_load_3d(sa, mapA, &full[s], kx, t.m0, t.a_z);
        else tma_load_2d(sa, mapA, &full[s], kx, t.m0);
    };
    auto load_b = [&](int it) {
        const int s = it % kStages;
        uint8_t *sa = ring + (size_t)s * stage_bytes;
        const int kx = (t.kb0 + it) * kBlockK;
#pragma unroll
        for (int j = 0; j < NSPLIT; ++j) {
            uint8_t *sb = sa + kTileABytes + j * b_bytes;
            const int bx = j * op.b_split_stride + kx;
            if (t.b_z >= 0) tma_load_3d(sb, &mapB, &full[s], bx, t.n0, t.b_z);
            else tma_load_2d(sb, &mapB, &full[s], bx, t.n0);
        }
    };
    if (threadIdx.x == 0)
        for (int it = 0; it < pre; ++it) load_a(it);
    pdl_wait();
    // TMEM is taken only after the wait: a kernel that waits never holds
    // columns that a CTA of an earlier kernel could still be waiting for
    if (warp == 0) tmem_alloc(&tmem_slot, ncols);
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = tmem_slot;
    pdl_trigger();

    // Roles: lane 0 of warp 0 produces, lane 0 of warp 1 issues the MMAs; the
    // other lanes of those warps wait at __syncwarp (not spinning on the
    // accumulator barrier, which would steal the role lane's issue slots).
    if (warp == 0) {
      if (lane == 0) {
        // producer: TMA loads of A (128 x 64) and NSPLIT B tiles (N x 64)
        for (int it = 0; it < pre; ++it) load_b(it);
        int it = pre;
        for (; it < t.nkb; ++it) {
            const int s = it % kStages;
            if (!mbar_wait(&empty[s], ((it / kStages) & 1) ^ 1)) {
                atomicOr(op.err, kErrTimeout);
                break;
            }
            load_a(it);
            load_b(it);
        }
        // loads still in flight (only after a timeout) land before exit
        for (int j = (it > kStages ? it - kStages : 0); j < it; ++j)
            mbar_wait(&full[j % kStages], (j / kStages) & 1);
      }
      __syncwarp();
    } else if (warp == 1) {
      if (lane == 0) {
        // MMA issuer.  Descriptors are built once per stage and advanced by
        // 32 bytes (2 in the >>4 address field) per 16-wide K step; the
        // accumulator of each step follows its rank chunk without division.
        const uint32_t idesc = idesc_bf16_f32(kTileM, n_tile);
        uint32_t started = 0;
        int acc = (t.kb0 * kBlockK) / op.acc_chunk;
        int next_chunk = (acc + 1) * op.acc_chunk;   // K index where acc advances
        for (int it = 0; it < t.nkb; ++it) {
            const int s = it % kStages;
            if (!mbar_wait(&full[s], (it / kStages) & 1)) {
                atomicOr(op.err, kErrTimeout);
                break;
            }
            tc_fence_after();
            const uint32_t sa = smem_u32(ring + (size_t)s * stage_bytes);
            const uint64_t ad0 = desc_k_sw128(sa);
            uint64_t bd0[NSPLIT];
#pragma unroll
            for (int j = 0; j < NSPLIT; ++j) bd0[j] = desc_k_sw128(sa + kTileABytes + j * b_bytes);
#pragma unroll
            for (int k16 = 0; k16 < kBlockK / 16; ++k16) {
                const int kg = (t.kb0 + it) * kBlockK + k16 * 16;
                while (kg >= next_chunk && acc < op.n_acc - 1) {
                    ++acc;
                    next_chunk += op.acc_chunk;
                }
                const uint32_t dt = tmem + (uint32_t)(acc * n_tile);
                const uint32_t acc_bit = 1u << acc;
#pragma unroll
                for (int j = 0; j < NSPLIT; ++j) {
                    mma_bf16(dt, ad0 + 2 * k16, bd0[j] + 2 * k16, idesc, started & acc_bit);
                    started |= acc_bit;
                }
            }
            mma_commit(&empty[s]);   // frees the stage once these MMAs are done
        }
        mma_commit(&accbar);
      }
      __syncwarp();
    }
    if (!mbar_wait(&accbar, 0)) atomicOr(op.err, kErrTimeout);
    tc_fence_after();

    // epilogue: thread = tile row (TMEM lane); warp halves take alternate
    // 32-column chunks, read with one wait for every accumulator.
    constexpr int kGroups = kThreads / 128;   // warps sharing each TMEM lane quarter
    const int quad = warp & 3, whalf = warp >> 2;
    const int row = quad * 32 + lane;
    const uint32_t lane_base = tmem + ((uint32_t)(quad * 32) << 16);
    const int S = op.cluster_splits();
    for (int c0 = whalf * 32; c0 < n_tile; c0 += 32 * kGroups) {
        uint32_t r[kMaxAcc][32];
#pragma unroll
        for (int a = 0; a < kMaxAcc; ++a)
            if (a < op.n_acc) tmem_ld32_nowait(lane_base + (uint32_t)(a * n_tile + c0), r[a]);
        tmem_ld_wait();
#pragma unroll
        for (int half = 0; half < 2; ++half) {
            if (c0 + half * 16 >= n_tile) break;
            float v[kMaxAcc][16];
#pragma unroll
            for (int a = 0; a < kMaxAcc; ++a)
#pragma unroll
                for (int i = 0; i < 16; ++i) v[a][i] = __uint_as_float(r[a][half * 16 + i]);
            if (S > 1) op.store_partial(t, row, c0 + half * 16, v);
            else op.store(t, row, c0 + half * 16, v);
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 0) tmem_dealloc(tmem, ncols);
    if (S > 1) {
        cluster_sync();   // every partial of the tile is written and visible
        // this CTA's columns (a multiple of 4 per warp group), split between
        // the groups of warps
        const int per = (((n_tile + S - 1) / S) + 4 * kGroups - 1) & ~(4 * kGroups - 1);
        const int nb = (int)cluster_ctarank() * per + whalf * (per / kGroups);
        const int ne = min(n_tile, nb + per / kGroups);
        for (int n = nb; n < ne; n += 4) {
            float part[4][kMaxSplits];
#pragma unroll
            for (int e = 0; e < 4; ++e)
#pragma unroll
                for (int q = 0; q < kMaxSplits; ++q)
                    part[e][q] = q < S ? op.load_partial(t, q, row, n + e) : 0.f;
#pragma unroll
            for (int e = 0; e < 4; ++e) {
                float sum = 0.f;
#pragma unroll
                for (int q = 0; q < kMaxSplits; ++q)
                    if (q < S) sum += part[e][q];
                op.store_sum(t, row, n + e, sum);
            }
        }
    }
}

// ---- S1: query projection, split over D_i --------------------------------
// q = W_q x is written in fp32 (q_part, split 0) for the selection and as
// the three bf16 terms of the scoring contraction (qs).
struct QueryOp {
    int n_tile, stages, n_acc, acc_chunk, b_split_stride;
    int *err;
    int B, HD, A, a, splits, kb_total, H, d_k, Bmax;
    float *q_part;        // [splits][A][B][HD]; the result is split 0
    __nv_bfloat16 *qs;    // [A*H][Bmax][3][D_k]
    __device__ int cluster_splits() const { return splits; }
    __device__ Tile tile() const {
        Tile t;
        t.m0 = blockIdx.x * kTileM;
        t.n0 = blockIdx.y * n_tile;
        t.a_sel = 0;
        t.a_z = -1;
        t.b_z = -1;
        const int split = blockIdx.z;
        const int per = (kb_total + splits - 1) / splits;
        t.kb0 = split * per;
        t.nkb = max(0, min(kb_total, t.kb0 + per) - t.kb0);
        return t;
    }
    __device__ void put(int m, int n, float q) const {
        q_part[((int64_t)a * B + n) * HD + m] = q;
        const __nv_bfloat16 q1 = __float2bfloat16_rn(q);
        const float r1 = q - __bfloat162float(q1);
        const __nv_bfloat16 q2 = __float2bfloat16_rn(r1);
        const float r2 = r1 - __bfloat162float(q2);
        const __nv_bfloat16 q3 = __float2bfloat16_rn(r2);
        const int h = m / d_k, c = m - h * d_k;
        __nv_bfloat16 *dst = qs + (((int64_t)(a * H + h) * Bmax + n) * 3) * d_k + c;
        dst[0] = q1;
        dst[d_k] = q2;
        dst[2 * d_k] = q3;
    }
    __device__ void store(const Tile &t, int row, int c, float (&v)[kMaxAcc][16]) const {
        const int m = t.m0 + row;
        if (m >= HD) return;
#pragma unroll
        for (int j = 0; j < 16; ++j) {
            const int n = t.n0 + c + j;
            if (n < B) put(m, n, t.nkb ? v[0][j] : 0.f);
        }
    }
    __device__ void store_sum(const Tile &t, int row, int c, float q) const {
        const int m = t.m0 + row, n = t.n0 + c;
        if (m < HD && n < B) put(m, n, q);
    }
    // split-K partials: q_part[split][a][n][m] (the sum later replaces split 0)
    __device__ void store_partial(const Tile &t, int row, int c, float (&v)[kMaxAcc][16]) const {
        const int m = t.m0 + row;
        if (m >= HD) return;
        float *dst = q_part + (((int64_t)blockIdx.z * A + a) * B + t.n0 + c) * HD + m;
#pragma unroll
        for (int j = 0; j < 16; ++j)
            if (t.n0 + c + j < B) dst[(int64_t)j * HD] = t.nkb ? v[0][j] : 0.f;
    }
    __device__ float load_partial(const Tile &t, int split, int row, int c) const {
        const int m = t.m0 + row, n = t.n0 + c;
        if (m >= HD || n >= B) return 0.f;
        return __ldcg(q_part + (((int64_t)split * A + a) * B + n) * HD + m);
    }
};

// ---- S2: row/column scores, one accumulator per rank chunk ------------------
// The epilogue folds the r chunk scores into the rank-1 score (Eq. 6-7),
// a = sum_alpha coef[alpha] S_alpha with coef = u (row keys) or t (column
// keys), and stores its order-preserving 32-bit key.
template <int R>
struct ScoreOp {
    int n_tile, stages, n_acc, acc_chunk, b_split_stride;
    int *err;
    int B, H, K, A, kb_total;
    const float *u, *t;   // [H][R]
    uint32_t *akey;       // [B][H][2][K]
    __device__ int cluster_splits() const { return 1; }
    __device__ void store_sum(const Tile &, int, int, float) const {}
    __device__ void store_partial(const Tile &, int, int, float (&)[kMaxAcc][16]) const {}
    __device__ float load_partial(const Tile &, int, int, int) const { return 0.f; }
    __device__ Tile tile() const {
        Tile tl;
        const int h = blockIdx.z >> 1, axis = blockIdx.z & 1;
        tl.m0 = blockIdx.x * kTileM;
        tl.n0 = blockIdx.y * n_tile;
        tl.a_sel = axis;
        tl.a_z = h;
        tl.b_z = (A == 2 && axis == 1 ? H : 0) + h;
        tl.kb0 = 0;
        tl.nkb = kb_total;
        return tl;
    }
    __device__ void store(const Tile &tl, int row, int c, float (&v)[kMaxAcc][16]) const {
        const int i = tl.m0 + row;
        if (i >= K) return;
        const int h = blockIdx.z >> 1, axis = blockIdx.z & 1;
        const float *coef = (axis == 0 ? u : t) + h * R;
        float cf[R];
#pragma unroll
        for (int a = 0; a < R; ++a) cf[a] = coef[a];
        const int n0 = tl.n0 + c;
        const int64_t tok_stride = (int64_t)H * 2 * K;   // akey elements per token
        uint32_t *dst = akey + ((int64_t)n0 * H + h) * 2 * K + (int64_t)axis * K + i;
        const int nj = min(16, B - n0);
#pragma unroll
        for (int j = 0; j < 16; ++j) {
            if (j >= nj) break;
            float a = cf[0] * v[0][j];
#pragma unroll
            for (int al = 1; al < R; ++al) a = fmaf(cf[al], v[al][j], a);
            dst[j * tok_stride] = f2ord(a);
        }
    }
};

// ---- S9: IVE projection, split over E*D_v --------------------------------
struct ProjOp {
    int n_tile, stages, n_acc, acc_chunk, b_split_stride;
    int *err;
    int B, d_out, kb_total, splits;
    __nv_bfloat16 *out;   // [B][d_out]
    float *part;          // [splits][B][d_out] split-K partials
    __device__ int cluster_splits() const { return splits; }
    __device__ void store_partial(const Tile &t, int row, int c, float (&v)[kMaxAcc][16]) const {
        const int o = t.m0 + row;
        if (o >= d_out) return;
        float *dst = part + ((int64_t)blockIdx.z * B + t.n0 + c) * d_out + o;
#pragma unroll
        for (int j = 0; j < 16; ++j)
            if (t.n0 + c + j < B) dst[(int64_t)j * d_out] = t.nkb ? v[0][j] : 0.f;
    }
    __device__ float load_partial(const Tile &t, int split, int row, int c) const {
        const int o = t.m0 + row, n = t.n0 + c;
        if (o >= d_out || n >= B) return 0.f;
        return __ldcg(part + ((int64_t)split * B + n) * d_out + o);
    }
    __device__ Tile tile() const {
        Tile t;
        t.m0 = blockIdx.x * kTileM;
        t.n0 = blockIdx.y * n_tile;
        t.a_sel = 0;
        t.a_z = -1;
        t.b_z = -1;
        const int per = (kb_total + splits - 1) / splits;
        t.kb0 = blockIdx.z * per;
        t.nkb = max(0, min(kb_total, t.kb0 + per) - t.kb0);
        return t;
    }
    __device__ void store(const Tile &t, int row, int c, float (&v)[kMaxAcc][16]) const {
        const int o = t.m0 + row;
        if (o >= d_out) return;
#pragma unroll
        for (int j = 0; j < 16; ++j) {
            const int n = t.n0 + c + j;
            if (n >= B) break;
            out[(int64_t)n * d_out + o] = __float2bfloat16_rn(t.nkb ? v[0][j] : 0.f);
        }
    }
    __device__ void store_sum(const Tile &t, int row, int c, float v) const {
        const int o = t.m0 + row, n = t.n0 + c;
        if (o < d_out && n < B) out[(int64_t)n * d_out + o] = __float2bfloat16_rn(v);
    }
};

// dst[c][r] = src[r][c] for a rows x cols bf16 matrix (32 x 32 tiles)
__global__ void transpose_kernel(const __nv_bfloat16 *__restrict__ src,
                                 __nv_bfloat16 *__restrict__ dst, int rows, int cols) {
    __shared__ __nv_bfloat16 tile[32][33];
    const int c0 = blockIdx.x * 32, r0 = blockIdx.y * 32;
    for (int i = threadIdx.y; i < 32; i += blockDim.y) {
        const int r = r0 + i, c = c0 + threadIdx.x;
        if (r < rows && c < cols) tile[i][threadIdx.x] = src[(int64_t)r * cols + c];
    }
    __syncthreads();
    for (int i = threadIdx.y; i < 32; i += blockDim.y) {
        const int c = c0 + i, r = r0 + threadIdx.x;
        if (r < rows && c < cols) dst[(int64_t)c * rows + r] = tile[threadIdx.x][i];
    }
}

PFN_cuTensorMapEncodeTiled_v12000 g_encode = nullptr;

}  // namespace

cudaError_t launch_transpose_bf16(const void *src, void *dst, int rows, int cols,
                                  cudaStream_t st) {
    dim3 grid((cols + 31) / 32, (rows + 31) / 32);
    transpose_kernel<<<grid, dim3(32, 8), 0, st>>>(static_cast<const __nv_bfloat16 *>(src),
                                                   static_cast<__nv_bfloat16 *>(dst), rows, cols);
    return cudaGetLastError();
}

// ---- host side ---------------------------------------------------------------

bool tc_init() {
    if (g_encode) return true;
    cudaDriverEntryPointQueryResult q;
    void *fn = nullptr;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault,
                                         &q) != cudaSuccess ||
        q != cudaDriverEntryPointSuccess || !fn) {
        cudaGetLastError();
        return false;
    }
    g_encode = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
    return true;
}

// bf16 tensor [outer][mid][inner] with inner contiguous, as a rank-2 map
// (inner, mid) or rank-3 map (inner, mid, outer); box = 64 x box_rows (x 1),
// 128-byte swizzle, zero fill out of bounds.
bool tc_encode(CUtensorMap *map, const void *base, uint64_t inner, uint64_t mid,
               uint64_t outer, uint32_t box_rows, int rank) {
    if (!g_encode || ((uintptr_t)base & 15) || (inner * 2) % 16) return false;
    cuuint64_t dims[3] = {inner, mid, outer};
    cuuint64_t strides[2] = {inner * 2, inner * 2 * mid};
    cuuint32_t box[3] = {(cuuint32_t)kBlockK, box_rows, 1};
    cuuint32_t estr[3] = {1, 1, 1};
    CUresult r = g_encode(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, (cuuint32_t)rank,
                          const_cast<void *>(base), dims, strides, box, estr,
                          CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                          CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS;
}

int tc_n_tile(int B, int n_acc) {
    int cap = 256 / n_acc;          // n_acc * N <= 512 TMEM columns, N <= 256
    if (cap > 256) cap = 256;
    int n = ((B + 15) / 16) * 16;
    return n < cap ? n : cap;
}

// grid.z = the split count, which is also the cluster's z extent when > 1
template <int NSPLIT, class Op>
static cudaError_t launch_gemm(dim3 grid, const CUtensorMap &a0, const CUtensorMap &a1,
                               const CUtensorMap &b, Op op, int nkb, bool pdl,
                               cudaStream_t st) {
    op.stages = stages_for(NSPLIT, op.n_tile, nkb);
    size_t ring = (size_t)op.stages * stage_bytes_of(NSPLIT, op.n_tile);
    const size_t smem = 1024 + ring;
    return launch_kernel(pdl, grid.z > 1 ? grid.z : 1u, tc_gemm_kernel<NSPLIT, Op>, grid,
                         kThreads, smem, st, a0, a1, b, op);
}

template <int NSPLIT, class Op> static cudaError_t allow_smem() {
    return cudaFuncSetAttribute(tc_gemm_kernel<NSPLIT, Op>,
                                cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kSmemBudget);
}

cudaError_t configure_tc() {
    cudaError_t e = allow_smem<1, QueryOp>();
    if (e == cudaSuccess) e = allow_smem<3, ScoreOp<1>>();
    if (e == cudaSuccess) e = allow_smem<3, ScoreOp<2>>();
    if (e == cudaSuccess) e = allow_smem<3, ScoreOp<3>>();
    if (e == cudaSuccess) e = allow_smem<3, ScoreOp<4>>();
    if (e == cudaSuccess) e = allow_smem<1, ProjOp>();
    return e;
}

cudaError_t launch_query_tc(const Dims &d, const Ptrs &p, const TcMaps &mp, int splits,
                            __nv_bfloat16 *qs, int Bmax, cudaStream_t st) {
    const int HD = d.H * d.d_k;
    const int n_tile = tc_n_tile(d.B, 1);
    const int kb_total = (d.d_in + kBlockK - 1) / kBlockK;
    if (splits > kMaxSplits) return cudaErrorInvalidValue;
    for (int a = 0; a < d.A; ++a) {
        QueryOp op;
        op.n_tile = n_tile;
        op.n_acc = 1;
        op.acc_chunk = 1 << 30;
        op.b_split_stride = 0;
        op.err = p.err;
        op.B = d.B;
        op.HD = HD;
        op.A = d.A;
        op.a = a;
        op.splits = splits;
        op.kb_total = kb_total;
        op.H = d.H;
        op.d_k = d.d_k;
        op.Bmax = Bmax;
        op.q_part = p.q_part;
        op.qs = qs;
        dim3 grid((HD + kTileM - 1) / kTileM, (d.B + n_tile - 1) / n_tile, splits);
        const int per = (kb_total + splits - 1) / splits;
        cudaError_t e = launch_gemm<1>(grid, a == 0 ? mp.w_q : mp.w_q_col, mp.w_q, mp.x, op, per,
                                       false, st);
        if (e != cudaSuccess) return e;
    }
    return cudaSuccess;
}

template <int R>
static cudaError_t launch_score_r(const Dims &d, const Ptrs &p, const TcMaps &mp,
                                  cudaStream_t st) {
    ScoreOp<R> op;
    op.n_tile = tc_n_tile(d.B, R);
    op.n_acc = R;
    op.acc_chunk = d.dk;
    op.b_split_stride = d.d_k;
    op.err = p.err;
    op.B = d.B;
    op.H = d.H;
    op.K = d.K;
    op.A = d.A;
    op.kb_total = (d.d_k + kBlockK - 1) / kBlockK;
    op.u = p.u;
    op.t = p.t;
    op.akey = p.akey;
    dim3 grid((d.K + kTileM - 1) / kTileM, (d.B + op.n_tile - 1) / op.n_tile, 2 * d.H);
    return launch_gemm<3>(grid, mp.k_row, mp.k_col, mp.qs, op, op.kb_total, d.pdl, st);
}

cudaError_t launch_score_tc(const Dims &d, const Ptrs &p, const TcMaps &mp, cudaStream_t st) {
    switch (d.r) {
    case 1: return launch_score_r<1>(d, p, mp, st);
    case 2: return launch_score_r<2>(d, p, mp, st);
    case 3: return launch_score_r<3>(d, p, mp, st);
    default: return launch_score_r<4>(d, p, mp, st);
    }
}

cudaError_t launch_proj_tc(const Dims &d, const Ptrs &p, const TcMaps &mp, cudaStream_t st) {
    if (d.p_splits > kMaxSplits) return cudaErrorInvalidValue;
    ProjOp op;
    op.n_tile = tc_n_tile(d.B, 1);
    op.n_acc = 1;
    op.acc_chunk = 1 << 30;
    op.b_split_stride = 0;
    op.err = p.err;
    op.B = d.B;
    op.d_out = d.d_out;
    op.kb_total = (d.E * d.d_v + kBlockK - 1) / kBlockK;
    op.splits = d.p_splits;
    op.out = static_cast<__nv_bfloat16 *>(p.out);
    op.part = p.proj_part;
    dim3 grid((d.d_out + kTileM - 1) / kTileM, (d.B + op.n_tile - 1) / op.n_tile, op.splits);
    const int per = (op.kb_total + op.splits - 1) / op.splits;
    return launch_gemm<1>(grid, mp.w_pt, mp.w_pt, mp.acc, op, per, d.pdl, st);
}

}  // namespace um
