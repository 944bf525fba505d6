// um_tc_gemm.cu -- the three dense contractions of the layer on tcgen05
// tensor cores (bf16 storage mode):
//   S1  q_part = W_q x            M = H*D_k outputs, N = tokens, K = D_i (split-K)
//   S2  S_alpha = K_chunk q_chunk M = keys, N = tokens, K = D_k in r chunks (Eq. 4)
//   S9  out = W_p^T acc           M = D'_v outputs, N = tokens, K = E*D_v (Eq. 15),
//                                 acc entering as two bf16 terms hi + lo
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
// weights): the S CTAs of one tile form a thread-block cluster and add up
// their fp32 partials through distributed shared memory.  Each stages its
// partial over its drained ring as S column slices; after one cluster
// barrier it sends slice j to CTA j with a single bulk copy (smem to peer
// smem, completing bytes of the peer's mbarrier), and each CTA adds its own
// columns over the S partials in split order (deterministic) and writes the
// result.  Measured on GB300 against partials staged in global memory (L2)
// behind a cluster barrier: the projection at 64 tokens 5.05 -> 4.61 us, at
// 256 tokens of the 20M-row layer 9.6 -> 7.8 us, the query there 12.4 ->
// 10.5 us.  (Per-element 16-byte st.async stores into the peers measured
// slower than either: each store updates the peer's mbarrier.)
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
    int z;             // the tile's third grid coordinate (split or head/axis)
};

// a_rows: rows of the staged A tile (128, or 256 for ops with kARows = 256)
__host__ __device__ inline size_t stage_bytes_of(int nsplit, int n_tile, int a_rows = kTileM) {
    return (size_t)a_rows * 128 + (size_t)nsplit * n_tile * 128;
}

// Split-K: CTA s of a tile's cluster adds up columns [s * per, (s + 1) * per)
// of the tile (per a multiple of 8).  Once its MMAs are done each CTA stages
// its partial over its ring as S slices (slice j: CTA j's columns, as
// [per / 4][128 rows] groups of 4 fp32, so that a warp's 16-byte stores and
// loads touch consecutive addresses) and receives the S - 1 other partials'
// slices of its own columns in as many slots after them.
__host__ __device__ inline int split_cols(int n_tile, int S) {
    return (((n_tile + S - 1) / S) + 7) & ~7;
}
__host__ __device__ inline size_t split_slice_bytes(int n_tile, int S) {
    return (size_t)kTileM * split_cols(n_tile, S) * 4;
}
// staged slices and receive slots together
__host__ __device__ inline size_t split_buf_bytes(int n_tile, int S) {
    return S > 1 ? (size_t)(2 * S - 1) * split_slice_bytes(n_tile, S) : 0;
}

// As many ring stages as fit (at most 4, never more than the K blocks).
inline int stages_for(int nsplit, int n_tile, int nkb, int a_rows = kTileM) {
    int s = (int)((kSmemBudget - 1024) / stage_bytes_of(nsplit, n_tile, a_rows));
    if (s > kMaxStages) s = kMaxStages;
    if (s > nkb) s = nkb;
    return s < 1 ? 1 : s;
}

// An op with kSwapAB = true multiplies with the roles of the staged tiles
// swapped: the B tiles (n_tile = 128 rows) are the MMA's A operand, so that
// they land on TMEM lanes, and the A tile is its B operand (one accumulator
// column per A row).  Loads, ring and barriers are the same.
template <class Op, class = void> struct SwapAB {
    static constexpr bool value = false;
};
template <class Op> struct SwapAB<Op, std::void_t<decltype(Op::kSwapAB)>> {
    static constexpr bool value = Op::kSwapAB;
};
// Rows of the staged A tile: 128, or Op::kARows (256: a swapped op's tile
// then carries twice the keys for the same 128-token operand, so half the
// tiles, half the operand bytes per key and 128 x 256 MMAs; measured on the
// candidate-list passes at mid_4m with 2048 tokens: 137 -> 118 us for both
// passes and their bound).  Loaded as 128-row TMA boxes.
template <class Op, class = void> struct ARows {
    static constexpr int value = kTileM;
};
template <class Op> struct ARows<Op, std::void_t<decltype(Op::kARows)>> {
    static constexpr int value = Op::kARows;
};

// An op with kGroupEpilogue = true (the candidate-list passes: swapped)
// reduces each group of 16 accumulator columns to one 32-bit value (group)
// and stores a thread's consecutive groups at once (store_groups): each
// epilogue warp half takes a contiguous half of the columns, so that a
// token's values leave as 16-byte stores instead of scattered 4-byte ones.
template <class Op, class = void> struct GroupEpi {
    static constexpr bool value = false;
};
template <class Op> struct GroupEpi<Op, std::void_t<decltype(Op::kGroupEpilogue)>> {
    static constexpr bool value = Op::kGroupEpilogue;
};

// The grouped epilogue of one TMEM lane (row) over its warp's columns
// [cb, cb + 16 NG): NG groups of 16 (NG a multiple of 4).
template <class Op, int NG>
__device__ __forceinline__ void group_epilogue(const Op &op, const Tile &t, int row, int cb,
                                               uint32_t lane_base) {
    static_assert(NG % 4 == 0, "whole 16-byte stores of group values");
    const uint32_t pre = op.prefetch(t, row, cb);
    uint32_t g[NG];
#pragma unroll
    for (int cc = 0; cc < NG / 2; ++cc) {
        uint32_t r[32];
        tmem_ld32_nowait(lane_base + (uint32_t)(cb + cc * 32), r);
        tmem_ld_wait();
#pragma unroll
        for (int half = 0; half < 2; ++half) {
            float v[16];
#pragma unroll
            for (int i = 0; i < 16; ++i) v[i] = __uint_as_float(r[half * 16 + i]);
            g[cc * 2 + half] = op.group(t, row, cb + cc * 32 + half * 16, v, pre);
        }
    }
    op.template store_groups<NG>(t, row, cb, g);
}

// accumulator columns of one MMA: n_tile, or the A rows when swapped
template <class Op> __host__ __device__ inline int acc_cols_of(const Op &op) {
    return SwapAB<Op>::value ? ARows<Op>::value : op.n_tile;
}

template <int NSPLIT, class Op>
__global__ void __launch_bounds__(kThreads, 1)
    tc_gemm_kernel(const __grid_constant__ CUtensorMap mapA0,
                   const __grid_constant__ CUtensorMap mapA1,
                   const __grid_constant__ CUtensorMap mapB, Op op, int probe) {
    extern __shared__ uint8_t smem_raw[];
    __shared__ __align__(8) uint64_t full[kMaxStages], empty[kMaxStages], accbar, never, recvbar;
    __shared__ uint32_t tmem_slot;
    uint8_t *ring = reinterpret_cast<uint8_t *>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const Tile t = op.tile_at(blockIdx.x, blockIdx.y, blockIdx.z);
    const int S = op.cluster_splits();
    const uint32_t me = S > 1 ? cluster_ctarank() : 0u;
    const int per = split_cols(op.n_tile, S);
    // columns this CTA adds up (none for a trailing CTA of a narrow tile)
    const int cnt_me = max(0, min(op.n_tile - (int)me * per, per));
    const size_t slice = split_slice_bytes(op.n_tile, S);
    const int n_tile = op.n_tile;
    const uint32_t b_bytes = (uint32_t)n_tile * 128;
    constexpr int kA = ARows<Op>::value;
    constexpr uint32_t a_bytes = (uint32_t)kA * 128;
    const uint32_t stage_bytes = a_bytes + NSPLIT * b_bytes;
    constexpr bool kSwap = SwapAB<Op>::value;
    const int acc_n = acc_cols_of(op);   // accumulator columns
    // the epilogue reads 32 columns at a time: cover the last such read
    const uint32_t ncols =
        tmem_cols_for((uint32_t)((op.n_acc - 1) * acc_n + ((acc_n - 1) / 32) * 32 + 32));
    const CUtensorMap *mapA = t.a_sel ? &mapA1 : &mapA0;
    const int kStages = op.stages;

    if (threadIdx.x == 0) {
        for (int s = 0; s < kStages; ++s) {
            mbar_init(&full[s], 1);
            mbar_init(&empty[s], 1);
        }
        mbar_init(&accbar, 1);
        mbar_init(&recvbar, 1);
        fence_mbar_init();
        // split-K: the S - 1 peers' copies of this CTA's columns complete
        // this transaction count (a phase of no bytes completes at once)
        if (S > 1) mbar_arrive_expect_tx(&recvbar, cnt_me > 0 ? (uint32_t)((S - 1) * slice) : 0u);
        prefetch_tensormap(mapA);
        prefetch_tensormap(&mapB);
    }
    __syncthreads();
    if (probe) {   // ultramem_debug_wait_probe: a bounded wait that runs out
        pdl_wait();
        if (probe_timeout(&never, op.err, kErrTimeout)) return;
    }

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
#pragma unroll
        for (int ab = 0; ab < kA / kTileM; ++ab) {
            uint8_t *sab = sa + ab * kTileABytes;
            if (t.a_z >= 0) tma_load_3d(sab, mapA, &full[s], kx, t.m0 + ab * kTileM, t.a_z);
            else tma_load_2d(sab, mapA, &full[s], kx, t.m0 + ab * kTileM);
        }
    };
    auto load_b = [&](int it) {
        const int s = it % kStages;
        uint8_t *sa = ring + (size_t)s * stage_bytes;
        const int kx = (t.kb0 + it) * kBlockK;
#pragma unroll
        for (int j = 0; j < NSPLIT; ++j) {
            uint8_t *sb = sa + a_bytes + j * b_bytes;
            const int bx = j * op.b_split_stride + kx;
            if (t.b_z >= 0) tma_load_3d(sb, &mapB, &full[s], bx, t.n0, t.b_z);
            else tma_load_2d(sb, &mapB, &full[s], bx, t.n0);
        }
    };
    if (threadIdx.x == 0)
        for (int it = 0; it < pre; ++it) load_a(it);
    pdl_wait();
    stamp_begin(op.stamp);
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
        const uint32_t idesc = kSwap ? idesc_bf16_f32(n_tile, kA) : idesc_bf16_f32(kTileM, n_tile);
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
            for (int j = 0; j < NSPLIT; ++j) bd0[j] = desc_k_sw128(sa + a_bytes + j * b_bytes);
#pragma unroll
            for (int k16 = 0; k16 < kBlockK / 16; ++k16) {
                const int kg = (t.kb0 + it) * kBlockK + k16 * 16;
                while (kg >= next_chunk && acc < op.n_acc - 1) {
                    ++acc;
                    next_chunk += op.acc_chunk;
                }
                const uint32_t dt = tmem + (uint32_t)(acc * acc_n);
                const uint32_t acc_bit = 1u << acc;
#pragma unroll
                for (int j = 0; j < NSPLIT; ++j) {
                    if constexpr (kSwap)
                        mma_bf16(dt, bd0[j] + 2 * k16, ad0 + 2 * k16, idesc, started & acc_bit);
                    else
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
    if constexpr (GroupEpi<Op>::value) {
        group_epilogue<Op, kA / 16 / kGroups>(op, t, row, whalf * (kA / kGroups), lane_base);
        tc_fence_before();
        __syncthreads();
        if (warp == 0) tmem_dealloc(tmem, ncols);
    } else if (S == 1) {
        // a per-chunk value the op fetches one chunk ahead (the candidate
        // lists' bounds), so that its latency overlaps the previous chunk
        uint32_t pre = op.prefetch(t, row, whalf * 32);
        for (int c0 = whalf * 32; c0 < acc_n; c0 += 32 * kGroups) {
            const uint32_t cur = pre;
            if (c0 + 32 * kGroups < acc_n) pre = op.prefetch(t, row, c0 + 32 * kGroups);
            uint32_t r[kMaxAcc][32];
#pragma unroll
            for (int a = 0; a < kMaxAcc; ++a)
                if (a < op.n_acc) tmem_ld32_nowait(lane_base + (uint32_t)(a * acc_n + c0), r[a]);
            tmem_ld_wait();
#pragma unroll
            for (int half = 0; half < 2; ++half) {
                if (c0 + half * 16 >= acc_n) break;
                float v[kMaxAcc][16];
#pragma unroll
                for (int a = 0; a < kMaxAcc; ++a)
#pragma unroll
                    for (int i = 0; i < 16; ++i) v[a][i] = __uint_as_float(r[a][half * 16 + i]);
                op.store(t, row, c0 + half * 16, v, cur);
            }
        }
        tc_fence_before();
        __syncthreads();
        if (warp == 0) tmem_dealloc(tmem, ncols);
    } else {
        // Split-K through distributed shared memory (one accumulator): each
        // CTA stages its partial; once every CTA of the cluster has staged
        // its own (so that every ring is drained), it sends slice j to CTA j
        // with one bulk copy into j's receive slot for it (completing bytes
        // of j's receive barrier), and adds up its own columns over the S
        // partials in split order (deterministic).
        uint8_t *recv = ring + (size_t)S * slice;   // slot of CTA q: q - (q > me)
        // column c's slice c / per as floor((c + 1/2) / per) in fp32: exact
        // while c < 2^22 (the rounding error, below 2^-23 c / per, stays under
        // the 1 / (2 per) between (c + 1/2) / per and the nearest integer)
        const float inv_per = 1.f / (float)per;
        for (int c0 = whalf * 32; c0 < n_tile; c0 += 32 * kGroups) {
            uint32_t r[32];
            tmem_ld32_nowait(lane_base + (uint32_t)c0, r);
            tmem_ld_wait();
#pragma unroll
            for (int g = 0; g < 8; ++g) {
                const int c = c0 + 4 * g;
                if (c >= n_tile) break;
                const int j = (int)(((float)c + 0.5f) * inv_per);
                float4 v = make_float4(__uint_as_float(r[4 * g]), __uint_as_float(r[4 * g + 1]),
                                       __uint_as_float(r[4 * g + 2]), __uint_as_float(r[4 * g + 3]));
                if (!t.nkb) v = make_float4(0.f, 0.f, 0.f, 0.f);   // an empty K range
                *reinterpret_cast<float4 *>(ring + j * slice +
                                            ((size_t)((c - j * per) >> 2) * kTileM + row) * 16) = v;
            }
        }
        fence_proxy_async_smem();   // the staged slices are read by bulk copies
        tc_fence_before();
        __syncthreads();
        if (warp == 0) tmem_dealloc(tmem, ncols);
        // every CTA has staged: its ring is drained and its receive barrier
        // initialised (fence.mbarrier_init above)
        cluster_arrive_relaxed();
        cluster_wait();
        if (threadIdx.x < (unsigned)S && threadIdx.x != me && (int)threadIdx.x * per < n_tile) {
            const uint32_t j = threadIdx.x;
            const uint32_t slot = me - (me > j ? 1u : 0u);
            bulk_copy_to_peer(mapa_shared(smem_u32(recv + slot * slice), j),
                              smem_u32(ring + j * slice), (uint32_t)slice,
                              mapa_shared(smem_u32(&recvbar), j));
        }
        if (cnt_me > 0 && !mbar_wait(&recvbar, 0)) atomicOr(op.err, kErrTimeout);
        // every copy into this CTA has landed, so every copy out of the
        // cluster's CTAs has been read once all have arrived: the wait
        // before exit keeps each CTA's shared memory alive until then
        cluster_arrive_relaxed();
        for (int it = threadIdx.x; it < kTileM * (cnt_me / 4); it += kThreads) {
            const size_t at = (size_t)it * 16;   // group it / 128, row it % 128
            float4 v[kMaxSplits];
#pragma unroll
            for (int q = 0; q < kMaxSplits; ++q)
                if (q < S)
                    v[q] = *reinterpret_cast<const float4 *>(
                        (q == (int)me ? ring + q * slice : recv + (q - (q > (int)me)) * slice) + at);
            float sums[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
            for (int q = 0; q < kMaxSplits; ++q) {
                if (q < S) {
                    sums[0] += v[q].x;
                    sums[1] += v[q].y;
                    sums[2] += v[q].z;
                    sums[3] += v[q].w;
                }
            }
            op.store_sums(t, it % kTileM, (int)me * per + 4 * (it / kTileM), sums);
        }
        cluster_wait();
    }
    stamp_end(op.stamp);
}

// ---- persistent variant (many tiles, no split-K) ----------------------------
// One CTA per SM loops over tiles i = blockIdx.x, + gridDim.x, ... (x fastest,
// then y, then z of the tile grid).  Warp 0 lane 0 streams A/B K-blocks of
// successive tiles through the ring; warp 1 lane 0 issues each tile's MMAs
// into one of two TMEM accumulator buffers; the epilogue warps (2 onwards)
// drain the other buffer meanwhile, so loads, MMAs and stores of
// consecutive tiles overlap.  Barriers: full/empty per ring stage; tfull
// (MMAs of a buffer done) and tempty (its epilogue done, one arrival per
// epilogue warp) per buffer.  Every wait is bounded; a timeout raises the
// error word and an abort flag that every role polls.
//
// Epilogue warps: 8 (two per TMEM lane quarter), or Op::kEpiWarps (16: four
// per quarter, each a quarter of the columns).  An epilogue whose work per
// column is a chain of dependent instructions (the candidate lists'
// appends) runs at a fraction of the issue rate with two warps per SM
// sub-partition; more warps hide that latency.
template <class Op, class = void> struct EpiWarps {
    static constexpr int value = 8;
};
template <class Op> struct EpiWarps<Op, std::void_t<decltype(Op::kEpiWarps)>> {
    static constexpr int value = Op::kEpiWarps;
};
template <class Op> constexpr int persistent_threads() { return 64 + 32 * EpiWarps<Op>::value; }

template <int NSPLIT, class Op>
__global__ void __launch_bounds__(persistent_threads<Op>(), 1)
    tc_gemm_persistent(const __grid_constant__ CUtensorMap mapA0,
                       const __grid_constant__ CUtensorMap mapA1,
                       const __grid_constant__ CUtensorMap mapB, Op op, int gx, int gy,
                       int tiles, uint32_t buf_cols, int probe) {
    extern __shared__ uint8_t smem_raw[];
    __shared__ __align__(8) uint64_t full[kMaxStages], empty[kMaxStages], tfull[2], tempty[2],
        drained, never;
    __shared__ uint32_t tmem_slot;
    __shared__ volatile int abort_flag;
    uint8_t *ring = reinterpret_cast<uint8_t *>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int n_tile = op.n_tile;
    const uint32_t b_bytes = (uint32_t)n_tile * 128;
    constexpr int kA = ARows<Op>::value;
    constexpr uint32_t a_bytes = (uint32_t)kA * 128;
    const uint32_t stage_bytes = a_bytes + NSPLIT * b_bytes;
    const int kStages = op.stages;
    auto tile_of = [&](int i) {
        const int bx = i % gx, r = i / gx;
        return op.tile_at(bx, r % gy, r / gy);
    };

    if (threadIdx.x == 0) {
        for (int s = 0; s < kStages; ++s) {
            mbar_init(&full[s], 1);
            mbar_init(&empty[s], 1);
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(&tfull[b], 1);
            mbar_init(&tempty[b], EpiWarps<Op>::value);
        }
        mbar_init(&drained, 1);
        abort_flag = 0;
        fence_mbar_init();
        prefetch_tensormap(&mapA0);
        prefetch_tensormap(&mapA1);
        prefetch_tensormap(&mapB);
    }
    pdl_wait();
    if (probe) {   // ultramem_debug_wait_probe: a bounded wait that runs out
        __syncthreads();
        if (probe_timeout(&never, op.err, kErrTimeout)) return;
    }
    stamp_begin(op.stamp);
    if (warp == 0) tmem_alloc(&tmem_slot, 2 * buf_cols);
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = tmem_slot;
    pdl_trigger();
    auto fail = [&]() {
        atomicOr(op.err, kErrTimeout);
        abort_flag = 1;
    };

    if (warp == 0) {
        if (lane == 0) {
            // producer
            int it = 0;
            for (int i = blockIdx.x; i < tiles && !abort_flag; i += gridDim.x) {
                const Tile t = tile_of(i);
                const CUtensorMap *mapA = t.a_sel ? &mapA1 : &mapA0;
                for (int kb = 0; kb < t.nkb; ++kb, ++it) {
                    const int s = it % kStages;
                    if (it >= kStages && !mbar_wait(&empty[s], ((it / kStages) & 1) ^ 1)) {
                        fail();
                        break;
                    }
                    uint8_t *sa = ring + (size_t)s * stage_bytes;
                    mbar_arrive_expect_tx(&full[s], stage_bytes);
                    const int kx = (t.kb0 + kb) * kBlockK;
#pragma unroll
                    for (int ab = 0; ab < kA / kTileM; ++ab) {
                        uint8_t *sab = sa + ab * kTileABytes;
                        if (t.a_z >= 0)
                            tma_load_3d(sab, mapA, &full[s], kx, t.m0 + ab * kTileM, t.a_z);
                        else tma_load_2d(sab, mapA, &full[s], kx, t.m0 + ab * kTileM);
                    }
#pragma unroll
                    for (int j = 0; j < NSPLIT; ++j) {
                        uint8_t *sb = sa + a_bytes + j * b_bytes;
                        const int bx = j * op.b_split_stride + kx;
                        if (t.b_z >= 0) tma_load_3d(sb, &mapB, &full[s], bx, t.n0, t.b_z);
                        else tma_load_2d(sb, &mapB, &full[s], bx, t.n0);
                    }
                }
            }
            // loads still in flight (only after an abort) land before exit
            for (int j = (it > kStages ? it - kStages : 0); j < it; ++j)
                mbar_wait(&full[j % kStages], (j / kStages) & 1);
        }
        __syncwarp();
    } else if (warp == 1) {
        if (lane == 0) {
            // MMA issuer
            constexpr bool kSwap = SwapAB<Op>::value;
            const uint32_t idesc = kSwap ? idesc_bf16_f32(n_tile, kA) : idesc_bf16_f32(kTileM, n_tile);
            const int acc_n = acc_cols_of(op);
            int it = 0, lt = 0;
            for (int i = blockIdx.x; i < tiles && !abort_flag; i += gridDim.x, ++lt) {
                const Tile t = tile_of(i);
                const int buf = lt & 1;
                if (lt >= 2 && !mbar_wait(&tempty[buf], ((lt >> 1) - 1) & 1)) {
                    fail();
                    break;
                }
                tc_fence_after();
                const uint32_t dbase = tmem + (uint32_t)buf * buf_cols;
                uint32_t started = 0;
                int acc = (t.kb0 * kBlockK) / op.acc_chunk;
                int next_chunk = (acc + 1) * op.acc_chunk;
                bool ok = true;
                for (int kb = 0; kb < t.nkb; ++kb, ++it) {
                    const int s = it % kStages;
                    if (!mbar_wait(&full[s], (it / kStages) & 1)) {
                        fail();
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    const uint32_t sa = smem_u32(ring + (size_t)s * stage_bytes);
                    const uint64_t ad0 = desc_k_sw128(sa);
                    uint64_t bd0[NSPLIT];
#pragma unroll
                    for (int j = 0; j < NSPLIT; ++j)
                        bd0[j] = desc_k_sw128(sa + a_bytes + j * b_bytes);
#pragma unroll
                    for (int k16 = 0; k16 < kBlockK / 16; ++k16) {
                        const int kg = (t.kb0 + kb) * kBlockK + k16 * 16;
                        while (kg >= next_chunk && acc < op.n_acc - 1) {
                            ++acc;
                            next_chunk += op.acc_chunk;
                        }
                        const uint32_t dt = dbase + (uint32_t)(acc * acc_n);
                        const uint32_t acc_bit = 1u << acc;
#pragma unroll
                        for (int j = 0; j < NSPLIT; ++j) {
                            if constexpr (kSwap)
                                mma_bf16(dt, bd0[j] + 2 * k16, ad0 + 2 * k16, idesc,
                                         started & acc_bit);
                            else
                                mma_bf16(dt, ad0 + 2 * k16, bd0[j] + 2 * k16, idesc,
                                         started & acc_bit);
                            started |= acc_bit;
                        }
                    }
                    mma_commit(&empty[s]);
                }
                if (!ok) break;
                mma_commit(&tfull[buf]);
            }
            // every MMA issued has completed before TMEM is released
            mma_commit(&drained);
            mbar_wait(&drained, 0);
        }
        __syncwarp();
    } else {
        // epilogue warps: warp w reads TMEM lane quarter w % 4; the kEG warps
        // of a quarter take interleaved 32-column chunks (grouped ops: one
        // contiguous share of the columns each)
        constexpr int kEG = EpiWarps<Op>::value / 4;
        const int quad = warp & 3, grp = (warp - 2) >> 2;
        const int row = quad * 32 + lane;
        int lt = 0;
        for (int i = blockIdx.x; i < tiles && !abort_flag; i += gridDim.x, ++lt) {
            const Tile t = tile_of(i);
            const int buf = lt & 1;
            if (!mbar_wait(&tfull[buf], (lt >> 1) & 1)) {
                if (lane == 0) fail();
                break;
            }
            tc_fence_after();
            const uint32_t lane_base =
                tmem + (uint32_t)buf * buf_cols + ((uint32_t)(quad * 32) << 16);
            const int acc_n = acc_cols_of(op);
            if constexpr (GroupEpi<Op>::value) {
                group_epilogue<Op, kA / 16 / kEG>(op, t, row, grp * (kA / kEG), lane_base);
            } else {
                uint32_t pre = op.prefetch(t, row, grp * 32);   // one chunk ahead, as above
                for (int c0 = grp * 32; c0 < acc_n; c0 += 32 * kEG) {
                    const uint32_t cur = pre;
                    if (c0 + 32 * kEG < acc_n) pre = op.prefetch(t, row, c0 + 32 * kEG);
                    uint32_t r[kMaxAcc][32];
#pragma unroll
                    for (int a = 0; a < kMaxAcc; ++a)
                        if (a < op.n_acc)
                            tmem_ld32_nowait(lane_base + (uint32_t)(a * acc_n + c0), r[a]);
                    tmem_ld_wait();
#pragma unroll
                    for (int half = 0; half < 2; ++half) {
                        if (c0 + half * 16 >= acc_n) break;
                        float v[kMaxAcc][16];
#pragma unroll
                        for (int a = 0; a < kMaxAcc; ++a)
#pragma unroll
                            for (int q = 0; q < 16; ++q)
                                v[a][q] = __uint_as_float(r[a][half * 16 + q]);
                        op.store(t, row, c0 + half * 16, v, cur);
                    }
                }
            }
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(&tempty[buf]);
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 0) tmem_dealloc(tmem, 2 * buf_cols);
    stamp_end(op.stamp);
}

// ---- S1: query projection, split over D_i --------------------------------
// q = W_q x is written in fp32 (q_part, split 0) for the selection and as
// the three bf16 terms of the scoring contraction (qs).
struct QueryOp {
    static constexpr int kEpiWarps = 16;
    int n_tile, stages, n_acc, acc_chunk, b_split_stride;
    int *err;
    unsigned long long *stamp;   // profiling stamps of the stage, or null
    int B, HD, A, a, splits, kb_total, H, d_k, dk, r, Bmax;
    int write_qs;         // 0: the query LayerNorm writes the splits later
    float *q_part;        // [A][B][HD] (split 0 of the partial buffer)
    __nv_bfloat16 *qs;    // [2][H][Bmax][3][D_k] scaled split queries
    const float *u, *t;   // [H][r]
    __device__ int cluster_splits() const { return splits; }
    int cluster_splits_host() const { return splits; }
    __device__ Tile tile_at(int bx, int by, int bz) const {
        Tile t;
        t.m0 = bx * kTileM;
        t.n0 = by * n_tile;
        t.a_sel = 0;
        t.a_z = -1;
        t.b_z = -1;
        t.z = bz;   // the split
        const int per = (kb_total + splits - 1) / splits;
        t.kb0 = bz * per;
        t.nkb = max(0, min(kb_total, t.kb0 + per) - t.kb0);
        return t;
    }
    // q (fp32) and its two scaled splits for output row m over columns
    // n0 .. n0 + cnt - 1 of the tile (the row's coefficients looked up once)
    template <int CNT>
    __device__ void put_row(int m, int n0, const float (&v)[CNT]) const {
        const int h = m / d_k, c = m - h * d_k;
        const int k = h * r + c / dk;
        const bool row_axis = A == 1 || a == 0, col_axis = A == 1 || a == 1;
        const float cu = row_axis ? u[k] : 0.f, ct = col_axis ? t[k] : 0.f;
#pragma unroll
        for (int j = 0; j < CNT; ++j) {
            const int n = n0 + j;
            if (n >= B) break;
            q_part[((int64_t)a * B + n) * HD + m] = v[j];
            if (!write_qs) continue;
            // a shared query feeds both axes; a separate column query only axis 1
            if (row_axis) put_split_query(qs, 0, h, c, n, v[j] * cu, H, Bmax, d_k);
            if (col_axis) put_split_query(qs, 1, h, c, n, v[j] * ct, H, Bmax, d_k);
        }
    }
    __device__ uint32_t prefetch(const Tile &, int, int) const { return 0u; }
    __device__ void store(const Tile &tl, int row, int c, float (&v)[kMaxAcc][16],
                          uint32_t) const {
        const int m = tl.m0 + row;
        if (m >= HD) return;
        float w[16];
#pragma unroll
        for (int j = 0; j < 16; ++j) w[j] = tl.nkb ? v[0][j] : 0.f;
        put_row<16>(m, tl.n0 + c, w);
    }
    __device__ void store_sums(const Tile &tl, int row, int c, const float (&s4)[4]) const {
        const int m = tl.m0 + row;
        if (m < HD) put_row<4>(m, tl.n0 + c, s4);
    }
};

// ---- S2: row/column scores ---------------------------------------------------
// The B operand is the query already scaled by the axis' rank-1 coefficients
// (u or t per rank chunk), so one fp32 accumulator holds the folded score
// a = sum_alpha coef[alpha] S_alpha (Eq. 4 with Eq. 6-7) and the epilogue
// stores its order-preserving 32-bit key.
//
struct ScoreOp {
    static constexpr int kEpiWarps = 16;
    int n_tile, stages, n_acc, acc_chunk, b_split_stride;
    int *err;
    unsigned long long *stamp;   // profiling stamps of the stage, or null
    int B, H, K, kb_total;
    uint32_t *akey;       // [B][H][2][K]
    __device__ int cluster_splits() const { return 1; }
    int cluster_splits_host() const { return 1; }
    __device__ void store_sums(const Tile &, int, int, const float (&)[4]) const {}
    __device__ Tile tile_at(int bx, int by, int bz) const {
        Tile tl;
        const int h = bz >> 1, axis = bz & 1;
        tl.z = bz;   // head and axis
        tl.m0 = bx * kTileM;
        tl.n0 = by * n_tile;
        tl.a_sel = axis;
        tl.a_z = h;
        tl.b_z = axis * H + h;
        tl.kb0 = 0;
        tl.nkb = kb_total;
        return tl;
    }
    __device__ uint32_t prefetch(const Tile &, int, int) const { return 0u; }
    __device__ void store(const Tile &tl, int row, int c, float (&v)[kMaxAcc][16],
                          uint32_t) const {
        const int i = tl.m0 + row;
        if (i >= K) return;
        const int h = tl.z >> 1, axis = tl.z & 1;
        const int n0 = tl.n0 + c;
        const int64_t tok_stride = (int64_t)H * 2 * K;   // akey elements per token
        uint32_t *dst = akey + ((int64_t)n0 * H + h) * 2 * K + (int64_t)axis * K + i;
        const int nj = min(16, B - n0);
#pragma unroll
        for (int j = 0; j < 16; ++j) {
            if (j >= nj) break;
            dst[j * tok_stride] = f2ord(v[0][j]);
        }
    }
};

// Candidate lists (long grids): instead of every key, the contraction runs
// twice, with the roles of the tiles swapped (kSwapAB): 128 tokens on the
// TMEM lanes and 256 keys on the columns, so that each epilogue thread owns
// one token's scores of consecutive keys and needs no other lane.  The
// first pass (kListGroupMax) stores, per (token, head, axis), the largest
// key of each group of 16 keys.  A small kernel takes tau <= the k-th
// largest of those group maxima: k distinct groups hold a key >= tau, so
// every key of the axis' top k is >= tau.  The second pass (kListCandidates)
// recomputes the same keys (the same tiles, MMAs and order, so bit for bit)
// and writes each key >= tau, as a (key, position) composite, into its
// group's 16-entry segment of the (token, head, axis) list, and the group's
// count over its maximum.  About 2 % of the keys land in the lists, and the
// selection gets 17-25 % shorter.  Measured on GB300 (step times, graph
// replays): with 16 epilogue warps and 256-key tiles the two passes and
// the bound cost less than that saves once each SM has about 3.5 of their
// tiles (prefill of 16384 tokens 3255 -> 3083 us a step), more below (mid_4m
// with 128 tokens 65.7 -> 80.4 us), so the layer picks the form by grid.
enum { kListGroupMax = 1, kListCandidates = 2 };
constexpr int kListGroup = 16;   // keys of a group; entries of a list segment

template <int Mode>
struct ScoreListOp {
    static constexpr bool kSwapAB = true;
    static constexpr int kARows = 256;   // keys a tile: 128 x 256 MMAs
    static constexpr int kEpiWarps = 16;
    int n_tile, stages, n_acc, acc_chunk, b_split_stride;   // n_tile = 128 tokens
    int *err;
    unsigned long long *stamp;   // profiling stamps of the stage, or null
    int B, H, K, kb_total;
    int G;                        // groups of 16 keys an axis
    uint32_t *gstat;              // [B][H][2][G] group maxima, then group counts
    const uint32_t *tau;          // [B][H][2]
    unsigned long long *cand;     // [B][H][2][G][16] composites
    __device__ int cluster_splits() const { return 1; }
    int cluster_splits_host() const { return 1; }
    __device__ void store_sums(const Tile &, int, int, const float (&)[4]) const {}
    __device__ Tile tile_at(int bx, int by, int bz) const {
        Tile tl;
        const int h = bz >> 1, axis = bz & 1;
        tl.z = bz;   // head and axis
        tl.m0 = bx * kARows;   // first key
        tl.n0 = by * n_tile;   // first token
        tl.a_sel = axis;
        tl.a_z = h;
        tl.b_z = axis * H + h;
        tl.kb0 = 0;
        tl.nkb = kb_total;
        return tl;
    }
    // the bound of this thread's token (the same for every chunk)
    __device__ uint32_t prefetch(const Tile &tl, int row, int) const {
        if constexpr (Mode != kListCandidates) return 0u;
        const int n = tl.n0 + row;
        return n < B ? tau[(int64_t)n * H * 2 + tl.z] : 0xffffffffu;
    }
    static constexpr bool kGroupEpilogue = true;
    // row: the token (TMEM lane); c: the tile column of the group's first
    // key.  Returns the group's largest key (group maxima), or its count
    // after writing its keys >= t to its segment (candidates).
    __device__ uint32_t group(const Tile &tl, int row, int c, const float (&v)[16],
                              uint32_t t) const {
        const int n = tl.n0 + row;
        const int i0 = tl.m0 + c;
        if (n >= B || i0 >= K) return 0u;
        const int valid = min(kListGroup, K - i0);
        // f2ord is monotone (-0 and +0 share a key), so the maximum and the
        // comparisons are taken on the fp32 scores and only kept keys are
        // converted
        if constexpr (Mode == kListGroupMax) {
            float mx = v[0];   // valid >= 1
#pragma unroll
            for (int j = 1; j < kListGroup; ++j)
                if (j < valid) mx = fmaxf(mx, v[j]);
            return f2ord(mx);
        } else {
            const float tf = ord2f(t);   // v >= tf  <=>  f2ord(v) >= t
            unsigned long long *seg =
                cand + (((int64_t)n * H * 2 + tl.z) * G + i0 / kListGroup) * kListGroup;
            uint32_t cnt = 0u;
#pragma unroll
            for (int j = 0; j < kListGroup; ++j)
                if (j < valid && v[j] >= tf) seg[cnt++] = comp_of(f2ord(v[j]), (uint32_t)(i0 + j));
            return cnt;
        }
    }
    // the NG groups from tile column c (a multiple of 16 NG): 16-byte stores
    // when every row of gstat starts on 16 bytes (G a multiple of 4), else
    // one store per group
    template <int NG>
    __device__ void store_groups(const Tile &tl, int row, int c, const uint32_t (&g)[NG]) const {
        const int n = tl.n0 + row;
        const int gi = (tl.m0 + c) / kListGroup;
        if (n >= B || gi >= G) return;
        uint32_t *dst = gstat + ((int64_t)n * H * 2 + tl.z) * G + gi;
        if ((G & 3) == 0) {
#pragma unroll
            for (int q = 0; q < NG / 4; ++q)
                if (gi + 4 * q < G)
                    *reinterpret_cast<uint4 *>(dst + 4 * q) =
                        make_uint4(g[4 * q], g[4 * q + 1], g[4 * q + 2], g[4 * q + 3]);
        } else {
#pragma unroll
            for (int q = 0; q < NG; ++q)
                if (gi + q < G) dst[q] = g[q];
        }
    }
};


// ---- S9: IVE projection, split over E*D_v --------------------------------
struct ProjOp {
    static constexpr int kEpiWarps = 16;
    int n_tile, stages, n_acc, acc_chunk, b_split_stride;
    int *err;
    unsigned long long *stamp;   // profiling stamps of the stage, or null
    int B, d_out, kb_total, splits;
    __nv_bfloat16 *out;   // [B][d_out]
    __device__ int cluster_splits() const { return splits; }
    int cluster_splits_host() const { return splits; }
    __device__ Tile tile_at(int bx, int by, int bz) const {
        Tile t;
        t.m0 = bx * kTileM;
        t.n0 = by * n_tile;
        t.a_sel = 0;
        t.a_z = -1;
        t.b_z = -1;
        t.z = bz;   // the split
        const int per = (kb_total + splits - 1) / splits;
        t.kb0 = bz * per;
        t.nkb = max(0, min(kb_total, t.kb0 + per) - t.kb0);
        return t;
    }
    __device__ uint32_t prefetch(const Tile &, int, int) const { return 0u; }
    __device__ void store(const Tile &t, int row, int c, float (&v)[kMaxAcc][16],
                          uint32_t) const {
        const int o = t.m0 + row;
        if (o >= d_out) return;
#pragma unroll
        for (int j = 0; j < 16; ++j) {
            const int n = t.n0 + c + j;
            if (n >= B) break;
            out[(int64_t)n * d_out + o] = __float2bfloat16_rn(t.nkb ? v[0][j] : 0.f);
        }
    }
    __device__ void store_sums(const Tile &t, int row, int c, const float (&s4)[4]) const {
        const int o = t.m0 + row;
        if (o >= d_out) return;
#pragma unroll
        for (int e = 0; e < 4; ++e) {
            const int n = t.n0 + c + e;
            if (n < B) out[(int64_t)n * d_out + o] = __float2bfloat16_rn(s4[e]);
        }
    }
};

// The backward's dacc = W_p g (the projectors as stored, [E D_v][D'_v], are
// the K-major A operand; the gradient rows g [B][D'_v] the B operand): fp32
// rows dacc[B][E D_v], unsplit.
struct DaccOp {
    int n_tile, stages, n_acc, acc_chunk, b_split_stride;
    int *err;
    unsigned long long *stamp;   // profiling stamps of the stage, or null
    int B, M, kb_total;
    float *out;   // [B][M]
    __device__ int cluster_splits() const { return 1; }
    int cluster_splits_host() const { return 1; }
    __device__ void store_sums(const Tile &, int, int, const float (&)[4]) const {}
    __device__ Tile tile_at(int bx, int by, int) const {
        Tile t;
        t.m0 = bx * kTileM;
        t.n0 = by * n_tile;
        t.a_sel = 0;
        t.a_z = -1;
        t.b_z = -1;
        t.z = 0;
        t.kb0 = 0;
        t.nkb = kb_total;
        return t;
    }
    __device__ uint32_t prefetch(const Tile &, int, int) const { return 0u; }
    __device__ void store(const Tile &t, int row, int c, float (&v)[kMaxAcc][16],
                          uint32_t) const {
        const int o = t.m0 + row;
        if (o >= M) return;
#pragma unroll
        for (int j = 0; j < 16; ++j) {
            const int n = t.n0 + c + j;
            if (n >= B) break;
            out[(int64_t)n * M + o] = t.nkb ? v[0][j] : 0.f;
        }
    }
};

// The backward's dW_p = sum_tokens acc_p g^T, computed transposed: A = the
// gradient rows transposed ([D'_v][B] bf16, K = tokens), B = the pooled rows
// transposed as two bf16 terms hi + lo ([E D_v][2 B], the lo term at column
// offset B), both terms multiplying each A tile into one accumulator (the
// pooled rows to 2^-16 relative, as in the forward's projection).  Tile
// rows are outputs o, columns are pooled entries c; fp32 dW [E D_v][D'_v]
// row-major, unsplit.
struct DwOp {
    int n_tile, stages, n_acc, acc_chunk, b_split_stride;
    int *err;
    unsigned long long *stamp;   // profiling stamps of the stage, or null
    int M, N, kb_total;   // M = D'_v (rows o), N = E D_v (columns c)
    float *out;           // [N][M]
    __device__ int cluster_splits() const { return 1; }
    int cluster_splits_host() const { return 1; }
    __device__ void store_sums(const Tile &, int, int, const float (&)[4]) const {}
    __device__ Tile tile_at(int bx, int by, int) const {
        Tile t;
        t.m0 = bx * kTileM;
        t.n0 = by * n_tile;
        t.a_sel = 0;
        t.a_z = -1;
        t.b_z = -1;
        t.z = 0;
        t.kb0 = 0;
        t.nkb = kb_total;
        return t;
    }
    __device__ uint32_t prefetch(const Tile &, int, int) const { return 0u; }
    __device__ void store(const Tile &t, int row, int c, float (&v)[kMaxAcc][16],
                          uint32_t) const {
        const int o = t.m0 + row;
        if (o >= M) return;
        // dW[n][o]: a warp's 32 rows o are contiguous for each column n
#pragma unroll
        for (int j = 0; j < 16; ++j) {
            const int n = t.n0 + c + j;
            if (n < N) out[(int64_t)n * M + o] = t.nkb ? v[0][j] : 0.f;
        }
    }
};

// dst[c][r] = src[r][c] for a rows x cols bf16 matrix (32 x 32 tiles), with
// row strides ld_src (>= cols) and ld_dst (>= rows) in elements
__global__ void transpose_kernel(const __nv_bfloat16 *__restrict__ src,
                                 __nv_bfloat16 *__restrict__ dst, int rows, int cols,
                                 int64_t ld_src, int64_t ld_dst) {
    __shared__ __nv_bfloat16 tile[32][33];
    const int c0 = blockIdx.x * 32, r0 = blockIdx.y * 32;
    for (int i = threadIdx.y; i < 32; i += blockDim.y) {
        const int r = r0 + i, c = c0 + threadIdx.x;
        if (r < rows && c < cols) tile[i][threadIdx.x] = src[(int64_t)r * ld_src + c];
    }
    __syncthreads();
    for (int i = threadIdx.y; i < 32; i += blockDim.y) {
        const int c = c0 + i, r = r0 + threadIdx.x;
        if (r < rows && c < cols) dst[(int64_t)c * ld_dst + r] = tile[threadIdx.x][i];
    }
}

PFN_cuTensorMapEncodeTiled_v12000 g_encode = nullptr;

}  // namespace

cudaError_t launch_transpose_bf16(const void *src, void *dst, int rows, int cols,
                                  cudaStream_t st, int64_t ld_src, int64_t ld_dst) {
    dim3 grid((cols + 31) / 32, (rows + 31) / 32);
    transpose_kernel<<<grid, dim3(32, 8), 0, st>>>(static_cast<const __nv_bfloat16 *>(src),
                                                   static_cast<__nv_bfloat16 *>(dst), rows, cols,
                                                   ld_src > 0 ? ld_src : cols,
                                                   ld_dst > 0 ? ld_dst : rows);
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

static int sm_count() { return device_sm_count(); }

// TMEM columns of one accumulator buffer: the epilogue reads 32 columns at a
// time, so cover the last such read, rounded to 32.
static uint32_t buf_cols_of(int n_acc, int n_tile) {
    const uint32_t c = (uint32_t)((n_acc - 1) * n_tile + ((n_tile - 1) / 32) * 32 + 32);
    return (c + 31) & ~31u;
}

// The persistent kernel serves grids with more tiles than SMs, no split-K and
// two accumulator buffers within TMEM's 512 columns; returns false when it
// does not apply.
template <int NSPLIT, class Op>
static bool persistent_ok(dim3 grid, const Op &op) {
    const uint32_t bc = buf_cols_of(op.n_acc, acc_cols_of(op));
    return grid.z >= 1 && op.cluster_splits_host() == 1 &&
           (int)(grid.x * grid.y * grid.z) > sm_count() && 2 * bc <= 512 &&
           tmem_cols_for(2 * bc) == 2 * bc;
}

template <int NSPLIT, class Op>
static cudaError_t launch_gemm_persistent(dim3 grid, const CUtensorMap &a0, const CUtensorMap &a1,
                                          const CUtensorMap &b, Op op, int nkb, bool pdl,
                                          cudaStream_t st, int probe) {
    (void)nkb;   // the ring runs across tiles: as many stages as fit
    constexpr int kA = ARows<Op>::value;
    op.stages = stages_for(NSPLIT, op.n_tile, kMaxStages, kA);
    const size_t smem = 1024 + (size_t)op.stages * stage_bytes_of(NSPLIT, op.n_tile, kA);
    const int tiles = (int)(grid.x * grid.y * grid.z);
    const int ctas = tiles < sm_count() ? tiles : sm_count();
    return launch_kernel(pdl, tc_gemm_persistent<NSPLIT, Op>, dim3(ctas),
                         persistent_threads<Op>(), smem, st, a0,
                         a1, b, op, (int)grid.x, (int)grid.y, tiles,
                         buf_cols_of(op.n_acc, acc_cols_of(op)), probe);
}

// grid.z = the split count (S1, S9; also the cluster's z extent when > 1) or
// the head/axis (S2)
template <int NSPLIT, class Op>
static cudaError_t launch_gemm(dim3 grid, const CUtensorMap &a0, const CUtensorMap &a1,
                               const CUtensorMap &b, Op op, int nkb, bool pdl,
                               cudaStream_t st, int probe = 0) {
    if (persistent_ok<NSPLIT>(grid, op))
        return launch_gemm_persistent<NSPLIT>(grid, a0, a1, b, op, nkb, pdl, st, probe);
    // the split-K epilogue adds up one accumulator
    if (op.cluster_splits_host() > 1 && op.n_acc != 1) return cudaErrorInvalidValue;
    constexpr int kA = ARows<Op>::value;
    op.stages = stages_for(NSPLIT, op.n_tile, nkb, kA);
    const size_t ring = (size_t)op.stages * stage_bytes_of(NSPLIT, op.n_tile, kA);
    const size_t split = split_buf_bytes(op.n_tile, op.cluster_splits_host());
    const size_t smem = 1024 + (ring > split ? ring : split);
    if (smem > kSmemBudget) return cudaErrorInvalidValue;   // the split buffers do not fit
    return launch_kernel(pdl, grid.z > 1 ? grid.z : 1u, tc_gemm_kernel<NSPLIT, Op>, grid,
                         kThreads, smem, st, a0, a1, b, op, probe);
}

template <int NSPLIT, class Op> static cudaError_t allow_smem() {
    cudaError_t e = cudaFuncSetAttribute(tc_gemm_kernel<NSPLIT, Op>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)kSmemBudget);
    if (e == cudaSuccess)
        e = cudaFuncSetAttribute(tc_gemm_persistent<NSPLIT, Op>,
                                 cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kSmemBudget);
    return e;
}

cudaError_t configure_tc() {
    cudaError_t e = allow_smem<1, QueryOp>();
    if (e == cudaSuccess) e = allow_smem<3, QueryOp>();
    if (e == cudaSuccess) e = allow_smem<3, ScoreOp>();
    if (e == cudaSuccess) e = allow_smem<3, ScoreListOp<kListGroupMax>>();
    if (e == cudaSuccess) e = allow_smem<3, ScoreListOp<kListCandidates>>();
    if (e == cudaSuccess) e = allow_smem<2, ProjOp>();
    if (e == cudaSuccess) e = allow_smem<1, DaccOp>();
    if (e == cudaSuccess) e = allow_smem<2, DwOp>();
    return e;
}

cudaError_t launch_dw_tc(const Dims &d, const CUtensorMap &g_t, const CUtensorMap &acc_t2,
                         float *dW, int *err, cudaStream_t st) {
    DwOp op;
    op.stamp = nullptr;
    op.M = d.d_out;
    op.N = d.E * d.d_v;
    op.n_tile = tc_n_tile(op.N, 1);
    op.n_acc = 1;
    op.acc_chunk = 1 << 30;
    op.b_split_stride = d.B;   // the lo term's columns follow the hi term's
    op.err = err;
    op.kb_total = (d.B + kBlockK - 1) / kBlockK;
    op.out = dW;
    dim3 grid((op.M + kTileM - 1) / kTileM, (op.N + op.n_tile - 1) / op.n_tile, 1);
    return launch_gemm<2>(grid, g_t, g_t, acc_t2, op, op.kb_total, false, st);
}

cudaError_t launch_dacc_tc(const Dims &d, const CUtensorMap &w_p, const CUtensorMap &g,
                           float *dacc, int *err, cudaStream_t st) {
    DaccOp op;
    op.stamp = nullptr;
    op.n_tile = tc_n_tile(d.B, 1);
    op.n_acc = 1;
    op.acc_chunk = 1 << 30;
    op.b_split_stride = 0;
    op.err = err;
    op.B = d.B;
    op.M = d.E * d.d_v;
    op.kb_total = (d.d_out + kBlockK - 1) / kBlockK;
    op.out = dacc;
    dim3 grid((op.M + kTileM - 1) / kTileM, (d.B + op.n_tile - 1) / op.n_tile, 1);
    return launch_gemm<1>(grid, w_p, w_p, g, op, op.kb_total, false, st);
}

// x_splits: the B operand is the convolved input as three bf16 terms (map
// xs over [B][3 D_i]), contracted as three MMAs into one accumulator
cudaError_t launch_query_tc(const Dims &d, const Ptrs &p, const TcMaps &mp, int splits,
                            __nv_bfloat16 *qs, int Bmax, bool x_splits, bool write_qs,
                            bool pdl, cudaStream_t st) {
    const int HD = d.H * d.d_k;
    const int n_tile = d.q_ntile ? d.q_ntile : tc_n_tile(d.B, 1);
    const int kb_total = (d.d_in + kBlockK - 1) / kBlockK;
    if (splits > kMaxSplits) return cudaErrorInvalidValue;
    for (int a = 0; a < d.A; ++a) {
        QueryOp op;
    op.stamp = p.stamp;
        op.n_tile = n_tile;
        op.n_acc = 1;
        op.acc_chunk = 1 << 30;
        op.b_split_stride = x_splits ? d.d_in : 0;
        op.write_qs = write_qs ? 1 : 0;
        op.err = p.err;
        op.B = d.B;
        op.HD = HD;
        op.A = d.A;
        op.a = a;
        op.splits = splits;
        op.kb_total = kb_total;
        op.H = d.H;
        op.d_k = d.d_k;
        op.dk = d.dk;
        op.r = d.r;
        op.Bmax = Bmax;
        op.q_part = p.q_part;
        op.qs = qs;
        op.u = p.u;
        op.t = p.t;
        dim3 grid((HD + kTileM - 1) / kTileM, (d.B + n_tile - 1) / n_tile, splits);
        const int per = (kb_total + splits - 1) / splits;
        const CUtensorMap &wa = a == 0 ? mp.w_q : mp.w_q_col;
        // the first query waits for all earlier work on the stream, unless it
        // follows this call's convolution
        cudaError_t e = x_splits ? launch_gemm<3>(grid, wa, mp.w_q, mp.xs, op, per, pdl && a == 0, st)
                                 : launch_gemm<1>(grid, wa, mp.w_q, mp.x, op, per, pdl && a == 0, st);
        if (e != cudaSuccess) return e;
    }
    return cudaSuccess;
}

cudaError_t launch_score_keys(const Dims &d, const Ptrs &p, const TcMaps &mp, int probe,
                              cudaStream_t st) {
    ScoreOp op;
    op.stamp = p.stamp;
    op.n_tile = tc_n_tile(d.B, 1);
    op.n_acc = 1;
    op.acc_chunk = 1 << 30;
    op.b_split_stride = d.d_k;
    op.err = p.err;
    op.B = d.B;
    op.H = d.H;
    op.K = d.K;
    op.kb_total = (d.d_k + kBlockK - 1) / kBlockK;
    op.akey = p.akey;
    dim3 grid((d.K + kTileM - 1) / kTileM, (d.B + op.n_tile - 1) / op.n_tile, 2 * d.H);
    return launch_gemm<3>(grid, mp.k_row, mp.k_col, mp.qs, op, op.kb_total, d.pdl, st, probe);
}

// one pass of the candidate-list scoring (128 tokens a tile, map qs_t)
template <int Mode>
static cudaError_t score_list_pass(const Dims &d, const Ptrs &p, const TcMaps &mp, int probe,
                                   cudaStream_t st) {
    ScoreListOp<Mode> op;
    op.stamp = p.stamp;
    op.n_tile = kTileM;
    op.n_acc = 1;
    op.acc_chunk = 1 << 30;
    op.b_split_stride = d.d_k;
    op.err = p.err;
    op.B = d.B;
    op.H = d.H;
    op.K = d.K;
    op.kb_total = (d.d_k + kBlockK - 1) / kBlockK;
    op.G = d.n_groups;
    op.gstat = p.gstat;
    op.tau = p.tau;
    op.cand = p.cand;
    constexpr int kA = ScoreListOp<Mode>::kARows;
    dim3 grid((d.K + kA - 1) / kA, (d.B + op.n_tile - 1) / op.n_tile, 2 * d.H);
    return launch_gemm<3>(grid, mp.k_row, mp.k_col, mp.qs_t, op, op.kb_total, d.pdl, st, probe);
}

cudaError_t launch_score_tc(const Dims &d, const Ptrs &p, const TcMaps &mp, cudaStream_t st) {
    if (d.cand) {
        // group maxima, the bound, then the lists (three dependent launches)
        cudaError_t e = score_list_pass<kListGroupMax>(d, p, mp, d.probe_wait, st);
        if (e == cudaSuccess) e = launch_cand_bound(d, p, st);
        if (e == cudaSuccess) e = score_list_pass<kListCandidates>(d, p, mp, 0, st);
        return e;
    }
    return launch_score_keys(d, p, mp, d.probe_wait, st);
}

cudaError_t launch_proj_tc(const Dims &d, const Ptrs &p, const TcMaps &mp, cudaStream_t st) {
    if (d.p_splits > kMaxSplits) return cudaErrorInvalidValue;
    ProjOp op;
    op.stamp = p.stamp;
    op.n_tile = d.p_ntile ? d.p_ntile : tc_n_tile(d.B, 1);
    op.n_acc = 1;
    op.acc_chunk = 1 << 30;
    // the pooled rows are two bf16 terms hi + lo ([B][2][E D_v]): both
    // multiply each projector tile into one fp32 accumulator, so the operand
    // carries the pooled value to 2^-16 relative instead of one rounding
    op.b_split_stride = d.E * d.d_v;
    op.err = p.err;
    op.B = d.B;
    op.d_out = d.d_out;
    op.kb_total = (d.E * d.d_v + kBlockK - 1) / kBlockK;
    op.splits = d.p_splits;
    op.out = static_cast<__nv_bfloat16 *>(p.out);
    dim3 grid((d.d_out + kTileM - 1) / kTileM, (d.B + op.n_tile - 1) / op.n_tile, op.splits);
    const int per = (op.kb_total + op.splits - 1) / op.splits;
    return launch_gemm<2>(grid, mp.w_pt, mp.w_pt, mp.acc, op, per, d.pdl, st);
}

}  // namespace um
