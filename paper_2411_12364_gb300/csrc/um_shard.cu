// um_shard.cu -- the local steps of the number-wise partitioned table
// (App. D): route the selected slots to the ranks that own their rows, look
// rows up in this rank's shard, and turn the rows returned by the owners
// into the per-slot (row, block, weight) the gather pools (Eq. 14-15).
// The exchanges between the steps are the caller's all-to-alls.
#include "um_internal.cuh"

namespace um {
namespace {

constexpr int kThreads = 256;
constexpr int kMaxOwners = 1024;

// The slot's physical row after the shuffle (Eq. 14); an address outside
// [0, E N) is recorded and read as address 0.
__device__ __forceinline__ uint64_t slot_row(const Dims &d, const Ptrs &p, int64_t s, bool *bad) {
    int64_t v = p.idx_in[s];
    *bad = v < 0 || (uint64_t)v >= d.M;
    if (*bad) v = 0;
    const uint64_t vs = shuffle_address(d, p.perm, (uint64_t)v);
    return vs % (uint64_t)d.N;
}

// counts[q] = slots whose row the owner q holds (counts zeroed before).
__global__ void route_count_kernel(Dims d, Ptrs p, int P, int64_t rows_per_rank, int *counts) {
    const int64_t S = (int64_t)d.B * d.H * d.m;
    for (int64_t s = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; s < S;
         s += (int64_t)gridDim.x * blockDim.x) {
        bool bad;
        const uint64_t row = slot_row(d, p, s, &bad);
        if (bad) atomicOr(p.err, kErrBadIndex);
        atomicAdd(&counts[(int)(row / (uint64_t)rows_per_rank)], 1);
    }
}

// Each slot takes the next free place in its owner's block of send_rows
// (the blocks in owner order, offsets from the counts; cursor zeroed before).
__global__ void route_scatter_kernel(Dims d, Ptrs p, int P, int64_t rows_per_rank,
                                     const int *counts, int *cursor, int32_t *send_rows,
                                     int32_t *slot_pos) {
    __shared__ int off[kMaxOwners];
    if (threadIdx.x == 0) {
        int run = 0;
        for (int q = 0; q < P; ++q) {
            off[q] = run;
            run += counts[q];
        }
    }
    __syncthreads();
    const int64_t S = (int64_t)d.B * d.H * d.m;
    for (int64_t s = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; s < S;
         s += (int64_t)gridDim.x * blockDim.x) {
        bool bad;
        const uint64_t row = slot_row(d, p, s, &bad);
        const int q = (int)(row / (uint64_t)rows_per_rank);
        const int pos = off[q] + atomicAdd(&cursor[q], 1);
        send_rows[pos] = (int32_t)(row - (uint64_t)q * (uint64_t)rows_per_rank);
        slot_pos[s] = pos;
    }
}

// out[i] = shard row rows[i], 16-byte vectors; a row outside [0, shard_rows)
// is recorded and returned as zeros.
__global__ void shard_lookup_kernel(const uint4 *__restrict__ V, int64_t shard_rows, int vpr,
                                    const int32_t *__restrict__ rows, int64_t n,
                                    uint4 *__restrict__ out, int *err) {
    const int64_t total = n * vpr;
    for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < total;
         i += (int64_t)gridDim.x * blockDim.x) {
        const int64_t r = i / vpr;
        const int c = (int)(i - r * vpr);
        const int32_t row = rows[r];
        const bool ok = row >= 0 && row < shard_rows;
        if (!ok && c == 0) atomicOr(err, kErrBadIndex);
        out[i] = ok ? V[(int64_t)row * vpr + c] : make_uint4(0, 0, 0, 0);
    }
}

// The gather's per-slot inputs for rows returned by their owners: slot s
// reads row slot_pos[s] of the returned rows, in block p of its shuffled
// address, with its weight(s); an address outside [0, E N) gets weight 0.
__global__ void shard_slots_kernel(Dims d, Ptrs p, const int32_t *slot_pos) {
    const int64_t S = (int64_t)d.B * d.H * d.m;
    for (int64_t s = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; s < S;
         s += (int64_t)gridDim.x * blockDim.x) {
        int64_t v = p.idx_in[s];
        const bool bad = v < 0 || (uint64_t)v >= d.M;
        if (bad) v = 0;
        const uint64_t vs = shuffle_address(d, p.perm, (uint64_t)v);
        p.sel_p[s] = (int32_t)(vs / (uint64_t)d.N);
        p.sel_row[s] = slot_pos[s];
        for (int ci = 0; ci < d.nc; ++ci)
            p.sel_w[s * d.nc + ci] = bad ? 0.f : p.w_in[s * d.nc + ci];
    }
}

int blocks_for(int64_t work) {
    int64_t b = (work + kThreads - 1) / kThreads;
    if (b > 4096) b = 4096;
    return b < 1 ? 1 : (int)b;
}

}  // namespace

cudaError_t launch_shard_route(const Dims &d, const Ptrs &p, int P, int64_t rows_per_rank,
                               int *counts, int *cursor, int32_t *send_rows, int32_t *slot_pos,
                               cudaStream_t st) {
    if (P < 1 || P > kMaxOwners) return cudaErrorInvalidValue;
    const int64_t S = (int64_t)d.B * d.H * d.m;
    cudaError_t e = cudaMemsetAsync(counts, 0, sizeof(int) * P, st);
    if (e == cudaSuccess) e = cudaMemsetAsync(cursor, 0, sizeof(int) * P, st);
    if (e != cudaSuccess) return e;
    route_count_kernel<<<blocks_for(S), kThreads, 0, st>>>(d, p, P, rows_per_rank, counts);
    route_scatter_kernel<<<blocks_for(S), kThreads, 0, st>>>(d, p, P, rows_per_rank, counts,
                                                            cursor, send_rows, slot_pos);
    return cudaGetLastError();
}

cudaError_t launch_shard_lookup(const void *values, int64_t shard_rows, int row_bytes,
                                const int32_t *rows, int64_t n, void *out, int *err,
                                cudaStream_t st) {
    const int vpr = row_bytes / 16;
    shard_lookup_kernel<<<blocks_for(n * vpr), kThreads, 0, st>>>(
        static_cast<const uint4 *>(values), shard_rows, vpr, rows, n, static_cast<uint4 *>(out),
        err);
    return cudaGetLastError();
}

cudaError_t launch_shard_slots(const Dims &d, const Ptrs &p, const int32_t *slot_pos,
                               cudaStream_t st) {
    const int64_t S = (int64_t)d.B * d.H * d.m;
    shard_slots_kernel<<<blocks_for(S), kThreads, 0, st>>>(d, p, slot_pos);
    return cudaGetLastError();
}

}  // namespace um
