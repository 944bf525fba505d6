// um_gather.cu -- S8 (weighted gather-sum grouped by virtual block, Eq. 15's
// inner V^T s^_p) and S9 on CUDA cores (the IVE projection o = sum_p W_p^T
// acc_p, used for fp32 storage; there with compensated sums, Dot2).
//
// Gather, one CTA per token.  Random 512-byte rows of a multi-GB table reach
// the HBM copy rate only with many rows in flight per SM (measured on GB300:
// about 6.8 TB/s from 32 warps per SM with 8 rows each), so the main kernel
// keeps few registers per thread:
//   * the token's H*m slots are bucketed by virtual block p with a stable
//     counting sort in shared memory (ballots per block, a scan over warps);
//   * each warp serves one block, so a lane owns 16 bytes of every row and
//     8 fp32 accumulators, and issues 8 row loads before using any;
//   * 16 warps per CTA, two CTAs per SM; the warps of a block are summed in a
//     fixed order at the end (deterministic).
// Wider rows or more slots take the per-lane multi-block kernels below.  Row
// loads bypass L1 (read-only path).
//
// fp32 storage accumulates in fp64 (products of two fp32 values are exact
// there): the fp32 mode's outputs carry the working precision element by
// element (see Dot2 in um_internal.cuh), and its projection reads fp32
// pooled rows that are rounded once.
//
// Multi-Core Scoring (Eq. 17): a slot has nc weights and weight i scales
// columns [i*D_v/nc, (i+1)*D_v/nc) of the row.  Slices are whole 16-byte
// vectors (D_v/nc is a multiple of 8), so a lane's vector lies in one slice
// and the lane picks that slice's weight.
#include "um_internal.cuh"

namespace um {
namespace {

constexpr int kThreads = 256;
constexpr int kWarps = kThreads / 32;
constexpr int kUnroll = 8;   // rows in flight per warp

__device__ __forceinline__ uint4 ld_stream(const void *ptr) {
    uint4 v;
    asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0,%1,%2,%3}, [%4];"
                 : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
                 : "l"(ptr));
    return v;
}

// The accumulator type of a gather: fp64 for fp32 storage, else fp32.
template <typename T>
using AccOf = typename std::conditional<std::is_same<T, float>::value, double, float>::type;

__device__ __forceinline__ float mul_add(float w, float v, float acc) { return fmaf(w, v, acc); }
__device__ __forceinline__ double mul_add(float w, float v, double acc) {
    return fma((double)w, (double)v, acc);
}

// add w * (8 bf16 or 4 fp32 packed in 16 bytes) into dst
template <typename A>
__device__ __forceinline__ void fma_vec(A *dst, uint4 v, float w, __nv_bfloat16) {
    const uint32_t u[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
    for (int q = 0; q < 4; ++q) {
        float lo = __uint_as_float(u[q] << 16), hi = __uint_as_float(u[q] & 0xffff0000u);
        dst[2 * q] = mul_add(w, lo, dst[2 * q]);
        dst[2 * q + 1] = mul_add(w, hi, dst[2 * q + 1]);
    }
}
template <typename A>
__device__ __forceinline__ void fma_vec(A *dst, uint4 v, float w, float) {
    dst[0] = mul_add(w, __uint_as_float(v.x), dst[0]);
    dst[1] = mul_add(w, __uint_as_float(v.y), dst[1]);
    dst[2] = mul_add(w, __uint_as_float(v.z), dst[2]);
    dst[3] = mul_add(w, __uint_as_float(v.w), dst[3]);
}

template <typename T>
__device__ __forceinline__ void unpack(uint4 v, float (&f)[16 / sizeof(T)]);
template <>
__device__ __forceinline__ void unpack<__nv_bfloat16>(uint4 v, float (&f)[8]) {
    const uint32_t u[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
    for (int q = 0; q < 4; ++q) {
        f[2 * q] = __uint_as_float(u[q] << 16);
        f[2 * q + 1] = __uint_as_float(u[q] & 0xffff0000u);
    }
}
template <>
__device__ __forceinline__ void unpack<float>(uint4 v, float (&f)[4]) {
    f[0] = __uint_as_float(v.x);
    f[1] = __uint_as_float(v.y);
    f[2] = __uint_as_float(v.z);
    f[3] = __uint_as_float(v.w);
}

// Register-accumulating gather for E <= EMAX blocks and rows of at most
// 32 vectors (one 16-byte vector per lane).  Each warp takes a contiguous
// run of the token's H*m slots; their (row, block, weight) are loaded once,
// one slot per lane, and broadcast by shuffle; 8 value loads per warp are
// in flight together.
template <typename T, int EMAX>
__global__ void __launch_bounds__(kThreads) gather_reg_kernel(Dims d, Ptrs p) {
    using A = AccOf<T>;
    extern __shared__ __align__(16) unsigned char red_raw[];
    A *red = reinterpret_cast<A *>(red_raw);   // [kWarps][E][D_v]
    constexpr int EPV = 16 / sizeof(T);
    const int b = blockIdx.x;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int EDv = d.E * d.d_v;
    const int VPR = d.d_v / EPV;          // vectors per row, <= 32 here
    const bool active = lane < VPR;
    const int hm = d.H * d.m;
    const int64_t base = (int64_t)b * hm;
    const T *V = static_cast<const T *>(p.values) + lane * EPV;
    const int per_warp = (hm + kWarps - 1) / kWarps;
    const int e_begin = min(hm, warp * per_warp), e_end = min(hm, e_begin + per_warp);
    pdl_wait();
    stamp_begin(p.stamp);
    pdl_trigger();
    A acc[EMAX][EPV];
#pragma unroll
    for (int q = 0; q < EMAX; ++q)
#pragma unroll
        for (int c = 0; c < EPV; ++c) acc[q][c] = 0;

    for (int c0 = e_begin; c0 < e_end; c0 += 32) {
        const int n = min(32, e_end - c0);
        int row_l = 0, blk_l = -1;
        float w_l = 0.f;
        if (lane < n) {
            row_l = p.sel_row[base + c0 + lane];
            blk_l = p.sel_p[base + c0 + lane];
            w_l = p.sel_w[base + c0 + lane];
        }
        for (int j0 = 0; j0 < n; j0 += kUnroll) {
            uint4 val[kUnroll];
#pragma unroll
            for (int u = 0; u < kUnroll; ++u) {
                const int j = j0 + u;
                const int row = __shfl_sync(0xffffffffu, row_l, j & 31);
                val[u] = (j < n && active) ? ld_stream(V + (int64_t)row * d.d_v)
                                           : make_uint4(0, 0, 0, 0);
            }
#pragma unroll
            for (int u = 0; u < kUnroll; ++u) {
                const int j = j0 + u;
                const int blk = __shfl_sync(0xffffffffu, blk_l, j & 31);
                const float w = j < n ? __shfl_sync(0xffffffffu, w_l, j & 31) : 0.f;
                float f[EPV];
                unpack<T>(val[u], f);
#pragma unroll
                for (int q = 0; q < EMAX; ++q) {
                    const float wq = blk == q ? w : 0.f;   // branch-free block select
#pragma unroll
                    for (int c = 0; c < EPV; ++c) acc[q][c] = mul_add(wq, f[c], acc[q][c]);
                }
            }
        }
    }
    // sum the warps' partial accumulators
    if (active)
#pragma unroll
        for (int q = 0; q < EMAX; ++q)
            if (q < d.E)
#pragma unroll
                for (int c = 0; c < EPV; ++c)
                    red[(size_t)warp * EDv + q * d.d_v + lane * EPV + c] = acc[q][c];
    __syncthreads();
    for (int i = threadIdx.x; i < EDv; i += kThreads) {
        A s = 0;
#pragma unroll
        for (int wv = 0; wv < kWarps; ++wv) s += red[(size_t)wv * EDv + i];
        store_pooled<T>(d, p, b, i, (float)s);
    }
    stamp_end(p.stamp);
}

constexpr int kBMaxE = 16;
constexpr int kMaxCores = 8;   // MCS component cores per head

// bytes of one accumulator of the layer's gather (fp64 for fp32 storage)
size_t acc_bytes(const Dims &d) { return d.dtype == ULTRAMEM_F32 ? 8 : 4; }

size_t bucket_smem_bytes(const Dims &d, int warps) {
    const int hm = d.H * d.m;
    return acc_bytes(d) * (size_t)warps * d.d_v + sizeof(int) * (size_t)hm +
           sizeof(float) * (size_t)hm * d.nc;
}

// THREADS = 512 (2 CTAs per SM) for batches up to about two CTAs per SM,
// where each token's latency matters; 256 (4 CTAs per SM) for longer
// grids, where CTAs in their bucketing or reduction phase overlap others'
// loads (measured: 6.5 TB/s over 2.15 GB at 16384 tokens, against 5.4 with
// 512).
template <typename T, int THREADS>
__global__ void __launch_bounds__(THREADS, 1024 / THREADS) gather_bucket_kernel(Dims d, Ptrs p) {
    constexpr int kBThreads = THREADS, kBWarps = THREADS / 32;
    extern __shared__ __align__(16) unsigned char gsm[];
    __shared__ int wcnt[kBWarps][kBMaxE];   // per warp and block: count, then offset
    __shared__ int tot[kBMaxE], start[kBMaxE];
    constexpr int EPV = 16 / sizeof(T);
    using A = AccOf<T>;
    const int b = blockIdx.x, E = d.E, hm = d.H * d.m, Dv = d.d_v;
    const int t = threadIdx.x, warp = t >> 5, lane = t & 31;
    const int64_t base = (int64_t)b * hm;
    A *red = reinterpret_cast<A *>(gsm);                         // [kBWarps][D_v]
    int *row_s = reinterpret_cast<int *>(red + kBWarps * Dv);    // [hm] bucketed rows
    float *w_s = reinterpret_cast<float *>(row_s + hm);          // [hm][nc] their weights
    const int nc = d.nc;
    pdl_wait();
    stamp_begin(p.stamp);
    pdl_trigger();

    // stable counting sort of the slots by block (slot order kept within a block)
    int row = 0, blk = -1;
    float w[kMaxCores];   // the slot's weight, or its nc slice weights (MCS)
#pragma unroll
    for (int ci = 0; ci < kMaxCores; ++ci) w[ci] = 0.f;
    if (t < hm) {
        row = p.sel_row[base + t];
        blk = p.sel_p[base + t];
#pragma unroll
        for (int ci = 0; ci < kMaxCores; ++ci)
            if (ci < nc) w[ci] = p.sel_w[(base + t) * nc + ci];
        if (blk < 0 || blk >= E) blk = -1;   // not a slot of this layer: skipped
    }
    int rank = 0;
    for (int q = 0; q < E; ++q) {
        const unsigned m = __ballot_sync(0xffffffffu, blk == q);
        if (blk == q) rank = __popc(m & ((1u << lane) - 1u));
        if (lane == 0) wcnt[warp][q] = __popc(m);
    }
    __syncthreads();
    if (t < E) {
        int run = 0;
        for (int wv = 0; wv < kBWarps; ++wv) {
            const int c = wcnt[wv][t];
            wcnt[wv][t] = run;
            run += c;
        }
        tot[t] = run;
    }
    __syncthreads();
    if (t == 0) {
        int run = 0;
        for (int q = 0; q < E; ++q) {
            start[q] = run;
            run += tot[q];
        }
    }
    __syncthreads();
    if (blk >= 0) {
        const int pos = start[blk] + wcnt[warp][blk] + rank;
        row_s[pos] = row;
#pragma unroll
        for (int ci = 0; ci < kMaxCores; ++ci)
            if (ci < nc) w_s[pos * nc + ci] = w[ci];
    }
    __syncthreads();

    // warps [q*wpb, (q+1)*wpb) serve block q, each a contiguous share
    const int wpb = kBWarps / E;
    const int q = warp / wpb, sub = warp - q * wpb;
    const bool active = lane * EPV < Dv;
    const int wsel = nc == 1 || !active ? 0 : (lane * EPV) / (Dv / nc);   // this lane's slice
    const T *V = static_cast<const T *>(p.values) + lane * EPV;
    A acc[EPV];
#pragma unroll
    for (int c = 0; c < EPV; ++c) acc[c] = 0;
    if (q < E) {
        const int n = tot[q], per = (n + wpb - 1) / wpb;
        const int lo = start[q] + min(n, sub * per), hi = start[q] + min(n, (sub + 1) * per);
        for (int j0 = lo; j0 < hi; j0 += kUnroll) {
            uint4 val[kUnroll];
            float wu[kUnroll];
#pragma unroll
            for (int u = 0; u < kUnroll; ++u) {
                const int j = j0 + u;
                const bool ok = j < hi;
                wu[u] = ok ? w_s[j * nc + wsel] : 0.f;
                val[u] = (ok && active) ? ld_stream(V + (int64_t)row_s[j] * Dv)
                                        : make_uint4(0, 0, 0, 0);
            }
#pragma unroll
            for (int u = 0; u < kUnroll; ++u) {
                float f[EPV];
                unpack<T>(val[u], f);
#pragma unroll
                for (int c = 0; c < EPV; ++c) acc[c] = mul_add(wu[u], f[c], acc[c]);
            }
        }
        if (active)
#pragma unroll
            for (int c = 0; c < EPV; ++c) red[warp * Dv + lane * EPV + c] = acc[c];
    }
    __syncthreads();
    const int EDv = E * Dv;
    for (int i = t; i < EDv; i += kBThreads) {
        const int qq = i / Dv, c = i - qq * Dv;
        A sum = 0;
        for (int sb = 0; sb < wpb; ++sb) sum += red[(qq * wpb + sb) * Dv + c];
        store_pooled<T>(d, p, b, i, (float)sum);
    }
    stamp_end(p.stamp);
}

// Shared-memory-accumulating gather for any E and row width (A: the
// accumulator, fp64 for fp32 storage while [kWarps][E][D_v] of it fits).
template <typename T, typename A>
__global__ void __launch_bounds__(kThreads) gather_kernel(Dims d, Ptrs p) {
    extern __shared__ __align__(16) unsigned char acc_raw[];
    A *acc_w = reinterpret_cast<A *>(acc_raw);   // [kWarps][E][D_v]
    const int b = blockIdx.x;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int EDv = d.E * d.d_v;
    pdl_wait();
    stamp_begin(p.stamp);
    pdl_trigger();
    A *mine = acc_w + (size_t)warp * EDv;
    for (int i = lane; i < EDv; i += 32) mine[i] = 0;
    __syncwarp();

    constexpr int EPV = 16 / sizeof(T);   // elements per 16-byte vector
    const int VPR = d.d_v / EPV;          // vectors per row
    const int hm = d.H * d.m;
    const int64_t base = (int64_t)b * hm;
    const T *V = static_cast<const T *>(p.values);
    for (int e0 = warp * kUnroll; e0 < hm; e0 += kWarps * kUnroll) {
        int row[kUnroll], blk[kUnroll];
        float w[kUnroll];
#pragma unroll
        for (int u = 0; u < kUnroll; ++u) {
            int e = e0 + u;
            bool ok = e < hm;
            row[u] = ok ? p.sel_row[base + e] : 0;
            blk[u] = ok ? p.sel_p[base + e] : 0;
            w[u] = ok && d.nc == 1 ? p.sel_w[base + e] : 0.f;
        }
        for (int vv = lane; vv < VPR; vv += 32) {
            uint4 val[kUnroll];
#pragma unroll
            for (int u = 0; u < kUnroll; ++u)
                val[u] = (e0 + u < hm) ? ld_stream(V + (int64_t)row[u] * d.d_v + vv * EPV)
                                       : make_uint4(0, 0, 0, 0);
            if (d.nc > 1) {   // MCS: the weight of this vector's value slice
                const int ws = (vv * EPV) / (d.d_v / d.nc);
#pragma unroll
                for (int u = 0; u < kUnroll; ++u)
                    if (e0 + u < hm) w[u] = p.sel_w[(base + e0 + u) * d.nc + ws];
            }
#pragma unroll
            for (int u = 0; u < kUnroll; ++u)
                if (e0 + u < hm) fma_vec(mine + blk[u] * d.d_v + vv * EPV, val[u], w[u], T());
        }
    }
    __syncthreads();
    for (int i = threadIdx.x; i < EDv; i += kThreads) {
        A s = 0;
#pragma unroll
        for (int wv = 0; wv < kWarps; ++wv) s += acc_w[(size_t)wv * EDv + i];
        store_pooled<T>(d, p, b, i, (float)s);
    }
    stamp_end(p.stamp);
}

// proj_part[split][b][o] = sum over this split's slice of E*D_v of acc[b][c] W[c][o]
// (W = the E projectors stacked: [E*D_v][D'_v]).  Tile 32 tokens x 64 outputs.
template <typename T>
__global__ void __launch_bounds__(kThreads) proj_kernel(Dims d, Ptrs p) {
    const int Kd = d.E * d.d_v;
    const int split = blockIdx.z;
    const int chunk = (Kd + d.p_splits - 1) / d.p_splits;
    const int kb = split * chunk, ke = min(Kd, kb + chunk);
    const int o0 = blockIdx.x * 64, b0 = blockIdx.y * 32;
    const T *W = static_cast<const T *>(p.w_proj);
    stamp_begin(p.stamp);
    __shared__ float as[32][33];   // [c][token]
    __shared__ float ws[32][65];   // [c][output]
    const int tid = threadIdx.x, tx = tid % 16, ty = tid / 16;
    // fp32 storage: compensated sums (Dot2), each partial to the working precision
    constexpr bool kExact = std::is_same<T, float>::value;
    float acc[2][4] = {};
    Dot2 ex[kExact ? 2 : 1][kExact ? 4 : 1];
    for (int k0 = kb; k0 < ke; k0 += 32) {
        for (int e = tid; e < 32 * 32; e += kThreads) {
            int bb = e / 32, kk = e % 32, b = b0 + bb, c = k0 + kk;
            as[kk][bb] = (b < d.B && c < ke) ? p.acc[(int64_t)b * Kd + c] : 0.f;
        }
        for (int e = tid; e < 32 * 64; e += kThreads) {
            int kk = e / 64, oo = e % 64, c = k0 + kk, o = o0 + oo;
            ws[kk][oo] = (c < ke && o < d.d_out) ? to_f(W[(int64_t)c * d.d_out + o]) : 0.f;
        }
        __syncthreads();
#pragma unroll 8
        for (int kk = 0; kk < 32; ++kk) {
            float a0 = as[kk][ty * 2], a1 = as[kk][ty * 2 + 1];
#pragma unroll
            for (int j = 0; j < 4; ++j) {
                float wv = ws[kk][tx * 4 + j];
                if constexpr (kExact) {
                    ex[0][j].add(a0, wv);
                    ex[1][j].add(a1, wv);
                } else {
                    acc[0][j] = fmaf(a0, wv, acc[0][j]);
                    acc[1][j] = fmaf(a1, wv, acc[1][j]);
                }
            }
        }
        __syncthreads();
    }
    for (int i = 0; i < 2; ++i)
        for (int j = 0; j < 4; ++j) {
            int b = b0 + ty * 2 + i, o = o0 + tx * 4 + j;
            float v = acc[i][j];
            if constexpr (kExact) v = ex[i][j].value();
            if (b < d.B && o < d.d_out)
                p.proj_part[((int64_t)split * d.B + b) * d.d_out + o] = v;
        }
    stamp_end(p.stamp);
}

// out = the sum of the split-K partials (in fp64 with fp32 storage: one
// rounding of the output)
template <typename T>
__global__ void proj_reduce_kernel(Dims d, Ptrs p) {
    pdl_wait();
    stamp_begin(p.stamp);
    pdl_trigger();
    using A = AccOf<T>;
    const int64_t total = (int64_t)d.B * d.d_out;
    for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < total;
         i += (int64_t)gridDim.x * blockDim.x) {
        A s = 0;
        for (int sp = 0; sp < d.p_splits; ++sp) s += (A)p.proj_part[(int64_t)sp * total + i];
        static_cast<T *>(p.out)[i] = from_f<T>((float)s);
    }
    stamp_end(p.stamp);
}

}  // namespace

size_t gather_smem_bytes(const Dims &d) { return acc_bytes(d) * kWarps * d.E * d.d_v; }

template <typename K> static cudaError_t allow(K kern, size_t bytes) {
    return cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)bytes);
}
// the per-CTA maximum of dynamic shared memory next to the kernel's static share
template <auto K> static cudaError_t allow_padded() {
    return allow(K, kSmemPerCta - static_smem_of<K>());
}

// Every gather kernel may use up to the per-CTA maximum of dynamic shared
// memory: a kernel's limit is a process-wide attribute, so it is only ever
// raised (set once to the maximum), never set to one layer's need, which
// would fail a later launch for a larger layer created earlier.
cudaError_t configure_gather(const Dims &) {
    cudaError_t e = allow_padded<gather_kernel<float, double>>();
    if (e == cudaSuccess) e = allow_padded<gather_kernel<float, float>>();
    if (e == cudaSuccess) e = allow_padded<gather_kernel<__nv_bfloat16, float>>();
    if (e == cudaSuccess) e = allow_padded<gather_reg_kernel<float, 1>>();
    if (e == cudaSuccess) e = allow_padded<gather_reg_kernel<float, 4>>();
    if (e == cudaSuccess) e = allow_padded<gather_reg_kernel<__nv_bfloat16, 1>>();
    if (e == cudaSuccess) e = allow_padded<gather_reg_kernel<__nv_bfloat16, 4>>();
    // the bucketed kernels may also be padded up to a whole SM's share (spread_smem)
    if (e == cudaSuccess) e = allow_padded<gather_bucket_kernel<float, 512>>();
    if (e == cudaSuccess) e = allow_padded<gather_bucket_kernel<__nv_bfloat16, 512>>();
    if (e == cudaSuccess) e = allow_padded<gather_bucket_kernel<float, 256>>();
    if (e == cudaSuccess) e = allow_padded<gather_bucket_kernel<__nv_bfloat16, 256>>();
    return e;
}

template <typename T>
static cudaError_t launch_gather_t(const Dims &d, const Ptrs &p, cudaStream_t st) {
    const size_t bytes = gather_smem_bytes(d);
    const bool fits_lanes = d.d_v / (16 / (int)sizeof(T)) <= 32;
    if (fits_lanes && d.d_v % (16 / (int)sizeof(T)) == 0 && d.E <= kBMaxE) {
        // spread over the SMs (see spread_smem)
        if (d.B <= 2 * 152 && d.H * d.m <= 512) {
            constexpr auto k = gather_bucket_kernel<T, 512>;
            return launch_kernel(d.pdl, k, d.B, 512,
                                 spread_smem(bucket_smem_bytes(d, 16), static_smem_of<k>(), d.B),
                                 st, d, p);
        }
        if (d.H * d.m <= 256 && d.E <= 8) {
            constexpr auto k = gather_bucket_kernel<T, 256>;
            return launch_kernel(d.pdl, k, d.B, 256,
                                 spread_smem(bucket_smem_bytes(d, 8), static_smem_of<k>(), d.B),
                                 st, d, p);
        }
    }
    // the shared-memory-accumulating kernel: fp64 accumulators (fp32 storage)
    // while they fit, else fp32 ones
    auto general = [&]() {
        if (std::is_same<T, float>::value && bytes <= kSmemPerCta)
            return launch_kernel(d.pdl, gather_kernel<T, AccOf<T>>, d.B, kThreads, bytes, st, d,
                                 p);
        return launch_kernel(d.pdl, gather_kernel<T, float>, d.B, kThreads,
                             sizeof(float) * kWarps * d.E * d.d_v, st, d, p);
    };
    if (d.nc > 1)   // MCS beyond the bucketed kernel's range
        return general();
    if (fits_lanes && d.E == 1)
        return launch_kernel(d.pdl, gather_reg_kernel<T, 1>, d.B, kThreads, bytes, st, d, p);
    if (fits_lanes && d.E <= 4)
        return launch_kernel(d.pdl, gather_reg_kernel<T, 4>, d.B, kThreads, bytes, st, d, p);
    return general();
}

cudaError_t launch_gather(const Dims &d, const Ptrs &p, cudaStream_t st) {
    if (d.dtype == ULTRAMEM_BF16) return launch_gather_t<__nv_bfloat16>(d, p, st);
    return launch_gather_t<float>(d, p, st);
}

cudaError_t launch_proj(const Dims &d, const Ptrs &p, cudaStream_t st) {
    dim3 grid((d.d_out + 63) / 64, (d.B + 31) / 32, d.p_splits);
    int64_t total = (int64_t)d.B * d.d_out;
    int rblocks = (int)((total + 255) / 256);
    if (rblocks > 4096) rblocks = 4096;
    if (d.dtype == ULTRAMEM_BF16) {
        proj_kernel<__nv_bfloat16><<<grid, kThreads, 0, st>>>(d, p);
        proj_reduce_kernel<__nv_bfloat16><<<rblocks, 256, 0, st>>>(d, p);
    } else {
        proj_kernel<float><<<grid, kThreads, 0, st>>>(d, p);
        proj_reduce_kernel<float><<<rblocks, 256, 0, st>>>(d, p);
    }
    return cudaGetLastError();
}

}  // namespace um
