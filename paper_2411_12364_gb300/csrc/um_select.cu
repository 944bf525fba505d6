// um_select.cu -- S3..S7 for one (token, head) per CTA, in shared memory:
//   rank-1 scores a = u^T S_row, b = t^T S_col          (Eq. 6-7)
//   top-k of each axis by radix select                  (Eq. 8-9)
//   exact Tucker score g on the k*k survivors           (Eq. 10)
//   top-m of g, ordered by (score desc, v asc)          (Eq. 10)
//   weights (raw scores, or PKM's softmax), shuffle     (Trick 1, Eq. 3, Eq. 14)
// No K*K grid is ever formed.  Scores are compared as order-preserving 32-bit
// keys of their fp32 values; ties go to the smaller index.
#include "um_internal.cuh"

namespace um {
namespace {

constexpr int kThreads = 256;
constexpr int kWarps = kThreads / 32;

struct SelShared {
    int hist[256];
    int warp_tot[kWarps];
    int digit;
    int remaining;
    float scalar;
};

// fp32 -> uint32 whose unsigned order is the float order (-0 folded into +0).
__device__ __forceinline__ uint32_t f2ord(float f) {
    uint32_t u = __float_as_uint(f + 0.0f);
    return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}
__device__ __forceinline__ float ord2f(uint32_t o) {
    uint32_t u = (o & 0x80000000u) ? (o & 0x7fffffffu) : ~o;
    return __uint_as_float(u);
}

// Exclusive prefix sum of one int per thread over the block; also syncs.
__device__ int block_exclusive_scan(int v, SelShared &sh, int *total) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    int incl = v;
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
        int y = __shfl_up_sync(0xffffffffu, incl, off);
        if (lane >= off) incl += y;
    }
    if (lane == 31) sh.warp_tot[warp] = incl;
    __syncthreads();
    int before = 0, all = 0;
    for (int w = 0; w < kWarps; ++w) {
        int t = sh.warp_tot[w];
        if (w < warp) before += t;
        all += t;
    }
    __syncthreads();
    if (total) *total = all;
    return before + incl - v;
}

// Radix select (8-bit digits, most significant first) of the kk-th largest
// key among key[0..n).  Returns that key T; *need_eq = how many keys equal to
// T belong to the top kk (count(key > T) = kk - *need_eq).
__device__ uint32_t select_kth_largest(const uint32_t *key, int n, int kk, SelShared &sh,
                                       int *need_eq) {
    uint32_t prefix = 0, mask = 0;
    int remaining = kk;
    for (int shift = 24; shift >= 0; shift -= 8) {
        for (int i = threadIdx.x; i < 256; i += kThreads) sh.hist[i] = 0;
        __syncthreads();
        for (int i = threadIdx.x; i < n; i += kThreads) {
            uint32_t v = key[i];
            if ((v & mask) == prefix) atomicAdd(&sh.hist[(v >> shift) & 255u], 1);
        }
        __syncthreads();
        if (threadIdx.x < 32) {
            const int lane = threadIdx.x;
            int cnt[8], s = 0;
#pragma unroll
            for (int j = 0; j < 8; ++j) {
                cnt[j] = sh.hist[255 - 8 * lane - j];
                s += cnt[j];
            }
            int incl = s;
#pragma unroll
            for (int off = 1; off < 32; off <<= 1) {
                int y = __shfl_up_sync(0xffffffffu, incl, off);
                if (lane >= off) incl += y;
            }
            int before = incl - s;
            if (before < remaining && remaining <= incl) {
                int acc = before;
                for (int j = 0; j < 8; ++j) {
                    if (acc + cnt[j] >= remaining) {
                        sh.digit = 255 - 8 * lane - j;
                        sh.remaining = remaining - acc;
                        break;
                    }
                    acc += cnt[j];
                }
            }
        }
        __syncthreads();
        prefix |= (uint32_t)sh.digit << shift;
        mask |= 255u << shift;
        remaining = sh.remaining;
        __syncthreads();
    }
    *need_eq = remaining;
    return prefix;
}

// Writes to out[], in increasing position order, every i < n with key > T
// and the first need_eq positions with key == T (at most cap entries).
__device__ void ordered_select(const uint32_t *key, int n, uint32_t T, int need_eq, int *out,
                               int cap, SelShared &sh) {
    const int per = (n + kThreads - 1) / kThreads;
    const int beg = min(n, (int)threadIdx.x * per), end = min(n, beg + per);
    int eq = 0;
    for (int i = beg; i < end; ++i) eq += key[i] == T;
    const int eq_before = block_exclusive_scan(eq, sh, nullptr);
    int take = 0;
    for (int i = beg, e = eq_before; i < end; ++i) {
        uint32_t v = key[i];
        if (v > T) ++take;
        else if (v == T) take += (e++ < need_eq);
    }
    int o = block_exclusive_scan(take, sh, nullptr);
    for (int i = beg, e = eq_before; i < end; ++i) {
        uint32_t v = key[i];
        bool sel = v > T;
        if (v == T) sel = (e++ < need_eq);
        if (sel && o < cap) out[o] = i;
        o += sel;
    }
    __syncthreads();
}

// Ascending bitonic sort of P (a power of two) 64-bit words in shared memory.
__device__ void bitonic_sort(unsigned long long *a, int P) {
    for (int size = 2; size <= P; size <<= 1)
        for (int stride = size >> 1; stride > 0; stride >>= 1) {
            for (int i = threadIdx.x; i < P / 2; i += kThreads) {
                int lo = 2 * i - (i & (stride - 1));
                int hi = lo + stride;
                bool up = ((lo & size) == 0);
                unsigned long long x = a[lo], y = a[hi];
                if ((x > y) == up) { a[lo] = y; a[hi] = x; }
            }
            __syncthreads();
        }
}

__device__ __forceinline__ int pow2_at_least(int m) {
    int P = 1;
    while (P < m) P <<= 1;
    return P;
}

struct SelLayout {
    uint32_t *key;
    int *sel_i, *sel_j, *win;
    float *srow, *scol, *R;
    unsigned long long *sortbuf;
};

__device__ SelLayout carve(const Dims &d, unsigned char *base) {
    SelLayout L;
    const int nkey = max(d.K, d.k * d.k);
    size_t off = 0;
    L.key = reinterpret_cast<uint32_t *>(base + off);
    off += sizeof(uint32_t) * nkey;
    off = (off + 15) & ~size_t(15);
    L.sortbuf = reinterpret_cast<unsigned long long *>(base + off);
    off += sizeof(unsigned long long) * pow2_at_least(d.m);
    L.sel_i = reinterpret_cast<int *>(base + off);
    off += sizeof(int) * d.k;
    L.sel_j = reinterpret_cast<int *>(base + off);
    off += sizeof(int) * d.k;
    L.win = reinterpret_cast<int *>(base + off);
    off += sizeof(int) * d.m;
    L.srow = reinterpret_cast<float *>(base + off);
    off += sizeof(float) * d.k * d.r;
    L.scol = reinterpret_cast<float *>(base + off);
    off += sizeof(float) * d.k * d.r;
    L.R = reinterpret_cast<float *>(base + off);
    return L;
}

__global__ void __launch_bounds__(kThreads) select_kernel(Dims d, Ptrs p) {
    extern __shared__ __align__(16) unsigned char smem_raw[];
    __shared__ SelShared sh;
    const int b = blockIdx.x / d.H, h = blockIdx.x % d.H;
    SelLayout L = carve(d, smem_raw);
    const int r = d.r, K = d.K, k = d.k, m = d.m;
    const float *C = p.core + (int64_t)h * r * r;

    // Eq. 6-9 per axis: rank-1 score, top-k, survivors in increasing index
    for (int axis = 0; axis < 2; ++axis) {
        const float *coef = (axis == 0 ? p.u : p.t) + (int64_t)h * r;
        const float *S = p.s + (((int64_t)b * d.H + h) * 2 + axis) * (int64_t)K * r;
        for (int i = threadIdx.x; i < K; i += kThreads) {
            float a = 0.f;
            for (int al = 0; al < r; ++al) a = fmaf(coef[al], S[(int64_t)i * r + al], a);
            L.key[i] = f2ord(a);
        }
        __syncthreads();
        int need_eq;
        uint32_t T = select_kth_largest(L.key, K, k, sh, &need_eq);
        int *sel = axis == 0 ? L.sel_i : L.sel_j;
        ordered_select(L.key, K, T, need_eq, sel, k, sh);
        float *keep = axis == 0 ? L.srow : L.scol;
        for (int e = threadIdx.x; e < k * r; e += kThreads)
            keep[e] = S[(int64_t)sel[e / r] * r + (e % r)];
        __syncthreads();
    }

    // Eq. 10: g(i,j) = sum_ab S_row[a,i] C[a,b] S_col[b,j] on I x J, as
    // R[i][b] = sum_a S_row[a,i] C[a,b] then g = sum_b R[i][b] S_col[b,j].
    for (int e = threadIdx.x; e < k * r; e += kThreads) {
        int ii = e / r, be = e % r;
        float acc = 0.f;
        for (int al = 0; al < r; ++al) acc = fmaf(L.srow[ii * r + al], C[al * r + be], acc);
        L.R[e] = acc;
    }
    __syncthreads();
    const int k2 = k * k;
    for (int c = threadIdx.x; c < k2; c += kThreads) {
        int ii = c / k, jj = c - ii * k;
        float g = 0.f;
        for (int be = 0; be < r; ++be) g = fmaf(L.R[ii * r + be], L.scol[jj * r + be], g);
        L.key[c] = f2ord(g);   // candidate c = ii*k + jj: increasing c is increasing v
    }
    __syncthreads();
    int need_eq;
    uint32_t T = select_kth_largest(L.key, k2, m, sh, &need_eq);
    ordered_select(L.key, k2, T, need_eq, L.win, m, sh);

    // order the m winners by (score desc, v asc)
    const int P = pow2_at_least(m);
    for (int e = threadIdx.x; e < P; e += kThreads)
        L.sortbuf[e] = e < m ? ((unsigned long long)(~L.key[L.win[e]]) << 32) |
                                   (unsigned)L.win[e]
                             : ~0ull;
    __syncthreads();
    bitonic_sort(L.sortbuf, P);

    // PKM's softmax over the m selected scores (Eq. 3); Trick 1 skips it
    if (d.act == ULTRAMEM_ACT_SOFTMAX) {
        if (threadIdx.x < 32) {
            float gmax = ord2f(L.key[(int)(L.sortbuf[0] & 0xffffffffu)]);
            float z = 0.f;
            for (int e = threadIdx.x; e < m; e += 32)
                z += __expf(ord2f(L.key[(int)(L.sortbuf[e] & 0xffffffffu)]) - gmax);
#pragma unroll
            for (int off = 16; off > 0; off >>= 1) z += __shfl_xor_sync(0xffffffffu, z, off);
            if (threadIdx.x == 0) sh.scalar = z;
        }
        __syncthreads();
    }
    const float gmax = ord2f(L.key[(int)(L.sortbuf[0] & 0xffffffffu)]);
    const int64_t base = ((int64_t)b * d.H + h) * m;
    for (int e = threadIdx.x; e < m; e += kThreads) {
        int c = (int)(L.sortbuf[e] & 0xffffffffu);
        int ii = c / k, jj = c - ii * k;
        uint64_t v = (uint64_t)L.sel_i[ii] * (uint64_t)K + (uint64_t)L.sel_j[jj];
        float g = ord2f(L.key[c]);
        float w = d.act == ULTRAMEM_ACT_SOFTMAX ? __expf(g - gmax) / sh.scalar : g;
        uint64_t vs = shuffle_address(d, p.perm, v);   // Eq. 14
        uint64_t pb = vs / (uint64_t)d.N;
        p.sel_row[base + e] = (int32_t)(vs - pb * (uint64_t)d.N);
        p.sel_p[base + e] = (int32_t)pb;
        p.sel_w[base + e] = w;
        if (p.idx_out) p.idx_out[base + e] = (int64_t)v;
        if (p.w_out) p.w_out[base + e] = w;
    }
}

// lookup_reduce input: given virtual addresses and weights -> (row, p, w).
// An address outside [0, E*N) is recorded in the error word and skipped
// (weight 0, row 0).
__global__ void slots_kernel(Dims d, Ptrs p) {
    const int64_t total = (int64_t)d.B * d.H * d.m;
    for (int64_t e = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; e < total;
         e += (int64_t)gridDim.x * blockDim.x) {
        int64_t v = p.idx_in[e];
        float w = p.w_in[e];
        if (v < 0 || (uint64_t)v >= d.M) {
            atomicOr(p.err, kErrBadIndex);
            v = 0;
            w = 0.f;
        }
        uint64_t vs = shuffle_address(d, p.perm, (uint64_t)v);
        uint64_t pb = vs / (uint64_t)d.N;
        p.sel_row[e] = (int32_t)(vs - pb * (uint64_t)d.N);
        p.sel_p[e] = (int32_t)pb;
        p.sel_w[e] = w;
    }
}

}  // namespace

size_t select_smem_bytes(const Dims &d) {
    size_t nkey = (size_t)(d.K > d.k * d.k ? d.K : d.k * d.k);
    size_t P = 1;
    while ((int)P < d.m) P <<= 1;
    size_t off = sizeof(uint32_t) * nkey;
    off = (off + 15) & ~size_t(15);
    off += sizeof(unsigned long long) * P;
    off += sizeof(int) * (2 * d.k + d.m);
    off += sizeof(float) * 3 * d.k * d.r;
    return (off + 15) & ~size_t(15);
}

cudaError_t launch_select(const Dims &d, const Ptrs &p, cudaStream_t st) {
    select_kernel<<<d.B * d.H, kThreads, select_smem_bytes(d), st>>>(d, p);
    return cudaGetLastError();
}

cudaError_t launch_slots_from_addresses(const Dims &d, const Ptrs &p, cudaStream_t st) {
    int64_t total = (int64_t)d.B * d.H * d.m;
    int blocks = (int)((total + 255) / 256);
    if (blocks > 4096) blocks = 4096;
    if (blocks < 1) blocks = 1;
    slots_kernel<<<blocks, 256, 0, st>>>(d, p);
    return cudaGetLastError();
}

cudaError_t configure_select(const Dims &d) {
    return cudaFuncSetAttribute(select_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                (int)select_smem_bytes(d));
}

}  // namespace um
