// um_exact.cu -- Eq. 5 (or Eq. 2 with product keys) by brute force: the
// exact top-m of the whole K x K grid of each (token, head).  It is not on
// the forward path; it measures the recall of the approximate search of
// Eq. 6-10 (which the forward runs) against the exact one.
//
// One CTA of 512 threads per (token, head):
//   1. the head's chunk scores (Eq. 4) of all K row and K column keys, from
//      its query and the key rows (a warp per key, coalesced), kept in
//      shared memory as R[i] = S_row[:,i]^T C and S_col[:,j] (product keys:
//      s_row[i] and s_col[j]), so that g(i,j) = R[i] . S_col[j] (or the sum)
//      with the forward's own arithmetic;
//   2. an exact radix select of the m-th largest order-preserving key over
//      the K^2 scores, recomputed on the fly (4 passes of 8 bits, histograms
//      built with one shared atomic per distinct bin and warp); when several
//      slots share that key, 4 more passes select the largest address among
//      the tied ones that is still taken (ties go to the smaller address);
//   3. one pass collects the m winners, which are then ordered by (score
//      desc, address asc).
// Shared memory is 8 (K r + D_k) bytes plus 9 KB (K r <= 25600 fits).
#include "um_internal.cuh"

namespace um {
namespace {

constexpr int kThreads = 512;
constexpr int kWarps = kThreads / 32;
constexpr int kMaxM = 1024;
constexpr int kMaxR = 8;
constexpr unsigned kFull = 0xffffffffu;

typedef unsigned long long u64;

struct ExactShared {
    u64 win[kMaxM];       // the m winners as (key, ~v) composites
    int hist[256];
    int count;            // winners collected so far
    uint32_t prefix;      // key bits fixed so far
    int need;             // how many of the remaining keys are still to take
    int ties;             // slots whose key equals the threshold
    uint32_t vcut;        // largest tied address taken
    float core[kMaxR * kMaxR];
};

template <typename T>
__device__ __forceinline__ float elem(const T *p, int i) { return to_f(p[i]); }

// The grid score of slot (i, j) from the chunk scores in shared memory.
struct Grid {
    const float *R, *S;   // [K][r] each
    int K, r, pkm;
    __device__ __forceinline__ float score(int i, int j) const {
        if (pkm) return R[i] + S[j];
        const float *a = R + i * r, *b = S + j * r;
        if (r == 2) return fmaf(a[1], b[1], a[0] * b[0]);
        float g = 0.f;
        for (int be = 0; be < r; ++be) g = fmaf(a[be], b[be], g);
        return g;
    }
};

// Adds one count for `bin` (0..255; 256 = none) with one atomic per distinct
// bin of the warp.
__device__ __forceinline__ void warp_hist(int *hist, int bin) {
    const unsigned peers = __match_any_sync(kFull, bin);
    const int lane = threadIdx.x & 31;
    if (bin < 256 && lane == __ffs(peers) - 1) atomicAdd(&hist[bin], __popc(peers));
}

// The bin, counted from the top, that holds the need-th largest entry;
// updates need to the rank within that bin.  One warp; returns the bin.
__device__ int pick_bin_from_top(const int *hist, int &need) {
    const int lane = threadIdx.x & 31;
    // lane l owns bins 255 - 8 l .. 248 - 8 l (descending)
    int c[8], s = 0;
#pragma unroll
    for (int q = 0; q < 8; ++q) {
        c[q] = hist[255 - 8 * lane - q];
        s += c[q];
    }
    int incl = s;
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
        const int y = __shfl_up_sync(kFull, incl, off);
        if (lane >= off) incl += y;
    }
    const int excl = incl - s;
    const unsigned hit = __ballot_sync(kFull, excl < need && incl >= need);
    const int owner = __ffs(hit) - 1;
    int bin = 0, above = 0;
    if (lane == owner) {
        int run = excl;
#pragma unroll
        for (int q = 0; q < 8; ++q) {
            if (run + c[q] >= need) {
                bin = 255 - 8 * lane - q;
                above = run;
                break;
            }
            run += c[q];
        }
    }
    bin = __shfl_sync(kFull, bin, owner);
    above = __shfl_sync(kFull, above, owner);
    need -= above;
    return bin;
}

// The same from the bottom (the need-th smallest).
__device__ int pick_bin_from_bottom(const int *hist, int &need) {
    const int lane = threadIdx.x & 31;
    int c[8], s = 0;
#pragma unroll
    for (int q = 0; q < 8; ++q) {
        c[q] = hist[8 * lane + q];
        s += c[q];
    }
    int incl = s;
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
        const int y = __shfl_up_sync(kFull, incl, off);
        if (lane >= off) incl += y;
    }
    const int excl = incl - s;
    const unsigned hit = __ballot_sync(kFull, excl < need && incl >= need);
    const int owner = __ffs(hit) - 1;
    int bin = 0, below = 0;
    if (lane == owner) {
        int run = excl;
#pragma unroll
        for (int q = 0; q < 8; ++q) {
            if (run + c[q] >= need) {
                bin = 8 * lane + q;
                below = run;
                break;
            }
            run += c[q];
        }
    }
    bin = __shfl_sync(kFull, bin, owner);
    below = __shfl_sync(kFull, below, owner);
    need -= below;
    return bin;
}

template <typename T>
__global__ void __launch_bounds__(kThreads, 1) exact_kernel(Dims d, Ptrs p, int64_t *idx_out,
                                                            float *w_out) {
    extern __shared__ __align__(16) float rs[];   // R [K][r], S_col [K][r], q [2][D_k]
    __shared__ ExactShared sh;
    const int b = blockIdx.x / d.H, h = blockIdx.x % d.H;
    const int K = d.K, r = d.r, D = d.d_k, dk = d.dk, m = d.m;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    float *R = rs, *S = rs + (size_t)K * r, *qv = S + (size_t)K * r;
    pdl_wait();
    pdl_trigger();

    const int HD = d.H * D;
    const int64_t split_stride = (int64_t)d.A * d.B * HD;
    for (int e = threadIdx.x; e < 2 * D; e += kThreads) {   // summed over the D_i splits
        const int axis = e / D, c = e - axis * D;
        const int a = (axis == 1 && d.A == 2) ? 1 : 0;
        const float *src = p.q_part + ((int64_t)a * d.B + b) * HD + h * D + c;
        float q = 0.f;
        for (int sp = 0; sp < d.q_splits; ++sp) q += src[sp * split_stride];
        qv[e] = q;
    }
    if (threadIdx.x < r * r) sh.core[threadIdx.x] = p.core[(int64_t)h * r * r + threadIdx.x];
    if (threadIdx.x == 0) {
        sh.count = 0;
        sh.prefix = 0;
        sh.need = m;
    }
    __syncthreads();

    // 1. chunk scores of every key (Eq. 4), a warp per key
    for (int key = warp; key < 2 * K; key += kWarps) {
        const int axis = key >= K, i = key - axis * K;
        const T *row = static_cast<const T *>(axis ? p.k_col : p.k_row) + ((int64_t)h * K + i) * D;
        const float *q = qv + axis * D;
        float s[kMaxR];
#pragma unroll
        for (int a = 0; a < kMaxR; ++a) s[a] = 0.f;
        for (int c = lane; c < D; c += 32) {
            const float pr = elem(row, c) * q[c];
            const int al = c / dk;
#pragma unroll
            for (int a = 0; a < kMaxR; ++a) s[a] += a == al ? pr : 0.f;
        }
#pragma unroll
        for (int a = 0; a < kMaxR; ++a) {
            if (a < r)
#pragma unroll
                for (int off = 16; off > 0; off >>= 1) s[a] += __shfl_xor_sync(kFull, s[a], off);
        }
        if (lane == 0) {
            if (axis == 0) {   // R = S_row^T C
                for (int be = 0; be < r; ++be) {
                    float acc = 0.f;
                    for (int a = 0; a < r; ++a) acc = fmaf(s[a], sh.core[a * r + be], acc);
                    R[i * r + be] = acc;
                }
            } else {
                for (int be = 0; be < r; ++be) S[i * r + be] = s[be];
            }
        }
    }
    __syncthreads();

    const Grid gd{R, S, K, r, d.pkm};
    const int64_t total = (int64_t)K * K;
    const int64_t iters = (total + kThreads - 1) / kThreads;
    // slot c = it * kThreads + tid, as (i, j) stepped without division
    const int di = kThreads / K, dj = kThreads % K;

    // 2. the m-th largest key, 8 bits a pass
    for (int shift = 24; shift >= 0; shift -= 8) {
        for (int e = threadIdx.x; e < 256; e += kThreads) sh.hist[e] = 0;
        __syncthreads();
        const uint32_t pre = sh.prefix;
        const uint32_t hi_mask = shift == 24 ? 0u : ~0u << (shift + 8);
        int i = threadIdx.x / K, j = threadIdx.x % K;
        for (int64_t it = 0; it < iters; ++it) {
            int bin = 256;
            if (i < K) {
                const uint32_t key = f2ord(gd.score(i, j));
                if ((key & hi_mask) == (pre & hi_mask)) bin = (key >> shift) & 255;
            }
            warp_hist(sh.hist, bin);
            i += di;
            j += dj;
            if (j >= K) { j -= K; ++i; }
        }
        __syncthreads();
        if (warp == 0) {
            int need = sh.need;
            const int bin = pick_bin_from_top(sh.hist, need);
            if (lane == 0) {
                sh.prefix = pre | ((uint32_t)bin << shift);
                sh.need = need;
                sh.ties = sh.hist[bin];
            }
        }
        __syncthreads();
    }
    const uint32_t thr = sh.prefix;   // the m-th largest key
    // ties at the threshold: the need-th smallest address among them
    uint32_t vcut = ~0u;
    if (sh.ties > sh.need) {
        if (threadIdx.x == 0) sh.vcut = 0;
        for (int shift = 24; shift >= 0; shift -= 8) {
            for (int e = threadIdx.x; e < 256; e += kThreads) sh.hist[e] = 0;
            __syncthreads();
            const uint32_t pre = sh.vcut;
            const uint32_t hi_mask = shift == 24 ? 0u : ~0u << (shift + 8);
            int i = threadIdx.x / K, j = threadIdx.x % K;
            for (int64_t it = 0; it < iters; ++it) {
                int bin = 256;
                if (i < K && f2ord(gd.score(i, j)) == thr) {
                    const uint32_t v = (uint32_t)i * (uint32_t)K + (uint32_t)j;
                    if ((v & hi_mask) == (pre & hi_mask)) bin = (v >> shift) & 255;
                }
                warp_hist(sh.hist, bin);
                i += di;
                j += dj;
                if (j >= K) { j -= K; ++i; }
            }
            __syncthreads();
            if (warp == 0) {
                int need = sh.need;
                const int bin = pick_bin_from_bottom(sh.hist, need);
                if (lane == 0) {
                    sh.vcut = pre | ((uint32_t)bin << shift);
                    sh.need = need;
                }
            }
            __syncthreads();
        }
        vcut = sh.vcut;
    }

    // 3. the winners: keys above the threshold, and the tied ones up to vcut
    {
        int i = threadIdx.x / K, j = threadIdx.x % K;
        for (int64_t it = 0; it < iters; ++it) {
            bool take = false;
            uint32_t key = 0, v = 0;
            if (i < K) {
                key = f2ord(gd.score(i, j));
                v = (uint32_t)i * (uint32_t)K + (uint32_t)j;
                take = key > thr || (key == thr && v <= vcut);
            }
            const unsigned bal = __ballot_sync(kFull, take);
            if (bal) {
                int base = 0;
                if (lane == 0) base = atomicAdd(&sh.count, __popc(bal));
                base = __shfl_sync(kFull, base, 0);
                const int pos = base + __popc(bal & ((1u << lane) - 1u));
                if (take && pos < kMaxM) sh.win[pos] = ((u64)key << 32) | (u64)(~v);
            }
            i += di;
            j += dj;
            if (j >= K) { j -= K; ++i; }
        }
    }
    __syncthreads();
    const int n = min(sh.count, m);
    if (sh.count != m && threadIdx.x == 0) atomicOr(p.err, kErrInternal);   // never expected

    // 4. ranks by (key desc, v asc): the number of composites above each
    const int64_t base = ((int64_t)b * d.H + h) * m;
    for (int e = threadIdx.x; e < n; e += kThreads) {
        const u64 x = sh.win[e];
        int rank = 0;
        for (int f = 0; f < n; ++f) rank += sh.win[f] > x;
        const uint32_t v = ~(uint32_t)x;
        idx_out[base + rank] = (int64_t)v;
        if (w_out) w_out[base + rank] = ord2f((uint32_t)(x >> 32));
    }
}

}  // namespace

size_t exact_smem_bytes(const Dims &d) {
    return sizeof(float) * 2 * ((size_t)d.K * d.r + (size_t)d.d_k);
}

bool exact_fits(const Dims &d) {
    return d.m <= kMaxM && d.r <= kMaxR &&
           exact_smem_bytes(d) + sizeof(ExactShared) <= kSmemPerCta;
}

cudaError_t configure_exact(const Dims &d) {
    const cudaFuncAttribute a = cudaFuncAttributeMaxDynamicSharedMemorySize;
    const int bytes = (int)exact_smem_bytes(d);
    cudaError_t e = cudaFuncSetAttribute(exact_kernel<float>, a, bytes);
    if (e == cudaSuccess) e = cudaFuncSetAttribute(exact_kernel<__nv_bfloat16>, a, bytes);
    return e;
}

cudaError_t launch_exact(const Dims &d, const Ptrs &p, int64_t *idx_out, float *w_out,
                         cudaStream_t st) {
    const size_t smem = exact_smem_bytes(d);
    if (d.dtype == ULTRAMEM_BF16)
        return launch_kernel(d.pdl, exact_kernel<__nv_bfloat16>, d.B * d.H, kThreads, smem, st,
                             d, p, idx_out, w_out);
    return launch_kernel(d.pdl, exact_kernel<float>, d.B * d.H, kThreads, smem, st, d, p,
                         idx_out, w_out);
}

}  // namespace um
