// um_select.cu -- S3..S7 for one (token, head) per CTA, in shared memory:
//   rank-1 scores a = u^T S_row, b = t^T S_col          (Eq. 6-7)
//   top-k of each axis                                  (Eq. 8-9)
//   exact Tucker score g on the k*k survivors           (Eq. 10)
//   top-m of g, ordered by (score desc, v asc)          (Eq. 10)
//   weights (raw scores, or PKM's softmax), shuffle     (Trick 1, Eq. 3, Eq. 14)
// No K*K grid is ever formed.  Scores are compared as order-preserving 32-bit
// keys of their fp32 values; ties go to the smaller index.
//
// Top-k of n keys (topk_positions): each thread takes the maximum of its
// strided share of the keys; tau = the kk-th largest of those 256 maxima is
// a lower bound of the kk-th largest key for any input (kk threads each own
// a key >= tau).  Keys > tau are gathered, plus -- only when fewer than kk
// keys exceed tau -- the first ties at tau in position order; these
// candidates (typically one to three times kk) are ranked exactly.  If more
// than kCap keys exceed tau, a radix select over all n keys is used instead.
#include "um_internal.cuh"

namespace um {
namespace {

constexpr int kThreads = 256;
constexpr int kWarps = kThreads / 32;
constexpr int kCap = 2048;       // candidate capacity of the threshold path
constexpr int kMaxOut = 1024;    // largest k or m

struct SelShared {
    int hist[256];
    int warp_tot[kWarps];
    int digit;
    int remaining;
    float scalar;
    uint32_t vt[kThreads];
    uint32_t cand_key[kCap];
    int cand_pos[kCap];
    uint32_t win_key[kMaxOut];
    int win_pos[kMaxOut];
    int n_gt;
    uint32_t tau;
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
__device__ int block_exclusive_scan(int v, SelShared &sh) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    int incl = v;
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
        int y = __shfl_up_sync(0xffffffffu, incl, off);
        if (lane >= off) incl += y;
    }
    if (lane == 31) sh.warp_tot[warp] = incl;
    __syncthreads();
    int before = 0;
    for (int w = 0; w < warp; ++w) before += sh.warp_tot[w];
    __syncthreads();
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

// Appends to sh.cand_*[base..] the first `need` positions (in position
// order) with key == T, using contiguous per-thread ranges.
__device__ void gather_ties_in_order(const uint32_t *key, int n, uint32_t T, int need, int base,
                                     SelShared &sh) {
    const int per = (n + kThreads - 1) / kThreads;
    const int beg = min(n, (int)threadIdx.x * per), end = min(n, beg + per);
    int eq = 0;
    for (int i = beg; i < end; ++i) eq += key[i] == T;
    int e = block_exclusive_scan(eq, sh);
    for (int i = beg; i < end && e < need; ++i)
        if (key[i] == T) {
            sh.cand_key[base + e] = T;
            sh.cand_pos[base + e] = i;
            ++e;
        }
    __syncthreads();
}

enum { kOrderByPosition = 0, kOrderByScore = 1 };

// Positions of the kk largest keys of key[0..n) (ties: smaller position
// first).  Leaves them in sh.win_pos / sh.win_key ordered by (key desc,
// position asc); with kOrderByPosition, also writes the positions in
// increasing order to out[0..kk).
__device__ void topk_positions(const uint32_t *key, int n, int kk, int *out, int order,
                               SelShared &sh) {
    // tau = kk-th largest per-thread maximum (0 when fewer than kk threads own
    // a key, which makes every key a candidate)
    uint32_t vmax = 0;
    for (int i = threadIdx.x; i < n; i += kThreads) vmax = max(vmax, key[i]);
    sh.vt[threadIdx.x] = vmax;
    if (threadIdx.x == 0) { sh.n_gt = 0; sh.tau = 0; }
    __syncthreads();
    {
        int rank = 0;
        for (int t = 0; t < kThreads; ++t) {
            uint32_t o = sh.vt[t];
            rank += (o > vmax) || (o == vmax && t < (int)threadIdx.x);
        }
        if (rank == kk - 1) sh.tau = vmax;
    }
    __syncthreads();
    const uint32_t tau = sh.tau;
    for (int i = threadIdx.x; i < n; i += kThreads) {
        uint32_t v = key[i];
        if (v > tau) {
            int slot = atomicAdd(&sh.n_gt, 1);
            if (slot < kCap) { sh.cand_key[slot] = v; sh.cand_pos[slot] = i; }
        }
    }
    __syncthreads();
    int c = sh.n_gt;
    if (c > kCap) {
        int need_eq;
        uint32_t T = select_kth_largest(key, n, kk, sh, &need_eq);
        // every key > T, then the first need_eq ties at T
        if (threadIdx.x == 0) sh.n_gt = 0;
        __syncthreads();
        for (int i = threadIdx.x; i < n; i += kThreads) {
            uint32_t v = key[i];
            if (v > T) {
                int slot = atomicAdd(&sh.n_gt, 1);
                sh.cand_key[slot] = v;   // fewer than kk <= kCap of them
                sh.cand_pos[slot] = i;
            }
        }
        __syncthreads();
        gather_ties_in_order(key, n, T, need_eq, kk - need_eq, sh);
        c = kk;
    } else if (c < kk) {
        gather_ties_in_order(key, n, tau, kk - c, c, sh);
        c = kk;
    }
    // exact rank of every candidate by (key desc, position asc)
    for (int e = threadIdx.x; e < c; e += kThreads) {
        const uint32_t ke = sh.cand_key[e];
        const int pe = sh.cand_pos[e];
        int rank = 0;
        for (int f = 0; f < c; ++f) {
            uint32_t kf = sh.cand_key[f];
            rank += (kf > ke) || (kf == ke && sh.cand_pos[f] < pe);
        }
        if (rank < kk) {
            sh.win_key[rank] = ke;
            sh.win_pos[rank] = pe;
        }
    }
    __syncthreads();
    if (order == kOrderByPosition) {
        for (int e = threadIdx.x; e < kk; e += kThreads) {
            const int pe = sh.win_pos[e];
            int r = 0;
            for (int f = 0; f < kk; ++f) r += sh.win_pos[f] < pe;
            out[r] = pe;
        }
        __syncthreads();
    }
}

struct SelLayout {
    uint32_t *key;
    int *sel_i, *sel_j;
    float *srow, *scol, *R;
};

__device__ SelLayout carve(const Dims &d, unsigned char *base) {
    SelLayout L;
    const int nkey = max(d.K, d.k * d.k);
    size_t off = 0;
    L.key = reinterpret_cast<uint32_t *>(base + off);
    off += sizeof(uint32_t) * nkey;
    L.sel_i = reinterpret_cast<int *>(base + off);
    off += sizeof(int) * d.k;
    L.sel_j = reinterpret_cast<int *>(base + off);
    off += sizeof(int) * d.k;
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

    // Eq. 6-9 per axis: rank-1 score, top-k; survivors in increasing index
    for (int axis = 0; axis < 2; ++axis) {
        const float *coef = (axis == 0 ? p.u : p.t) + (int64_t)h * r;
        const float *S = p.s + (((int64_t)b * d.H + h) * 2 + axis) * (int64_t)K * r;
        for (int i = threadIdx.x; i < K; i += kThreads) {
            float a = 0.f;
            for (int al = 0; al < r; ++al) a = fmaf(coef[al], S[(int64_t)i * r + al], a);
            L.key[i] = f2ord(a);
        }
        __syncthreads();
        int *sel = axis == 0 ? L.sel_i : L.sel_j;
        topk_positions(L.key, K, k, sel, kOrderByPosition, sh);
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
        L.key[c] = f2ord(g);   // I and J ascending: increasing c is increasing v
    }
    __syncthreads();
    topk_positions(L.key, k2, m, nullptr, kOrderByScore, sh);

    // PKM's softmax over the m selected scores (Eq. 3); Trick 1 skips it
    const float gmax = ord2f(sh.win_key[0]);
    if (d.act == ULTRAMEM_ACT_SOFTMAX) {
        if (threadIdx.x < 32) {
            float z = 0.f;
            for (int e = threadIdx.x; e < m; e += 32) z += __expf(ord2f(sh.win_key[e]) - gmax);
#pragma unroll
            for (int off = 16; off > 0; off >>= 1) z += __shfl_xor_sync(0xffffffffu, z, off);
            if (threadIdx.x == 0) sh.scalar = z;
        }
        __syncthreads();
    }
    const int64_t base = ((int64_t)b * d.H + h) * m;
    for (int e = threadIdx.x; e < m; e += kThreads) {
        int c = sh.win_pos[e];
        int ii = c / k, jj = c - ii * k;
        uint64_t v = (uint64_t)L.sel_i[ii] * (uint64_t)K + (uint64_t)L.sel_j[jj];
        float g = ord2f(sh.win_key[e]);
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
    size_t off = sizeof(uint32_t) * nkey + sizeof(int) * 2 * d.k + sizeof(float) * 3 * d.k * d.r;
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
