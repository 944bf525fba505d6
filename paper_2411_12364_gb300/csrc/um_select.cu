// um_select.cu -- S4..S7 for one (token, head) per CTA:
//   top-k of each axis on the rank-1 score keys         (Eq. 8-9)
//   exact chunk scores S_alpha of the 2k survivors      (Eq. 4)
//   exact Tucker score g on the k*k survivor pairs      (Eq. 10)
//   top-m of g, ordered by (score desc, v asc)          (Eq. 10)
//   weights (raw scores, or PKM's softmax), shuffle     (Trick 1, Eq. 3, Eq. 14)
// No K*K grid is ever formed.  The scoring kernel leaves, per key, the
// order-preserving 32-bit key of its fp32 rank-1 score; the exact chunk
// scores of the k survivors of each axis are recomputed here from q and the
// key rows.  Ties go to the smaller index.
//
// Top-k of n keys, in two stages.  Candidates (whole block): each thread
// takes the maximum of its strided share of the keys; each warp takes the
// j-th largest of its 32 lane maxima (j = ceil(k / 8), a register bitonic
// sort) and tau is the smallest of the 8 warp values.  Every warp owns at
// least j keys >= tau, so at least k keys are >= tau whatever the input:
// every key of the top k is >= tau.  Each warp appends its keys >= tau to its
// own region (ballot, no atomics); when more than 2k survive, the same bound
// is taken again over the survivors.  Order (one warp): the candidates, as
// 64-bit composites (key, ~position) whose descending order is key
// descending then position ascending, are sorted in registers by a bitonic
// network (shuffles across lanes, swaps across registers).  Rare inputs with
// too many candidates (heavy ties) take an exact radix select instead.
#include "um_internal.cuh"

namespace um {
namespace {

constexpr int kThreads = 256;
constexpr int kWarps = kThreads / 32;
constexpr int kRegion = 128;               // candidates per warp region
constexpr int kCap = kWarps * kRegion;     // 1024 per selection
constexpr int kMaxK = 128;
constexpr int kMaxM = 1024;
constexpr unsigned kFull = 0xffffffffu;

typedef unsigned long long u64;

struct SelShared {
    u64 cand[2][kCap];      // per selection: kWarps regions of kRegion (or one flat list)
    u64 fwin[kMaxM];        // final winners by rank
    int wcnt[2][kWarps];    // region fill counts
    uint32_t vt[2][kWarps];
    int hist[256];
    int warp_tot[kWarps];
    int digit, remaining;
    float scalar;
};

__device__ __forceinline__ u64 comp_of(uint32_t key, uint32_t pos) {
    return ((u64)key << 32) | (u64)(~pos);
}
__device__ __forceinline__ uint32_t key_of(u64 c) { return (uint32_t)(c >> 32); }
__device__ __forceinline__ uint32_t pos_of(u64 c) { return ~(uint32_t)c; }

template <typename T>
__device__ __forceinline__ void unpack16(uint4 v, float (&f)[16 / sizeof(T)]);
template <>
__device__ __forceinline__ void unpack16<__nv_bfloat16>(uint4 v, float (&f)[8]) {
    const uint32_t u[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
    for (int q = 0; q < 4; ++q) {
        f[2 * q] = __uint_as_float(u[q] << 16);
        f[2 * q + 1] = __uint_as_float(u[q] & 0xffff0000u);
    }
}
template <>
__device__ __forceinline__ void unpack16<float>(uint4 v, float (&f)[4]) {
    f[0] = __uint_as_float(v.x);
    f[1] = __uint_as_float(v.y);
    f[2] = __uint_as_float(v.z);
    f[3] = __uint_as_float(v.w);
}

// j-th largest (1-based, j <= 32) of one value per lane: descending bitonic
// sort across the warp.
__device__ __forceinline__ uint32_t warp_jth_largest(uint32_t v, int j) {
    const int lane = threadIdx.x & 31;
#pragma unroll
    for (int blk = 2; blk <= 32; blk <<= 1)
#pragma unroll
        for (int st = blk >> 1; st > 0; st >>= 1) {
            const uint32_t o = __shfl_xor_sync(kFull, v, st);
            const bool keep_max = ((lane & st) == 0) == ((lane & blk) == 0);
            v = keep_max ? max(v, o) : min(v, o);
        }
    return __shfl_sync(kFull, v, j - 1);
}

// Exclusive prefix sum of one int per thread over the block; also syncs.
__device__ int block_exclusive_scan(int v, SelShared &sh) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    int incl = v;
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
        int y = __shfl_up_sync(kFull, incl, off);
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
                int y = __shfl_up_sync(kFull, incl, off);
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

// Exact fallback for selection s: a flat list of exactly kk candidates (every
// key > T, then the first ties at T in position order) in cand[s], counted
// in region 0.  Kept out of line: it only runs when a region overflows.
__device__ __noinline__ void radix_fallback(const uint32_t *key, int n, int kk, int s,
                                            SelShared &sh) {
    int need_eq;
    const uint32_t T = select_kth_largest(key, n, kk, sh, &need_eq);
    const int n_gt = kk - need_eq;
    const int per = (n + kThreads - 1) / kThreads;
    const int beg = min(n, (int)threadIdx.x * per), end = min(n, beg + per);
    int gt = 0, eq = 0;
    for (int i = beg; i < end; ++i) {
        gt += key[i] > T;
        eq += key[i] == T;
    }
    int o = block_exclusive_scan(gt, sh);
    int e = block_exclusive_scan(eq, sh);
    for (int i = beg; i < end; ++i) {
        const uint32_t v = key[i];
        if (v > T) sh.cand[s][o++] = comp_of(v, (uint32_t)i);
        else if (v == T && e < need_eq) sh.cand[s][n_gt + e++] = comp_of(v, (uint32_t)i);
        else if (v == T) ++e;
    }
    if (threadIdx.x < kWarps) sh.wcnt[s][threadIdx.x] = threadIdx.x == 0 ? kk : 0;
    __syncthreads();
}

// Tightens selection s: the same bound over the survivors of each region.
__device__ void tighten(int s, int kk, SelShared &sh) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    constexpr int kPer = kRegion / 32;
    const int mycnt = sh.wcnt[s][warp];
    u64 mine[kPer];
    uint32_t vm = 0;
#pragma unroll
    for (int q = 0; q < kPer; ++q) {
        const int f = lane + 32 * q;
        mine[q] = f < mycnt ? sh.cand[s][warp * kRegion + f] : 0ull;
        vm = max(vm, key_of(mine[q]));
    }
    const int j = (kk + kWarps - 1) / kWarps;
    const uint32_t tw = j <= 32 ? warp_jth_largest(vm, j) : 0u;
    if (lane == 0) sh.vt[s][warp] = tw;
    __syncthreads();
    uint32_t tau = sh.vt[s][0];
    for (int w = 1; w < kWarps; ++w) tau = min(tau, sh.vt[s][w]);
    u64 *region = sh.cand[s] + warp * kRegion;
    int cnt = 0;
#pragma unroll
    for (int q = 0; q < kPer; ++q) {
        const bool pr = lane + 32 * q < mycnt && key_of(mine[q]) >= tau;
        const unsigned bal = __ballot_sync(kFull, pr);
        if (pr) region[cnt + __popc(bal & ((1u << lane) - 1u))] = mine[q];
        cnt += __popc(bal);
    }
    __syncthreads();   // everyone has read wcnt before it changes
    if (lane == 0) sh.wcnt[s][warp] = cnt;
    __syncthreads();
}

// Candidates of ns (1 or 2) selections of n keys each, key[s][0..n), for
// their top kk: thresholds, per-warp compaction, tightening or the radix
// fallback.  Leaves them in sh.cand[s] (kWarps regions counted by
// sh.wcnt[s][w], or a flat list in region 0 when sh.wcnt[s][0] > kRegion).
// vmax[s] is this thread's maximum over its strided share of key[s].  Every
// thread of the block calls it; it ends with a barrier.
__device__ void select_candidates(const uint32_t *key0, const uint32_t *key1, int ns, int n,
                                  int kk, uint32_t vmax0, uint32_t vmax1, SelShared &sh) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int j = (kk + kWarps - 1) / kWarps;
#pragma unroll 1
    for (int s = 0; s < ns; ++s) {
        const uint32_t tw = j <= 32 ? warp_jth_largest(s ? vmax1 : vmax0, j) : 0u;
        if (lane == 0) sh.vt[s][warp] = tw;
    }
    __syncthreads();
    // each warp appends its keys >= tau to its own region
#pragma unroll 1
    for (int s = 0; s < ns; ++s) {
        const uint32_t *key = s ? key1 : key0;
        uint32_t tau = sh.vt[s][0];
        for (int w = 1; w < kWarps; ++w) tau = min(tau, sh.vt[s][w]);
        u64 *region = sh.cand[s] + warp * kRegion;
        int cnt = 0;
        for (int b0 = warp * 32; b0 < n; b0 += kThreads) {
            const int i = b0 + lane;
            const uint32_t v = i < n ? key[i] : 0u;
            const bool pr = i < n && v >= tau;
            const unsigned bal = __ballot_sync(kFull, pr);
            const int slot = cnt + __popc(bal & ((1u << lane) - 1u));
            if (pr && slot < kRegion) region[slot] = comp_of(v, (uint32_t)i);
            cnt += __popc(bal);
        }
        if (lane == 0) sh.wcnt[s][warp] = cnt;
    }
    __syncthreads();
#pragma unroll 1
    for (int s = 0; s < ns; ++s) {
        int total = 0;
        bool over = false;
        for (int w = 0; w < kWarps; ++w) {
            total += sh.wcnt[s][w];
            over |= sh.wcnt[s][w] > kRegion;
        }
        __syncthreads();
        if (!over && total > 2 * kk) {
            tighten(s, kk, sh);
            total = 0;
            for (int w = 0; w < kWarps; ++w) total += sh.wcnt[s][w];
            __syncthreads();
            over = total > 8 * 32 && kk <= 8 * 32;   // too many to sort in registers
        }
        if (over) radix_fallback(s ? key1 : key0, n, kk, s, sh);   // rare, exact
    }
}

__device__ __forceinline__ int candidate_count(int s, const SelShared &sh) {
    if (sh.wcnt[s][0] > kRegion) return sh.wcnt[s][0];   // flat list
    int total = 0;
    for (int w = 0; w < kWarps; ++w) total += sh.wcnt[s][w];
    return total;
}

// Descending bitonic sort of 32*R values held as v[q] on lane l = element
// q*32 + l: shuffles for strides below 32, register swaps above.
template <int R>
__device__ __forceinline__ void warp_sort_desc(u64 (&v)[R]) {
    const int lane = threadIdx.x & 31;
#pragma unroll 1
    for (int size = 2; size <= 32 * R; size <<= 1) {
#pragma unroll 1
        for (int j = size >> 1; j > 0; j >>= 1) {
            if (j < 32) {
#pragma unroll
                for (int q = 0; q < R; ++q) {
                    const u64 o = __shfl_xor_sync(kFull, v[q], j);
                    const int e = q * 32 + lane;
                    const bool keep_max = ((e & j) == 0) == ((e & size) == 0);
                    v[q] = keep_max ? (v[q] > o ? v[q] : o) : (v[q] < o ? v[q] : o);
                }
            } else {
                const int jq = j >> 5;
#pragma unroll
                for (int m = 1; m < R; m <<= 1) {
                    if (jq != m) continue;
#pragma unroll
                    for (int q = 0; q < R; ++q) {
                        if (q & m) continue;
                        const bool desc = ((q * 32 + lane) & size) == 0;
                        const u64 a = v[q], b = v[q | m];
                        const bool sw = desc ? (a < b) : (a > b);
                        v[q] = sw ? b : a;
                        v[q | m] = sw ? a : b;
                    }
                }
            }
        }
    }
}

// One warp: the candidates of selection s (at most 32*R) sorted descending
// into v; element e = q*32 + lane, zero-padded.
template <int R>
__device__ __forceinline__ void warp_gather_sorted(int s, const SelShared &sh, u64 (&v)[R]) {
    const int lane = threadIdx.x & 31;
    const bool flat = sh.wcnt[s][0] > kRegion;
    int pref[kWarps + 1];
    pref[0] = 0;
#pragma unroll
    for (int w = 0; w < kWarps; ++w)
        pref[w + 1] = pref[w] + (flat ? (w == 0 ? sh.wcnt[s][0] : 0) : sh.wcnt[s][w]);
#pragma unroll
    for (int q = 0; q < R; ++q) {
        const int f = q * 32 + lane;
        u64 val = 0ull;
        if (f < pref[kWarps]) {
            int w = 0, before = 0;
#pragma unroll
            for (int x = 1; x < kWarps; ++x)
                if (f >= pref[x]) { w = x; before = pref[x]; }
            val = sh.cand[s][(flat ? 0 : w * kRegion) + f - before];
        }
        v[q] = val;
    }
    warp_sort_desc<R>(v);
}

// Block-level exact ranks of selection s's candidates (any count up to
// kCap) into win[rank] for rank < kk; each warp ranks its own region's
// entries against all entries (a flat list is split w, w+8, ... over warps).
__device__ void block_rank(int s, int kk, u64 *win, SelShared &sh) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const bool flat = sh.wcnt[s][0] > kRegion;
    const int mine_n = flat ? (sh.wcnt[s][0] + kWarps - 1 - warp) / kWarps : sh.wcnt[s][warp];
    for (int q = lane; q < mine_n; q += 32) {
        const u64 ce = sh.cand[s][flat ? warp + q * kWarps : warp * kRegion + q];
        int before = 0;
#pragma unroll 1
        for (int w = 0; w < (flat ? 1 : kWarps); ++w) {
            const u64 *reg = sh.cand[s] + w * kRegion;
            const int cw = sh.wcnt[s][w];
            int f = 0;
            for (; f + 4 <= cw; f += 4) {
                const u64 a0 = reg[f], a1 = reg[f + 1], a2 = reg[f + 2], a3 = reg[f + 3];
                before += (a0 > ce) + (a1 > ce) + (a2 > ce) + (a3 > ce);
            }
            for (; f < cw; ++f) before += reg[f] > ce;
        }
        if (before < kk) win[before] = ce;
    }
}

// Final top-m: candidates sorted by one warp when they fit its registers,
// else ranked by the whole block; win[rank] for rank < kk.  Ends with a
// barrier.
__device__ void finish_top(int s, int kk, u64 *win, SelShared &sh) {
    const int c = candidate_count(s, sh);
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    if (c <= 256) {
        if (warp == 0) {
            if (c <= 64) {
                u64 v[2];
                warp_gather_sorted<2>(s, sh, v);
#pragma unroll
                for (int q = 0; q < 2; ++q)
                    if (q * 32 + lane < kk) win[q * 32 + lane] = v[q];
            } else if (c <= 128) {
                u64 v[4];
                warp_gather_sorted<4>(s, sh, v);
#pragma unroll
                for (int q = 0; q < 4; ++q)
                    if (q * 32 + lane < kk) win[q * 32 + lane] = v[q];
            } else {
                u64 v[8];
                warp_gather_sorted<8>(s, sh, v);
#pragma unroll
                for (int q = 0; q < 8; ++q)
                    if (q * 32 + lane < kk) win[q * 32 + lane] = v[q];
            }
        }
    } else {
        block_rank(s, kk, win, sh);
    }
    __syncthreads();
}

// Exact chunk scores of one key row against q (fp32 in shared memory):
// out[alpha] = sum_{c < dk} row[alpha*dk + c] * q[alpha*dk + c]  (Eq. 4).
// 16-byte loads, up to 8 in flight, when the row and chunks are aligned.
template <typename T>
__device__ void row_scores(const T *row, const float *q, const Dims &d, float *out) {
    constexpr int EPV = 16 / sizeof(T);
    const int dk = d.dk;
    const bool vec = d.d_k % EPV == 0 && dk % EPV == 0 && ((uintptr_t)row & 15) == 0;
#pragma unroll 1
    for (int al = 0; al < d.r; ++al) {
        const int c0 = al * dk;
        float acc = 0.f;
        if (vec) {
            const uint4 *rv = reinterpret_cast<const uint4 *>(row + c0);
            const int nv = dk / EPV;
#pragma unroll 1
            for (int v0 = 0; v0 < nv; v0 += 8) {
                uint4 buf[8];
#pragma unroll
                for (int u = 0; u < 8; ++u)
                    buf[u] = v0 + u < nv ? rv[v0 + u] : make_uint4(0, 0, 0, 0);
#pragma unroll
                for (int u = 0; u < 8; ++u) {
                    if (v0 + u >= nv) break;
                    float f[EPV];
                    unpack16<T>(buf[u], f);
                    const float *qq = q + c0 + (v0 + u) * EPV;
#pragma unroll
                    for (int e = 0; e < EPV; ++e) acc = fmaf(f[e], qq[e], acc);
                }
            }
        } else {
#pragma unroll 4
            for (int c = 0; c < dk; ++c) acc = fmaf(to_f(row[c0 + c]), q[c0 + c], acc);
        }
        out[al] = acc;
    }
}

// One warp per axis: the top-k of the axis' candidates, in increasing key
// index (so that enumerating I x J row-major is increasing v = i*K + j), and
// each survivor's exact chunk scores, one lane per survivor.
template <typename T, int R>
__device__ void finish_axis(const Dims &d, const Ptrs &p, int h, int axis, const float *qv,
                            const SelShared &sh, int *sel, float *S_out) {
    const int lane = threadIdx.x & 31;
    const int k = d.k;
    u64 v[R];
    warp_gather_sorted<R>(axis, sh, v);
    u64 pk[R];   // winners keyed by ~position: descending order = increasing index
#pragma unroll
    for (int q = 0; q < R; ++q)
        pk[q] = q * 32 + lane < k ? (u64)(uint32_t)(~pos_of(v[q])) : 0ull;
    warp_sort_desc<R>(pk);
    const T *keys = static_cast<const T *>(axis == 0 ? p.k_row : p.k_col);
#pragma unroll
    for (int q = 0; q < R; ++q) {
        const int e = q * 32 + lane;
        if (e < k) {
            const uint32_t pos = ~(uint32_t)pk[q];
            sel[e] = (int)pos;
            row_scores<T>(keys + ((int64_t)h * d.K + pos) * d.d_k, qv + axis * d.d_k, d,
                          S_out + e * d.r);
        }
    }
}

template <typename T>
__device__ void finish_axes(const Dims &d, const Ptrs &p, int h, const float *qv,
                            const SelShared &sh, int *sel_i, int *sel_j, float *srow,
                            float *scol) {
    const int warp = threadIdx.x >> 5;
    if (warp >= 2) return;
    const int c = candidate_count(warp, sh);   // <= 256 (see select_candidates)
    int *sel = warp == 0 ? sel_i : sel_j;
    float *So = warp == 0 ? srow : scol;
    if (c <= 64) finish_axis<T, 2>(d, p, h, warp, qv, sh, sel, So);
    else if (c <= 128) finish_axis<T, 4>(d, p, h, warp, qv, sh, sel, So);
    else finish_axis<T, 8>(d, p, h, warp, qv, sh, sel, So);
}

struct SelLayout {
    uint32_t *key0, *key1;
    float *qv;          // [2][D_k] row and column query of this (token, head)
    int *sel_i, *sel_j;
    float *srow, *scol, *R;
};

__device__ SelLayout carve(const Dims &d, unsigned char *base) {
    SelLayout L;
    size_t off = 0;
    L.key0 = reinterpret_cast<uint32_t *>(base + off);
    off += sizeof(uint32_t) * max(d.K, d.k * d.k);
    L.key1 = reinterpret_cast<uint32_t *>(base + off);
    off += sizeof(uint32_t) * d.K;
    L.qv = reinterpret_cast<float *>(base + off);
    off += sizeof(float) * 2 * d.d_k;
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

template <typename T>
__global__ void __launch_bounds__(kThreads) select_kernel(Dims d, Ptrs p) {
    extern __shared__ __align__(16) unsigned char smem_raw[];
    __shared__ SelShared sh;
    const int b = blockIdx.x / d.H, h = blockIdx.x % d.H;
    SelLayout L = carve(d, smem_raw);
    const int r = d.r, K = d.K, k = d.k, m = d.m;
    const float *C = p.core + (int64_t)h * r * r;
    const uint32_t *A0 = p.akey + (((int64_t)b * d.H + h) * 2) * (int64_t)K;
    const uint32_t *A1 = A0 + K;

    // rank-1 score keys of both axes (Eq. 6-7, from the scoring kernel) and
    // the row/column query of this (token, head), summed over its D_i splits
    uint32_t vm0 = 0, vm1 = 0;
    for (int i0 = threadIdx.x; i0 < K; i0 += 4 * kThreads) {
        uint32_t a[4], c2[4];
#pragma unroll
        for (int q = 0; q < 4; ++q) {
            const int i = i0 + q * kThreads;
            a[q] = i < K ? A0[i] : 0u;
            c2[q] = i < K ? A1[i] : 0u;
        }
#pragma unroll
        for (int q = 0; q < 4; ++q) {
            const int i = i0 + q * kThreads;
            if (i < K) {
                L.key0[i] = a[q];
                L.key1[i] = c2[q];
                vm0 = max(vm0, a[q]);
                vm1 = max(vm1, c2[q]);
            }
        }
    }
    {
        const int HD = d.H * d.d_k;
        for (int e = threadIdx.x; e < 2 * d.d_k; e += kThreads) {
            const int axis = e / d.d_k, c = e % d.d_k;
            const int a = (axis == 1 && d.A == 2) ? 1 : 0;
            const float *src = p.q_part + ((int64_t)a * d.B + b) * HD + h * d.d_k + c;
            const int64_t split_stride = (int64_t)d.A * d.B * HD;
            float q = 0.f;
            for (int s = 0; s < d.q_splits; ++s) q += src[s * split_stride];
            L.qv[e] = q;
        }
    }
    // (the first barrier of select_candidates orders these shared-memory writes)

    // Eq. 8-9: top-k of both axes
    select_candidates(L.key0, L.key1, 2, K, k, vm0, vm1, sh);
    // survivors in increasing index, with their exact chunk scores (Eq. 4)
    finish_axes<T>(d, p, h, L.qv, sh, L.sel_i, L.sel_j, L.srow, L.scol);
    __syncthreads();

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
    uint32_t vmg = 0;
    const int dii = kThreads / k, djj = kThreads % k;   // (ii, jj) step per c += kThreads
    int ii = threadIdx.x / k, jj = threadIdx.x % k;
    for (int c = threadIdx.x; c < k2; c += kThreads) {
        float g = 0.f;
        for (int be = 0; be < r; ++be) g = fmaf(L.R[ii * r + be], L.scol[jj * r + be], g);
        const uint32_t kg = f2ord(g);
        L.key0[c] = kg;
        vmg = max(vmg, kg);
        ii += dii;
        jj += djj;
        if (jj >= k) { jj -= k; ++ii; }
    }
    select_candidates(L.key0, nullptr, 1, k2, m, vmg, 0u, sh);
    finish_top(0, m, sh.fwin, sh);

    // PKM's softmax over the m selected scores (Eq. 3); Trick 1 skips it
    const float gmax = ord2f(key_of(sh.fwin[0]));
    if (d.act == ULTRAMEM_ACT_SOFTMAX) {
        if (threadIdx.x < 32) {
            float z = 0.f;
            for (int e = threadIdx.x; e < m; e += 32) z += __expf(ord2f(key_of(sh.fwin[e])) - gmax);
#pragma unroll
            for (int off = 16; off > 0; off >>= 1) z += __shfl_xor_sync(kFull, z, off);
            if (threadIdx.x == 0) sh.scalar = z;
        }
        __syncthreads();
    }
    const int64_t base = ((int64_t)b * d.H + h) * m;
    for (int e = threadIdx.x; e < m; e += kThreads) {
        const u64 wc = sh.fwin[e];
        const int c = (int)pos_of(wc);
        const int ii = c / k, jj = c - ii * k;
        const uint64_t v = (uint64_t)L.sel_i[ii] * (uint64_t)K + (uint64_t)L.sel_j[jj];
        const float g = ord2f(key_of(wc));
        const float w = d.act == ULTRAMEM_ACT_SOFTMAX ? __expf(g - gmax) / sh.scalar : g;
        const uint64_t vs = shuffle_address(d, p.perm, v);   // Eq. 14
        const uint64_t pb = vs / (uint64_t)d.N;
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
    size_t nkey0 = (size_t)(d.K > d.k * d.k ? d.K : d.k * d.k);
    size_t off = sizeof(uint32_t) * (nkey0 + d.K) + sizeof(float) * 2 * d.d_k +
                 sizeof(int) * 2 * d.k + sizeof(float) * 3 * d.k * d.r;
    return (off + 15) & ~size_t(15);
}

cudaError_t launch_select(const Dims &d, const Ptrs &p, cudaStream_t st) {
    if (d.dtype == ULTRAMEM_BF16)
        select_kernel<__nv_bfloat16><<<d.B * d.H, kThreads, select_smem_bytes(d), st>>>(d, p);
    else
        select_kernel<float><<<d.B * d.H, kThreads, select_smem_bytes(d), st>>>(d, p);
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
    const int bytes = (int)select_smem_bytes(d);
    cudaError_t e = cudaFuncSetAttribute(select_kernel<float>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
    if (e != cudaSuccess) return e;
    return cudaFuncSetAttribute(select_kernel<__nv_bfloat16>,
                                cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
}

}  // namespace um
