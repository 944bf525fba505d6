// um_select.cu -- S4..S7 for one (token, head) per CTA:
//   top-k of each axis on the rank-1 score keys         (Eq. 8-9)
//   exact chunk scores S_alpha of the 2k survivors      (Eq. 4)
//   exact Tucker score g on the k*k survivor pairs      (Eq. 10; with product
//                                                         keys s_row + s_col, Eq. 2)
//   top-m of g, ordered by (score desc, v asc)          (Eq. 10)
//   weights (raw scores, or PKM's softmax), shuffle     (Trick 1, Eq. 3, Eq. 14)
//   with h component cores (MCS), the h individual scores of each winner
//                                                        (Eq. 16-17)
// No K*K grid is ever formed.  The scoring kernel leaves, per key, the
// order-preserving 32-bit key of its fp32 rank-1 score; the exact chunk
// scores of the k survivors of each axis are recomputed here from q and the
// key rows.  Ties go to the smaller index.
//
// Top-k of n keys, in two stages.  Candidates: each thread keeps the two
// largest of its share of the keys; each warp takes the j-th largest of its
// lanes' 64 values (j = ceil(k / 8): j rounds of a warp max that removes one
// instance) and tau is the smallest of the 8 warp values.  Every warp owns at
// least j keys >= tau, so at least k keys are >= tau whatever the input:
// every key of the top k is >= tau.  The keys >= tau are appended to one
// flat list per selection (a hit mask per lane, a warp scan, one shared
// atomic per warp).  When the list is long the same bound is taken again over
// it; when it overflows (heavy ties) an exact radix select replaces it.
// Order: the candidates are 64-bit composites (key, ~position) whose
// descending order is key descending then position ascending; the rank of
// each is the number of candidates above it (counted by a group of lanes per
// candidate, or by binary searches in sorted warp runs on long grids), and the
// ones ranked below k are the winners, in rank order.
#include "um_internal.cuh"

namespace um {
namespace {

constexpr int kThreads = 256;
constexpr int kWarps = kThreads / 32;
constexpr int kCap = 1024;                 // candidates per selection
constexpr int kPerThread = kCap / kThreads;
constexpr int kMaxK = 128;
constexpr int kMaxM = 1024;
static_assert(kMaxM <= kCap, "the final winners reuse a candidate list");
constexpr int kMaxR = 8;
constexpr int kRankSort = 256;             // longer lists are tightened first
constexpr uint32_t kPairMix = 421;         // prime > kMaxK: the order of the Tucker pairs
static_assert(kWarps == 8, "the Tucker pairs' assignment spreads rows over 8 warps");
static_assert(kPairMix > kMaxK, "kPairMix must be coprime with every k^2");
// value rows of a batch beyond this are not prefetched into L2 by the
// selection: they would be evicted before the gather reads them
constexpr uint64_t kPrefetchMaxBytes = 64ull << 20;
constexpr unsigned kFull = 0xffffffffu;

// counter slots of SelShared::cnt
constexpr int kCntAxis = 0;      // +s: first pass of axis s
constexpr int kCntAxisT = 2;     // +s: tightened axis s
constexpr int kCntTop = 4;       // final top-m
constexpr int kCntTopT = 5;      // tightened final top-m

typedef unsigned long long u64;

struct SelShared {
    __align__(16) u64 cand[2][kCap];   // flat candidate lists, one per selection; the
                                       // final winners by rank reuse list 1
    __align__(16) u64 win[2][kMaxK];   // axis winners by rank
    float core[kMaxR * kMaxR];         // C of this head
    int cnt[8];                        // list lengths (may exceed kCap: overflow)
    uint32_t vt[2][kWarps];
    __align__(16) u64 runs[kThreads];  // sorted warp runs of rank_sorted
    int hist[256];
    int warp_tot[kWarps];
    int digit, remaining;
    float scalar;
    double dscalar;   // fp32 storage: the softmax denominator in fp64
    unsigned long long xbar;   // paired selection: the row CTA's exchange mbarrier
};

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

// Inserts v into a lane's two largest values m1 >= m2.
__device__ __forceinline__ void top2(uint32_t v, uint32_t &m1, uint32_t &m2) {
    m2 = max(m2, min(v, m1));
    m1 = max(m1, v);
}

// The j-th largest (1 <= j <= 32) of the warp's 64 values {m1, m2}: j rounds
// of a warp maximum, each removing one instance (the lowest lane holding it).
__device__ __forceinline__ uint32_t warp_jth_top2(uint32_t m1, uint32_t m2, int j) {
    const int lane = threadIdx.x & 31;
    uint32_t t = 0u;
#pragma unroll 1
    for (int r = 0; r < j; ++r) {
        t = __reduce_max_sync(kFull, m1);
        const unsigned bal = __ballot_sync(kFull, m1 == t);
        if (lane == __ffs(bal) - 1) {
            m1 = m2;
            m2 = 0u;
        }
    }
    return t;
}

// Each warp's bound for a top-kk selection into sh.vt[s][warp] from its
// lanes' two largest keys (a0 >= a1 of selection 0, b0 >= b1 of selection 1).
// No barrier.
__device__ __forceinline__ void warp_bounds(uint32_t a0, uint32_t a1, uint32_t b0, uint32_t b1,
                                            int ns, int kk, SelShared &sh) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int j = (kk + kWarps - 1) / kWarps;
    const uint32_t t0 = j <= 32 ? warp_jth_top2(a0, a1, j) : 0u;
    const uint32_t t1 = ns > 1 && j <= 32 ? warp_jth_top2(b0, b1, j) : 0u;
    if (lane == 0) {
        sh.vt[0][warp] = t0;
        sh.vt[1][warp] = t1;
    }
}

__device__ __forceinline__ uint32_t block_bound(int s, const SelShared &sh) {
    uint32_t tau = sh.vt[s][0];
#pragma unroll
    for (int w = 1; w < kWarps; ++w) tau = min(tau, sh.vt[s][w]);
    return tau;
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

// One digit of a radix select: given the histogram of the current digit
// over the entries that match the digits chosen so far, warp 0 finds the
// digit that holds the `remaining`-th largest entry and leaves it, and the
// rank still to go within it, in sh.digit and sh.remaining.
__device__ __forceinline__ void radix_digit(int remaining, SelShared &sh) {
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
        radix_digit(remaining, sh);
        __syncthreads();
        prefix |= (uint32_t)sh.digit << shift;
        mask |= 255u << shift;
        remaining = sh.remaining;
        __syncthreads();
    }
    *need_eq = remaining;
    return prefix;
}

// Exact replacement of an overflowed list: exactly kk candidates (every key
// > T, then the first ties at T in position order) into cand[s], length in
// cnt[slot].  Out of line: it only runs on heavy ties.
__device__ __noinline__ void radix_fallback(const uint32_t *key, int n, int kk, int s, int slot,
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
    if (threadIdx.x == 0) sh.cnt[slot] = kk;
    __syncthreads();
}

// Appends the lanes' composites with pr set to list (length counter *cnt):
// one shared atomic per warp.  Entries past kCap are dropped (the counter
// still counts them, which marks the overflow).
__device__ __forceinline__ void warp_append(bool pr, u64 comp, u64 *list, int *cnt) {
    const int lane = threadIdx.x & 31;
    const unsigned bal = __ballot_sync(kFull, pr);
    if (bal == 0u) return;
    int base = 0;
    if (lane == 0) base = atomicAdd(cnt, __popc(bal));
    base = __shfl_sync(kFull, base, 0);
    const int slot = base + __popc(bal & ((1u << lane) - 1u));
    if (pr && slot < kCap) list[slot] = comp;
}

// The scoring's candidate list of axis s (Dims::cand): every key of the
// axis' top k is in it, with the keys above a bound, as composites.  The
// list is G segments of 16 entries (one per group of 16 keys); segment g
// holds its group's candidates in its first cnt[g] entries (the counts
// replace the group maxima in gstat).  Up to kCap entries are gathered
// into cand[s] (placed by a block scan of the threads' counts); a longer
// list (heavy ties) is replaced by its exact top kk, a radix select over the
// 64-bit composites (distinct: exactly kk are >= the kk-th largest).
// Length in cnt[slot].  Whole block; ends with a barrier.
constexpr int kSeg = 16;               // entries of a list segment (keys of a group)
constexpr int kMaxSegPerThread = 4;   // G <= 1024 segments
__device__ __noinline__ void cand_fallback(const u64 *seg, const uint32_t *cnt, int G, int kk,
                                           int s, int slot, SelShared &sh) {
    const int n = kSeg * G;
    auto entry = [&](int i) -> u64 {   // 0 for an empty slot (below every composite kept)
        return i % kSeg < (int)min(cnt[i / kSeg], (uint32_t)kSeg) ? seg[i] : 0ull;
    };
    u64 prefix = 0, mask = 0;
    int remaining = kk;
    for (int shift = 56; shift >= 0; shift -= 8) {
        for (int i = threadIdx.x; i < 256; i += kThreads) sh.hist[i] = 0;
        __syncthreads();
        for (int i = threadIdx.x; i < n; i += kThreads) {
            const u64 v = entry(i);
            if (v && (v & mask) == prefix) atomicAdd(&sh.hist[(int)((v >> shift) & 255u)], 1);
        }
        __syncthreads();
        radix_digit(remaining, sh);
        __syncthreads();
        prefix |= (u64)sh.digit << shift;
        mask |= (u64)255 << shift;
        remaining = sh.remaining;
        __syncthreads();
    }
    if (threadIdx.x == 0) sh.cnt[slot] = 0;
    __syncthreads();
    for (int i0 = 0; i0 < n; i0 += kThreads) {   // uniform trip count
        const int i = i0 + threadIdx.x;
        const u64 v = i < n ? entry(i) : 0ull;
        warp_append(v && v >= prefix, v, sh.cand[s], &sh.cnt[slot]);
    }
    __syncthreads();
}

// Both axes' lists of one (token, head) (lists `list0` and `list0 + 1`)
// into cand[0] and cand[1], lengths in cnt[kCntAxis + s].  One block scan
// places both (the two axes' counts packed in the low and high 16 bits:
// each total is at most 16 G <= 16384), and each thread loads the first
// entry of all its segments before it stores any, so that the copies cost
// one round trip to memory, not one per segment.  Whole block; ends with a
// barrier.
__device__ void load_lists(const Ptrs &p, int64_t list0, int G, int kk, SelShared &sh) {
    const uint32_t *cnt[2] = {p.gstat + list0 * G, p.gstat + (list0 + 1) * G};
    const u64 *seg[2] = {p.cand + list0 * (int64_t)G * kSeg, p.cand + (list0 + 1) * (int64_t)G * kSeg};
    int mine[2][kMaxSegPerThread], tot = 0;
#pragma unroll
    for (int s = 0; s < 2; ++s) {
#pragma unroll
        for (int q = 0; q < kMaxSegPerThread; ++q) {
            const int g = threadIdx.x + q * kThreads;
            mine[s][q] = g < G ? (int)min(cnt[s][g], (uint32_t)kSeg) : 0;
            tot += mine[s][q] << (16 * s);
        }
    }
    const int o = block_exclusive_scan(tot, sh);
    if (threadIdx.x == kThreads - 1) {
        sh.cnt[kCntAxis] = (o + tot) & 0xffff;
        sh.cnt[kCntAxis + 1] = (o + tot) >> 16;
    }
    __syncthreads();
    const int c[2] = {sh.cnt[kCntAxis], sh.cnt[kCntAxis + 1]};
    // the first entry of every segment of this thread, then the rest
    u64 first[2][kMaxSegPerThread];
#pragma unroll
    for (int s = 0; s < 2; ++s)
#pragma unroll
        for (int q = 0; q < kMaxSegPerThread; ++q)
            first[s][q] = mine[s][q] > 0 && c[s] <= kCap
                              ? seg[s][(int64_t)(threadIdx.x + q * kThreads) * kSeg]
                              : 0ull;
#pragma unroll
    for (int s = 0; s < 2; ++s) {
        if (c[s] > kCap) continue;   // uniform: the radix select below replaces it
        int at = (o >> (16 * s)) & 0xffff;
#pragma unroll
        for (int q = 0; q < kMaxSegPerThread; ++q) {
            if (mine[s][q] == 0) continue;
            const u64 *sg = seg[s] + (int64_t)(threadIdx.x + q * kThreads) * kSeg;
            sh.cand[s][at++] = first[s][q];
            for (int e = 1; e < mine[s][q]; ++e) sh.cand[s][at++] = sg[e];
        }
        // fewer than kk is impossible (the bound guarantees kk); should it
        // happen, positions past K mark the missing entries (recorded)
        for (int f = c[s] + threadIdx.x; f < kk; f += kThreads)
            sh.cand[s][f] = comp_of(0u, 0xffffffffu - (uint32_t)f);
    }
    __syncthreads();
#pragma unroll
    for (int s = 0; s < 2; ++s) {
        if (c[s] > kCap) {
            cand_fallback(seg[s], cnt[s], G, kk, s, kCntAxis + s, sh);
        } else if (c[s] < kk) {
            if (threadIdx.x == 0) {
                sh.cnt[kCntAxis + s] = kk;
                atomicOr(p.err, kErrInternal);
            }
        }
    }
    __syncthreads();
}

// Appends key[i] >= tau_s (i < n) of NS selections to their lists.  A round
// covers 4 kThreads 16-byte groups of keys; lane l of warp w reads groups
// (q kWarps + w) 32 + l, q < 4, so that a warp's loads are contiguous, and
// marks its hits in a 16-bit mask.  A warp scan of the lanes' hit counts
// places them, one shared atomic per warp and selection reserves the room,
// and each lane writes its hits by walking its mask (re-reading a hit's key).
// The last group may extend past n (up to the 16-byte end of the array's
// section); its extra entries are masked.
template <int NS>
__device__ void compact(const uint32_t *key0, const uint32_t *key1, int n, uint32_t tau0,
                        uint32_t tau1, SelShared &sh, int slot0, int slot1) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int n4 = (n + 3) >> 2;
#pragma unroll 1
    for (int r0 = 0; r0 < n4; r0 += 4 * kThreads) {
#pragma unroll
        for (int s = 0; s < NS; ++s) {
            const uint32_t *key = s ? key1 : key0;
            const uint4 *k4 = reinterpret_cast<const uint4 *>(key);
            const uint32_t tau = s ? tau1 : tau0;
            uint32_t mask = 0u;
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                const int g = r0 + (q * kWarps + warp) * 32 + lane;
                if (g < n4) {
                    const uint4 v = k4[g];
                    uint32_t m4 = (uint32_t)(v.x >= tau) | (uint32_t)(v.y >= tau) << 1 |
                                  (uint32_t)(v.z >= tau) << 2 | (uint32_t)(v.w >= tau) << 3;
                    const int valid = n - 4 * g;   // >= 1
                    if (valid < 4) m4 &= (1u << valid) - 1u;
                    mask |= m4 << (4 * q);
                }
            }
            const int cnt = __popc(mask);
            int incl = cnt;
#pragma unroll
            for (int off = 1; off < 32; off <<= 1) {
                const int y = __shfl_up_sync(kFull, incl, off);
                if (lane >= off) incl += y;
            }
            const int tot = __shfl_sync(kFull, incl, 31);
            if (tot == 0) continue;   // warp-uniform
            int base = 0;
            if (lane == 31) base = atomicAdd(&sh.cnt[s ? slot1 : slot0], tot);
            int slot = __shfl_sync(kFull, base, 31) + incl - cnt;
            u64 *list = sh.cand[s];
            while (mask) {
                const int b = __ffs(mask) - 1;
                mask &= mask - 1u;
                const int i = 4 * (r0 + ((b >> 2) * kWarps + warp) * 32 + lane) + (b & 3);
                if (slot < kCap) list[slot] = comp_of(key[i], (uint32_t)i);
                ++slot;
            }
        }
    }
}

// The same bound taken again over list s (c entries, c <= kCap); the
// survivors replace the list, length in cnt[slot_out].  Whole block; ends
// with a barrier.
__device__ void tighten(int s, int c, int kk, int slot_out, SelShared &sh) {
    u64 mine[kPerThread];
    uint32_t m1 = 0u, m2 = 0u;
#pragma unroll
    for (int q = 0; q < kPerThread; ++q) {
        const int f = threadIdx.x + q * kThreads;
        mine[q] = f < c ? sh.cand[s][f] : 0ull;
        top2(key_of(mine[q]), m1, m2);
    }
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int j = (kk + kWarps - 1) / kWarps;
    const uint32_t tw = j <= 32 ? warp_jth_top2(m1, m2, j) : 0u;
    if (lane == 0) sh.vt[s][warp] = tw;
    __syncthreads();   // also: every list entry has been read
    const uint32_t tau = block_bound(s, sh);
#pragma unroll
    for (int q = 0; q < kPerThread; ++q) {
        const bool pr = threadIdx.x + q * kThreads < c && key_of(mine[q]) >= tau;
        warp_append(pr, mine[q], sh.cand[s], &sh.cnt[slot_out]);
    }
    __syncthreads();
}

// Length of list s once it can be ranked: the radix select replaces an
// overflowed list, a long one is tightened.  Uniform; may sync.
__device__ int settle(int s, const uint32_t *key, int n, int kk, int slot, int slot_t,
                      SelShared &sh) {
    const int c = sh.cnt[slot];
    if (c > kCap) {
        radix_fallback(key, n, kk, s, slot, sh);
        return kk;
    }
    if (c > kRankSort && c > 2 * kk) {
        tighten(s, c, kk, slot_t, sh);
        return sh.cnt[slot_t];
    }
    return c;
}

// Ranks of the c entries of list (threads [0, nt) of the selection, nt a
// power of two, tid the thread's index among them): a group of G lanes per
// entry counts the entries above it; entries of rank < kk go to win[rank].
__device__ __forceinline__ void rank_list(const u64 *list, int c, int kk, u64 *win, int tid,
                                          int nt) {
    int G = 1;
    while (G < 32 && 2 * G * c <= nt) G <<= 1;
    const int sub = tid & (G - 1), slots = nt / G;
    const int span = (((c + G - 1) / G) + 7) & ~7;
    const int lo = min(c, sub * span), hi = min(c, lo + span);
    const ulonglong2 *l2 = reinterpret_cast<const ulonglong2 *>(list);
#pragma unroll 1
    for (int f0 = 0; f0 < c; f0 += slots) {
        const int f = f0 + tid / G;
        const u64 me = f < c ? list[f] : ~0ull;
        int before = 0, g = lo;
#pragma unroll 1
        for (; g + 8 <= hi; g += 8) {
            const ulonglong2 a = l2[g / 2], b = l2[g / 2 + 1], x = l2[g / 2 + 2],
                             y = l2[g / 2 + 3];
            before += (a.x > me) + (a.y > me) + (b.x > me) + (b.y > me) + (x.x > me) +
                      (x.y > me) + (y.x > me) + (y.y > me);
        }
        for (; g < hi; ++g) before += list[g] > me;
        for (int off = G >> 1; off > 0; off >>= 1) before += __shfl_xor_sync(kFull, before, off);
        if (sub == 0 && f < c && before < kk) win[before] = me;
    }
}

// Prefetch of [ptr, ptr + bytes) into L2, one 128-byte line per request.
__device__ __forceinline__ void prefetch_l2(const void *ptr, uint32_t bytes) {
    const char *c = static_cast<const char *>(ptr);
    for (uint32_t o = 0; o < bytes; o += 128) asm volatile("prefetch.global.L2 [%0];" ::"l"(c + o));
}

template <int ID>
__device__ __forceinline__ void named_barrier(int nthreads) {
    asm volatile("bar.sync %0, %1;" ::"n"(ID), "r"(nthreads) : "memory");
}

// Exact ranks of the c <= nt entries of list (distinct composites) for
// threads [0, nt) of the selection (tid the thread's index among them, nt a
// multiple of 32): each warp sorts its run of 32 in registers (descending
// bitonic network), the runs go to runs[nt], and an entry's rank is its place
// in its own run plus, per other run, the number of entries above it (a
// 5-step binary search).  Entries of rank < kk go to win[rank].  BAR: the
// named barrier of these nt threads.
template <int BAR, int NT>
__device__ void rank_sorted(const u64 *list, int c, int kk, u64 *win, u64 *runs, int tid) {
    constexpr int nt = NT, nw = NT / 32;
    const int lane = tid & 31, w = tid >> 5;
    u64 x = tid < c ? list[tid] : 0ull;   // padding sorts below every entry
#pragma unroll
    for (int blk = 2; blk <= 32; blk <<= 1)
#pragma unroll
        for (int st = blk >> 1; st > 0; st >>= 1) {
            const u64 o = __shfl_xor_sync(kFull, x, st);
            const bool keep_max = ((lane & st) == 0) == ((lane & blk) == 0);
            x = keep_max ? (x > o ? x : o) : (x < o ? x : o);
        }
    runs[w * 32 + lane] = x;
    named_barrier<BAR>(nt);
    const int cw = min(32, max(0, c - 32 * w));   // real entries of this run
    if (lane < cw) {
        // the searches of the other runs are independent: interleaved steps
        int pos[nw];
#pragma unroll
        for (int v = 0; v < nw; ++v) pos[v] = 0;
#pragma unroll
        for (int step = 16; step > 0; step >>= 1)
#pragma unroll
            for (int v = 0; v < nw; ++v)
                if (runs[v * 32 + pos[v] + step - 1] > x) pos[v] += step;
        int rank = lane;
#pragma unroll
        for (int v = 0; v < nw; ++v) {
            // entries of the descending run above x: 0 .. 32 (the steps reach 31)
            const int cnt = pos[v] + (runs[v * 32 + pos[v]] > x);
            rank += v == w ? 0 : cnt;
        }
        if (rank < kk) win[rank] = x;
    }
}

struct SelLayout {
    float *qv;          // [2][D_k] row and column query of this (token, head)
    uint32_t *key0;     // [max(K, k*k)] axis-0 keys, then the g keys
    uint32_t *key1;     // [K] axis-1 keys (free once the axis winners are ranked)
    int *sel_i, *sel_j; // [k] surviving rows / columns in increasing index
    float *R, *scol;    // [k][r] R = S_row^T C and S_col of the survivors
    float *srow;        // MCS, fp32: [k][r] S_row of the row survivors } in key1's
    float *cparts;      // MCS: [nc][r][r] component cores of this head } space
};

// Dynamic shared memory layout; every section starts on 16 bytes.
struct SelOffsets {
    size_t qv, key0, key1, sel_i, sel_j, R, scol, srow, cparts, total;
};
__host__ __device__ inline SelOffsets sel_offsets(const Dims &d) {
    auto up = [](size_t x) { return (x + 15) & ~size_t(15); };
    SelOffsets o;
    size_t off = 0;
    o.qv = off;    off = up(off + sizeof(float) * 2 * d.d_k);
    // streamed keys: the axes' keys stay in L2 (read twice), not in shared
    // memory; candidate lists: the selection reads no keys
    const int Ka = d.stream_keys || d.cand ? 0 : d.K;
    o.key0 = off;  off = up(off + sizeof(uint32_t) * (Ka > d.k * d.k ? Ka : d.k * d.k));
    // with MCS (and with fp32 storage), key1's space later holds S_row of the
    // row survivors and the component cores (so that the block's shared
    // memory does not grow)
    const bool mcs = d.nc > 1;
    const bool keep_srow = mcs || d.dtype == ULTRAMEM_F32;
    const int mcs_floats = keep_srow ? d.k * d.r + (mcs ? d.nc * d.r * d.r : 0) : 0;
    o.key1 = off;  off = up(off + sizeof(uint32_t) * (Ka > mcs_floats ? Ka : mcs_floats));
    o.srow = o.key1;
    o.cparts = o.key1 + sizeof(float) * d.k * d.r;
    o.sel_i = off; off = up(off + sizeof(int) * d.k);
    o.sel_j = off; off = up(off + sizeof(int) * d.k);
    o.R = off;     off = up(off + sizeof(float) * d.k * d.r);
    o.scol = off;  off = up(off + sizeof(float) * d.k * d.r);
    o.total = off;
    return o;
}

__device__ SelLayout carve(const Dims &d, unsigned char *base) {
    const SelOffsets o = sel_offsets(d);
    SelLayout L;
    L.qv = reinterpret_cast<float *>(base + o.qv);
    L.key0 = reinterpret_cast<uint32_t *>(base + o.key0);
    L.key1 = reinterpret_cast<uint32_t *>(base + o.key1);
    L.sel_i = reinterpret_cast<int *>(base + o.sel_i);
    L.sel_j = reinterpret_cast<int *>(base + o.sel_j);
    L.R = reinterpret_cast<float *>(base + o.R);
    L.scol = reinterpret_cast<float *>(base + o.scol);
    L.srow = reinterpret_cast<float *>(base + o.srow);
    L.cparts = reinterpret_cast<float *>(base + o.cparts);
    return L;
}

// Loads the rank-1 score keys of both axes (Eq. 6-7, written by the scoring
// kernel) into shared memory and returns this thread's two largest of each
// axis (padding reads as 0, below every key); all loads of a round are
// issued before any store.  Each key is read once: the loads are streaming
// (L2 evict-first), so that a long batch's keys do not push the key rows,
// which every (token, head) reads again, out of L2.  With `stream` the keys
// are not stored (the compaction reads them again from L2) and are loaded
// with the L2 caching kept.
__device__ __forceinline__ uint4 ld_key4(const uint4 *p, bool stream) {
    return stream ? __ldcg(p) : __ldcs(p);
}
__device__ __forceinline__ uint32_t ld_key(const uint32_t *p, bool stream) {
    return stream ? __ldcg(p) : __ldcs(p);
}
template <int NS = 2>   // axes loaded: both, or (NS = 1) the one in A0
__device__ __forceinline__ void load_keys(const uint32_t *A0, const uint32_t *A1, int K,
                                          const SelLayout &L, uint32_t (&top)[2][2],
                                          bool stream) {
    uint32_t a1 = 0u, a2 = 0u, b1 = 0u, b2 = 0u;
    if ((K & 3) == 0) {
        const uint4 *V0 = reinterpret_cast<const uint4 *>(A0);
        const uint4 *V1 = reinterpret_cast<const uint4 *>(A1);
        uint4 *S0 = reinterpret_cast<uint4 *>(L.key0), *S1 = reinterpret_cast<uint4 *>(L.key1);
        const int nv = K >> 2;
#pragma unroll 1
        for (int v0 = threadIdx.x; v0 < nv; v0 += 4 * kThreads) {
            uint4 a[4], c[4];
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                const int i = v0 + q * kThreads;
                a[q] = i < nv ? ld_key4(V0 + i, stream) : make_uint4(0, 0, 0, 0);
                c[q] = NS > 1 && i < nv ? ld_key4(V1 + i, stream) : make_uint4(0, 0, 0, 0);
            }
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                const int i = v0 + q * kThreads;
                if (i < nv && !stream) {
                    S0[i] = a[q];
                    if (NS > 1) S1[i] = c[q];
                }
                top2(a[q].x, a1, a2);
                top2(a[q].y, a1, a2);
                top2(a[q].z, a1, a2);
                top2(a[q].w, a1, a2);
                top2(c[q].x, b1, b2);
                top2(c[q].y, b1, b2);
                top2(c[q].z, b1, b2);
                top2(c[q].w, b1, b2);
            }
        }
    } else {
#pragma unroll 1
        for (int i0 = threadIdx.x; i0 < K; i0 += 4 * kThreads) {
            uint32_t a[4], c[4];
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                const int i = i0 + q * kThreads;
                a[q] = i < K ? ld_key(A0 + i, stream) : 0u;
                c[q] = NS > 1 && i < K ? ld_key(A1 + i, stream) : 0u;
            }
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                const int i = i0 + q * kThreads;
                if (i < K && !stream) {
                    L.key0[i] = a[q];
                    if (NS > 1) L.key1[i] = c[q];
                }
                top2(a[q], a1, a2);
                top2(c[q], b1, b2);
            }
        }
    }
    top[0][0] = a1;
    top[0][1] = a2;
    top[1][0] = b1;
    top[1][1] = b2;
}

// A 16-byte load of a key row with the L2 evict-last policy: the rows are
// read again by the other (token, head) pairs of the batch.
__device__ __forceinline__ uint4 ld_key_row(const uint4 *ptr) {
    uint64_t pol;
    asm volatile("createpolicy.fractional.L2::evict_last.b64 %0, 1.0;" : "=l"(pol));
    uint4 v;
    asm volatile("ld.global.nc.L2::cache_hint.v4.u32 {%0, %1, %2, %3}, [%4], %5;"
                 : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
                 : "l"(ptr), "l"(pol));
    return v;
}

// The paired decode selection's cluster barrier (arrive, then wait).
__device__ __forceinline__ void cl_arrive_relaxed() {
    asm volatile("barrier.cluster.arrive.relaxed.aligned;" ::: "memory");
}
__device__ __forceinline__ void cl_wait() {
    asm volatile("barrier.cluster.wait.acquire.aligned;" ::: "memory");
}
// The exchange mbarrier of the paired selection (in the row CTA): one
// arrival, which also expects the column CTA's survivors' bytes; the init is
// published to the pair by a release fence and the pair's first cluster
// barrier.
__device__ __forceinline__ void xbar_init(unsigned long long *bar, uint32_t bytes) {
    const uint32_t a = (uint32_t)__cvta_generic_to_shared(bar);
    asm volatile("mbarrier.init.shared::cta.b64 [%0], 1;" ::"r"(a) : "memory");
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(a), "r"(bytes)
                 : "memory");
}
// A 32-bit store into the same shared-memory location of CTA `rank`, which
// completes 4 bytes of that CTA's mbarrier at the same offset as `bar`.
__device__ __forceinline__ void st_async_u32(const void *local, uint32_t rank, uint32_t v,
                                             const unsigned long long *bar) {
    const uint32_t a = (uint32_t)__cvta_generic_to_shared(local);
    const uint32_t b = (uint32_t)__cvta_generic_to_shared(bar);
    uint32_t ra, rb;
    asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(ra) : "r"(a), "r"(rank));
    asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(rb) : "r"(b), "r"(rank));
    asm volatile("st.async.shared::cluster.mbarrier::complete_tx::bytes.b32 [%0], %1, [%2];" ::"r"(ra),
                 "r"(v), "r"(rb)
                 : "memory");
}
// Bounded wait (about a second of SM cycles) for phase 0 of the exchange
// mbarrier, with cluster-scope acquire: the column CTA's stores are then
// visible.  Returns false when it gave up.
__device__ __forceinline__ bool xbar_wait(unsigned long long *bar) {
    const uint32_t a = (uint32_t)__cvta_generic_to_shared(bar);
    const long long start = clock64();
    for (;;) {
        uint32_t ok;
        asm volatile(
            "{\n\t.reg .pred p;\n\t"
            "mbarrier.try_wait.parity.acquire.cluster.shared::cta.b64 p, [%1], 0;\n\t"
            "selp.u32 %0, 1, 0, p;\n\t}"
            : "=r"(ok)
            : "r"(a)
            : "memory");
        if (ok) return true;
        if (clock64() - start > (1ll << 31)) return false;
    }
}

// The 2k axis survivors, one group of G lanes each: the survivor's place in
// increasing key index (so that enumerating I x J row-major is increasing
// v = i*K + j), and its exact chunk scores S_alpha (Eq. 4) from 16-byte
// loads of its key row split over the group.  Row survivors store
// R[i][b] = sum_a S_row[a,i] C[a,b], column survivors S_col[j][b].
// RM >= r bounds the rank at compile time (2 for the common ranks, else 8).
// gax < 0: both axes (winners of axis s in win[s]); gax = 0 or 1 (the
// paired decode selection): only axis gax, whose winners are in win[0].
template <typename T, int RM>
__device__ void axis_survivors(const Dims &d, const Ptrs &p, int h, const SelLayout &L,
                               const SelShared &sh, int gax = -1) {
    constexpr int EPV = 16 / sizeof(T);
    const int k = d.k, r = d.r, dk = d.dk, D = d.d_k;
    const int nl = gax < 0 ? 2 : 1;   // lists
    // G = 2^lg lanes per survivor, sized for two lists in either case: the
    // lanes' partial sums (and so the scores' roundings) are then the same
    // whether one CTA takes both axes or a pair one each
    int lg = 0;
    while (lg < 5 && 2 * k * (2 << lg) <= kThreads) ++lg;
    const int G = 1 << lg;
    const int lane = threadIdx.x & 31, sub = lane & (G - 1);
    const int sv = threadIdx.x >> lg;   // 2k G <= kThreads: one pass
    const bool active = sv < nl * k;
    const int ls = active && sv >= k ? 1 : 0;   // the list
    const int s = gax < 0 ? ls : gax;           // its axis
    const int qi = active ? sv - ls * k : 0;
    uint32_t pos = active ? pos_of(sh.win[ls][qi]) : 0u;
    if (active && pos >= (uint32_t)d.K) {   // never expected: record and skip
        if (sub == 0) atomicOr(p.err, kErrInternal);
        pos = 0u;
    }

    const T *row = static_cast<const T *>(s ? p.k_col : p.k_row) + ((int64_t)h * d.K + pos) * D;
    const float *q = L.qv + s * D;
    const bool vec = D % EPV == 0 && dk % EPV == 0 && ((uintptr_t)row & 15) == 0;
    const uint4 *rv = reinterpret_cast<const uint4 *>(row);
    const int nvec = vec ? D / EPV : 0;
    // the first batch of the row's 16-byte loads is issued before the order
    // scan below, which reads shared memory only
    uint4 buf[8];
#pragma unroll
    for (int u = 0; u < 8; ++u) {
        const int iv = sub + u * G;
        buf[u] = active && iv < nvec ? ld_key_row(rv + iv) : make_uint4(0, 0, 0, 0);
    }

    int ord = 0;
    if (active) {
        int g = sub;
        for (; g + 3 * G < k; g += 4 * G) {
            const uint32_t a = pos_of(sh.win[ls][g]), b = pos_of(sh.win[ls][g + G]),
                           c = pos_of(sh.win[ls][g + 2 * G]), e = pos_of(sh.win[ls][g + 3 * G]);
            ord += (a < pos) + (b < pos) + (c < pos) + (e < pos);
        }
        for (; g < k; g += G) ord += pos_of(sh.win[ls][g]) < pos;
    }
    for (int off = G >> 1; off > 0; off >>= 1) ord += __shfl_xor_sync(kFull, ord, off);

    float S[RM];
#pragma unroll
    for (int a = 0; a < RM; ++a) S[a] = 0.f;
    // fp32 storage: each chunk score as a compensated dot product (Dot2),
    // so that the weights carry the working precision (see Dot2)
    constexpr bool kExact = std::is_same<T, float>::value;
    Dot2 SX[kExact ? RM : 1];
    if (vec) {
        // 16-byte group iv of the row belongs to chunk iv / cpv
        const int cpv = dk / EPV;
        // (rank > 2) chunk of element x = floor(x / dk), as floor((x + 1/2) /
        // dk) in fp32: exact while x, dk < 2^20 (the error stays below 1/(2 dk))
        const float inv_dk = 1.f / (float)dk;
#pragma unroll 1
        for (int u0 = sub; u0 < nvec; u0 += 8 * G) {
            if (u0 != sub) {
#pragma unroll
                for (int u = 0; u < 8; ++u) {
                    const int iv = u0 + u * G;
                    buf[u] = active && iv < nvec ? ld_key_row(rv + iv) : make_uint4(0, 0, 0, 0);
                }
            }
#pragma unroll
            for (int u = 0; u < 8; ++u) {
                const int iv = u0 + u * G;
                if (iv < nvec) {
                    float f[EPV];
                    unpack16<T>(buf[u], f);
                    // q + iv*EPV is 16-byte aligned: qv is, and D % EPV == 0
                    const float4 *qq = reinterpret_cast<const float4 *>(q + iv * EPV);
                    if constexpr (kExact) {
                        // the vector lies in one chunk: add its products there
                        const int al = RM == 2 ? (iv >= cpv ? RM - 1 : 0)
                                               : (int)(((float)(iv * EPV) + 0.5f) * inv_dk);
#pragma unroll
                        for (int a = 0; a < RM; ++a) {
                            if (a == al) {
#pragma unroll
                                for (int e4 = 0; e4 < EPV / 4; ++e4) {
                                    const float4 q4 = qq[e4];
                                    SX[a].add(f[4 * e4], q4.x);
                                    SX[a].add(f[4 * e4 + 1], q4.y);
                                    SX[a].add(f[4 * e4 + 2], q4.z);
                                    SX[a].add(f[4 * e4 + 3], q4.w);
                                }
                            }
                        }
                        continue;
                    }
                    float pv = 0.f;
#pragma unroll
                    for (int e4 = 0; e4 < EPV / 4; ++e4) {
                        const float4 q4 = qq[e4];
                        pv = fmaf(f[4 * e4], q4.x, pv);
                        pv = fmaf(f[4 * e4 + 1], q4.y, pv);
                        pv = fmaf(f[4 * e4 + 2], q4.z, pv);
                        pv = fmaf(f[4 * e4 + 3], q4.w, pv);
                    }
                    if (RM == 2) {   // rank 1 or 2: the second chunk starts at cpv
                        const bool hi = iv >= cpv;
                        S[0] += hi ? 0.f : pv;
                        S[RM - 1] += hi ? pv : 0.f;
                    } else {
                        const int al = (int)(((float)(iv * EPV) + 0.5f) * inv_dk);
#pragma unroll
                        for (int a = 0; a < RM; ++a)
                            if (a < r) S[a] += a == al ? pv : 0.f;   // r is uniform
                    }
                }
            }
        }
    } else {
#pragma unroll
        for (int a = 0; a < RM; ++a) {
            if (a < r && active) {
                float acc = 0.f;
                for (int c = a * dk + sub; c < (a + 1) * dk; c += G) {
                    if constexpr (kExact) SX[a].add(to_f(row[c]), q[c]);
                    else acc = fmaf(to_f(row[c]), q[c], acc);
                }
                S[a] = acc;
            }
        }
    }
    if constexpr (kExact) {
        // the group's partial sums merged with their error terms
#pragma unroll
        for (int a = 0; a < RM; ++a) {
            if (a < r) {
                for (int off = G >> 1; off > 0; off >>= 1) {
                    Dot2 o;
                    o.s = __shfl_xor_sync(kFull, SX[a].s, off);
                    o.c = __shfl_xor_sync(kFull, SX[a].c, off);
                    SX[a].merge(o);
                }
                S[a] = SX[a].value();
            }
        }
    } else {
#pragma unroll
        for (int a = 0; a < RM; ++a) {
            if (a < r)
                for (int off = G >> 1; off > 0; off >>= 1) S[a] += __shfl_xor_sync(kFull, S[a], off);
        }
    }
    if (active && sub == 0) {
        if (s == 0) {
            L.sel_i[ord] = (int)pos;
            // MCS (the individual scores) and fp32 storage (the weights in
            // fp64) need S_row itself
            if (d.nc > 1 || kExact)
#pragma unroll
                for (int a = 0; a < RM; ++a)
                    if (a < r) L.srow[ord * r + a] = S[a];
#pragma unroll
            for (int b = 0; b < RM; ++b) {
                if (b < r) {
                    float acc = 0.f;
#pragma unroll
                    for (int a = 0; a < RM; ++a)
                        if (a < r) acc = fmaf(S[a], sh.core[a * r + b], acc);
                    L.R[ord * r + b] = acc;
                }
            }
        } else {
            L.sel_j[ord] = (int)pos;
#pragma unroll
            for (int b = 0; b < RM; ++b)
                if (b < r) L.scol[ord * r + b] = S[b];
        }
    }
}

// MINB: resident CTAs per SM the registers are sized for (3: about 80
// registers, for grids of up to about three CTAs per SM, where a CTA's
// latency matters; 4: 64 registers, for long grids, where occupancy does).
// RM >= r: the rank bound of the survivor phase (2, or 8 for larger ranks),
// one per kernel so that each carries a single copy of it.
// PAIR (decode grids of at most one (token, head) per SM): a cluster of two
// CTAs per (token, head), blockIdx.z = its axis.  Each takes one axis through
// the key load, bound, compaction, rank and survivors (half the work a warp
// does in those phases); the column CTA then sends its survivors (indices
// and S_col) into the row CTA's shared memory with asynchronous stores that
// complete bytes of the row CTA's exchange mbarrier, and the row CTA, once
// that barrier completes, goes on alone (Tucker scores, top-m, outputs).
template <typename T, int MINB, int RM, bool PAIR = false>
__global__ void __launch_bounds__(kThreads, MINB) select_kernel(Dims d, Ptrs p) {
    extern __shared__ __align__(16) unsigned char smem_raw[];
    __shared__ SelShared sh;
    const int b = blockIdx.x / d.H, h = blockIdx.x % d.H;
    const int ax = PAIR ? (int)blockIdx.z : 0;   // the cluster's rank (cluster 1 x 1 x 2)
    const SelLayout L = carve(d, smem_raw);
    const int r = d.r, K = d.K, k = d.k, m = d.m;
    const uint32_t *A0 = p.akey + (((int64_t)b * d.H + h) * 2 + ax) * (int64_t)K;
    const uint32_t *A1 = A0 + K;   // (not read when PAIR)

    if (threadIdx.x < 8) sh.cnt[threadIdx.x] = 0;
    if constexpr (PAIR) {
        // the row CTA's exchange barrier, expecting the column CTA's
        // survivors (k indices and k r scores); the pair's cluster barrier
        // arrival publishes it, its wait comes just before the exchange
        if (ax == 0 && threadIdx.x == 0) xbar_init(&sh.xbar, (uint32_t)(d.k + d.k * d.r) * 4u);
        cl_arrive_relaxed();
    }
    // C of this head (a weight: read before the dependency wait) and the
    // row/column query of this (token, head), summed over its D_i splits:
    // loaded before the keys, stored after them
    const float core_e = threadIdx.x < r * r ? p.core[(int64_t)h * r * r + threadIdx.x] : 0.f;
    // MCS component cores (nc r^2 <= 2 kThreads), stored once key1 is free
    const int ncrr = d.nc > 1 ? d.nc * r * r : 0;
    const float *cp = p.cores + (int64_t)h * ncrr;
    const float cp0 = threadIdx.x < ncrr ? cp[threadIdx.x] : 0.f;
    const float cp1 = threadIdx.x + kThreads < ncrr ? cp[threadIdx.x + kThreads] : 0.f;
    pdl_wait();
    stamp_begin(p.stamp);
    pdl_trigger();
    const int HD = d.H * d.d_k;
    const int64_t split_stride = (int64_t)d.A * d.B * HD;
    auto q_src = [&](int e) {
        const int axis = e / d.d_k, c = e - axis * d.d_k;
        const int a = (axis == 1 && d.A == 2) ? 1 : 0;
        return p.q_part + ((int64_t)a * d.B + b) * HD + h * d.d_k + c;
    };
    // the split-K partials of q, summed in fp64 with fp32 storage (one
    // rounding of the query the weights are computed from)
    auto q_of = [&](int e) {
        const float *src = q_src(e);
        if constexpr (std::is_same<T, float>::value) {
            double q = 0.0;
            for (int s = 0; s < d.q_splits; ++s) q += (double)src[s * split_stride];
            return (float)q;
        } else {
            float q = 0.f;
            for (int s = 0; s < d.q_splits; ++s) q += src[s * split_stride];
            return q;
        }
    };
    const bool one_split = d.q_splits == 1;
    // the query elements this CTA needs: both axes', or its own axis'
    const int e0 = PAIR ? ax * d.d_k : 0, ne = PAIR ? d.d_k : 2 * d.d_k;
    float q0 = 0.f;
    if (threadIdx.x < ne) q0 = one_split ? *q_src(e0 + threadIdx.x) : q_of(e0 + threadIdx.x);
    uint32_t top[2][2];
    const bool stream = d.stream_keys != 0;   // uniform
    // candidate lists: only the long-grid instantiation reads them (the
    // launch picks it whenever they are on)
    const bool lists = MINB >= 4 && d.cand;
    if constexpr (PAIR) load_keys<1>(A0, A1, K, L, top, stream);
    else if (!lists) load_keys(A0, A1, K, L, top, stream);
    // the axes' keys: in shared memory, or (streamed) in L2, where the
    // compaction reads them a second time
    const uint32_t *KA = stream ? A0 : L.key0, *KB = stream ? A1 : L.key1;
    if (threadIdx.x < r * r) sh.core[threadIdx.x] = core_e;
    if (threadIdx.x < ne) L.qv[e0 + threadIdx.x] = q0;
    for (int e = threadIdx.x + kThreads; e < ne; e += kThreads) L.qv[e0 + e] = q_of(e0 + e);

    // Eq. 8-9: top-k of both axes
    if constexpr (PAIR) {   // this CTA's axis as list 0
        warp_bounds(top[0][0], top[0][1], 0u, 0u, 1, k, sh);
        __syncthreads();
        compact<1>(KA, nullptr, K, block_bound(0, sh), 0u, sh, kCntAxis, kCntAxis);
        __syncthreads();
    } else if (lists) {   // the scoring left each axis' candidates
        __syncthreads();
        load_lists(p, ((int64_t)b * d.H + h) * 2, d.n_groups, k, sh);
    } else {
        warp_bounds(top[0][0], top[0][1], top[1][0], top[1][1], 2, k, sh);
        __syncthreads();
        compact<2>(KA, KB, K, block_bound(0, sh), block_bound(1, sh), sh, kCntAxis,
                   kCntAxis + 1);
        __syncthreads();
    }
    const int c0 = settle(0, KA, K, k, kCntAxis, kCntAxisT, sh);
    const int c1 = PAIR ? 0 : settle(1, KB, K, k, kCntAxis + 1, kCntAxisT + 1, sh);
    if constexpr (PAIR) {
        rank_list(sh.cand[0], c0, k, sh.win[0], threadIdx.x, kThreads);
    } else {
        const int s = threadIdx.x >= kThreads / 2, cs = s ? c1 : c0;
        const int tid = threadIdx.x & (kThreads / 2 - 1);
        // long grids (issue-bound) rank by sorted runs, which execute fewer
        // instructions; decode grids (latency-bound) by counting, which
        // has the shorter dependency chain
        if (MINB >= 4 && c0 <= kThreads / 2 && c1 <= kThreads / 2) {   // uniform
            if (s)   // warp-uniform: each half of the block has its own barrier
                rank_sorted<2, kThreads / 2>(sh.cand[1], cs, k, sh.win[1], sh.runs + kThreads / 2,
                                             tid);
            else
                rank_sorted<1, kThreads / 2>(sh.cand[0], cs, k, sh.win[0], sh.runs, tid);
        } else
            rank_list(sh.cand[s], cs, k, sh.win[s], tid, kThreads / 2);
    }
    __syncthreads();
    if (threadIdx.x < ncrr) L.cparts[threadIdx.x] = cp0;   // key1 is free now
    if (threadIdx.x + kThreads < ncrr) L.cparts[threadIdx.x + kThreads] = cp1;
    // survivors in increasing index with their exact chunk scores (Eq. 4)
    axis_survivors<T, RM>(d, p, h, L, sh, PAIR ? ax : -1);
    __syncthreads();
    if constexpr (PAIR) {
        // the column CTA sends its survivors into the row CTA with
        // asynchronous stores that complete bytes of the row CTA's exchange
        // mbarrier, and is done; the row CTA waits on that barrier
        cl_wait();   // the exchange barrier is initialised
        if (ax == 1) {
            for (int i = threadIdx.x; i < k; i += kThreads)
                st_async_u32(L.sel_j + i, 0u, (uint32_t)L.sel_j[i], &sh.xbar);
            for (int i = threadIdx.x; i < k * r; i += kThreads)
                st_async_u32(L.scol + i, 0u, __float_as_uint(L.scol[i]), &sh.xbar);
            stamp_end(p.stamp);
            return;
        }
        if (!xbar_wait(&sh.xbar) && threadIdx.x == 0) atomicOr(p.err, kErrTimeout);
    }

    u64 *const fwin = sh.cand[1];   // final winners by rank (list 1 is free now)

    // Eq. 10: g(i,j) = sum_b R[i][b] S_col[b,j] on I x J, R = S_row^T C.
    // Which thread computes which pair decides how tight the bound below is:
    // it is the smallest of the 8 warps' values, so every warp should hold a
    // spread sample of rows and columns.  In index order (pair c to thread
    // c mod 256) a warp holds a few rows and half of the columns, and about
    // twice as many candidates pass (final list at decode_1m, median over
    // CTAs: 126 of 1024 for m = 32; 49 with a spread assignment).
    const int k2 = k * k;
    uint32_t g1 = 0u, g2 = 0u;
    if (!d.pkm && r == 2 && (k & 31) == 0) {   // uniform
        // lane l of warp w owns columns l + 32 h (h < k/32; S_col in
        // registers) and, of each, the rows ((w + l) mod 8) + 8 i (i < k/8):
        // a warp holds every row and every column (8 warps, kThreads = 256)
        const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
        const int i0 = (w + lane) & 7;
        for (int jj = lane; jj < k; jj += 32) {
            const float2 b2 = *reinterpret_cast<const float2 *>(L.scol + jj * 2);
            for (int ii = i0; ii < k; ii += 8) {
                const float2 a2 = *reinterpret_cast<const float2 *>(L.R + ii * 2);
                const uint32_t kg = f2ord(fmaf(a2.y, b2.y, a2.x * b2.x));
                L.key0[ii * k + jj] = kg;
                top2(kg, g1, g2);
            }
        }
    } else {
        // any shape: thread t visits the pairs p = t, t + kThreads, ... as
        // pair index pp = p kPairMix mod k^2 (a bijection: kPairMix is a
        // prime above kMaxK)
        const uint32_t uk2 = (uint32_t)k2;
        const uint32_t step = (uint32_t)(((uint64_t)kThreads * kPairMix) % uk2);
        uint32_t pp = (uint32_t)(((uint64_t)threadIdx.x * kPairMix) % uk2);
        // ii = pp / k as floor((pp + 1/2) / k) in fp32: pp < 2^14 and k <= 128,
        // so the rounding error (< 2^-16) stays below the 1/(2k) margin
        const float inv_k = 1.f / (float)k;
        for (int c = threadIdx.x; c < k2; c += kThreads) {
            const int ii = (int)(((float)pp + 0.5f) * inv_k);
            const int jj = (int)pp - ii * k;
            float g;
            if (d.pkm) {    // product keys (Eq. 2): s_row[i] + s_col[j]
                g = L.R[ii] + L.scol[jj];
            } else if (r == 2) {   // the common rank, without the loop
                const float2 a2 = *reinterpret_cast<const float2 *>(L.R + ii * 2);
                const float2 b2 = *reinterpret_cast<const float2 *>(L.scol + jj * 2);
                g = fmaf(a2.y, b2.y, a2.x * b2.x);
            } else {
                g = 0.f;
                for (int be = 0; be < r; ++be) g = fmaf(L.R[ii * r + be], L.scol[jj * r + be], g);
            }
            const uint32_t kg = f2ord(g);
            L.key0[pp] = kg;
            top2(kg, g1, g2);
            pp += step;
            if (pp >= uk2) pp -= uk2;
        }
    }
    warp_bounds(g1, g2, 0u, 0u, 1, m, sh);
    __syncthreads();
    compact<1>(L.key0, nullptr, k2, block_bound(0, sh), 0u, sh, kCntTop, kCntTop);
    __syncthreads();
    const int cf = settle(0, L.key0, k2, m, kCntTop, kCntTopT, sh);
    if (MINB >= 4 && cf <= kThreads)
        rank_sorted<3, kThreads>(sh.cand[0], cf, m, fwin, sh.runs, threadIdx.x);
    else rank_list(sh.cand[0], cf, m, fwin, threadIdx.x, kThreads);
    __syncthreads();

    // fp32 storage: the weights are the winners' scores recomputed in fp64
    // from the exact chunk scores (S_row, S_col) and the core, rounded once;
    // the fp32 scores above only decided the order
    constexpr bool kExact = std::is_same<T, float>::value;
    auto exact_g = [&](int ii, int jj, const float *Cm) -> double {
        if (d.pkm) return (double)L.srow[ii] + (double)L.scol[jj];   // Eq. 2: r = 1
        double g = 0.0;
        for (int a = 0; a < r; ++a) {
            double cs = 0.0;
            for (int be = 0; be < r; ++be)
                cs += (double)Cm[a * r + be] * (double)L.scol[jj * r + be];
            g += (double)L.srow[ii * r + a] * cs;
        }
        return g;
    };
    auto pair_of = [&](u64 wc, int &ii, int &jj) {
        int c = (int)pos_of(wc);
        if ((uint32_t)c >= (uint32_t)k2) c = 0;   // recorded below
        ii = c / k;
        jj = c - ii * k;
    };
    double gmax_d = 0.0;
    if constexpr (kExact) {
        int i0, j0;
        pair_of(fwin[0], i0, j0);
        gmax_d = exact_g(i0, j0, sh.core);
        if (d.act == ULTRAMEM_ACT_SOFTMAX) {
            if (threadIdx.x < 32) {
                double z = 0.0;
                for (int e = threadIdx.x; e < m; e += 32) {
                    int ii, jj;
                    pair_of(fwin[e], ii, jj);
                    z += exp(exact_g(ii, jj, sh.core) - gmax_d);
                }
#pragma unroll
                for (int off = 16; off > 0; off >>= 1) z += __shfl_xor_sync(kFull, z, off);
                if (threadIdx.x == 0) sh.dscalar = z;
            }
            __syncthreads();
        }
    }

    // PKM's softmax over the m selected scores (Eq. 3); Trick 1 skips it
    const float gmax = ord2f(key_of(fwin[0]));
    if (!kExact && d.act == ULTRAMEM_ACT_SOFTMAX) {
        if (threadIdx.x < 32) {
            float z = 0.f;
            for (int e = threadIdx.x; e < m; e += 32) z += __expf(ord2f(key_of(fwin[e])) - gmax);
#pragma unroll
            for (int off = 16; off > 0; off >>= 1) z += __shfl_xor_sync(kFull, z, off);
            if (threadIdx.x == 0) sh.scalar = z;
        }
        __syncthreads();
    }
    const int64_t base = ((int64_t)b * d.H + h) * m;
    const uint32_t N = (uint32_t)d.N;
    const uint32_t row_bytes = (uint32_t)d.d_v * (d.dtype == ULTRAMEM_BF16 ? 2u : 4u);
    const bool prefetch = (uint64_t)d.B * d.H * m * row_bytes <= kPrefetchMaxBytes;
    for (int e = threadIdx.x; e < m; e += kThreads) {
        const u64 wc = fwin[e];
        int c = (int)pos_of(wc);
        if ((uint32_t)c >= (uint32_t)k2) {   // never expected: record and skip
            atomicOr(p.err, kErrInternal);
            c = 0;
        }
        const int ii = c / k, jj = c - ii * k;
        const uint64_t v = (uint64_t)L.sel_i[ii] * (uint64_t)K + (uint64_t)L.sel_j[jj];
        const float g = ord2f(key_of(wc));
        float w;
        if constexpr (kExact) {
            const double gd = exact_g(ii, jj, sh.core);
            w = (float)(d.act == ULTRAMEM_ACT_SOFTMAX ? exp(gd - gmax_d) / sh.dscalar : gd);
        } else {
            w = d.act == ULTRAMEM_ACT_SOFTMAX ? __expf(g - gmax) / sh.scalar : g;
        }
        const uint32_t vs = (uint32_t)shuffle_address(d, p.perm, v);   // Eq. 14, < M < 2^32
        const uint32_t pb = vs / N;
        const uint32_t prow = vs - pb * N;
        p.sel_row[base + e] = (int32_t)prow;
        p.sel_p[base + e] = (int32_t)pb;
        if (p.idx_out) p.idx_out[base + e] = (int64_t)v;
        if (d.nc == 1) {
            p.sel_w[base + e] = w;
            if (p.w_out) p.w_out[base + e] = w;
        } else {
            // MCS (Eq. 16-17): the individual scores S_row^T C^(i) S_col of
            // this slot, one per value slice (the softmax is not allowed here)
            float sr[RM], sc[RM];
#pragma unroll
            for (int a = 0; a < RM; ++a) {
                sr[a] = a < r ? L.srow[ii * r + a] : 0.f;
                sc[a] = a < r ? L.scol[jj * r + a] : 0.f;
            }
            for (int ci = 0; ci < d.nc; ++ci) {
                const float *Cc = L.cparts + ci * r * r;
                if constexpr (kExact) {   // fp32 storage: in fp64, rounded once
                    const float gx = (float)exact_g(ii, jj, Cc);
                    p.sel_w[(base + e) * d.nc + ci] = gx;
                    if (p.w_out) p.w_out[(base + e) * d.nc + ci] = gx;
                    continue;
                }
                float gi = 0.f;
#pragma unroll
                for (int a = 0; a < RM; ++a) {
                    if (a < r) {
                        float cs = 0.f;
#pragma unroll
                        for (int be = 0; be < RM; ++be)
                            if (be < r) cs = fmaf(Cc[a * r + be], sc[be], cs);
                        gi = fmaf(sr[a], cs, gi);
                    }
                }
                p.sel_w[(base + e) * d.nc + ci] = gi;
                if (p.w_out) p.w_out[(base + e) * d.nc + ci] = gi;
            }
        }
    }
    // The gather will read the winners' value rows: start moving them into
    // L2 (unless the batch's rows would not stay there until then).  Winner
    // e's row is fetched by a thread of the warps after those that stored
    // the slots (for m <= 128), which works out the slot again: a prefetch
    // holds its warp for about 1300 cycles (the row's address translation,
    // measured at decode), and this way the stores above do not wait behind
    // it.
    if (prefetch) {
        const int sw = (m + 31) / 32;   // warps that stored slots
        const int shift = 2 * sw * 32 <= kThreads ? 32 * sw : 32;
        for (int e = (threadIdx.x + kThreads - shift) % kThreads; e < m; e += kThreads) {
            int c = (int)pos_of(fwin[e]);
            if ((uint32_t)c >= (uint32_t)k2) c = 0;   // recorded above
            const int ii = c / k, jj = c - ii * k;
            const uint64_t v = (uint64_t)L.sel_i[ii] * (uint64_t)K + (uint64_t)L.sel_j[jj];
            const uint32_t vs = (uint32_t)shuffle_address(d, p.perm, v);
            const uint32_t prow = vs - (vs / N) * N;
            prefetch_l2(static_cast<const unsigned char *>(p.values) + (size_t)prow * row_bytes,
                        row_bytes);
        }
    }
    stamp_end(p.stamp);
}

// Candidate lists (Dims::cand), between the two scoring passes: the bound of
// one (token, head, axis) per warp.  tau is the largest T whose low 16 bits
// are zero with at least k of the axis' G group maxima (groups of 16 keys)
// >= T, found bit by bit from the top: k distinct groups hold a key >= tau,
// so the axis' top k is among the keys >= tau.  tau is at most the k-th
// largest group maximum and agrees with it in the sign, the exponent and
// the first 7 mantissa bits of the score; the low bits would tighten the
// lists by a few keys for twice the rounds.
constexpr int kBoundWarps = 8;
constexpr int kMaxGroupsPerLane = 32;   // G <= 1024 groups (K <= 16384 keys)
static_assert(32 * kMaxGroupsPerLane == kMaxSegPerThread * kThreads, "one limit on G");
template <int NQ>   // group maxima a lane holds, 32 NQ >= G
__global__ void __launch_bounds__(32 * kBoundWarps) cand_bound_kernel(Dims d, Ptrs p) {
    pdl_wait();
    stamp_begin(p.stamp);
    pdl_trigger();
    const int lane = threadIdx.x & 31;
    const int64_t w = (int64_t)blockIdx.x * kBoundWarps + (threadIdx.x >> 5);
    if (w < (int64_t)d.B * d.H * 2) {   // warp-uniform
        const int G = d.n_groups;
        const uint32_t *g = p.gstat + w * G;
        uint32_t v[NQ];
#pragma unroll
        for (int q = 0; q < NQ; ++q) {
            const int e = lane + 32 * q;
            v[q] = e < G ? g[e] : 0u;   // 0: below every score's key
        }
        uint32_t T = 0u;
#pragma unroll 4
        for (int bit = 31; bit >= 16; --bit) {
            const uint32_t c = T | (1u << bit);
            int n = 0;
#pragma unroll
            for (int q = 0; q < NQ; ++q) n += v[q] >= c;
            if (__reduce_add_sync(kFull, n) >= d.k) T = c;
        }
        if (lane == 0) p.tau[w] = T;
    }
    stamp_end(p.stamp);
}

// lookup_reduce input: given virtual addresses and weights -> (row, p, w).
// An address outside [0, E*N) is recorded in the error word and skipped
// (weights 0, row 0).  With MCS each slot has nc weights.
__global__ void slots_kernel(Dims d, Ptrs p) {
    const int64_t total = (int64_t)d.B * d.H * d.m;
    for (int64_t e = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; e < total;
         e += (int64_t)gridDim.x * blockDim.x) {
        int64_t v = p.idx_in[e];
        const bool bad = v < 0 || (uint64_t)v >= d.M;
        if (bad) {
            atomicOr(p.err, kErrBadIndex);
            v = 0;
        }
        for (int ci = 0; ci < d.nc; ++ci)
            p.sel_w[e * d.nc + ci] = bad ? 0.f : p.w_in[e * d.nc + ci];
        uint64_t vs = shuffle_address(d, p.perm, (uint64_t)v);
        uint64_t pb = vs / (uint64_t)d.N;
        p.sel_row[e] = (int32_t)(vs - pb * (uint64_t)d.N);
        p.sel_p[e] = (int32_t)pb;
    }
}

}  // namespace

size_t select_smem_bytes(const Dims &d) { return sel_offsets(d).total; }

template <typename T, int RM>
static cudaError_t launch_select_t(const Dims &d, const Ptrs &p, size_t smem, cudaStream_t st) {
    if (d.B * d.H > 3 * 152 || d.cand)
        return launch_kernel(d.pdl, select_kernel<T, 4, RM>, d.B * d.H, kThreads, smem, st, d, p);
    if (d.B * d.H <= device_sm_count()) {
        // at most one (token, head) per SM: a CTA pair per (token, head), the
        // pairs spread over the SMs
        const size_t sm =
            spread_smem(smem, static_smem_of<select_kernel<T, 3, RM, true>>(), 2 * d.B * d.H);
        return launch_kernel(d.pdl, 2u, select_kernel<T, 3, RM, true>, dim3(d.B * d.H, 1, 2),
                             kThreads, sm, st, d, p);
    }
    // decode grids: spread over the SMs (see spread_smem)
    const size_t sm = spread_smem(smem, static_smem_of<select_kernel<T, 3, RM>>(), d.B * d.H);
    return launch_kernel(d.pdl, select_kernel<T, 3, RM>, d.B * d.H, kThreads, sm, st, d, p);
}

cudaError_t launch_select(const Dims &d, const Ptrs &p, cudaStream_t st) {
    const size_t smem = select_smem_bytes(d);
    if (d.dtype == ULTRAMEM_BF16)
        return d.r <= 2 ? launch_select_t<__nv_bfloat16, 2>(d, p, smem, st)
                        : launch_select_t<__nv_bfloat16, kMaxR>(d, p, smem, st);
    return d.r <= 2 ? launch_select_t<float, 2>(d, p, smem, st)
                    : launch_select_t<float, kMaxR>(d, p, smem, st);
}

cudaError_t launch_cand_bound(const Dims &d, const Ptrs &p, cudaStream_t st) {
    if (d.n_groups < d.k || d.n_groups > 32 * kMaxGroupsPerLane) return cudaErrorInvalidValue;
    const int64_t warps = (int64_t)d.B * d.H * 2;
    const int blocks = (int)((warps + kBoundWarps - 1) / kBoundWarps);
    const int nq = (d.n_groups + 31) / 32;
    auto go = [&](auto kernel) {
        return launch_kernel(d.pdl, kernel, blocks, 32 * kBoundWarps, 0, st, d, p);
    };
    if (nq <= 1) return go(cand_bound_kernel<1>);
    if (nq <= 2) return go(cand_bound_kernel<2>);
    if (nq <= 4) return go(cand_bound_kernel<4>);
    if (nq <= 8) return go(cand_bound_kernel<8>);
    if (nq <= 16) return go(cand_bound_kernel<16>);
    return go(cand_bound_kernel<kMaxGroupsPerLane>);
}

cudaError_t launch_slots_from_addresses(const Dims &d, const Ptrs &p, cudaStream_t st) {
    int64_t total = (int64_t)d.B * d.H * d.m;
    int blocks = (int)((total + 255) / 256);
    if (blocks > 4096) blocks = 4096;
    if (blocks < 1) blocks = 1;
    slots_kernel<<<blocks, 256, 0, st>>>(d, p);
    return cudaGetLastError();
}

// Each selection kernel may use up to the per-CTA maximum of dynamic shared
// memory (the decode-grid one is padded to spread its CTAs; see
// spread_smem).  The limit is a process-wide attribute of the kernel, so it
// is set once to the maximum, never lowered to one layer's need.
template <typename T, int RM> static cudaError_t allow_select() {
    const cudaFuncAttribute a = cudaFuncAttributeMaxDynamicSharedMemorySize;
    cudaError_t e = cudaFuncSetAttribute(
        select_kernel<T, 3, RM>, a, (int)(kSmemPerCta - static_smem_of<select_kernel<T, 3, RM>>()));
    if (e == cudaSuccess)
        e = cudaFuncSetAttribute(
            select_kernel<T, 3, RM, true>, a,
            (int)(kSmemPerCta - static_smem_of<select_kernel<T, 3, RM, true>>()));
    if (e == cudaSuccess)
        e = cudaFuncSetAttribute(select_kernel<T, 4, RM>, a,
                                 (int)(kSmemPerCta - static_smem_of<select_kernel<T, 4, RM>>()));
    return e;
}

cudaError_t configure_select(const Dims &) {
    cudaError_t e = allow_select<float, 2>();
    if (e == cudaSuccess) e = allow_select<float, kMaxR>();
    if (e == cudaSuccess) e = allow_select<__nv_bfloat16, 2>();
    if (e == cudaSuccess) e = allow_select<__nv_bfloat16, kMaxR>();
    return e;
}

}  // namespace um
