// um_small.cu -- the query projection (S1) for small token batches, on CUDA
// cores.
//
// At decode batches the contraction is a few hundred KB of weights times a
// handful of tokens.  The tensor-core kernel needs 128 weight rows
// per CTA, which leaves too few CTAs to stream the weights unless K is split,
// and the split-K reduction then dominates.  Here a CTA takes 16 weight rows
// x 8 tokens: its operand rows (bf16, K contiguous) arrive by 1-D bulk
// copies (TMA) into shared memory in one round trip, 256 threads compute the
// 128 dot products (2 x 2 outputs per thread over one of 8 interleaved
// K-slices, then a fixed 3-step shuffle sum: deterministic), and the
// epilogue writes the result in place.  No partial sums leave the CTA.
// When the query input is the convolved x~ (Trick 4), its token rows are
// fp32 (staged the same way, 4 bytes a value), so the contraction sees x~
// exactly.
//
//   Y[n][o] = sum_d x[n][d] W_q[o][d]  -> q (fp32), and q scaled by u (row
//   keys) and by t (column keys) as 3-term bf16 splits for the scoring
// (The tile re-reads each weight row once per 8 tokens, so from about 128
// tokens on, and for the larger IVE projector, the tensor-core kernel wins.)
#include <type_traits>

#include "um_internal.cuh"
#include "um_tc.cuh"

namespace um {
namespace {

using namespace tc;

constexpr int kThreads = 256;
constexpr int kRows = 16;        // weight rows per CTA
constexpr int kToks = 8;         // tokens per CTA
constexpr int kSlices = 8;       // interleaved K slices per output block
// K elements staged per round: 96 KB of bf16 rows, or 64 KB with fp32 tokens
template <bool XF> constexpr int chunk_of() { return XF ? 1024 : 2048; }

struct SmallArgs {
    const __nv_bfloat16 *W;      // [O][Kd]
    const void *X;               // [N][Kd] bf16, or fp32 (the convolved input)
    int O, N, Kd;
    int *err;
    // S1 epilogue
    float *q;                    // [A][B][HD] at a * B * HD (split 0 of q_part)
    __nv_bfloat16 *qs;           // [2][H][Bmax][3][D_k], the scaled split queries
    const float *u, *t;          // [H][r] rank-1 coefficients of row / column keys
    int a, A, H, d_k, dk, r, Bmax;
    int write_qs;                // 0: the query LayerNorm writes the splits later
    unsigned long long *stamp;   // profiling stamps of the stage, or null
};

// Per output row o: its head, column and the rank-1 coefficients of its
// chunk (loaded once, before the weights arrive).
struct RowScale {
    int h, c;
    float cu, ct;
};
__device__ __forceinline__ RowScale row_scale(const SmallArgs &g, int o) {
    RowScale rs;
    rs.h = o / g.d_k;
    rs.c = o - rs.h * g.d_k;
    const int k = rs.h * g.r + rs.c / g.dk;
    rs.cu = (g.A == 1 || g.a == 0) ? g.u[k] : 0.f;
    rs.ct = (g.A == 1 || g.a == 1) ? g.t[k] : 0.f;
    return rs;
}

struct QueryEp {
    __device__ static void put(const SmallArgs &g, int o, int n, float v, const RowScale &rs) {
        g.q[(int64_t)n * g.O + o] = v;
        if (!g.write_qs) return;
        // a shared query feeds both axes; a separate column query only axis 1
        if (g.A == 1 || g.a == 0) put_split_query(g.qs, 0, rs.h, rs.c, n, v * rs.cu, g.H, g.Bmax, g.d_k);
        if (g.A == 1 || g.a == 1) put_split_query(g.qs, 1, rs.h, rs.c, n, v * rs.ct, g.H, g.Bmax, g.d_k);
    }
};

__device__ __forceinline__ void bulk_g2s(void *dst, const void *src, uint32_t bytes,
                                         uint64_t *bar) {
    asm volatile(
        "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];"
        ::"r"(smem_u32(dst)), "l"(src), "r"(bytes), "r"(smem_u32(bar))
        : "memory");
}

__device__ __forceinline__ void bf16x8(uint4 v, float (&f)[8]) {
    const uint32_t u[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
    for (int q = 0; q < 4; ++q) {
        f[2 * q] = __uint_as_float(u[q] << 16);
        f[2 * q + 1] = __uint_as_float(u[q] & 0xffff0000u);
    }
}

__device__ __forceinline__ void load8(const __nv_bfloat16 *p, float (&f)[8]) {
    bf16x8(*reinterpret_cast<const uint4 *>(p), f);
}
__device__ __forceinline__ void load8(const float *p, float (&f)[8]) {
    const float4 a = reinterpret_cast<const float4 *>(p)[0], b = reinterpret_cast<const float4 *>(p)[1];
    f[0] = a.x; f[1] = a.y; f[2] = a.z; f[3] = a.w;
    f[4] = b.x; f[5] = b.y; f[6] = b.z; f[7] = b.w;
}

// XF: the token rows are fp32 (the convolved input) instead of bf16
template <class Ep, bool XF>
__global__ void __launch_bounds__(kThreads) small_gemm_kernel(SmallArgs g) {
    using TX = typename std::conditional<XF, float, __nv_bfloat16>::type;
    extern __shared__ __align__(128) unsigned char smem_raw[];
    __shared__ __align__(8) uint64_t bar;
    constexpr int kChunk = chunk_of<XF>();
    const int stride = min(kChunk, g.Kd);                                // elements per staged row
    __nv_bfloat16 *Ws = reinterpret_cast<__nv_bfloat16 *>(smem_raw);   // [kRows][stride]
    TX *Xs = reinterpret_cast<TX *>(Ws + kRows * stride);                // [kToks][stride]
    const TX *X = static_cast<const TX *>(g.X);
    const int o0 = blockIdx.x * kRows, n0 = blockIdx.y * kToks;
    const int nrows = min(kRows, g.O - o0), ntoks = min(kToks, g.N - n0);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int blk = warp * 4 + (lane >> 3), s = lane & 7;
    const int r0 = 2 * (blk & 7), t0 = 2 * (blk >> 3);   // 8 row pairs x 4 token pairs

    if (threadIdx.x == 0) {
        mbar_init(&bar, 1);
        fence_mbar_init();
    }
    RowScale rs[2];
#pragma unroll
    for (int i = 0; i < 2; ++i) rs[i] = row_scale(g, min(o0 + r0 + i, g.O - 1));
    __syncthreads();
    float acc[2][2] = {};
    uint32_t phase = 0;
    bool ok = true;
    for (int k0 = 0; k0 < g.Kd; k0 += kChunk) {
        const int kc = min(kChunk, g.Kd - k0);
        const uint32_t row_bytes = (uint32_t)kc * 2, x_bytes = (uint32_t)(kc * sizeof(TX));
        if (threadIdx.x == 0) {
            // weights first (no dependency), the tokens after the wait
            mbar_arrive_expect_tx(&bar, row_bytes * (uint32_t)nrows + x_bytes * (uint32_t)ntoks);
            for (int r = 0; r < nrows; ++r)
                bulk_g2s(Ws + r * stride, g.W + (int64_t)(o0 + r) * g.Kd + k0, row_bytes, &bar);
        }
        if (k0 == 0) {
            pdl_wait();
            stamp_begin(g.stamp);
            // the scoring kernel's CTAs may now start streaming its keys
            pdl_trigger();
        }
        if (threadIdx.x == 0)
            for (int t = 0; t < ntoks; ++t)
                bulk_g2s(Xs + t * stride, X + (int64_t)(n0 + t) * g.Kd + k0, x_bytes, &bar);
        const bool timed_out = !mbar_wait(&bar, phase);
        if (__syncthreads_or(timed_out)) {   // block-uniform
            // give the copies in flight one more bounded wait before the
            // shared memory is released, then stop
            if (threadIdx.x == 0) atomicOr(g.err, kErrTimeout);
            mbar_wait(&bar, phase);
            ok = false;
            break;
        }
        phase ^= 1;
        {
            // rows/tokens past the edge read whatever the buffer holds; their
            // results are never written
            const __nv_bfloat16 *w0 = Ws + r0 * stride, *w1 = w0 + stride;
            const TX *x0 = Xs + t0 * stride, *x1 = x0 + stride;
#pragma unroll 4
            for (int kk = s * 8; kk < kc; kk += kSlices * 8) {
                float a0[8], a1[8], b0[8], b1[8];
                load8(w0 + kk, a0);
                load8(w1 + kk, a1);
                load8(x0 + kk, b0);
                load8(x1 + kk, b1);
#pragma unroll
                for (int e = 0; e < 8; ++e) {
                    acc[0][0] = fmaf(a0[e], b0[e], acc[0][0]);
                    acc[0][1] = fmaf(a0[e], b1[e], acc[0][1]);
                    acc[1][0] = fmaf(a1[e], b0[e], acc[1][0]);
                    acc[1][1] = fmaf(a1[e], b1[e], acc[1][1]);
                }
            }
        }
        __syncthreads();   // the buffers are refilled by the next round
    }
#pragma unroll
    for (int i = 0; i < 2; ++i)
#pragma unroll
        for (int j = 0; j < 2; ++j)
#pragma unroll
            for (int off = 1; off < kSlices; off <<= 1)
                acc[i][j] += __shfl_xor_sync(0xffffffffu, acc[i][j], off);
    if (s == 0 && ok) {
#pragma unroll
        for (int i = 0; i < 2; ++i)
#pragma unroll
            for (int j = 0; j < 2; ++j)
                if (r0 + i < nrows && t0 + j < ntoks)
                    Ep::put(g, o0 + r0 + i, n0 + t0 + j, acc[i][j], rs[i]);
    }
    stamp_end(g.stamp);
}

template <bool XF> constexpr size_t smem_row_bytes() {   // W row + token row, one element
    return (size_t)kRows * 2 + (size_t)kToks * (XF ? 4 : 2);
}
template <class Ep, bool XF>
cudaError_t launch_small(const SmallArgs &g, bool pdl, cudaStream_t st) {
    dim3 grid((g.O + kRows - 1) / kRows, (g.N + kToks - 1) / kToks);
    constexpr int kChunk = chunk_of<XF>();
    const size_t smem = smem_row_bytes<XF>() * (g.Kd < kChunk ? g.Kd : kChunk);
    constexpr auto k = small_gemm_kernel<Ep, XF>;
    // spread over the SMs when launched as a dependent (see spread_smem)
    const size_t sm = pdl ? spread_smem(smem, static_smem_of<k>(), (int64_t)grid.x * grid.y) : smem;
    return launch_kernel(pdl, k, grid, kThreads, sm, st, g);
}

}  // namespace

cudaError_t configure_small() {
    // up to a whole SM's share: launches may be padded (spread_smem)
    cudaError_t e = cudaFuncSetAttribute(
        small_gemm_kernel<QueryEp, false>, cudaFuncAttributeMaxDynamicSharedMemorySize,
        (int)(kSmemPerCta - static_smem_of<small_gemm_kernel<QueryEp, false>>()));
    if (e == cudaSuccess)
        e = cudaFuncSetAttribute(
            small_gemm_kernel<QueryEp, true>, cudaFuncAttributeMaxDynamicSharedMemorySize,
            (int)(kSmemPerCta - static_smem_of<small_gemm_kernel<QueryEp, true>>()));
    return e;
}

cudaError_t launch_query_small(const Dims &d, const Ptrs &p, __nv_bfloat16 *qs, int Bmax,
                               bool x_f32, bool write_qs, bool pdl, cudaStream_t st) {
    const int HD = d.H * d.d_k;
    for (int a = 0; a < d.A; ++a) {
        SmallArgs g = {};
        g.W = static_cast<const __nv_bfloat16 *>(a == 0 ? p.w_q : p.w_q_col);
        g.X = x_f32 ? p.xs : p.x;
        g.O = HD;
        g.N = d.B;
        g.Kd = d.d_in;
        g.err = p.err;
        g.q = p.q_part + (int64_t)a * d.B * HD;
        g.qs = qs;
        g.u = p.u;
        g.t = p.t;
        g.a = a;
        g.A = d.A;
        g.H = d.H;
        g.d_k = d.d_k;
        g.dk = d.dk;
        g.r = d.r;
        g.Bmax = Bmax;
        g.write_qs = write_qs ? 1 : 0;
        g.stamp = p.stamp;
        // the first query waits for all earlier work on the stream, unless it
        // follows this call's convolution
        cudaError_t e = x_f32 ? launch_small<QueryEp, true>(g, pdl && a == 0, st)
                              : launch_small<QueryEp, false>(g, pdl && a == 0, st);
        if (e != cudaSuccess) return e;
    }
    return cudaSuccess;
}

}  // namespace um
