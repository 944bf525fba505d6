// um_score.cu -- query projection (S1) and row/column scores (S2-S3, Eq. 4
// and 6) on CUDA cores in fp32, the path of fp32 storage.  The query
// projection is split over D_i so that enough CTAs stream W_q; the partial
// sums are added when the score kernel loads the query (and, in fp64, when
// the selection loads it for the weights).  With fp32 storage each partial
// is a compensated dot product (Dot2); the scores here only decide which
// keys survive, and the selection recomputes the survivors' exactly.
#include "um_internal.cuh"

namespace um {
namespace {

constexpr int kThreads = 256;

// q_part[split][a][b][o] = sum over this split's slice of D_i of x[b][d] W[o][d]
// Tile: 32 tokens x 64 outputs; each thread owns 2 tokens x 4 outputs.  TX:
// the token rows' type (T, or fp32 for the convolved input x~ of Trick 4,
// which the caller then passes as p.x).
template <typename T, typename TX>
__global__ void __launch_bounds__(kThreads) query_kernel(Dims d, Ptrs p) {
    pdl_wait();
    stamp_begin(p.stamp);
    pdl_trigger();
    const int a = blockIdx.z / d.q_splits, split = blockIdx.z % d.q_splits;
    const TX *X = static_cast<const TX *>(p.x);
    const T *W = static_cast<const T *>(a == 0 ? p.w_q : p.w_q_col);
    const int HD = d.H * d.d_k;
    const int o0 = blockIdx.x * 64, b0 = blockIdx.y * 32;
    const int chunk = (d.d_in + d.q_splits - 1) / d.q_splits;
    const int kb = split * chunk, ke = min(d.d_in, kb + chunk);

    __shared__ float xs[32][33];  // [d][token]
    __shared__ float ws[32][65];  // [d][output]
    const int tid = threadIdx.x, tx = tid % 16, ty = tid / 16;
    // fp32 storage: compensated sums (Dot2), each partial to the working precision
    constexpr bool kExact = std::is_same<T, float>::value;
    float acc[2][4] = {};
    Dot2 ex[kExact ? 2 : 1][kExact ? 4 : 1];
    for (int k0 = kb; k0 < ke; k0 += 32) {
        for (int e = tid; e < 32 * 32; e += kThreads) {
            int bb = e / 32, kk = e % 32, b = b0 + bb, k = k0 + kk;
            xs[kk][bb] = (b < d.B && k < ke) ? to_f(X[(int64_t)b * d.d_in + k]) : 0.f;
        }
        for (int e = tid; e < 64 * 32; e += kThreads) {
            int oo = e / 32, kk = e % 32, o = o0 + oo, k = k0 + kk;
            ws[kk][oo] = (o < HD && k < ke) ? to_f(W[(int64_t)o * d.d_in + k]) : 0.f;
        }
        __syncthreads();
#pragma unroll 8
        for (int kk = 0; kk < 32; ++kk) {
            float xv0 = xs[kk][ty * 2], xv1 = xs[kk][ty * 2 + 1];
#pragma unroll
            for (int j = 0; j < 4; ++j) {
                float wv = ws[kk][tx * 4 + j];
                if constexpr (kExact) {
                    ex[0][j].add(xv0, wv);
                    ex[1][j].add(xv1, wv);
                } else {
                    acc[0][j] = fmaf(xv0, wv, acc[0][j]);
                    acc[1][j] = fmaf(xv1, wv, acc[1][j]);
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
            if (b < d.B && o < HD)
                p.q_part[(((int64_t)split * d.A + a) * d.B + b) * HD + o] = v;
        }
    stamp_end(p.stamp);
}

// For each rank chunk alpha, S_alpha[b][i] = sum_{c < dk} key[h][i][alpha*dk + c]
// * q[b][h][alpha*dk + c] (Eq. 4 with the r x K x (D_k/r) reshape); the chunk
// scores are folded into the rank-1 score a = sum_alpha coef[alpha] S_alpha
// (coef = u for row keys, t for column keys, Eq. 6-7) and its
// order-preserving key is stored: akey[b][h][axis][i].
// Tile: 64 keys x 32 tokens; each thread owns 4 keys x 2 tokens.
template <typename T>
__global__ void __launch_bounds__(kThreads) score_kernel(Dims d, Ptrs p) {
    stamp_begin(p.stamp);
    const int h = blockIdx.z >> 1, axis = blockIdx.z & 1;
    const int a = (axis == 1 && d.A == 2) ? 1 : 0;
    const T *keys = static_cast<const T *>(axis == 0 ? p.k_row : p.k_col) +
                    (int64_t)h * d.K * d.d_k;
    const float *coef = (axis == 0 ? p.u : p.t) + (int64_t)h * d.r;
    const int i0 = blockIdx.x * 64, b0 = blockIdx.y * 32;
    const int HD = d.H * d.d_k;

    __shared__ float ks[32][65];  // [c][key]
    __shared__ float qs[32][33];  // [c][token]
    const int tid = threadIdx.x, tx = tid % 16, ty = tid / 16;
    float folded[4][2] = {};
    for (int al = 0; al < d.r; ++al) {
        float acc[4][2] = {};
        for (int c0 = 0; c0 < d.dk; c0 += 32) {
            for (int e = tid; e < 64 * 32; e += kThreads) {
                int kk = e / 32, cc = e % 32, i = i0 + kk, c = c0 + cc;
                ks[cc][kk] = (i < d.K && c < d.dk)
                                 ? to_f(keys[(int64_t)i * d.d_k + al * d.dk + c]) : 0.f;
            }
            for (int e = tid; e < 32 * 32; e += kThreads) {
                int bb = e / 32, cc = e % 32, b = b0 + bb, c = c0 + cc;
                float q = 0.f;
                if (b < d.B && c < d.dk) {
                    int64_t off = (int64_t)b * HD + h * d.d_k + al * d.dk + c;
                    for (int s = 0; s < d.q_splits; ++s)
                        q += p.q_part[((int64_t)s * d.A + a) * d.B * HD + off];
                }
                qs[cc][bb] = q;
            }
            __syncthreads();
#pragma unroll 8
            for (int cc = 0; cc < 32; ++cc) {
                float q0 = qs[cc][ty * 2], q1 = qs[cc][ty * 2 + 1];
#pragma unroll
                for (int j = 0; j < 4; ++j) {
                    float kv = ks[cc][tx * 4 + j];
                    acc[j][0] = fmaf(kv, q0, acc[j][0]);
                    acc[j][1] = fmaf(kv, q1, acc[j][1]);
                }
            }
            __syncthreads();
        }
        const float cf = coef[al];
        for (int j = 0; j < 4; ++j)
            for (int t = 0; t < 2; ++t)
                folded[j][t] = al == 0 ? cf * acc[j][t] : fmaf(cf, acc[j][t], folded[j][t]);
    }
    for (int j = 0; j < 4; ++j)
        for (int t = 0; t < 2; ++t) {
            int i = i0 + tx * 4 + j, b = b0 + ty * 2 + t;
            if (i < d.K && b < d.B)
                p.akey[(((int64_t)b * d.H + h) * 2 + axis) * d.K + i] = f2ord(folded[j][t]);
        }
    stamp_end(p.stamp);
}

}  // namespace

cudaError_t launch_query(const Dims &d, const Ptrs &p, bool x_f32, cudaStream_t st) {
    const int HD = d.H * d.d_k;
    dim3 grid((HD + 63) / 64, (d.B + 31) / 32, d.A * d.q_splits);
    if (d.dtype == ULTRAMEM_BF16)
        return x_f32 ? launch_kernel(d.pdl, query_kernel<__nv_bfloat16, float>, grid, kThreads,
                                     0, st, d, p)
                     : launch_kernel(d.pdl, query_kernel<__nv_bfloat16, __nv_bfloat16>, grid,
                                     kThreads, 0, st, d, p);
    return launch_kernel(d.pdl, query_kernel<float, float>, grid, kThreads, 0, st, d, p);
}

cudaError_t launch_score(const Dims &d, const Ptrs &p, cudaStream_t st) {
    dim3 grid((d.K + 63) / 64, (d.B + 31) / 32, d.H * 2);
    if (d.dtype == ULTRAMEM_BF16)
        score_kernel<__nv_bfloat16><<<grid, kThreads, 0, st>>>(d, p);
    else
        score_kernel<float><<<grid, kThreads, 0, st>>>(d, p);
    return cudaGetLastError();
}

}  // namespace um
