// um_query_extras.cu -- the query side of the final UltraMem (Sec. 3.1):
//   Trick 4: a causal depthwise convolution of the input before the query
//            linear,  x~[t][c] = b[c] + sum_j w[j][c] x[t - j][c], the taps
//            reaching back into the conv state before each sequence;
//   Trick 2: LayerNorm of each head's query over its D_k entries, after the
//            projection and before the key scores (and a LayerNorm of stored
//            key rows, which at inference folds into the key table).
//
// The convolution is elementwise over (token, channel) and HBM-light (at a
// decode batch it reads a few KB), so it is one short kernel that also
// writes the state after the call.  Its output feeds the query contraction
// exactly: on the tensor path as three bf16 terms x~ = t1 + t2 + t3 (each
// the rounding of what the previous ones leave, residual <= 2^-24 |x~|),
// which the contraction reads as three B operands into one accumulator; on
// the CUDA-core path as fp32.  The LayerNorm is one warp per (query, token,
// head): two passes over the head's D_k values for the mean and the
// variance, a third writes the normalised query back in place and, on the
// tensor path, its scaled three-term splits for the key scores.
#include "um_internal.cuh"

namespace um {
namespace {

constexpr int kThreads = 256;
constexpr unsigned kFull = 0xffffffffu;

// Input c of the token j positions before token b: from its own sequence,
// else from the state before the sequence (zero without one).
template <typename T>
__device__ __forceinline__ T input_back(const Dims &d, const Ptrs &p, int b, int j, int c) {
    const int s = b / d.seq_len, pos = b - s * d.seq_len - j;
    if (pos >= 0) return static_cast<const T *>(p.x)[(int64_t)(b - j) * d.d_in + c];
    if (!p.state_in) return from_f<T>(0.f);
    const int kk = d.conv_k - 1;
    return static_cast<const T *>(p.state_in)[((int64_t)s * kk + kk + pos) * d.d_in + c];
}

// grid (B + sequences * (conv_k - 1), ceil(D_i / kThreads)): rows below B
// are tokens, the rest are rows of the state after the call.
template <typename T>
__global__ void __launch_bounds__(kThreads) conv_kernel(Dims d, Ptrs p, int splits) {
    pdl_wait();
    stamp_begin(p.stamp);
    pdl_trigger();
    const int c = blockIdx.y * kThreads + threadIdx.x;
    if (c >= d.d_in) return;
    const int row = blockIdx.x;
    if (row < d.B) {
        // fp32 storage: the taps summed in fp64, one rounding of x~
        using A = typename std::conditional<std::is_same<T, float>::value, double, float>::type;
        A acc = p.conv_b ? (A)p.conv_b[c] : (A)0;
        for (int j = 0; j < d.conv_k; ++j)
            acc += (A)p.conv_w[(int64_t)j * d.d_in + c] * (A)to_f(input_back<T>(d, p, row, j, c));
        if (splits) {
            __nv_bfloat16 *dst = static_cast<__nv_bfloat16 *>(p.xs) + (int64_t)row * 3 * d.d_in + c;
            const __nv_bfloat16 t1 = __float2bfloat16_rn((float)acc);
            const float r1 = (float)acc - __bfloat162float(t1);
            const __nv_bfloat16 t2 = __float2bfloat16_rn(r1);
            const float r2 = r1 - __bfloat162float(t2);
            dst[0] = t1;
            dst[d.d_in] = t2;
            dst[2 * d.d_in] = __float2bfloat16_rn(r2);
        } else {
            static_cast<float *>(p.xs)[(int64_t)row * d.d_in + c] = (float)acc;
        }
    } else {
        // state row i of sequence s: input seq_len - kk + i of it (a copy)
        const int kk = d.conv_k - 1, e = row - d.B, s = e / kk, i = e - s * kk;
        static_cast<T *>(p.state_out)[((int64_t)s * kk + i) * d.d_in + c] =
            input_back<T>(d, p, s * d.seq_len + d.seq_len - 1, kk - 1 - i, c);
    }
    stamp_end(p.stamp);
}

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) v += __shfl_xor_sync(kFull, v, off);
    return v;
}

constexpr int kLnMax = 8;   // values per lane: D_k <= 256 with the LayerNorm

// One warp per (query a, token b, head h); lane l owns entries l + 32 i.
// The gain, bias and rank-1 coefficients (weights) are loaded before the
// dependency wait, and the next kernel is released only after it: released
// at the start, the key-score kernel measured 2.4x slower at decode.
__global__ void __launch_bounds__(kThreads) query_ln_kernel(Dims d, Ptrs p, __nv_bfloat16 *qs,
                                                            int Bmax) {
    const int lane = threadIdx.x & 31;
    const int64_t id = (int64_t)blockIdx.x * (kThreads / 32) + (threadIdx.x >> 5);
    const bool live = id < (int64_t)d.A * d.B * d.H;
    const int h = live ? (int)(id % d.H) : 0;
    const int b = live ? (int)((id / d.H) % d.B) : 0;
    const int a = live ? (int)(id / ((int64_t)d.H * d.B)) : 0;
    const int HD = d.H * d.d_k;
    const float *g = p.ln_g + (int64_t)a * HD + (int64_t)h * d.d_k;
    const float *bb = p.ln_b ? p.ln_b + (int64_t)a * HD + (int64_t)h * d.d_k : nullptr;
    float gv[kLnMax], bv[kLnMax], uv[kLnMax], tv[kLnMax];
#pragma unroll
    for (int i = 0; i < kLnMax; ++i) {
        const int c = lane + 32 * i;
        const bool in = live && c < d.d_k;
        const int k = h * d.r + (in ? c / d.dk : 0);
        gv[i] = in ? g[c] : 0.f;
        bv[i] = in && bb ? bb[c] : 0.f;
        uv[i] = in && qs ? p.u[k] : 0.f;
        tv[i] = in && qs ? p.t[k] : 0.f;
    }
    pdl_wait();
    stamp_begin(p.stamp);
    pdl_trigger();
    if (!live) return;
    const int64_t split_stride = (int64_t)d.A * d.B * HD;
    float *q = p.q_part + ((int64_t)a * d.B + b) * HD + (int64_t)h * d.d_k;
    if (d.dtype == ULTRAMEM_F32) {
        // fp32 storage (CUDA-core path, no splits to write): the partial
        // sums, mean, variance and normalisation in fp64, one rounding
        double vd[kLnMax];
        double sum = 0.0;
#pragma unroll
        for (int i = 0; i < kLnMax; ++i) {
            const int c = lane + 32 * i;
            vd[i] = 0.0;
            if (c < d.d_k) {
                for (int s = 0; s < d.q_splits; ++s) vd[i] += (double)q[s * split_stride + c];
                sum += vd[i];
            }
        }
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) sum += __shfl_xor_sync(kFull, sum, off);
        const double mean = sum / (double)d.d_k;
        double sq = 0.0;
#pragma unroll
        for (int i = 0; i < kLnMax; ++i) {
            const double e = lane + 32 * i < d.d_k ? vd[i] - mean : 0.0;
            sq += e * e;
        }
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) sq += __shfl_xor_sync(kFull, sq, off);
        const double inv = 1.0 / sqrt(sq / (double)d.d_k + (double)d.ln_eps);
#pragma unroll
        for (int i = 0; i < kLnMax; ++i) {
            const int c = lane + 32 * i;
            if (c >= d.d_k) break;
            q[c] = (float)((vd[i] - mean) * inv * (double)gv[i] + (double)bv[i]);
        }
        stamp_end(p.stamp);
        return;
    }
    float v[kLnMax];
    float sum = 0.f;
#pragma unroll
    for (int i = 0; i < kLnMax; ++i) {
        const int c = lane + 32 * i;
        v[i] = 0.f;
        if (c < d.d_k) {
            for (int s = 0; s < d.q_splits; ++s) v[i] += q[s * split_stride + c];
            sum += v[i];
        }
    }
    const float mean = warp_sum(sum) / (float)d.d_k;
    float sq = 0.f;
#pragma unroll
    for (int i = 0; i < kLnMax; ++i) {
        const float e = lane + 32 * i < d.d_k ? v[i] - mean : 0.f;
        sq = fmaf(e, e, sq);
    }
    const float inv = 1.f / sqrtf(warp_sum(sq) / (float)d.d_k + d.ln_eps);
    const bool row_axis = d.A == 1 || a == 0, col_axis = d.A == 1 || a == 1;
#pragma unroll
    for (int i = 0; i < kLnMax; ++i) {
        const int c = lane + 32 * i;
        if (c >= d.d_k) break;
        const float y = (v[i] - mean) * inv * gv[i] + bv[i];
        q[c] = y;   // split 0 now holds the normalised query
        if (qs) {
            if (row_axis) put_split_query(qs, 0, h, c, b, y * uv[i], d.H, Bmax, d.d_k);
            if (col_axis) put_split_query(qs, 1, h, c, b, y * tv[i], d.H, Bmax, d.d_k);
        }
    }
    stamp_end(p.stamp);
}

// One warp per stored row.
template <typename T>
__global__ void __launch_bounds__(kThreads) key_ln_kernel(const T *keys, int64_t n_rows, int dd,
                                                          const float *g, const float *bb,
                                                          float eps, T *out) {
    const int lane = threadIdx.x & 31;
    const int64_t row = (int64_t)blockIdx.x * (kThreads / 32) + (threadIdx.x >> 5);
    if (row >= n_rows) return;
    const T *x = keys + row * dd;
    float sum = 0.f;
    for (int c = lane; c < dd; c += 32) sum += to_f(x[c]);
    const float mean = warp_sum(sum) / (float)dd;
    float sq = 0.f;
    for (int c = lane; c < dd; c += 32) {
        const float e = to_f(x[c]) - mean;
        sq = fmaf(e, e, sq);
    }
    const float inv = 1.f / sqrtf(warp_sum(sq) / (float)dd + eps);
    __syncwarp();   // in place: every lane has read the row before writing
    for (int c = lane; c < dd; c += 32) {
        const float y = (to_f(x[c]) - mean) * inv * g[c] + (bb ? bb[c] : 0.f);
        out[row * dd + c] = from_f<T>(y);
    }
}

}  // namespace

cudaError_t launch_query_conv(const Dims &d, const Ptrs &p, bool splits, cudaStream_t st) {
    const int seqs = d.B / d.seq_len;
    const int state_rows = p.state_out ? seqs * (d.conv_k - 1) : 0;
    dim3 grid(d.B + state_rows, (d.d_in + kThreads - 1) / kThreads);
    if (d.dtype == ULTRAMEM_BF16)
        return launch_kernel(d.pdl, conv_kernel<__nv_bfloat16>, grid, kThreads, 0, st, d, p,
                             splits ? 1 : 0);
    return launch_kernel(d.pdl, conv_kernel<float>, grid, kThreads, 0, st, d, p, splits ? 1 : 0);
}

cudaError_t launch_query_ln(const Dims &d, const Ptrs &p, __nv_bfloat16 *qs, int Bmax,
                            cudaStream_t st) {
    const int64_t warps = (int64_t)d.A * d.B * d.H;
    const int blocks = (int)((warps + kThreads / 32 - 1) / (kThreads / 32));
    return launch_kernel(d.pdl, query_ln_kernel, blocks, kThreads, 0, st, d, p, qs, Bmax);
}

cudaError_t launch_key_ln(const void *keys, int dtype, int64_t n_rows, int dd, const float *g,
                          const float *b, float eps, void *out, cudaStream_t st) {
    const int64_t blocks = (n_rows + kThreads / 32 - 1) / (kThreads / 32);
    if (blocks == 0) return cudaSuccess;
    if (dtype == ULTRAMEM_BF16)
        key_ln_kernel<__nv_bfloat16><<<(unsigned)blocks, kThreads, 0, st>>>(
            static_cast<const __nv_bfloat16 *>(keys), n_rows, dd, g, b, eps,
            static_cast<__nv_bfloat16 *>(out));
    else
        key_ln_kernel<float><<<(unsigned)blocks, kThreads, 0, st>>>(
            static_cast<const float *>(keys), n_rows, dd, g, b, eps, static_cast<float *>(out));
    return cudaGetLastError();
}

}  // namespace um
