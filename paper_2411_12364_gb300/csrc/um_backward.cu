// um_backward.cu -- the backward of the lookup-reduce (Eq. 14-15; App. D's
// fused lookup-reduce operator), for training the value table, the slot
// weights and the IVE projectors.  With dL/do = g:
//   dacc_p = W_p g                                         (dacc_kernel)
//   dV[row_e] += w_e (.) dacc_{p_e},  dw_e = dacc_{p_e} . V[row_e]  per slice
//                                                          (rows_kernel)
//   dW_p = sum_tokens acc_p g^T                            (dwp_kernel)
// The forward's pooled rows acc_p, needed for dW_p, are recomputed by the
// forward gather (one more read of the selected rows).  dV is accumulated
// with fp32 vector atomics (rows repeat across tokens and heads; their
// summation order is not fixed), and so is dacc over its split-K slices.
// dacc and dW_p are CUDA-core tiled contractions; with fp32 storage they
// are compensated dot products (Dot2) and dacc is unsplit, so that the
// fp32 mode's gradients carry the working precision.
#include "um_internal.cuh"

namespace um {
namespace {

constexpr int kThreads = 256;
constexpr int kWarps = kThreads / 32;
constexpr unsigned kFull = 0xffffffffu;

// dacc[b][c] = sum_o W[c][o] g[b][o], W = the projectors [E D_v][D'_v].
// Tile: 32 tokens x 64 rows c; each thread 2 tokens x 4 rows; blockIdx.z
// takes one of gridDim.z slices of o and adds its partial sums into dacc
// (zeroed before), so that small batches still fill the SMs.
template <typename T>
__global__ void __launch_bounds__(kThreads) dacc_kernel(Dims d, const T *g, const T *W,
                                                        float *dacc) {
    const int Mc = d.E * d.d_v, Kfull = d.d_out;
    const int per = (((Kfull + gridDim.z - 1) / gridDim.z) + 31) & ~31;
    const int kb = blockIdx.z * per, Kd = min(Kfull, kb + per);
    const int c0 = blockIdx.x * 64, b0 = blockIdx.y * 32;
    __shared__ float gs[32][33];   // [o][token]
    __shared__ float wsm[32][65];  // [o][row c]
    const int tid = threadIdx.x, tx = tid % 16, ty = tid / 16;
    // fp32 storage: compensated sums (Dot2) over the whole of D'_v (one slice)
    constexpr bool kExact = std::is_same<T, float>::value;
    float acc[2][4] = {};
    Dot2 ex[kExact ? 2 : 1][kExact ? 4 : 1];
    for (int k0 = kb; k0 < Kd; k0 += 32) {
        for (int e = tid; e < 32 * 32; e += kThreads) {
            const int bb = e / 32, kk = e % 32, b = b0 + bb, k = k0 + kk;
            gs[kk][bb] = (b < d.B && k < Kd) ? to_f(g[(int64_t)b * Kfull + k]) : 0.f;
        }
        for (int e = tid; e < 64 * 32; e += kThreads) {
            const int cc = e / 32, kk = e % 32, c = c0 + cc, k = k0 + kk;
            wsm[kk][cc] = (c < Mc && k < Kd) ? to_f(W[(int64_t)c * Kfull + k]) : 0.f;
        }
        __syncthreads();
#pragma unroll 8
        for (int kk = 0; kk < 32; ++kk) {
            const float g0 = gs[kk][ty * 2], g1 = gs[kk][ty * 2 + 1];
#pragma unroll
            for (int j = 0; j < 4; ++j) {
                const float wv = wsm[kk][tx * 4 + j];
                if constexpr (kExact) {
                    ex[0][j].add(g0, wv);
                    ex[1][j].add(g1, wv);
                } else {
                    acc[0][j] = fmaf(g0, wv, acc[0][j]);
                    acc[1][j] = fmaf(g1, wv, acc[1][j]);
                }
            }
        }
        __syncthreads();
    }
    for (int i = 0; i < 2; ++i)
        for (int j = 0; j < 4; ++j) {
            const int b = b0 + ty * 2 + i, c = c0 + tx * 4 + j;
            if (b >= d.B || c >= Mc) continue;
            if constexpr (kExact) dacc[(int64_t)b * Mc + c] = ex[i][j].value();   // one slice
            else atomicAdd(&dacc[(int64_t)b * Mc + c], acc[i][j]);
        }
}

// dW[c][o] = sum_b acc[b][c] g[b][o].  Tile: 64 rows c x 64 outputs o, 4 x 4
// a thread, K over the tokens in steps of 32.
template <typename T>
__global__ void __launch_bounds__(kThreads) dwp_kernel(Dims d, const float *acc, const T *g,
                                                       float *dW) {
    const int Mc = d.E * d.d_v, No = d.d_out;
    const int c0 = blockIdx.x * 64, o0 = blockIdx.y * 64;
    __shared__ float as[32][65];   // [token][c]
    __shared__ float gsm[32][65];  // [token][o]
    const int tid = threadIdx.x, tx = tid % 16, ty = tid / 16;
    constexpr bool kExact = std::is_same<T, float>::value;   // fp32 storage: Dot2
    float r[4][4] = {};
    Dot2 ex[kExact ? 4 : 1][kExact ? 4 : 1];
    for (int b0 = 0; b0 < d.B; b0 += 32) {
        for (int e = tid; e < 32 * 64; e += kThreads) {
            const int bb = e / 64, cc = e % 64, b = b0 + bb;
            as[bb][cc] = (b < d.B && c0 + cc < Mc) ? acc[(int64_t)b * Mc + c0 + cc] : 0.f;
            gsm[bb][cc] = (b < d.B && o0 + cc < No) ? to_f(g[(int64_t)b * No + o0 + cc]) : 0.f;
        }
        __syncthreads();
#pragma unroll 4
        for (int bb = 0; bb < 32; ++bb) {
            float a[4], q[4];
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                a[i] = as[bb][ty * 4 + i];
                q[i] = gsm[bb][tx * 4 + i];
            }
#pragma unroll
            for (int i = 0; i < 4; ++i)
#pragma unroll
                for (int j = 0; j < 4; ++j) {
                    if constexpr (kExact) ex[i][j].add(a[i], q[j]);
                    else r[i][j] = fmaf(a[i], q[j], r[i][j]);
                }
        }
        __syncthreads();
    }
    for (int i = 0; i < 4; ++i)
        for (int j = 0; j < 4; ++j) {
            const int c = c0 + ty * 4 + i, o = o0 + tx * 4 + j;
            float v = r[i][j];
            if constexpr (kExact) v = ex[i][j].value();
            if (c < Mc && o < No) dW[(int64_t)c * No + o] = v;
        }
}

__device__ __forceinline__ void unpack16(uint4 v, float (&f)[8], __nv_bfloat16) {
    const uint32_t u[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
    for (int q = 0; q < 4; ++q) {
        f[2 * q] = __uint_as_float(u[q] << 16);
        f[2 * q + 1] = __uint_as_float(u[q] & 0xffff0000u);
    }
}
__device__ __forceinline__ void unpack16(uint4 v, float (&f)[8], float) {
    f[0] = __uint_as_float(v.x);
    f[1] = __uint_as_float(v.y);
    f[2] = __uint_as_float(v.z);
    f[3] = __uint_as_float(v.w);
}

// A warp per slot over the whole grid (every slot's two row loads in flight
// at once), a lane per 16-byte vector of the value row (D_v <= 32 vectors).
// dacc_src: the dacc buffer (fp32), or, without a projector, g itself.
template <typename T>
__global__ void __launch_bounds__(kThreads) rows_kernel(Dims d, Ptrs p, const void *dacc_src,
                                                        float *dV, float *dw) {
    constexpr int EPV = 16 / sizeof(T);
    const int Dv = d.d_v, EDv = d.E * Dv, nc = d.nc, hm = d.H * d.m;
    const int lane = threadIdx.x & 31;
    const int64_t slot = (int64_t)blockIdx.x * kWarps + (threadIdx.x >> 5);
    if (slot >= (int64_t)d.B * hm) return;   // warp-uniform
    const int64_t b = slot / hm;
    const bool active = lane * EPV < Dv;
    const int wsel = nc == 1 || !active ? 0 : (lane * EPV) / (Dv / nc);   // this lane's slice
    const int64_t v = p.idx_in[slot];
    if (v < 0 || (uint64_t)v >= d.M) {   // not an address of this layer
        if (lane == 0) atomicOr(p.err, kErrBadIndex);
        if (dw && lane < nc) dw[slot * nc + lane] = 0.f;
        return;
    }
    const uint64_t vs = shuffle_address(d, p.perm, (uint64_t)v);
    const int pb = (int)(vs / (uint64_t)d.N);
    const int64_t row = (int64_t)(vs - (uint64_t)pb * (uint64_t)d.N);
    const float we = p.w_in[slot * nc + wsel];
    // the slice dot products: fp64 for fp32 storage (one rounding of dw)
    using A = typename std::conditional<std::is_same<T, float>::value, double, float>::type;
    A part = 0;
    if (active) {
        float f[8], dac[8];
        unpack16(*reinterpret_cast<const uint4 *>(static_cast<const T *>(p.values) + row * Dv +
                                                  lane * EPV),
                 f, T());
        const int64_t o = b * EDv + (int64_t)pb * Dv + lane * EPV;
        if (d.has_proj) {
            const float4 *src = reinterpret_cast<const float4 *>(static_cast<const float *>(dacc_src) + o);
#pragma unroll
            for (int c = 0; c < EPV; c += 4) {
                const float4 q = src[c / 4];
                dac[c] = q.x; dac[c + 1] = q.y; dac[c + 2] = q.z; dac[c + 3] = q.w;
            }
        } else {
            unpack16(*reinterpret_cast<const uint4 *>(static_cast<const T *>(dacc_src) + o), dac,
                     T());
        }
#pragma unroll
        for (int c = 0; c < EPV; ++c) part += (A)dac[c] * (A)f[c];
        if (dV) {
            float *dst = dV + row * Dv + lane * EPV;
#pragma unroll
            for (int c = 0; c < EPV; c += 4)
                atomicAdd(reinterpret_cast<float4 *>(dst + c),
                          make_float4(we * dac[c], we * dac[c + 1], we * dac[c + 2],
                                      we * dac[c + 3]));
        }
    }
    // dw: the sum of the slice's lanes (nc <= 8 warp sums, fixed order)
    if (dw)
        for (int i = 0; i < nc; ++i) {
            A sv = wsel == i && active ? part : (A)0;
#pragma unroll
            for (int off = 16; off > 0; off >>= 1) sv += __shfl_xor_sync(kFull, sv, off);
            if (lane == 0) dw[slot * nc + i] = (float)sv;
        }
}

}  // namespace

bool backward_fits(const Dims &d) {
    const int epv = d.dtype == ULTRAMEM_BF16 ? 8 : 4;
    return d.d_v % epv == 0 && d.d_v / epv <= 32;
}

cudaError_t configure_backward(const Dims &) { return cudaSuccess; }

// dacc (with a projector) then dV and dw; g [B][D'_v] in the storage type.
cudaError_t launch_backward_rows(const Dims &d, const Ptrs &p, const void *g, float *dacc,
                                 bool dacc_ready, float *dV, float *dw, cudaStream_t st) {
    const bool bf = d.dtype == ULTRAMEM_BF16;
    if (d.has_proj && !dacc_ready) {
        // slices of D'_v so that about two waves of CTAs run
        const int tiles = ((d.E * d.d_v + 63) / 64) * ((d.B + 31) / 32);
        int ks = (2 * device_sm_count() + tiles - 1) / tiles;
        ks = max(1, min(ks, (d.d_out + 127) / 128));
        if (!bf) ks = 1;   // fp32 storage: one compensated sum, stored (no atomics)
        dim3 grid((d.E * d.d_v + 63) / 64, (d.B + 31) / 32, ks);
        cudaError_t z = cudaMemsetAsync(dacc, 0, sizeof(float) * d.B * d.E * d.d_v, st);
        if (z != cudaSuccess) return z;
        if (bf)
            dacc_kernel<__nv_bfloat16><<<grid, kThreads, 0, st>>>(
                d, static_cast<const __nv_bfloat16 *>(g),
                static_cast<const __nv_bfloat16 *>(p.w_proj), dacc);
        else
            dacc_kernel<float><<<grid, kThreads, 0, st>>>(d, static_cast<const float *>(g),
                                                          static_cast<const float *>(p.w_proj),
                                                          dacc);
        cudaError_t e = cudaGetLastError();
        if (e != cudaSuccess) return e;
    }
    const void *src = d.has_proj ? static_cast<const void *>(dacc) : g;
    const int64_t slots = (int64_t)d.B * d.H * d.m;
    const unsigned blocks = (unsigned)((slots + kWarps - 1) / kWarps);
    if (bf)
        rows_kernel<__nv_bfloat16><<<blocks, kThreads, 0, st>>>(d, p, src, dV, dw);
    else
        rows_kernel<float><<<blocks, kThreads, 0, st>>>(d, p, src, dV, dw);
    return cudaGetLastError();
}

// dW_p from the forward's pooled rows acc (fp32 [B][E D_v]) and g.
cudaError_t launch_backward_proj(const Dims &d, const float *acc, const void *g, float *dW,
                                 cudaStream_t st) {
    dim3 grid((d.E * d.d_v + 63) / 64, (d.d_out + 63) / 64);
    if (d.dtype == ULTRAMEM_BF16)
        dwp_kernel<__nv_bfloat16><<<grid, kThreads, 0, st>>>(
            d, acc, static_cast<const __nv_bfloat16 *>(g), dW);
    else
        dwp_kernel<float><<<grid, kThreads, 0, st>>>(d, acc, static_cast<const float *>(g), dW);
    return cudaGetLastError();
}

}  // namespace um
