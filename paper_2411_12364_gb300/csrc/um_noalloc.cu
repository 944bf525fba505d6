// um_noalloc.cu -- ultramem_lookup_reduce_noalloc: the lookup-reduce (S7-S9)
// for callers that must not allocate device memory, such as code running
// where the allocator is owned by someone else, inside a fixed memory budget,
// or at a point where an allocation could block or fail.  It takes no layer
// handle and calls no allocating routine.  Its scratch (the per-slot rows,
// blocks and weights, the per-block pooled rows and the projection partial
// sums) lives in one file-scope __device__ array of kScratchBytes that every
// GPU loading this library holds until the process exits.  The kernels are
// the ones the layer handle uses.
#include <math.h>
#include <string.h>

#include <mutex>

#include "um_internal.cuh"

namespace um {
cudaError_t configure_gather(const Dims &d);
void host_shuffle_params(uint64_t seed, uint64_t M, uint64_t *a, uint64_t *c);
}  // namespace um

namespace {

constexpr size_t kScratchBytes = 8u << 20;   // 8 MiB
constexpr int kMaxDevices = 64;

static __device__ __align__(256) unsigned char g_scratch[kScratchBytes];

std::mutex g_mu;
void *g_scratch_addr[kMaxDevices];     // device address of g_scratch per device
bool g_configured[kMaxDevices];        // the gather kernels' shared memory limit set

size_t align256(size_t x) { return (x + 255) & ~size_t(255); }

ultramem_status status_of(cudaError_t e) {
    if (e == cudaSuccess) return ULTRAMEM_OK;
    cudaGetLastError();
    return e == cudaErrorMemoryAllocation ? ULTRAMEM_ENOMEM : ULTRAMEM_ECUDA;
}

int splits_for(int B, int d_out, int kd) {
    int tiles = ((d_out + 63) / 64) * ((B + 31) / 32);
    int s = (304 + tiles - 1) / tiles;
    int cap = kd / 64 > 0 ? kd / 64 : 1;
    if (s > 8) s = 8;
    if (s > cap) s = cap;
    return s < 1 ? 1 : s;
}

}  // namespace

extern "C" ultramem_status ultramem_lookup_reduce_noalloc(const ultramem_config *cfg,
                                                          const void *values,
                                                          const void *w_proj,
                                                          const uint32_t *perm,
                                                          const int64_t *idx, const float *w,
                                                          int32_t B, void *out, void *stream) {
    if (!cfg || B < 0) return ULTRAMEM_EINVAL;
    if (B == 0) return ULTRAMEM_OK;
    const ultramem_config &c = *cfg;
    const int s = (int)lround(sqrt((double)c.expand_e));
    if (c.heads <= 0 || c.topm <= 0 || c.n <= 0 || c.d_v <= 0 || c.d_v % 8 ||
        c.expand_e < 1 || c.expand_e > 16 || s * s != c.expand_e ||
        (c.dtype != ULTRAMEM_F32 && c.dtype != ULTRAMEM_BF16) ||
        (c.has_proj != 0 && c.has_proj != 1) ||
        (!c.has_proj && (c.expand_e != 1 || c.d_out != c.d_v)) || (c.has_proj && c.d_out <= 0) ||
        c.cores < 0 || c.cores > 8 || (c.cores > 1 && c.d_v % (8 * c.cores)))
        return ULTRAMEM_EINVAL;
    const uint64_t N = (uint64_t)c.n * c.n, M = (uint64_t)c.expand_e * N;
    if (M >= (1ull << 32)) return ULTRAMEM_EINVAL;
    if (!values || !idx || !w || !out || (c.has_proj && !w_proj)) return ULTRAMEM_EINVAL;
    if ((uintptr_t)values % 16) return ULTRAMEM_EINVAL;

    um::Dims d;
    memset(&d, 0, sizeof d);
    d.B = B;
    d.H = c.heads;
    d.m = c.topm;
    d.nc = c.cores > 1 ? c.cores : 1;
    d.N = (int64_t)N;
    d.M = M;
    d.E = c.expand_e;
    d.d_v = c.d_v;
    d.d_out = c.d_out;
    d.dtype = c.dtype;
    d.has_proj = c.has_proj;
    d.q_splits = 1;
    const int kd = d.E * d.d_v;
    d.p_splits = c.has_proj ? splits_for(B, d.d_out, kd) : 1;
    um::host_shuffle_params(c.shuffle_seed, M, &d.shuf_a, &d.shuf_c);
    d.shuf_mu = um::barrett_mu(M);

    // scratch layout: error word | rows | blocks | weights | acc | partials
    const size_t slots = (size_t)B * d.H * d.m;
    size_t off = 0;
    const size_t o_err = off;
    off = align256(off + sizeof(int));
    const size_t o_row = off;
    off = align256(off + slots * sizeof(int32_t));
    const size_t o_blk = off;
    off = align256(off + slots * sizeof(int32_t));
    const size_t o_w = off;
    off = align256(off + slots * d.nc * sizeof(float));
    const size_t o_acc = off;
    if (c.has_proj) off = align256(off + (size_t)B * kd * sizeof(float));
    const size_t o_part = off;
    if (c.has_proj) off = align256(off + (size_t)d.p_splits * B * d.d_out * sizeof(float));
    if (off > kScratchBytes) return ULTRAMEM_EINVAL;   // batch too large for the scratch

    // once per device, with that device current: the array's device address
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) {
        cudaGetLastError();
        return ULTRAMEM_ENODEV;
    }
    if (dev < 0 || dev >= kMaxDevices) return ULTRAMEM_EINVAL;
    unsigned char *base;
    {
        std::lock_guard<std::mutex> lock(g_mu);
        if (!g_scratch_addr[dev]) {
            void *ptr = nullptr;
            cudaError_t e = cudaGetSymbolAddress(&ptr, g_scratch);
            if (e != cudaSuccess || !ptr) return status_of(e);
            g_scratch_addr[dev] = ptr;
        }
        if (!g_configured[dev]) {   // once per device: the kernels' maximum, never lowered
            cudaError_t e = um::configure_gather(d);
            if (e != cudaSuccess) return status_of(e);
            g_configured[dev] = true;
        }
        base = static_cast<unsigned char *>(g_scratch_addr[dev]);
    }

    um::Ptrs p;
    memset(&p, 0, sizeof p);
    p.values = values;
    p.w_proj = w_proj;
    p.perm = perm;
    p.idx_in = idx;
    p.w_in = w;
    p.out = out;
    p.err = reinterpret_cast<int *>(base + o_err);
    p.sel_row = reinterpret_cast<int32_t *>(base + o_row);
    p.sel_p = reinterpret_cast<int32_t *>(base + o_blk);
    p.sel_w = reinterpret_cast<float *>(base + o_w);
    p.acc = c.has_proj ? reinterpret_cast<float *>(base + o_acc) : nullptr;
    p.proj_part = c.has_proj ? reinterpret_cast<float *>(base + o_part) : nullptr;

    cudaStream_t st = static_cast<cudaStream_t>(stream);
    cudaGetLastError();
    cudaError_t e = cudaMemsetAsync(p.err, 0, sizeof(int), st);   // the one word that starts at 0
    if (e == cudaSuccess) e = um::launch_slots_from_addresses(d, p, st);
    if (e == cudaSuccess) e = um::launch_gather(d, p, st);
    if (e == cudaSuccess && c.has_proj) e = um::launch_proj(d, p, st);
    return status_of(e);
}
