// Jurisdiction-masked reachability (Sec. 3.3 forbidden-vertex policy over
// G = (V, E); Sec. 4.2 graph search over the current topology).
//
// R(s, m) is the least set that contains s when region(s) is permitted by m
// and is closed under edges u -> v into permitted v.  One block computes it
// for one mask and a batch of 64 sources at once: vertex v holds a 64-bit
// word whose bit j says "v is in R(src_j, m)" (multi-source, bit-parallel
// frontier propagation).  Sweeps pull over in-edges,
//     vis[v] |= OR_{u -> v} vis[u]      for permitted v,
// in place, until a sweep changes nothing; in-place updates only speed up
// convergence and the fixpoint is exactly the closure, so the result equals
// a breadth-first search per source.  At most V + 1 sweeps run (each sweep
// extends every search by at least one level).  The vertex-major words are
// transposed with __ballot_sync into the caller's source-major bitset rows,
// written with 128-bit stores.
#include <cuda_runtime.h>

#include <algorithm>
#include <mutex>

#include "pv_internal.cuh"

namespace {

constexpr uint32_t kReachMaxV = 16384;
constexpr int kReachThreads = 512;
constexpr int kGridThreads = 256;

inline size_t align256(size_t x) { return (x + 255) & ~(size_t)255; }

// In-degree count with validation of the caller's CSR.
__global__ void reach_indeg_kernel(uint32_t V, uint32_t E, const uint32_t *__restrict__ offs,
                                   const uint32_t *__restrict__ cols, const uint8_t *__restrict__ region,
                                   uint32_t *__restrict__ indeg, int32_t *status) {
    for (uint32_t u = blockIdx.x * blockDim.x + threadIdx.x; u < V; u += gridDim.x * blockDim.x) {
        if (region[u] >= 32) pv_device_error(status, PV_EINVAL);
        const uint32_t a = offs[u], b = offs[u + 1];
        if (b < a || b > E) {
            pv_device_error(status, PV_EINVAL);
            continue;
        }
        for (uint32_t e = a; e < b; ++e) {
            const uint32_t v = cols[e];
            if (v >= V) {
                pv_device_error(status, PV_EINVAL);
                continue;
            }
            atomicAdd(&indeg[v], 1u);
        }
    }
}

// Single block: in_offs = exclusive scan of indeg (V+1 entries); cursor copy.
__global__ void __launch_bounds__(1024) reach_scan_kernel(uint32_t V, const uint32_t *__restrict__ indeg,
                                                          uint32_t *__restrict__ in_offs,
                                                          uint32_t *__restrict__ cursor) {
    __shared__ uint32_t s_warp[32];
    __shared__ uint32_t s_carry;
    const uint32_t t = threadIdx.x, lane = t & 31, warp = t >> 5;
    if (t == 0) s_carry = 0;
    __syncthreads();
    for (uint32_t c0 = 0; c0 < V; c0 += 1024) {
        const uint32_t i = c0 + t;
        const uint32_t x = i < V ? indeg[i] : 0;
        uint32_t incl = x;
        for (int d = 1; d < 32; d <<= 1) {
            uint32_t y = __shfl_up_sync(PV_FULL_MASK, incl, d);
            if (lane >= (uint32_t)d) incl += y;
        }
        if (lane == 31) s_warp[warp] = incl;
        __syncthreads();
        if (warp == 0) {
            uint32_t v = s_warp[lane], vi = v;
            for (int d = 1; d < 32; d <<= 1) {
                uint32_t y = __shfl_up_sync(PV_FULL_MASK, vi, d);
                if (lane >= (uint32_t)d) vi += y;
            }
            s_warp[lane] = vi - v;
        }
        __syncthreads();
        const uint32_t excl = s_carry + s_warp[warp] + incl - x;
        if (i < V) {
            in_offs[i] = excl;
            cursor[i] = excl;
        }
        __syncthreads();
        if (t == 1023) s_carry = excl + x;
        __syncthreads();
    }
    if (t == 0) in_offs[V] = s_carry;
}

__global__ void reach_fill_kernel(uint32_t V, uint32_t E, const uint32_t *__restrict__ offs,
                                  const uint32_t *__restrict__ cols, uint32_t *__restrict__ cursor,
                                  uint32_t *__restrict__ in_cols) {
    for (uint32_t u = blockIdx.x * blockDim.x + threadIdx.x; u < V; u += gridDim.x * blockDim.x) {
        const uint32_t a = offs[u], b = offs[u + 1];
        if (b < a || b > E) continue;
        for (uint32_t e = a; e < b; ++e) {
            const uint32_t v = cols[e];
            if (v < V) in_cols[atomicAdd(&cursor[v], 1u)] = u;
        }
    }
}

__global__ void __launch_bounds__(kReachThreads) reach_msbfs_kernel(
    uint32_t V, const uint32_t *__restrict__ in_offs, const uint32_t *__restrict__ in_cols,
    const uint8_t *__restrict__ region, uint32_t num_src, const uint32_t *__restrict__ src,
    const uint32_t *__restrict__ masks, uint32_t *__restrict__ reach, uint32_t W) {
    extern __shared__ uint64_t s_vis[];                 // [V]
    __shared__ uint32_t s_allow[kReachMaxV / 32];
    const uint32_t t = threadIdx.x, lane = t & 31, warp = t >> 5;
    const uint32_t m = blockIdx.y;
    const uint32_t j0 = blockIdx.x * 64, nb = min(64u, num_src - j0);
    const uint32_t mask = masks[m];
    volatile uint64_t *vis = s_vis;
    for (uint32_t v0 = 0; v0 < V; v0 += kReachThreads) {
        const uint32_t v = v0 + t;
        bool ok = false;
        if (v < V) {
            const uint32_t r = region[v];
            ok = r < 32 && ((mask >> r) & 1u);
            s_vis[v] = 0;
        }
        const uint32_t b = __ballot_sync(PV_FULL_MASK, ok);
        if (lane == 0 && v0 + warp * 32 < V) s_allow[(v0 >> 5) + warp] = b;
    }
    __syncthreads();
    if (t < nb) {
        const uint32_t s = src[j0 + t];
        if (s < V && ((s_allow[s >> 5] >> (s & 31)) & 1u)) atomicOr((unsigned long long *)&s_vis[s], 1ull << t);
    }
    __syncthreads();
    for (uint32_t iter = 0; iter <= V; ++iter) {
        int changed = 0;
        for (uint32_t v = t; v < V; v += kReachThreads) {
            if (!((s_allow[v >> 5] >> (v & 31)) & 1u)) continue;
            const uint64_t old = vis[v];
            uint64_t acc = old;
            const uint32_t a = __ldg(in_offs + v), b = __ldg(in_offs + v + 1);
            for (uint32_t e = a; e < b; ++e) acc |= vis[__ldg(in_cols + e)];
            if (acc != old) {
                vis[v] = acc;
                changed = 1;
            }
        }
        if (!__syncthreads_or(changed)) break;
    }
    // transpose: warp handles 128 vertices (4 words) per step
    const uint32_t groups = W / 4;
    for (uint32_t q = warp; q < groups; q += kReachThreads / 32) {
        uint64_t x[4];
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            const uint32_t v = q * 128 + i * 32 + lane;
            x[i] = v < V ? vis[v] : 0ull;
        }
        uint4 lo = make_uint4(0, 0, 0, 0), hi = make_uint4(0, 0, 0, 0);
        for (uint32_t j = 0; j < 64; ++j) {
            uint32_t b[4];
#pragma unroll
            for (int i = 0; i < 4; ++i) b[i] = __ballot_sync(PV_FULL_MASK, (x[i] >> j) & 1ull);
            if (lane == (j & 31)) {
                if (j < 32) lo = make_uint4(b[0], b[1], b[2], b[3]);
                else hi = make_uint4(b[0], b[1], b[2], b[3]);
            }
        }
        if (lane < nb)
            reinterpret_cast<uint4 *>(reach + ((size_t)m * num_src + j0 + lane) * W)[q] = lo;
        if (lane + 32 < nb)
            reinterpret_cast<uint4 *>(reach + ((size_t)m * num_src + j0 + lane + 32) * W)[q] = hi;
    }
}

}  // namespace

extern "C" int pv_compliant_reach(pv_ctx *ctx, uint32_t V, const uint32_t *d_offs, uint32_t num_edges,
                                  const uint32_t *d_cols, const uint8_t *d_region, uint32_t num_src,
                                  const uint32_t *d_src, uint32_t num_masks, const uint32_t *d_masks,
                                  uint32_t *d_reach, uint32_t words_per_row, pv_stream stream) {
    if (!ctx) return PV_EINVAL;
    if (V == 0 || V > kReachMaxV) return pv_fail(ctx, PV_EINVAL, "pv_compliant_reach: V must be 1..%u", kReachMaxV);
    if (words_per_row % 4 != 0 || words_per_row < (V + 31) / 32)
        return pv_fail(ctx, PV_EINVAL, "pv_compliant_reach: words_per_row must be >= ceil(V/32) and a multiple of 4");
    if (num_src == 0 || num_masks == 0) return PV_OK;
    if (!d_offs || !d_region || !d_src || !d_masks || !d_reach || (num_edges && !d_cols))
        return pv_fail(ctx, PV_EINVAL, "pv_compliant_reach: NULL device pointer");
    if (((uintptr_t)d_reach & 15) != 0) return pv_fail(ctx, PV_EINVAL, "pv_compliant_reach: d_reach must be 16-byte aligned");
    if (num_masks > 65535) return pv_fail(ctx, PV_EINVAL, "pv_compliant_reach: num_masks must be <= 65535");
    const size_t o_indeg = 0, o_in_offs = align256((size_t)(V + 1) * 4);
    const size_t o_cursor = o_in_offs + align256((size_t)(V + 1) * 4);
    const size_t o_cols = o_cursor + align256((size_t)V * 4);
    const size_t total = o_cols + align256((size_t)num_edges * 4 + 4);
    uint8_t *base = (uint8_t *)pv_scratch(ctx, total);
    if (!base) return PV_ENOMEM;
    uint32_t *indeg = (uint32_t *)(base + o_indeg), *in_offs = (uint32_t *)(base + o_in_offs);
    uint32_t *cursor = (uint32_t *)(base + o_cursor), *in_cols = (uint32_t *)(base + o_cols);
    cudaStream_t st = (cudaStream_t)stream;
    PV_TRY_CUDA(ctx, cudaMemsetAsync(indeg, 0, (size_t)(V + 1) * 4, st), "indeg clear");
    const uint32_t grid = std::min<uint32_t>((V + kGridThreads - 1) / kGridThreads, (uint32_t)ctx->num_sms * 8);
    const int pr = pv_prof_start(ctx, st, PV_K_REACH);
    reach_indeg_kernel<<<grid, kGridThreads, 0, st>>>(V, num_edges, d_offs, d_cols, d_region, indeg, ctx->d_status);
    reach_scan_kernel<<<1, 1024, 0, st>>>(V, indeg, in_offs, cursor);
    reach_fill_kernel<<<grid, kGridThreads, 0, st>>>(V, num_edges, d_offs, d_cols, cursor, in_cols);
    const size_t smem = (size_t)V * 8;
    PV_TRY_CUDA(ctx, cudaFuncSetAttribute(reach_msbfs_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem),
                "reach smem");
    dim3 g2((num_src + 63) / 64, num_masks);
    reach_msbfs_kernel<<<g2, kReachThreads, smem, st>>>(V, in_offs, in_cols, d_region, num_src, d_src, d_masks,
                                                       d_reach, words_per_row);
    pv_prof_stop(ctx, st, pr, 4);
    return pv_check_launch(ctx, "reach kernels");
}

// -----------------------------------------------------------------------------
// Compliant reach that allocates nothing.
//
// For callers that must not allocate device memory themselves or through this
// library: a host program whose device memory is owned by another framework's
// pool or held to a fixed budget, or a latency-critical caller that cannot
// afford the device-wide synchronisation cudaMalloc / cudaFree may imply.
// The in-edge CSR this path builds lives in one static device array below;
// every GPU that loads the library holds it until the process exits.
// -----------------------------------------------------------------------------
namespace {

constexpr size_t up256(size_t x) { return (x + 255) & ~(size_t)255; }

constexpr uint32_t kNoAllocMaxEdges = 1u << 18;   // directed edges accepted by the no-allocation call
constexpr size_t kNoAllocIndeg = 256;              // [0, 256): status word
constexpr size_t kNoAllocInOffs = kNoAllocIndeg + up256((size_t)(kReachMaxV + 1) * 4);
constexpr size_t kNoAllocCursor = kNoAllocInOffs + up256((size_t)(kReachMaxV + 1) * 4);
constexpr size_t kNoAllocCols = kNoAllocCursor + up256((size_t)kReachMaxV * 4);
constexpr size_t kNoAllocBytes = kNoAllocCols + up256((size_t)kNoAllocMaxEdges * 4);   // about 1.2 MB

__device__ __align__(256) uint8_t g_reach_noalloc_scratch[kNoAllocBytes];

constexpr int kNoAllocMaxDevices = 64;
std::mutex g_noalloc_mutex;
uint8_t *g_noalloc_base[kNoAllocMaxDevices] = {};

// Device address of the static array on the current device, looked up once
// per device (in host code the array's name is not a device address).
int noalloc_scratch(uint8_t **out) {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return PV_ECUDA;
    if (dev < 0 || dev >= kNoAllocMaxDevices) return PV_EINVAL;
    std::lock_guard<std::mutex> lock(g_noalloc_mutex);
    if (!g_noalloc_base[dev]) {
        void *p = nullptr;
        if (cudaGetSymbolAddress(&p, g_reach_noalloc_scratch) != cudaSuccess || !p) return PV_ECUDA;
        g_noalloc_base[dev] = static_cast<uint8_t *>(p);
    }
    *out = g_noalloc_base[dev];
    return PV_OK;
}

}  // namespace

extern "C" int pv_compliant_reach_noalloc(uint32_t V, const uint32_t *d_offs, uint32_t num_edges,
                                          const uint32_t *d_cols, const uint8_t *d_region, uint32_t num_src,
                                          const uint32_t *d_src, uint32_t num_masks, const uint32_t *d_masks,
                                          uint32_t *d_reach, uint32_t words_per_row, pv_stream stream) {
    if (V == 0 || V > kReachMaxV) return PV_EINVAL;
    if (num_edges > kNoAllocMaxEdges) return PV_EINVAL;
    if (words_per_row % 4 != 0 || words_per_row < (V + 31) / 32) return PV_EINVAL;
    if (num_src == 0 || num_masks == 0) return PV_OK;
    if (!d_offs || !d_region || !d_src || !d_masks || !d_reach || (num_edges && !d_cols)) return PV_EINVAL;
    if (((uintptr_t)d_reach & 15) != 0 || num_masks > 65535) return PV_EINVAL;
    uint8_t *base = nullptr;
    const int rc = noalloc_scratch(&base);
    if (rc != PV_OK) return rc;
    int32_t *status = reinterpret_cast<int32_t *>(base);
    uint32_t *indeg = reinterpret_cast<uint32_t *>(base + kNoAllocIndeg);
    uint32_t *in_offs = reinterpret_cast<uint32_t *>(base + kNoAllocInOffs);
    uint32_t *cursor = reinterpret_cast<uint32_t *>(base + kNoAllocCursor);
    uint32_t *in_cols = reinterpret_cast<uint32_t *>(base + kNoAllocCols);
    cudaStream_t st = (cudaStream_t)stream;
    // the array keeps the previous call's contents: clear what must start at zero
    if (cudaMemsetAsync(base, 0, kNoAllocIndeg + (size_t)(V + 1) * 4, st) != cudaSuccess) return PV_ECUDA;
    int dev = 0, sms = 0;
    if (cudaGetDevice(&dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
        return PV_ECUDA;
    const uint32_t grid = std::min<uint32_t>((V + kGridThreads - 1) / kGridThreads, (uint32_t)sms * 8);
    reach_indeg_kernel<<<grid, kGridThreads, 0, st>>>(V, num_edges, d_offs, d_cols, d_region, indeg, status);
    reach_scan_kernel<<<1, 1024, 0, st>>>(V, indeg, in_offs, cursor);
    reach_fill_kernel<<<grid, kGridThreads, 0, st>>>(V, num_edges, d_offs, d_cols, cursor, in_cols);
    const size_t smem = (size_t)V * 8;
    if (cudaFuncSetAttribute(reach_msbfs_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem) !=
        cudaSuccess)
        return PV_ECUDA;
    dim3 g2((num_src + 63) / 64, num_masks);
    reach_msbfs_kernel<<<g2, kReachThreads, smem, st>>>(V, in_offs, in_cols, d_region, num_src, d_src, d_masks,
                                                       d_reach, words_per_row);
    return cudaGetLastError() == cudaSuccess ? PV_OK : PV_ECUDA;
}
