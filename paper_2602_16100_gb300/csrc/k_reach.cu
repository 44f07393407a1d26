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
//
// Symmetric graphs (every edge u -> v has its reverse v -> u) take an exact
// shortcut: there a path s -> v inside the permitted vertices exists iff s
// and v lie in the same connected component of the subgraph induced by the
// permitted vertices, so R(s, m) is that component (or empty when s itself
// is not permitted).  One block labels the components of one mask with a
// lock-free union-find in shared memory, materialises the bitset of each
// component its sources fall in, and copies those rows out: the output
// write is the whole cost.  A device-side check decides per call which of
// the two paths runs; both are launched and the other one returns at once.
#include <cuda_runtime.h>

#include <algorithm>
#include <mutex>

#include "pv_internal.cuh"

namespace {

constexpr uint32_t kReachMaxV = 16384;
constexpr int kReachThreads = 512;
constexpr int kGridThreads = 256;

inline size_t align256(size_t x) { return (x + 255) & ~(size_t)255; }

// A CSR whose offsets are malformed (some row with offs[u + 1] < offs[u] or
// offs[u + 1] > E) counts as having no edges at all: its well-formed rows
// could overlap, so their lengths could add up past E, the size of every
// edge-indexed scratch array.  indeg[V] (cleared with the counts, never
// counted into) is that per-call flag; every later kernel of the call reads
// it before it touches an edge.
__device__ __forceinline__ bool csr_offsets_bad(const uint32_t *bad) {
    return *(volatile const uint32_t *)bad != 0;
}

// In-degree count with validation of the caller's CSR.  An out-of-range
// column skips that edge; malformed offsets set the flag at indeg[V] (the
// counts of this pass are then unused).
__global__ void reach_indeg_kernel(uint32_t V, uint32_t E, const uint32_t *__restrict__ offs,
                                   const uint32_t *__restrict__ cols, const uint8_t *__restrict__ region,
                                   uint32_t *__restrict__ indeg, int32_t *status) {
    for (uint32_t u = blockIdx.x * blockDim.x + threadIdx.x; u < V; u += gridDim.x * blockDim.x) {
        if (region[u] >= 32) pv_device_error(status, PV_EINVAL);
        const uint32_t a = offs[u], b = offs[u + 1];
        if (b < a || b > E) {
            pv_device_error(status, PV_EINVAL);
            atomicOr(&indeg[V], 1u);
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
// With malformed offsets every in-edge list is empty.
__global__ void __launch_bounds__(1024) reach_scan_kernel(uint32_t V, const uint32_t *__restrict__ indeg,
                                                          uint32_t *__restrict__ in_offs,
                                                          uint32_t *__restrict__ cursor, const uint32_t *asym) {
    if (asym && *(volatile const uint32_t *)asym == 0) return;   // symmetric: in-edges unused
    __shared__ uint32_t s_warp[32];
    __shared__ uint32_t s_carry;
    const bool bad = csr_offsets_bad(indeg + V);
    const uint32_t t = threadIdx.x, lane = t & 31, warp = t >> 5;
    if (t == 0) s_carry = 0;
    __syncthreads();
    for (uint32_t c0 = 0; c0 < V; c0 += 1024) {
        const uint32_t i = c0 + t;
        const uint32_t x = i < V && !bad ? indeg[i] : 0;
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
                                  uint32_t *__restrict__ in_cols, const uint32_t *asym, const uint32_t *bad) {
    if (asym && *(volatile const uint32_t *)asym == 0) return;   // symmetric: in-edges unused
    if (csr_offsets_bad(bad)) return;                            // no edges
    for (uint32_t u = blockIdx.x * blockDim.x + threadIdx.x; u < V; u += gridDim.x * blockDim.x) {
        const uint32_t a = offs[u], b = offs[u + 1];
        if (b < a || b > E) continue;
        for (uint32_t e = a; e < b; ++e) {
            const uint32_t v = cols[e];
            if (v < V) in_cols[atomicAdd(&cursor[v], 1u)] = u;
        }
    }
}

// Symmetry check of the caller's out-edge CSR, one warp per vertex:
// *asym != 0 unless every edge u -> v (v < V, both lists well formed) has
// its reverse v -> u.  Vertices whose list is longer than kSymScanMax make
// the graph count as asymmetric (the sweep path then runs; still exact).
// With malformed offsets (flag set by the in-degree pass) the graph has no
// edges, which is symmetric: nothing is listed.
// The same pass lists each undirected edge once, as pairs[] = u << 16 | v
// with v < u (*npairs of them, in no particular order).
constexpr uint32_t kSymScanMax = 64;

__global__ void reach_symcheck_kernel(uint32_t V, uint32_t E, const uint32_t *__restrict__ offs,
                                      const uint32_t *__restrict__ cols, uint32_t *asym, uint32_t *pairs,
                                      uint32_t *npairs, const uint32_t *bad) {
    if (csr_offsets_bad(bad)) return;   // no edges: symmetric, no pairs
    const uint32_t lane = threadIdx.x & 31;
    const uint32_t nwarps = gridDim.x * (blockDim.x / 32);
    for (uint32_t u = blockIdx.x * (blockDim.x / 32) + threadIdx.x / 32; u < V; u += nwarps) {
        // warp-uniform early exit (lane 0's read decides for the warp)
        if (__shfl_sync(PV_FULL_MASK, *(volatile uint32_t *)asym, 0)) return;
        const uint32_t a = offs[u], b = offs[u + 1];
        if (b < a || b > E) continue;
        if (b - a > kSymScanMax) {
            if (lane == 0) atomicOr(asym, 1u);
            return;
        }
        for (uint32_t e0 = a; e0 < b; e0 += 32) {
            const uint32_t e = e0 + lane;
            uint32_t v = V;
            bool ok = true;
            if (e < b) {
                v = cols[e];
                if (v < V && v != u) {
                    const uint32_t c = offs[v], d = offs[v + 1];
                    bool found = false;
                    if (!(d < c || d > E) && d - c <= kSymScanMax)
                        for (uint32_t f = c; f < d && !found; ++f) found = cols[f] == u;
                    ok = found;
                }
            }
            if (__any_sync(PV_FULL_MASK, !ok)) {
                if (lane == 0) atomicOr(asym, 1u);
                return;
            }
            const bool keep = v < u;   // v < V too
            const uint32_t bal = __ballot_sync(PV_FULL_MASK, keep);
            uint32_t base = 0;
            if (lane == 0 && bal) base = atomicAdd(npairs, (uint32_t)__popc(bal));
            base = __shfl_sync(PV_FULL_MASK, base, 0);
            if (keep) pairs[base + __popc(bal & ((1u << lane) - 1u))] = (u << 16) | v;
        }
    }
}

// Union-find over shared memory with parent[x] <= x at all times: roots are
// hooked under smaller roots by compare-and-swap, finds halve paths (a
// racing write only ever stores an ancestor).  A failed hook means the root
// gained a parent, so the next attempt starts from a smaller root: at most
// 2V attempts.
__device__ __forceinline__ uint32_t uf_find(volatile uint32_t *parent, uint32_t x) {
    for (;;) {
        const uint32_t p = parent[x];
        if (p == x) return x;
        const uint32_t gp = parent[p];
        if (gp != p) parent[x] = gp;
        x = gp;
    }
}

__device__ __forceinline__ void uf_union(volatile uint32_t *parent, uint32_t a, uint32_t b, uint32_t limit,
                                         int32_t *status) {
    for (uint32_t it = 0; it < limit; ++it) {
        a = uf_find(parent, a);
        b = uf_find(parent, b);
        if (a == b) return;
        if (a < b) {
            const uint32_t x = a;
            a = b;
            b = x;
        }
        if (atomicCAS(const_cast<uint32_t *>(parent + a), a, b) == a) return;
    }
    // not reachable by the argument above; should it happen all the same,
    // the row would be wrong, so the call reports it rather than pass
    pv_device_error(status, PV_ETIMEOUT);
}

constexpr int kCompThreads = 512;
constexpr uint32_t kNoComp = 0xFFFFFFFFu;
constexpr uint16_t kNoLabel = 0xFFFF;
constexpr uint16_t kSlotNone = 0xFFFF, kSlotWanted = 0xFFFE, kSlotOverflow = 0xFFFD;

__host__ __device__ inline uint32_t up16u(uint32_t x) { return (x + 15u) & ~15u; }

// Component labels of one mask per block: lab[m][v] = the smallest vertex
// of v's component in the permitted subgraph, kNoLabel for a vertex whose
// region the mask does not permit.  One pass over the pair list (from L2)
// points every permitted vertex at its smallest permitted neighbour below
// it (a valid forest of the same components, so most unions then find one
// root) and copies the pairs inside the permitted subgraph, usually a small
// share of them, to shared memory; the union pass then runs over that
// compact list (over the whole list again when it did not fit).
constexpr int kLabelThreads = 1024;
constexpr size_t kLabelSmemTarget = 100 * 1024;   // two label blocks per SM

// Layout of the labels kernel's dynamic shared memory for V vertices:
// parent[V], the permitted-vertex bitmap, then the compact pair list.
struct LabelSmem {
    uint32_t allow, pairs, cap;
    size_t total;
    __host__ __device__ explicit LabelSmem(uint32_t V) {
        allow = up16u(V * 4);
        pairs = allow + up16u(((V + 31) / 32) * 4);
        const size_t left = kLabelSmemTarget > pairs ? kLabelSmemTarget - pairs : 0;
        cap = (uint32_t)(left / 4) & ~3u;
        total = (size_t)pairs + (size_t)cap * 4;
    }
};

__global__ void __launch_bounds__(kLabelThreads) reach_labels_kernel(
    uint32_t V, const uint32_t *__restrict__ pairs, const uint32_t *__restrict__ npairs,
    const uint8_t *__restrict__ region, const uint32_t *__restrict__ masks, uint16_t *__restrict__ lab,
    const uint32_t *asym, int32_t *status) {
    if (*(volatile const uint32_t *)asym) return;       // not symmetric: the sweep kernel runs
    extern __shared__ __align__(16) uint8_t s_dyn[];
    __shared__ uint32_t s_np;                                                      // compact pairs
    const LabelSmem L(V);
    volatile uint32_t *parent = reinterpret_cast<uint32_t *>(s_dyn);              // [V]
    uint32_t *s_allow = reinterpret_cast<uint32_t *>(s_dyn + L.allow);            // [ceil(V / 32)]
    uint32_t *s_pairs = reinterpret_cast<uint32_t *>(s_dyn + L.pairs);            // [L.cap]
    const uint32_t t = threadIdx.x, lane = t & 31, warp = t >> 5, nt = blockDim.x;
    const uint32_t m = blockIdx.x, mask = masks[m];
    auto allowed = [&](uint32_t v) { return (s_allow[v >> 5] >> (v & 31)) & 1u; };
    // every vertex its own root; permitted-vertex bitmap
    for (uint32_t v0 = 0; v0 < V; v0 += nt) {
        const uint32_t v = v0 + t;
        bool ok = false;
        if (v < V) {
            const uint32_t r = region[v];
            ok = r < 32 && ((mask >> r) & 1u);
            parent[v] = v;
        }
        const uint32_t bal = __ballot_sync(PV_FULL_MASK, ok);
        if (lane == 0 && v0 + warp * 32 < V) s_allow[(v0 >> 5) + warp] = bal;
    }
    if (t == 0) s_np = 0;
    __syncthreads();
    // each permitted vertex under its smallest permitted neighbour; the
    // pairs inside the permitted subgraph copied to the compact list
    const uint32_t np = *npairs;
    for (uint32_t i0 = 0; i0 < np; i0 += 4 * nt) {
        const uint32_t i = i0 + 4 * t;
        uint32_t pq[4] = {0, 0, 0, 0};
        if (i < np) {
            const uint4 q = *reinterpret_cast<const uint4 *>(pairs + i);
            pq[0] = q.x;
            pq[1] = q.y;
            pq[2] = q.z;
            pq[3] = q.w;
        }
#pragma unroll
        for (int k = 0; k < 4; ++k) {
            const uint32_t u = pq[k] >> 16, v = pq[k] & 0xFFFFu;   // v < u
            const bool in = i + k < np && allowed(u) && allowed(v);
            if (in) atomicMin(const_cast<uint32_t *>(parent + u), v);
            const uint32_t bal = __ballot_sync(PV_FULL_MASK, in);
            uint32_t base = 0;
            if (lane == 0 && bal) base = atomicAdd(&s_np, (uint32_t)__popc(bal));
            base = __shfl_sync(PV_FULL_MASK, base, 0) + __popc(bal & ((1u << lane) - 1u));
            if (in && base < L.cap) s_pairs[base] = pq[k];
        }
    }
    __syncthreads();
    // union the endpoints of every undirected edge inside the permitted
    // vertices (each pair once): from the compact list, or from the whole
    // list again when the compact one overflowed
    const uint32_t nc = s_np;
    if (nc <= L.cap) {
        for (uint32_t i = t; i < nc; i += nt) {
            const uint32_t p = s_pairs[i];
            uf_union(parent, p >> 16, p & 0xFFFFu, 2 * V + 2, status);
        }
    } else {
        for (uint32_t i = 4 * t; i < np; i += 4 * nt) {
            const uint4 q = *reinterpret_cast<const uint4 *>(pairs + i);
            const uint32_t pq[4] = {q.x, q.y, q.z, q.w};
#pragma unroll
            for (int k = 0; k < 4; ++k) {
                const uint32_t u = pq[k] >> 16, v = pq[k] & 0xFFFFu;
                if (i + k < np && allowed(u) && allowed(v)) uf_union(parent, u, v, 2 * V + 2, status);
            }
        }
    }
    __syncthreads();
    uint16_t *out = lab + (size_t)m * V;
    for (uint32_t v = t; v < V; v += nt) out[v] = allowed(v) ? (uint16_t)uf_find(parent, v) : kNoLabel;
}

struct RowSmem {   // dynamic shared-memory layout of reach_rows_kernel
    uint32_t slot, slot_comp, rows, total;
    __host__ __device__ RowSmem(uint32_t V, uint32_t W, uint32_t cap) {
        slot = up16u(V * 4);
        slot_comp = slot + up16u(V * 2);
        rows = slot_comp + up16u(cap * 4);
        total = rows + cap * W * 4;
    }
};

// The bitset row of component c (all v < V with lab[v] == c; words past V
// are zero), W / 4 uint4s written by one warp to dst (shared or global).
__device__ __forceinline__ void comp_row(const uint32_t *lab, uint32_t V, uint32_t W, uint32_t c, uint4 *dst,
                                         uint32_t lane) {
    const uint32_t groups = W / 4;
    for (uint32_t g0 = 0; g0 < groups; g0 += 32) {
        uint4 mine = make_uint4(0, 0, 0, 0);
        const uint32_t n = min(32u, groups - g0);
        for (uint32_t i = 0; i < n; ++i) {
            const uint32_t base = (g0 + i) * 128 + lane;
            uint32_t bits[4];
#pragma unroll
            for (int k = 0; k < 4; ++k) {
                const uint32_t v = base + 32 * k;
                bits[k] = __ballot_sync(PV_FULL_MASK, v < V && lab[v] == c);
            }
            if (lane == i) mine = make_uint4(bits[0], bits[1], bits[2], bits[3]);
        }
        if (lane < n) dst[g0 + lane] = mine;
    }
}

// Rows of one mask for a slice of sources: R(s, m) = the bitset of s's
// component (empty when s is not permitted or out of range).  The
// components the slice's sources fall in get a shared-memory row each
// (first come, up to cap), built in one pass over the vertices; each output
// row is then a 128-bit copy, or, past cap, built from ballots directly.
__global__ void __launch_bounds__(kCompThreads) reach_rows_kernel(
    uint32_t V, const uint16_t *__restrict__ lab_all, uint32_t num_src, const uint32_t *__restrict__ src,
    uint32_t *__restrict__ reach, uint32_t W, uint32_t src_per_block, uint32_t cap, const uint32_t *asym) {
    if (*(volatile const uint32_t *)asym) return;
    extern __shared__ __align__(16) uint8_t s_dyn[];
    const RowSmem L(V, W, cap);
    uint32_t *s_lab = reinterpret_cast<uint32_t *>(s_dyn);
    uint16_t *s_slot = reinterpret_cast<uint16_t *>(s_dyn + L.slot);
    uint32_t *s_slot_comp = reinterpret_cast<uint32_t *>(s_dyn + L.slot_comp);
    uint4 *s_rows = reinterpret_cast<uint4 *>(s_dyn + L.rows);
    __shared__ uint32_t s_nslots;
    const uint32_t t = threadIdx.x, lane = t & 31, warp = t >> 5, nt = blockDim.x, nw = nt / 32;
    const uint32_t m = blockIdx.y;
    const uint32_t j0 = blockIdx.x * src_per_block, j1 = min(num_src, j0 + src_per_block);
    const uint16_t *lab = lab_all + (size_t)m * V;
    for (uint32_t v = t; v < V; v += nt) {
        const uint16_t l = lab[v];
        s_lab[v] = l == kNoLabel ? kNoComp : l;
        s_slot[v] = kSlotNone;
    }
    if (t == 0) s_nslots = 0;
    __syncthreads();
    for (uint32_t j = j0 + t; j < j1; j += nt) {
        const uint32_t s = src[j];
        if (s < V && s_lab[s] != kNoComp) s_slot[s_lab[s]] = kSlotWanted;
    }
    __syncthreads();
    for (uint32_t v = t; v < V; v += nt)
        if (s_slot[v] == kSlotWanted) {
            const uint32_t k = atomicAdd(&s_nslots, 1u);
            s_slot[v] = k < cap ? (uint16_t)k : kSlotOverflow;
            if (k < cap) s_slot_comp[k] = v;
        }
    __syncthreads();
    const uint32_t nsl = min(s_nslots, cap);
    // slot rows: cleared, then every word written once by the lanes of the
    // slot's component among its 32 vertices
    for (uint32_t q = t; q < nsl * (W / 4); q += nt) s_rows[q] = make_uint4(0, 0, 0, 0);
    __syncthreads();
    uint32_t *s_words = reinterpret_cast<uint32_t *>(s_rows);
    for (uint32_t v0 = warp * 32; v0 < V; v0 += nt) {
        const uint32_t v = v0 + lane;
        const uint32_t c = v < V ? s_lab[v] : kNoComp;
        const uint32_t k = c != kNoComp ? s_slot[c] : kSlotNone;
        const uint32_t peers = __match_any_sync(PV_FULL_MASK, k);
        if (k < cap && lane == (uint32_t)(__ffs(peers) - 1)) s_words[(size_t)k * W + (v0 >> 5)] = peers;
    }
    __syncthreads();
    for (uint32_t j = j0 + warp; j < j1; j += nw) {
        const uint32_t s = src[j];
        const uint32_t c = s < V ? s_lab[s] : kNoComp;
        uint4 *out = reinterpret_cast<uint4 *>(reach + ((size_t)m * num_src + j) * W);
        if (c == kNoComp) {
            for (uint32_t q = lane; q < W / 4; q += 32) out[q] = make_uint4(0, 0, 0, 0);
        } else if (s_slot[c] < cap) {
            const uint4 *row = s_rows + (size_t)s_slot[c] * (W / 4);
            for (uint32_t q = lane; q < W / 4; q += 32) out[q] = row[q];
        } else {
            comp_row(s_lab, V, W, c, out, lane);
        }
    }
}

// One work item of the sweep kernel: mask m, sources j0 .. j0 + 63.
__device__ __forceinline__ void msbfs_item(uint32_t V, const uint32_t *__restrict__ in_offs,
                                           const uint32_t *__restrict__ in_cols, const uint8_t *__restrict__ region,
                                           uint32_t num_src, const uint32_t *__restrict__ src, uint32_t mask,
                                           uint32_t *__restrict__ reach, uint32_t W, uint32_t m, uint32_t j0,
                                           uint64_t *s_vis, uint32_t *s_allow) {
    const uint32_t t = threadIdx.x, lane = t & 31, warp = t >> 5;
    const uint32_t nb = min(64u, num_src - j0);
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


__global__ void __launch_bounds__(kReachThreads) reach_msbfs_kernel(
    uint32_t V, const uint32_t *__restrict__ in_offs, const uint32_t *__restrict__ in_cols,
    const uint8_t *__restrict__ region, uint32_t num_src, const uint32_t *__restrict__ src, uint32_t num_masks,
    const uint32_t *__restrict__ masks, uint32_t *__restrict__ reach, uint32_t W, const uint32_t *asym) {
    // the component path has written the rows of a symmetric graph
    if (asym && *(volatile const uint32_t *)asym == 0) return;
    extern __shared__ uint64_t s_vis[];                 // [V]
    __shared__ uint32_t s_allow[kReachMaxV / 32];
    const uint32_t nbatch = (num_src + 63) / 64;
    const uint64_t items = (uint64_t)nbatch * num_masks;   // (mask, source batch) pairs
    for (uint64_t item = blockIdx.x; item < items; item += gridDim.x) {
        const uint32_t m = (uint32_t)(item / nbatch);
        msbfs_item(V, in_offs, in_cols, region, num_src, src, masks[m], reach, W, m,
                   (uint32_t)(item % nbatch) * 64, s_vis, s_allow);
        __syncthreads();
    }
}

// The dynamic shared-memory limits of the three block-wide kernels are
// process-wide settings per device.  They are raised once per device to the
// largest size any call can ask for (under a mutex), so that no call lowers
// the limit between another thread's setting and launch.
constexpr int kSmemAttrMaxDevices = 64;
std::mutex g_smem_attr_mutex;
bool g_smem_attr_set[kSmemAttrMaxDevices] = {};

cudaError_t reach_smem_limits() {
    int dev = 0, optin = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= kSmemAttrMaxDevices) return cudaErrorInvalidDevice;
    std::lock_guard<std::mutex> lock(g_smem_attr_mutex);
    if (g_smem_attr_set[dev]) return cudaSuccess;
    e = cudaDeviceGetAttribute(&optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev);
    if (e != cudaSuccess) return e;
    const int rows_max = optin - 1024;
    const int lab_max = (int)LabelSmem(kReachMaxV).total;
    const int bfs_max = (int)(kReachMaxV * 8);
    if ((e = cudaFuncSetAttribute(reach_rows_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, rows_max)) !=
            cudaSuccess ||
        (e = cudaFuncSetAttribute(reach_labels_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                  std::min(lab_max, rows_max))) != cudaSuccess ||
        (e = cudaFuncSetAttribute(reach_msbfs_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                  std::min(bfs_max, rows_max))) != cudaSuccess)
        return e;
    g_smem_attr_set[dev] = true;
    return cudaSuccess;
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
    const size_t o_pairs = o_cols + align256((size_t)num_edges * 4 + 4);   // undirected pairs (+ count)
    const size_t o_lab = o_pairs + align256((size_t)num_edges * 4 + 16) + 256;   // component labels
    const bool comp = ctx->opt_reach == 0;
    const size_t total = o_lab + (comp ? align256((size_t)num_masks * V * 2) : 0);
    uint8_t *base = (uint8_t *)pv_scratch(ctx, total);
    if (!base) return PV_ENOMEM;
    uint32_t *indeg = (uint32_t *)(base + o_indeg), *in_offs = (uint32_t *)(base + o_in_offs);
    uint32_t *cursor = (uint32_t *)(base + o_cursor), *in_cols = (uint32_t *)(base + o_cols);
    uint32_t *pairs = (uint32_t *)(base + o_pairs);
    uint32_t *npairs = (uint32_t *)(base + o_pairs + align256((size_t)num_edges * 4 + 16));
    cudaStream_t st = (cudaStream_t)stream;
    // component path: row-slot cache sized to keep 3 blocks per SM when the
    // fixed part allows it, at least one slot otherwise, none if even that
    // does not fit (rows then come straight from the ballots)
    uint32_t cap = 0;
    size_t rows_smem = 0;
    const size_t lab_smem = LabelSmem(V).total;
    const size_t limit = ctx->max_smem_optin - 1024;
    if (comp) {
        const size_t fixed = RowSmem(V, words_per_row, 0).total;
        const size_t row = (size_t)words_per_row * 4 + 4;
        const size_t budget = std::max<size_t>(72 * 1024, fixed + 16 * row);
        if (fixed + row <= limit) cap = (uint32_t)std::min<size_t>((std::min(budget, limit) - fixed) / row, 0xFFF0);
        rows_smem = RowSmem(V, words_per_row, cap).total;
        if (rows_smem > limit) {
            cap = 0;
            rows_smem = RowSmem(V, words_per_row, 0).total;
        }
        if (rows_smem > limit) return pv_fail(ctx, PV_EINVAL, "pv_compliant_reach: words_per_row too large");
    }
    uint16_t *lab = (uint16_t *)(base + o_lab);   // [num_masks][V] (component path only)
    PV_TRY_CUDA(ctx, reach_smem_limits(), "reach shared-memory limits");
    if (comp && !ctx->reach_side) {   // first call: the sweep path's side stream
        PV_TRY_CUDA(ctx, cudaStreamCreateWithFlags(&ctx->reach_side, cudaStreamNonBlocking), "reach side stream");
        PV_TRY_CUDA(ctx, cudaEventCreateWithFlags(&ctx->reach_fork, cudaEventDisableTiming), "reach fork event");
        PV_TRY_CUDA(ctx, cudaEventCreateWithFlags(&ctx->reach_join, cudaEventDisableTiming), "reach join event");
    }
    PV_TRY_CUDA(ctx, cudaMemsetAsync(indeg, 0, (size_t)(V + 1) * 4, st), "indeg clear");
    if (comp) {
        PV_TRY_CUDA(ctx, cudaMemsetAsync(ctx->d_reach_asym, 0, 4, st), "symmetry flag clear");
        PV_TRY_CUDA(ctx, cudaMemsetAsync(npairs, 0, 4, st), "pair count clear");
    }
    ctx->last_reach_comp = comp;
    const uint32_t *sym_flag = comp ? ctx->d_reach_asym : nullptr;
    const uint32_t grid = std::min<uint32_t>((V + kGridThreads - 1) / kGridThreads, (uint32_t)ctx->num_sms * 8);
    const int pr = pv_prof_start(ctx, st, PV_K_REACH);
    uint32_t launches = 4;
    reach_indeg_kernel<<<grid, kGridThreads, 0, st>>>(V, num_edges, d_offs, d_cols, d_region, indeg, ctx->d_status);
    if (comp) {
        const uint32_t wgrid = std::min<uint32_t>((V + kGridThreads / 32 - 1) / (kGridThreads / 32),
                                                  (uint32_t)ctx->num_sms * 8);
        reach_symcheck_kernel<<<wgrid, kGridThreads, 0, st>>>(V, num_edges, d_offs, d_cols, ctx->d_reach_asym, pairs,
                                                              npairs, indeg + V);
        launches += 3;
        // Both paths are launched and the symmetry flag picks the one that
        // works: on the component path's calls the sweep path's kernels go to
        // the side stream (they need only the in-degrees and the flag), so
        // their launches overlap the labels and rows kernels instead of
        // queueing behind them; the caller's stream joins it at the end.
        PV_TRY_CUDA(ctx, cudaEventRecord(ctx->reach_fork, st), "reach fork");
        PV_TRY_CUDA(ctx, cudaStreamWaitEvent(ctx->reach_side, ctx->reach_fork, 0), "reach fork");
    }
    cudaStream_t sw = comp ? ctx->reach_side : st;   // the sweep path's stream
    reach_scan_kernel<<<1, 1024, 0, sw>>>(V, indeg, in_offs, cursor, sym_flag);
    reach_fill_kernel<<<grid, kGridThreads, 0, sw>>>(V, num_edges, d_offs, d_cols, cursor, in_cols, sym_flag,
                                                     indeg + V);
    if (comp) {
        reach_labels_kernel<<<num_masks, kLabelThreads, lab_smem, st>>>(V, pairs, npairs, d_region, d_masks, lab,
                                                                         ctx->d_reach_asym, ctx->d_status);
        int per_sm = 1;
        cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, reach_rows_kernel, kCompThreads, rows_smem);
        // one wave of resident blocks over masks x source slices
        const uint64_t want = (uint64_t)std::max(per_sm, 1) * ctx->num_sms;
        const uint32_t slices = (uint32_t)std::max<uint64_t>(1, std::min<uint64_t>(num_src, want / num_masks));
        const uint32_t spb = (num_src + slices - 1) / slices;
        dim3 gc((num_src + spb - 1) / spb, num_masks);
        reach_rows_kernel<<<gc, kCompThreads, rows_smem, st>>>(V, lab, num_src, d_src, d_reach, words_per_row, spb,
                                                               cap, ctx->d_reach_asym);
    }
    const size_t smem = (size_t)V * 8;
    int bfs_per_sm = 1;
    cudaOccupancyMaxActiveBlocksPerMultiprocessor(&bfs_per_sm, reach_msbfs_kernel, kReachThreads, smem);
    const uint64_t items = (uint64_t)((num_src + 63) / 64) * num_masks;
    const uint32_t g2 = (uint32_t)std::min<uint64_t>(items, (uint64_t)std::max(bfs_per_sm, 1) * ctx->num_sms);
    reach_msbfs_kernel<<<g2, kReachThreads, smem, sw>>>(V, in_offs, in_cols, d_region, num_src, d_src, num_masks,
                                                       d_masks, d_reach, words_per_row,
                                                       comp ? ctx->d_reach_asym : nullptr);
    if (comp) {
        PV_TRY_CUDA(ctx, cudaEventRecord(ctx->reach_join, ctx->reach_side), "reach join");
        PV_TRY_CUDA(ctx, cudaStreamWaitEvent(st, ctx->reach_join, 0), "reach join");
    }
    pv_prof_stop(ctx, st, pr, launches);
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
// per device (in host code the array's name is not a device address) and
// kept for the life of the process: after a cudaDeviceReset the module is
// loaded again and the kept address would be stale, so the library is not
// to be used on a device after a reset.
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
    reach_scan_kernel<<<1, 1024, 0, st>>>(V, indeg, in_offs, cursor, nullptr);
    reach_fill_kernel<<<grid, kGridThreads, 0, st>>>(V, num_edges, d_offs, d_cols, cursor, in_cols, nullptr,
                                                     indeg + V);
    const size_t smem = (size_t)V * 8;
    if (reach_smem_limits() != cudaSuccess) return PV_ECUDA;
    const uint64_t items = (uint64_t)((num_src + 63) / 64) * num_masks;
    const uint32_t g2 = (uint32_t)std::min<uint64_t>(items, (uint64_t)sms * 4);
    reach_msbfs_kernel<<<g2, kReachThreads, smem, st>>>(V, in_offs, in_cols, d_region, num_src, d_src, num_masks,
                                                       d_masks, d_reach, words_per_row, nullptr);
    return cudaGetLastError() == cudaSuccess ? PV_OK : PV_ECUDA;
}
