// Placement constraints Phi_C: node-label loading and batched node-selector
// evaluation (Sec. 3.3 satisfaction (i); Sec. 4.1 placement directives;
// Sec. 5.5 compute check; Sec. 6.3 hallucinated identifiers; Sec. 5.3
// fail-closed unenforceable intents).
//
// Two exact kernels compute the same feasible-node bitsets:
//  * sel_cmp_kernel: label columns of a node tile are staged in shared
//    memory; a warp per pod sweeps 32 nodes at a time, tests each
//    expression against the node's value and emits one bitset word per
//    sweep with __ballot_sync.
//  * sel_rows_kernel: pv_load_cluster builds, for every (key, carried
//    value), the bitset of nodes carrying it, plus one "key present" row
//    per key.  An In expression is then the OR of its values' rows, NotIn
//    its complement, Exists / DoesNotExist the present row or its
//    complement, and a pod's row the AND over its expressions -- 32 nodes
//    per word operation, rows read from L2 with 128-bit loads.
#include <cuda_runtime.h>

#include <algorithm>
#include <vector>

#include "pv_internal.cuh"

namespace {

constexpr uint32_t kInvWords = 2048;                  // 65536 value ids / 32
constexpr uint64_t kRowBudgetBytes = 2ull << 30;      // value-row memory budget
constexpr uint32_t kMaxKeys = 4096;

__host__ __device__ inline uint32_t words_for(uint32_t n) { return ((n + 127) / 128) * 4; }

// ---------------------------------------------------------------------------
// loading
// ---------------------------------------------------------------------------
__global__ void build_inventory_kernel(uint32_t N, uint32_t K, const uint16_t *__restrict__ labels,
                                       uint32_t *__restrict__ inv) {
    size_t total = (size_t)N * K;
    for (size_t i = blockIdx.x * (size_t)blockDim.x + threadIdx.x; i < total; i += (size_t)gridDim.x * blockDim.x) {
        uint32_t k = (uint32_t)(i / N);
        uint16_t v = labels[i];
        if (v != PV_ABSENT) atomicOr(&inv[(size_t)k * kInvWords + (v >> 5)], 1u << (v & 31));
    }
}

// One block (1024 threads) per key: exclusive prefix popcount over the key's
// 2048 inventory words; count[k] = number of carried values.
__global__ void __launch_bounds__(1024) inventory_rank_kernel(const uint32_t *__restrict__ inv,
                                                              uint32_t *__restrict__ rank,
                                                              uint32_t *__restrict__ count) {
    __shared__ uint32_t s_warp[32];
    const uint32_t k = blockIdx.x, t = threadIdx.x, lane = t & 31, warp = t >> 5;
    const uint32_t *w = inv + (size_t)k * kInvWords;
    uint32_t a = __popc(w[2 * t]), b = __popc(w[2 * t + 1]);
    uint32_t x = a + b, incl = x;
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
        if (lane == 31) count[k] = vi;
    }
    __syncthreads();
    uint32_t excl = s_warp[warp] + incl - x;
    rank[(size_t)k * kInvWords + 2 * t] = excl;
    rank[(size_t)k * kInvWords + 2 * t + 1] = excl + a;
}

// Single block: key_base = exclusive scan of count[0..K), key_base[K] = total.
__global__ void __launch_bounds__(1024) key_base_kernel(uint32_t K, const uint32_t *__restrict__ count,
                                                        uint32_t *__restrict__ base) {
    __shared__ uint32_t s_carry;
    __shared__ uint32_t s_warp[32];
    const uint32_t t = threadIdx.x, lane = t & 31, warp = t >> 5;
    if (t == 0) s_carry = 0;
    __syncthreads();
    for (uint32_t c0 = 0; c0 < K; c0 += 1024) {
        uint32_t i = c0 + t;
        uint32_t x = i < K ? count[i] : 0, incl = x;
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
        uint32_t excl = s_carry + s_warp[warp] + incl - x;
        if (i < K) base[i] = excl;
        __syncthreads();
        if (t == 1023) s_carry = excl + x;
        __syncthreads();
    }
    if (t == 0) base[K] = s_carry;
}

__device__ __forceinline__ uint32_t value_row(const uint32_t *__restrict__ inv, const uint32_t *__restrict__ rank,
                                              const uint32_t *__restrict__ key_base, uint32_t k, uint32_t v,
                                              bool *carried) {
    uint32_t w = inv[(size_t)k * kInvWords + (v >> 5)];
    uint32_t bit = v & 31;
    *carried = (w >> bit) & 1u;
    return key_base[k] + rank[(size_t)k * kInvWords + (v >> 5)] + __popc(w & ((1u << bit) - 1u));
}

// Value rows and present rows.  One warp covers 32 consecutive nodes of one
// key; present rows are written with a ballot, value rows with atomicOr.
__global__ void build_rows_kernel(uint32_t N, uint32_t K, const uint16_t *__restrict__ labels,
                                  const uint32_t *__restrict__ inv, const uint32_t *__restrict__ rank,
                                  const uint32_t *__restrict__ key_base, uint32_t num_value_rows,
                                  uint32_t row_words, uint32_t *__restrict__ rows) {
    const uint32_t lane = threadIdx.x & 31;
    const uint32_t words = (N + 31) / 32;
    const size_t total_warps = (size_t)K * words;
    const size_t gw = (blockIdx.x * (size_t)blockDim.x + threadIdx.x) >> 5;
    const size_t nw = ((size_t)gridDim.x * blockDim.x) >> 5;
    for (size_t i = gw; i < total_warps; i += nw) {
        uint32_t k = (uint32_t)(i / words), wd = (uint32_t)(i % words);
        uint32_t n = wd * 32 + lane;
        uint16_t v = n < N ? labels[(size_t)k * N + n] : (uint16_t)PV_ABSENT;
        uint32_t pres = __ballot_sync(PV_FULL_MASK, v != PV_ABSENT);
        if (lane == 0) rows[((size_t)num_value_rows + k) * row_words + wd] = pres;
        if (v != PV_ABSENT) {
            bool carried;
            uint32_t r = value_row(inv, rank, key_base, k, v, &carried);
            atomicOr(&rows[(size_t)r * row_words + wd], 1u << lane);
        }
    }
}

// ---------------------------------------------------------------------------
// expression checks shared by both kernels
// ---------------------------------------------------------------------------
__device__ __forceinline__ bool expr_valid(const pv_expr &x, uint32_t K) {
    if (x.key >= K) return false;
    if (x.op == PV_IN || x.op == PV_NOTIN) {
        if (x.nvals < 1 || x.nvals > 8) return false;
        for (int j = 0; j < 8; ++j)
            if (j < x.nvals && x.vals[j] == PV_ABSENT) return false;
        return true;
    }
    if (x.op == PV_EXISTS || x.op == PV_DOESNOTEXIST) return x.nvals == 0;
    return false;
}

// Lane-parallel validation and hallucinated-value scan of pod p's list.
// Returns bit0 = bad, bit1 = unknown value.
__device__ __forceinline__ uint32_t pod_prescan(uint32_t lo, uint32_t hi, uint32_t num_exprs,
                                                const pv_expr *__restrict__ exprs, uint32_t K,
                                                const uint32_t *__restrict__ inv, uint32_t lane) {
    bool bad = hi < lo || hi > num_exprs;
    bool unknown = false;
    if (!bad) {
        for (uint32_t e = lo + lane; e < hi; e += 32) {
            pv_expr x = exprs[e];
            if (!expr_valid(x, K)) {
                bad = true;
                continue;
            }
            if (x.op == PV_IN)
                for (int j = 0; j < 8; ++j)
                    if (j < x.nvals) {
                        uint32_t v = x.vals[j];
                        if (!((inv[(size_t)x.key * kInvWords + (v >> 5)] >> (v & 31)) & 1u)) unknown = true;
                    }
        }
    }
    bad = __any_sync(PV_FULL_MASK, bad);
    unknown = __any_sync(PV_FULL_MASK, unknown);
    return (bad ? 1u : 0u) | (unknown ? 2u : 0u);
}

__device__ __forceinline__ uint8_t pod_flags(bool nonempty, bool unknown, bool has_assign, bool assign_ok) {
    uint8_t f = 0;
    if (!nonempty) f |= PV_F_EMPTY;
    if (unknown) f |= PV_F_UNKNOWN_VALUE;
    if (has_assign && assign_ok) {
        f |= PV_F_ASSIGN_OK;
        if (!unknown) f |= PV_F_PASS;
    }
    return f;
}

// ---------------------------------------------------------------------------
// kernel 1: per-node comparison over shared-memory label tiles
// ---------------------------------------------------------------------------
constexpr int kCmpThreads = 512;
constexpr int kCmpWarps = kCmpThreads / 32;
constexpr int kCmpPods = 128;   // pods per block
constexpr int kCmpCache = 8;    // expressions cached per warp

__global__ void __launch_bounds__(kCmpThreads) sel_cmp_kernel(
    uint32_t N, uint32_t K, const uint16_t *__restrict__ labels, uint32_t tile, uint32_t P,
    const uint32_t *__restrict__ offs, uint32_t num_exprs, const pv_expr *__restrict__ exprs,
    const uint32_t *__restrict__ assign, uint32_t *__restrict__ bits, uint32_t W, uint8_t *__restrict__ flags,
    const uint32_t *__restrict__ inv, const uint32_t *__restrict__ rep_of) {
    extern __shared__ uint16_t s_lab[];   // [K][tile]
    __shared__ uint8_t s_state[kCmpPods]; // bit0 nonempty, bit1 assign ok, bit2 bad, bit3 unknown
    __shared__ pv_expr s_ex[kCmpWarps][kCmpCache];
    const uint32_t lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const uint32_t p0 = blockIdx.x * kCmpPods;
    if (p0 >= P) return;
    const uint32_t np = min((uint32_t)kCmpPods, P - p0);
    const uint32_t nvalid_words = (N + 31) / 32;

    // per-pod validation / unknown scan (warp per pod)
    for (uint32_t pl = warp; pl < np; pl += kCmpWarps) {
        uint32_t p = p0 + pl;
        if (rep_of && rep_of[p] != p) continue;   // a duplicate: sel_copy_kernel writes it
        uint32_t r = pod_prescan(offs[p], offs[p + 1], num_exprs, exprs, K, inv, lane);
        if (lane == 0) s_state[pl] = (uint8_t)(((r & 1u) ? 4u : 0u) | ((r & 2u) ? 8u : 0u));
    }

    for (uint32_t n0 = 0; n0 < N; n0 += tile) {
        const uint32_t tn = min(tile, N - n0);
        __syncthreads();
        for (uint32_t i = threadIdx.x; i < K * tile; i += kCmpThreads) {
            uint32_t k = i / tile, j = i - k * tile;
            s_lab[i] = j < tn ? labels[(size_t)k * N + n0 + j] : (uint16_t)PV_ABSENT;
        }
        __syncthreads();
        const uint32_t groups = (tn + 31) / 32;
        for (uint32_t pl = warp; pl < np; pl += kCmpWarps) {
            const uint32_t p = p0 + pl;
            if (rep_of && rep_of[p] != p) continue;
            const uint8_t st = s_state[pl];
            uint32_t *row = bits + (size_t)p * W + (n0 >> 5);
            if (st & 4u) {
                for (uint32_t g = lane; g < groups; g += 32) row[g] = 0;
                continue;
            }
            const uint32_t lo = offs[p], E = offs[p + 1] - lo;
            const bool cached = E <= (uint32_t)kCmpCache;
            if (cached) {
                if (lane < E) s_ex[warp][lane] = exprs[lo + lane];
                __syncwarp();
            }
            const uint32_t a = assign ? assign[p] : PV_UNPLACED;
            bool any = false, aok = false;
            for (uint32_t gb = 0; gb < groups; gb += 32) {
                uint32_t mine = 0;
                const uint32_t gend = min(groups, gb + 32);
                for (uint32_t g = gb; g < gend; ++g) {
                    const uint32_t j = g * 32 + lane;   // node offset within the tile
                    bool ok = j < tn;
                    for (uint32_t e = 0; e < E; ++e) {
                        const pv_expr &x = cached ? s_ex[warp][e] : exprs[lo + e];
                        const uint16_t v = s_lab[(uint32_t)x.key * tile + j];
                        const bool present = v != PV_ABSENT;
                        bool inset = false;
                        const uint32_t nv = x.nvals;
                        for (uint32_t q = 0; q < nv; ++q) inset |= (v == x.vals[q]);
                        bool m;
                        switch (x.op) {
                        case PV_IN: m = present && inset; break;
                        case PV_NOTIN: m = !present || !inset; break;
                        case PV_EXISTS: m = present; break;
                        default: m = !present; break;
                        }
                        ok = ok && m;
                    }
                    const uint32_t w = __ballot_sync(PV_FULL_MASK, ok);
                    if (lane == g - gb) mine = w;
                    const uint32_t node_base = n0 + g * 32;
                    if (a >= node_base && a < node_base + 32) aok = (w >> (a - node_base)) & 1u;
                }
                if (lane < gend - gb) row[gb + lane] = mine;
                any = any || __any_sync(PV_FULL_MASK, mine != 0);
            }
            __syncwarp();
            if (lane == 0) s_state[pl] = st | (any ? 1u : 0u) | (aok ? 2u : 0u);
        }
    }
    __syncthreads();
    // padding words and flags
    for (uint32_t pl = warp; pl < np; pl += kCmpWarps) {
        const uint32_t p = p0 + pl;
        if (rep_of && rep_of[p] != p) continue;
        for (uint32_t w = nvalid_words + lane; w < W; w += 32) bits[(size_t)p * W + w] = 0;
        if (lane == 0) {
            const uint8_t st = s_state[pl];
            flags[p] = (st & 4u) ? (uint8_t)PV_F_BAD_EXPR
                                 : pod_flags(st & 1u, st & 8u, assign != nullptr, st & 2u);
        }
    }
}

// ---------------------------------------------------------------------------
// kernel 2: per-(key, value) node-bitset rows
// ---------------------------------------------------------------------------
constexpr int kRowsThreads = 256;

// Four words (128 nodes from word w0) of the node set matching expression x:
// In = OR of its values' rows, NotIn its complement, Exists the key's
// present row, DoesNotExist its complement.  Words past the rows read 0
// before the complement.
__device__ __forceinline__ uint4 expr_rows4(const pv_expr &x, uint32_t w0, bool in_rows,
                                            const uint32_t *__restrict__ inv, const uint32_t *__restrict__ rank,
                                            const uint32_t *__restrict__ key_base, const uint32_t *__restrict__ rows,
                                            uint32_t row_words, uint32_t num_value_rows) {
    const uint32_t k = x.key, op = x.op;
    uint4 r;
    if (op == PV_IN || op == PV_NOTIN) {
        r = make_uint4(0, 0, 0, 0);
        const uint32_t nv = x.nvals;
        for (uint32_t j = 0; j < nv; ++j) {
            bool carried;
            const uint32_t row = value_row(inv, rank, key_base, k, x.vals[j], &carried);
            if (carried && in_rows) {
                const uint4 v = __ldg(reinterpret_cast<const uint4 *>(rows + (size_t)row * row_words + w0));
                r.x |= v.x; r.y |= v.y; r.z |= v.z; r.w |= v.w;
            }
        }
    } else {
        r = in_rows ? __ldg(reinterpret_cast<const uint4 *>(rows + ((size_t)num_value_rows + k) * row_words + w0))
                    : make_uint4(0, 0, 0, 0);
    }
    if (op == PV_NOTIN || op == PV_DOESNOTEXIST) { r.x = ~r.x; r.y = ~r.y; r.z = ~r.z; r.w = ~r.w; }
    return r;
}

// A pod's expressions resolved once, one expression per lane (lists of at
// most 32): each lane validates its expression, flags In values that no
// node carries, and leaves the word offsets of the rows to OR (the key's
// present row for Exists / DoesNotExist) in the warp's shared slots.  The
// row sweep then reads only rows.  Returns bit0 = a bad expression, bit1 =
// an unknown value (as pod_prescan).
constexpr int kRowsWarps = kRowsThreads / 32;
struct ResolvedExprs {
    uint32_t meta[kRowsWarps][32];     // op | rows << 8
    uint32_t off[kRowsWarps][32][8];   // word offset of each row in the row array
    uint8_t order[kRowsWarps][32];     // evaluation order of the expressions (sel_rows_kernel)
};

template <bool kOrder>
__device__ __forceinline__ uint32_t resolve_exprs(ResolvedExprs &rx, uint32_t warp, uint32_t lane, uint32_t lo,
                                                  uint32_t E, const pv_expr *__restrict__ exprs, uint32_t K,
                                                  const uint32_t *__restrict__ inv, const uint32_t *__restrict__ rank,
                                                  const uint32_t *__restrict__ key_base, uint32_t num_value_rows,
                                                  uint32_t row_words) {
    bool bad = false, unknown = false;
    if (lane < E) {
        const pv_expr *xp = exprs + lo + lane;
        const uint32_t k = xp->key, op = xp->op, nv = xp->nvals;
        uint32_t n = 0;
        if (k >= K) {
            bad = true;
        } else if (op == PV_IN || op == PV_NOTIN) {
            bad = nv < 1 || nv > 8;
#pragma unroll
            for (uint32_t j = 0; j < 8; ++j) {
                if (j >= nv || bad) continue;
                const uint32_t v = xp->vals[j];
                if (v == PV_ABSENT) {
                    bad = true;
                    continue;
                }
                const uint32_t w = inv[(size_t)k * kInvWords + (v >> 5)], bit = v & 31;
                if ((w >> bit) & 1u) {
                    const uint32_t row = key_base[k] + rank[(size_t)k * kInvWords + (v >> 5)] +
                                         __popc(w & ((1u << bit) - 1u));
                    rx.off[warp][lane][n++] = row * row_words;
                } else if (op == PV_IN) {
                    unknown = true;
                }
            }
        } else if (op == PV_EXISTS || op == PV_DOESNOTEXIST) {
            bad = nv != 0;
            rx.off[warp][lane][n++] = (num_value_rows + k) * row_words;
        } else {
            bad = true;
        }
        rx.meta[warp][lane] = op | n << 8;
    }
    // Evaluation order (the AND of the expressions' sets does not depend on
    // it): In expressions with the fewest carried values first, then
    // DoesNotExist, Exists and NotIn, the sparsest sets first, so that a pod
    // whose row empties early stops reading rows.  Ties keep list order.
    uint32_t key = 0xFFFFFFFFu;
    if (kOrder && lane < E) {
        const uint32_t op = rx.meta[warp][lane] & 0xFFu, n = rx.meta[warp][lane] >> 8;
        const uint32_t cls = op == PV_IN ? 0u : op == PV_DOESNOTEXIST ? 1u : op == PV_EXISTS ? 2u : 3u;
        key = cls << 8 | n;
    }
    uint32_t place = 0;
    for (uint32_t j = 0; kOrder && j < E; ++j) {
        const uint32_t kj = __shfl_sync(PV_FULL_MASK, key, j);
        place += (kj < key || (kj == key && j < lane)) ? 1u : 0u;
    }
    if (kOrder && lane < E) rx.order[warp][place] = (uint8_t)lane;
    __syncwarp();
    bad = __any_sync(PV_FULL_MASK, bad);
    unknown = __any_sync(PV_FULL_MASK, unknown);
    return (bad ? 1u : 0u) | (unknown ? 2u : 0u);
}

// The same resolution with one lane per (expression, value) slot: lanes
// 0 .. E - 1 read their expression's header word, a warp scan lays the
// slots out (an In or NotIn expression takes one slot per listed value,
// any other one slot), and every slot's lane resolves its value's row in
// one step.  For lists of at most 32 slots (returns bit2 and resolves
// nothing when there are more).  Same results, flags and order as
// resolve_exprs<true>.
__device__ __forceinline__ uint32_t expr_header(const pv_expr *__restrict__ exprs, uint32_t lo, uint32_t lane) {
    return __ldg(reinterpret_cast<const uint32_t *>(exprs + lo + lane));
}

__device__ __forceinline__ uint32_t resolve_slots(ResolvedExprs &rx, uint32_t warp, uint32_t lane, uint32_t lo,
                                                  uint32_t E, const pv_expr *__restrict__ exprs, uint32_t K,
                                                  const uint32_t *__restrict__ inv, const uint32_t *__restrict__ rank,
                                                  const uint32_t *__restrict__ key_base, uint32_t num_value_rows,
                                                  uint32_t row_words, uint32_t lane_hdr) {
    // header word (expr_header, fetched by the caller): key (bits 0..15),
    // op (16..23), nvals (24..31)
    uint32_t hdr = 0, m = 0;
    bool bad = false;
    if (lane < E) {
        hdr = lane_hdr;
        const uint32_t k = hdr & 0xFFFFu, op = (hdr >> 16) & 0xFFu, nv = hdr >> 24;
        const bool listed = op == PV_IN || op == PV_NOTIN;
        bad = k >= K || (listed ? (nv < 1 || nv > 8) : (op == PV_EXISTS || op == PV_DOESNOTEXIST) ? nv != 0 : true);
        m = (listed && !bad) ? nv : 1u;
    }
    uint32_t incl = m;   // slots of expressions 0 .. lane
    for (int d = 1; d < 32; d <<= 1) {
        const uint32_t y = __shfl_up_sync(PV_FULL_MASK, incl, d);
        if (lane >= (uint32_t)d) incl += y;
    }
    const uint32_t T = __shfl_sync(PV_FULL_MASK, incl, 31);
    if (T > 32) return 4u;
    const uint32_t pre = incl - m;
    const uint32_t starts = __reduce_or_sync(PV_FULL_MASK, lane < E ? 1u << pre : 0u);
    // slot lane: expression e, value j
    const uint32_t upto = lane == 31 ? ~0u : (2u << lane) - 1u;
    const uint32_t e = lane < T ? (uint32_t)__popc(starts & upto) - 1u : 0u;
    const uint32_t pre_e = __shfl_sync(PV_FULL_MASK, pre, e);
    const uint32_t hdr_e = __shfl_sync(PV_FULL_MASK, hdr, e);
    const uint32_t m_e = __shfl_sync(PV_FULL_MASK, m, e);
    const bool bad_e = __shfl_sync(PV_FULL_MASK, bad ? 1u : 0u, e) != 0;
    const uint32_t k = hdr_e & 0xFFFFu, op = (hdr_e >> 16) & 0xFFu;
    bool carried = false, unknown = false;
    uint32_t off = 0;
    if (lane < T && !bad_e) {
        if (op == PV_IN || op == PV_NOTIN) {
            const uint32_t v = __ldg(&exprs[lo + e].vals[lane - pre_e]);
            if (v == PV_ABSENT) {
                bad = true;
            } else {
                const uint32_t w = __ldg(inv + (size_t)k * kInvWords + (v >> 5)), bit = v & 31;
                carried = (w >> bit) & 1u;
                if (carried)
                    off = (__ldg(key_base + k) + __ldg(rank + (size_t)k * kInvWords + (v >> 5)) +
                           __popc(w & ((1u << bit) - 1u))) * row_words;
                else if (op == PV_IN)
                    unknown = true;
            }
        } else {
            carried = true;
            off = (num_value_rows + k) * row_words;
        }
    }
    // carried rows of each expression, packed in slot order
    const uint32_t C = __ballot_sync(PV_FULL_MASK, carried);
    const uint32_t below = (1u << lane) - 1u;
    if (carried) rx.off[warp][e][__popc(C & below & ~((1u << pre_e) - 1u))] = off;
    uint32_t key = 0xFFFFFFFFu;
    if (lane < E) {
        const uint32_t span = (m >= 32 ? ~0u : (1u << m) - 1u) << pre;
        const uint32_t n = __popc(C & span), opl = (hdr >> 16) & 0xFFu;
        rx.meta[warp][lane] = opl | n << 8;
        const uint32_t cls = opl == PV_IN ? 0u : opl == PV_DOESNOTEXIST ? 1u : opl == PV_EXISTS ? 2u : 3u;
        key = cls << 8 | n;
    }
    (void)m_e;
    uint32_t place = 0;
    for (uint32_t j = 0; j < E; ++j) {
        const uint32_t kj = __shfl_sync(PV_FULL_MASK, key, j);
        place += (kj < key || (kj == key && j < lane)) ? 1u : 0u;
    }
    if (lane < E) rx.order[warp][place] = (uint8_t)lane;
    __syncwarp();
    bad = __any_sync(PV_FULL_MASK, bad);
    unknown = __any_sync(PV_FULL_MASK, unknown);
    return (bad ? 1u : 0u) | (unknown ? 2u : 0u);
}

// ANDs resolved expression e's node set into a 160-word span's accumulators
// of one lane: chunk q (four words, loaded when l0) and word w (loaded when
// l1); words past the rows read 0 before the complement.
__device__ __forceinline__ void and_resolved5(const ResolvedExprs &rx, uint32_t warp, uint32_t e,
                                              const uint32_t *__restrict__ rows, uint32_t q, uint32_t w, bool l0,
                                              bool l1, uint4 &a0, uint32_t &a1) {
    const uint32_t meta = rx.meta[warp][e], op = meta & 0xFFu, n = meta >> 8;
    uint4 v0 = make_uint4(0, 0, 0, 0);
    uint32_t v1 = 0;
    uint32_t j = 0;
    for (; j + 1 < n; j += 2) {   // two rows per step: four loads in flight
        const uint32_t *rp = rows + rx.off[warp][e][j], *rq = rows + rx.off[warp][e][j + 1];
        uint4 x0 = make_uint4(0, 0, 0, 0), y0 = x0;
        uint32_t x1 = 0, y1 = 0;
        if (l0) {
            x0 = __ldg(reinterpret_cast<const uint4 *>(rp) + q);
            y0 = __ldg(reinterpret_cast<const uint4 *>(rq) + q);
        }
        if (l1) {
            x1 = __ldg(rp + w);
            y1 = __ldg(rq + w);
        }
        v0.x |= x0.x | y0.x; v0.y |= x0.y | y0.y; v0.z |= x0.z | y0.z; v0.w |= x0.w | y0.w;
        v1 |= x1 | y1;
    }
    if (j < n) {
        const uint32_t *rp = rows + rx.off[warp][e][j];
        if (l0) {
            const uint4 x = __ldg(reinterpret_cast<const uint4 *>(rp) + q);
            v0.x |= x.x; v0.y |= x.y; v0.z |= x.z; v0.w |= x.w;
        }
        if (l1) v1 |= __ldg(rp + w);
    }
    if (op == PV_NOTIN || op == PV_DOESNOTEXIST) {
        a0.x &= ~v0.x; a0.y &= ~v0.y; a0.z &= ~v0.z; a0.w &= ~v0.w;
        a1 &= ~v1;
    } else {
        a0.x &= v0.x; a0.y &= v0.y; a0.z &= v0.z; a0.w &= v0.w;
        a1 &= v1;
    }
}

// Clears the bits of nodes >= N in the four words from w0.
__device__ __forceinline__ void clip_rows4(uint4 &acc, uint32_t w0, uint32_t N) {
    const uint32_t full_words = N >> 5, tail_bits = N & 31;
    uint32_t *aw = &acc.x;
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const uint32_t w = w0 + i;
        if (w > full_words || (w == full_words && tail_bits == 0)) aw[i] = 0;
        else if (w == full_words) aw[i] &= (1u << tail_bits) - 1u;
    }
}

__global__ void __launch_bounds__(kRowsThreads) sel_rows_kernel(
    uint32_t N, uint32_t K, uint32_t P, const uint32_t *__restrict__ offs, uint32_t num_exprs,
    const pv_expr *__restrict__ exprs, const uint32_t *__restrict__ assign, uint32_t *__restrict__ bits,
    uint32_t W, uint8_t *__restrict__ flags, const uint32_t *__restrict__ inv, const uint32_t *__restrict__ rank,
    const uint32_t *__restrict__ key_base, const uint32_t *__restrict__ rows, uint32_t row_words,
    uint32_t num_value_rows, const uint32_t *__restrict__ pod_list, const uint32_t *__restrict__ list_len) {
    __shared__ ResolvedExprs rx;
    const uint32_t lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const uint32_t gw = (blockIdx.x * kRowsThreads + threadIdx.x) >> 5;
    const uint32_t nw = (gridDim.x * kRowsThreads) >> 5;
    const uint32_t n = pod_list ? *list_len : P;   // with a list: only the pods it names
    // The next pod's offsets are loaded while this pod is resolved, and its
    // expression headers while this pod's rows are swept, so a pod's chain
    // of dependent loads starts at its values.
    auto pod_at = [&](uint32_t i) { return pod_list ? pod_list[i] : i; };
    auto headed = [&](uint32_t lo, uint32_t hi) { return hi >= lo && hi <= num_exprs && hi - lo <= 32; };
    uint32_t p = 0, lo = 0, hi = 0, hdr = 0;
    if (gw < n) {
        p = pod_at(gw);
        lo = offs[p];
        hi = offs[p + 1];
        hdr = headed(lo, hi) && lane < hi - lo ? expr_header(exprs, lo, lane) : 0u;
    }
    for (uint32_t i = gw; i < n; i += nw) {
        uint32_t np = 0, nlo = 0, nhi = 0;
        if (i + nw < n) {
            np = pod_at(i + nw);
            nlo = offs[np];
            nhi = offs[np + 1];
        }
        const uint32_t a = assign ? assign[p] : PV_UNPLACED;
        const uint32_t E = hi - lo;
        const bool resolved = headed(lo, hi);
        uint32_t pre = resolved ? resolve_slots(rx, warp, lane, lo, E, exprs, K, inv, rank, key_base, num_value_rows,
                                                row_words, hdr)
                                : pod_prescan(lo, hi, num_exprs, exprs, K, inv, lane);
        if (resolved && (pre & 4u))   // more than 32 slots: one lane per expression
            pre = resolve_exprs<true>(rx, warp, lane, lo, E, exprs, K, inv, rank, key_base, num_value_rows,
                                      row_words);
        const uint32_t nhdr = i + nw < n && headed(nlo, nhi) && lane < nhi - nlo ? expr_header(exprs, nlo, lane) : 0u;
        uint4 *out = reinterpret_cast<uint4 *>(bits + (size_t)p * W);
        const uint32_t pc = p, lc = lo;   // this pod (the names below move on to the next one)
        p = np;
        lo = nlo;
        hi = nhi;
        hdr = nhdr;
        if (pre & 1u) {
            for (uint32_t q = lane; q < W / 4; q += 32) out[q] = make_uint4(0, 0, 0, 0);
            if (lane == 0) flags[pc] = PV_F_BAD_EXPR;
            continue;
        }
        bool any = false, aok = false;
        auto finish = [&](uint4 acc, uint32_t q) {
            const uint32_t w0 = q * 4;
            if (w0 + 4 > (N >> 5)) clip_rows4(acc, w0, N);   // only chunks reaching node N - 1 or past it
            out[q] = acc;
            any = any || (acc.x | acc.y | acc.z | acc.w) != 0;
            if (a < N && (a >> 7) == q) {   // the assigned node's word is in this chunk
                const uint32_t wsel = (a >> 5) & 3u;
                const uint32_t word = wsel == 0 ? acc.x : wsel == 1 ? acc.y : wsel == 2 ? acc.z : acc.w;
                aok = (word >> (a & 31)) & 1u;
            }
        };
        if (resolved) {
            // of each 160-word span a lane takes chunk lane (words 4 lane ..
            // 4 lane + 3) and word 128 + lane: five words per lane, so a row
            // of up to 5,120 nodes keeps every lane busy in one pass over the
            // resolved rows
            for (uint32_t sb = 0; sb < W; sb += 160) {
                const uint32_t q = sb / 4 + lane, w = sb + 128 + lane;
                const bool h0 = q * 4 < W, h1 = w < W;
                const bool l0 = h0 && q * 4 < row_words, l1 = h1 && w < row_words;
                uint4 a0 = make_uint4(~0u, ~0u, ~0u, ~0u);
                uint32_t a1 = ~0u;
                for (uint32_t i = 0; i < E; ++i) {
                    and_resolved5(rx, warp, rx.order[warp][i], rows, q, w, l0, l1, a0, a1);
                    // every node of the span rejected: the remaining sets
                    // cannot add any back (words past the rows hold no nodes)
                    const bool nz = (l0 && (a0.x | a0.y | a0.z | a0.w)) || (l1 && a1);
                    if (!__any_sync(PV_FULL_MASK, nz)) {
                        a0 = make_uint4(0, 0, 0, 0);
                        a1 = 0;
                        break;
                    }
                }
                if (h0) finish(a0, q);
                if (h1) {
                    const uint32_t full_words = N >> 5, tail_bits = N & 31;
                    if (w > full_words || (w == full_words && tail_bits == 0)) a1 = 0;
                    else if (w == full_words) a1 &= (1u << tail_bits) - 1u;
                    bits[(size_t)pc * W + w] = a1;
                    any = any || a1 != 0;
                    if (a < N && (a >> 5) == w) aok = (a1 >> (a & 31)) & 1u;
                }
            }
        } else {
            for (uint32_t q = lane; q < W / 4; q += 32) {
                const uint32_t w0 = q * 4;
                uint4 acc = make_uint4(~0u, ~0u, ~0u, ~0u);
                const bool in_rows = w0 < row_words;
                for (uint32_t e = 0; e < E; ++e) {
                    const uint4 r = expr_rows4(exprs[lc + e], w0, in_rows, inv, rank, key_base, rows, row_words,
                                               num_value_rows);
                    acc.x &= r.x; acc.y &= r.y; acc.z &= r.z; acc.w &= r.w;
                }
                finish(acc, q);
            }
        }
        any = __any_sync(PV_FULL_MASK, any);   // also keeps the warp's resolved rows until all lanes are done
        aok = __any_sync(PV_FULL_MASK, aok);
        if (lane == 0) flags[pc] = pod_flags(any, pre & 2u, assign != nullptr, aok);
    }
}

// Multi-term selectors (Kubernetes required node affinity): a pod's row is
// the OR over its terms of the AND over each term's expressions.  A pod
// without terms admits every node; a term without expressions matches none.
// Warp per pod; every term's list is validated and scanned for values no
// node carries, as in sel_rows_kernel.
__global__ void __launch_bounds__(kRowsThreads) sel_terms_kernel(
    uint32_t N, uint32_t K, uint32_t P, const uint32_t *__restrict__ pod_terms, uint32_t num_terms,
    const uint32_t *__restrict__ term_offs, uint32_t num_exprs, const pv_expr *__restrict__ exprs,
    const uint32_t *__restrict__ assign, uint32_t *__restrict__ bits, uint32_t W, uint8_t *__restrict__ flags,
    const uint32_t *__restrict__ inv, const uint32_t *__restrict__ rank, const uint32_t *__restrict__ key_base,
    const uint32_t *__restrict__ rows, uint32_t row_words, uint32_t num_value_rows) {
    __shared__ ResolvedExprs rx;
    const uint32_t lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const uint32_t gw = (blockIdx.x * kRowsThreads + threadIdx.x) >> 5;
    const uint32_t nw = (gridDim.x * kRowsThreads) >> 5;
    for (uint32_t p = gw; p < P; p += nw) {
        const uint32_t t0 = pod_terms[p], t1 = pod_terms[p + 1];
        uint32_t pre = (t1 < t0 || t1 > num_terms) ? 1u : 0u;
        // the terms' expressions form one range; lists of at most 32 are resolved once
        uint32_t e0 = 0, E = 0;
        bool resolved = false;
        if (!(pre & 1u) && t1 > t0) {
            e0 = term_offs[t0];
            const uint32_t e1 = term_offs[t1];
            bool mono = e1 >= e0;
            for (uint32_t t = t0; t < t1 && mono; ++t) mono = term_offs[t + 1] >= term_offs[t];
            resolved = mono && e1 <= num_exprs && e1 - e0 <= 32;
            E = resolved ? e1 - e0 : 0u;
        }
        if (resolved)
            pre |= resolve_exprs<false>(rx, warp, lane, e0, E, exprs, K, inv, rank, key_base, num_value_rows, row_words);
        else
            for (uint32_t t = t0; t < t1 && !(pre & 1u); ++t)
                pre |= pod_prescan(term_offs[t], term_offs[t + 1], num_exprs, exprs, K, inv, lane);
        uint4 *out = reinterpret_cast<uint4 *>(bits + (size_t)p * W);
        if (pre & 1u) {
            for (uint32_t q = lane; q < W / 4; q += 32) out[q] = make_uint4(0, 0, 0, 0);
            if (lane == 0) flags[p] = PV_F_BAD_EXPR;
            continue;
        }
        const uint32_t a = assign ? assign[p] : PV_UNPLACED;
        bool any = false, aok = false;
        auto finish = [&](uint4 res, uint32_t q) {
            const uint32_t w0 = q * 4;
            if (w0 + 4 > (N >> 5)) clip_rows4(res, w0, N);   // only chunks reaching node N - 1 or past it
            out[q] = res;
            any = any || (res.x | res.y | res.z | res.w) != 0;
            if (a < N && (a >> 7) == q) {   // the assigned node's word is in this chunk
                const uint32_t wsel = (a >> 5) & 3u;
                const uint32_t word = wsel == 0 ? res.x : wsel == 1 ? res.y : wsel == 2 ? res.z : res.w;
                aok = (word >> (a & 31)) & 1u;
            }
        };
        const uint4 none = make_uint4(0, 0, 0, 0), all = make_uint4(~0u, ~0u, ~0u, ~0u);
        if (resolved) {   // a 160-word span per pass, five words per lane, as in sel_rows_kernel
            for (uint32_t sb = 0; sb < W; sb += 160) {
                const uint32_t q = sb / 4 + lane, w = sb + 128 + lane;
                const bool h0 = q * 4 < W, h1 = w < W;
                const bool l0 = h0 && q * 4 < row_words, l1 = h1 && w < row_words;
                uint4 r0 = t0 == t1 ? all : none;
                uint32_t r1 = t0 == t1 ? ~0u : 0u;
                for (uint32_t t = t0; t < t1; ++t) {
                    const uint32_t lo = term_offs[t] - e0, hi = term_offs[t + 1] - e0;
                    uint4 a0 = hi > lo ? all : none;
                    uint32_t a1 = hi > lo ? ~0u : 0u;
                    for (uint32_t e = lo; e < hi; ++e) and_resolved5(rx, warp, e, rows, q, w, l0, l1, a0, a1);
                    r0.x |= a0.x; r0.y |= a0.y; r0.z |= a0.z; r0.w |= a0.w;
                    r1 |= a1;
                }
                if (h0) finish(r0, q);
                if (h1) {
                    const uint32_t full_words = N >> 5, tail_bits = N & 31;
                    if (w > full_words || (w == full_words && tail_bits == 0)) r1 = 0;
                    else if (w == full_words) r1 &= (1u << tail_bits) - 1u;
                    bits[(size_t)p * W + w] = r1;
                    any = any || r1 != 0;
                    if (a < N && (a >> 5) == w) aok = (r1 >> (a & 31)) & 1u;
                }
            }
        } else {
            for (uint32_t q = lane; q < W / 4; q += 32) {
                const uint32_t w0 = q * 4;
                const bool in_rows = w0 < row_words;
                uint4 res = t0 == t1 ? all : none;
                for (uint32_t t = t0; t < t1; ++t) {
                    const uint32_t lo = term_offs[t], hi = term_offs[t + 1];
                    uint4 acc = hi > lo ? all : none;
                    for (uint32_t e = lo; e < hi; ++e) {
                        const uint4 r = expr_rows4(exprs[e], w0, in_rows, inv, rank, key_base, rows, row_words,
                                                   num_value_rows);
                        acc.x &= r.x; acc.y &= r.y; acc.z &= r.z; acc.w &= r.w;
                    }
                    res.x |= acc.x; res.y |= acc.y; res.z |= acc.z; res.w |= acc.w;
                }
                finish(res, q);
            }
        }
        any = __any_sync(PV_FULL_MASK, any);
        aok = __any_sync(PV_FULL_MASK, aok);
        if (lane == 0) flags[p] = pod_flags(any, pre & 2u, assign != nullptr, aok);
    }
}

// ---------------------------------------------------------------------------
// identical selectors evaluated once (pods sharing an expression list, such
// as the replicas of one deployment, or intents with the same selector)
// ---------------------------------------------------------------------------
// A list's canonical form: per expression its key / operator / count word
// and its value words with the unused value slots zeroed (evaluation never
// reads them), so equal canonical lists give equal rows and flags.  Each
// pod's list is hashed (splitmix64's finalizer over the words, mixed with
// the expression's position) into an open-addressing table whose entries
// keep the smallest pod with that hash; every other pod with the hash is
// compared word by word with it, so a hash collision costs only an extra
// evaluation, never a wrong row.  Representatives are evaluated as usual;
// each duplicate then copies its representative's row and flags and redoes
// its own placement check.
__device__ __forceinline__ uint64_t mix64(uint64_t z) {
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
    z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
    return z ^ (z >> 31);
}

__device__ __forceinline__ void canon_expr(const pv_expr *x, uint32_t w[5]) {
    const uint32_t *raw = reinterpret_cast<const uint32_t *>(x);   // 20-byte records, 4-byte aligned
    w[0] = raw[0];
    const bool listed = (x->op == PV_IN || x->op == PV_NOTIN) && x->nvals <= 8;
    const uint32_t nv = listed ? x->nvals : 0u;
#pragma unroll
    for (uint32_t i = 0; i < 4; ++i) {
        const uint32_t v = raw[1 + i];
        w[1 + i] = (2 * i < nv ? (v & 0xFFFFu) : 0u) | (2 * i + 1 < nv ? (v & 0xFFFF0000u) : 0u);
    }
}

__device__ __forceinline__ uint64_t warp_sum64(uint64_t v) {
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(PV_FULL_MASK, v, o);
    return v;
}

// Warp per pod: hashes[p] (0 for a malformed range, which is never shared)
// and the pod's entry in the table (keys: hash, 0 = free; reps: smallest pod).
__global__ void __launch_bounds__(256) sel_hash_kernel(uint32_t P, const uint32_t *__restrict__ offs,
                                                       uint32_t num_exprs, const pv_expr *__restrict__ exprs,
                                                       unsigned long long *__restrict__ keys,
                                                       uint32_t *__restrict__ reps, uint32_t cap_mask,
                                                       uint32_t weak, unsigned long long *__restrict__ hashes) {
    const uint32_t lane = threadIdx.x & 31;
    const uint32_t gw = (blockIdx.x * blockDim.x + threadIdx.x) >> 5, nw = (gridDim.x * blockDim.x) >> 5;
    for (uint32_t p = gw; p < P; p += nw) {
        const uint32_t lo = offs[p], hi = offs[p + 1];
        if (hi < lo || hi > num_exprs) {
            if (lane == 0) hashes[p] = 0;
            continue;
        }
        const uint32_t E = hi - lo;
        uint64_t acc = 0;
        for (uint32_t e = lane; e < E; e += 32) {
            uint32_t w[5];
            canon_expr(exprs + lo + e, w);
            uint64_t h = mix64(((uint64_t)e << 32) ^ w[0]);
#pragma unroll
            for (uint32_t i = 1; i < 5; ++i) h = mix64(h ^ ((uint64_t)i << 40) ^ w[i]);
            acc += h;
        }
        acc = warp_sum64(acc);
        uint64_t h = mix64(acc ^ ((uint64_t)E * 0x9E3779B97F4A7C15ull)) | 1ull;
        if (weak) h = (h & 7ull) + 1ull;   // test mode: eight hash values, so most lists collide
        if (lane == 0) {
            hashes[p] = h;
            // popular lists share a slot: read first, and take an atomic only
            // to claim a free slot or to lower the slot's pod
            uint32_t slot = (uint32_t)(h * 0x9E3779B97F4A7C15ull >> 32) & cap_mask;
            for (uint32_t probe = 0; probe <= cap_mask; ++probe) {   // the table has room for every pod
                unsigned long long k = *(volatile unsigned long long *)(keys + slot);
                if (k == 0ull) k = atomicCAS(keys + slot, 0ull, (unsigned long long)h);
                if (k == 0ull || k == h) {
                    if (*(volatile uint32_t *)(reps + slot) > p) atomicMin(reps + slot, p);
                    break;
                }
                slot = (slot + 1) & cap_mask;
            }
        }
    }
}

// Warp per pod: rep_of[p] = the table's pod for p's hash when its canonical
// list equals p's, else p.
__global__ void __launch_bounds__(256) sel_rep_kernel(uint32_t P, const uint32_t *__restrict__ offs,
                                                      const pv_expr *__restrict__ exprs,
                                                      const unsigned long long *__restrict__ keys,
                                                      const uint32_t *__restrict__ reps, uint32_t cap_mask,
                                                      const unsigned long long *__restrict__ hashes,
                                                      uint32_t *__restrict__ rep_of, uint32_t *__restrict__ rep_list,
                                                      uint32_t *__restrict__ rep_count) {
    const uint32_t lane = threadIdx.x & 31;
    const uint32_t gw = (blockIdx.x * blockDim.x + threadIdx.x) >> 5, nw = (gridDim.x * blockDim.x) >> 5;
    for (uint32_t p = gw; p < P; p += nw) {
        const uint64_t h = hashes[p];
        uint32_t r = p;
        if (h != 0) {
            uint32_t slot = (uint32_t)(h * 0x9E3779B97F4A7C15ull >> 32) & cap_mask;
            for (uint32_t probe = 0; probe <= cap_mask && keys[slot] != h; ++probe) slot = (slot + 1) & cap_mask;
            r = keys[slot] == h ? reps[slot] : p;
        }
        if (r != p) {
            const uint32_t lo = offs[p], E = offs[p + 1] - lo, lr = offs[r], Er = offs[r + 1] - lr;
            bool same = E == Er;
            for (uint32_t e = lane; same && e < E; e += 32) {
                uint32_t a[5], b[5];
                canon_expr(exprs + lo + e, a);
                canon_expr(exprs + lr + e, b);
#pragma unroll
                for (int i = 0; i < 5; ++i) same = same && a[i] == b[i];
            }
            if (!__all_sync(PV_FULL_MASK, same)) r = p;
        }
        if (lane == 0) {
            rep_of[p] = r;
            if (r == p) rep_list[atomicAdd(rep_count, 1u)] = p;
        }
    }
}

// Warp per duplicate pod: its representative's row, flags without the
// placement bits, and its own placement check.
__global__ void __launch_bounds__(256) sel_copy_kernel(uint32_t P, uint32_t N, uint32_t W,
                                                       const uint32_t *__restrict__ rep_of,
                                                       const uint32_t *__restrict__ assign, uint32_t *__restrict__ bits,
                                                       uint8_t *__restrict__ flags) {
    const uint32_t lane = threadIdx.x & 31;
    const uint32_t gw = (blockIdx.x * blockDim.x + threadIdx.x) >> 5, nw = (gridDim.x * blockDim.x) >> 5;
    for (uint32_t p = gw; p < P; p += nw) {
        const uint32_t r = rep_of[p];
        if (r == p) continue;
        const uint4 *src = reinterpret_cast<const uint4 *>(bits + (size_t)r * W);
        uint4 *dst = reinterpret_cast<uint4 *>(bits + (size_t)p * W);
        for (uint32_t q = lane; q < W / 4; q += 32) dst[q] = src[q];
        if (lane == 0) {
            uint8_t f = flags[r] & (uint8_t)(PV_F_EMPTY | PV_F_UNKNOWN_VALUE | PV_F_BAD_EXPR);
            const uint32_t a = assign ? assign[p] : PV_UNPLACED;
            if (a < N && ((bits[(size_t)r * W + (a >> 5)] >> (a & 31)) & 1u)) {
                f |= PV_F_ASSIGN_OK;
                if (!(f & PV_F_UNKNOWN_VALUE)) f |= PV_F_PASS;
            }
            flags[p] = f;
        }
    }
}

}  // namespace

// -----------------------------------------------------------------------------
// C ABI
// -----------------------------------------------------------------------------
extern "C" int pv_load_cluster(pv_ctx *ctx, uint32_t num_nodes, uint32_t num_keys, const uint16_t *labels) {
    if (!ctx) return PV_EINVAL;
    if (num_nodes == 0 || num_keys == 0 || !labels)
        return pv_fail(ctx, PV_EINVAL, "pv_load_cluster: empty cluster or NULL labels");
    if (num_keys > kMaxKeys) return pv_fail(ctx, PV_EINVAL, "pv_load_cluster: num_keys > %u", kMaxKeys);
    if (int rc0 = pv_load_begin(ctx)) return rc0;
    cudaStream_t ls = ctx->load_stream;
    pv_cluster_state c;   // the new state (the loaded one stays in use until it is complete)
    const size_t nl = (size_t)num_nodes * num_keys;
    int rc;
    if ((rc = pv_pool_alloc(ctx, (void **)&c.d_labels, nl * 2, "labels")) ||
        (rc = pv_pool_alloc(ctx, (void **)&c.d_inv, (size_t)num_keys * kInvWords * 4, "inventory")) ||
        (rc = pv_pool_alloc(ctx, (void **)&c.d_inv_rank, (size_t)num_keys * kInvWords * 4, "inventory rank")) ||
        (rc = pv_pool_alloc(ctx, (void **)&c.d_key_base, ((size_t)num_keys + 1) * 4 * 2, "key base"))) {
        pv_free_cluster(ctx, c);
        return rc;
    }
    uint32_t *d_count = c.d_key_base + (num_keys + 1);
    PV_TRY_CUDA(ctx, cudaMemcpyAsync(c.d_labels, labels, nl * 2, cudaMemcpyHostToDevice, ls), "labels upload");
    PV_TRY_CUDA(ctx, cudaMemsetAsync(c.d_inv, 0, (size_t)num_keys * kInvWords * 4, ls), "inventory clear");
    build_inventory_kernel<<<ctx->num_sms * 8, 256, 0, ls>>>(num_nodes, num_keys, c.d_labels, c.d_inv);
    inventory_rank_kernel<<<num_keys, 1024, 0, ls>>>(c.d_inv, c.d_inv_rank, d_count);
    key_base_kernel<<<1, 1024, 0, ls>>>(num_keys, d_count, c.d_key_base);
    if ((rc = pv_check_launch(ctx, "inventory kernels"))) { pv_free_cluster(ctx, c); return rc; }
    uint32_t nvr = 0;
    cudaError_t e = cudaMemcpyAsync(&nvr, c.d_key_base + num_keys, 4, cudaMemcpyDeviceToHost, ls);
    if (e == cudaSuccess) e = cudaStreamSynchronize(ls);
    if (e != cudaSuccess) {
        pv_free_cluster(ctx, c);
        return pv_cuda_fail(ctx, e, "value count");
    }
    c.num_nodes = num_nodes;
    c.num_keys = num_keys;
    c.row_words = words_for(num_nodes);
    c.num_value_rows = nvr;
    const uint64_t row_bytes = ((uint64_t)nvr + num_keys) * c.row_words * 4;
    if (row_bytes <= kRowBudgetBytes) {
        if (pv_pool_alloc(ctx, (void **)&c.d_rows, row_bytes, "value rows") == PV_OK) {
            if ((e = cudaMemsetAsync(c.d_rows, 0, row_bytes, ls)) != cudaSuccess) {
                pv_free_cluster(ctx, c);
                return pv_cuda_fail(ctx, e, "value rows clear");
            }
            build_rows_kernel<<<ctx->num_sms * 8, 256, 0, ls>>>(num_nodes, num_keys, c.d_labels, c.d_inv, c.d_inv_rank,
                                                          c.d_key_base, nvr, c.row_words, c.d_rows);
            if ((rc = pv_check_launch(ctx, "value rows"))) { pv_free_cluster(ctx, c); return rc; }
            c.rows_built = true;
        } else {
            ctx->err.clear();   // rows are optional; fall back to the comparison kernel
        }
    }
    c.loaded = true;
    pv_retire_begin(ctx);
    pv_free_cluster(ctx, ctx->cl);
    pv_retire_end(ctx);
    ctx->cl = c;
    return pv_load_end(ctx);
}

extern "C" int pv_eval_selectors(pv_ctx *ctx, uint32_t num_pods, const uint32_t *d_expr_offs, uint32_t num_exprs,
                                 const pv_expr *d_exprs, const uint32_t *d_assign, uint32_t *d_bits,
                                 uint32_t words_per_row, uint8_t *d_flags, pv_stream stream) {
    if (!ctx) return PV_EINVAL;
    const pv_cluster_state &c = ctx->cl;
    if (!c.loaded) return pv_fail(ctx, PV_ESTATE, "pv_eval_selectors: no cluster loaded");
    if (num_pods == 0) return PV_OK;
    if (!d_expr_offs || !d_bits || !d_flags || (num_exprs > 0 && !d_exprs))
        return pv_fail(ctx, PV_EINVAL, "pv_eval_selectors: NULL device pointer");
    if (words_per_row % 4 != 0 || words_per_row < (c.num_nodes + 31) / 32)
        return pv_fail(ctx, PV_EINVAL, "pv_eval_selectors: words_per_row must be >= ceil(N/32) and a multiple of 4");
    if (((uintptr_t)d_bits & 15) != 0) return pv_fail(ctx, PV_EINVAL, "pv_eval_selectors: d_bits must be 16-byte aligned");
    if (((uintptr_t)d_exprs & 3) != 0)   // expressions are read a 32-bit word at a time
        return pv_fail(ctx, PV_EINVAL, "pv_eval_selectors: d_exprs must be 4-byte aligned");
    int which = ctx->opt_selector;
    if (which == 0) which = c.rows_built ? 2 : 1;
    if (which == 2 && !c.rows_built)
        return pv_fail(ctx, PV_EINVAL, "pv_eval_selectors: value rows were not built for this cluster");
    cudaStream_t st = (cudaStream_t)stream;
    const uint32_t wblocks = std::min<uint32_t>((num_pods + 7) / 8, (uint32_t)ctx->num_sms * 16);   // warp per pod
    // comparison kernel: node tiles of as many nodes (multiple of 32) as fit 96 KB of label columns
    uint32_t tile = (uint32_t)((96 * 1024) / (2ull * c.num_keys)) / 32 * 32;
    if (which == 1 && tile < 32)
        return pv_fail(ctx, PV_EINVAL, "pv_eval_selectors: too many keys for the comparison kernel");
    tile = min(tile, ((c.num_nodes + 31) / 32) * 32);
    uint32_t *rep_of = nullptr, *rep_list = nullptr, *rep_count = nullptr;
    pv_use_begin(ctx, st);
    const int pr = pv_prof_start(ctx, st, PV_K_SELECTOR);
    if (ctx->opt_selector_dedupe && num_pods <= (1u << 30)) {
        uint32_t cap = 1;
        while ((uint64_t)cap < 2ull * num_pods) cap <<= 1;
        const size_t o_reps = (size_t)cap * 8, o_hash = o_reps + (((size_t)cap * 4 + 255) & ~(size_t)255);
        const size_t o_rep = o_hash + (size_t)num_pods * 8, o_list = o_rep + (((size_t)num_pods * 4 + 255) & ~(size_t)255);
        const size_t total = o_list + (size_t)num_pods * 4 + 256;
        uint8_t *base = (uint8_t *)pv_scratch(ctx, total);
        if (!base) {
            pv_prof_stop(ctx, st, pr, 0);
            return PV_ENOMEM;
        }
        auto *keys = reinterpret_cast<unsigned long long *>(base);
        auto *reps = reinterpret_cast<uint32_t *>(base + o_reps);
        auto *hashes = reinterpret_cast<unsigned long long *>(base + o_hash);
        rep_of = reinterpret_cast<uint32_t *>(base + o_rep);
        rep_list = reinterpret_cast<uint32_t *>(base + o_list);
        rep_count = rep_list + num_pods;
        PV_TRY_CUDA(ctx, cudaMemsetAsync(rep_count, 0, 4, st), "selector list clear");
        PV_TRY_CUDA(ctx, cudaMemsetAsync(keys, 0, (size_t)cap * 8, st), "selector table clear");
        PV_TRY_CUDA(ctx, cudaMemsetAsync(reps, 0xFF, (size_t)cap * 4, st), "selector table clear");
        sel_hash_kernel<<<wblocks, 256, 0, st>>>(num_pods, d_expr_offs, num_exprs, d_exprs, keys, reps, cap - 1,
                                                  ctx->opt_selector_dedupe == 2 ? 1u : 0u, hashes);
        sel_rep_kernel<<<wblocks, 256, 0, st>>>(num_pods, d_expr_offs, d_exprs, keys, reps, cap - 1, hashes, rep_of,
                                                 rep_list, rep_count);
    }
    if (which == 2) {
        sel_rows_kernel<<<wblocks, kRowsThreads, 0, st>>>(c.num_nodes, c.num_keys, num_pods, d_expr_offs, num_exprs,
                                                          d_exprs, d_assign, d_bits, words_per_row, d_flags, c.d_inv,
                                                          c.d_inv_rank, c.d_key_base, c.d_rows, c.row_words,
                                                          c.num_value_rows, rep_list, rep_count);
    } else {
        const size_t smem = (size_t)tile * c.num_keys * 2;
        PV_TRY_CUDA(ctx, cudaFuncSetAttribute(sel_cmp_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem),
                    "sel_cmp_kernel smem");
        const uint32_t blocks = (num_pods + kCmpPods - 1) / kCmpPods;
        sel_cmp_kernel<<<blocks, kCmpThreads, smem, st>>>(c.num_nodes, c.num_keys, c.d_labels, tile, num_pods,
                                                          d_expr_offs, num_exprs, d_exprs, d_assign, d_bits,
                                                          words_per_row, d_flags, c.d_inv, rep_of);
    }
    if (rep_of)
        sel_copy_kernel<<<wblocks, 256, 0, st>>>(num_pods, c.num_nodes, words_per_row, rep_of, d_assign, d_bits,
                                                 d_flags);
    pv_prof_stop(ctx, st, pr, rep_of ? 4 : 1);
    pv_mark_use(ctx, st);
    return pv_check_launch(ctx, "selector kernels");
}

extern "C" int pv_eval_selector_terms(pv_ctx *ctx, uint32_t num_pods, const uint32_t *d_pod_terms, uint32_t num_terms,
                                      const uint32_t *d_term_offs, uint32_t num_exprs, const pv_expr *d_exprs,
                                      const uint32_t *d_assign, uint32_t *d_bits, uint32_t words_per_row,
                                      uint8_t *d_flags, pv_stream stream) {
    if (!ctx) return PV_EINVAL;
    const pv_cluster_state &c = ctx->cl;
    if (!c.loaded) return pv_fail(ctx, PV_ESTATE, "pv_eval_selector_terms: no cluster loaded");
    if (num_pods == 0) return PV_OK;
    if (!d_pod_terms || !d_bits || !d_flags || (num_terms > 0 && !d_term_offs) || (num_exprs > 0 && !d_exprs))
        return pv_fail(ctx, PV_EINVAL, "pv_eval_selector_terms: NULL device pointer");
    if (words_per_row % 4 != 0 || words_per_row < (c.num_nodes + 31) / 32)
        return pv_fail(ctx, PV_EINVAL,
                       "pv_eval_selector_terms: words_per_row must be >= ceil(N/32) and a multiple of 4");
    if (((uintptr_t)d_bits & 15) != 0)
        return pv_fail(ctx, PV_EINVAL, "pv_eval_selector_terms: d_bits must be 16-byte aligned");
    if (!c.rows_built)
        return pv_fail(ctx, PV_EINVAL, "pv_eval_selector_terms: value rows were not built for this cluster");
    cudaStream_t st = (cudaStream_t)stream;
    const uint32_t blocks = std::min<uint32_t>((num_pods + 7) / 8, (uint32_t)ctx->num_sms * 16);
    pv_use_begin(ctx, st);
    const int pr = pv_prof_start(ctx, st, PV_K_SELECTOR);
    sel_terms_kernel<<<blocks, kRowsThreads, 0, st>>>(c.num_nodes, c.num_keys, num_pods, d_pod_terms, num_terms,
                                                      d_term_offs, num_exprs, d_exprs, d_assign, d_bits,
                                                      words_per_row, d_flags, c.d_inv, c.d_inv_rank, c.d_key_base,
                                                      c.d_rows, c.row_words, c.num_value_rows);
    pv_prof_stop(ctx, st, pr, 1);
    pv_mark_use(ctx, st);
    return pv_check_launch(ctx, "sel_terms_kernel");
}
