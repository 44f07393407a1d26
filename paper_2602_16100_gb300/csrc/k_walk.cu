// Routing constraints Phi_N on realised paths: flow-table loading and
// hop-synchronous probe walks (Sec. 3.3 satisfaction (ii) and the "for all v
// on the path" example; Sec. 4.2 per-hop flow rules; Sec. 5.5 network check;
// Sec. 6.3 item 4: every transit switch is checked).
//
// Loading sorts each switch's rules by (priority desc, input index asc) on
// the device (bitonic sort of packed keys, one block per switch) and
// compiles them into a matching-friendly form, padded to a multiple of 32
// rules with never-matching entries:
//   A = {src & m_src, m_src, dst & m_dst, m_dst}       (uint4, 16 B)
//   B = {dport_lo | dport_hi << 16,
//        in_port_val | in_port_mask << 8 | action << 16} (uint2, 8 B)
// so a rule matches iff ((src^A.x)&A.y | (dst^A.z)&A.w | (in^B.y)&mask) == 0
// and lo <= dport <= hi.
//
// A walk runs one hop for all live probes per step:
//   regroup  : histogram of live probes by current switch, exclusive scan,
//              block-aggregated scatter into switch-contiguous order;
//   hop      : each block takes a contiguous range of that order, stages
//              the range's switch tables into shared memory with a
//              (non-multicast) cp.async.bulk copy completed on an mbarrier,
//              and each warp resolves first-match for one probe at a time,
//              32 rules per step, with __ballot_sync / __ffs.  Terminated
//              probes write their result; live ones are appended (block-
//              aggregated) to the next hop's list.
#include <cuda_runtime.h>

#include <algorithm>
#include <vector>

#include "pv_internal.cuh"

namespace {

constexpr int kHopThreads = 256;
constexpr int kHopWarps = kHopThreads / 32;
constexpr uint32_t kMinPerBlock = 512;       // live probes per active hop block
constexpr int kGridThreads = 256;
constexpr uint32_t kSmemHistMax = 12288;     // switches for shared-memory histograms
constexpr uint32_t kWaitLimit = 1u << 24;    // bounded mbarrier polls

// ---------------------------------------------------------------------------
// PTX helpers: mbarrier + bulk copy (non-multicast, own CTA)
// ---------------------------------------------------------------------------
__device__ __forceinline__ uint32_t smem_u32(const void *p) {
    return (uint32_t)__cvta_generic_to_shared(p);
}
__device__ __forceinline__ void mbar_init(uint64_t *bar, uint32_t count) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count) : "memory");
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}
__device__ __forceinline__ void mbar_arrive_expect_tx(uint64_t *bar, uint32_t bytes) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)), "r"(bytes)
                 : "memory");
}
// Bulk copy global -> shared completed on an mbarrier, asking L2 to keep the
// source lines (evict_last): the flow-table blobs are re-read every hop while
// the probe lists stream through L2.
__device__ __forceinline__ void bulk_g2s_keep(void *dst, const void *src, uint32_t bytes, uint64_t *bar) {
    asm volatile(
        "{\n\t.reg .b64 pol;\n\t"
        "createpolicy.fractional.L2::evict_last.b64 pol, 1.0;\n\t"
        "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint [%0], [%1], %2, [%3], pol;\n\t}"
        ::"r"(smem_u32(dst)),
        "l"(src), "r"(bytes), "r"(smem_u32(bar))
        : "memory");
}
__device__ __forceinline__ bool mbar_try_wait(uint64_t *bar, uint32_t parity) {
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(smem_u32(bar)), "r"(parity)
        : "memory");
    return ok != 0;
}
__device__ __forceinline__ uint64_t global_ns() {
    uint64_t t;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
    return t;
}
// Waits for the phase with the given parity; gives up after limit_ns
// nanoseconds of the global timer (or kWaitLimit polls, whichever is first).
__device__ __forceinline__ bool mbar_wait_bounded(uint64_t *bar, uint32_t parity, uint64_t limit_ns) {
    const uint64_t t0 = global_ns();
    for (uint32_t it = 0; it < kWaitLimit; ++it) {
        if (mbar_try_wait(bar, parity)) return true;
        if (global_ns() - t0 > limit_ns) break;
    }
    return false;
}

// ---------------------------------------------------------------------------
// load: per-switch stable priority sort + compile
// ---------------------------------------------------------------------------
// Also validates every rule of the switch against its port count; the lowest
// offending global rule index goes to *bad (0xFFFFFFFF when all are valid).
__global__ void __launch_bounds__(1024) compile_tables_kernel(const uint32_t *__restrict__ rule_offs,
                                                              const pv_rule *__restrict__ raw,
                                                              const uint32_t *__restrict__ port_offs,
                                                              const uint32_t *__restrict__ tab_offs,
                                                              uint4 *__restrict__ A, uint2 *__restrict__ B,
                                                              uint32_t *__restrict__ bad) {
    extern __shared__ uint32_t s_keys[];
    const uint32_t s = blockIdx.x, t = threadIdx.x;
    const uint32_t base = rule_offs[s], n = rule_offs[s + 1] - base;
    const uint32_t nports = port_offs[s + 1] - port_offs[s];
    for (uint32_t i = t; i < n; i += blockDim.x) {
        const pv_rule r = raw[base + i];
        const bool ok = (r.in_port == PV_ANY_PORT || r.in_port < nports) &&
                        (r.action == PV_DROP || r.action < nports) && r.src_len <= 32 && r.dst_len <= 32 &&
                        r.dport_lo <= r.dport_hi;
        if (!ok) atomicMin(bad, base + i);
    }
    uint32_t npow = 1;
    while (npow < n) npow <<= 1;
    for (uint32_t i = t; i < npow; i += blockDim.x)
        s_keys[i] = i < n ? ((uint32_t)(65535u - raw[base + i].priority) << 16) | i : 0xFFFFFFFFu;
    __syncthreads();
    for (uint32_t k = 2; k <= npow; k <<= 1)
        for (uint32_t j = k >> 1; j > 0; j >>= 1) {
            for (uint32_t i = t; i < npow; i += blockDim.x) {
                uint32_t ixj = i ^ j;
                if (ixj > i) {
                    uint32_t a = s_keys[i], b = s_keys[ixj];
                    bool up = (i & k) == 0;
                    if ((a > b) == up) {
                        s_keys[i] = b;
                        s_keys[ixj] = a;
                    }
                }
            }
            __syncthreads();
        }
    const uint32_t out = tab_offs[s], npad = tab_offs[s + 1] - out;
    for (uint32_t i = t; i < npad; i += blockDim.x) {
        uint4 a;
        uint2 b;
        if (i < n) {
            const pv_rule r = raw[base + (s_keys[i] & 0xFFFFu)];
            const uint32_t ms = pv_prefix_mask(min(32u, (uint32_t)r.src_len));
            const uint32_t md = pv_prefix_mask(min(32u, (uint32_t)r.dst_len));
            a = make_uint4(r.src_ip & ms, ms, r.dst_ip & md, md);
            const bool any = r.in_port == PV_ANY_PORT;
            b.x = (uint32_t)r.dport_lo | ((uint32_t)r.dport_hi << 16);
            b.y = (any ? 0u : (r.in_port & 0xFFu)) | (any ? 0u : 0xFF00u) | ((uint32_t)r.action << 16);
        } else {
            a = make_uint4(0, 0, 0, 0);
            b.x = 1u;   // lo = 1 > hi = 0: never matches
            b.y = 0u;
        }
        A[out + i] = a;
        B[out + i] = b;
    }
}

// ---------------------------------------------------------------------------
// load: first-match index
// ---------------------------------------------------------------------------
// A switch's blob (sections 16-byte aligned):
//   header   uint4 {npad | n_plain << 16, n_items, n_segs, n_bnd}
//   A[n_plain] uint4, B[n_plain] uint2   the plain rules (those not in a
//                                    segment, the only ones items name), in
//                                    first-match order (records as above)
//   boff[kBuckets + 1] u32           item range of each destination-port bucket
//   items[n_items] u16               per bucket, in first-match order: a plain
//                                    rule's position, or kSegItem | segment id
//   segs[n_segs] uint2               {first boundary, number of boundaries}
//   bnd[n_bnd] u32, win[n_bnd] u32   per segment: ascending elementary-interval
//                                    starts (the first is 0) and the interval's
//                                    winner (kWinFound | action, or 0 = none)
//   jmp[n_segs]                      per segment, kJumpBytes: {base, shift,
//                                    J[kJumpSlots + 1] u16}: base = the
//                                    segment's second boundary (its first
//                                    non-zero one), and J[j] = the last
//                                    boundary index <= base + (j << shift)
//                                    (J[kJumpSlots] = the last index), so an
//                                    address's interval is searched among
//                                    J[j] .. J[j + 1] only
//   A[npad] uint4, B[npad] uint2     all rules in first-match order, padded to a
//                                    multiple of 32 (linear scan, statistics)
// The indexed kernel stages everything before the full rule list; the
// linear kernel stages the header and the full rule list.
// Exactness.  A header whose dport lies in bucket k can only match rules whose
// port range meets bucket k; bucket k's list keeps the first-match order, so
// its first hit is the first match of the whole table.  A segment is a run of
// consecutive rules that constrain nothing but the destination prefix (any
// in_port, no source prefix, full port range); every rule's address range is
// a union of the segment's elementary intervals (each range contributes its
// start and end + 1 as boundaries), so within a segment the first match of
// address d is the precomputed winner of d's interval.
constexpr uint32_t kBuckets = 256;          // dport >> kBucketShift
constexpr uint32_t kBucketShift = 8;
constexpr uint32_t kMinSegment = 4;         // shorter destination-only runs stay plain items
constexpr uint32_t kTailEarlyItems = 12;    // candidate items per bucket below which the tail starts at hop 5
constexpr uint32_t kMaxSegment = 4096;      // longer runs are split (in order: still exact)
constexpr uint32_t kSegItem = 0x8000u;
constexpr uint32_t kWinFound = 0x80000000u;
constexpr uint32_t kJumpSlots = 256;
constexpr uint32_t kJumpBytes = (8 + (kJumpSlots + 1) * 2 + 15) / 16 * 16;   // 528
static_assert(kJumpBytes % 16 == 0, "jump blocks keep the blob's later sections 16-byte aligned");
constexpr int kIndexThreads = 512;
static_assert(kIndexThreads / 32 == 16, "bucket fill counts are laid out for 16 warps");

// Shared-memory layout of index_build_kernel, sized for the largest table
// of a load (max_rules rules): sort keys (also the staged port ranges),
// interval winners (also the bucket pairs' rule offsets), scan positions,
// rule classes, segment bounds, one segment's prefixes and actions, and the
// bucket fill's per-warp counts and cursors.
constexpr uint32_t kIndexWarps = 512 / 32;
static_assert(PV_MAX_RULES * 4 <= kMaxSegment * 10, "plain-rule ranks overlay one segment's staging area");
static_assert(PV_MAX_RULES < kSegItem, "plain-rule positions fit an item below the segment flag");
struct IndexSmem {
    uint32_t sort_cap, key_cap, rules_cap, segs_cap, seg_cap;
    size_t bytes;
    __host__ __device__ IndexSmem() : sort_cap(0), key_cap(0), rules_cap(0), segs_cap(0), seg_cap(0), bytes(0) {}
    __host__ __device__ explicit IndexSmem(uint32_t max_rules) {
        const uint32_t n = max_rules < 1 ? 1 : max_rules;
        seg_cap = n < kMaxSegment ? n : kMaxSegment;
        const uint32_t need = 2 * seg_cap + 1 > n ? 2 * seg_cap + 1 : n;
        sort_cap = 1;
        while (sort_cap < need) sort_cap <<= 1;
        key_cap = 2 * seg_cap + 8 > kBuckets + 8 ? 2 * seg_cap + 8 : kBuckets + 8;
        key_cap = (key_cap + 1) & ~1u;
        rules_cap = (n + 7) & ~7u;
        segs_cap = n / kMinSegment + n / kMaxSegment + 2;   // runs of >= 4, long runs split
        bytes = (size_t)sort_cap * 4 + (size_t)key_cap * 8 + (size_t)rules_cap * 2 + (size_t)segs_cap * 8 +
                (size_t)seg_cap * 10;
        bytes = (bytes + 15) & ~(size_t)15;
        bytes += (size_t)kIndexWarps * kBuckets * 2 + (size_t)kBuckets * 4;
    }
};

__host__ __device__ inline uint32_t up16(uint32_t b) { return (b + 15u) & ~15u; }

struct BlobLayout {
    uint32_t a, b, boff, items, segs, bnd, win, jmp, fa, fb, total;
    __host__ __device__ BlobLayout(uint32_t npad, uint32_t n_plain, uint32_t n_items, uint32_t n_segs,
                                   uint32_t n_bnd) {
        a = 16;
        b = a + up16(n_plain * 16);
        boff = b + up16(n_plain * 8);
        items = boff + up16((kBuckets + 1) * 4);
        segs = items + up16(n_items * 2);
        bnd = segs + up16(n_segs * 8);
        win = bnd + up16(n_bnd * 4);
        jmp = win + up16(n_bnd * 4);
        fa = jmp + n_segs * kJumpBytes;
        fb = fa + npad * 16;
        total = fb + npad * 8;
    }
    __host__ __device__ explicit BlobLayout(uint4 hdr)
        : BlobLayout(hdr.x & 0xFFFFu, hdr.x >> 16, hdr.y, hdr.z, hdr.w) {}
};

// Bytes of the hop kernel's staged port table ({peer, aux} per port).
inline size_t port_stage_bytes(uint32_t max_ports) { return ((size_t)max_ports * 8 + 15) & ~(size_t)15; }

// Rules as the linear kernel stages them: the header, then all rules' A and B
// records from the blob's end.
__host__ __device__ inline uint32_t linear_bytes(uint32_t npad) { return 16 + npad * 24; }

__device__ __forceinline__ bool rule_dst_only(uint4 a, uint2 b) {
    return a.y == 0 && b.x == 0xFFFF0000u && ((b.y >> 8) & 0xFFu) == 0;
}

// In-place exclusive scan of v[0..n) by the whole block; returns the total.
__device__ uint32_t block_exclusive_scan(uint32_t *v, uint32_t n, uint32_t *s_warp) {
    const uint32_t t = threadIdx.x, lane = t & 31, warp = t >> 5, nt = blockDim.x;
    const uint32_t per = (n + nt - 1) / nt, b0 = t * per;
    uint32_t local = 0;
    for (uint32_t i = 0; i < per; ++i)
        if (b0 + i < n) local += v[b0 + i];
    uint32_t incl = local;
    for (int d = 1; d < 32; d <<= 1) {
        const uint32_t y = __shfl_up_sync(PV_FULL_MASK, incl, d);
        if (lane >= (uint32_t)d) incl += y;
    }
    if (lane == 31) s_warp[warp] = incl;
    __syncthreads();
    if (warp == 0) {
        const uint32_t x = lane < nt / 32 ? s_warp[lane] : 0u;
        uint32_t xi = x;
        for (int d = 1; d < 32; d <<= 1) {
            const uint32_t y = __shfl_up_sync(PV_FULL_MASK, xi, d);
            if (lane >= (uint32_t)d) xi += y;
        }
        s_warp[lane] = xi - x;
        if (lane == 31) s_warp[32] = xi;
    }
    __syncthreads();
    uint32_t run = s_warp[warp] + incl - local;
    for (uint32_t i = 0; i < per; ++i)
        if (b0 + i < n) {
            const uint32_t x = v[b0 + i];
            v[b0 + i] = run;
            run += x;
        }
    const uint32_t total = s_warp[32];
    __syncthreads();
    return total;
}

// Pass 1 (kFill = false) writes sizes[4s..4s+3] = {n_items, n_segs, n_bnd,
// n_plain}; pass 2 writes the blob at blob_offs[s].  One kIndexThreads-thread block per switch.
template <bool kFill>
__global__ void __launch_bounds__(kIndexThreads) index_build_kernel(const uint32_t *__restrict__ rule_offs,
                                                           const uint32_t *__restrict__ tab_offs,
                                                           const uint4 *__restrict__ A, const uint2 *__restrict__ B,
                                                           uint32_t *__restrict__ sizes,
                                                           const uint64_t *__restrict__ blob_offs,
                                                           uint8_t *__restrict__ blob, IndexSmem sm) {
    extern __shared__ __align__(16) uint32_t s_mem[];
    uint32_t *s_keys = s_mem;                                            // [sort_cap]
    uint32_t *s_win = s_keys + sm.sort_cap;                              // [key_cap]
    uint32_t *s_pos = s_win + sm.key_cap;                                // [key_cap]
    int16_t *s_cls = reinterpret_cast<int16_t *>(s_pos + sm.key_cap);     // [rules_cap]
    uint32_t *s_segs = reinterpret_cast<uint32_t *>(s_cls + sm.rules_cap);  // [segs_cap][2]
    uint2 *s_rules = reinterpret_cast<uint2 *>(s_segs + 2 * sm.segs_cap);   // [seg_cap] {value, mask}
    uint16_t *s_act = reinterpret_cast<uint16_t *>(s_rules + sm.seg_cap);    // [seg_cap]
    uint8_t *s_tail = reinterpret_cast<uint8_t *>(s_mem) +
                      (((size_t)sm.sort_cap * 4 + (size_t)sm.key_cap * 8 + (size_t)sm.rules_cap * 2 +
                        (size_t)sm.segs_cap * 8 + (size_t)sm.seg_cap * 10 + 15) & ~(size_t)15);
    uint16_t *s_wcnt = reinterpret_cast<uint16_t *>(s_tail);                        // [16][kBuckets]
    uint32_t *s_cur = reinterpret_cast<uint32_t *>(s_tail + kIndexWarps * kBuckets * 2);  // [kBuckets]
    __shared__ uint32_t s_warp[33];
    const uint32_t s = blockIdx.x, t = threadIdx.x, lane = t & 31, warp = t >> 5, nt = blockDim.x;
    const uint32_t n = rule_offs[s + 1] - rule_offs[s];
    const uint32_t t0 = tab_offs[s], npad = tab_offs[s + 1] - t0;
    const uint4 *a = A + t0;
    const uint2 *b = B + t0;

    // 1. destination-only runs -> segments.  The rules are classified and
    //    their port ranges staged (s_keys is free until the segment sort of
    //    step 3); block scans then number the runs of destination-only rules
    //    and their segments (runs shorter than kMinSegment stay plain rules,
    //    longer ones are cut every kMaxSegment rules).
    for (uint32_t i = t; i < n; i += nt) {
        const uint2 bi = b[i];
        s_cls[i] = rule_dst_only(a[i], bi) ? 1 : -1;
        s_keys[i] = bi.x;   // dport lo | hi << 16
    }
    __syncthreads();
    auto run_start = [&](uint32_t i) { return s_cls[i] > 0 && (i == 0 || s_cls[i - 1] < 0); };
    for (uint32_t i = t; i < n; i += nt) s_pos[i] = run_start(i) ? 1u : 0u;
    __syncthreads();
    const uint32_t R = block_exclusive_scan(s_pos, n, s_warp);   // s_pos[i]: runs starting before i
    uint32_t *s_run = s_win;                                     // [2R]: start, end of each run
    for (uint32_t i = t; i < n; i += nt) {
        if (s_cls[i] < 0) continue;
        const bool st = run_start(i);
        const uint32_t r = s_pos[i] + (st ? 1u : 0u) - 1u;
        if (st) s_run[2 * r] = i;
        if (i + 1 == n || s_cls[i + 1] < 0) s_run[2 * r + 1] = i + 1;
    }
    __syncthreads();
    for (uint32_t r = t; r < R; r += nt) {
        const uint32_t len = s_run[2 * r + 1] - s_run[2 * r];
        s_pos[r] = len < kMinSegment ? 0u : (len + kMaxSegment - 1) / kMaxSegment;
    }
    __syncthreads();
    const uint32_t nsegs = block_exclusive_scan(s_pos, R, s_warp);   // s_pos[r]: first segment of run r
    for (uint32_t r = t; r < R; r += nt) {
        const uint32_t r0 = s_run[2 * r], r1 = s_run[2 * r + 1];
        if (r1 - r0 < kMinSegment) continue;
        uint32_t seg = s_pos[r];
        for (uint32_t k0 = r0; k0 < r1; k0 += kMaxSegment, ++seg) {
            s_segs[2 * seg] = k0;
            s_segs[2 * seg + 1] = min(r1, k0 + kMaxSegment);
        }
    }
    // each rule's class: its segment, or -1 (a thread reads and writes only
    // its own rules' flags from here on)
    for (uint32_t i = t; i < n; i += nt) {
        if (s_cls[i] < 0) continue;
        uint32_t lo = 0, hi = R;   // the run holding i: last start <= i
        while (hi - lo > 1) {
            const uint32_t mid = (lo + hi) >> 1;
            if (s_run[2 * mid] <= i) lo = mid;
            else hi = mid;
        }
        const uint32_t r0 = s_run[2 * lo], r1 = s_run[2 * lo + 1];
        s_cls[i] = r1 - r0 < kMinSegment ? (int16_t)-1 : (int16_t)(s_pos[lo] + (i - r0) / kMaxSegment);
    }
    __syncthreads();
    // plain rules (not in a segment) and their positions among themselves;
    // the ranks sit in the segment staging area (s_rules and s_act, free
    // until step 3: seg_cap * 10 bytes hold n words for n <= PV_MAX_RULES)
    uint32_t *s_plain = reinterpret_cast<uint32_t *>(s_rules);   // [n]
    for (uint32_t i = t; i < n; i += nt) s_plain[i] = s_cls[i] < 0 ? 1u : 0u;
    __syncthreads();
    const uint32_t n_plain = block_exclusive_scan(s_plain, n, s_warp);
    uint8_t *out = nullptr;
    BlobLayout L(npad, n_plain, 0, 0, 0);
    if (kFill) {
        out = blob + blob_offs[s];
        L = BlobLayout(npad, n_plain, sizes[4 * s], sizes[4 * s + 1], sizes[4 * s + 2]);
        uint4 *ca = reinterpret_cast<uint4 *>(out + L.a);
        uint2 *cb = reinterpret_cast<uint2 *>(out + L.b);
        for (uint32_t i = t; i < n; i += nt)
            if (s_cls[i] < 0) {
                ca[s_plain[i]] = a[i];
                cb[s_plain[i]] = b[i];
            }
    }

    // 2. bucket lists.  Rule i puts one item into each bucket its port range
    //    meets (a segment's token, at the segment's first rule, goes into
    //    every bucket); the items of rule i take pair positions poff[i] ..
    //    poff[i] + nb(i) - 1, so pairs run in rule order, and a stable
    //    counting sort of the pairs by bucket leaves each bucket's items in
    //    first-match order.
    auto bucket_range = [&](uint32_t i, uint32_t *b0) -> uint32_t {   // number of buckets
        const int c = s_cls[i];
        if (c >= 0) {
            *b0 = 0;
            return s_segs[2 * c] == i ? kBuckets : 0u;
        }
        const uint32_t pr = s_keys[i];
        *b0 = (pr & 0xFFFFu) >> kBucketShift;
        return ((pr >> 16) >> kBucketShift) - *b0 + 1u;
    };
    uint32_t *s_poff = s_win;   // [n]: first pair of rule i (s_win is free until step 3)
    for (uint32_t k = t; k < kBuckets; k += nt) s_pos[k] = 0;
    for (uint32_t x = t; x < kIndexWarps * kBuckets; x += nt) s_wcnt[x] = 0;
    __syncthreads();
    for (uint32_t i = t; i < n; i += nt) {
        uint32_t b0;
        const uint32_t nb = bucket_range(i, &b0);
        s_poff[i] = nb;
        for (uint32_t k = b0; k < b0 + nb; ++k) atomicAdd(&s_pos[k], 1u);
    }
    __syncthreads();
    const uint32_t n_items = block_exclusive_scan(s_pos, kBuckets, s_warp);   // s_pos[k] = first item of bucket k
    if (kFill) {
        uint32_t *boff = reinterpret_cast<uint32_t *>(out + L.boff);
        uint16_t *items = reinterpret_cast<uint16_t *>(out + L.items);
        for (uint32_t k = t; k < kBuckets; k += nt) {
            boff[k] = s_pos[k];
            s_cur[k] = s_pos[k];
        }
        if (t == 0) boff[kBuckets] = n_items;
        block_exclusive_scan(s_poff, n, s_warp);
        const uint32_t lt = (1u << lane) - 1u;
        for (uint32_t c0 = 0; c0 < n_items; c0 += nt) {
            const uint32_t p = c0 + t;
            const bool on = p < n_items;
            uint32_t k = 0xFFFFFFFFu, i = 0;
            if (on) {
                uint32_t lo = 0, hi = n;   // rule of pair p: last i with poff[i] <= p
                while (hi - lo > 1) {
                    const uint32_t mid = (lo + hi) >> 1;
                    if (s_poff[mid] <= p) lo = mid;
                    else hi = mid;
                }
                i = lo;
                uint32_t b0;
                bucket_range(i, &b0);
                k = b0 + (p - s_poff[i]);
            }
            // rank among this warp's pairs of the same bucket (lanes run in
            // pair order), then this warp's count per bucket for the others
            const uint32_t peers = __match_any_sync(PV_FULL_MASK, k);
            const uint32_t rank = __popc(peers & lt);
            const bool leader = (peers & lt) == 0;
            if (on && leader) s_wcnt[warp * kBuckets + k] = (uint16_t)__popc(peers);
            __syncthreads();
            if (on) {
                uint32_t pos = s_cur[k] + rank;
                for (uint32_t w = 0; w < warp; ++w) pos += s_wcnt[w * kBuckets + k];
                const int c = s_cls[i];
                items[pos] = (uint16_t)(c >= 0 ? (kSegItem | (uint32_t)c) : s_plain[i]);
            }
            __syncthreads();
            if (on && leader) {
                atomicAdd(&s_cur[k], (uint32_t)__popc(peers));
                s_wcnt[warp * kBuckets + k] = 0;
            }
            __syncthreads();
        }
    }
    __syncthreads();

    // 3. per segment: sorted unique boundaries, interval winners, merged runs
    uint32_t n_bnd = 0;
    for (uint32_t j = 0; j < nsegs; ++j) {
        const uint32_t k0 = s_segs[2 * j], k1 = s_segs[2 * j + 1], m = k1 - k0;
        const uint32_t nk = 2 * m + 1;
        uint32_t npow = 1;
        while (npow < nk) npow <<= 1;
        for (uint32_t x = t; x < npow; x += nt) {
            uint32_t key = 0xFFFFFFFFu;
            if (x == 0) {
                key = 0;
            } else if (x < nk) {
                const uint4 r = a[k0 + (x - 1) / 2];
                if (x & 1u) {
                    key = r.z;
                } else {
                    const uint64_t end1 = (uint64_t)r.z + (uint64_t)(~r.w) + 1ull;
                    key = end1 < (1ull << 32) ? (uint32_t)end1 : 0u;
                }
            }
            s_keys[x] = key;
        }
        __syncthreads();
        for (uint32_t kk = 2; kk <= npow; kk <<= 1)
            for (uint32_t jj = kk >> 1; jj > 0; jj >>= 1) {
                for (uint32_t i = t; i < npow; i += nt) {
                    const uint32_t ixj = i ^ jj;
                    if (ixj > i) {
                        const uint32_t p = s_keys[i], q = s_keys[ixj];
                        if ((p > q) == ((i & kk) == 0)) {
                            s_keys[i] = q;
                            s_keys[ixj] = p;
                        }
                    }
                }
                __syncthreads();
            }
        for (uint32_t x = t; x < nk; x += nt) s_pos[x] = (x == 0 || s_keys[x] != s_keys[x - 1]) ? 1u : 0u;
        __syncthreads();
        for (uint32_t x = t; x < nk; x += nt) s_win[x] = s_keys[x];   // keep sorted copy
        __syncthreads();
        const uint32_t K = block_exclusive_scan(s_pos, nk, s_warp);
        for (uint32_t x = t; x < nk; x += nt)
            if (x == 0 || s_win[x] != s_win[x - 1]) s_keys[s_pos[x]] = s_win[x];
        __syncthreads();
        // the segment's prefixes and actions, staged in shared memory
        for (uint32_t r = t; r < m; r += nt) {
            const uint4 ar = a[k0 + r];
            s_rules[r] = make_uint2(ar.z, ar.w);
            s_act[r] = (uint16_t)(b[k0 + r].y >> 16);
        }
        __syncthreads();
        // winners of the K elementary intervals: the first rule (in
        // first-match order) whose address range contains the interval.
        // Each rule's range [v, v + size) starts and ends on boundaries, so
        // it covers intervals ia .. ib - 1 exactly; the smallest rule index
        // covering an interval wins.
        for (uint32_t x = t; x < K; x += nt) s_win[x] = 0xFFFFFFFFu;
        __syncthreads();
        for (uint32_t r = t; r < m; r += nt) {
            const uint2 ar = s_rules[r];
            const uint64_t end1 = (uint64_t)ar.x + (uint64_t)(~ar.y) + 1ull;   // exclusive end
            uint32_t lo = 0, hi = K;   // first x with s_keys[x] >= ar.x
            while (lo < hi) {
                const uint32_t mid = (lo + hi) >> 1;
                if (s_keys[mid] < ar.x) lo = mid + 1;
                else hi = mid;
            }
            const uint32_t ia = lo;
            uint32_t ib = K;
            if (end1 < (1ull << 32)) {
                lo = ia;
                hi = K;
                while (lo < hi) {
                    const uint32_t mid = (lo + hi) >> 1;
                    if (s_keys[mid] < (uint32_t)end1) lo = mid + 1;
                    else hi = mid;
                }
                ib = lo;
            }
            for (uint32_t x = ia; x < ib; ++x) atomicMin(&s_win[x], r);
        }
        __syncthreads();
        for (uint32_t x = t; x < K; x += nt) {
            const uint32_t r = s_win[x];
            s_win[x] = r == 0xFFFFFFFFu ? 0u : (kWinFound | s_act[r]);
        }
        __syncthreads();
        // merge adjacent intervals with the same winner
        for (uint32_t x = t; x < K; x += nt) s_pos[x] = (x == 0 || s_win[x] != s_win[x - 1]) ? 1u : 0u;
        __syncthreads();
        // keep flags must be read before the scan overwrites them
        uint32_t keep_mask = 0;
        for (uint32_t x = t, q = 0; x < K && q < 32; x += nt, ++q)
            if (s_pos[x]) keep_mask |= 1u << q;
        __syncthreads();
        const uint32_t K2 = block_exclusive_scan(s_pos, K, s_warp);
        if (kFill) {
            uint2 *segs = reinterpret_cast<uint2 *>(out + L.segs);
            uint32_t *bnd = reinterpret_cast<uint32_t *>(out + L.bnd);
            uint32_t *win = reinterpret_cast<uint32_t *>(out + L.win);
            if (t == 0) segs[j] = make_uint2(n_bnd, K2);
            for (uint32_t x = t, q = 0; x < K; x += nt, ++q)
                if ((keep_mask >> q) & 1u) {
                    bnd[n_bnd + s_pos[x]] = s_keys[x];
                    win[n_bnd + s_pos[x]] = s_win[x];
                }
            __syncthreads();   // the segment's boundaries are in the blob
            uint8_t *jb = out + L.jmp + j * kJumpBytes;
            const uint32_t *bb = bnd + n_bnd;
            const uint32_t base = K2 > 1 ? bb[1] : 0xFFFFFFFFu, top = bb[K2 - 1];
            uint32_t shift = 0;
            while (shift < 32 && ((uint64_t)(top - (K2 > 1 ? base : top)) >> shift) >= kJumpSlots) ++shift;
            if (t == 0) {
                reinterpret_cast<uint32_t *>(jb)[0] = base;
                reinterpret_cast<uint32_t *>(jb)[1] = shift;
            }
            uint16_t *J = reinterpret_cast<uint16_t *>(jb + 8);
            for (uint32_t x = t; x <= kJumpSlots; x += nt) {
                const uint64_t start = (uint64_t)base + ((uint64_t)x << shift);
                uint32_t v = K2 - 1;   // last index with bb[v] <= start
                if (x < kJumpSlots && start < 0xFFFFFFFFull) {
                    uint32_t lo = 0, hi = K2;   // bb[lo] <= start < bb[hi]
                    while (hi - lo > 1) {
                        const uint32_t mid = (lo + hi) >> 1;
                        if (bb[mid] <= (uint32_t)start) lo = mid;
                        else hi = mid;
                    }
                    v = lo;
                }
                J[x] = (uint16_t)v;
            }
        }
        n_bnd += K2;
        __syncthreads();
    }

    // 4. header and the full rule list
    if (kFill) {
        if (t == 0) *reinterpret_cast<uint4 *>(out) = make_uint4(npad | n_plain << 16, n_items, nsegs, n_bnd);
        uint4 *oa = reinterpret_cast<uint4 *>(out + L.fa);
        uint2 *ob = reinterpret_cast<uint2 *>(out + L.fb);
        for (uint32_t i = t; i < npad; i += nt) {
            oa[i] = a[i];
            ob[i] = b[i];
        }
    } else if (t == 0) {
        sizes[4 * s] = n_items;
        sizes[4 * s + 1] = nsegs;
        sizes[4 * s + 2] = n_bnd;
        sizes[4 * s + 3] = n_plain;
    }
}

// ---------------------------------------------------------------------------
// walk kernels
// ---------------------------------------------------------------------------
// Live lists are written in per-block slices: block b of the producing kernel
// owns list[desc[b].x .. desc[b].x + desc[b].y); consumers take one slice
// per block.  Warps reserve slots of their block's slice with shared-memory
// atomics, so producing a list needs neither a global counter nor barriers.
// Entry: x = probe id, y = location (switch << 8 | in_port).
// Walk result i as one 32-bit store {status, hops, last_switch} (the
// struct's own alignment is 2, so a member-wise store would be two or three
// narrow writes, each a separate sector write at L2; walks require a 4-byte
// aligned result array).
__device__ __forceinline__ void put_result(pv_result *out, uint32_t i, uint32_t status, uint32_t hops,
                                           uint32_t last) {
    reinterpret_cast<uint32_t *>(out)[i] = status | hops << 8 | last << 16;
}

__device__ __forceinline__ uint32_t warp_reserve(bool want, uint32_t *s_count) {
    const uint32_t lane = threadIdx.x & 31;
    const uint32_t m = __ballot_sync(PV_FULL_MASK, want);
    uint32_t base = 0;
    if (lane == 0 && m) base = atomicAdd(s_count, (uint32_t)__popc(m));
    base = __shfl_sync(PV_FULL_MASK, base, 0);
    return base + __popc(m & ((1u << lane) - 1u));
}

// Path constraints of the walk (Sec. 4.2 constraint object; Sec. 5.3 and
// Sec. 5.5 waypoint and forbidden-switch checks).  Probe k follows policy
// probe_pol[k] (or first + k / per when probe_pol is null); an index >= num means
// none.  A forbidden switch is judged like a forbidden jurisdiction (checked
// when the probe is handed to it, so it never enters); hits[k] bit i is set
// once the probe has entered waypoint i of its policy.
struct PolicyArgs {
    const uint4 *hdr;          // [num] {forbid offset, count, waypoint offset, count}
    const uint16_t *sw;        // switch ids
    uint32_t num;
    const uint32_t *probe_pol; // [M] or null
    uint32_t per;              // probes per policy when probe_pol is null
    uint32_t first;            // policy of probe 0 when probe_pol is null
    uint32_t *hits;            // [M] waypoint bits (output)
};

__device__ __forceinline__ uint4 policy_of(const PolicyArgs &pa, uint32_t k) {
    const uint32_t p = pa.probe_pol ? pa.probe_pol[k] : (pa.per ? pa.first + k / pa.per : 0xFFFFFFFFu);
    return p < pa.num ? pa.hdr[p] : make_uint4(0, 0, 0, 0);
}

__device__ __forceinline__ bool switch_listed(const uint16_t *list, uint32_t n, uint32_t s) {
    for (uint32_t i = 0; i < n; ++i)
        if (list[i] == s) return true;
    return false;
}

// First visit of every probe: NOSRC for an absent source host, VIOLATION at
// the attachment switch when its region is not permitted (or, with path
// constraints, the switch is forbidden to the probe), otherwise listed.
// It also counts the listed probes per switch into hist (the first hop's
// histogram; per block in shared memory when S <= kSmemHistMax).  With
// kBind, the probe records are first built from compact flows and the
// placement (the binding of pv_bind_flows) and written for the later hops.
struct BindArgs {
    // flow i: destination address dst[i * dst_stride], port dport[i * dport_stride]
    // (records {dst_ip, dport, 0}: strides 2 and 4; columns: 1 and 1)
    const uint32_t *dst;
    const uint16_t *dport;
    uint32_t dst_stride, dport_stride;
    uint32_t ppg, pods;          // probes and pods per group
    const uint32_t *assign;      // [groups * pods]
    const uint32_t *group_mask;  // [groups]
    const uint32_t *host_ip;     // [H]
};

// Flow i as {dst_ip, dport}.
__device__ __forceinline__ uint2 flow_at(const BindArgs &ba, uint32_t i) {
    return make_uint2(__ldg(ba.dst + (size_t)i * ba.dst_stride), __ldg(ba.dport + (size_t)i * ba.dport_stride));
}

__device__ __forceinline__ uint32_t flow_dport(const BindArgs &ba, uint32_t i) {
    return __ldg(ba.dport + (size_t)i * ba.dport_stride);
}

template <bool kPolicy, bool kBind>
__global__ void __launch_bounds__(kGridThreads) walk_init_kernel(
    uint32_t M, pv_probe *__restrict__ probes, uint32_t H, const uint16_t *__restrict__ host_switch,
    const uint16_t *__restrict__ host_port, const uint8_t *__restrict__ region, pv_result *__restrict__ out,
    uint2 *__restrict__ list, uint2 *__restrict__ desc, PolicyArgs pa, uint32_t S, uint32_t *__restrict__ hist,
    BindArgs ba) {
    extern __shared__ uint32_t s_hist[];   // [S] when S <= kSmemHistMax
    const bool smem_hist = S <= kSmemHistMax;
    if (smem_hist)
        for (uint32_t j = threadIdx.x; j < S; j += kGridThreads) s_hist[j] = 0;
    __shared__ uint32_t s_count;
    const uint32_t c0 = (uint32_t)(((uint64_t)M * blockIdx.x) / gridDim.x);
    const uint32_t c1 = (uint32_t)(((uint64_t)M * (blockIdx.x + 1)) / gridDim.x);
    if (threadIdx.x == 0) s_count = 0;
    __syncthreads();
    for (uint32_t base = c0; base < c1; base += kGridThreads) {
        const uint32_t i = base + threadIdx.x;
        bool live = false;
        uint32_t loc = 0;
        if (i < c1) {
            // probe record {src_ip, dst_ip, dport | src_host << 16, allowed_mask}
            uint4 pr;
            if (kBind) {
                const uint32_t grp = i / ba.ppg;
                const uint32_t node = ba.assign[grp * ba.pods + (i - grp * ba.ppg) % ba.pods];
                const uint2 f = flow_at(ba, i);
                const bool placed = node < H;
                pr = make_uint4(placed ? ba.host_ip[node] : 0u, f.x,
                                (f.y & 0xFFFFu) | (placed ? node : (uint32_t)PV_NO_HOST) << 16, ba.group_mask[grp]);
                reinterpret_cast<uint4 *>(probes)[i] = pr;
            } else {
                pr = __ldg(reinterpret_cast<const uint4 *>(probes) + i);
            }
            const uint32_t h = pr.z >> 16;
            if (kPolicy) pa.hits[i] = 0;
            if (h < H) {
                const uint32_t s = host_switch[h];
                const uint32_t reg = region[s];
                bool ok = reg < 32 && ((pr.w >> reg) & 1u);
                if (kPolicy && ok) {
                    const uint4 ph = policy_of(pa, i);
                    ok = !switch_listed(pa.sw + ph.x, ph.y, s);
                }
                if (ok) {
                    live = true;
                    loc = (s << 8) | host_port[h];
                } else {
                    put_result(out, i, PV_VIOLATION, 1, s);
                }
            } else {
                put_result(out, i, PV_NOSRC, 0, 0xFFFF);
            }
        }
        const uint32_t slot = warp_reserve(live, &s_count);
        if (live) {
            list[c0 + slot] = make_uint2(i, loc);
            atomicAdd(smem_hist ? &s_hist[loc >> 8] : &hist[loc >> 8], 1u);
        }
    }
    __syncthreads();
    if (threadIdx.x == 0) desc[blockIdx.x] = make_uint2(c0, s_count);
    if (smem_hist)
        for (uint32_t j = threadIdx.x; j < S; j += kGridThreads)
            if (s_hist[j]) atomicAdd(&hist[j], s_hist[j]);
}

// First visit of compact flows, placed directly (pv_verify_flows).  The
// probes of one (group, pod) pair share their source host, mask and path
// constraint, so a pair is listed or judged as a whole: flow_groups_kernel
// adds each listed pair's probe count to its source switch (the first hop's
// per-switch counts) and keeps the pair's offset within that switch; after
// the scan, the walk's first kernel binds every probe and writes its walk
// record straight to its slot in the first hop's switch order (switch start
// + pair offset + rank within the pair), so the first hop needs neither a
// regroup nor a list: it reads records by position and takes each in_port
// from the record's source host.  walk_init_group_kernel (below) does so one group per
// block with each pair's run in bucket order; walk_init_direct_kernel is the
// grid-stride form for groups too large for its shared memory.  Probe i
// belongs to group i / ppg and pod (i mod ppg) mod pods; the caller
// guarantees one path constraint per group.
template <bool kPolicy>
__device__ __forceinline__ bool first_switch_permitted(const PolicyArgs &pa, uint32_t k, uint32_t s, uint32_t reg,
                                                       uint32_t mask) {
    bool ok = reg < 32 && ((mask >> reg) & 1u);
    if (kPolicy && ok) {
        const uint4 ph = policy_of(pa, k);
        ok = !switch_listed(pa.sw + ph.x, ph.y, s);
    }
    return ok;
}

template <bool kPolicy>
__global__ void __launch_bounds__(kGridThreads) flow_groups_kernel(uint32_t M, uint32_t H,
                                                                   const uint16_t *__restrict__ host_switch,
                                                                   const uint8_t *__restrict__ region, PolicyArgs pa,
                                                                   BindArgs ba, uint32_t G, uint32_t *__restrict__ hist,
                                                                   uint32_t *__restrict__ pair_off) {
    for (uint32_t g = blockIdx.x * blockDim.x + threadIdx.x; g < G; g += gridDim.x * blockDim.x) {
        const uint32_t grp = g / ba.pods, q = g - grp * ba.pods;
        const uint32_t first = grp * ba.ppg, len = min(ba.ppg, M - first);
        const uint32_t cnt = len > q ? (len - q + ba.pods - 1) / ba.pods : 0u;
        const uint32_t node = ba.assign[g];
        uint32_t off = 0;
        if (cnt && node < H) {
            const uint32_t s = host_switch[node];
            if (first_switch_permitted<kPolicy>(pa, first + q, s, region[s], ba.group_mask[grp]))
                off = atomicAdd(&hist[s], cnt);
        }
        pair_off[g] = off;
    }
}

template <bool kPolicy>
__global__ void __launch_bounds__(kGridThreads) walk_init_direct_kernel(
    uint32_t M, pv_probe *__restrict__ probes, uint32_t H, const uint16_t *__restrict__ host_switch,
    const uint8_t *__restrict__ region, pv_result *__restrict__ out, uint4 *__restrict__ recs,
    const uint32_t *__restrict__ seg,
    const uint32_t *__restrict__ pair_off, PolicyArgs pa, BindArgs ba) {
    for (uint32_t i = blockIdx.x * blockDim.x + threadIdx.x; i < M; i += gridDim.x * blockDim.x) {
        const uint32_t grp = i / ba.ppg, r = i - grp * ba.ppg, g = grp * ba.pods + r % ba.pods;
        const uint32_t node = ba.assign[g];
        const uint2 f = flow_at(ba, i);
        const bool placed = node < H;
        const uint32_t mask = ba.group_mask[grp];
        const uint32_t z = (f.y & 0xFFFFu) | (placed ? node : (uint32_t)PV_NO_HOST) << 16;
        if (probes)   // the caller's copy of the bound record {src_ip, dst_ip, dport | src_host << 16, mask}
            reinterpret_cast<uint4 *>(probes)[i] = make_uint4(placed ? ba.host_ip[node] : 0u, f.x, z, mask);
        if (kPolicy) pa.hits[i] = 0;
        if (!placed) {
            put_result(out, i, PV_NOSRC, 0, 0xFFFF);
            continue;
        }
        const uint32_t s = host_switch[node];
        if (first_switch_permitted<kPolicy>(pa, i, s, region[s], mask)) {
            const uint32_t slot = seg[s] + pair_off[g] + r / ba.pods;
            recs[slot] = make_uint4(i, f.x, z, mask);
        } else {
            put_result(out, i, PV_VIOLATION, 1, s);
        }
    }
}

// The same placement by one block per group, with each pair's run ordered
// by destination-port bucket of the first-match index, so the lanes of a
// first-hop warp mostly read the same few candidate lists.  The block brings
// its group's slice of the flows into shared memory with bulk copies (one
// per column, or one for records; the few elements outside the copies'
// 16-byte-aligned middles by plain loads), counts its probes per (pod,
// bucket), binds and judges them in one pass that drops each listed probe's
// rank into its pod's run (the next slot of its bucket), then writes every
// run out whole as walk records, so each sector of the records is written
// at once.  Used when the counts, ranks and flow slices fit
// kGroupInitSmem.
constexpr uint32_t kGroupInitMaxPods = 16;
constexpr uint32_t kGroupInitThreads = 512;
constexpr size_t kGroupInitSmem = 64 * 1024;   // ppg <= 65535 also fits the rank's 16 bits

// Shared-memory layout of walk_init_group_kernel: bucket counts / run
// slots [pods][kBuckets], ranks [ppg], then the destination slice and the
// port slice (the same slice for records), each with 16 bytes of slack so
// that its elements keep their global address modulo 16.
struct GroupInitSmem {
    uint32_t rank, dst, dport, total;
    __host__ __device__ GroupInitSmem(uint32_t pods, uint32_t ppg, bool records) {
        rank = pods * kBuckets * 4;
        dst = rank + ((ppg * 2 + 15) & ~15u);
        dport = dst + (records ? 0u : ((ppg * 4 + 16 + 15) & ~15u));
        total = dport + (records ? ppg * 8 + 16 : ((ppg * 2 + 16 + 15) & ~15u));
    }
};

// A slice of n elements of es bytes at global address src, staged in
// shared memory from s_base + (src mod 16), so that its 16-byte-aligned
// middle [b0, b1) can come by one bulk copy; the elements outside it
// (at most 15 bytes at each end, or all of them when there is no middle)
// come by plain loads.
struct Slice {
    uintptr_t a0, b0, b1;
    uint32_t n, es;
    __device__ Slice(const void *src, uint32_t n_, uint32_t es_) : n(n_), es(es_) {
        a0 = reinterpret_cast<uintptr_t>(src);
        b0 = (a0 + 15) & ~(uintptr_t)15;
        b1 = (a0 + (uintptr_t)n * es) & ~(uintptr_t)15;
        if (b1 < b0) b1 = b0;
    }
    __device__ uint32_t bulk_bytes() const { return (uint32_t)(b1 - b0); }
    __device__ uint8_t *staged(uint8_t *s_base) const { return s_base + (a0 & 15); }
};

// Thread 0 (after the barrier's expect-tx): the slice's bulk copy on bar.
__device__ __forceinline__ void slice_copy(const Slice &sl, uint8_t *s_base, uint64_t *bar) {
    if (sl.b1 > sl.b0)
        bulk_g2s_keep(sl.staged(s_base) + (sl.b0 - sl.a0), reinterpret_cast<const void *>(sl.b0), sl.bulk_bytes(),
                      bar);
}

// All threads: the slice's elements outside the bulk copy.
__device__ __forceinline__ void slice_edges(const Slice &sl, uint8_t *s_base) {
    const uint32_t n = sl.n, es = sl.es;
    const bool body = sl.b1 > sl.b0;
    const uint32_t lo = body ? (uint32_t)((sl.b0 - sl.a0) / es) : n;
    const uint32_t hi = body ? (uint32_t)((sl.b1 - sl.a0) / es) : n;
    uint8_t *dst = sl.staged(s_base);
    const void *src = reinterpret_cast<const void *>(sl.a0);
    for (uint32_t k = threadIdx.x; k < lo; k += blockDim.x) {
        if (es == 2) reinterpret_cast<uint16_t *>(dst)[k] = __ldg(reinterpret_cast<const uint16_t *>(src) + k);
        else reinterpret_cast<uint32_t *>(dst)[k * (es / 4)] = __ldg(reinterpret_cast<const uint32_t *>(src) + k * (es / 4));
        if (es == 8)
            reinterpret_cast<uint32_t *>(dst)[2 * k + 1] = __ldg(reinterpret_cast<const uint32_t *>(src) + 2 * k + 1);
    }
    for (uint32_t k = hi + threadIdx.x; k < n; k += blockDim.x) {
        if (es == 2) reinterpret_cast<uint16_t *>(dst)[k] = __ldg(reinterpret_cast<const uint16_t *>(src) + k);
        else reinterpret_cast<uint32_t *>(dst)[k * (es / 4)] = __ldg(reinterpret_cast<const uint32_t *>(src) + k * (es / 4));
        if (es == 8)
            reinterpret_cast<uint32_t *>(dst)[2 * k + 1] = __ldg(reinterpret_cast<const uint32_t *>(src) + 2 * k + 1);
    }
}

template <bool kPolicy>
__global__ void __launch_bounds__(kGroupInitThreads) walk_init_group_kernel(
    uint32_t M, pv_probe *__restrict__ probes, uint32_t H, const uint16_t *__restrict__ host_switch,
    const uint8_t *__restrict__ region, pv_result *__restrict__ out, uint4 *__restrict__ recs,
    const uint32_t *__restrict__ seg,
    const uint32_t *__restrict__ pair_off, PolicyArgs pa, BindArgs ba, uint64_t wait_ns, int32_t *status) {
    extern __shared__ __align__(16) uint8_t s_raw[];
    __shared__ uint32_t s_pair[kGroupInitMaxPods][3];   // per pod: {node, switch, listed}
    __shared__ uint64_t s_bar;
    const uint32_t grp = blockIdx.x, P = ba.pods, t = threadIdx.x, lane = t & 31, warp = t >> 5;
    const bool records = ba.dst_stride == 2;
    const GroupInitSmem L(P, ba.ppg, records);
    uint32_t *s_cur = reinterpret_cast<uint32_t *>(s_raw);                  // [pods][kBuckets] counts, then slots
    uint16_t *s_rank = reinterpret_cast<uint16_t *>(s_raw + L.rank);        // pod runs: ranks in the group
    const uint32_t first = grp * ba.ppg, len = min(ba.ppg, M - first);
    // the group's flows: destination and port slices (one slice for records)
    const Slice sa = records ? Slice(ba.dst + (size_t)first * 2, len, 8) : Slice(ba.dst + first, len, 4);
    const Slice sb = records ? Slice(ba.dst, 0, 8) : Slice(ba.dport + first, len, 2);
    if (t == 0) {
        mbar_init(&s_bar, 1);
        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
        mbar_arrive_expect_tx(&s_bar, sa.bulk_bytes() + sb.bulk_bytes());
        slice_copy(sa, s_raw + L.dst, &s_bar);
        slice_copy(sb, s_raw + L.dport, &s_bar);
    }
    slice_edges(sa, s_raw + L.dst);
    slice_edges(sb, s_raw + L.dport);
    const uint32_t *s_dst = reinterpret_cast<const uint32_t *>(sa.staged(s_raw + L.dst));
    const uint16_t *s_dport = records ? reinterpret_cast<const uint16_t *>(s_dst) + 2
                                      : reinterpret_cast<const uint16_t *>(sb.staged(s_raw + L.dport));
    const uint32_t ds = records ? 2u : 1u, ps = records ? 4u : 1u;
    const uint32_t mask = ba.group_mask[grp];
    for (uint32_t x = t; x < P * kBuckets; x += kGroupInitThreads) s_cur[x] = 0;
    if (t < P) {
        const uint32_t node = ba.assign[grp * P + t];
        const bool placed = node < H;
        const uint32_t sw = placed ? host_switch[node] : 0u;
        s_pair[t][0] = node;
        s_pair[t][1] = sw;
        s_pair[t][2] = placed && t < len && first_switch_permitted<kPolicy>(pa, first + t, sw, region[sw], mask);
    }
    __syncthreads();   // barrier initialised before anyone waits on it
    const bool ok = mbar_wait_bounded(&s_bar, 0, wait_ns);
    if (__syncthreads_or(!ok)) {
        // the flows did not arrive in time: report it (the call's results are
        // not to be used), wait for the copies once more (bounded), and bind
        // from global memory, so the later hops still read valid records
        if (t == 0) pv_device_error(status, PV_ETIMEOUT);
        mbar_wait_bounded(&s_bar, 0, wait_ns);
        s_dst = records ? ba.dst + (size_t)first * 2 : ba.dst + first;
        s_dport = records ? ba.dport + (size_t)first * 4 : ba.dport + first;
    }
    for (uint32_t r = t; r < len; r += kGroupInitThreads)
        atomicAdd(&s_cur[(r % P) * kBuckets + (s_dport[r * ps] >> kBucketShift)], 1u);
    __syncthreads();
    // exclusive scan of each pod's buckets, offset by the runs of the pods
    // before it (pod q holds probes q, q + P, ...: ceil((len - q) / P) of them)
    for (uint32_t q = warp; q < P; q += kGroupInitThreads / 32) {
        uint32_t *c = s_cur + q * kBuckets;
        constexpr uint32_t kPer = kBuckets / 32;
        uint32_t v[kPer], sum = 0;
        for (uint32_t j = 0; j < kPer; ++j) {
            v[j] = c[lane * kPer + j];
            sum += v[j];
        }
        uint32_t incl = sum;
        for (int d = 1; d < 32; d <<= 1) {
            const uint32_t y = __shfl_up_sync(PV_FULL_MASK, incl, d);
            if (lane >= (uint32_t)d) incl += y;
        }
        uint32_t before = 0;   // probes of pods 0 .. q - 1
        for (uint32_t q2 = 0; q2 < q; ++q2) before += len > q2 ? (len - q2 + P - 1) / P : 0u;
        uint32_t run = before + incl - sum;
        for (uint32_t j = 0; j < kPer; ++j) {
            c[lane * kPer + j] = run;
            run += v[j];
        }
    }
    __syncthreads();
    for (uint32_t r = t; r < len; r += kGroupInitThreads) {
        const uint32_t i = first + r, q = r % P;
        const uint32_t node = s_pair[q][0], sw = s_pair[q][1];
        const bool placed = node < H;
        const uint32_t dport = s_dport[r * ps];
        if (probes)   // the caller's copy of the bound record {src_ip, dst_ip, dport | src_host << 16, mask}
            reinterpret_cast<uint4 *>(probes)[i] = make_uint4(placed ? ba.host_ip[node] : 0u, s_dst[r * ds],
                                                              dport | (placed ? node : (uint32_t)PV_NO_HOST) << 16,
                                                              mask);
        if (kPolicy) pa.hits[i] = 0;
        if (s_pair[q][2]) {
            s_rank[atomicAdd(&s_cur[q * kBuckets + (dport >> kBucketShift)], 1u)] = (uint16_t)r;
        } else {
            put_result(out, i, placed ? PV_VIOLATION : PV_NOSRC, placed ? 1u : 0u, placed ? sw : 0xFFFFu);
        }
    }
    __syncthreads();
    uint32_t before = 0;
    for (uint32_t q = 0; q < P && q < len; ++q) {
        const uint32_t n = (len - q + P - 1) / P;
        if (s_pair[q][2]) {
            const uint32_t sw = s_pair[q][1];
            const uint32_t node = s_pair[q][0];
            const uint32_t base = seg[sw] + pair_off[grp * P + q];
            for (uint32_t k = t; k < n; k += kGroupInitThreads) {
                const uint32_t r = s_rank[before + k];
                recs[base + k] = make_uint4(first + r, s_dst[r * ds], s_dport[r * ps] | node << 16, mask);
            }
        }
        before += n;
    }
}

// A live-list entry is uint2 {probe id, loc}: loc bits 0..7 in_port, 8..23
// switch, 24..31 the hop at which a probe caught in a forwarding cycle is
// finished (plus one; 0 = not known to cycle).
__device__ __forceinline__ uint32_t entry_switch(uint32_t loc) { return (loc >> 8) & 0xFFFFu; }

// Forwarding-cycle shortcut.  For a fixed header the next location depends
// only on the current one (first match, action, port map, region check), so
// once a probe is back at a location it visited, its walk repeats with that
// period until the hop cap: it ends LOOP, hops = cap, at the switch it holds
// at hop cap - 1.  Locations are compared with a checkpoint taken at hops 4,
// 8, 16, ... (Brent's cycle detection); with period p found at hop h the
// probe walks only (cap - 1 - h) mod p more hops and is then finished with
// exactly the result the full walk gives.
constexpr uint32_t kCycleCheckFrom = 4;
// Bits 24..31 of a list entry's location hold the visit after which a probe
// in a known forwarding cycle finishes (1 .. cap - 1), 0, or kBounced: the
// probe left its last switch by the port it had entered through (a bounce).
// With symmetric cabling a bounce at the next switch too proves a two-switch
// cycle: state (switch, in_port) after the second bounce equals the state
// before the first, and the walk is a function of that state, so the visits
// alternate between the two switches until the hop cap.
constexpr uint32_t kBounced = 0xFFu;
__device__ __forceinline__ uint32_t loc_finish(uint32_t loc) {
    const uint32_t f = loc >> 24;
    return f == kBounced ? 0u : f;
}

// One block per list slice: per-switch histogram of the live probes.
__global__ void __launch_bounds__(kGridThreads) walk_hist_kernel(const uint2 *__restrict__ list,
                                                                 const uint2 *__restrict__ desc, uint32_t S,
                                                                 uint32_t *__restrict__ hist) {
    extern __shared__ uint32_t s_hist[];
    const uint2 d = desc[blockIdx.x];
    if (d.y == 0) return;
    const bool use_smem = S <= kSmemHistMax;
    if (use_smem) {
        for (uint32_t j = threadIdx.x; j < S; j += kGridThreads) s_hist[j] = 0;
        __syncthreads();
    }
    for (uint32_t i = d.x + threadIdx.x; i < d.x + d.y; i += kGridThreads) {
        const uint32_t s = entry_switch(list[i].y);
        if (use_smem) atomicAdd(&s_hist[s], 1u);
        else atomicAdd(&hist[s], 1u);
    }
    if (use_smem) {
        __syncthreads();
        for (uint32_t j = threadIdx.x; j < S; j += kGridThreads)
            if (s_hist[j]) atomicAdd(&hist[j], s_hist[j]);
    }
}

// Single block: seg[s] = exclusive prefix of hist, seg[S] = total,
// seg[S + 1] = switches holding at least one probe; cursor[s] = seg[s];
// hist cleared for the next hop.
__global__ void __launch_bounds__(1024) walk_scan_kernel(uint32_t S, uint32_t *__restrict__ hist,
                                                         uint32_t *__restrict__ seg, uint32_t *__restrict__ cursor) {
    __shared__ uint32_t s_warp[32];
    __shared__ uint32_t s_carry;
    const uint32_t t = threadIdx.x, lane = t & 31, warp = t >> 5;
    uint32_t nonempty = 0;
    if (t == 0) s_carry = 0;
    __syncthreads();
    for (uint32_t c0 = 0; c0 < S; c0 += 1024) {
        const uint32_t i = c0 + t;
        const uint32_t x = i < S ? hist[i] : 0;
        nonempty += (uint32_t)__syncthreads_count(x > 0);
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
        if (i < S) {
            seg[i] = excl;
            cursor[i] = excl;
            hist[i] = 0;
        }
        __syncthreads();
        if (t == 1023) s_carry = excl + x;
        __syncthreads();
    }
    if (t == 0) {
        seg[S] = s_carry;
        seg[S + 1] = nonempty;
    }
}

// One block per list slice: block-aggregated counting-sort scatter (one
// atomicAdd per (block, switch) reserves a contiguous run).
__global__ void __launch_bounds__(kGridThreads) walk_scatter_kernel(const uint2 *__restrict__ list,
                                                                    const uint2 *__restrict__ desc, uint32_t S,
                                                                    uint32_t *__restrict__ cursor,
                                                                    uint2 *__restrict__ sorted) {
    extern __shared__ uint32_t s_cnt[];   // [S] counts, then [S] bases
    const uint2 d = desc[blockIdx.x];
    if (d.y == 0) return;
    const uint32_t b0 = d.x, b1 = d.x + d.y;
    if (S > kSmemHistMax) {
        for (uint32_t i = b0 + threadIdx.x; i < b1; i += kGridThreads) {
            const uint2 e = list[i];
            sorted[atomicAdd(&cursor[entry_switch(e.y)], 1u)] = e;
        }
        return;
    }
    uint32_t *s_base = s_cnt + S;
    for (uint32_t j = threadIdx.x; j < S; j += kGridThreads) s_cnt[j] = 0;
    __syncthreads();
    // both passes keep four independent list loads in flight per thread
    constexpr uint32_t kU = 4, kStep = kU * kGridThreads;
    for (uint32_t i0 = b0 + threadIdx.x; i0 < b1; i0 += kStep) {
        uint32_t loc[kU];
#pragma unroll
        for (uint32_t j = 0; j < kU; ++j) loc[j] = i0 + j * kGridThreads < b1 ? list[i0 + j * kGridThreads].y : 0u;
#pragma unroll
        for (uint32_t j = 0; j < kU; ++j)
            if (i0 + j * kGridThreads < b1) atomicAdd(&s_cnt[entry_switch(loc[j])], 1u);
    }
    __syncthreads();
    for (uint32_t j = threadIdx.x; j < S; j += kGridThreads) {
        const uint32_t c = s_cnt[j];
        s_base[j] = c ? atomicAdd(&cursor[j], c) : 0;
        s_cnt[j] = 0;
    }
    __syncthreads();
    for (uint32_t i0 = b0 + threadIdx.x; i0 < b1; i0 += kStep) {
        uint2 e[kU];
#pragma unroll
        for (uint32_t j = 0; j < kU; ++j) e[j] = i0 + j * kGridThreads < b1 ? list[i0 + j * kGridThreads] : make_uint2(0, 0);
#pragma unroll
        for (uint32_t j = 0; j < kU; ++j)
            if (i0 + j * kGridThreads < b1) {
                const uint32_t s = entry_switch(e[j].y);
                sorted[s_base[s] + atomicAdd(&s_cnt[s], 1u)] = e[j];
            }
    }
}

struct HopArgs {
    const uint2 *sorted;
    uint32_t hop, cap;
    const uint32_t *seg;
    uint32_t S, H;
    const uint8_t *blob;
    const uint64_t *blob_offs;
    const uint8_t *region;
    const uint32_t *port_offs;
    const int32_t *port_peer;
    const uint32_t *host_ip;
    const pv_probe *probes;
    const uint4 *recs;   // walk records (kRec kernels)
    pv_result *out;
    uint2 *next_list;
    uint2 *next_desc;
    int32_t *status;
    uint32_t lane_max;   // longest candidate list handled one probe per lane
    uint32_t wait_extra; // bytes the staging barrier expects beyond the copy (0; > 0 only in failure tests)
    uint64_t wait_ns;    // bound on each staging wait
    uint32_t *hop_live;  // [cap]: live probes processed at each hop (statistics)
    uint32_t *ck;        // [M]: cycle-detection checkpoint location per probe
    uint32_t cycles;     // 1: finish probes caught in forwarding cycles early
    uint32_t bounce;     // 1: finish two-switch cycles at their second bounce (symmetric cabling)
    PolicyArgs pa;       // path constraints (used by the kPolicy kernels)
    uint32_t *hist_next; // per-switch counts of the next hop's list (null: a separate pass counts)
    uint32_t hist_off;   // byte offset of the block's count array in dynamic shared memory
    uint32_t port_off;   // byte offset of the staged port table in dynamic shared memory
    uint32_t recs_at_position;   // 1: no list, entry i is record i (first hop of directly placed flows)
    const uint2 *host_addr;      // [H] {address, attachment port} of each host
    const uint2 *port_stage;     // [ports] {peer, aux} as the hop kernel stages them
    unsigned long long *stats;   // [PV_WALK_STATS] counters of the statistics kernels (kStats)
};

// Walk statistics (kStats kernels): first matches resolved, index rule
// tests, interval lookups, the rules a scan in first-match order tests
// before its first hit (all of the switch's rules on a miss), and first
// matches where that scan and the kernel disagree.
enum { kStFirstMatches = 0, kStRuleTests, kStLookups, kStLinearDepth, kStMismatch, kStCount };

// First match by a plain scan of the compiled rules in first-match order
// (smem or global): the statistics kernels' reference for depth and result.
// *depth = position of the hit + 1, or the number of rules on a miss.
__device__ __forceinline__ uint32_t scan_first_match(const uint4 *A, const uint2 *Bv, uint32_t npad, uint32_t src,
                                                     uint32_t dst, uint32_t dport, uint32_t in_port,
                                                     uint32_t *depth) {
    for (uint32_t r = 0; r < npad; ++r) {
        const uint2 b = Bv[r];
        if (b.x == 1u) {   // padding (lo 1 > hi 0): the table has r rules
            *depth = r;
            return 0u;
        }
        const uint4 a = A[r];
        const uint32_t diff = ((src ^ a.x) & a.y) | ((dst ^ a.z) & a.w) | ((in_port ^ b.y) & ((b.y >> 8) & 0xFFu));
        if (diff == 0 && dport >= (b.x & 0xFFFFu) && dport <= (b.x >> 16)) {
            *depth = r + 1;
            return kWinFound | (b.y >> 16);
        }
    }
    *depth = npad;
    return 0u;
}

// Adds one thread's statistics to the walk's counters (one atomic per warp
// and counter).
__device__ __forceinline__ void flush_stats(unsigned long long *stats, const uint32_t (&c)[kStCount]) {
    const uint32_t lane = threadIdx.x & 31;
#pragma unroll
    for (int i = 0; i < kStCount; ++i) {
        unsigned long long v = c[i];
        for (int o = 16; o > 0; o >>= 1) v += __shfl_down_sync(PV_FULL_MASK, v, o);
        if (lane == 0 && v) atomicAdd(stats + i, v);
    }
}

// Linear first match: 32 consecutive rules per warp step.
// Both first-match routines return kWinFound | action, or 0 for a table miss.
// A walk reads a probe's header through its list entry's first field: the
// caller's probe record (pv_verify_probes; the field is the probe id) or,
// for compact flows placed directly, the walk record the first kernel wrote
// at the probe's first-hop slot, {probe id, dst_ip, dport | src_host << 16,
// allowed_mask}, whose source address comes from the host table (kRec): the
// first hop then reads its records in list order.
template <bool kRec>
__device__ __forceinline__ uint4 load_header(const HopArgs &g, uint32_t x, uint32_t *id) {
    if (kRec) {
        const uint4 r = __ldg(g.recs + x);
        *id = r.x;
        return make_uint4(__ldg(g.host_ip + (r.z >> 16)), r.y, r.z, r.w);
    }
    *id = x;
    return __ldg(reinterpret_cast<const uint4 *>(g.probes) + x);
}

// The same in two steps, so the record's load can run ahead of its use:
// the record (or probe) at index x, then the header and probe id from it.
template <bool kRec>
__device__ __forceinline__ uint4 load_raw(const HopArgs &g, uint32_t x) {
    return kRec ? __ldg(g.recs + x) : __ldg(reinterpret_cast<const uint4 *>(g.probes) + x);
}

template <bool kRec>
__device__ __forceinline__ uint4 header_of(const HopArgs &g, uint4 raw, uint32_t x, uint32_t *id,
                                           uint32_t *src_port) {
    if (kRec) {
        *id = raw.x;
        const uint2 ha = __ldg(g.host_addr + (raw.z >> 16));   // the source host's address and port
        *src_port = ha.y;
        return make_uint4(ha.x, raw.y, raw.z, raw.w);
    }
    *id = x;
    return raw;
}

template <bool kStats>
__device__ __forceinline__ uint32_t first_match_linear(const uint8_t *sm, uint32_t npad, uint32_t lane, uint32_t src,
                                                       uint32_t dst, uint32_t dport, uint32_t in_port,
                                                       uint32_t &tests) {
    const uint4 *sA = reinterpret_cast<const uint4 *>(sm + 16);               // staged by the linear kernel
    const uint2 *sB = reinterpret_cast<const uint2 *>(sm + 16 + npad * 16);
    for (uint32_t base = 0; base < npad; base += 32) {
        const uint4 a = sA[base + lane];
        const uint2 b = sB[base + lane];
        const uint32_t diff = ((src ^ a.x) & a.y) | ((dst ^ a.z) & a.w) | ((in_port ^ b.y) & ((b.y >> 8) & 0xFFu));
        const bool hit = diff == 0 && dport >= (b.x & 0xFFFFu) && dport <= (b.x >> 16);
        const uint32_t m = __ballot_sync(PV_FULL_MASK, hit);
        if (kStats) tests += 32;
        if (m) return kWinFound | __shfl_sync(PV_FULL_MASK, b.y >> 16, __ffs(m) - 1);
    }
    return 0u;
}

// The boundary range of a segment that holds dst's interval, from the
// segment's jump block jb (shared or global memory): the answer (the last
// boundary <= dst) is in [*lo, *lo + *len).
__device__ __forceinline__ void jump_range(const uint8_t *jb, uint32_t dst, uint32_t *lo, uint32_t *len) {
    const uint2 bs = *reinterpret_cast<const uint2 *>(jb);   // {base, shift}
    if (dst < bs.x) {
        *lo = 0;
        *len = 1;
        return;
    }
    const uint32_t j = min((dst - bs.x) >> bs.y, kJumpSlots - 1);
    const uint16_t *J = reinterpret_cast<const uint16_t *>(jb + 8);
    const uint32_t a = J[j], b = J[j + 1];
    *lo = a;
    *len = b - a + 1;
}

// Winner of the elementary interval holding dst: the warp narrows the range
// 32-ways per step (bnd ascending, bnd[0] = 0 <= dst).
__device__ __forceinline__ uint32_t segment_lookup(const uint32_t *bnd, const uint32_t *win, uint32_t cnt,
                                                   uint32_t dst, uint32_t lane) {
    uint32_t lo = 0, len = cnt;
    while (len > 32) {
        const uint32_t stride = (len + 31) / 32;
        const bool le = lane * stride < len && bnd[lo + lane * stride] <= dst;
        const uint32_t c = __popc(__ballot_sync(PV_FULL_MASK, le));
        lo += (c - 1) * stride;
        len = min(stride, len - (c - 1) * stride);
    }
    const bool le = lane < len && bnd[lo + lane] <= dst;
    const uint32_t c = __popc(__ballot_sync(PV_FULL_MASK, le));
    return win[lo + c - 1];
}

// Indexed first match: walk the dport bucket's candidate list in first-match
// order, 32 items per step; segment items are answered by interval lookup.
template <bool kStats>
__device__ __forceinline__ uint32_t first_match_indexed(const uint8_t *sm, const uint4 hdr, uint32_t lane,
                                                        uint32_t src, uint32_t dst, uint32_t dport, uint32_t in_port,
                                                        uint32_t &tests, uint32_t &lookups) {
    const BlobLayout L(hdr);
    const uint4 *sA = reinterpret_cast<const uint4 *>(sm + L.a);
    const uint2 *sB = reinterpret_cast<const uint2 *>(sm + L.b);
    const uint32_t *boff = reinterpret_cast<const uint32_t *>(sm + L.boff);
    const uint16_t *items = reinterpret_cast<const uint16_t *>(sm + L.items);
    const uint2 *segs = reinterpret_cast<const uint2 *>(sm + L.segs);
    const uint32_t *bnd = reinterpret_cast<const uint32_t *>(sm + L.bnd);
    const uint32_t *win = reinterpret_cast<const uint32_t *>(sm + L.win);
    const uint32_t k = dport >> kBucketShift;
    const uint32_t i0 = boff[k], i1 = boff[k + 1];
    for (uint32_t c0 = i0; c0 < i1; c0 += 32) {
        const uint32_t idx = c0 + lane;
        const uint32_t it = idx < i1 ? items[idx] : 0xFFFFu;
        const bool valid = it != 0xFFFFu;
        const bool is_seg = valid && (it & kSegItem);
        bool hit = false;
        uint32_t action = 0;
        if (valid && !is_seg) {
            const uint4 a = sA[it];
            const uint2 b = sB[it];
            const uint32_t diff = ((src ^ a.x) & a.y) | ((dst ^ a.z) & a.w) | ((in_port ^ b.y) & ((b.y >> 8) & 0xFFu));
            hit = diff == 0 && dport >= (b.x & 0xFFFFu) && dport <= (b.x >> 16);
            action = b.y >> 16;
        }
        uint32_t G = __ballot_sync(PV_FULL_MASK, hit);
        uint32_t Sg = __ballot_sync(PV_FULL_MASK, is_seg);
        if (kStats) tests += __popc(__ballot_sync(PV_FULL_MASK, valid && !is_seg));
        while (true) {
            const uint32_t pg = G ? (uint32_t)__ffs(G) - 1 : 32u;
            const uint32_t ps = Sg ? (uint32_t)__ffs(Sg) - 1 : 32u;
            if (ps < pg) {
                const uint2 sd = segs[__shfl_sync(PV_FULL_MASK, it, ps) & 0x7FFFu];
                const uint32_t w = segment_lookup(bnd + sd.x, win + sd.x, sd.y, dst, lane);
                if (kStats) ++lookups;
                if (w & kWinFound) return w;
                Sg &= Sg - 1u;
            } else if (pg < 32u) {
                return kWinFound | __shfl_sync(PV_FULL_MASK, action, pg);
            } else {
                break;
            }
        }
    }
    return 0u;
}

// Scalar first match, one probe per lane (called by all 32 lanes; inactive
// lanes return 0): each lane walks its bucket's candidate list in order.
// Plain rules are tested until a hit or a segment token; the warp then
// reconverges and the lanes parked on a segment token run their interval
// binary searches together (a segment miss resumes the walk after the token).
template <bool kStats>
__device__ __forceinline__ uint32_t first_match_lane(const uint8_t *sm, const BlobLayout &L, bool active,
                                                     uint32_t src, uint32_t dst, uint32_t dport, uint32_t in_port,
                                                     uint32_t &tests, uint32_t &lookups) {
    const uint4 *sA = reinterpret_cast<const uint4 *>(sm + L.a);
    const uint2 *sB = reinterpret_cast<const uint2 *>(sm + L.b);
    const uint32_t *boff = reinterpret_cast<const uint32_t *>(sm + L.boff);
    const uint16_t *items = reinterpret_cast<const uint16_t *>(sm + L.items);
    const uint2 *segs = reinterpret_cast<const uint2 *>(sm + L.segs);
    const uint32_t *bnd = reinterpret_cast<const uint32_t *>(sm + L.bnd);
    const uint32_t *win = reinterpret_cast<const uint32_t *>(sm + L.win);
    const uint32_t k = dport >> kBucketShift;
    uint32_t i = active ? boff[k] : 0u, i1 = active ? boff[k + 1] : 0u;
    uint32_t result = 0;
    bool done = !active;
    while (__any_sync(PV_FULL_MASK, !done)) {
        uint32_t seg = 0xFFFFFFFFu;
        if (!done) {
            // two items per step, both rules loaded before either is tested
            // (a segment token's slot loads rule 0, unused)
            auto hit = [&](uint4 a, uint2 bb) {
                const uint32_t diff =
                    ((src ^ a.x) & a.y) | ((dst ^ a.z) & a.w) | ((in_port ^ bb.y) & ((bb.y >> 8) & 0xFFu));
                return diff == 0 && dport >= (bb.x & 0xFFFFu) && dport <= (bb.x >> 16);
            };
            for (; i < i1; i += 2) {
                const uint32_t it0 = items[i];
                const bool has1 = i + 1 < i1;
                const uint32_t it1 = has1 ? items[i + 1] : 0u;
                const uint32_t r0 = (it0 & kSegItem) ? 0u : it0, r1 = (it1 & kSegItem) ? 0u : it1;
                const uint4 a0 = sA[r0], a1 = sA[r1];
                const uint2 b0 = sB[r0], b1 = sB[r1];
                if (it0 & kSegItem) {
                    seg = it0 & 0x7FFFu;
                    break;
                }
                if (kStats) ++tests;
                if (hit(a0, b0)) {
                    result = kWinFound | (b0.y >> 16);
                    done = true;
                    break;
                }
                if (!has1) break;
                if (it1 & kSegItem) {
                    seg = it1 & 0x7FFFu;
                    ++i;   // i names the token, so a segment miss resumes after it
                    break;
                }
                if (kStats) ++tests;
                if (hit(a1, b1)) {
                    result = kWinFound | (b1.y >> 16);
                    done = true;
                    break;
                }
            }
            if (!done && seg == 0xFFFFFFFFu) done = true;   // list exhausted: table miss
        }
        __syncwarp();
        if (seg != 0xFFFFFFFFu) {
            const uint2 sd = segs[seg];
            const uint32_t *b = bnd + sd.x;
            uint32_t lo, len;   // b[lo] <= dst; answer in [lo, lo + len)
            jump_range(sm + L.jmp + seg * kJumpBytes, dst, &lo, &len);
            while (len > 1) {
                const uint32_t half = len >> 1;
                lo = b[lo + half] <= dst ? lo + half : lo;
                len -= half;
            }
            const uint32_t w = win[sd.x + lo];
            if (kStats) ++lookups;
            if (w & kWinFound) {
                result = w;
                done = true;
            } else {
                ++i;
            }
        }
    }
    return result;
}

// Outcome of one hop at a permitted switch given the first match fm
// (kWinFound | action, or 0): a terminal status, kViolationNext (the next
// switch is outside the probe's jurisdictions: the walk ends there, one hop
// later), or kAlive with the next location.  Checking the next switch's
// region here, when the probe is handed on, is the region check of the next
// visit done early, so live lists only hold probes permitted where they are.
constexpr uint32_t kAlive = 0xFFu;
constexpr uint32_t kViolationNext = 0xFEu;

__device__ __forceinline__ void hop_outcome(const HopArgs &g, uint32_t hop, uint32_t fm, uint32_t dst, uint32_t mask,
                                            uint32_t pbase, uint32_t nports, uint32_t *status, uint32_t *next) {
    *next = 0;
    const uint32_t act = fm & 0xFFFFu;
    if (!(fm & kWinFound) || act == PV_DROP || act >= nports) {
        *status = PV_DROPPED;
        return;
    }
    const int32_t peer = g.port_peer[pbase + act];
    if (peer < 0) {
        *status = PV_DROPPED;
    } else if (peer & PV_PEER_HOST) {
        const uint32_t q = (uint32_t)(peer & ~PV_PEER_HOST);
        *status = (q < g.H && g.host_ip[q] == dst) ? PV_COMPLIANT : PV_MISDELIVERED;
    } else if (hop + 1 >= g.cap) {
        *status = PV_LOOP;
    } else {
        const uint32_t r2 = g.region[(uint32_t)peer >> 8];
        *status = (r2 < 32 && ((mask >> r2) & 1u)) ? kAlive : kViolationNext;
        *next = (uint32_t)peer;
    }
}

// The hop kernel stages the current switch's ports once per table from the
// port stage the table loader builds (port_stage_kernel): port p as {peer,
// aux}, aux = the region of the peer switch, or the address of the attached
// host, so a hop's outcome reads shared memory only.
// hop_outcome with the port table staged in shared memory (same outcomes).
__device__ __forceinline__ void hop_outcome_staged(const HopArgs &g, const uint2 *s_port, uint32_t hop, uint32_t fm,
                                                   uint32_t dst, uint32_t mask, uint32_t nports, uint32_t *status,
                                                   uint32_t *next) {
    *next = 0;
    const uint32_t act = fm & 0xFFFFu;
    if (!(fm & kWinFound) || act == PV_DROP || act >= nports) {
        *status = PV_DROPPED;
        return;
    }
    const uint2 pe = s_port[act];
    const int32_t peer = (int32_t)pe.x;
    if (peer < 0) {
        *status = PV_DROPPED;
    } else if (peer & PV_PEER_HOST) {
        const uint32_t q = (uint32_t)(peer & ~PV_PEER_HOST);
        *status = (q < g.H && pe.y == dst) ? PV_COMPLIANT : PV_MISDELIVERED;
    } else if (hop + 1 >= g.cap) {
        *status = PV_LOOP;
    } else {
        const uint32_t r2 = pe.y;
        *status = (r2 < 32 && ((mask >> r2) & 1u)) ? kAlive : kViolationNext;
        *next = (uint32_t)peer;
    }
}

// kFirst: the walk's first hop, where every entry's finish field is 0, its
// in_port is the source host's port (so a live probe never bounces) and no
// cycle check is due, so all of that is left out.
template <bool kIndexed, bool kPolicy, bool kStats, bool kRec, bool kFirst>
__global__ void __launch_bounds__(kHopThreads, 4) walk_hop_kernel(HopArgs g) {
    extern __shared__ __align__(128) uint8_t s_raw[];
    __shared__ uint64_t s_bar;
    __shared__ uint32_t s_count;
    const uint32_t lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const uint32_t n = g.seg[g.S];   // live probes this hop
    if (blockIdx.x == 0 && threadIdx.x == 0) g.hop_live[g.hop] = n;
    // blocks: enough for kMinPerBlock probes each (a block stages a whole
    // switch table, which small shares would not repay), but at least one per
    // switch holding probes (else few blocks stage many tables one by one)
    const uint32_t want = max((n + kMinPerBlock - 1) / kMinPerBlock, g.seg[g.S + 1]);
    const uint32_t active = max(1u, min(gridDim.x, want));
    const uint32_t r0 = blockIdx.x < active ? (uint32_t)(((uint64_t)n * blockIdx.x) / active) : n;
    const uint32_t r1 = blockIdx.x < active ? (uint32_t)(((uint64_t)n * (blockIdx.x + 1)) / active) : n;
    if (r0 >= r1) {
        if (threadIdx.x == 0) g.next_desc[blockIdx.x] = make_uint2(r0, 0);
        return;
    }
    if (threadIdx.x == 0) {
        mbar_init(&s_bar, 1);
        s_count = 0;
    }
    uint32_t *s_hist = reinterpret_cast<uint32_t *>(s_raw + g.hist_off);   // [S] when g.hist_next
    uint2 *s_port = reinterpret_cast<uint2 *>(s_raw + g.port_off);        // [ports of the current switch]
    if (g.hist_next)
        for (uint32_t j = threadIdx.x; j < g.S; j += kHopThreads) s_hist[j] = 0;
    __syncthreads();
    uint32_t parity = 0;
    uint32_t pos = r0;
    uint32_t stc[kStCount] = {};
    while (pos < r1) {
        // switch owning position pos: the last s with seg[s] <= pos (empty
        // switches repeat their successor's start), found by each warp with
        // a 32-way search (two rounds of loads for 512 switches)
        uint32_t lo = 0, len = g.S;   // seg[lo] <= pos; answer in [lo, lo + len)
        while (len > 1) {
            const uint32_t stride = (len + 31) >> 5;
            const bool le = lane * stride < len && __ldg(g.seg + lo + lane * stride) <= pos;
            const uint32_t c = __popc(__ballot_sync(PV_FULL_MASK, le));   // lane 0 always
            lo += (c - 1) * stride;
            len = min(stride, len - (c - 1) * stride);
        }
        const uint32_t s = lo;
        const uint32_t seg_end = min(r1, g.seg[s + 1]);
        const uint8_t *src_blob = g.blob + g.blob_offs[s];
        const uint4 hdr = __ldg(reinterpret_cast<const uint4 *>(src_blob));
        const BlobLayout L(hdr);
        const uint32_t npad = hdr.x & 0xFFFFu;
        const uint32_t pbase = g.port_offs[s], nports = g.port_offs[s + 1] - pbase;
        __syncthreads();   // everyone is done with the previous table and ports
        if (threadIdx.x == 0) {
            asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
            if (kIndexed) {   // header, plain rules, index
                mbar_arrive_expect_tx(&s_bar, L.fa + g.wait_extra);
                bulk_g2s_keep(s_raw, src_blob, L.fa, &s_bar);
            } else {          // header and the full rule list
                mbar_arrive_expect_tx(&s_bar, linear_bytes(npad) + g.wait_extra);
                bulk_g2s_keep(s_raw, src_blob, 16, &s_bar);
                if (npad) bulk_g2s_keep(s_raw + 16, src_blob + L.fa, npad * 24, &s_bar);
            }
        }
        for (uint32_t p = threadIdx.x; p < nports; p += kHopThreads) s_port[p] = __ldg(g.port_stage + pbase + p);
        const bool ok = mbar_wait_bounded(&s_bar, parity, g.wait_ns);
        if (__syncthreads_or(!ok)) {
            // give up: record the timeout, leave an empty slice for the next
            // hop, let the copy in flight land (bounded again), return.
            // Accepted edge case: a copy still in flight after both bounds
            // (4 s for a copy of at most a few hundred KB) may land after
            // the block has exited; the call then reports PV_ETIMEOUT and
            // its results are not to be used.
            if (threadIdx.x == 0) {
                pv_device_error(g.status, PV_ETIMEOUT);
                g.next_desc[blockIdx.x] = make_uint2(r0, 0);
            }
            mbar_wait_bounded(&s_bar, parity, g.wait_ns);
            return;
        }
        parity ^= 1u;   // the barrier above also published s_port
        // Lane j handles probe j of each batch of 32.  Loads run ahead of the
        // batch in hand: the list entry two batches ahead and the record one
        // batch ahead (its index comes from the entry fetched a batch
        // earlier), so neither waits on the other or on the batch's work.
        constexpr uint32_t kStride = 32 * kHopWarps;
        const uint32_t wb0 = pos + warp * 32;
        // At the first hop of directly placed flows there is no list: entry
        // i is record i, and its in_port is its source host's port.
        const bool at_pos = kRec && g.recs_at_position != 0;
        uint2 e1 = make_uint2(0, 0), e2 = make_uint2(0, 0);   // entries of batches wb, wb + kStride
        uint4 raw1 = make_uint4(0, 0, 0, 0);                  // record of batch wb
        if (wb0 + lane < seg_end) {
            e1 = at_pos ? make_uint2(wb0 + lane, 0) : g.sorted[wb0 + lane];
            raw1 = load_raw<kRec>(g, e1.x);
        }
        if (wb0 + kStride + lane < seg_end)
            e2 = at_pos ? make_uint2(wb0 + kStride + lane, 0) : g.sorted[wb0 + kStride + lane];
        for (uint32_t wb = wb0; wb < seg_end; wb += kStride) {
            const uint32_t cnt = min(32u, seg_end - wb);
            uint2 e = e1;
            const uint4 raw = raw1;
            if (wb + kStride + lane < seg_end) raw1 = load_raw<kRec>(g, e2.x);
            e1 = e2;
            if (wb + 2 * kStride + lane < seg_end)
                e2 = at_pos ? make_uint2(wb + 2 * kStride + lane, 0) : g.sorted[wb + 2 * kStride + lane];
            uint4 pr = make_uint4(0, 0, 0, 0);   // {src_ip, dst_ip, dport | src_host << 16, allowed_mask}
            uint32_t pid = 0;                     // probe id
            if (lane < cnt) {
                uint32_t src_port = 0;
                pr = header_of<kRec>(g, raw, e.x, &pid, &src_port);
                if (at_pos) e.y = src_port;
            }
            // a probe in a known forwarding cycle that has reached its finish hop
            const uint32_t fin = kFirst ? 0u : loc_finish(e.y);
            const bool fin_now = !kFirst && lane < cnt && fin != 0 && fin - 1 == g.hop;
            const uint32_t fin_lanes = kFirst ? 0u : __ballot_sync(PV_FULL_MASK, fin_now);
            uint32_t my_status = fin_now ? (uint32_t)PV_LOOP : kAlive, my_next = 0, my_fm = 0;
            // Every listed probe is permitted at s (checked when it was handed
            // on).  Lane-per-probe when every candidate list of the batch is short.
            bool lane_mode = false;
            if (kIndexed) {
                const uint32_t *boff = reinterpret_cast<const uint32_t *>(s_raw + L.boff);
                uint32_t len = 0;
                if (lane < cnt) {
                    const uint32_t k = (pr.z & 0xFFFFu) >> kBucketShift;
                    len = boff[k + 1] - boff[k];
                }
                lane_mode = __reduce_max_sync(PV_FULL_MASK, len) <= g.lane_max;
            }
            if (lane_mode) {
                const bool act = lane < cnt && !fin_now;
                const uint32_t fm = first_match_lane<kStats>(s_raw, L, act, pr.x, pr.y, pr.z & 0xFFFFu, e.y & 0xFFu,
                                                             stc[kStRuleTests], stc[kStLookups]);
                my_fm = fm;
                if (act) hop_outcome_staged(g, s_port, g.hop, fm, pr.y, pr.w, nports, &my_status, &my_next);
            } else {
                for (uint32_t j = 0; j < cnt; ++j) {
                    if ((fin_lanes >> j) & 1u) continue;
                    const uint32_t in_port = __shfl_sync(PV_FULL_MASK, e.y, j) & 0xFFu;
                    const uint32_t src = __shfl_sync(PV_FULL_MASK, pr.x, j);
                    const uint32_t dst = __shfl_sync(PV_FULL_MASK, pr.y, j);
                    const uint32_t dport = __shfl_sync(PV_FULL_MASK, pr.z, j) & 0xFFFFu;
                    const uint32_t mask = __shfl_sync(PV_FULL_MASK, pr.w, j);
                    uint32_t tests = 0, lookups = 0;
                    const uint32_t fm =
                        kIndexed ? first_match_indexed<kStats>(s_raw, hdr, lane, src, dst, dport, in_port, tests, lookups)
                                 : first_match_linear<kStats>(s_raw, npad, lane, src, dst, dport, in_port, tests);
                    uint32_t status, next;
                    hop_outcome_staged(g, s_port, g.hop, fm, dst, mask, nports, &status, &next);
                    if (lane == j) {
                        my_status = status;
                        my_next = next;
                        my_fm = fm;
                        if (kStats) {
                            stc[kStRuleTests] += tests;
                            stc[kStLookups] += lookups;
                        }
                    }
                }
            }
            if (kStats && lane < cnt && !fin_now) {
                uint32_t depth = 0;
                // the full rule list: staged by the linear kernel, read from
                // the blob by the indexed one
                const uint4 *fa = reinterpret_cast<const uint4 *>(kIndexed ? src_blob + L.fa : s_raw + 16);
                const uint2 *fb = reinterpret_cast<const uint2 *>(kIndexed ? src_blob + L.fb : s_raw + 16 + npad * 16);
                const uint32_t ref = scan_first_match(fa, fb, npad, pr.x, pr.y, pr.z & 0xFFFFu, e.y & 0xFFu, &depth);
                ++stc[kStFirstMatches];
                stc[kStLinearDepth] += depth;
                stc[kStMismatch] += ref != my_fm ? 1u : 0u;
            }
            if (kPolicy && lane < cnt && !fin_now) {
                const uint4 ph = policy_of(g.pa, pid);
                uint32_t bits = 0;   // waypoints of the probe's policy at this switch
                for (uint32_t i = 0; i < ph.w; ++i)
                    if (g.pa.sw[ph.z + i] == s) bits |= 1u << i;
                if (bits) g.pa.hits[pid] |= bits;
                if (my_status == kAlive && switch_listed(g.pa.sw + ph.x, ph.y, my_next >> 8))
                    my_status = kViolationNext;   // the next switch is forbidden to this flow
            }
            // a bounce (out by the port it came in by) right after a bounce: a
            // two-switch cycle, whose visit cap - 1 (the walk's last) is at s
            // or at the next switch by parity
            const bool bounce = !kFirst && (my_fm & 0xFFFFu) == (e.y & 0xFFu);
            const bool pingpong = !kFirst && (e.y >> 24) == kBounced && lane < cnt && my_status == kAlive && bounce;
            if (lane < cnt && my_status != kAlive) {
                const bool at_next = my_status == kViolationNext;
                put_result(g.out, pid, at_next ? (uint32_t)PV_VIOLATION : my_status,
                           fin_now ? g.cap : g.hop + (at_next ? 2u : 1u), at_next ? (my_next >> 8) : s);
            } else if (pingpong) {
                put_result(g.out, pid, PV_LOOP, g.cap, ((g.cap - 1u - g.hop) & 1u) ? (my_next >> 8) : s);
            }
            const bool live = lane < cnt && my_status == kAlive && !pingpong;
            uint32_t nloc = my_next;
            if (live) {
                uint32_t nfin = fin;
                const uint32_t h1 = g.hop + 1;   // hop of the next visit (< cap)
                if (!kFirst && g.cycles && nfin == 0 && h1 >= kCycleCheckFrom) {
                    if ((h1 & (h1 - 1u)) == 0) {
                        g.ck[e.x] = my_next;   // new checkpoint
                    } else if (g.ck[e.x] == my_next) {
                        const uint32_t period = h1 - (1u << (31 - __clz(h1)));
                        nfin = h1 + (g.cap - 1u - h1) % period + 1u;
                        if (nfin >= g.cap) nfin = 0;   // finishing at visit cap - 1 is the plain walk's end
                    }
                }
                if (nfin == 0 && g.bounce && bounce) nfin = kBounced;
                nloc = my_next | (nfin << 24);
            }
            const uint32_t slot = warp_reserve(live, &s_count);
            if (live) {
                g.next_list[r0 + slot] = make_uint2(e.x, nloc);
                if (g.hist_next) atomicAdd(&s_hist[entry_switch(nloc)], 1u);
            }
        }
        pos = seg_end;
    }
    if (kStats) flush_stats(g.stats, stc);
    __syncthreads();
    if (threadIdx.x == 0) g.next_desc[blockIdx.x] = make_uint2(r0, s_count);
    if (g.hist_next)
        for (uint32_t j = threadIdx.x; j < g.S; j += kHopThreads)
            if (s_hist[j]) atomicAdd(&g.hist_next[j], s_hist[j]);
}

// First match of one probe by one thread, reading the switch's blob from
// global memory (L2-resident tables): the per-lane walk of first_match_lane
// without its warp phases.  The candidate list is read four items at a time
// and the four candidates' rules are loaded together before any is tested,
// so a probe's chain of dependent L2 round trips per hop shrinks about as
// many times (a tail walk is as long as its slowest probe's chain).
constexpr uint32_t kTailBatch = 4;

template <bool kStats>
__device__ __forceinline__ uint32_t first_match_thread(const uint8_t *__restrict__ blob, const BlobLayout &L,
                                                       uint32_t src, uint32_t dst, uint32_t dport,
                                                       uint32_t in_port, uint32_t &tests, uint32_t &lookups) {
    const uint4 *A = reinterpret_cast<const uint4 *>(blob + L.a);
    const uint2 *Bv = reinterpret_cast<const uint2 *>(blob + L.b);
    const uint32_t *boff = reinterpret_cast<const uint32_t *>(blob + L.boff);
    const uint16_t *items = reinterpret_cast<const uint16_t *>(blob + L.items);
    const uint2 *segs = reinterpret_cast<const uint2 *>(blob + L.segs);
    const uint32_t *bnd = reinterpret_cast<const uint32_t *>(blob + L.bnd);
    const uint32_t *win = reinterpret_cast<const uint32_t *>(blob + L.win);
    const uint32_t k = dport >> kBucketShift;
    const uint32_t i1 = __ldg(boff + k + 1);
    for (uint32_t i = __ldg(boff + k); i < i1; i += kTailBatch) {
        uint32_t it[kTailBatch];
        uint4 a[kTailBatch];
        uint2 bb[kTailBatch];
#pragma unroll
        for (uint32_t j = 0; j < kTailBatch; ++j) it[j] = i + j < i1 ? __ldg(items + i + j) : 0xFFFFu;
#pragma unroll
        for (uint32_t j = 0; j < kTailBatch; ++j) {
            const bool rule = it[j] != 0xFFFFu && !(it[j] & kSegItem);
            a[j] = rule ? __ldg(A + it[j]) : make_uint4(0, 0, 0, 0);
            bb[j] = rule ? __ldg(Bv + it[j]) : make_uint2(1u, 0u);   // lo 1 > hi 0: never matches
        }
#pragma unroll
        for (uint32_t j = 0; j < kTailBatch; ++j) {
            if (it[j] == 0xFFFFu) return 0u;   // past the list's end: table miss
            if (it[j] & kSegItem) {
                const uint2 sd = __ldg(segs + (it[j] & 0x7FFFu));
                uint32_t lo = 0, len = sd.y;   // bnd[sd.x] = 0 <= dst
                while (len > 1) {
                    const uint32_t half = len >> 1;
                    lo = __ldg(bnd + sd.x + lo + half) <= dst ? lo + half : lo;
                    len -= half;
                }
                const uint32_t w = __ldg(win + sd.x + lo);
                if (kStats) ++lookups;
                if (w & kWinFound) return w;
                continue;
            }
            if (kStats) ++tests;
            const uint32_t diff = ((src ^ a[j].x) & a[j].y) | ((dst ^ a[j].z) & a[j].w) |
                                  ((in_port ^ bb[j].y) & ((bb[j].y >> 8) & 0xFFu));
            if (diff == 0 && dport >= (bb[j].x & 0xFFFFu) && dport <= (bb[j].x >> 16))
                return kWinFound | (bb[j].y >> 16);
        }
    }
    return 0u;
}

// The walk's last hops, first_hop .. cap - 1, in one launch: one thread per
// probe still walking (the unsorted list the last hop kernel wrote, read
// through its per-block slices), each thread taking its probe hop after hop
// to the end with the tables read from L2.  Few probes are left by then, so
// regrouping them by switch every hop would cost more in launches than the
// table staging saves.  Results, cycle finishing, path constraints and the
// per-hop live counts are those of walk_hop_kernel.
template <bool kPolicy, bool kStats, bool kRec>
__global__ void __launch_bounds__(256) walk_tail_kernel(HopArgs g, const uint2 *__restrict__ list,
                                                        const uint2 *__restrict__ desc, uint32_t nslices,
                                                        uint32_t first_hop) {
    const uint32_t lane = threadIdx.x & 31;
    uint32_t stc[kStCount] = {};
    for (uint32_t sl = blockIdx.x; sl < nslices; sl += gridDim.x) {
        const uint2 d = desc[sl];
        for (uint32_t base = d.x; base < d.x + d.y; base += blockDim.x) {
            const uint32_t i = base + threadIdx.x;
            bool active = i < d.x + d.y;
            uint2 e = make_uint2(0, 0);
            uint4 pr = make_uint4(0, 0, 0, 0);
            uint32_t pid = 0;
            if (active) {
                e = list[i];
                pr = load_header<kRec>(g, e.x, &pid);
            }
            uint32_t loc = e.y;
            for (uint32_t h = first_hop; h < g.cap; ++h) {
                const uint32_t live = __ballot_sync(PV_FULL_MASK, active);
                if (!live) break;
                if (lane == 0) atomicAdd(&g.hop_live[h], (uint32_t)__popc(live));
                if (!active) continue;
                const uint32_t s = (loc >> 8) & 0xFFFFu, in_port = loc & 0xFFu, fin = loc_finish(loc);
                uint32_t *out = reinterpret_cast<uint32_t *>(g.out) + pid;   // {status, hops, last_switch}
                if (fin != 0 && fin - 1 == h) {   // finished at its cycle position
                    *out = (uint32_t)PV_LOOP | g.cap << 8 | s << 16;
                    active = false;
                    continue;
                }
                const uint8_t *blob = g.blob + g.blob_offs[s];
                const uint4 hdr = __ldg(reinterpret_cast<const uint4 *>(blob));
                const BlobLayout L(hdr);
                const uint32_t fm = first_match_thread<kStats>(blob, L, pr.x, pr.y, pr.z & 0xFFFFu, in_port,
                                                               stc[kStRuleTests], stc[kStLookups]);
                if (kStats) {
                    uint32_t depth = 0;
                    const uint32_t ref = scan_first_match(reinterpret_cast<const uint4 *>(blob + L.fa),
                                                          reinterpret_cast<const uint2 *>(blob + L.fb),
                                                          hdr.x & 0xFFFFu, pr.x, pr.y, pr.z & 0xFFFFu, in_port, &depth);
                    ++stc[kStFirstMatches];
                    stc[kStLinearDepth] += depth;
                    stc[kStMismatch] += ref != fm ? 1u : 0u;
                }
                const uint32_t pbase = g.port_offs[s], nports = g.port_offs[s + 1] - pbase;
                uint32_t status, next;
                hop_outcome(g, h, fm, pr.y, pr.w, pbase, nports, &status, &next);
                if (kPolicy) {
                    const uint4 ph = policy_of(g.pa, pid);
                    uint32_t bits = 0;
                    for (uint32_t k = 0; k < ph.w; ++k)
                        if (g.pa.sw[ph.z + k] == s) bits |= 1u << k;
                    if (bits) g.pa.hits[pid] |= bits;
                    if (status == kAlive && switch_listed(g.pa.sw + ph.x, ph.y, next >> 8)) status = kViolationNext;
                }
                if (status != kAlive) {
                    const bool at_next = status == kViolationNext;
                    *out = (at_next ? (uint32_t)PV_VIOLATION : status) | (h + (at_next ? 2u : 1u)) << 8 |
                           (at_next ? (next >> 8) : s) << 16;
                    active = false;
                    continue;
                }
                const bool bounce = g.bounce && (fm & 0xFFFFu) == in_port;
                if (bounce && (loc >> 24) == kBounced) {   // two bounces in a row: a two-switch cycle
                    *out = (uint32_t)PV_LOOP | g.cap << 8 | (((g.cap - 1u - h) & 1u) ? (next >> 8) : s) << 16;
                    active = false;
                    continue;
                }
                uint32_t nfin = fin;
                const uint32_t h1 = h + 1;
                if (g.cycles && nfin == 0 && h1 >= kCycleCheckFrom) {
                    if ((h1 & (h1 - 1u)) == 0) {
                        g.ck[e.x] = next;
                    } else if (g.ck[e.x] == next) {
                        const uint32_t period = h1 - (1u << (31 - __clz(h1)));
                        nfin = h1 + (g.cap - 1u - h1) % period + 1u;
                        if (nfin >= g.cap) nfin = 0;
                    }
                }
                if (nfin == 0 && bounce) nfin = kBounced;
                loc = next | (nfin << 24);
            }
        }
    }
    if (kStats) flush_stats(g.stats, stc);
}

inline size_t align256(size_t x) { return (x + 255) & ~(size_t)255; }

// stage[p] = port p's {peer, aux} as walk_hop_kernel stages it: aux = the
// peer switch's region, or the attached host's address (0 for a host index
// out of range, which the outcome rejects by its index).
__global__ void port_stage_kernel(uint32_t P, const int32_t *__restrict__ peer, const uint8_t *__restrict__ region,
                                  uint32_t H, const uint32_t *__restrict__ host_ip, uint2 *__restrict__ stage) {
    const uint32_t p = blockIdx.x * blockDim.x + threadIdx.x;
    if (p >= P) return;
    const int32_t x = peer[p];
    uint32_t aux = 0;
    if (x >= 0) {
        if (x & PV_PEER_HOST) {
            const uint32_t q = (uint32_t)(x & ~PV_PEER_HOST);
            aux = q < H ? host_ip[q] : 0u;
        } else {
            aux = region[(uint32_t)x >> 8];
        }
    }
    stage[p] = make_uint2((uint32_t)x, aux);
}

// addr[h] = {host_ip[h], host_port[h]}.
__global__ void host_addr_kernel(uint32_t H, const uint32_t *__restrict__ ip, const uint16_t *__restrict__ port,
                                 uint2 *__restrict__ addr) {
    const uint32_t h = blockIdx.x * blockDim.x + threadIdx.x;
    if (h < H) addr[h] = make_uint2(ip[h], port[h]);
}

}  // namespace

// A flow-table load between its two halves: the first has validated the
// structure on the host and queued the uploads and the index-size pass; the
// second reads the sizes back, builds the blobs and installs the tables.
struct pv_table_load {
    uint32_t S = 0, H = 0, P = 0, max_pad = 0, max_rules = 0, max_ports = 0;
    const uint32_t *rule_offs = nullptr, *port_offs = nullptr, *host_ip = nullptr;
    const pv_rule *rules = nullptr;
    const uint8_t *switch_region = nullptr;
    const int32_t *port_peer = nullptr;
    const uint16_t *host_switch = nullptr, *host_port = nullptr;
    std::vector<uint32_t> tab;   // first compiled rule of each switch (tables padded to 32 rules)
    pv_table_state t;            // the new tables (the loaded ones stay in use until these are complete)
    uint32_t *d_rule_offs = nullptr, *d_tab_offs = nullptr, *d_sizes = nullptr;
    uint4 *d_rule_a = nullptr;
    uint2 *d_rule_b = nullptr;
    void free_temps(pv_ctx *ctx) {
        pv_pool_free(ctx, d_rule_offs);
        pv_pool_free(ctx, d_tab_offs);
        pv_pool_free(ctx, d_rule_a);
        pv_pool_free(ctx, d_rule_b);
        pv_pool_free(ctx, d_sizes);
        d_rule_offs = d_tab_offs = d_sizes = nullptr;
        d_rule_a = nullptr;
        d_rule_b = nullptr;
    }
};

void pv_discard_table_load(pv_ctx *ctx) {
    if (!ctx->table_load) return;
    ctx->table_load->free_temps(ctx);
    pv_free_tables(ctx, ctx->table_load->t);
    delete ctx->table_load;
    ctx->table_load = nullptr;
}

namespace {

// First half: host validation of the structure, every upload, rule
// compilation and the index-size pass, all queued on the load stream; the
// host does not wait for the device.
int tables_begin(pv_ctx *ctx, pv_table_load &L, uint32_t S, const uint32_t *rule_offs, const pv_rule *rules,
                 const uint8_t *switch_region, const uint32_t *port_offs, const int32_t *port_peer,
                 uint32_t H, const uint16_t *host_switch, const uint16_t *host_port, const uint32_t *host_ip) {
    if (!ctx) return PV_EINVAL;
    if (S == 0 || S > PV_MAX_SWITCHES) return pv_fail(ctx, PV_EINVAL, "num_switches must be 1..%d", PV_MAX_SWITCHES);
    if (H > PV_MAX_HOSTS) return pv_fail(ctx, PV_EINVAL, "num_hosts must be <= %d", PV_MAX_HOSTS);
    if (!rule_offs || !switch_region || !port_offs || (H && (!host_switch || !host_port || !host_ip)))
        return pv_fail(ctx, PV_EINVAL, "pv_load_flow_tables: NULL host pointer");
    if (rule_offs[0] != 0 || port_offs[0] != 0) return pv_fail(ctx, PV_EINVAL, "offsets must start at 0");
    std::vector<uint32_t> &tab = L.tab;
    tab.assign(S + 1, 0);
    uint32_t &max_pad = L.max_pad;
    max_pad = 0;
    L.max_ports = 0;
    for (uint32_t s = 0; s < S; ++s) {
        if (rule_offs[s + 1] < rule_offs[s] || port_offs[s + 1] < port_offs[s])
            return pv_fail(ctx, PV_EINVAL, "offsets not monotone at switch %u", s);
        const uint32_t nr = rule_offs[s + 1] - rule_offs[s], np = port_offs[s + 1] - port_offs[s];
        if (nr > PV_MAX_RULES) return pv_fail(ctx, PV_EINVAL, "switch %u has %u rules (max %d)", s, nr, PV_MAX_RULES);
        if (np > PV_MAX_PORTS) return pv_fail(ctx, PV_EINVAL, "switch %u has %u ports (max %d)", s, np, PV_MAX_PORTS);
        if (switch_region[s] >= 32) return pv_fail(ctx, PV_EINVAL, "switch %u region %u >= 32", s, switch_region[s]);
        const uint32_t pad = (nr + 31) / 32 * 32;
        tab[s + 1] = tab[s] + pad;
        max_pad = std::max(max_pad, pad);
        L.max_ports = std::max(L.max_ports, np);
    }
    const uint32_t R = rule_offs[S], P = port_offs[S];
    if (R && !rules) return pv_fail(ctx, PV_EINVAL, "NULL rules");
    if (P && !port_peer) return pv_fail(ctx, PV_EINVAL, "NULL port_peer");
    // per-rule fields are checked on the device by compile_tables_kernel
    for (uint32_t s = 0; s < S; ++s) {
        for (uint32_t p = port_offs[s]; p < port_offs[s + 1]; ++p) {
            const int32_t peer = port_peer[p];
            if (peer == PV_PEER_NONE) continue;
            if (peer < 0) return pv_fail(ctx, PV_EINVAL, "port %u: bad peer %d", p, peer);
            if (peer & PV_PEER_HOST) {
                if ((uint32_t)(peer & ~PV_PEER_HOST) >= H) return pv_fail(ctx, PV_EINVAL, "port %u: host out of range", p);
            } else {
                const uint32_t s2 = (uint32_t)peer >> 8, p2 = (uint32_t)peer & 0xFFu;
                if (s2 >= S || p2 >= port_offs[s2 + 1] - port_offs[s2])
                    return pv_fail(ctx, PV_EINVAL, "port %u: peer switch port out of range", p);
            }
        }
    }
    for (uint32_t h = 0; h < H; ++h)
        if (host_switch[h] >= S || host_port[h] >= port_offs[host_switch[h] + 1] - port_offs[host_switch[h]])
            return pv_fail(ctx, PV_EINVAL, "host %u attachment out of range", h);

    if (int rc0 = pv_load_begin(ctx)) return rc0;
    cudaStream_t ls = ctx->load_stream;
    pv_table_state &t = L.t;
    const uint32_t T = tab[S];
    uint32_t *&d_rule_offs = L.d_rule_offs, *&d_tab_offs = L.d_tab_offs, *&d_sizes = L.d_sizes;
    uint4 *&d_rule_a = L.d_rule_a;
    uint2 *&d_rule_b = L.d_rule_b;
    auto free_temps = [&]() { L.free_temps(ctx); };
    int rc;
    if ((rc = pv_pool_alloc(ctx, (void **)&d_tab_offs, (S + 1) * 4, "table offsets")) ||
        (rc = pv_pool_alloc(ctx, (void **)&d_rule_a, (size_t)T * 16, "rules A")) ||
        (rc = pv_pool_alloc(ctx, (void **)&d_rule_b, (size_t)T * 8, "rules B")) ||
        (rc = pv_pool_alloc(ctx, (void **)&d_sizes, (size_t)S * 16 + 4, "index sizes")) ||
        (rc = pv_pool_alloc(ctx, (void **)&t.d_blob_offs, ((size_t)S + 1) * 8, "blob offsets")) ||
        (rc = pv_pool_alloc(ctx, (void **)&t.d_region, S, "regions")) ||
        (rc = pv_pool_alloc(ctx, (void **)&t.d_port_offs, (S + 1) * 4, "port offsets")) ||
        (rc = pv_pool_alloc(ctx, (void **)&t.d_port_peer, (size_t)P * 4, "port peers")) ||
        (rc = pv_pool_alloc(ctx, (void **)&t.d_host_switch, (size_t)H * 2, "host switch")) ||
        (rc = pv_pool_alloc(ctx, (void **)&t.d_host_port, (size_t)H * 2, "host port")) ||
        (rc = pv_pool_alloc(ctx, (void **)&t.d_host_ip, (size_t)H * 4, "host ip")) ||
        (rc = pv_pool_alloc(ctx, (void **)&t.d_host_addr, (size_t)H * 8, "host addresses")) ||
        (rc = pv_pool_alloc(ctx, (void **)&t.d_port_stage, std::max<size_t>((size_t)P, 1) * 8, "port stage")) ||
        (rc = pv_pool_alloc(ctx, (void **)&d_rule_offs, (S + 1) * 4, "rule offsets")) ||
        (rc = pv_pool_alloc(ctx, (void **)&t.d_raw, (size_t)R * sizeof(pv_rule), "raw rules"))) {
        free_temps();
        pv_free_tables(ctx, t);
        return rc;
    }
    cudaError_t e = cudaSuccess;
    e = e ? e : cudaMemcpyAsync(d_tab_offs, tab.data(), (S + 1) * 4, cudaMemcpyHostToDevice, ls);
    e = e ? e : cudaMemcpyAsync(t.d_region, switch_region, S, cudaMemcpyHostToDevice, ls);
    e = e ? e : cudaMemcpyAsync(t.d_port_offs, port_offs, (S + 1) * 4, cudaMemcpyHostToDevice, ls);
    if (P) e = e ? e : cudaMemcpyAsync(t.d_port_peer, port_peer, (size_t)P * 4, cudaMemcpyHostToDevice, ls);
    if (H) {
        e = e ? e : cudaMemcpyAsync(t.d_host_switch, host_switch, (size_t)H * 2, cudaMemcpyHostToDevice, ls);
        e = e ? e : cudaMemcpyAsync(t.d_host_port, host_port, (size_t)H * 2, cudaMemcpyHostToDevice, ls);
        e = e ? e : cudaMemcpyAsync(t.d_host_ip, host_ip, (size_t)H * 4, cudaMemcpyHostToDevice, ls);
        if (e == cudaSuccess)
            host_addr_kernel<<<(H + 255) / 256, 256, 0, ls>>>(H, t.d_host_ip, t.d_host_port, t.d_host_addr);
        e = e ? e : cudaGetLastError();
    }
    if (P && e == cudaSuccess) {
        port_stage_kernel<<<(P + 255) / 256, 256, 0, ls>>>(P, t.d_port_peer, t.d_region, H, t.d_host_ip,
                                                            t.d_port_stage);
        e = cudaGetLastError();
    }
    e = e ? e : cudaMemcpyAsync(d_rule_offs, rule_offs, (S + 1) * 4, cudaMemcpyHostToDevice, ls);
    if (R) e = e ? e : cudaMemcpyAsync(t.d_raw, rules, (size_t)R * sizeof(pv_rule), cudaMemcpyHostToDevice, ls);
    if (e != cudaSuccess) {
        free_temps();
        pv_free_tables(ctx, t);
        return pv_cuda_fail(ctx, e, "pv_load_flow_tables uploads");
    }
    // links into each switch, sorted by (source switch, source port); uploaded
    // here, ahead of the index-size read-back, so no pageable copy (which
    // waits for the stream) follows the index fill
    {
        std::vector<uint32_t> in_offs(S + 1, 0), links;
        for (uint32_t u = 0; u < S; ++u)
            for (uint32_t p = port_offs[u]; p < port_offs[u + 1]; ++p) {
                const int32_t peer = port_peer[p];
                if (peer >= 0 && !(peer & PV_PEER_HOST)) ++in_offs[((uint32_t)peer >> 8) + 1];
            }
        for (uint32_t v = 0; v < S; ++v) in_offs[v + 1] += in_offs[v];
        links.resize(std::max<uint32_t>(in_offs[S], 1));
        std::vector<uint32_t> cur(in_offs.begin(), in_offs.end() - 1);
        for (uint32_t u = 0; u < S; ++u)   // ascending u, then p: each list ends up sorted
            for (uint32_t p = port_offs[u]; p < port_offs[u + 1]; ++p) {
                const int32_t peer = port_peer[p];
                if (peer < 0 || (peer & PV_PEER_HOST)) continue;
                const uint32_t v = (uint32_t)peer >> 8;
                links[cur[v]++] = u << 16 | (p - port_offs[u]) << 8 | ((uint32_t)peer & 0xFFu);
            }
        int rc2;
        if ((rc2 = pv_pool_alloc(ctx, (void **)&t.d_in_offs, (S + 1) * 4, "in-link offsets")) ||
            (rc2 = pv_pool_alloc(ctx, (void **)&t.d_in_links, links.size() * 4, "in-links"))) {
            t.num_links = 0;
            free_temps();
            pv_free_tables(ctx, t);
            return rc2;
        }
        cudaError_t e2 = cudaMemcpyAsync(t.d_in_offs, in_offs.data(), (S + 1) * 4, cudaMemcpyHostToDevice, ls);
        if (e2 == cudaSuccess)
            e2 = cudaMemcpyAsync(t.d_in_links, links.data(), links.size() * 4, cudaMemcpyHostToDevice, ls);
        t.num_links = in_offs[S];
        // symmetric cabling (port p of u leads to port q of v exactly when q
        // of v leads back to p of u) lets a walk recognise a two-switch
        // forwarding cycle from two bounces in a row (walk_hop_kernel)
        bool sym = true;
        for (uint32_t u = 0; u < S && sym; ++u)
            for (uint32_t p = port_offs[u]; p < port_offs[u + 1] && sym; ++p) {
                const int32_t peer = port_peer[p];
                if (peer < 0 || (peer & PV_PEER_HOST)) continue;
                const uint32_t v = (uint32_t)peer >> 8, q = (uint32_t)peer & 0xFFu;
                sym = port_peer[port_offs[v] + q] == (int32_t)(u << 8 | (p - port_offs[u]));
            }
        t.links_symmetric = sym;

        if (e2 != cudaSuccess) {
            free_temps();
            pv_free_tables(ctx, t);
            return pv_cuda_fail(ctx, e2, "in-links upload");
        }
    }
    uint32_t maxn = 0;
    for (uint32_t s = 0; s < S; ++s) maxn = std::max(maxn, rule_offs[s + 1] - rule_offs[s]);
    L.max_rules = maxn;
    const IndexSmem ism(maxn);
    if (e == cudaSuccess) {
        uint32_t npow = 1;
        while (npow < maxn) npow <<= 1;
        uint32_t *d_bad = d_sizes + (size_t)S * 4;   // lowest invalid rule index
        e = cudaMemsetAsync(d_bad, 0xFF, 4, ls);
        if (e == cudaSuccess) {
            compile_tables_kernel<<<S, 1024, npow * 4, ls>>>(d_rule_offs, t.d_raw, t.d_port_offs, d_tab_offs,
                                                             d_rule_a, d_rule_b, d_bad);
            e = cudaGetLastError();
        }
        if (e == cudaSuccess &&
            (pv_smem_limit(ctx, (const void *)index_build_kernel<false>, "index_build_kernel smem") ||
             pv_smem_limit(ctx, (const void *)index_build_kernel<true>, "index_build_kernel smem"))) {
            free_temps();
            pv_free_tables(ctx, t);
            return PV_ECUDA;
        }
        if (e == cudaSuccess) {
            index_build_kernel<false><<<S, kIndexThreads, ism.bytes, ls>>>(d_rule_offs, d_tab_offs, d_rule_a,
                                                                           d_rule_b, d_sizes, nullptr, nullptr, ism);
            e = cudaGetLastError();
        }
    }
    if (e != cudaSuccess) {
        free_temps();
        pv_free_tables(ctx, t);
        return pv_cuda_fail(ctx, e, "pv_load_flow_tables");
    }
    L.S = S;
    L.H = H;
    L.P = P;
    L.rule_offs = rule_offs;
    L.rules = rules;
    L.switch_region = switch_region;
    L.port_offs = port_offs;
    L.port_peer = port_peer;
    L.host_switch = host_switch;
    L.host_port = host_port;
    L.host_ip = host_ip;
    return PV_OK;
}

// Second half: waits for the index sizes (and the device-side rule
// validation), lays out and fills the blobs, installs the tables.
int tables_end(pv_ctx *ctx, pv_table_load &L) {
    const uint32_t S = L.S, H = L.H, P = L.P, max_pad = L.max_pad;
    const uint32_t *rule_offs = L.rule_offs, *port_offs = L.port_offs, *host_ip = L.host_ip;
    const pv_rule *rules = L.rules;
    const uint8_t *switch_region = L.switch_region;
    const int32_t *port_peer = L.port_peer;
    const uint16_t *host_switch = L.host_switch, *host_port = L.host_port;
    const std::vector<uint32_t> &tab = L.tab;
    const IndexSmem ism(L.max_rules);
    pv_table_state &t = L.t;
    uint32_t *d_rule_offs = L.d_rule_offs, *d_tab_offs = L.d_tab_offs, *d_sizes = L.d_sizes;
    uint4 *d_rule_a = L.d_rule_a;
    uint2 *d_rule_b = L.d_rule_b;
    auto free_temps = [&]() { L.free_temps(ctx); };
    if (int rc0 = pv_load_begin(ctx)) {
        free_temps();
        pv_free_tables(ctx, t);
        return rc0;
    }
    cudaStream_t ls = ctx->load_stream;
    cudaError_t e = cudaSuccess;
    int rc = PV_OK;
    // blob layout from the index sizes (and the device-side rule validation)
    std::vector<uint32_t> sizes((size_t)S * 4 + 1);
    std::vector<uint64_t> boffs(S + 1, 0);
    if (e == cudaSuccess) e = cudaMemcpyAsync(sizes.data(), d_sizes, (size_t)S * 16 + 4, cudaMemcpyDeviceToHost, ls);
    if (e == cudaSuccess) e = cudaStreamSynchronize(ls);
    if (e == cudaSuccess && sizes[(size_t)S * 4] != 0xFFFFFFFFu) {
        const uint32_t i = sizes[(size_t)S * 4];
        const uint32_t s = (uint32_t)(std::upper_bound(rule_offs, rule_offs + S + 1, i) - rule_offs) - 1;
        const pv_rule &r = rules[i];
        free_temps();
        pv_free_tables(ctx, t);
        return pv_fail(ctx, PV_EINVAL,
                       "rule %u (switch %u, %u ports): in_port %u, action %u, prefix lengths %u/%u, dport %u..%u "
                       "out of range",
                       i, s, port_offs[s + 1] - port_offs[s], r.in_port, r.action, r.src_len, r.dst_len,
                       r.dport_lo, r.dport_hi);
    }
    uint32_t max_blob = 0, max_linear = 0;
    uint64_t all_items = 0;
    if (e == cudaSuccess) {
        for (uint32_t s = 0; s < S; ++s) {
            const uint32_t npad = tab[s + 1] - tab[s];
            all_items += sizes[4 * s];
            const BlobLayout L(npad, sizes[4 * s + 3], sizes[4 * s], sizes[4 * s + 1], sizes[4 * s + 2]);
            boffs[s + 1] = boffs[s] + L.total;
            max_blob = std::max(max_blob, L.fa);             // staged by the indexed kernel
            max_linear = std::max(max_linear, linear_bytes(npad));
        }
        e = cudaMemcpyAsync(t.d_blob_offs, boffs.data(), ((size_t)S + 1) * 8, cudaMemcpyHostToDevice, ls);
    }
    if (e == cudaSuccess) {
        rc = pv_pool_alloc(ctx, (void **)&t.d_blob, boffs[S], "flow table blobs");
        if (rc) {
            free_temps();
            pv_free_tables(ctx, t);
            return rc;
        }
        index_build_kernel<true><<<S, kIndexThreads, ism.bytes, ls>>>(d_rule_offs, d_tab_offs, d_rule_a, d_rule_b,
                                                                      d_sizes, t.d_blob_offs, t.d_blob, ism);
        e = cudaGetLastError();
    }
    free_temps();
    if (e != cudaSuccess) {
        pv_free_tables(ctx, t);
        return pv_cuda_fail(ctx, e, "pv_load_flow_tables");
    }
    t.num_switches = S;
    t.num_hosts = H;
    // The tail launch walks each probe's candidate lists from L2, one thread
    // per probe: with short lists (at most kTailEarlyItems items per bucket
    // on average) it pays from hop 5 on, with long ones only from hop 8.
    t.tail_hop = all_items <= (uint64_t)kTailEarlyItems * kBuckets * S ? 5u : 8u;
    t.max_rules_padded = max_pad;
    t.max_ports = L.max_ports;
    t.max_blob_bytes = max_blob;
    t.max_linear_bytes = max_linear;
    // the hop kernel stages the port table after the table (16-byte aligned)
    const size_t smem_cap = ctx->max_smem_optin - 1024 - 16 - port_stage_bytes(t.max_ports);
    t.index_fits = max_blob <= smem_cap;
    if (max_linear > smem_cap) {
        pv_free_tables(ctx, t);
        return pv_fail(ctx, PV_EINVAL, "largest flow table needs %u bytes of shared memory", max_linear);
    }
    {
        const int rc3 = pv_smem_limit(ctx, (const void *)walk_scatter_kernel, "walk_scatter_kernel smem");
        if (rc3) {
            pv_free_tables(ctx, t);
            return rc3;
        }
    }
    // host copy for rule installation
    pv_table_host &h = ctx->tbh;
    h.rule_offs.assign(rule_offs, rule_offs + S + 1);
    h.region.assign(switch_region, switch_region + S);
    h.port_offs.assign(port_offs, port_offs + S + 1);
    h.port_peer.assign(port_peer, port_peer + P);
    h.host_switch.assign(host_switch, host_switch + H);
    h.host_port.assign(host_port, host_port + H);
    h.host_ip.assign(host_ip, host_ip + H);
    t.loaded = true;
    pv_retire_begin(ctx);
    pv_free_tables(ctx, ctx->tb);
    pv_retire_end(ctx);
    ctx->tb = t;
    return pv_load_end(ctx);
}

}  // namespace

// -----------------------------------------------------------------------------
// C ABI
// -----------------------------------------------------------------------------
extern "C" int pv_load_flow_tables(pv_ctx *ctx, uint32_t S, const uint32_t *rule_offs, const pv_rule *rules,
                                   const uint8_t *switch_region, const uint32_t *port_offs,
                                   const int32_t *port_peer, uint32_t H, const uint16_t *host_switch,
                                   const uint16_t *host_port, const uint32_t *host_ip) {
    if (!ctx) return PV_EINVAL;
    if (ctx->table_load) return pv_fail(ctx, PV_ESTATE, "pv_load_flow_tables: a two-part table load is in progress");
    pv_table_load L;
    if (int rc = tables_begin(ctx, L, S, rule_offs, rules, switch_region, port_offs, port_peer, H, host_switch,
                              host_port, host_ip))
        return rc;
    return tables_end(ctx, L);
}

extern "C" int pv_load_flow_tables_begin(pv_ctx *ctx, uint32_t S, const uint32_t *rule_offs, const pv_rule *rules,
                                         const uint8_t *switch_region, const uint32_t *port_offs,
                                         const int32_t *port_peer, uint32_t H, const uint16_t *host_switch,
                                         const uint16_t *host_port, const uint32_t *host_ip) {
    if (!ctx) return PV_EINVAL;
    if (ctx->table_load) return pv_fail(ctx, PV_ESTATE, "pv_load_flow_tables_begin: a table load is in progress");
    pv_table_load *L = new pv_table_load;
    if (int rc = tables_begin(ctx, *L, S, rule_offs, rules, switch_region, port_offs, port_peer, H, host_switch,
                              host_port, host_ip)) {
        delete L;
        return rc;
    }
    ctx->table_load = L;
    return PV_OK;
}

extern "C" int pv_load_flow_tables_end(pv_ctx *ctx) {
    if (!ctx) return PV_EINVAL;
    pv_table_load *L = ctx->table_load;
    if (!L) return pv_fail(ctx, PV_ESTATE, "pv_load_flow_tables_end: no table load in progress");
    ctx->table_load = nullptr;
    const int rc = tables_end(ctx, *L);
    delete L;
    return rc;
}

namespace {

// The walk of pv_verify_probes; with pa, under the path constraints of
// pv_verify_probes_constrained.
using HopKernel = void (*)(HopArgs);
using TailKernel = void (*)(HopArgs, const uint2 *, const uint2 *, uint32_t, uint32_t);

// first: the kernel for the walk's first hop (the statistics kernels serve
// every hop with the general form)
template <bool kRec, bool kFirst>
HopKernel pick_hop_form(bool indexed, bool pol) {
    if (indexed)
        return pol ? walk_hop_kernel<true, true, false, kRec, kFirst> : walk_hop_kernel<true, false, false, kRec, kFirst>;
    return pol ? walk_hop_kernel<false, true, false, kRec, kFirst> : walk_hop_kernel<false, false, false, kRec, kFirst>;
}

template <bool kRec>
HopKernel pick_hop(bool indexed, bool pol, bool stats, bool first) {
    if (stats) {
        if (indexed)
            return pol ? walk_hop_kernel<true, true, true, kRec, false> : walk_hop_kernel<true, false, true, kRec, false>;
        return pol ? walk_hop_kernel<false, true, true, kRec, false> : walk_hop_kernel<false, false, true, kRec, false>;
    }
    return first ? pick_hop_form<kRec, true>(indexed, pol) : pick_hop_form<kRec, false>(indexed, pol);
}

template <bool kRec>
TailKernel pick_tail(bool pol, bool stats) {
    return pol ? (stats ? walk_tail_kernel<true, true, kRec> : walk_tail_kernel<true, false, kRec>)
               : (stats ? walk_tail_kernel<false, true, kRec> : walk_tail_kernel<false, false, kRec>);
}

int walk_probes(pv_ctx *ctx, uint32_t M, const pv_probe *d_probes, uint32_t hop_cap, pv_result *d_out,
                const PolicyArgs *pa, pv_stream stream, const BindArgs *ba = nullptr) {
    const pv_table_state &t = ctx->tb;
    const bool pol = pa != nullptr;
    if (!t.loaded) return pv_fail(ctx, PV_ESTATE, "pv_verify_probes: no flow tables loaded");
    if (hop_cap == 0 || hop_cap > PV_MAX_HOP_CAP) return pv_fail(ctx, PV_EINVAL, "hop_cap must be 1..255");
    if (M == 0) return PV_OK;
    if ((!d_probes && !ba) || !d_out) return pv_fail(ctx, PV_EINVAL, "pv_verify_probes: NULL device pointer");
    if (((uintptr_t)d_probes & 15) != 0) return pv_fail(ctx, PV_EINVAL, "pv_verify_probes: d_probes must be 16-byte aligned");
    if (((uintptr_t)d_out & 3) != 0) return pv_fail(ctx, PV_EINVAL, "pv_verify_probes: d_out must be 4-byte aligned");
    const uint32_t S = t.num_switches;
    int which = ctx->opt_walk;
    if (which == 0) which = t.index_fits ? 2 : 1;
    if (which == 2 && !t.index_fits)
        return pv_fail(ctx, PV_EINVAL, "pv_verify_probes: the first-match index does not fit shared memory");
    const bool indexed = which == 2;
    const size_t table_smem = indexed ? t.max_blob_bytes : t.max_linear_bytes;
    // the next hop's per-switch counts ride in the hop kernel's shared memory
    // after the staged table, when they fit
    // (and the current switch's port table after both)
    const size_t hist_off = (table_smem + 15) & ~(size_t)15;
    const size_t port_bytes = port_stage_bytes(t.max_ports);
    const bool fuse_hist =
        S <= kSmemHistMax && hist_off + (size_t)S * 4 + 16 + port_bytes <= ctx->max_smem_optin - 1024;
    const size_t port_off = fuse_hist ? ((hist_off + (size_t)S * 4 + 15) & ~(size_t)15) : hist_off;
    const size_t hop_smem = port_off + port_bytes;
    int hop_blocks_per_sm = 0;
    const bool stats = ctx->opt_walk_stats != 0;
    // compact flows with one path constraint per group are placed directly
    // (and walked through walk records)
    const bool direct = ba && (!pol || (pa->probe_pol == nullptr && (pa->per == 0 || pa->per % ba->ppg == 0)));
    const HopKernel hop_fn = direct ? pick_hop<true>(indexed, pol, stats, false) : pick_hop<false>(indexed, pol, stats, false);
    const HopKernel hop_fn0 = direct ? pick_hop<true>(indexed, pol, stats, true) : pick_hop<false>(indexed, pol, stats, true);
    const TailKernel tail_fn = direct ? pick_tail<true>(pol, stats) : pick_tail<false>(pol, stats);
    if (int rc = pv_smem_limit(ctx, (const void *)hop_fn, "walk_hop_kernel smem")) return rc;
    if (int rc = pv_smem_limit(ctx, (const void *)hop_fn0, "walk_hop_kernel smem")) return rc;
    hop_blocks_per_sm = pv_blocks_per_sm(ctx, (const void *)hop_fn, kHopThreads, hop_smem);
    const uint32_t hop_grid = (uint32_t)ctx->num_sms * (uint32_t)std::max(1, hop_blocks_per_sm);
    const uint32_t init_grid = (uint32_t)ctx->num_sms * 8;
    const uint32_t max_desc = std::max(hop_grid, init_grid);
    const size_t o_a = 0, o_b = align256((size_t)M * 8), o_sorted = o_b + align256((size_t)M * 8);
    const size_t o_hist = o_sorted + align256((size_t)M * 8);
    const size_t o_seg = o_hist + align256((size_t)S * 4);
    const size_t o_cur = o_seg + align256((size_t)(S + 2) * 4);
    const size_t o_desc = o_cur + align256((size_t)S * 4);
    const size_t o_ck = o_desc + 2 * align256((size_t)max_desc * 8);
    const bool cycles = ctx->opt_walk_cycles == 0 && hop_cap > kCycleCheckFrom;
    const uint64_t groups = ba ? ((uint64_t)M + ba->ppg - 1) / ba->ppg : 0;
    const uint64_t G64 = groups * (ba ? ba->pods : 0);
    if (direct && G64 > 0xFFFFFFFFull) return pv_fail(ctx, PV_EINVAL, "pv_verify_flows: too many (group, pod) pairs");
    const uint32_t G = (uint32_t)G64;
    const size_t o_pair = o_ck + (cycles ? align256((size_t)M * 4) : 0);
    // walk records (direct placement), or bound records the caller did not ask for
    const bool own_recs = direct || (ba && !d_probes);
    const size_t o_recs = o_pair + (direct ? align256((size_t)G * 4) : 0);
    const size_t total = o_recs + (own_recs ? align256((size_t)M * 16) : 0);
    uint8_t *base = (uint8_t *)pv_scratch(ctx, total);
    if (!base) return PV_ENOMEM;
    uint2 *listA = (uint2 *)(base + o_a), *listB = (uint2 *)(base + o_b), *sorted = (uint2 *)(base + o_sorted);
    uint32_t *hist = (uint32_t *)(base + o_hist), *seg = (uint32_t *)(base + o_seg);
    uint32_t *cursor = (uint32_t *)(base + o_cur);
    uint2 *descA = (uint2 *)(base + o_desc), *descB = (uint2 *)(base + o_desc + align256((size_t)max_desc * 8));
    cudaStream_t st = (cudaStream_t)stream;
    pv_use_begin(ctx, st);
    PV_TRY_CUDA(ctx, cudaMemsetAsync(hist, 0, (size_t)S * 4, st), "hist clear");
    if (stats)
        PV_TRY_CUDA(ctx, cudaMemsetAsync(ctx->d_walk_stats, 0, PV_WALK_STATS * sizeof(unsigned long long), st),
                    "walk statistics clear");
    int pr = pv_prof_start(ctx, st, PV_K_WALK_INIT);
    const PolicyArgs no_policy = {nullptr, nullptr, 0, nullptr, 0, 0, nullptr};
    const size_t init_smem = S <= kSmemHistMax ? (size_t)S * 4 : 0;
    const BindArgs no_bind = {nullptr, nullptr, 0, 0, 1, 1, nullptr, nullptr, nullptr};
    pv_probe *probes_rw = const_cast<pv_probe *>(d_probes);   // written only when binding
    uint4 *recs = (uint4 *)(base + o_recs);
    if (ba && !direct && !d_probes) probes_rw = reinterpret_cast<pv_probe *>(recs);   // the walk's own copy
    const PolicyArgs &pa0 = pol ? *pa : no_policy;
    const BindArgs &ba0 = ba ? *ba : no_bind;
    uint32_t *pair_off = (uint32_t *)(base + o_pair);
    if (direct) {
        const uint32_t gb = (uint32_t)std::min<uint64_t>((G + kGridThreads - 1) / kGridThreads, init_grid);
        if (pol)
            flow_groups_kernel<true><<<gb, kGridThreads, 0, st>>>(M, t.num_hosts, t.d_host_switch, t.d_region, pa0,
                                                                 ba0, G, hist, pair_off);
        else
            flow_groups_kernel<false><<<gb, kGridThreads, 0, st>>>(M, t.num_hosts, t.d_host_switch, t.d_region, pa0,
                                                                  ba0, G, hist, pair_off);
        walk_scan_kernel<<<1, 1024, 0, st>>>(S, hist, seg, cursor);
        const uint32_t groups32 = (uint32_t)groups;
        const size_t gsm = ba->ppg <= 0xFFFFu ? GroupInitSmem(ba->pods, ba->ppg, ba->dst_stride == 2).total : ~(size_t)0;
        const bool by_group = ba->pods <= kGroupInitMaxPods && gsm <= kGroupInitSmem && groups <= 0x7FFFFFFFull;
        const uint64_t wait_ns = ctx->opt_test_stall_staging ? 50ull * 1000 * 1000 : 2ull * 1000 * 1000 * 1000;
        if (by_group) {
            const int rc2 = pol ? pv_smem_limit(ctx, (const void *)walk_init_group_kernel<true>, "walk_init_group_kernel smem")
                                : pv_smem_limit(ctx, (const void *)walk_init_group_kernel<false>, "walk_init_group_kernel smem");
            if (rc2) return rc2;
        }
        if (by_group && pol)
            walk_init_group_kernel<true><<<groups32, kGroupInitThreads, gsm, st>>>(
                M, probes_rw, t.num_hosts, t.d_host_switch, t.d_region, d_out, recs, seg,
                pair_off, pa0, ba0, wait_ns, ctx->d_status);
        else if (by_group)
            walk_init_group_kernel<false><<<groups32, kGroupInitThreads, gsm, st>>>(
                M, probes_rw, t.num_hosts, t.d_host_switch, t.d_region, d_out, recs, seg,
                pair_off, pa0, ba0, wait_ns, ctx->d_status);
        else if (pol)
            walk_init_direct_kernel<true><<<init_grid, kGridThreads, 0, st>>>(
                M, probes_rw, t.num_hosts, t.d_host_switch, t.d_region, d_out, recs, seg,
                pair_off, pa0, ba0);
        else
            walk_init_direct_kernel<false><<<init_grid, kGridThreads, 0, st>>>(
                M, probes_rw, t.num_hosts, t.d_host_switch, t.d_region, d_out, recs, seg,
                pair_off, pa0, ba0);
    } else if (pol && ba)
        walk_init_kernel<true, true><<<init_grid, kGridThreads, init_smem, st>>>(
            M, probes_rw, t.num_hosts, t.d_host_switch, t.d_host_port, t.d_region, d_out, listA, descA, pa0, S, hist,
            ba0);
    else if (pol)
        walk_init_kernel<true, false><<<init_grid, kGridThreads, init_smem, st>>>(
            M, probes_rw, t.num_hosts, t.d_host_switch, t.d_host_port, t.d_region, d_out, listA, descA, pa0, S, hist,
            ba0);
    else if (ba)
        walk_init_kernel<false, true><<<init_grid, kGridThreads, init_smem, st>>>(
            M, probes_rw, t.num_hosts, t.d_host_switch, t.d_host_port, t.d_region, d_out, listA, descA, pa0, S, hist,
            ba0);
    else
        walk_init_kernel<false, false><<<init_grid, kGridThreads, init_smem, st>>>(
            M, probes_rw, t.num_hosts, t.d_host_switch, t.d_host_port, t.d_region, d_out, listA, descA, pa0, S, hist,
            ba0);
    pv_prof_stop(ctx, st, pr, direct ? 3 : 1);
    const size_t hist_smem = S <= kSmemHistMax ? (size_t)S * 4 : 0;
    const size_t scat_smem = S <= kSmemHistMax ? (size_t)S * 8 : 0;
    HopArgs g;
    g.cap = hop_cap;
    g.seg = seg;
    g.S = S;
    g.H = t.num_hosts;
    g.blob = t.d_blob;
    g.blob_offs = t.d_blob_offs;
    g.region = t.d_region;
    g.port_offs = t.d_port_offs;
    g.port_peer = t.d_port_peer;
    g.host_ip = t.d_host_ip;
    g.probes = probes_rw;
    g.recs = recs;
    g.out = d_out;
    g.status = ctx->d_status;
    g.lane_max = (uint32_t)ctx->opt_walk_lane_max;
    g.hop_live = ctx->d_walk_live;
    g.ck = (uint32_t *)(base + o_ck);
    g.cycles = cycles ? 1u : 0u;
    g.bounce = ctx->opt_walk_cycles == 0 && ctx->tb.links_symmetric ? 1u : 0u;   // any cap: no checkpoints needed
    g.pa = pol ? *pa : no_policy;
    g.hist_next = nullptr;
    g.hist_off = (uint32_t)hist_off;
    g.port_off = (uint32_t)port_off;
    g.recs_at_position = 0;
    g.host_addr = t.d_host_addr;
    g.port_stage = t.d_port_stage;
    g.stats = ctx->d_walk_stats;
    ctx->last_walk_cap = hop_cap;
    g.wait_extra = ctx->opt_test_stall_staging ? 16u : 0u;
    g.wait_ns = ctx->opt_test_stall_staging ? 50ull * 1000 * 1000 : 2ull * 1000 * 1000 * 1000;
    uint32_t in_slices = init_grid;
    // hops from tail_hop on run in one walk_tail_kernel launch (indexed tables only)
    const uint32_t opt_tail = ctx->opt_walk_tail_hop < 0 ? t.tail_hop : (uint32_t)ctx->opt_walk_tail_hop;
    const uint32_t tail_hop = (indexed && opt_tail > 0 && opt_tail < hop_cap) ? opt_tail : hop_cap;
    for (uint32_t h = 0; h < tail_hop; ++h) {
        uint2 *cur = (h & 1) ? listB : listA;
        uint2 *nxt = (h & 1) ? listA : listB;
        uint2 *dcur = (h & 1) ? descB : descA;
        uint2 *dnxt = (h & 1) ? descA : descB;
        if (!(direct && h == 0)) {   // directly placed flows start switch-sorted
            pr = pv_prof_start(ctx, st, PV_K_WALK_REGROUP);
            // hop 0's counts come from the init kernel, later hops' from the
            // previous hop kernel when fused
            const bool counted = h == 0 || fuse_hist;
            if (!counted) walk_hist_kernel<<<in_slices, kGridThreads, hist_smem, st>>>(cur, dcur, S, hist);
            walk_scan_kernel<<<1, 1024, 0, st>>>(S, hist, seg, cursor);
            walk_scatter_kernel<<<in_slices, kGridThreads, scat_smem, st>>>(cur, dcur, S, cursor, sorted);
            pv_prof_stop(ctx, st, pr, counted ? 2 : 3);
        }
        g.hist_next = (fuse_hist && h + 1 < tail_hop) ? hist : nullptr;
        g.sorted = sorted;
        g.hop = h;
        g.recs_at_position = (direct && h == 0) ? 1u : 0u;
        g.next_list = nxt;
        g.next_desc = dnxt;
        pr = pv_prof_start(ctx, st, PV_K_WALK_HOP);
        (h == 0 ? hop_fn0 : hop_fn)<<<hop_grid, kHopThreads, hop_smem, st>>>(g);
        pv_prof_stop(ctx, st, pr, 1);
        in_slices = hop_grid;
    }
    if (tail_hop < hop_cap) {
        const uint32_t h = tail_hop - 1;   // the last regrouped hop wrote this list
        uint2 *lst = (h & 1) ? listA : listB;
        uint2 *dsc = (h & 1) ? descA : descB;
        PV_TRY_CUDA(ctx, cudaMemsetAsync(ctx->d_walk_live + tail_hop, 0, (hop_cap - tail_hop) * sizeof(uint32_t), st),
                    "tail live counts");
        g.hop = tail_hop;
        pr = pv_prof_start(ctx, st, PV_K_WALK_HOP);
        tail_fn<<<hop_grid, 256, 0, st>>>(g, lst, dsc, hop_grid, tail_hop);
        pv_prof_stop(ctx, st, pr, 1);
    }
    pv_mark_use(ctx, st);
    return pv_check_launch(ctx, "probe walk kernels");
}

}  // namespace

extern "C" int pv_verify_probes(pv_ctx *ctx, uint32_t M, const pv_probe *d_probes, uint32_t hop_cap,
                                pv_result *d_out, pv_stream stream) {
    if (!ctx) return PV_EINVAL;
    return walk_probes(ctx, M, d_probes, hop_cap, d_out, nullptr, stream);
}

extern "C" int pv_verify_probes_constrained(pv_ctx *ctx, uint32_t M, const pv_probe *d_probes, uint32_t hop_cap,
                                            const uint32_t *d_probe_policy, uint32_t probes_per_policy,
                                            uint32_t first_policy, pv_result *d_out, uint32_t *d_waypoints,
                                            pv_stream stream) {
    if (!ctx) return PV_EINVAL;
    if (!ctx->pol.loaded) return pv_fail(ctx, PV_ESTATE, "pv_verify_probes_constrained: no path policies loaded");
    if (M && !d_waypoints) return pv_fail(ctx, PV_EINVAL, "pv_verify_probes_constrained: NULL waypoint output");
    const PolicyArgs pa = {ctx->pol.d_hdr, ctx->pol.d_sw, ctx->pol.num, d_probe_policy, probes_per_policy,
                           first_policy, d_waypoints};
    return walk_probes(ctx, M, d_probes, hop_cap, d_out, &pa, stream);
}

namespace {

// Checks shared by the compact-flow walks (records or columns).
int check_flow_call(pv_ctx *ctx, const char *fn, uint32_t M, const void *d_dst, const void *d_dport, uint32_t ppg,
                    uint32_t pods, const uint32_t *d_assign, const uint32_t *d_group_mask) {
    if (M && (!d_dst || !d_dport || !d_assign || !d_group_mask))
        return pv_fail(ctx, PV_EINVAL, "%s: NULL device pointer", fn);
    if (M && (ppg == 0 || pods == 0)) return pv_fail(ctx, PV_EINVAL, "%s: group sizes must be > 0", fn);
    return PV_OK;
}

BindArgs flow_records(const pv_ctx *ctx, const pv_flow *f, uint32_t ppg, uint32_t pods, const uint32_t *assign,
                      const uint32_t *group_mask) {
    return {reinterpret_cast<const uint32_t *>(f), reinterpret_cast<const uint16_t *>(f) + 2, 2, 4, ppg, pods,
            assign, group_mask, ctx->tb.d_host_ip};
}

BindArgs flow_columns(const pv_ctx *ctx, const uint32_t *dst, const uint16_t *dport, uint32_t ppg, uint32_t pods,
                      const uint32_t *assign, const uint32_t *group_mask) {
    return {dst, dport, 1, 1, ppg, pods, assign, group_mask, ctx->tb.d_host_ip};
}

int verify_flows_policies(pv_ctx *ctx, const char *fn, uint32_t M, const BindArgs &ba, uint32_t hop_cap,
                          const uint32_t *d_probe_policy, uint32_t probes_per_policy, uint32_t first_policy,
                          pv_probe *d_probes, pv_result *d_out, uint32_t *d_waypoints, pv_stream stream) {
    if (!ctx->pol.loaded) return pv_fail(ctx, PV_ESTATE, "%s: no path policies loaded", fn);
    if (M && !d_waypoints) return pv_fail(ctx, PV_EINVAL, "%s: NULL device pointer", fn);
    const PolicyArgs pa = {ctx->pol.d_hdr, ctx->pol.d_sw, ctx->pol.num, d_probe_policy, probes_per_policy,
                           first_policy, d_waypoints};
    return walk_probes(ctx, M, d_probes, hop_cap, d_out, &pa, stream, &ba);
}

}  // namespace

extern "C" int pv_verify_flows(pv_ctx *ctx, uint32_t M, const pv_flow *d_flows, uint32_t ppg, uint32_t pods,
                               const uint32_t *d_assign, const uint32_t *d_group_mask, uint32_t hop_cap,
                               pv_probe *d_probes, pv_result *d_out, pv_stream stream) {
    if (!ctx) return PV_EINVAL;
    if (int rc = check_flow_call(ctx, "pv_verify_flows", M, d_flows, d_flows, ppg, pods, d_assign, d_group_mask))
        return rc;
    if (((uintptr_t)d_flows & 7) != 0) return pv_fail(ctx, PV_EINVAL, "pv_verify_flows: d_flows must be 8-byte aligned");
    const BindArgs ba = flow_records(ctx, d_flows, ppg, pods, d_assign, d_group_mask);
    return walk_probes(ctx, M, d_probes, hop_cap, d_out, nullptr, stream, &ba);
}

extern "C" int pv_verify_flows_constrained(pv_ctx *ctx, uint32_t M, const pv_flow *d_flows, uint32_t ppg,
                                           uint32_t pods, const uint32_t *d_assign, const uint32_t *d_group_mask,
                                           uint32_t hop_cap, const uint32_t *d_probe_policy,
                                           uint32_t probes_per_policy, uint32_t first_policy, pv_probe *d_probes,
                                           pv_result *d_out, uint32_t *d_waypoints, pv_stream stream) {
    if (!ctx) return PV_EINVAL;
    if (int rc = check_flow_call(ctx, "pv_verify_flows_constrained", M, d_flows, d_flows, ppg, pods, d_assign,
                                 d_group_mask))
        return rc;
    if (((uintptr_t)d_flows & 7) != 0)
        return pv_fail(ctx, PV_EINVAL, "pv_verify_flows_constrained: d_flows must be 8-byte aligned");
    const BindArgs ba = flow_records(ctx, d_flows, ppg, pods, d_assign, d_group_mask);
    return verify_flows_policies(ctx, "pv_verify_flows_constrained", M, ba, hop_cap, d_probe_policy,
                                 probes_per_policy, first_policy, d_probes, d_out, d_waypoints, stream);
}

extern "C" int pv_verify_flow_columns(pv_ctx *ctx, uint32_t M, const uint32_t *d_dst_ip, const uint16_t *d_dport,
                                      uint32_t ppg, uint32_t pods, const uint32_t *d_assign,
                                      const uint32_t *d_group_mask, uint32_t hop_cap, pv_probe *d_probes,
                                      pv_result *d_out, pv_stream stream) {
    if (!ctx) return PV_EINVAL;
    if (int rc = check_flow_call(ctx, "pv_verify_flow_columns", M, d_dst_ip, d_dport, ppg, pods, d_assign,
                                 d_group_mask))
        return rc;
    if (((uintptr_t)d_dst_ip & 3) != 0 || ((uintptr_t)d_dport & 1) != 0)
        return pv_fail(ctx, PV_EINVAL, "pv_verify_flow_columns: d_dst_ip must be 4-byte and d_dport 2-byte aligned");
    const BindArgs ba = flow_columns(ctx, d_dst_ip, d_dport, ppg, pods, d_assign, d_group_mask);
    return walk_probes(ctx, M, d_probes, hop_cap, d_out, nullptr, stream, &ba);
}

extern "C" int pv_verify_flow_columns_constrained(pv_ctx *ctx, uint32_t M, const uint32_t *d_dst_ip,
                                                  const uint16_t *d_dport, uint32_t ppg, uint32_t pods,
                                                  const uint32_t *d_assign, const uint32_t *d_group_mask,
                                                  uint32_t hop_cap, const uint32_t *d_probe_policy,
                                                  uint32_t probes_per_policy, uint32_t first_policy,
                                                  pv_probe *d_probes, pv_result *d_out, uint32_t *d_waypoints,
                                                  pv_stream stream) {
    if (!ctx) return PV_EINVAL;
    if (int rc = check_flow_call(ctx, "pv_verify_flow_columns_constrained", M, d_dst_ip, d_dport, ppg, pods,
                                 d_assign, d_group_mask))
        return rc;
    if (((uintptr_t)d_dst_ip & 3) != 0 || ((uintptr_t)d_dport & 1) != 0)
        return pv_fail(ctx, PV_EINVAL,
                       "pv_verify_flow_columns_constrained: d_dst_ip must be 4-byte and d_dport 2-byte aligned");
    const BindArgs ba = flow_columns(ctx, d_dst_ip, d_dport, ppg, pods, d_assign, d_group_mask);
    return verify_flows_policies(ctx, "pv_verify_flow_columns_constrained", M, ba, hop_cap, d_probe_policy,
                                 probes_per_policy, first_policy, d_probes, d_out, d_waypoints, stream);
}

extern "C" int pv_load_path_policies(pv_ctx *ctx, uint32_t num_policies, const uint32_t *forbid_offs,
                                     const uint16_t *forbid, const uint32_t *must_offs, const uint16_t *must,
                                     const uint8_t *concrete) {
    if (!ctx) return PV_EINVAL;
    if (!ctx->tb.loaded) return pv_fail(ctx, PV_ESTATE, "pv_load_path_policies: load the flow tables first");
    if (num_policies == 0 || !forbid_offs || !must_offs || !concrete)
        return pv_fail(ctx, PV_EINVAL, "pv_load_path_policies: need num_policies > 0 and offset arrays");
    if (forbid_offs[0] != 0 || must_offs[0] != 0)
        return pv_fail(ctx, PV_EINVAL, "pv_load_path_policies: offsets must start at 0");
    const uint32_t S = ctx->tb.num_switches;
    std::vector<uint4> hdr(num_policies);
    const uint32_t nf = forbid_offs[num_policies], nm = must_offs[num_policies];
    if ((nf && !forbid) || (nm && !must)) return pv_fail(ctx, PV_EINVAL, "pv_load_path_policies: NULL switch list");
    if ((uint64_t)nf + nm > 0xFFFFFFFFull) return pv_fail(ctx, PV_EINVAL, "pv_load_path_policies: lists too long");
    for (uint32_t p = 0; p < num_policies; ++p) {
        if (forbid_offs[p + 1] < forbid_offs[p] || must_offs[p + 1] < must_offs[p])
            return pv_fail(ctx, PV_EINVAL, "pv_load_path_policies: policy %u: decreasing offsets", p);
        const uint32_t fl = forbid_offs[p + 1] - forbid_offs[p], ml = must_offs[p + 1] - must_offs[p];
        if (ml > 32) return pv_fail(ctx, PV_EINVAL, "pv_load_path_policies: policy %u has %u > 32 waypoints", p, ml);
        hdr[p] = make_uint4(forbid_offs[p], fl, nf + must_offs[p], ml);
    }
    std::vector<uint16_t> sw((size_t)nf + nm);
    for (uint32_t i = 0; i < nf; ++i) sw[i] = forbid[i];
    for (uint32_t i = 0; i < nm; ++i) sw[(size_t)nf + i] = must[i];
    for (size_t i = 0; i < sw.size(); ++i)
        if (sw[i] >= S)
            return pv_fail(ctx, PV_EINVAL, "pv_load_path_policies: switch id %u >= %u switches", (unsigned)sw[i], S);
    if (int rc0 = pv_load_begin(ctx)) return rc0;
    cudaStream_t ls = ctx->load_stream;
    pv_policy_state p;
    int rc;
    if ((rc = pv_pool_alloc(ctx, (void **)&p.d_hdr, (size_t)num_policies * 16, "policy headers")) ||
        (rc = pv_pool_alloc(ctx, (void **)&p.d_sw, std::max<size_t>(sw.size(), 1) * 2, "policy switches")) ||
        (rc = pv_pool_alloc(ctx, (void **)&p.d_concrete, num_policies, "policy flags"))) {
        pv_free_policies(ctx, p);
        return rc;
    }
    cudaError_t e = cudaMemcpyAsync(p.d_hdr, hdr.data(), (size_t)num_policies * 16, cudaMemcpyHostToDevice, ls);
    if (e == cudaSuccess && !sw.empty()) e = cudaMemcpyAsync(p.d_sw, sw.data(), sw.size() * 2, cudaMemcpyHostToDevice, ls);
    if (e == cudaSuccess) e = cudaMemcpyAsync(p.d_concrete, concrete, num_policies, cudaMemcpyHostToDevice, ls);
    if (e != cudaSuccess) {
        pv_free_policies(ctx, p);
        return pv_cuda_fail(ctx, e, "pv_load_path_policies");
    }
    p.loaded = true;
    p.num = num_policies;
    pv_retire_begin(ctx);
    pv_free_policies(ctx, ctx->pol);
    pv_retire_end(ctx);
    ctx->pol = p;
    return pv_load_end(ctx);
}
