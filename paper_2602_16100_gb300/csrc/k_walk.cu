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

constexpr int kHopThreads = 512;
constexpr int kHopWarps = kHopThreads / 32;
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
__device__ __forceinline__ void bulk_g2s(void *dst, const void *src, uint32_t bytes, uint64_t *bar) {
    asm volatile(
        "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
            smem_u32(dst)),
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
__device__ __forceinline__ bool mbar_wait_bounded(uint64_t *bar, uint32_t parity) {
    for (uint32_t it = 0; it < kWaitLimit; ++it)
        if (mbar_try_wait(bar, parity)) return true;
    return false;
}

// ---------------------------------------------------------------------------
// load: per-switch stable priority sort + compile
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(1024) compile_tables_kernel(const uint32_t *__restrict__ rule_offs,
                                                              const pv_rule *__restrict__ raw,
                                                              const uint32_t *__restrict__ tab_offs,
                                                              uint4 *__restrict__ A, uint2 *__restrict__ B) {
    extern __shared__ uint32_t s_keys[];
    const uint32_t s = blockIdx.x, t = threadIdx.x;
    const uint32_t base = rule_offs[s], n = rule_offs[s + 1] - base;
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
            const uint32_t ms = pv_prefix_mask(r.src_len), md = pv_prefix_mask(r.dst_len);
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
// walk kernels
// ---------------------------------------------------------------------------
// Every thread of the block calls this; threads with want append one slot of
// the shared output list.  Returns the slot (undefined when !want).
__device__ __forceinline__ uint32_t block_append(bool want, uint32_t *count, uint32_t *s_tmp) {
    const uint32_t lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nwarps = blockDim.x >> 5;
    const uint32_t m = __ballot_sync(PV_FULL_MASK, want);
    const uint32_t rank = __popc(m & ((1u << lane) - 1u));
    if (lane == 0) s_tmp[warp] = __popc(m);
    __syncthreads();
    if (threadIdx.x == 0) {
        uint32_t run = 0;
        for (uint32_t w = 0; w < nwarps; ++w) {
            uint32_t c = s_tmp[w];
            s_tmp[w] = run;
            run += c;
        }
        s_tmp[32] = run ? atomicAdd(count, run) : 0;
    }
    __syncthreads();
    const uint32_t pos = s_tmp[32] + s_tmp[warp] + rank;
    __syncthreads();
    return pos;
}

// Live list entry: x = probe id, y = location (switch << 8 | in_port).
__global__ void __launch_bounds__(kGridThreads) walk_init_kernel(
    uint32_t M, const pv_probe *__restrict__ probes, uint32_t H, const uint16_t *__restrict__ host_switch,
    const uint16_t *__restrict__ host_port, pv_result *__restrict__ out, uint2 *__restrict__ list,
    uint32_t *__restrict__ count) {
    __shared__ uint32_t s_tmp[40];
    const uint32_t stride = gridDim.x * kGridThreads;
    for (uint32_t base = blockIdx.x * kGridThreads; base < M; base += stride) {
        const uint32_t i = base + threadIdx.x;
        bool live = false;
        uint32_t loc = 0;
        if (i < M) {
            const uint32_t h = probes[i].src_host;
            if (h < H) {
                live = true;
                loc = ((uint32_t)host_switch[h] << 8) | host_port[h];
            } else {
                pv_result r;
                r.status = PV_NOSRC;
                r.hops = 0;
                r.last_switch = 0xFFFF;
                out[i] = r;
            }
        }
        const uint32_t pos = block_append(live, count, s_tmp);
        if (live) list[pos] = make_uint2(i, loc);
    }
}

__global__ void __launch_bounds__(kGridThreads) walk_hist_kernel(const uint2 *__restrict__ list,
                                                                 const uint32_t *__restrict__ count_ptr,
                                                                 uint32_t S, uint32_t *__restrict__ hist) {
    extern __shared__ uint32_t s_hist[];
    const uint32_t n = *count_ptr;
    const bool use_smem = S <= kSmemHistMax;
    if (use_smem) {
        for (uint32_t j = threadIdx.x; j < S; j += kGridThreads) s_hist[j] = 0;
        __syncthreads();
    }
    for (uint32_t i = blockIdx.x * kGridThreads + threadIdx.x; i < n; i += gridDim.x * kGridThreads) {
        const uint32_t s = list[i].y >> 8;
        if (use_smem) atomicAdd(&s_hist[s], 1u);
        else atomicAdd(&hist[s], 1u);
    }
    if (use_smem) {
        __syncthreads();
        for (uint32_t j = threadIdx.x; j < S; j += kGridThreads)
            if (s_hist[j]) atomicAdd(&hist[j], s_hist[j]);
    }
}

// Single block: seg[s] = exclusive prefix of hist, seg[S] = total;
// cursor[s] = seg[s]; hist cleared for the next hop.
__global__ void __launch_bounds__(1024) walk_scan_kernel(uint32_t S, uint32_t *__restrict__ hist,
                                                         uint32_t *__restrict__ seg, uint32_t *__restrict__ cursor) {
    __shared__ uint32_t s_warp[32];
    __shared__ uint32_t s_carry;
    const uint32_t t = threadIdx.x, lane = t & 31, warp = t >> 5;
    if (t == 0) s_carry = 0;
    __syncthreads();
    for (uint32_t c0 = 0; c0 < S; c0 += 1024) {
        const uint32_t i = c0 + t;
        const uint32_t x = i < S ? hist[i] : 0;
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
    if (t == 0) seg[S] = s_carry;
}

// Block-aggregated counting-sort scatter: each block reserves, per switch,
// one contiguous run of its items with a single atomicAdd.
__global__ void __launch_bounds__(kGridThreads) walk_scatter_kernel(const uint2 *__restrict__ list,
                                                                    const uint32_t *__restrict__ count_ptr,
                                                                    uint32_t S, uint32_t *__restrict__ cursor,
                                                                    uint2 *__restrict__ sorted) {
    extern __shared__ uint32_t s_cnt[];   // [S] counts, then [S] bases
    const uint32_t n = *count_ptr;
    const uint32_t per = (n + gridDim.x - 1) / gridDim.x;
    const uint32_t b0 = min(n, blockIdx.x * per), b1 = min(n, b0 + per);
    if (b0 >= b1) return;
    if (S > kSmemHistMax) {
        for (uint32_t i = b0 + threadIdx.x; i < b1; i += kGridThreads) {
            const uint2 e = list[i];
            sorted[atomicAdd(&cursor[e.y >> 8], 1u)] = e;
        }
        return;
    }
    uint32_t *s_base = s_cnt + S;
    for (uint32_t j = threadIdx.x; j < S; j += kGridThreads) s_cnt[j] = 0;
    __syncthreads();
    for (uint32_t i = b0 + threadIdx.x; i < b1; i += kGridThreads) atomicAdd(&s_cnt[list[i].y >> 8], 1u);
    __syncthreads();
    for (uint32_t j = threadIdx.x; j < S; j += kGridThreads) {
        const uint32_t c = s_cnt[j];
        s_base[j] = c ? atomicAdd(&cursor[j], c) : 0;
        s_cnt[j] = 0;
    }
    __syncthreads();
    for (uint32_t i = b0 + threadIdx.x; i < b1; i += kGridThreads) {
        const uint2 e = list[i];
        const uint32_t s = e.y >> 8;
        sorted[s_base[s] + atomicAdd(&s_cnt[s], 1u)] = e;
    }
}

struct HopArgs {
    const uint2 *sorted;
    const uint32_t *counts;
    uint32_t hop, cap;
    const uint32_t *seg;
    uint32_t S, H;
    const uint32_t *tab_offs;
    const uint4 *rule_a;
    const uint2 *rule_b;
    uint32_t max_pad;
    const uint8_t *region;
    const uint32_t *port_offs;
    const int32_t *port_peer;
    const uint32_t *host_ip;
    const pv_probe *probes;
    pv_result *out;
    uint2 *next_list;
    uint32_t *next_count;
    int32_t *status;
};

__global__ void __launch_bounds__(kHopThreads) walk_hop_kernel(HopArgs g) {
    extern __shared__ __align__(128) uint8_t s_raw[];
    uint4 *sA = reinterpret_cast<uint4 *>(s_raw);
    uint2 *sB = reinterpret_cast<uint2 *>(s_raw + (size_t)g.max_pad * 16);
    __shared__ uint64_t s_bar;
    __shared__ uint32_t s_tmp[40];
    const uint32_t lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const uint32_t n = g.counts[g.hop];
    const uint32_t r0 = (uint32_t)(((uint64_t)n * blockIdx.x) / gridDim.x);
    const uint32_t r1 = (uint32_t)(((uint64_t)n * (blockIdx.x + 1)) / gridDim.x);
    if (r0 >= r1) return;
    if (threadIdx.x == 0) mbar_init(&s_bar, 1);
    __syncthreads();
    uint32_t parity = 0;
    uint32_t pos = r0;
    while (pos < r1) {
        // switch owning position pos: last s with seg[s] <= pos
        uint32_t lo = 0, hi = g.S;   // seg[lo] <= pos < seg[hi]
        while (hi - lo > 1) {
            const uint32_t mid = (lo + hi) >> 1;
            if (g.seg[mid] <= pos) lo = mid;
            else hi = mid;
        }
        const uint32_t s = lo;
        const uint32_t seg_end = min(r1, g.seg[s + 1]);
        const uint32_t t0 = g.tab_offs[s], npad = g.tab_offs[s + 1] - t0;
        __syncthreads();   // everyone is done with the previous table
        if (npad > 0) {
            if (threadIdx.x == 0) {
                asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
                mbar_arrive_expect_tx(&s_bar, npad * 24u);
                bulk_g2s(sA, g.rule_a + t0, npad * 16u, &s_bar);
                bulk_g2s(sB, g.rule_b + t0, npad * 8u, &s_bar);
            }
            const bool ok = mbar_wait_bounded(&s_bar, parity);
            if (__syncthreads_or(!ok)) {
                if (threadIdx.x == 0) pv_device_error(g.status, PV_ETIMEOUT);
                mbar_wait_bounded(&s_bar, parity);   // let copies in flight land
                return;
            }
            parity ^= 1u;
        }
        const uint32_t reg = g.region[s];
        const uint32_t pbase = g.port_offs[s], nports = g.port_offs[s + 1] - pbase;
        for (uint32_t rb = pos; rb < seg_end; rb += 32 * kHopWarps) {
            const uint32_t wb = rb + warp * 32;
            const uint32_t cnt = wb < seg_end ? min(32u, seg_end - wb) : 0u;
            bool my_live = false;
            uint2 my_entry = make_uint2(0, 0);
            for (uint32_t j = 0; j < cnt; ++j) {
                const uint2 e = g.sorted[wb + j];
                const uint32_t pid = e.x, in_port = e.y & 0xFFu;
                // probe record {src_ip, dst_ip, dport | src_host << 16, allowed_mask}
                const uint4 pr = __ldg(reinterpret_cast<const uint4 *>(g.probes) + pid);
                uint32_t status = 0xFFu;   // alive
                uint32_t next = 0;
                if (reg >= 32 || !((pr.w >> reg) & 1u)) {
                    status = PV_VIOLATION;
                } else {
                    const uint32_t src = pr.x, dst = pr.y, dport = pr.z & 0xFFFFu;
                    uint32_t act = PV_DROP;
                    bool found = false;
                    for (uint32_t base = 0; base < npad; base += 32) {
                        const uint4 a = sA[base + lane];
                        const uint2 b = sB[base + lane];
                        const uint32_t diff = ((src ^ a.x) & a.y) | ((dst ^ a.z) & a.w) |
                                              ((in_port ^ b.y) & ((b.y >> 8) & 0xFFu));
                        const bool hit = diff == 0 && dport >= (b.x & 0xFFFFu) && dport <= (b.x >> 16);
                        const uint32_t m = __ballot_sync(PV_FULL_MASK, hit);
                        if (m) {
                            const int l = __ffs(m) - 1;
                            act = __shfl_sync(PV_FULL_MASK, b.y >> 16, l);
                            found = true;
                            break;
                        }
                    }
                    if (!found || act == PV_DROP || act >= nports) {
                        status = PV_DROPPED;
                    } else {
                        const int32_t peer = g.port_peer[pbase + act];
                        if (peer < 0) {
                            status = PV_DROPPED;
                        } else if (peer & PV_PEER_HOST) {
                            const uint32_t q = (uint32_t)(peer & ~PV_PEER_HOST);
                            status = (q < g.H && g.host_ip[q] == dst) ? PV_COMPLIANT : PV_MISDELIVERED;
                        } else if (g.hop + 1 >= g.cap) {
                            status = PV_LOOP;
                        } else {
                            next = (uint32_t)peer;
                        }
                    }
                }
                if (status != 0xFFu) {
                    if (lane == 0) {
                        pv_result r;
                        r.status = (uint8_t)status;
                        r.hops = (uint8_t)(g.hop + 1);
                        r.last_switch = (uint16_t)s;
                        g.out[pid] = r;
                    }
                } else if (lane == j) {
                    my_live = true;
                    my_entry = make_uint2(pid, next);
                }
            }
            const uint32_t slot = block_append(my_live, g.next_count, s_tmp);
            if (my_live) g.next_list[slot] = my_entry;
        }
        pos = seg_end;
    }
}

inline size_t align256(size_t x) { return (x + 255) & ~(size_t)255; }

}  // namespace

// -----------------------------------------------------------------------------
// C ABI
// -----------------------------------------------------------------------------
extern "C" int pv_load_flow_tables(pv_ctx *ctx, uint32_t S, const uint32_t *rule_offs, const pv_rule *rules,
                                   const uint8_t *switch_region, const uint32_t *port_offs,
                                   const int32_t *port_peer, uint32_t H, const uint16_t *host_switch,
                                   const uint16_t *host_port, const uint32_t *host_ip) {
    if (!ctx) return PV_EINVAL;
    if (S == 0 || S > PV_MAX_SWITCHES) return pv_fail(ctx, PV_EINVAL, "num_switches must be 1..%d", PV_MAX_SWITCHES);
    if (H > PV_MAX_HOSTS) return pv_fail(ctx, PV_EINVAL, "num_hosts must be <= %d", PV_MAX_HOSTS);
    if (!rule_offs || !switch_region || !port_offs || (H && (!host_switch || !host_port || !host_ip)))
        return pv_fail(ctx, PV_EINVAL, "pv_load_flow_tables: NULL host pointer");
    if (rule_offs[0] != 0 || port_offs[0] != 0) return pv_fail(ctx, PV_EINVAL, "offsets must start at 0");
    std::vector<uint32_t> tab(S + 1, 0);
    uint32_t max_pad = 0;
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
    }
    const uint32_t R = rule_offs[S], P = port_offs[S];
    if (R && !rules) return pv_fail(ctx, PV_EINVAL, "NULL rules");
    if (P && !port_peer) return pv_fail(ctx, PV_EINVAL, "NULL port_peer");
    for (uint32_t s = 0; s < S; ++s) {
        const uint32_t np = port_offs[s + 1] - port_offs[s];
        for (uint32_t i = rule_offs[s]; i < rule_offs[s + 1]; ++i) {
            const pv_rule &r = rules[i];
            if (r.in_port != PV_ANY_PORT && r.in_port >= np)
                return pv_fail(ctx, PV_EINVAL, "rule %u: in_port %u >= %u ports", i, r.in_port, np);
            if (r.action != PV_DROP && r.action >= np)
                return pv_fail(ctx, PV_EINVAL, "rule %u: action %u >= %u ports", i, r.action, np);
            if (r.src_len > 32 || r.dst_len > 32) return pv_fail(ctx, PV_EINVAL, "rule %u: prefix length > 32", i);
            if (r.dport_lo > r.dport_hi) return pv_fail(ctx, PV_EINVAL, "rule %u: dport_lo > dport_hi", i);
        }
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

    PV_TRY_CUDA(ctx, cudaSetDevice(ctx->device), "cudaSetDevice");
    PV_TRY_CUDA(ctx, cudaDeviceSynchronize(), "pv_load_flow_tables sync");
    pv_free_tables(ctx->tb);
    pv_table_state &t = ctx->tb;
    const uint32_t T = tab[S];
    uint32_t *d_rule_offs = nullptr;
    pv_rule *d_raw = nullptr;
    int rc;
    if ((rc = pv_device_alloc(ctx, (void **)&t.d_tab_offs, (S + 1) * 4, "table offsets")) ||
        (rc = pv_device_alloc(ctx, (void **)&t.d_rule_a, (size_t)T * 16, "rules A")) ||
        (rc = pv_device_alloc(ctx, (void **)&t.d_rule_b, (size_t)T * 8, "rules B")) ||
        (rc = pv_device_alloc(ctx, (void **)&t.d_region, S, "regions")) ||
        (rc = pv_device_alloc(ctx, (void **)&t.d_port_offs, (S + 1) * 4, "port offsets")) ||
        (rc = pv_device_alloc(ctx, (void **)&t.d_port_peer, (size_t)P * 4, "port peers")) ||
        (rc = pv_device_alloc(ctx, (void **)&t.d_host_switch, (size_t)H * 2, "host switch")) ||
        (rc = pv_device_alloc(ctx, (void **)&t.d_host_port, (size_t)H * 2, "host port")) ||
        (rc = pv_device_alloc(ctx, (void **)&t.d_host_ip, (size_t)H * 4, "host ip")) ||
        (rc = pv_device_alloc(ctx, (void **)&d_rule_offs, (S + 1) * 4, "rule offsets")) ||
        (rc = pv_device_alloc(ctx, (void **)&d_raw, (size_t)R * sizeof(pv_rule), "raw rules"))) {
        pv_device_free(d_rule_offs);
        pv_device_free(d_raw);
        pv_free_tables(t);
        return rc;
    }
    cudaError_t e = cudaSuccess;
    e = e ? e : cudaMemcpy(t.d_tab_offs, tab.data(), (S + 1) * 4, cudaMemcpyHostToDevice);
    e = e ? e : cudaMemcpy(t.d_region, switch_region, S, cudaMemcpyHostToDevice);
    e = e ? e : cudaMemcpy(t.d_port_offs, port_offs, (S + 1) * 4, cudaMemcpyHostToDevice);
    if (P) e = e ? e : cudaMemcpy(t.d_port_peer, port_peer, (size_t)P * 4, cudaMemcpyHostToDevice);
    if (H) {
        e = e ? e : cudaMemcpy(t.d_host_switch, host_switch, (size_t)H * 2, cudaMemcpyHostToDevice);
        e = e ? e : cudaMemcpy(t.d_host_port, host_port, (size_t)H * 2, cudaMemcpyHostToDevice);
        e = e ? e : cudaMemcpy(t.d_host_ip, host_ip, (size_t)H * 4, cudaMemcpyHostToDevice);
    }
    e = e ? e : cudaMemcpy(d_rule_offs, rule_offs, (S + 1) * 4, cudaMemcpyHostToDevice);
    if (R) e = e ? e : cudaMemcpy(d_raw, rules, (size_t)R * sizeof(pv_rule), cudaMemcpyHostToDevice);
    if (e == cudaSuccess) {
        uint32_t maxn = 0;
        for (uint32_t s = 0; s < S; ++s) maxn = std::max(maxn, rule_offs[s + 1] - rule_offs[s]);
        uint32_t npow = 1;
        while (npow < maxn) npow <<= 1;
        compile_tables_kernel<<<S, 1024, npow * 4>>>(d_rule_offs, d_raw, t.d_tab_offs, t.d_rule_a, t.d_rule_b);
        e = cudaGetLastError();
        if (e == cudaSuccess) e = cudaDeviceSynchronize();
    }
    pv_device_free(d_rule_offs);
    pv_device_free(d_raw);
    if (e != cudaSuccess) {
        pv_free_tables(t);
        return pv_cuda_fail(ctx, e, "pv_load_flow_tables");
    }
    t.num_switches = S;
    t.num_hosts = H;
    t.max_rules_padded = max_pad;
    const size_t smem = (size_t)max_pad * 24;
    if (smem > ctx->max_smem_optin - 1024) {
        pv_free_tables(t);
        return pv_fail(ctx, PV_EINVAL, "largest flow table needs %zu bytes of shared memory", smem);
    }
    PV_TRY_CUDA(ctx, cudaFuncSetAttribute(walk_hop_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem),
                "walk_hop_kernel smem");
    PV_TRY_CUDA(ctx, cudaFuncSetAttribute(walk_scatter_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                          (int)(2 * kSmemHistMax * 4)),
                "walk_scatter_kernel smem");
    t.loaded = true;
    return PV_OK;
}

extern "C" int pv_verify_probes(pv_ctx *ctx, uint32_t M, const pv_probe *d_probes, uint32_t hop_cap,
                                pv_result *d_out, pv_stream stream) {
    if (!ctx) return PV_EINVAL;
    const pv_table_state &t = ctx->tb;
    if (!t.loaded) return pv_fail(ctx, PV_ESTATE, "pv_verify_probes: no flow tables loaded");
    if (hop_cap == 0 || hop_cap > PV_MAX_HOP_CAP) return pv_fail(ctx, PV_EINVAL, "hop_cap must be 1..255");
    if (M == 0) return PV_OK;
    if (!d_probes || !d_out) return pv_fail(ctx, PV_EINVAL, "pv_verify_probes: NULL device pointer");
    if (((uintptr_t)d_probes & 15) != 0) return pv_fail(ctx, PV_EINVAL, "pv_verify_probes: d_probes must be 16-byte aligned");
    const uint32_t S = t.num_switches;
    const size_t o_a = 0, o_b = align256((size_t)M * 8), o_sorted = o_b + align256((size_t)M * 8);
    const size_t o_hist = o_sorted + align256((size_t)M * 8);
    const size_t o_seg = o_hist + align256((size_t)S * 4);
    const size_t o_cur = o_seg + align256((size_t)(S + 1) * 4);
    const size_t o_cnt = o_cur + align256((size_t)S * 4);
    const size_t total = o_cnt + align256((size_t)(hop_cap + 2) * 4);
    uint8_t *base = (uint8_t *)pv_scratch(ctx, total);
    if (!base) return PV_ENOMEM;
    uint2 *listA = (uint2 *)(base + o_a), *listB = (uint2 *)(base + o_b), *sorted = (uint2 *)(base + o_sorted);
    uint32_t *hist = (uint32_t *)(base + o_hist), *seg = (uint32_t *)(base + o_seg);
    uint32_t *cursor = (uint32_t *)(base + o_cur), *counts = (uint32_t *)(base + o_cnt);
    cudaStream_t st = (cudaStream_t)stream;
    PV_TRY_CUDA(ctx, cudaMemsetAsync(counts, 0, (size_t)(hop_cap + 2) * 4, st), "counts clear");
    PV_TRY_CUDA(ctx, cudaMemsetAsync(hist, 0, (size_t)S * 4, st), "hist clear");
    const uint32_t grid = (uint32_t)ctx->num_sms * 8;
    int pr = pv_prof_start(ctx, st, PV_K_WALK_INIT);
    walk_init_kernel<<<grid, kGridThreads, 0, st>>>(M, d_probes, t.num_hosts, t.d_host_switch, t.d_host_port, d_out,
                                                    listA, counts);
    pv_prof_stop(ctx, st, pr, 1);
    const size_t hist_smem = S <= kSmemHistMax ? (size_t)S * 4 : 0;
    const size_t scat_smem = S <= kSmemHistMax ? (size_t)S * 8 : 0;
    const size_t hop_smem = (size_t)t.max_rules_padded * 24;
    int hop_blocks_per_sm = 0;
    cudaOccupancyMaxActiveBlocksPerMultiprocessor(&hop_blocks_per_sm, walk_hop_kernel, kHopThreads, hop_smem);
    const uint32_t hop_grid = (uint32_t)ctx->num_sms * (uint32_t)std::max(1, hop_blocks_per_sm);
    HopArgs g;
    g.cap = hop_cap;
    g.seg = seg;
    g.S = S;
    g.H = t.num_hosts;
    g.tab_offs = t.d_tab_offs;
    g.rule_a = t.d_rule_a;
    g.rule_b = t.d_rule_b;
    g.max_pad = t.max_rules_padded;
    g.region = t.d_region;
    g.port_offs = t.d_port_offs;
    g.port_peer = t.d_port_peer;
    g.host_ip = t.d_host_ip;
    g.probes = d_probes;
    g.out = d_out;
    g.status = ctx->d_status;
    g.counts = counts;
    for (uint32_t h = 0; h < hop_cap; ++h) {
        uint2 *cur = (h & 1) ? listB : listA;
        uint2 *nxt = (h & 1) ? listA : listB;
        pr = pv_prof_start(ctx, st, PV_K_WALK_REGROUP);
        walk_hist_kernel<<<grid, kGridThreads, hist_smem, st>>>(cur, counts + h, S, hist);
        walk_scan_kernel<<<1, 1024, 0, st>>>(S, hist, seg, cursor);
        walk_scatter_kernel<<<grid, kGridThreads, scat_smem, st>>>(cur, counts + h, S, cursor, sorted);
        pv_prof_stop(ctx, st, pr, 3);
        g.sorted = sorted;
        g.hop = h;
        g.next_list = nxt;
        g.next_count = counts + h + 1;
        pr = pv_prof_start(ctx, st, PV_K_WALK_HOP);
        walk_hop_kernel<<<hop_grid, kHopThreads, hop_smem, st>>>(g);
        pv_prof_stop(ctx, st, pr, 1);
    }
    return pv_check_launch(ctx, "probe walk kernels");
}
