// Path scheduling (Sec. 4.2: the flow scheduling module computes paths that
// respect the constraint object -- weighted Dijkstra, breadth-first when no
// weights are given -- and turns each path into per-hop flow rules).
//
// A request asks for a path from a source host to a destination host over
// the switches its jurisdiction mask permits and its policy does not forbid,
// through the policy's waypoints in order.  The path is the concatenation of
// shortest segments, each made canonical: walking back from the segment's
// end, every switch takes the predecessor link with the smallest (source
// switch, source port) among those on a shortest path.  Any exact shortest-
// path algorithm therefore yields the same path; one block per request runs
// in-place Bellman-Ford pull sweeps over the links into each switch (every
// sweep only lowers upper bounds, so the fixpoint is exact), all in shared
// memory, and one thread walks the predecessors back.
#include <cuda_runtime.h>

#include <algorithm>
#include <vector>

#include "pv_internal.cuh"

namespace {

constexpr int kSchedThreads = 256;
constexpr uint32_t kSchedMaxSwitches = 16384;
constexpr uint32_t kInf = 0xFFFFFFFFu;

struct SchedArgs {
    uint32_t S, H;
    const uint8_t *region;
    const uint32_t *port_offs;
    const uint16_t *host_switch, *host_port;
    const uint32_t *in_offs, *in_links;
    const uint16_t *weights;       // [ports] or null (unit weights)
    const uint4 *pol_hdr;          // path policies (null: none loaded)
    const uint16_t *pol_sw;
    uint32_t num_pol;
    const pv_path_req *req;
    uint32_t R, max_len;
    uint32_t *visits;              // [R][max_len]: switch << 16 | in_port << 8 | out_port
    uint8_t *len, *status;
};

__device__ __forceinline__ uint32_t link_weight(const SchedArgs &a, uint32_t u, uint32_t p) {
    if (!a.weights) return 1u;
    const uint32_t w = a.weights[a.port_offs[u] + p];
    return w ? w : 1u;   // a weight of 0 counts as 1
}

// With kStaged the block first copies the links into each switch, with their
// weights resolved, to shared memory, where every sweep and the predecessor
// pass read them.
template <bool kStaged>
__global__ void __launch_bounds__(kSchedThreads) sched_paths_kernel(SchedArgs a) {
    extern __shared__ uint32_t s_mem[];
    const uint32_t S = a.S, okw = (S + 31) / 32;
    volatile uint32_t *dist = s_mem;                 // [S]
    uint32_t *ok = s_mem + S;                        // [okw] permitted switches
    uint32_t *vis = ok + okw;                        // [max_len] visits
    uint32_t *back = vis + a.max_len;                // [max_len] links of a segment, last first
    uint32_t *pred = back + a.max_len;               // [S] canonical predecessor link (kStaged)
    uint32_t *g_offs = pred + (kStaged ? S : 0u);    // [S + 1]
    const uint32_t L = a.in_offs[S];
    uint32_t *g_links = g_offs + (kStaged ? S + 1 : 0u);   // [L]
    uint16_t *g_w = reinterpret_cast<uint16_t *>(g_links + (kStaged ? L : 0u));   // [L] link weights
    __shared__ uint32_t s_st, s_n;
    const uint32_t t = threadIdx.x, nt = blockDim.x;
    auto allowed = [&](uint32_t s) { return (ok[s >> 5] >> (s & 31)) & 1u; };
    const uint32_t *in_offs = a.in_offs, *in_links = a.in_links;
    if (kStaged) {
        for (uint32_t v = t; v <= S; v += nt) g_offs[v] = a.in_offs[v];
        for (uint32_t l = t; l < L; l += nt) {
            const uint32_t x = a.in_links[l];
            g_links[l] = x;
            g_w[l] = (uint16_t)link_weight(a, x >> 16, (x >> 8) & 0xFFu);
        }
        __syncthreads();
        in_offs = g_offs;
        in_links = g_links;
    }
    // weight of in-link l = (u, p) of switch v
    auto lw = [&](uint32_t l, uint32_t x) -> uint32_t {
        return kStaged ? (uint32_t)g_w[l] : link_weight(a, x >> 16, (x >> 8) & 0xFFu);
    };
    for (uint32_t r = blockIdx.x; r < a.R; r += gridDim.x) {
        const pv_path_req q = a.req[r];
        if (q.src_host >= a.H || q.dst_host >= a.H) {
            if (t == 0) {
                a.status[r] = PV_PATH_NOSRC;
                a.len[r] = 0;
            }
            continue;
        }
        uint4 ph = make_uint4(0, 0, 0, 0);
        if (a.pol_hdr && q.policy < a.num_pol) ph = a.pol_hdr[q.policy];
        for (uint32_t w = t; w < okw; w += nt) {
            uint32_t bits = 0;
            for (uint32_t b = 0; b < 32; ++b) {
                const uint32_t s = w * 32 + b;
                if (s >= S) break;
                const uint32_t reg = a.region[s];
                bool fine = reg < 32 && ((q.allowed_mask >> reg) & 1u);
                for (uint32_t i = 0; i < ph.y && fine; ++i) fine = a.pol_sw[ph.x + i] != s;
                if (fine) bits |= 1u << b;
            }
            ok[w] = bits;
        }
        __syncthreads();
        const uint32_t src_sw = a.host_switch[q.src_host], dst_sw = a.host_switch[q.dst_host];
        uint32_t st = (allowed(src_sw) && allowed(dst_sw)) ? PV_PATH_OK : PV_PATH_BLOCKED;
        for (uint32_t i = 0; i < ph.w && st == PV_PATH_OK; ++i)
            if (!allowed(a.pol_sw[ph.z + i])) st = PV_PATH_BLOCKED;
        uint32_t n = 1, cur = src_sw;
        if (t == 0) vis[0] = src_sw << 16 | (uint32_t)a.host_port[q.src_host] << 8;
        for (uint32_t i = 0; i <= ph.w && st == PV_PATH_OK; ++i) {
            const uint32_t tgt = i < ph.w ? a.pol_sw[ph.z + i] : dst_sw;
            if (tgt == cur) continue;
            for (uint32_t v = t; v < S; v += nt) dist[v] = v == cur ? 0u : kInf;
            __syncthreads();
            // pull sweeps until nothing changes (at most S are needed)
            for (uint32_t round = 0; round <= S; ++round) {
                int changed = 0;
                for (uint32_t v = t; v < S; v += nt) {
                    if (v == cur || !allowed(v)) continue;
                    uint32_t best = dist[v];
                    for (uint32_t l = in_offs[v]; l < in_offs[v + 1]; ++l) {
                        const uint32_t x = in_links[l], u = x >> 16;
                        if (!allowed(u)) continue;
                        const uint32_t du = dist[u];
                        if (du == kInf) continue;
                        const uint32_t c = du + lw(l, x);
                        if (c < best) best = c;
                    }
                    if (best < dist[v]) {
                        dist[v] = best;
                        changed = 1;
                    }
                }
                if (!__syncthreads_or(changed)) break;
            }
            if (dist[tgt] == kInf) {
                st = PV_PATH_BLOCKED;
                break;
            }
            if (kStaged) {
                // every switch's canonical predecessor at once: the first link
                // (smallest (u, p)) on a shortest path into it
                for (uint32_t v = t; v < S; v += nt) {
                    uint32_t pick = kInf;
                    if (v != cur && dist[v] != kInf)
                        for (uint32_t l = in_offs[v]; l < in_offs[v + 1] && pick == kInf; ++l) {
                            const uint32_t x = in_links[l], u = x >> 16;
                            if (allowed(u) && dist[u] != kInf && dist[u] + lw(l, x) == dist[v]) pick = x;
                        }
                    pred[v] = pick;
                }
                __syncthreads();
            }
            if (t == 0) {
                // canonical walk back from tgt: smallest (u, p) on a shortest path
                const uint32_t room = a.max_len - n;
                uint32_t k = 0, v = tgt, s_status = PV_PATH_OK;
                while (v != cur) {
                    uint32_t pick = kInf;
                    if (kStaged) {
                        pick = pred[v];
                    } else {
                        for (uint32_t l = in_offs[v]; l < in_offs[v + 1] && pick == kInf; ++l) {
                            const uint32_t x = in_links[l], u = x >> 16;
                            if (!allowed(u) || dist[u] == kInf) continue;
                            if (dist[u] + lw(l, x) == dist[v]) pick = x;
                        }
                    }
                    if (pick == kInf) {   // cannot happen once the distances are exact
                        s_status = PV_PATH_BLOCKED;
                        break;
                    }
                    if (k >= room) {
                        s_status = PV_PATH_TOO_LONG;
                        break;
                    }
                    // {source port, switch v, its in_port}
                    back[k++] = ((pick >> 8) & 0xFFu) << 24 | v << 8 | (pick & 0xFFu);
                    v = pick >> 16;
                }
                if (s_status == PV_PATH_OK)
                    while (k > 0) {
                        const uint32_t b = back[--k];
                        vis[n - 1] |= b >> 24;                              // out port toward the next switch
                        vis[n++] = ((b >> 8) & 0xFFFFu) << 16 | (b & 0xFFu) << 8;
                    }
                s_st = s_status;
                s_n = n;
            }
            __syncthreads();
            st = s_st;
            n = s_n;
            cur = tgt;
        }
        if (st == PV_PATH_OK) {
            if (t == 0) vis[n - 1] |= a.host_port[q.dst_host];
            if (t == 0) s_st = PV_PATH_OK;
            __syncthreads();
            // a recurring (switch, in_port) cannot be realised by header rules
            for (uint32_t i = t; i < n; i += nt)
                for (uint32_t j = i + 1; j < n; ++j)
                    if ((vis[i] >> 8) == (vis[j] >> 8)) s_st = PV_PATH_REPEAT;
            __syncthreads();
            st = s_st;
        }
        for (uint32_t i = t; i < n && st == PV_PATH_OK; i += nt) a.visits[(size_t)r * a.max_len + i] = vis[i];
        if (t == 0) {
            a.status[r] = (uint8_t)st;
            a.len[r] = (uint8_t)(st == PV_PATH_OK ? n : 0);
        }
        __syncthreads();   // shared state is rebuilt for the next request
    }
}

// Visit i of an OK request becomes, at its switch, the rule {priority,
// in_port, src /32, dst /32, any destination port, output port}, in slot
// r * max_len + i; unused slots get rule_switch 0xFFFF.
__global__ void compile_path_rules_kernel(uint32_t R, const pv_path_req *__restrict__ req,
                                          const uint32_t *__restrict__ host_ip, uint32_t H, uint32_t max_len,
                                          const uint32_t *__restrict__ visits, const uint8_t *__restrict__ len,
                                          const uint8_t *__restrict__ status, uint16_t priority,
                                          pv_rule *__restrict__ rules, uint16_t *__restrict__ rule_switch) {
    const size_t total = (size_t)R * max_len;
    for (size_t k = blockIdx.x * (size_t)blockDim.x + threadIdx.x; k < total; k += (size_t)gridDim.x * blockDim.x) {
        const uint32_t r = (uint32_t)(k / max_len), i = (uint32_t)(k % max_len);
        pv_rule x;
        x.priority = priority;
        x.in_port = 0;
        x.src_ip = x.dst_ip = 0;
        x.src_len = x.dst_len = 0;
        x.dport_lo = 0;
        x.dport_hi = 0xFFFF;
        x.action = PV_DROP;
        uint16_t sw = 0xFFFF;
        const pv_path_req q = req[r];
        if (status[r] == PV_PATH_OK && i < len[r] && q.src_host < H && q.dst_host < H) {
            const uint32_t h = visits[k];
            x.in_port = (uint16_t)((h >> 8) & 0xFFu);
            x.src_ip = host_ip[q.src_host];
            x.src_len = 32;
            x.dst_ip = host_ip[q.dst_host];
            x.dst_len = 32;
            x.action = (uint16_t)(h & 0xFFu);
            sw = (uint16_t)(h >> 16);
        } else {
            x.priority = 0;
        }
        rules[k] = x;
        rule_switch[k] = sw;
    }
}

}  // namespace

extern "C" int pv_schedule_paths(pv_ctx *ctx, uint32_t num_requests, const pv_path_req *d_requests,
                                 const uint16_t *d_link_weights, uint32_t max_len, uint32_t *d_visits,
                                 uint8_t *d_len, uint8_t *d_status, pv_stream stream) {
    if (!ctx) return PV_EINVAL;
    const pv_table_state &t = ctx->tb;
    if (!t.loaded) return pv_fail(ctx, PV_ESTATE, "pv_schedule_paths: no flow tables loaded");
    if (max_len == 0 || max_len > PV_MAX_HOP_CAP) return pv_fail(ctx, PV_EINVAL, "max_len must be 1..255");
    if (t.num_switches > kSchedMaxSwitches)
        return pv_fail(ctx, PV_EINVAL, "pv_schedule_paths: more than %u switches", kSchedMaxSwitches);
    if (num_requests == 0) return PV_OK;
    if (!d_requests || !d_visits || !d_len || !d_status)
        return pv_fail(ctx, PV_EINVAL, "pv_schedule_paths: NULL device pointer");
    SchedArgs a;
    a.S = t.num_switches;
    a.H = t.num_hosts;
    a.region = t.d_region;
    a.port_offs = t.d_port_offs;
    a.host_switch = t.d_host_switch;
    a.host_port = t.d_host_port;
    a.in_offs = t.d_in_offs;
    a.in_links = t.d_in_links;
    a.weights = d_link_weights;
    a.pol_hdr = ctx->pol.loaded ? ctx->pol.d_hdr : nullptr;
    a.pol_sw = ctx->pol.loaded ? ctx->pol.d_sw : nullptr;
    a.num_pol = ctx->pol.loaded ? ctx->pol.num : 0;
    a.req = d_requests;
    a.R = num_requests;
    a.max_len = max_len;
    a.visits = d_visits;
    a.len = d_len;
    a.status = d_status;
    const size_t base_smem = ((size_t)a.S + (a.S + 31) / 32 + 2 * (size_t)max_len) * 4;
    // the links (with weights) and the predecessors staged when they fit
    const uint32_t L = t.num_links;
    const size_t staged_smem = base_smem + ((size_t)a.S + (size_t)a.S + 1 + L) * 4 + ((size_t)L * 2 + 15) / 16 * 16;
    const int force = ctx->opt_sched_kernel;   // 0 automatic, 1 links from global memory, 2 staged
    const bool staged_fits = staged_smem <= std::min<size_t>(96 * 1024, ctx->max_smem_optin - 1024);
    if (force == 2 && !staged_fits)
        return pv_fail(ctx, PV_EINVAL, "pv_schedule_paths: the staged links do not fit shared memory");
    const bool staged = force == 2 || (force == 0 && staged_fits);
    const size_t smem = staged ? staged_smem : base_smem;
    const void *fn = staged ? (const void *)sched_paths_kernel<true> : (const void *)sched_paths_kernel<false>;
    PV_TRY_CUDA(ctx, cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem), "sched smem");
    int per_sm = 1;
    cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, fn, kSchedThreads, smem);
    const uint32_t grid = std::min<uint32_t>(num_requests, (uint32_t)std::max(per_sm, 1) * ctx->num_sms);
    pv_use_begin(ctx, (cudaStream_t)stream);
    const int pr = pv_prof_start(ctx, (cudaStream_t)stream, PV_K_SCHEDULE);
    if (staged)
        sched_paths_kernel<true><<<grid, kSchedThreads, smem, (cudaStream_t)stream>>>(a);
    else
        sched_paths_kernel<false><<<grid, kSchedThreads, smem, (cudaStream_t)stream>>>(a);
    pv_prof_stop(ctx, (cudaStream_t)stream, pr, 1);
    pv_mark_use(ctx, (cudaStream_t)stream);
    return pv_check_launch(ctx, "sched_paths_kernel");
}

extern "C" int pv_compile_path_rules(pv_ctx *ctx, uint32_t num_requests, const pv_path_req *d_requests,
                                     uint32_t max_len, const uint32_t *d_visits, const uint8_t *d_len,
                                     const uint8_t *d_status, uint16_t priority, pv_rule *d_rules,
                                     uint16_t *d_rule_switch, pv_stream stream) {
    if (!ctx) return PV_EINVAL;
    const pv_table_state &t = ctx->tb;
    if (!t.loaded) return pv_fail(ctx, PV_ESTATE, "pv_compile_path_rules: no flow tables loaded");
    if (max_len == 0 || max_len > PV_MAX_HOP_CAP) return pv_fail(ctx, PV_EINVAL, "max_len must be 1..255");
    if (num_requests == 0) return PV_OK;
    if (!d_requests || !d_visits || !d_len || !d_status || !d_rules || !d_rule_switch)
        return pv_fail(ctx, PV_EINVAL, "pv_compile_path_rules: NULL device pointer");
    const size_t total = (size_t)num_requests * max_len;
    const uint32_t grid = (uint32_t)std::min<size_t>((total + 255) / 256, (size_t)ctx->num_sms * 8);
    pv_use_begin(ctx, (cudaStream_t)stream);
    const int pr = pv_prof_start(ctx, (cudaStream_t)stream, PV_K_SCHEDULE);
    compile_path_rules_kernel<<<grid, 256, 0, (cudaStream_t)stream>>>(num_requests, d_requests, t.d_host_ip,
                                                                      t.num_hosts, max_len, d_visits, d_len,
                                                                      d_status, priority, d_rules, d_rule_switch);
    pv_prof_stop(ctx, (cudaStream_t)stream, pr, 1);
    pv_mark_use(ctx, (cudaStream_t)stream);
    return pv_check_launch(ctx, "compile_path_rules_kernel");
}

extern "C" int pv_install_path_rules(pv_ctx *ctx, uint32_t num_slots, const pv_rule *d_rules,
                                     const uint16_t *d_rule_switch) {
    if (!ctx) return PV_EINVAL;
    if (!ctx->tb.loaded) return pv_fail(ctx, PV_ESTATE, "pv_install_path_rules: no flow tables loaded");
    if (num_slots == 0) return PV_OK;
    if (!d_rules || !d_rule_switch) return pv_fail(ctx, PV_EINVAL, "pv_install_path_rules: NULL device pointer");
    std::vector<pv_rule> add(num_slots);
    std::vector<uint16_t> sw(num_slots);
    // the compiled rules come from an evaluation call: the load stream waits
    // for it, then reads them and the loaded rules
    if (int rc0 = pv_load_begin(ctx)) return rc0;
    cudaStream_t ls = ctx->load_stream;
    PV_TRY_CUDA(ctx, cudaStreamWaitEvent(ls, ctx->last_use, 0), "pv_install_path_rules");
    const pv_table_host h = ctx->tbh;   // copy: the reload below replaces ctx->tbh
    const uint32_t S = (uint32_t)h.region.size();
    std::vector<pv_rule> base(h.rule_offs[S]);
    PV_TRY_CUDA(ctx, cudaMemcpyAsync(add.data(), d_rules, (size_t)num_slots * sizeof(pv_rule),
                                     cudaMemcpyDeviceToHost, ls),
                "path rules download");
    PV_TRY_CUDA(ctx, cudaMemcpyAsync(sw.data(), d_rule_switch, (size_t)num_slots * 2, cudaMemcpyDeviceToHost, ls),
                "path rule switches download");
    if (!base.empty())
        PV_TRY_CUDA(ctx, cudaMemcpyAsync(base.data(), ctx->tb.d_raw, base.size() * sizeof(pv_rule),
                                         cudaMemcpyDeviceToHost, ls),
                    "loaded rules download");
    PV_TRY_CUDA(ctx, cudaStreamSynchronize(ls), "pv_install_path_rules");
    std::vector<uint32_t> count(S, 0);
    for (uint32_t k = 0; k < num_slots; ++k)
        if (sw[k] < S) ++count[sw[k]];
    std::vector<uint32_t> offs(S + 1, 0);
    for (uint32_t s = 0; s < S; ++s) offs[s + 1] = offs[s] + count[s] + (h.rule_offs[s + 1] - h.rule_offs[s]);
    std::vector<pv_rule> rules(offs[S]);
    std::vector<uint32_t> cur(offs.begin(), offs.end() - 1);
    for (uint32_t k = 0; k < num_slots; ++k)   // new rules first, in slot order: they win priority ties
        if (sw[k] < S) rules[cur[sw[k]]++] = add[k];
    for (uint32_t s = 0; s < S; ++s)
        for (uint32_t i = h.rule_offs[s]; i < h.rule_offs[s + 1]; ++i) rules[cur[s]++] = base[i];
    return pv_load_flow_tables(ctx, S, offs.data(), rules.data(), h.region.data(), h.port_offs.data(),
                               h.port_peer.data(), (uint32_t)h.host_ip.size(), h.host_switch.data(),
                               h.host_port.data(), h.host_ip.data());
}
