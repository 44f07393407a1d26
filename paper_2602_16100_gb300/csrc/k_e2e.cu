// End-to-end composition of the validator (Sec. 4.2 hybrid coordination:
// pods are placed first, then flows from their attachments are compiled and
// checked; Sec. 5.5: an intent passes only if all of its checks pass).
#include <cuda_runtime.h>

#include "pv_internal.cuh"

namespace {

constexpr int kThreads = 256;

// Warp per group: count the feasible nodes (< N) of the group's row, then for
// each pod select the r-th set bit, r = draw mod count.
__global__ void __launch_bounds__(kThreads) place_pods_kernel(uint32_t G, uint32_t pods, uint32_t N,
                                                              const uint32_t *__restrict__ bits, uint32_t W,
                                                              const uint64_t *__restrict__ draws,
                                                              uint32_t *__restrict__ assign) {
    const uint32_t lane = threadIdx.x & 31;
    const uint32_t nwords = (N + 31) / 32, tail = N & 31;
    for (uint32_t g = (blockIdx.x * kThreads + threadIdx.x) >> 5; g < G; g += (gridDim.x * kThreads) >> 5) {
        const uint32_t *row = bits + (size_t)g * W;
        auto word = [&](uint32_t w) -> uint32_t {
            uint32_t x = row[w];
            if (w == nwords - 1 && tail) x &= (1u << tail) - 1u;
            return x;
        };
        uint32_t c = 0;
        for (uint32_t w = lane; w < nwords; w += 32) c += __popc(word(w));
        for (int d = 16; d > 0; d >>= 1) c += __shfl_xor_sync(PV_FULL_MASK, c, d);
        for (uint32_t j = 0; j < pods; ++j) {
            const size_t pod = (size_t)g * pods + j;
            if (c == 0) {
                if (lane == 0) assign[pod] = PV_UNPLACED;
                continue;
            }
            uint32_t r = (uint32_t)(draws[pod] % c);   // rank among feasible nodes
            uint32_t result = PV_UNPLACED;
            for (uint32_t w0 = 0; w0 < nwords; w0 += 32) {
                const uint32_t w = w0 + lane;
                const uint32_t x = w < nwords ? word(w) : 0u;
                const uint32_t pc = __popc(x);
                uint32_t incl = pc;
                for (int d = 1; d < 32; d <<= 1) {
                    uint32_t y = __shfl_up_sync(PV_FULL_MASK, incl, d);
                    if (lane >= (uint32_t)d) incl += y;
                }
                const uint32_t total = __shfl_sync(PV_FULL_MASK, incl, 31);
                if (r < total) {
                    const uint32_t excl = incl - pc;
                    const bool here = r >= excl && r < incl;
                    const uint32_t who = __ffs(__ballot_sync(PV_FULL_MASK, here)) - 1;
                    if (lane == who) {
                        uint32_t y = x;
                        for (uint32_t k = r - excl; k > 0; --k) y &= y - 1u;
                        result = w * 32 + (__ffs(y) - 1);
                    }
                    result = __shfl_sync(PV_FULL_MASK, result, who);
                    break;
                }
                r -= total;
            }
            if (lane == 0) assign[pod] = result;
        }
    }
}

__global__ void __launch_bounds__(kThreads) bind_probes_kernel(uint32_t M, pv_probe *__restrict__ probes,
                                                               uint32_t ppg, uint32_t pods,
                                                               const uint32_t *__restrict__ assign, uint32_t H,
                                                               const uint32_t *__restrict__ host_ip) {
    for (uint32_t k = blockIdx.x * kThreads + threadIdx.x; k < M; k += gridDim.x * kThreads) {
        const uint32_t g = k / ppg;
        const uint32_t pod = g * pods + (k - g * ppg) % pods;
        const uint32_t node = assign[pod];
        if (node < H) {
            probes[k].src_host = (uint16_t)node;
            probes[k].src_ip = host_ip[node];
        } else {
            probes[k].src_host = PV_NO_HOST;
            probes[k].src_ip = 0;
        }
    }
}

// Warp per group: placement check of each pod against the group's row, probe
// status histogram, verdict.
__global__ void __launch_bounds__(kThreads) aggregate_kernel(uint32_t G, uint32_t pods, uint32_t N,
                                                             const uint32_t *__restrict__ bits, uint32_t W,
                                                             const uint8_t *__restrict__ gflags,
                                                             const uint32_t *__restrict__ assign, uint32_t ppg,
                                                             const pv_result *__restrict__ results,
                                                             uint8_t *__restrict__ pass, uint32_t *__restrict__ counts,
                                                             const uint32_t *__restrict__ hits,
                                                             const uint32_t *__restrict__ group_pol,
                                                             uint32_t first_pol, uint32_t num_pol,
                                                             const uint4 *__restrict__ pol_hdr,
                                                             const uint8_t *__restrict__ concrete) {
    const uint32_t lane = threadIdx.x & 31;
    for (uint32_t g = (blockIdx.x * kThreads + threadIdx.x) >> 5; g < G; g += (gridDim.x * kThreads) >> 5) {
        uint32_t placed = 0;
        for (uint32_t j = lane; j < pods; j += 32) {
            const uint32_t a = assign[(size_t)g * pods + j];
            placed += (a < N && ((bits[(size_t)g * W + (a >> 5)] >> (a & 31)) & 1u)) ? 1u : 0u;
        }
        uint32_t c[6] = {0, 0, 0, 0, 0, 0};
        const uint32_t *res = reinterpret_cast<const uint32_t *>(results + (size_t)g * ppg);
        if ((((uintptr_t)res) & 15) == 0) {
            // 16-byte loads, statuses counted in a packed histogram (8 bits per
            // status; flushed before any field could reach 256)
            const uint4 *res4 = reinterpret_cast<const uint4 *>(res);
            const uint32_t n4 = ppg / 4;
            uint64_t acc = 0;
            uint32_t since = 0;
            auto bump = [](uint32_t r) {   // statuses past PV_NOSRC are not counted
                const uint32_t st = r & 0xFFu;
                return st < 6u ? 1ull << (st * 8u) : 0ull;
            };
            auto flush = [&]() {
#pragma unroll
                for (int s = 0; s < 6; ++s) c[s] += (uint32_t)(acc >> (8 * s)) & 0xFFu;
                acc = 0;
                since = 0;
            };
            uint32_t k = lane;
            for (; k + 96 < n4; k += 128) {   // four loads in flight per lane
                const uint4 v0 = __ldg(res4 + k), v1 = __ldg(res4 + k + 32);
                const uint4 v2 = __ldg(res4 + k + 64), v3 = __ldg(res4 + k + 96);
                acc += bump(v0.x) + bump(v0.y) + bump(v0.z) + bump(v0.w) + bump(v1.x) + bump(v1.y) + bump(v1.z) +
                       bump(v1.w) + bump(v2.x) + bump(v2.y) + bump(v2.z) + bump(v2.w) + bump(v3.x) + bump(v3.y) +
                       bump(v3.z) + bump(v3.w);
                if (++since == 15) flush();   // at most 16 per field each step
            }
            flush();
            for (; k < n4; k += 32) {
                const uint4 v = __ldg(res4 + k);
                acc += bump(v.x) + bump(v.y) + bump(v.z) + bump(v.w);
            }
            flush();
            for (uint32_t k = 4 * n4 + lane; k < ppg; k += 32) {
                const uint32_t st = __ldg(res + k) & 0xFFu;
#pragma unroll
                for (int s = 0; s < 6; ++s) c[s] += st == (uint32_t)s;
            }
        } else {
            for (uint32_t k = lane; k < ppg; k += 32) {
                const uint32_t st = __ldg(res + k) & 0xFFu;
#pragma unroll
                for (int s = 0; s < 6; ++s) c[s] += st == (uint32_t)s;
            }
        }
        // path constraints: every probe must have entered all waypoints of the
        // group's policy, and the policy must name a concrete flow
        uint32_t missed = 0;
        bool policy_ok = true;
        if (pol_hdr) {
            const uint32_t p = group_pol ? group_pol[g] : first_pol + g;
            if (p < num_pol) {
                const uint32_t nm = pol_hdr[p].w;
                const uint32_t full = nm >= 32 ? 0xFFFFFFFFu : ((1u << nm) - 1u);
                for (uint32_t k = lane; k < ppg; k += 32) missed += hits[(size_t)g * ppg + k] != full;
                policy_ok = concrete[p] != 0;
            }
        }
        for (int d = 16; d > 0; d >>= 1) {
            missed += __shfl_xor_sync(PV_FULL_MASK, missed, d);
            placed += __shfl_xor_sync(PV_FULL_MASK, placed, d);
#pragma unroll
            for (int s = 0; s < 6; ++s) c[s] += __shfl_xor_sync(PV_FULL_MASK, c[s], d);
        }
        if (lane == 0) {
            uint32_t *out = counts + (size_t)g * 8;
#pragma unroll
            for (int s = 0; s < 6; ++s) out[s] = c[s];
            out[6] = placed;
            out[7] = missed;
            const bool ok = placed == pods && !(gflags[g] & (PV_F_UNKNOWN_VALUE | PV_F_BAD_EXPR)) && c[0] == ppg &&
                            policy_ok && missed == 0;
            pass[g] = ok ? 1 : 0;
        }
    }
}

uint32_t grid_for(const pv_ctx *ctx, size_t items, uint32_t per_block) {
    size_t b = (items + per_block - 1) / per_block;
    size_t cap = (size_t)ctx->num_sms * 16;
    if (b > cap) b = cap;
    return (uint32_t)(b ? b : 1);
}

}  // namespace

extern "C" int pv_place_pods(pv_ctx *ctx, uint32_t G, uint32_t pods, const uint32_t *d_bits, uint32_t W,
                             const uint64_t *d_draws, uint32_t *d_assign, pv_stream stream) {
    if (!ctx) return PV_EINVAL;
    if (!ctx->cl.loaded) return pv_fail(ctx, PV_ESTATE, "pv_place_pods: no cluster loaded");
    if (G == 0) return PV_OK;
    if (pods == 0) return pv_fail(ctx, PV_EINVAL, "pv_place_pods: pods_per_group must be > 0");
    if (!d_bits || !d_draws || !d_assign) return pv_fail(ctx, PV_EINVAL, "pv_place_pods: NULL device pointer");
    if (W < (ctx->cl.num_nodes + 31) / 32) return pv_fail(ctx, PV_EINVAL, "pv_place_pods: words_per_row too small");
    const int pr = pv_prof_start(ctx, (cudaStream_t)stream, PV_K_PLACE);
    place_pods_kernel<<<grid_for(ctx, (size_t)G * 32, kThreads), kThreads, 0, (cudaStream_t)stream>>>(
        G, pods, ctx->cl.num_nodes, d_bits, W, d_draws, d_assign);
    pv_prof_stop(ctx, (cudaStream_t)stream, pr, 1);
    return pv_check_launch(ctx, "place_pods_kernel");
}

// Probe records from compact flows: {src_ip, dst_ip, dport | src_host << 16,
// mask}, the source bound as in bind_probes_kernel.
__global__ void __launch_bounds__(kThreads) bind_flows_kernel(uint32_t M, const uint2 *__restrict__ flows,
                                                              uint32_t ppg, uint32_t pods,
                                                              const uint32_t *__restrict__ assign,
                                                              const uint32_t *__restrict__ group_mask, uint32_t H,
                                                              const uint32_t *__restrict__ host_ip,
                                                              uint4 *__restrict__ probes) {
    for (uint32_t k = blockIdx.x * kThreads + threadIdx.x; k < M; k += gridDim.x * kThreads) {
        const uint32_t g = k / ppg;
        const uint32_t node = assign[g * pods + (k - g * ppg) % pods];
        const uint2 f = __ldg(flows + k);
        const bool placed = node < H;
        probes[k] = make_uint4(placed ? host_ip[node] : 0u, f.x,
                               (f.y & 0xFFFFu) | (placed ? node : (uint32_t)PV_NO_HOST) << 16, group_mask[g]);
    }
}

extern "C" int pv_bind_flows(pv_ctx *ctx, uint32_t M, const pv_flow *d_flows, uint32_t ppg, uint32_t pods,
                             const uint32_t *d_assign, const uint32_t *d_group_mask, pv_probe *d_probes,
                             pv_stream stream) {
    if (!ctx) return PV_EINVAL;
    if (!ctx->tb.loaded) return pv_fail(ctx, PV_ESTATE, "pv_bind_flows: no flow tables loaded");
    if (M == 0) return PV_OK;
    if (ppg == 0 || pods == 0) return pv_fail(ctx, PV_EINVAL, "pv_bind_flows: group sizes must be > 0");
    if (!d_flows || !d_assign || !d_group_mask || !d_probes)
        return pv_fail(ctx, PV_EINVAL, "pv_bind_flows: NULL device pointer");
    if (((uintptr_t)d_probes & 15) != 0 || ((uintptr_t)d_flows & 7) != 0)
        return pv_fail(ctx, PV_EINVAL, "pv_bind_flows: d_probes must be 16-byte and d_flows 8-byte aligned");
    pv_use_begin(ctx, (cudaStream_t)stream);
    const int pr = pv_prof_start(ctx, (cudaStream_t)stream, PV_K_BIND);
    bind_flows_kernel<<<grid_for(ctx, M, kThreads), kThreads, 0, (cudaStream_t)stream>>>(
        M, reinterpret_cast<const uint2 *>(d_flows), ppg, pods, d_assign, d_group_mask, ctx->tb.num_hosts,
        ctx->tb.d_host_ip, reinterpret_cast<uint4 *>(d_probes));
    pv_prof_stop(ctx, (cudaStream_t)stream, pr, 1);
    pv_mark_use(ctx, (cudaStream_t)stream);
    return pv_check_launch(ctx, "bind_flows_kernel");
}

extern "C" int pv_bind_probes(pv_ctx *ctx, uint32_t M, pv_probe *d_probes, uint32_t ppg, uint32_t pods,
                              const uint32_t *d_assign, pv_stream stream) {
    if (!ctx) return PV_EINVAL;
    if (!ctx->tb.loaded) return pv_fail(ctx, PV_ESTATE, "pv_bind_probes: no flow tables loaded");
    if (M == 0) return PV_OK;
    if (ppg == 0 || pods == 0) return pv_fail(ctx, PV_EINVAL, "pv_bind_probes: group sizes must be > 0");
    if (!d_probes || !d_assign) return pv_fail(ctx, PV_EINVAL, "pv_bind_probes: NULL device pointer");
    pv_use_begin(ctx, (cudaStream_t)stream);
    const int pr = pv_prof_start(ctx, (cudaStream_t)stream, PV_K_BIND);
    bind_probes_kernel<<<grid_for(ctx, M, kThreads), kThreads, 0, (cudaStream_t)stream>>>(
        M, d_probes, ppg, pods, d_assign, ctx->tb.num_hosts, ctx->tb.d_host_ip);
    pv_prof_stop(ctx, (cudaStream_t)stream, pr, 1);
    pv_mark_use(ctx, (cudaStream_t)stream);
    return pv_check_launch(ctx, "bind_probes_kernel");
}

extern "C" int pv_aggregate_intents(pv_ctx *ctx, uint32_t G, uint32_t pods, const uint32_t *d_bits, uint32_t W,
                                    const uint8_t *d_gflags, const uint32_t *d_assign, uint32_t ppg,
                                    const pv_result *d_results, uint8_t *d_pass, uint32_t *d_counts,
                                    pv_stream stream) {
    if (!ctx) return PV_EINVAL;
    if (!ctx->cl.loaded) return pv_fail(ctx, PV_ESTATE, "pv_aggregate_intents: no cluster loaded");
    if (G == 0) return PV_OK;
    if (pods == 0) return pv_fail(ctx, PV_EINVAL, "pv_aggregate_intents: pods_per_group must be > 0");
    if (!d_bits || !d_gflags || !d_assign || !d_pass || !d_counts || (ppg && !d_results))
        return pv_fail(ctx, PV_EINVAL, "pv_aggregate_intents: NULL device pointer");
    if (W < (ctx->cl.num_nodes + 31) / 32) return pv_fail(ctx, PV_EINVAL, "pv_aggregate_intents: words_per_row too small");
    pv_use_begin(ctx, (cudaStream_t)stream);
    const int pr = pv_prof_start(ctx, (cudaStream_t)stream, PV_K_AGGREGATE);
    aggregate_kernel<<<grid_for(ctx, (size_t)G * 32, kThreads), kThreads, 0, (cudaStream_t)stream>>>(
        G, pods, ctx->cl.num_nodes, d_bits, W, d_gflags, d_assign, ppg, d_results, d_pass, d_counts, nullptr,
        nullptr, 0, 0, nullptr, nullptr);
    pv_prof_stop(ctx, (cudaStream_t)stream, pr, 1);
    pv_mark_use(ctx, (cudaStream_t)stream);
    return pv_check_launch(ctx, "aggregate_kernel");
}

extern "C" int pv_aggregate_constrained(pv_ctx *ctx, uint32_t G, uint32_t pods, const uint32_t *d_bits, uint32_t W,
                                        const uint8_t *d_gflags, const uint32_t *d_assign, uint32_t ppg,
                                        const pv_result *d_results, const uint32_t *d_waypoints,
                                        const uint32_t *d_group_policy, uint32_t first_policy, uint8_t *d_pass,
                                        uint32_t *d_counts, pv_stream stream) {
    if (!ctx) return PV_EINVAL;
    if (!ctx->cl.loaded) return pv_fail(ctx, PV_ESTATE, "pv_aggregate_constrained: no cluster loaded");
    if (!ctx->pol.loaded) return pv_fail(ctx, PV_ESTATE, "pv_aggregate_constrained: no path policies loaded");
    if (G == 0) return PV_OK;
    if (pods == 0) return pv_fail(ctx, PV_EINVAL, "pv_aggregate_constrained: pods_per_group must be > 0");
    if (!d_bits || !d_gflags || !d_assign || !d_pass || !d_counts || (ppg && (!d_results || !d_waypoints)))
        return pv_fail(ctx, PV_EINVAL, "pv_aggregate_constrained: NULL device pointer");
    if (W < (ctx->cl.num_nodes + 31) / 32)
        return pv_fail(ctx, PV_EINVAL, "pv_aggregate_constrained: words_per_row too small");
    pv_use_begin(ctx, (cudaStream_t)stream);
    const int pr = pv_prof_start(ctx, (cudaStream_t)stream, PV_K_AGGREGATE);
    aggregate_kernel<<<grid_for(ctx, (size_t)G * 32, kThreads), kThreads, 0, (cudaStream_t)stream>>>(
        G, pods, ctx->cl.num_nodes, d_bits, W, d_gflags, d_assign, ppg, d_results, d_pass, d_counts,
        d_waypoints, d_group_policy, first_policy, ctx->pol.num, ctx->pol.d_hdr, ctx->pol.d_concrete);
    pv_prof_stop(ctx, (cudaStream_t)stream, pr, 1);
    pv_mark_use(ctx, (cudaStream_t)stream);
    return pv_check_launch(ctx, "aggregate_kernel");
}
