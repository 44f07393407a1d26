// Context management, error reporting and the scratch arena of libpv.
#include <stdarg.h>
#include <stdio.h>

#include <mutex>
#include <new>
#include <utility>
#include <vector>

#include "pv_internal.cuh"

#define PV_VERSION 100

int pv_fail(pv_ctx *ctx, int code, const char *fmt, ...) {
    if (ctx) {
        char buf[512];
        va_list ap;
        va_start(ap, fmt);
        vsnprintf(buf, sizeof buf, fmt, ap);
        va_end(ap);
        ctx->err = buf;
    }
    return code;
}

int pv_cuda_fail(pv_ctx *ctx, cudaError_t e, const char *what) {
    if (e == cudaErrorMemoryAllocation) {
        cudaGetLastError();
        return pv_fail(ctx, PV_ENOMEM, "%s: out of device memory", what);
    }
    return pv_fail(ctx, PV_ECUDA, "%s: %s", what, cudaGetErrorString(e));
}

int pv_device_alloc(pv_ctx *ctx, void **p, size_t bytes, const char *what) {
    *p = nullptr;
    if (bytes == 0) bytes = 16;
    cudaError_t e = cudaMalloc(p, bytes);
    if (e != cudaSuccess) {
        *p = nullptr;
        return pv_cuda_fail(ctx, e, what);
    }
    return PV_OK;
}

void pv_device_free(void *p) {
    if (p) cudaFree(p);
}

int pv_pool_alloc(pv_ctx *ctx, void **p, size_t bytes, const char *what) {
    *p = nullptr;
    if (bytes == 0) bytes = 16;
    cudaError_t e = cudaMallocFromPoolAsync(p, bytes, ctx->pool, ctx->load_stream);
    if (e != cudaSuccess) {
        *p = nullptr;
        return pv_cuda_fail(ctx, e, what);
    }
    return PV_OK;
}

void pv_pool_free(pv_ctx *ctx, void *p) {
    if (p) cudaFreeAsync(p, ctx->retiring ? ctx->retire_stream : ctx->load_stream);
}

int pv_load_begin(pv_ctx *ctx) {
    PV_TRY_CUDA(ctx, cudaSetDevice(ctx->device), "cudaSetDevice");
    return PV_OK;
}

void pv_retire_begin(pv_ctx *ctx) {
    cudaEventRecord(ctx->retire_from, ctx->load_stream);
    cudaStreamWaitEvent(ctx->retire_stream, ctx->retire_from, 0);
    cudaStreamWaitEvent(ctx->retire_stream, ctx->last_use, 0);
    ctx->retiring = true;
}

void pv_retire_end(pv_ctx *ctx) { ctx->retiring = false; }

int pv_load_end(pv_ctx *ctx) {
    PV_TRY_CUDA(ctx, cudaEventRecord(ctx->load_done, ctx->load_stream), "load");
    return pv_check_launch(ctx, "load kernels");
}

void pv_use_begin(pv_ctx *ctx, cudaStream_t st) { cudaStreamWaitEvent(st, ctx->load_done, 0); }

void pv_mark_use(pv_ctx *ctx, cudaStream_t st) { cudaEventRecord(ctx->last_use, st); }

int pv_check_launch(pv_ctx *ctx, const char *what) {
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return pv_cuda_fail(ctx, e, what);
    return PV_OK;
}

int pv_smem_limit(pv_ctx *ctx, const void *fn, const char *what) {
    static std::mutex mu;
    static std::vector<std::pair<int, const void *>> done;
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return pv_cuda_fail(ctx, e, what);
    std::lock_guard<std::mutex> lock(mu);
    for (const auto &d : done)
        if (d.first == dev && d.second == fn) return PV_OK;
    // the dynamic limit plus the kernel's static shared memory may not exceed
    // the device's opt-in maximum
    cudaFuncAttributes fa;
    e = cudaFuncGetAttributes(&fa, fn);
    if (e != cudaSuccess) return pv_cuda_fail(ctx, e, what);
    const size_t lim = ctx->max_smem_optin > fa.sharedSizeBytes ? ctx->max_smem_optin - fa.sharedSizeBytes : 0;
    e = cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)lim);
    if (e != cudaSuccess) return pv_cuda_fail(ctx, e, what);
    done.emplace_back(dev, fn);
    return PV_OK;
}

int pv_blocks_per_sm(pv_ctx *ctx, const void *fn, int threads, size_t smem) {
    for (const auto &o : ctx->occ)
        if (o.fn == fn && o.threads == threads && o.smem == smem) return o.blocks;
    int n = 0;
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, fn, threads, smem) != cudaSuccess) {
        cudaGetLastError();
        n = 0;
    }
    if (ctx->occ.size() >= 64) ctx->occ.clear();   // table sets of many shapes: start over
    ctx->occ.push_back({fn, threads, smem, n});
    return n;
}

void *pv_scratch(pv_ctx *ctx, size_t bytes) {
    if (bytes <= ctx->scratch_bytes && ctx->scratch) return ctx->scratch;
    size_t want = bytes + bytes / 4 + (1u << 20);
    if (ctx->scratch) {
        cudaDeviceSynchronize();
        cudaFree(ctx->scratch);
        ctx->scratch = nullptr;
        ctx->scratch_bytes = 0;
    }
    void *p = nullptr;
    if (pv_device_alloc(ctx, &p, want, "scratch arena") != PV_OK) return nullptr;
    ctx->scratch = p;
    ctx->scratch_bytes = want;
    return p;
}

void pv_free_cluster(pv_ctx *ctx, pv_cluster_state &c) {
    pv_free_ptr(ctx, c.d_labels);
    pv_free_ptr(ctx, c.d_inv);
    pv_free_ptr(ctx, c.d_inv_rank);
    pv_free_ptr(ctx, c.d_key_base);
    pv_free_ptr(ctx, c.d_rows);
    c = pv_cluster_state();
}

void pv_free_policies(pv_ctx *ctx, pv_policy_state &p) {
    pv_free_ptr(ctx, p.d_hdr);
    pv_free_ptr(ctx, p.d_sw);
    pv_free_ptr(ctx, p.d_concrete);
    p = pv_policy_state();
}

void pv_free_tables(pv_ctx *ctx, pv_table_state &t) {
    pv_free_ptr(ctx, t.d_blob);
    pv_free_ptr(ctx, t.d_blob_offs);
    pv_free_ptr(ctx, t.d_region);
    pv_free_ptr(ctx, t.d_port_offs);
    pv_free_ptr(ctx, t.d_port_peer);
    pv_free_ptr(ctx, t.d_host_switch);
    pv_free_ptr(ctx, t.d_host_port);
    pv_free_ptr(ctx, t.d_host_ip);
    pv_free_ptr(ctx, t.d_host_addr);
    pv_free_ptr(ctx, t.d_port_stage);
    pv_free_ptr(ctx, t.d_in_offs);
    pv_free_ptr(ctx, t.d_in_links);
    pv_free_ptr(ctx, t.d_raw);
    t = pv_table_state();
}

int pv_prof_start(pv_ctx *ctx, cudaStream_t st, int group) {
    pv_prof_state &p = ctx->prof;
    if (!p.on) return -1;
    if (p.used * 2 + 2 > p.pool.size()) {
        for (int i = 0; i < 2; ++i) {
            cudaEvent_t e;
            if (cudaEventCreate(&e) != cudaSuccess) return -1;
            p.pool.push_back(e);
        }
        p.group.push_back(0);
        p.nlaunch.push_back(0);
    }
    const size_t i = p.used++;
    p.group[i] = group;
    p.nlaunch[i] = 0;
    cudaEventRecord(p.pool[2 * i], st);
    return (int)i;
}

void pv_prof_stop(pv_ctx *ctx, cudaStream_t st, int pair, uint32_t launches) {
    if (pair < 0) return;
    pv_prof_state &p = ctx->prof;
    p.nlaunch[pair] = launches;
    cudaEventRecord(p.pool[2 * (size_t)pair + 1], st);
}

extern "C" int pv_profile_enable(pv_ctx *ctx, int on) {
    if (!ctx) return PV_EINVAL;
    pv_prof_state &p = ctx->prof;
    if (on) {
        for (int g = 0; g < PV_K_COUNT; ++g) {
            p.ms[g] = 0;
            p.launches[g] = 0;
        }
        p.used = 0;
    }
    p.on = on != 0;
    return PV_OK;
}

extern "C" int pv_profile_collect(pv_ctx *ctx, pv_stream stream) {
    if (!ctx) return PV_EINVAL;
    pv_prof_state &p = ctx->prof;
    PV_TRY_CUDA(ctx, cudaStreamSynchronize((cudaStream_t)stream), "pv_profile_collect");
    for (size_t i = 0; i < p.used; ++i) {
        float ms = 0;
        PV_TRY_CUDA(ctx, cudaEventElapsedTime(&ms, p.pool[2 * i], p.pool[2 * i + 1]), "event elapsed");
        p.ms[p.group[i]] += ms;
        p.launches[p.group[i]] += p.nlaunch[i];
    }
    p.used = 0;
    return PV_OK;
}

extern "C" int pv_profile_read(const pv_ctx *ctx, int group, double *total_ms, uint64_t *launches) {
    if (!ctx || group < 0 || group >= PV_K_COUNT) return PV_EINVAL;
    if (total_ms) *total_ms = ctx->prof.ms[group];
    if (launches) *launches = ctx->prof.launches[group];
    return PV_OK;
}

extern "C" int pv_version(void) { return PV_VERSION; }

extern "C" int pv_create(pv_ctx **out, int cuda_device) {
    if (!out) return PV_EINVAL;
    *out = nullptr;
    pv_ctx *ctx = new (std::nothrow) pv_ctx();
    if (!ctx) return PV_ENOMEM;
    int ndev = 0;
    cudaError_t e = cudaGetDeviceCount(&ndev);
    if (e != cudaSuccess || cuda_device < 0 || cuda_device >= ndev) {
        delete ctx;
        return PV_ECUDA;
    }
    e = cudaSetDevice(cuda_device);
    if (e != cudaSuccess) {
        delete ctx;
        return PV_ECUDA;
    }
    ctx->device = cuda_device;
    cudaDeviceGetAttribute(&ctx->num_sms, cudaDevAttrMultiProcessorCount, cuda_device);
    int smem = 0;
    cudaDeviceGetAttribute(&smem, cudaDevAttrMaxSharedMemoryPerBlockOptin, cuda_device);
    ctx->max_smem_optin = (size_t)smem;
    cudaMemPoolProps props = {};
    props.allocType = cudaMemAllocationTypePinned;
    props.location.type = cudaMemLocationTypeDevice;
    props.location.id = cuda_device;
    uint64_t keep = ~0ull;   // keep freed blocks for the next load
    int no_reuse_deps = 0;
    if (cudaStreamCreateWithFlags(&ctx->load_stream, cudaStreamNonBlocking) != cudaSuccess ||
        cudaStreamCreateWithFlags(&ctx->retire_stream, cudaStreamNonBlocking) != cudaSuccess ||
        cudaEventCreateWithFlags(&ctx->retire_from, cudaEventDisableTiming) != cudaSuccess ||
        cudaMemPoolCreate(&ctx->pool, &props) != cudaSuccess ||
        cudaMemPoolSetAttribute(ctx->pool, cudaMemPoolAttrReleaseThreshold, &keep) != cudaSuccess ||
        // no reuse that would make the load stream wait for the retire stream
        // (and so for evaluation work): blocks freed there are reused once done
        cudaMemPoolSetAttribute(ctx->pool, cudaMemPoolReuseAllowInternalDependencies, &no_reuse_deps) !=
            cudaSuccess ||
        cudaEventCreateWithFlags(&ctx->last_use, cudaEventDisableTiming) != cudaSuccess ||
        cudaEventCreateWithFlags(&ctx->load_done, cudaEventDisableTiming) != cudaSuccess) {
        if (ctx->load_stream) cudaStreamDestroy(ctx->load_stream);
        if (ctx->retire_stream) cudaStreamDestroy(ctx->retire_stream);
        if (ctx->retire_from) cudaEventDestroy(ctx->retire_from);
        if (ctx->pool) cudaMemPoolDestroy(ctx->pool);
        delete ctx;
        return PV_ECUDA;
    }
    if (pv_device_alloc(ctx, (void **)&ctx->d_status, sizeof(int32_t), "status word") != PV_OK ||
        cudaMemset(ctx->d_status, 0, sizeof(int32_t)) != cudaSuccess ||
        pv_device_alloc(ctx, (void **)&ctx->d_walk_live, (PV_MAX_HOP_CAP + 1) * sizeof(uint32_t),
                        "walk statistics") != PV_OK ||
        cudaMemset(ctx->d_walk_live, 0, (PV_MAX_HOP_CAP + 1) * sizeof(uint32_t)) != cudaSuccess ||
        pv_device_alloc(ctx, (void **)&ctx->d_reach_asym, sizeof(uint32_t), "reach symmetry flag") != PV_OK ||
        pv_device_alloc(ctx, (void **)&ctx->d_walk_stats, PV_WALK_STATS * sizeof(unsigned long long),
                        "walk statistics counters") != PV_OK ||
        cudaMemset(ctx->d_walk_stats, 0, PV_WALK_STATS * sizeof(unsigned long long)) != cudaSuccess) {
        pv_device_free(ctx->d_status);
        pv_device_free(ctx->d_walk_live);
        pv_device_free(ctx->d_walk_stats);
        pv_device_free(ctx->d_reach_asym);
        cudaEventDestroy(ctx->last_use);
        cudaEventDestroy(ctx->load_done);
        cudaEventDestroy(ctx->retire_from);
        cudaStreamDestroy(ctx->load_stream);
        cudaStreamDestroy(ctx->retire_stream);
        cudaMemPoolDestroy(ctx->pool);
        delete ctx;
        return PV_ENOMEM;
    }
    *out = ctx;
    return PV_OK;
}

extern "C" void pv_destroy(pv_ctx *ctx) {
    if (!ctx) return;
    cudaDeviceSynchronize();
    pv_discard_table_load(ctx);
    pv_free_cluster(ctx, ctx->cl);
    pv_free_tables(ctx, ctx->tb);
    pv_free_policies(ctx, ctx->pol);
    cudaStreamSynchronize(ctx->load_stream);
    cudaStreamSynchronize(ctx->retire_stream);
    cudaEventDestroy(ctx->last_use);
    cudaEventDestroy(ctx->load_done);
    cudaEventDestroy(ctx->retire_from);
    cudaStreamDestroy(ctx->load_stream);
    cudaStreamDestroy(ctx->retire_stream);
    if (ctx->reach_side) cudaStreamDestroy(ctx->reach_side);
    if (ctx->reach_fork) cudaEventDestroy(ctx->reach_fork);
    if (ctx->reach_join) cudaEventDestroy(ctx->reach_join);
    cudaMemPoolDestroy(ctx->pool);
    for (cudaEvent_t e : ctx->prof.pool) cudaEventDestroy(e);
    pv_device_free(ctx->scratch);
    pv_device_free(ctx->d_status);
    pv_device_free(ctx->d_walk_live);
    pv_device_free(ctx->d_walk_stats);
    pv_device_free(ctx->d_reach_asym);
    delete ctx;
}

extern "C" const char *pv_last_error(const pv_ctx *ctx) {
    if (!ctx) return "null context";
    return ctx->err.c_str();
}

extern "C" int pv_sync(pv_ctx *ctx, pv_stream stream) {
    if (!ctx) return PV_EINVAL;
    PV_TRY_CUDA(ctx, cudaStreamSynchronize((cudaStream_t)stream), "pv_sync");
    int32_t st = 0;
    PV_TRY_CUDA(ctx, cudaMemcpy(&st, ctx->d_status, sizeof st, cudaMemcpyDeviceToHost), "pv_sync status");
    if (st != 0) {
        PV_TRY_CUDA(ctx, cudaMemset(ctx->d_status, 0, sizeof(int32_t)), "pv_sync reset");
        if (st == PV_ETIMEOUT) return pv_fail(ctx, PV_ETIMEOUT, "a bounded device-side wait gave up");
        return pv_fail(ctx, st, "device-detected error %d (malformed device-resident input)", (int)st);
    }
    return PV_OK;
}

extern "C" int pv_set_option(pv_ctx *ctx, int option, int64_t value) {
    if (!ctx) return PV_EINVAL;
    switch (option) {
    case PV_OPT_SELECTOR_KERNEL:
        if (value < 0 || value > 2) return pv_fail(ctx, PV_EINVAL, "selector kernel must be 0, 1 or 2");
        ctx->opt_selector = (int)value;
        return PV_OK;
    case PV_OPT_WALK_KERNEL:
        if (value < 0 || value > 2) return pv_fail(ctx, PV_EINVAL, "walk kernel must be 0, 1 or 2");
        ctx->opt_walk = (int)value;
        return PV_OK;
    case PV_OPT_WALK_LANE_MAX:
        if (value < 0 || value > 65535) return pv_fail(ctx, PV_EINVAL, "lane-mode list length must be 0..65535");
        ctx->opt_walk_lane_max = (int)value;
        return PV_OK;
    case PV_OPT_TEST_STALL_STAGING:
        if (value < 0 || value > 1) return pv_fail(ctx, PV_EINVAL, "stall-staging test switch must be 0 or 1");
        ctx->opt_test_stall_staging = (int)value;
        return PV_OK;
    case PV_OPT_WALK_CYCLES:
        if (value < 0 || value > 1) return pv_fail(ctx, PV_EINVAL, "walk cycle option must be 0 or 1");
        ctx->opt_walk_cycles = (int)value;
        return PV_OK;
    case PV_OPT_WALK_TAIL_HOP:
        if (value < -1 || value > PV_MAX_HOP_CAP) return pv_fail(ctx, PV_EINVAL, "tail hop must be -1..255");
        ctx->opt_walk_tail_hop = (int)value;
        return PV_OK;
    case PV_OPT_REACH_KERNEL:
        if (value < 0 || value > 1) return pv_fail(ctx, PV_EINVAL, "reach kernel must be 0 or 1");
        ctx->opt_reach = (int)value;
        return PV_OK;
    case PV_OPT_SCHED_KERNEL:
        if (value < 0 || value > 2) return pv_fail(ctx, PV_EINVAL, "scheduler kernel must be 0..2");
        ctx->opt_sched_kernel = (int)value;
        return PV_OK;
    case PV_OPT_SELECTOR_DEDUPE:
        if (value < 0 || value > 2) return pv_fail(ctx, PV_EINVAL, "selector dedupe switch must be 0, 1 or 2");
        ctx->opt_selector_dedupe = (int)value;
        return PV_OK;
    case PV_OPT_WALK_STATS:
        if (value < 0 || value > 1) return pv_fail(ctx, PV_EINVAL, "walk statistics switch must be 0 or 1");
        ctx->opt_walk_stats = (int)value;
        return PV_OK;
    default:
        return pv_fail(ctx, PV_EINVAL, "unknown option %d", option);
    }
}

extern "C" int pv_get_stat(const pv_ctx *ctx, int stat, int64_t *value) {
    if (!ctx || !value) return PV_EINVAL;
    switch (stat) {
    case PV_STAT_SELECTOR_ROWS_BUILT: *value = ctx->cl.rows_built ? 1 : 0; return PV_OK;
    case PV_STAT_SCRATCH_BYTES: *value = (int64_t)ctx->scratch_bytes; return PV_OK;
    case PV_STAT_WALK_INDEX_FITS: *value = ctx->tb.index_fits ? 1 : 0; return PV_OK;
    case PV_STAT_WALK_INDEX_BYTES: *value = (int64_t)ctx->tb.max_blob_bytes; return PV_OK;
    case PV_STAT_WALK_LIVE_TOTAL: {
        uint32_t live[PV_MAX_HOP_CAP + 1];
        const uint32_t cap = ctx->last_walk_cap;
        if (cap && cudaMemcpy(live, ctx->d_walk_live, cap * sizeof(uint32_t), cudaMemcpyDeviceToHost) !=
                       cudaSuccess)
            return PV_ECUDA;
        int64_t sum = 0;
        for (uint32_t h = 0; h < cap; ++h) sum += live[h];
        *value = sum;
        return PV_OK;
    }
    case PV_STAT_REACH_COMPONENTS: {
        uint32_t asym = 1;
        if (ctx->last_reach_comp &&
            cudaMemcpy(&asym, ctx->d_reach_asym, sizeof asym, cudaMemcpyDeviceToHost) != cudaSuccess)
            return PV_ECUDA;
        *value = (ctx->last_reach_comp && asym == 0) ? 1 : 0;
        return PV_OK;
    }
    case PV_STAT_WALK_FIRST_MATCHES:
    case PV_STAT_WALK_RULE_TESTS:
    case PV_STAT_WALK_INTERVAL_LOOKUPS:
    case PV_STAT_WALK_SCAN_DEPTH:
    case PV_STAT_WALK_INDEX_MISMATCHES: {
        unsigned long long c[PV_WALK_STATS];
        if (cudaMemcpy(c, ctx->d_walk_stats, sizeof c, cudaMemcpyDeviceToHost) != cudaSuccess) return PV_ECUDA;
        *value = (int64_t)c[stat - PV_STAT_WALK_FIRST_MATCHES];
        return PV_OK;
    }
    default: return PV_EINVAL;
    }
}
