// Internal declarations of libpv (not part of the C ABI).
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include <string>
#include <vector>

#include "pv.h"

#define PV_FULL_MASK 0xFFFFFFFFu
#define PV_WALK_STATS 8   // walk statistics counters (5 used)

// -----------------------------------------------------------------------------
// context
// -----------------------------------------------------------------------------
struct pv_cluster_state {
    bool loaded = false;
    uint32_t num_nodes = 0, num_keys = 0;
    uint16_t *d_labels = nullptr;     // [K][N]
    uint32_t *d_inv = nullptr;        // [K][2048]: bit v = some node carries value v of key k
    uint32_t *d_inv_rank = nullptr;   // [K][2048]: set bits of the key's inventory before word w
    uint32_t *d_key_base = nullptr;   // [K + 1]: first value row of key k; [K] = number of value rows
    // per-(key, value) node bitsets, then one "present" row per key
    bool rows_built = false;
    uint32_t row_words = 0;           // words per value row (multiple of 4)
    uint32_t num_value_rows = 0;
    uint32_t *d_rows = nullptr;       // [num_value_rows + K][row_words]
};

struct pv_table_state {
    bool loaded = false;
    uint32_t num_switches = 0, num_hosts = 0;
    uint32_t max_rules_padded = 0;    // largest per-switch table, in rules (multiple of 32)
    // One blob per switch (16-byte aligned): header, the plain rules, the
    // first-match index, then every rule in first-match order (see k_walk.cu).
    uint8_t *d_blob = nullptr;
    uint64_t *d_blob_offs = nullptr;  // [S + 1] byte offsets
    uint32_t max_blob_bytes = 0;      // largest stage of the indexed kernel (all but the full rule list)
    uint32_t tail_hop = 8;            // default first tail hop for these tables (see walk_probes)
    uint32_t max_linear_bytes = 0;    // largest header + full rule list (linear-scan kernel)
    uint32_t max_ports = 0;           // most ports on one switch
    bool index_fits = false;          // every blob fits shared memory
    uint8_t *d_region = nullptr;      // [S]
    uint32_t *d_port_offs = nullptr;  // [S + 1]
    int32_t *d_port_peer = nullptr;   // [ports]
    uint16_t *d_host_switch = nullptr, *d_host_port = nullptr;
    uint32_t *d_host_ip = nullptr;
    uint2 *d_host_addr = nullptr;     // [H] {address, attachment port}: one load for a walk's source host
    uint2 *d_port_stage = nullptr;    // [ports] {peer, peer's region or host address}: the hop kernel's port stage
    // switch-to-switch links into each switch, sorted by (source switch,
    // source port): u << 16 | p << 8 | q for port p of u cabled to port q
    uint32_t *d_in_offs = nullptr;    // [S + 1]
    uint32_t *d_in_links = nullptr;   // [links]
    uint32_t num_links = 0;           // switch-to-switch links
    bool links_symmetric = false;     // every switch port's peer port leads back to it
    pv_rule *d_raw = nullptr;         // [rules] as loaded (for rule installation)
};

// Host copy of the loaded flow tables except the rules, which stay on the
// device (the path scheduler's rule installation merges into them and
// reloads).
struct pv_table_host {
    std::vector<uint32_t> rule_offs, port_offs, host_ip;
    std::vector<uint8_t> region;
    std::vector<int32_t> port_peer;
    std::vector<uint16_t> host_switch, host_port;
};

// Path constraints of flow sets (pv_load_path_policies): per policy
// {forbidden offset, count, waypoint offset, count} into one switch list.
struct pv_policy_state {
    bool loaded = false;
    uint32_t num = 0;
    uint4 *d_hdr = nullptr;        // [num]
    uint16_t *d_sw = nullptr;      // forbidden and waypoint switch ids
    uint8_t *d_concrete = nullptr; // [num]: the constraint names a concrete flow
};

struct pv_prof_state {
    bool on = false;
    std::vector<cudaEvent_t> pool;     // event pairs: [2i] start, [2i+1] stop
    std::vector<int> group;            // group of pair i
    std::vector<uint32_t> nlaunch;     // kernel launches inside pair i
    size_t used = 0;                   // pairs recorded since the last collect
    double ms[PV_K_COUNT] = {};
    uint64_t launches[PV_K_COUNT] = {};
};

struct pv_table_load;   // a two-part flow-table load in progress (k_walk.cu)

struct pv_ctx {
    int device = 0;
    // Loads run on their own stream with memory from the context's pool, so
    // they wait only for the evaluation work that may still read the state
    // they replace (last_use), not for copies or kernels on other streams.
    cudaStream_t load_stream = nullptr;
    // The state a load replaces is freed on the retire stream, after the last
    // evaluation call that may read it (last_use) and the load's own work
    // before the replacement (retire_from); the load stream never waits for
    // evaluation work.
    cudaStream_t retire_stream = nullptr;
    cudaEvent_t retire_from = nullptr;
    bool retiring = false;            // pv_pool_free frees on the retire stream
    cudaMemPool_t pool = nullptr;
    cudaEvent_t last_use = nullptr;   // recorded by every call that reads loaded state
    cudaEvent_t load_done = nullptr;  // recorded at the end of every load (its device work)
    // compliant reach: the sweep path's kernels run on a side stream forked
    // from the caller's (created on the first call)
    cudaStream_t reach_side = nullptr;
    cudaEvent_t reach_fork = nullptr, reach_join = nullptr;
    pv_prof_state prof;
    // blocks per SM by (kernel, block size, dynamic shared memory): the
    // occupancy query runs once per combination
    struct occ_entry { const void *fn; int threads; size_t smem; int blocks; };
    std::vector<occ_entry> occ;
    int num_sms = 0;
    size_t max_smem_optin = 0;
    std::string err;
    int32_t *d_status = nullptr;      // first device-detected error (0 = none)
    int opt_selector = 0, opt_walk = 0;
    int opt_selector_dedupe = 0;      // 1: identical selectors evaluated once (2: with weak hashes, for tests)
    int opt_sched_kernel = 0;         // path scheduler kernel: 0 automatic, 1-2 forced (tests)
    int opt_walk_lane_max = 96;
    int opt_walk_cycles = 0;
    int opt_walk_tail_hop = -1;       // hops from here on run in one tail launch (0: never, -1: by the tables)
    int opt_walk_stats = 0;           // 1: walks run the statistics kernels
    unsigned long long *d_walk_stats = nullptr;   // [PV_WALK_STATS] counters of the last statistics walk
    int opt_test_stall_staging = 0;   // failure test: staging waits expect bytes that never come
    uint32_t *d_walk_live = nullptr;  // [PV_MAX_HOP_CAP + 1] live probes per hop of the last walk
    uint32_t last_walk_cap = 0;       // hop cap of the last walk
    int opt_reach = 0;                // 0: components on symmetric graphs, 1: sweeps only
    uint32_t *d_reach_asym = nullptr; // != 0: the last reach call's graph is not symmetric
    bool last_reach_comp = false;     // the last reach call launched the component path
    void *scratch = nullptr;
    size_t scratch_bytes = 0;
    pv_cluster_state cl;
    pv_table_state tb;
    pv_table_host tbh;
    pv_table_load *table_load = nullptr;   // between pv_load_flow_tables_begin and _end
    pv_policy_state pol;
};

// -----------------------------------------------------------------------------
// host helpers (pv_api.cu)
// -----------------------------------------------------------------------------
int pv_fail(pv_ctx *ctx, int code, const char *fmt, ...);
int pv_cuda_fail(pv_ctx *ctx, cudaError_t e, const char *what);
// Returns a device pointer to at least `bytes` of context scratch (grows the
// arena; growing synchronises the device).  nullptr on failure (error set).
void *pv_scratch(pv_ctx *ctx, size_t bytes);
int pv_device_alloc(pv_ctx *ctx, void **p, size_t bytes, const char *what);
void pv_device_free(void *p);
// Loaded-state memory: stream-ordered on the context's load stream and pool.
int pv_pool_alloc(pv_ctx *ctx, void **p, size_t bytes, const char *what);
void pv_pool_free(pv_ctx *ctx, void *p);
// A load builds its new state in fresh memory on the load stream, without
// waiting for the evaluation calls still reading the state it replaces.
// Between pv_retire_begin and pv_retire_end, pv_pool_free frees on the
// retire stream, which first waits (on the device) for the last of those
// calls and for the load stream's work so far.  pv_load_end records
// load_done on the load stream (the new state is complete) and returns
// without waiting for the load's device work.  A load that fails leaves
// the previous state loaded.
int pv_load_begin(pv_ctx *ctx);
void pv_retire_begin(pv_ctx *ctx);
void pv_retire_end(pv_ctx *ctx);
int pv_load_end(pv_ctx *ctx);
// Evaluation calls order their stream after the last load (pv_use_begin)
// and mark their use of the loaded state (pv_mark_use).
void pv_use_begin(pv_ctx *ctx, cudaStream_t st);
void pv_mark_use(pv_ctx *ctx, cudaStream_t st);
int pv_check_launch(pv_ctx *ctx, const char *what);
// Raises a kernel's dynamic shared-memory limit to the device maximum (less
// the kernel's static shared memory), once
// per (device, kernel).  The limit is a process-wide permission, not a
// reservation (occupancy follows each launch's own size), so one setting at
// the maximum serves every launch, and no thread lowers it between another
// thread's setting and launch; later calls only look the pair up.
int pv_smem_limit(pv_ctx *ctx, const void *fn, const char *what);
// Resident blocks per SM of fn at this block size and dynamic shared memory
// (0 when the query fails), cached in the context.
int pv_blocks_per_sm(pv_ctx *ctx, const void *fn, int threads, size_t smem);
// Kernel-group timing: no-ops unless profiling is enabled.  Returns the pair
// index to pass to pv_prof_stop (or -1).
int pv_prof_start(pv_ctx *ctx, cudaStream_t st, int group);
void pv_prof_stop(pv_ctx *ctx, cudaStream_t st, int pair, uint32_t launches);

#define PV_TRY_CUDA(ctx, call, what)                          \
    do {                                                      \
        cudaError_t _e = (call);                              \
        if (_e != cudaSuccess) return pv_cuda_fail(ctx, _e, what); \
    } while (0)

// -----------------------------------------------------------------------------
// device helpers
// -----------------------------------------------------------------------------
// Records the first device-detected error code in the context status word.
__device__ __forceinline__ void pv_device_error(int32_t *status, int32_t code) {
    atomicCAS(status, 0, code);
}

__host__ __device__ __forceinline__ uint32_t pv_div_up(uint32_t a, uint32_t b) { return (a + b - 1) / b; }

// Prefix mask with the top `len` bits set; len in 0..32 (len 0 -> 0, never a
// shift by 32).
__host__ __device__ __forceinline__ uint32_t pv_prefix_mask(uint32_t len) {
    return len == 0 ? 0u : (0xFFFFFFFFu << (32u - len));
}

// Releases loaded-state memory in the load stream's order.
template <typename T>
inline void pv_free_ptr(pv_ctx *ctx, T *&p) {
    if (p) pv_pool_free(ctx, (void *)p);
    p = nullptr;
}

void pv_free_cluster(pv_ctx *ctx, pv_cluster_state &c);
void pv_free_tables(pv_ctx *ctx, pv_table_state &t);
// Frees a two-part table load that was begun and not ended (pv_destroy).
void pv_discard_table_load(pv_ctx *ctx);
void pv_free_policies(pv_ctx *ctx, pv_policy_state &p);
