/*
 * pv.h -- C ABI of the GB300 privacy-intent validator library (libpv.so).
 *
 * The library checks, in batches on one GPU, whether a deployed
 * configuration C = <sigma, rho> satisfies compiled privacy intents
 * (Sec. 3.3, "Formal Model and Satisfaction"): (i) pod placements sigma
 * against Kubernetes node selectors over the node labels lambda_N, and
 * (ii) the realised paths of ONOS-style flow rules against per-flow
 * permitted-jurisdiction sets over the switch labels lambda_V.  It also
 * answers jurisdiction-masked reachability over the topology G = (V, E).
 *
 * Conventions shared by every call
 * --------------------------------
 *  - Return value: PV_OK (0) or a PV_E* code; pv_last_error() gives a
 *    message.  Nothing throws across the ABI.
 *  - Ownership: a pv_ctx owns all state loaded by pv_load_* (copied from
 *    HOST pointers into library-owned device memory) and a scratch arena
 *    that grows on demand.  Evaluation calls take CALLER-OWNED DEVICE
 *    pointers and a CUDA stream (NULL = legacy default stream); they only
 *    enqueue work and return before it completes.
 *  - Device-detected errors (malformed device-resident inputs, a bounded
 *    wait that gave up) are recorded in a device status word and returned
 *    by the next pv_sync() on that context.  Device kernels never read or
 *    write out of bounds on malformed inputs.
 *  - Bitsets: item i is bit (i & 31) of 32-bit word (i >> 5) (LSB first);
 *    rows hold words_per_row words, words_per_row >= ceil(n / 32) and a
 *    multiple of 4 (rows are 16-byte aligned); padding bits are written 0.
 *  - A context is not thread-safe; use one context per host thread.
 */
#ifndef PV_H
#define PV_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct CUstream_st *pv_stream; /* same type as cudaStream_t */
typedef struct pv_ctx pv_ctx;

enum {
    PV_OK = 0,
    PV_EINVAL = 1,    /* argument or input out of range / malformed      */
    PV_ENOMEM = 2,    /* device or host allocation failed                */
    PV_ECUDA = 3,     /* a CUDA runtime call failed                      */
    PV_ESTATE = 4,    /* required pv_load_* has not been called          */
    PV_ETIMEOUT = 5,  /* a bounded device-side wait gave up              */
    PV_ENOTIMPL = 6
};

/* label / selector encodings (Sec. 3.3 label functions; Sec. 4.1) */
#define PV_ABSENT 0xFFFFu          /* node does not carry the key           */
enum { PV_IN = 0, PV_NOTIN = 1, PV_EXISTS = 2, PV_DOESNOTEXIST = 3 };

/* flow-rule / topology encodings (Sec. 4.2 per-hop flow rules) */
#define PV_ANY_PORT 0xFFFFu        /* rule.in_port wildcard                 */
#define PV_DROP 0xFFFFu            /* rule.action: drop                     */
#define PV_NO_HOST 0xFFFFu         /* probe.src_host: no source host        */
#define PV_PEER_NONE (-1)          /* port_peer: unconnected port           */
#define PV_PEER_HOST 0x40000000    /* port_peer: PV_PEER_HOST | host id     */
#define PV_UNPLACED 0xFFFFFFFFu    /* assign[]: pod has no feasible node    */

/* limits */
#define PV_MAX_PORTS 256           /* ports per switch (port ids 0..255)    */
#define PV_MAX_RULES 8192          /* rules per switch                      */
#define PV_MAX_SWITCHES 65535
#define PV_MAX_HOSTS 65535
#define PV_MAX_HOP_CAP 255

/* probe walk statuses */
enum {
    PV_COMPLIANT = 0,     /* delivered to the destination host, every switch permitted */
    PV_VIOLATION = 1,     /* visited a switch whose region is not permitted             */
    PV_DROPPED = 2,       /* table miss, drop action, or unconnected output port       */
    PV_LOOP = 3,          /* not terminated within hop_cap switch visits                */
    PV_MISDELIVERED = 4,  /* delivered to a host that does not own dst_ip               */
    PV_NOSRC = 5          /* src_host is PV_NO_HOST or out of range                      */
};

/* per-pod selector flags */
enum {
    PV_F_ASSIGN_OK = 1,      /* assign[p] < num_nodes and that node is feasible          */
    PV_F_EMPTY = 2,          /* no feasible node: the intent is unenforceable, fail closed */
    PV_F_UNKNOWN_VALUE = 4,  /* an In value is carried by no node (hallucinated id)       */
    PV_F_PASS = 8,           /* placement check passes: ASSIGN_OK and not UNKNOWN_VALUE   */
    PV_F_BAD_EXPR = 16       /* malformed expression list: row empty, check fails         */
};

typedef struct {           /* one matchExpression, 20 bytes                             */
    uint16_t key;          /* label key id < num_keys                                     */
    uint8_t op;            /* PV_IN, PV_NOTIN, PV_EXISTS, PV_DOESNOTEXIST                 */
    uint8_t nvals;         /* 1..8 for In/NotIn, 0 for Exists/DoesNotExist                */
    uint16_t vals[8];      /* value ids (not PV_ABSENT); entries >= nvals are ignored    */
} pv_expr;

typedef struct {           /* one flow rule, 20 bytes                                    */
    uint16_t priority;     /* higher wins; ties go to the lower input index               */
    uint16_t in_port;      /* port id or PV_ANY_PORT                                      */
    uint32_t src_ip, dst_ip;  /* prefix values; bits beyond the length are ignored       */
    uint8_t src_len, dst_len; /* prefix lengths 0..32 (0 matches everything)             */
    uint16_t dport_lo, dport_hi; /* inclusive destination-port range, lo <= hi          */
    uint16_t action;       /* output port id or PV_DROP                                   */
} pv_rule;

typedef struct {           /* one probe packet, 16 bytes                                 */
    uint32_t src_ip, dst_ip;
    uint16_t dport;
    uint16_t src_host;     /* injecting host id, or PV_NO_HOST                            */
    uint32_t allowed_mask; /* bit r set = switches of region r are permitted              */
} pv_probe;

typedef struct {           /* one walk result, 4 bytes                                   */
    uint8_t status;        /* PV_COMPLIANT .. PV_NOSRC                                    */
    uint8_t hops;          /* switch visits made (hop_cap for PV_LOOP, 0 for PV_NOSRC)   */
    uint16_t last_switch;  /* last switch visited (0xFFFF for PV_NOSRC)                   */
} pv_result;
typedef struct {           /* one flow of an intent, 8 bytes                             */
    uint32_t dst_ip;       /* destination address                                        */
    uint16_t dport;        /* destination port                                           */
    uint16_t reserved;     /* 0                                                          */
} pv_flow;
typedef struct {           /* one path request of the scheduler, 16 bytes                */
    uint16_t src_host;     /* source host id                                             */
    uint16_t dst_host;     /* destination host id                                        */
    uint32_t allowed_mask; /* permitted regions (bit r = region r)                       */
    uint32_t policy;       /* path policy index (>= loaded policies: none)               */
    uint32_t reserved;     /* 0                                                          */
} pv_path_req;
enum { PV_PATH_OK = 0, PV_PATH_NOSRC = 1, PV_PATH_BLOCKED = 2, PV_PATH_TOO_LONG = 3, PV_PATH_REPEAT = 4 };

/* ---------------------------------------------------------------------------
 * Context.
 * pv_create: binds the context to CUDA device `cuda_device` (the device must
 * be current on the calling thread for every later call).  Returns PV_ECUDA
 * if the device cannot be used.  pv_destroy frees all device state; it
 * accepts NULL.  pv_sync waits for `stream` and returns (and clears) the
 * first device-detected error since the previous pv_sync.
 * ------------------------------------------------------------------------- */
int pv_create(pv_ctx **out, int cuda_device);
void pv_destroy(pv_ctx *ctx);
const char *pv_last_error(const pv_ctx *ctx);
int pv_sync(pv_ctx *ctx, pv_stream stream);
int pv_version(void);

/* ---------------------------------------------------------------------------
 * pv_load_cluster -- the node label function lambda_N (Sec. 3.3; label
 * schema of Sec. 5.2, e.g. location, provider, security-level, zone).
 *
 * labels: HOST pointer, key-major (structure of arrays):
 *   labels[k * num_nodes + n] = value id of key k on node n, or PV_ABSENT.
 * Copied to the device; the library also builds the per-key inventory of
 * carried values (for the hallucinated-identifier check of Sec. 6.3) and,
 * when it fits its memory budget, per-(key, value) node bitsets.
 * Errors: PV_EINVAL if num_nodes == 0, num_keys == 0 or num_keys > 4096;
 * PV_ENOMEM.  Replaces any previously loaded cluster.
 * ------------------------------------------------------------------------- */
int pv_load_cluster(pv_ctx *ctx, uint32_t num_nodes, uint32_t num_keys, const uint16_t *labels);

/* ---------------------------------------------------------------------------
 * pv_eval_selectors -- placement constraints Phi_C (Sec. 3.3 satisfaction
 * (i) and worked example; Sec. 4.1 placement directives; Sec. 5.5 compute
 * check "a pod is scheduled only onto nodes whose labels satisfy the
 * placement constraints").
 *
 * For pod p, feasible(p) = { n : every expression of p matches node n },
 * with Kubernetes matchExpressions semantics (In: key carried and value in
 * set; NotIn: key absent or value not in set; Exists; DoesNotExist).  An
 * empty expression list admits every node.
 *
 * Device inputs: d_expr_offs[num_pods + 1] (CSR offsets into d_exprs,
 * num_exprs entries, 4-byte aligned), d_assign[num_pods] or NULL (the
 * placement sigma).  Device outputs: d_bits[num_pods][words_per_row]
 * (16-byte aligned) feasible-node bitsets; d_flags[num_pods] PV_F_* bits
 * (ASSIGN_OK and PASS need d_assign).
 * Malformed expression lists (offsets decreasing or beyond num_exprs, key
 * >= num_keys, unknown op, bad nvals, PV_ABSENT as a value) give an empty
 * row and PV_F_BAD_EXPR for that pod; they are not call errors.
 * Errors: PV_ESTATE (no cluster), PV_EINVAL (words_per_row too small or
 * not a multiple of 4, NULL or misaligned pointers with num_pods > 0).
 * ------------------------------------------------------------------------- */
int pv_eval_selectors(pv_ctx *ctx, uint32_t num_pods, const uint32_t *d_expr_offs, uint32_t num_exprs,
                      const pv_expr *d_exprs, const uint32_t *d_assign, uint32_t *d_bits,
                      uint32_t words_per_row, uint8_t *d_flags, pv_stream stream);

/* ---------------------------------------------------------------------------
 * pv_eval_selector_terms -- the node-affinity form of placement constraints
 * (Sec. 3.3 and Sec. 4.1: node selectors / affinities): Kubernetes required
 * node affinity, a list of selector terms that are ORed, each term a list of
 * expressions that are ANDed (the same pv_expr semantics as above):
 *     feasible(p) = union over p's terms t of { n : every expression of t
 *                   matches node n }.
 * A pod with no terms admits every node; a term with no expressions matches
 * no node (Kubernetes: an empty selector term matches nothing).
 *
 * Device inputs: d_pod_terms[num_pods + 1] (CSR: pod p's terms are
 * pod_terms[p] .. pod_terms[p+1]), d_term_offs[num_terms + 1] (CSR into
 * d_exprs), d_exprs[num_exprs], d_assign[num_pods] or NULL.  Outputs and
 * flags as pv_eval_selectors; an In value carried by no node in any term
 * sets PV_F_UNKNOWN_VALUE; a malformed term range or expression gives an
 * empty row and PV_F_BAD_EXPR.  Needs the per-(key, value) rows
 * (PV_STAT_SELECTOR_ROWS_BUILT).
 * Errors: PV_ESTATE (no cluster), PV_EINVAL (words_per_row, alignment, NULL
 * pointers, rows not built).
 * ------------------------------------------------------------------------- */
int pv_eval_selector_terms(pv_ctx *ctx, uint32_t num_pods, const uint32_t *d_pod_terms, uint32_t num_terms,
                           const uint32_t *d_term_offs, uint32_t num_exprs, const pv_expr *d_exprs,
                           const uint32_t *d_assign, uint32_t *d_bits, uint32_t words_per_row, uint8_t *d_flags,
                           pv_stream stream);

/* ---------------------------------------------------------------------------
 * pv_load_flow_tables -- the installed per-hop flow rules rho (Sec. 4.2
 * flow scheduling module; each path becomes per-hop rules pushed to ONOS)
 * and the switch labels lambda_V reduced to a region id per switch
 * (Sec. 5.2 label schema, device_labels.location).
 *
 * HOST inputs:
 *   rule_offs[num_switches + 1], rules[rule_offs[num_switches]]: switch s
 *     owns rules[rule_offs[s] .. rule_offs[s+1]) in input order;
 *   switch_region[num_switches]: region id < 32;
 *   port_offs[num_switches + 1], port_peer[port_offs[num_switches]]: port p
 *     of switch s (p < port_offs[s+1]-port_offs[s] <= PV_MAX_PORTS) leads to
 *     PV_PEER_NONE, PV_PEER_HOST | h, or the switch port (s2 << 8) | p2;
 *   host_switch[num_hosts], host_port[num_hosts]: attachment of host h;
 *   host_ip[num_hosts]: the address host h owns.
 * The library sorts each switch's rules by (priority desc, input index asc)
 * on the device and compiles them for the walk kernels.
 * Errors: PV_EINVAL for any out-of-range field (in_port / action >= the
 * switch's port count unless wildcard/drop, prefix length > 32, lo > hi,
 * region >= 32, offsets not monotone, more than PV_MAX_RULES rules or
 * PV_MAX_PORTS ports on a switch, peers out of range); PV_ENOMEM.
 * Replaces any previously loaded tables.
 * ------------------------------------------------------------------------- */
int pv_load_flow_tables(pv_ctx *ctx, uint32_t num_switches, const uint32_t *rule_offs, const pv_rule *rules,
                        const uint8_t *switch_region, const uint32_t *port_offs, const int32_t *port_peer,
                        uint32_t num_hosts, const uint16_t *host_switch, const uint16_t *host_port,
                        const uint32_t *host_ip);

/* ---------------------------------------------------------------------------
 * pv_load_flow_tables_begin / pv_load_flow_tables_end -- pv_load_flow_tables
 * in two halves, so that a caller can queue its own transfers between them.
 * begin takes the same arguments and does the host checks (the same errors),
 * queues every upload of the tables and the first device passes on the
 * context's load stream, and returns without waiting for the device.  end
 * waits for those passes, reports the device-side rule errors (PV_EINVAL,
 * as pv_load_flow_tables), builds the index and installs the tables.
 * Between the two:
 *   - every host array given to begin stays allocated and unchanged (end
 *     reads them again);
 *   - evaluation calls keep using the tables installed before begin, and
 *     the other loads work as usual;
 *   - a second begin, pv_load_flow_tables or pv_install_path_rules (which
 *     loads tables) fails with PV_ESTATE.
 * end without a begin fails with PV_ESTATE.  If begin fails nothing is in
 * progress; if end fails the previous tables stay installed.  pv_destroy
 * frees a load that was begun and not ended.
 * ------------------------------------------------------------------------- */
int pv_load_flow_tables_begin(pv_ctx *ctx, uint32_t num_switches, const uint32_t *rule_offs, const pv_rule *rules,
                              const uint8_t *switch_region, const uint32_t *port_offs, const int32_t *port_peer,
                              uint32_t num_hosts, const uint16_t *host_switch, const uint16_t *host_port,
                              const uint32_t *host_ip);
int pv_load_flow_tables_end(pv_ctx *ctx);

/* ---------------------------------------------------------------------------
 * pv_verify_probes -- routing constraints Phi_N on the realised paths
 * (Sec. 3.3 satisfaction (ii): "for all v on the path"; Sec. 5.5 network
 * check; Sec. 6.3 item 4: transit switches are checked hop by hop).
 *
 * Each probe starts at (host_switch[src_host], host_port[src_host]); at each
 * visited switch s: (1) region(s) not in allowed_mask -> PV_VIOLATION;
 * (2) first matching rule by priority (no match or drop -> PV_DROPPED);
 * (3) the output port's peer: unconnected -> PV_DROPPED, a host ->
 * PV_COMPLIANT if it owns dst_ip else PV_MISDELIVERED, a switch port ->
 * next hop.  Not terminated within hop_cap visits -> PV_LOOP.
 *
 * Device input d_probes[num_probes] (16-byte aligned); device output
 * d_out[num_probes] (4-byte aligned; every walk call writes each result as
 * one 32-bit word).
 * Errors: PV_ESTATE (no tables), PV_EINVAL (hop_cap 0 or > 255, NULL or
 * misaligned pointers with num_probes > 0).  Out-of-range src_host gives
 * PV_NOSRC.
 * ------------------------------------------------------------------------- */
int pv_verify_probes(pv_ctx *ctx, uint32_t num_probes, const pv_probe *d_probes, uint32_t hop_cap,
                     pv_result *d_out, pv_stream stream);

/* ---------------------------------------------------------------------------
 * pv_compliant_reach -- jurisdiction-masked reachability over G = (V, E)
 * (Sec. 3.3 forbidden-vertex policy; Sec. 4.2 graph search over the current
 * topology).  R(s, m) = { v : some path s -> v has every vertex, s included,
 * in a region permitted by m }; empty when region(s) is not permitted.
 *
 * Device inputs: d_offs[V + 1], d_cols[num_edges] (CSR of directed edges
 * u -> v: the out-neighbours of u are d_cols[d_offs[u] .. d_offs[u+1])),
 * d_region[V] (< 32), d_src[num_src] (vertex ids), d_masks[num_masks].
 * Device output: d_reach[num_masks][num_src][words_per_row] bitsets over V.
 * Malformed inputs are reported as PV_EINVAL by the next pv_sync() and never
 * cause an access outside the arrays above: malformed offsets (some row
 * with d_offs[u+1] < d_offs[u] or d_offs[u+1] > num_edges) make the graph
 * count as having no edges at all (so R(s, m) = {s} for a permitted s); an
 * edge with cols >= V is skipped; a vertex with region >= 32 is in no
 * permitted set.  Out-of-range sources give empty rows.  When every remaining edge has its reverse (and
 * no vertex has more than 64 out-edges) the rows are taken from the
 * connected components of the permitted subgraph, which on such a graph is
 * the same set (PV_OPT_REACH_KERNEL).  The call enqueues on `stream`; with
 * the component path enabled, the other path's kernels (which return at
 * once on a symmetric graph) run on a side stream of the context that
 * `stream` waits for before the call returns (created on the first call).
 * Errors: PV_EINVAL (V == 0, V > 16384, words_per_row too small or not a
 * multiple of 4, NULL pointers); PV_ENOMEM (scratch).
 * ------------------------------------------------------------------------- */
int pv_compliant_reach(pv_ctx *ctx, uint32_t V, const uint32_t *d_offs, uint32_t num_edges,
                       const uint32_t *d_cols, const uint8_t *d_region, uint32_t num_src, const uint32_t *d_src, uint32_t num_masks,
                       const uint32_t *d_masks, uint32_t *d_reach, uint32_t words_per_row, pv_stream stream);

/* ---------------------------------------------------------------------------
 * pv_compliant_reach_noalloc -- the same computation and output as
 * pv_compliant_reach, for callers that cannot allocate device memory: a
 * program whose device memory belongs to another framework's pool or is held
 * to a fixed budget, or a latency-critical caller that cannot absorb the
 * device-wide synchronisation cudaMalloc / cudaFree may imply.  (The paper
 * has no counterpart; this is a property of the library, not of the method.)
 *
 * It needs no pv_ctx and allocates nothing: its working memory (a status
 * word and the in-edge CSR) is one static device array of about 1.2 MB that
 * every GPU which loads the library holds until the process exits.  Limits:
 * V <= 16384 and num_edges <= 262144; larger inputs return PV_EINVAL before
 * any work is queued.  Arguments, layouts and the result are those of
 * pv_compliant_reach; the call runs on `stream` on the current device.
 * The first call on a device looks up the array's device address (no
 * allocation); make that first call before any stream capture.
 * All calls share the one array and each call overwrites it, so calls whose
 * work overlaps on the GPU (different streams, or host threads without
 * ordering) race; order them on one stream.  The address looked up on a
 * device's first call is kept for the life of the process, so the library
 * must not be used on a device after cudaDeviceReset.  Malformed inputs get
 * the rows pv_compliant_reach gives them (malformed offsets: no edges;
 * columns >= V skipped), but no error is reported for them here.
 * Returns PV_OK, PV_EINVAL (limits, NULL or misaligned pointers) or
 * PV_ECUDA.
 * ------------------------------------------------------------------------- */
int pv_compliant_reach_noalloc(uint32_t V, const uint32_t *d_offs, uint32_t num_edges, const uint32_t *d_cols,
                               const uint8_t *d_region, uint32_t num_src, const uint32_t *d_src,
                               uint32_t num_masks, const uint32_t *d_masks, uint32_t *d_reach,
                               uint32_t words_per_row, pv_stream stream);

/* ---------------------------------------------------------------------------
 * End-to-end composition (Sec. 4.2 hybrid coordination: pods are placed
 * first, then flows from their attachments are checked; Sec. 5.5: an intent
 * passes only if all of its checks pass).  A "group" is one intent: one
 * selector row, pods_per_group pods, probes_per_group probes.  Cluster node
 * n is network host n.
 *
 * pv_place_pods: pod j of group g gets the r-th feasible node of row g in
 *   ascending order, r = d_draws[g * pods_per_group + j] mod |feasible|, or
 *   PV_UNPLACED if the row is empty.  d_assign[num_groups * pods_per_group].
 * pv_bind_probes: probe k of group g = k / probes_per_group is sent from
 *   the host of pod (k mod probes_per_group) mod pods_per_group of g:
 *   src_host and src_ip are rewritten in place (PV_NO_HOST / 0 when that pod
 *   is unplaced or not a host).  Needs the flow tables (host_ip).
 * pv_bind_flows: the same binding from the compact form of an intent's
 *   flows: d_flows[k] = {dst_ip, dport} and the group's jurisdiction mask
 *   d_group_mask[g] give the whole probe record d_probes[k] (16-byte
 *   aligned), its source bound as above.
 * pv_verify_flows: pv_bind_flows followed by pv_verify_probes in one call,
 *   with the same results: the walk's first kernel binds each flow, writes
 *   its record to d_probes when d_probes is not NULL (NULL: the bound
 *   records are not returned), and starts its walk.  When every group has
 *   one path constraint (always for pv_verify_flows; for the constrained
 *   call, no d_probe_policy and probes_per_policy 0 or a multiple of
 *   probes_per_group), the probes of each (group, pod) pair, which share
 *   their first switch, are counted per switch from the pairs alone and
 *   written straight into the first hop's switch order, with a compact
 *   walk record in the library's scratch; otherwise the first hop is
 *   regrouped like any other.  pv_verify_flows_constrained is the same with
 *   the path constraints of pv_verify_probes_constrained.
 * pv_verify_flow_columns(_constrained): the same calls with the flows as two
 *   columns, d_dst_ip[k] (4-byte aligned) and d_dport[k] (2-byte aligned):
 *   6 bytes per flow instead of the 8 of a pv_flow record, which is what a
 *   caller uploading its flows from host memory pays for.  Same results.
 * pv_aggregate_intents: d_pass[g] = 1 iff every pod of g has d_assign in
 *   row g, d_group_flags[g] has neither PV_F_UNKNOWN_VALUE nor
 *   PV_F_BAD_EXPR, and every probe of g is PV_COMPLIANT.
 *   d_counts[g][8]: [0..5] probe status histogram, [6] pods placed on a
 *   feasible node, [7] zero.
 * Errors: PV_ESTATE, PV_EINVAL (zero group sizes, NULL pointers).
 * ------------------------------------------------------------------------- */
int pv_bind_flows(pv_ctx *ctx, uint32_t num_probes, const pv_flow *d_flows, uint32_t probes_per_group,
                  uint32_t pods_per_group, const uint32_t *d_assign, const uint32_t *d_group_mask,
                  pv_probe *d_probes, pv_stream stream);
int pv_verify_flows(pv_ctx *ctx, uint32_t num_probes, const pv_flow *d_flows, uint32_t probes_per_group,
                    uint32_t pods_per_group, const uint32_t *d_assign, const uint32_t *d_group_mask, uint32_t hop_cap,
                    pv_probe *d_probes, pv_result *d_out, pv_stream stream);
int pv_verify_flows_constrained(pv_ctx *ctx, uint32_t num_probes, const pv_flow *d_flows, uint32_t probes_per_group,
                                uint32_t pods_per_group, const uint32_t *d_assign, const uint32_t *d_group_mask,
                                uint32_t hop_cap, const uint32_t *d_probe_policy, uint32_t probes_per_policy,
                                uint32_t first_policy, pv_probe *d_probes, pv_result *d_out, uint32_t *d_waypoints,
                                pv_stream stream);
int pv_verify_flow_columns(pv_ctx *ctx, uint32_t num_probes, const uint32_t *d_dst_ip, const uint16_t *d_dport,
                           uint32_t probes_per_group, uint32_t pods_per_group, const uint32_t *d_assign,
                           const uint32_t *d_group_mask, uint32_t hop_cap, pv_probe *d_probes, pv_result *d_out,
                           pv_stream stream);
int pv_verify_flow_columns_constrained(pv_ctx *ctx, uint32_t num_probes, const uint32_t *d_dst_ip,
                                       const uint16_t *d_dport, uint32_t probes_per_group, uint32_t pods_per_group,
                                       const uint32_t *d_assign, const uint32_t *d_group_mask, uint32_t hop_cap,
                                       const uint32_t *d_probe_policy, uint32_t probes_per_policy,
                                       uint32_t first_policy, pv_probe *d_probes, pv_result *d_out,
                                       uint32_t *d_waypoints, pv_stream stream);
int pv_place_pods(pv_ctx *ctx, uint32_t num_groups, uint32_t pods_per_group, const uint32_t *d_bits,
                  uint32_t words_per_row, const uint64_t *d_draws, uint32_t *d_assign, pv_stream stream);
int pv_bind_probes(pv_ctx *ctx, uint32_t num_probes, pv_probe *d_probes, uint32_t probes_per_group,
                   uint32_t pods_per_group, const uint32_t *d_assign, pv_stream stream);
int pv_aggregate_intents(pv_ctx *ctx, uint32_t num_groups, uint32_t pods_per_group, const uint32_t *d_bits,
                         uint32_t words_per_row, const uint8_t *d_group_flags, const uint32_t *d_assign,
                         uint32_t probes_per_group, const pv_result *d_results, uint8_t *d_pass,
                         uint32_t *d_counts, pv_stream stream);

/* ---------------------------------------------------------------------------
 * Path constraints (Sec. 4.2: the constraint object the flow scheduler gets
 * lists forbidden switches and must_go switches; Sec. 5.3, networking
 * intent: the realised path must include the waypoint; Sec. 5.5: network
 * checks assert that realised paths avoid forbidden switches and include
 * required waypoints; Sec. 6.3, failure mode 2: a constraint without a
 * concrete src/dst applies to no flow, a no-op policy, and its intent is not
 * enforced).
 *
 * pv_load_path_policies: policy p forbids the switches
 *   forbid[forbid_offs[p] .. forbid_offs[p+1]) and requires the waypoints
 *   must[must_offs[p] .. must_offs[p+1]) (at most 32); concrete[p] != 0 when
 *   the constraint names at least one concrete (src, dst) flow.  HOST arrays,
 *   copied; offsets start at 0.  Needs the flow tables (switch ids < S).
 *   Replaces previously loaded policies.  Errors: PV_ESTATE, PV_EINVAL
 *   (decreasing offsets, > 32 waypoints, switch id out of range), PV_ENOMEM.
 * pv_verify_probes_constrained: pv_verify_probes with path constraints.
 *   Probe k follows policy d_probe_policy[k] (device, or NULL: policy
 *   first_policy + k / probes_per_policy, so a slice of a larger batch can
 *   keep its policies); an index >= num_policies means none.  A forbidden
 *   switch is judged like a switch outside the probe's jurisdictions
 *   (PV_VIOLATION there; the walk stops).  Device output d_waypoints[M]: bit
 *   i set iff the probe entered waypoint i of its policy (a switch it was
 *   refused does not count).  Errors: as pv_verify_probes; PV_ESTATE (no
 *   policies), PV_EINVAL (NULL d_waypoints).
 * pv_aggregate_constrained: pv_aggregate_intents plus, for group g with
 *   policy p = d_group_policy[g] (device, or NULL: p = first_policy + g;
 *   p >= num_policies: none): g fails unless concrete[p] and every probe of g has all of p's
 *   waypoint bits; d_counts[g][7] = probes of g that missed a waypoint.
 * ------------------------------------------------------------------------- */
int pv_load_path_policies(pv_ctx *ctx, uint32_t num_policies, const uint32_t *forbid_offs, const uint16_t *forbid,
                          const uint32_t *must_offs, const uint16_t *must, const uint8_t *concrete);
int pv_verify_probes_constrained(pv_ctx *ctx, uint32_t num_probes, const pv_probe *d_probes, uint32_t hop_cap,
                                 const uint32_t *d_probe_policy, uint32_t probes_per_policy, uint32_t first_policy,
                                 pv_result *d_out, uint32_t *d_waypoints, pv_stream stream);
int pv_aggregate_constrained(pv_ctx *ctx, uint32_t num_groups, uint32_t pods_per_group, const uint32_t *d_bits,
                             uint32_t words_per_row, const uint8_t *d_group_flags, const uint32_t *d_assign,
                             uint32_t probes_per_group, const pv_result *d_results, const uint32_t *d_waypoints,
                             const uint32_t *d_group_policy, uint32_t first_policy, uint8_t *d_pass,
                             uint32_t *d_counts, pv_stream stream);

/* ---------------------------------------------------------------------------
 * Path scheduling -- the enforcement side (Sec. 4.2: the flow scheduling
 * module computes paths respecting the constraint object with weighted
 * Dijkstra, breadth-first when no weights are given, and turns each path
 * into per-hop flow rules).
 *
 * pv_schedule_paths: request r asks for a path from host src_host to host
 *   dst_host over switches whose region allowed_mask permits and that its
 *   policy (pv_load_path_policies; none when the index is out of range or no
 *   policies are loaded) does not forbid, through the policy's waypoints in
 *   their listed order.  The path is the concatenation of shortest segments
 *   src switch -> waypoint 1 -> ... -> dst switch; link u --port p--> costs
 *   d_link_weights[port_offs[u] + p] (device, 0 counts as 1; NULL: 1 each).
 *   A segment is made canonical by walking back from its end and taking, at
 *   every switch, the predecessor link with the smallest source switch, then
 *   the smallest source port, among those on a shortest path.  Device
 *   outputs: d_visits[r][max_len] = switch << 16 | in_port << 8 | out_port
 *   for the d_len[r] visits (in_port of the first = the source host's port,
 *   out_port of the last = the destination host's port), d_status[r] =
 *   PV_PATH_OK, NOSRC (a host id out of range), BLOCKED (an endpoint or
 *   waypoint not permitted, or no path), TOO_LONG (more than max_len visits),
 *   REPEAT (a (switch, in_port) pair recurs: rules matching header and
 *   in_port cannot realise it).  Needs <= 16,384 switches.
 * pv_compile_path_rules: visit i of an OK request becomes, at its switch,
 *   the rule {priority, in_port, src /32, dst /32, ports 0..65535, out_port}
 *   in d_rules[r * max_len + i], d_rule_switch[...] = its switch (0xFFFF for
 *   unused slots).
 * pv_install_path_rules: adds the compiled rules ahead of each switch's
 *   loaded rules (they win priority ties) and reloads the tables
 *   (synchronous, like pv_load_flow_tables; slots with switch 0xFFFF or out
 *   of range are skipped).
 * Errors: PV_ESTATE (no tables), PV_EINVAL (max_len not 1..255, NULL
 * pointers, too many switches), PV_ENOMEM.
 * ------------------------------------------------------------------------- */
int pv_schedule_paths(pv_ctx *ctx, uint32_t num_requests, const pv_path_req *d_requests,
                      const uint16_t *d_link_weights, uint32_t max_len, uint32_t *d_visits, uint8_t *d_len,
                      uint8_t *d_status, pv_stream stream);
int pv_compile_path_rules(pv_ctx *ctx, uint32_t num_requests, const pv_path_req *d_requests, uint32_t max_len,
                          const uint32_t *d_visits, const uint8_t *d_len, const uint8_t *d_status,
                          uint16_t priority, pv_rule *d_rules, uint16_t *d_rule_switch, pv_stream stream);
int pv_install_path_rules(pv_ctx *ctx, uint32_t num_slots, const pv_rule *d_rules, const uint16_t *d_rule_switch);

/* ---------------------------------------------------------------------------
 * Tuning knobs (no counterpart in the paper).
 * PV_OPT_SELECTOR_KERNEL: 0 = automatic, 1 = per-node label comparison over
 *   shared-memory label tiles, 2 = per-(key, value) node-bitset rows
 *   (needs the rows to have been built by pv_load_cluster).
 * PV_OPT_SELECTOR_DEDUPE: 0 (default) or 1 = pv_eval_selectors evaluates
 *   each distinct expression list once: pods whose lists are equal (the
 *   same expressions in the same order, unused value slots ignored), such as
 *   the replicas of one deployment or intents sharing a selector, get their
 *   representative's row (the smallest such pod) and flags, with their own
 *   placement check.  Same results; pays off when lists repeat.  2 = the
 *   same with deliberately weak hashes (tests: every collision is resolved
 *   by comparing the lists).  Not used by pv_eval_selector_terms.
 * PV_OPT_SCHED_KERNEL: pv_schedule_paths' kernel (one block per request):
 *   0 = automatic (the links into each switch, with their weights, staged
 *   in shared memory when they fit, else read from global memory); 1 =
 *   links from global memory; 2 = staged (PV_EINVAL if they do not fit).
 *   Both give the same paths.
 * PV_OPT_WALK_KERNEL: 0 = automatic, 1 = linear first-match scan of the
 *   staged table, 2 = indexed first match (per-dport-bucket candidate lists
 *   and destination-interval maps built by pv_load_flow_tables; needs every
 *   switch's index to fit shared memory).
 * PV_OPT_WALK_LANE_MAX: with kernel 2, a batch of 32 probes is resolved one
 *   probe per lane when its longest candidate list has at most this many
 *   items (default 96), else one probe at a time by the whole warp.
 * PV_OPT_WALK_CYCLES: 0 (default) = a probe found back at a (switch,
 *   in_port) it already held is in a forwarding cycle (its header is fixed,
 *   so its walk repeats); it walks only to the cycle position of hop
 *   hop_cap - 1 and is finished there with the PV_LOOP result the full walk
 *   gives (checkpoints at hops 4, 8, 16, ...).  When every switch port's
 *   peer port leads back to it, a probe that leaves two switches in a row by
 *   the port it came in by (two bounces) is in a two-switch cycle and is
 *   finished at the second bounce.  1 = walk every hop to the cap.
 *   Both give the same results; PV_STAT_WALK_LIVE_TOTAL differs.
 * PV_OPT_WALK_TAIL_HOP: with the indexed kernel, the walk's hops from this
 *   one on (0 = none) run in a single launch, one thread per probe still
 *   walking, tables read from L2 instead of staged per switch.  Same
 *   results.  Default (-1): chosen by pv_load_flow_tables from the loaded
 *   index, hop 5 when its candidate lists hold at most 12 items per
 *   destination-port bucket on average, else hop 8.
 * PV_OPT_REACH_KERNEL: 0 = automatic (on a symmetric graph, rows are the
 *   connected components of the permitted subgraph; otherwise multi-source
 *   pull sweeps), 1 = sweeps always.  Both give the same rows.
 * PV_OPT_WALK_STATS: 0 (default) or 1 = walks run counting versions of the
 *   hop kernels (same results, slower: a diagnostic, not a timed path).
 *   For every first match they also scan the switch's compiled rules in
 *   first-match order and record, for the walk: first matches resolved,
 *   index rule tests (candidate rules whose match was evaluated; the linear
 *   kernel evaluates 32 per step), interval lookups (destination-only rule
 *   runs answered by interval search), the scan depth (rules the ordered
 *   scan tests before its first hit, every rule of the switch on a miss), and
 *   index mismatches (first matches where the scan and the kernel disagree;
 *   0 unless the index is wrong).  Read them with pv_get_stat
 *   (PV_STAT_WALK_FIRST_MATCHES .. PV_STAT_WALK_INDEX_MISMATCHES; each read
 *   synchronises with the device).
 * PV_OPT_TEST_STALL_STAGING: failure-injection switch for tests (0 or 1).
 *   When 1, each hop block's table-staging barrier expects 16 bytes more
 *   than its copy delivers, so its bounded wait runs out (after 50 ms rather
 *   than the normal 2 s); the walk then reports PV_ETIMEOUT through pv_sync
 *   and the context stays usable.  Never set it outside a test.
 * pv_get_stat: PV_STAT_SELECTOR_ROWS_BUILT (1 if value rows exist),
 *   PV_STAT_SCRATCH_BYTES, PV_STAT_WALK_INDEX_FITS (1 if kernel 2 is
 *   usable), PV_STAT_WALK_INDEX_BYTES (largest shared-memory
 *   stage of an indexed table: header, plain rules and index),
 *   PV_STAT_WALK_LIVE_TOTAL (probe-hop entries the last pv_verify_probes
 *   processed: the sum over its hops of the probes still walking; reading it
 *   synchronises with the device), PV_STAT_REACH_COMPONENTS (1 if the last
 *   pv_compliant_reach found its graph symmetric and wrote the rows from
 *   components; synchronises).
 * ------------------------------------------------------------------------- */
enum {
    PV_OPT_SELECTOR_KERNEL = 1, PV_OPT_WALK_KERNEL = 2, PV_OPT_WALK_LANE_MAX = 3, PV_OPT_TEST_STALL_STAGING = 4,
    PV_OPT_REACH_KERNEL = 5, PV_OPT_WALK_CYCLES = 6, PV_OPT_WALK_TAIL_HOP = 7, PV_OPT_WALK_STATS = 8,
    PV_OPT_SELECTOR_DEDUPE = 9, PV_OPT_SCHED_KERNEL = 10
};
enum {
    PV_STAT_SELECTOR_ROWS_BUILT = 1, PV_STAT_SCRATCH_BYTES = 2, PV_STAT_WALK_INDEX_FITS = 3,
    PV_STAT_WALK_INDEX_BYTES = 4, PV_STAT_WALK_LIVE_TOTAL = 5, PV_STAT_REACH_COMPONENTS = 6,
    PV_STAT_WALK_FIRST_MATCHES = 7, PV_STAT_WALK_RULE_TESTS = 8, PV_STAT_WALK_INTERVAL_LOOKUPS = 9,
    PV_STAT_WALK_SCAN_DEPTH = 10, PV_STAT_WALK_INDEX_MISMATCHES = 11
};
int pv_set_option(pv_ctx *ctx, int option, int64_t value);
int pv_get_stat(const pv_ctx *ctx, int stat, int64_t *value);

/* ---------------------------------------------------------------------------
 * Kernel timing (no counterpart in the paper).  While enabled, every kernel
 * group the library launches is bracketed by CUDA events recorded on the
 * caller's stream.  pv_profile_enable(ctx, 1) clears the totals and starts
 * recording, (ctx, 0) stops; pv_profile_collect synchronises `stream` and
 * folds the recorded event pairs into per-group totals; pv_profile_read
 * returns a group's total device milliseconds and number of kernel
 * launches.  Groups: PV_K_* below (REGROUP = histogram + scan + scatter).
 * ------------------------------------------------------------------------- */
enum {
    PV_K_SELECTOR = 0, PV_K_PLACE = 1, PV_K_BIND = 2, PV_K_WALK_INIT = 3, PV_K_WALK_REGROUP = 4,
    PV_K_WALK_HOP = 5, PV_K_AGGREGATE = 6, PV_K_REACH = 7, PV_K_SCHEDULE = 8, PV_K_COUNT = 9
};
int pv_profile_enable(pv_ctx *ctx, int on);
int pv_profile_collect(pv_ctx *ctx, pv_stream stream);
int pv_profile_read(const pv_ctx *ctx, int group, double *total_ms, uint64_t *launches);

#ifdef __cplusplus
}
#endif
#endif /* PV_H */
