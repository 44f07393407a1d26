/*
 * Plain, slow, single-threaded CPU oracle of the cross-layer privacy
 * validator.  TEST INFRASTRUCTURE ONLY: the test suite, the package's smoke
 * check and the benchmark's CPU-baseline leg may call it; the product path
 * never does.  It shares no code, header or table with the CUDA library.
 *
 * Every function computes a plain definition directly, in the order the
 * paper states it:
 *
 *  - Satisfaction C |=_lambda I (Sec. 3.3, "Formal Model and Satisfaction"):
 *    (i) placement constraints hold for sigma under lambda_N, (ii) routing
 *    constraints hold on the realised paths under lambda_V.
 *  - Placement constraints are Kubernetes node selectors / affinities
 *    (Sec. 3.3 worked example; Sec. 4.1 "Placement Directives"): the
 *    matchExpressions operators In, NotIn, Exists, DoesNotExist, ANDed
 *    within one pod (or within one selector term, the terms ORed, for the
 *    node-affinity form).  An equality nodeSelector is In with one value.
 *  - Hallucinated identifiers (Sec. 6.3, failure mode 3): a value referenced
 *    by an In expression that no node carries fails the check.
 *  - Unenforceable intents fail closed (Sec. 5.3, intent examples table): a
 *    selector with no feasible node fails.
 *  - Realised paths are the hop-by-hop walk of OpenFlow/ONOS first-match-
 *    by-priority flow rules (Sec. 4.2, flow scheduling module and per-hop
 *    rules); every traversed vertex must carry a permitted jurisdiction
 *    (Sec. 3.3 example "for all v on the path"; Sec. 6.3 failure mode 4:
 *    transit switches are checked, not just endpoints).
 *  - Compliant reach: the set of vertices reachable from a source over
 *    vertices whose region is permitted (Sec. 3.3 forbidden-vertex policy
 *    over G = (V, E); Sec. 4.2 graph search over the topology).
 *  - Path constraints (Sec. 4.2 constraint object; Sec. 5.3 waypoint
 *    intent; Sec. 5.5 network checks): forbidden switches are judged like
 *    forbidden jurisdictions, required waypoints must be on the path; a
 *    constraint naming no concrete flow is a no-op policy and fails
 *    (Sec. 6.3, failure mode 2).
 *  - An intent passes only if all its checks pass (Sec. 5.5, validator
 *    check definition).
 *
 * Readings where the paper is silent (operator set, absent labels, priority
 * direction, ties, table miss, loop definition, statuses) are documented
 * beside each function.
 *
 * Parity pins: selectors against a string-keyed brute force and the paper's
 * 5-worker label table; first-match against a sort-then-scan formulation and
 * hand cases; walks against hand-built topologies, a recursive path trace
 * and path invariants; constrained walks against a path recorded without
 * constraints and judged afterwards, and a hand-built waypoint case; reach
 * against simple-path enumeration, union-find
 * components and monotonicity/symmetry; placement/aggregation by
 * composition and invariants.
 */
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#define OR_ABSENT 0xFFFFu
#define OR_OP_IN 0
#define OR_OP_NOTIN 1
#define OR_OP_EXISTS 2
#define OR_OP_DOESNOTEXIST 3
#define OR_ANY_PORT 0xFFFFu
#define OR_DROP 0xFFFFu
#define OR_NO_HOST 0xFFFFu
#define OR_PEER_NONE (-1)
#define OR_HOST_BIT (1 << 30)
#define OR_UNPLACED 0xFFFFFFFFu

enum { OR_COMPLIANT = 0, OR_VIOLATION = 1, OR_DROPPED = 2, OR_LOOP = 3, OR_MISDELIVERED = 4, OR_NOSRC = 5 };
enum { OR_F_ASSIGN_OK = 1, OR_F_EMPTY = 2, OR_F_UNKNOWN = 4, OR_F_PASS = 8, OR_F_BAD = 16 };

typedef struct { uint16_t key; uint8_t op; uint8_t nvals; uint16_t vals[8]; } or_expr;
typedef struct {
    uint16_t priority, in_port;
    uint32_t src_ip, dst_ip;
    uint8_t src_len, dst_len;
    uint16_t dport_lo, dport_hi, action;
} or_rule;
typedef struct { uint32_t src_ip, dst_ip; uint16_t dport, src_host; uint32_t allowed_mask; } or_probe;
typedef struct { uint8_t status, hops; uint16_t last_switch; } or_result;

void oracle_struct_sizes(uint32_t *out) {
    out[0] = sizeof(or_expr);
    out[1] = sizeof(or_rule);
    out[2] = sizeof(or_probe);
    out[3] = sizeof(or_result);
}

/* ------------------------------------------------------------------------
 * Selectors (placement constraints Phi_C).
 *
 * Kubernetes matchExpressions semantics:
 *   In(k, S):         node carries key k and its value is in S
 *   NotIn(k, S):      node does not carry k, or its value is not in S
 *   Exists(k):        node carries k
 *   DoesNotExist(k):  node does not carry k
 * The expressions of one pod are ANDed; an empty list admits every node.
 * A value id of 0xFFFF means "key absent" in the label matrix; it is not a
 * valid value inside an expression (the expression is malformed).
 * ---------------------------------------------------------------------- */
static int expr_is_valid(const or_expr *e, uint32_t num_keys) {
    if (e->key >= num_keys) return 0;
    if (e->op == OR_OP_IN || e->op == OR_OP_NOTIN) {
        if (e->nvals < 1 || e->nvals > 8) return 0;
        for (int j = 0; j < e->nvals; ++j)
            if (e->vals[j] == OR_ABSENT) return 0;
        return 1;
    }
    if (e->op == OR_OP_EXISTS || e->op == OR_OP_DOESNOTEXIST) return e->nvals == 0;
    return 0;
}

static int value_in_set(uint16_t v, const or_expr *e) {
    for (int j = 0; j < e->nvals; ++j)
        if (e->vals[j] == v) return 1;
    return 0;
}

static int expr_matches(const or_expr *e, uint16_t label) {
    int present = label != OR_ABSENT;
    switch (e->op) {
    case OR_OP_IN: return present && value_in_set(label, e);
    case OR_OP_NOTIN: return !present || !value_in_set(label, e);
    case OR_OP_EXISTS: return present;
    default: return !present; /* DoesNotExist */
    }
}

/* carried[k][v] = 1 iff some node carries value v for key k (the "live node
 * label inventory" the hallucinated-identifier check consults). */
static uint8_t *build_inventory(uint32_t num_nodes, uint32_t num_keys, const uint16_t *labels) {
    uint8_t *inv = (uint8_t *)calloc((size_t)num_keys * 65536u, 1);
    if (!inv) return NULL;
    for (uint32_t k = 0; k < num_keys; ++k)
        for (uint32_t n = 0; n < num_nodes; ++n) {
            uint16_t v = labels[(size_t)k * num_nodes + n];
            if (v != OR_ABSENT) inv[(size_t)k * 65536u + v] = 1;
        }
    return inv;
}

/* bits[p][words_per_row]: node n -> word n>>5, bit n&31; padding zero.
 * flags[p]: ASSIGN_OK = assign[p] < N and that node is feasible;
 *           EMPTY = no feasible node (fail closed);
 *           UNKNOWN = an In value is carried by no node;
 *           PASS = ASSIGN_OK and not UNKNOWN (the placement check);
 *           BAD = malformed expression list (row left empty, check fails).
 * Returns 0, or -1 if the inventory could not be allocated. */
int oracle_eval_selectors(uint32_t num_nodes, uint32_t num_keys, const uint16_t *labels,
                          uint32_t num_pods, const uint32_t *expr_offs, uint32_t num_exprs,
                          const or_expr *exprs, const uint32_t *assign,
                          uint32_t *bits, uint32_t words_per_row, uint8_t *flags) {
    uint8_t *inv = build_inventory(num_nodes, num_keys, labels);
    if (!inv) return -1;
    for (uint32_t p = 0; p < num_pods; ++p) {
        uint32_t *row = bits + (size_t)p * words_per_row;
        memset(row, 0, (size_t)words_per_row * 4);
        uint32_t lo = expr_offs[p], hi = expr_offs[p + 1];
        int bad = hi < lo || hi > num_exprs;
        for (uint32_t e = lo; !bad && e < hi; ++e)
            if (!expr_is_valid(&exprs[e], num_keys)) bad = 1;
        if (bad) { flags[p] = OR_F_BAD; continue; }
        uint32_t count = 0;
        for (uint32_t n = 0; n < num_nodes; ++n) {
            int ok = 1;
            for (uint32_t e = lo; e < hi && ok; ++e)
                ok = expr_matches(&exprs[e], labels[(size_t)exprs[e].key * num_nodes + n]);
            if (ok) { row[n >> 5] |= 1u << (n & 31); ++count; }
        }
        int unknown = 0;
        for (uint32_t e = lo; e < hi; ++e)
            if (exprs[e].op == OR_OP_IN)
                for (int j = 0; j < exprs[e].nvals; ++j)
                    if (!inv[(size_t)exprs[e].key * 65536u + exprs[e].vals[j]]) unknown = 1;
        uint8_t f = 0;
        if (count == 0) f |= OR_F_EMPTY;
        if (unknown) f |= OR_F_UNKNOWN;
        if (assign) {
            uint32_t a = assign[p];
            if (a < num_nodes && ((row[a >> 5] >> (a & 31)) & 1u)) f |= OR_F_ASSIGN_OK;
            if ((f & OR_F_ASSIGN_OK) && !unknown) f |= OR_F_PASS;
        }
        flags[p] = f;
    }
    free(inv);
    return 0;
}

/* ------------------------------------------------------------------------
 * Flow rules: OpenFlow first match by priority.  A rule matches a header
 * (in_port, src, dst, dport) iff its in_port is ANY or equal, both address
 * prefixes match, and lo <= dport <= hi.  The first match is the matching
 * rule of highest priority; among equal priorities the lowest input index.
 * ---------------------------------------------------------------------- */
static int prefix_match(uint32_t addr, uint32_t value, uint32_t len) {
    if (len == 0) return 1;                 /* never shift by 32 */
    return ((addr ^ value) >> (32 - len)) == 0;
}

static int rule_matches(const or_rule *r, uint32_t in_port, uint32_t src, uint32_t dst, uint32_t dport) {
    if (r->in_port != OR_ANY_PORT && r->in_port != in_port) return 0;
    if (!prefix_match(src, r->src_ip, r->src_len)) return 0;
    if (!prefix_match(dst, r->dst_ip, r->dst_len)) return 0;
    return r->dport_lo <= dport && dport <= r->dport_hi;
}

int32_t oracle_first_match(const or_rule *rules, uint32_t num_rules, uint32_t in_port,
                           uint32_t src, uint32_t dst, uint32_t dport) {
    int32_t best = -1;
    for (uint32_t i = 0; i < num_rules; ++i) {
        if (!rule_matches(&rules[i], in_port, src, dst, dport)) continue;
        if (best < 0 || rules[i].priority > rules[best].priority) best = (int32_t)i;
    }
    return best;
}

/* ------------------------------------------------------------------------
 * Probe walk.  From the source host's attachment (switch, port), for hop
 * h = 0 .. cap-1 at switch s:
 *   1. if region(s) is not in the probe's permitted mask -> VIOLATION
 *      (the region check comes first: reaching a forbidden switch violates
 *      the intent even if that switch would then drop the packet);
 *   2. first-matching rule; no match or action DROP -> DROP (a table miss
 *      drops, as with no table-miss entry);
 *   3. output port: unconnected -> DROP; a host -> COMPLIANT if that host
 *      owns the destination address, else MISDELIVERED; a switch port ->
 *      continue there with that in_port.
 * A probe not terminated within cap switch visits is LOOP.  hops = switch
 * visits made; last_switch = the last switch visited.  A probe whose source
 * host id is out of range (e.g. its pod was not placed) is NOSRC with
 * hops 0 and last_switch 0xFFFF.
 * ---------------------------------------------------------------------- */
static or_result walk_one(uint32_t num_switches, const uint32_t *rule_offs, const or_rule *rules,
                          const uint8_t *switch_region, const uint32_t *port_offs, const int32_t *port_peer,
                          uint32_t num_hosts, const uint16_t *host_switch, const uint16_t *host_port,
                          const uint32_t *host_ip, const or_probe *pr, uint32_t hop_cap) {
    or_result res;
    (void)num_switches;
    if (pr->src_host >= num_hosts) {
        res.status = OR_NOSRC; res.hops = 0; res.last_switch = 0xFFFF;
        return res;
    }
    uint32_t s = host_switch[pr->src_host];
    uint32_t in_port = host_port[pr->src_host];
    uint32_t last = s;
    for (uint32_t h = 0; h < hop_cap; ++h) {
        last = s;
        res.hops = (uint8_t)(h + 1);
        res.last_switch = (uint16_t)s;
        uint32_t region = switch_region[s];
        if (region >= 32 || !((pr->allowed_mask >> region) & 1u)) { res.status = OR_VIOLATION; return res; }
        uint32_t r0 = rule_offs[s], nr = rule_offs[s + 1] - r0;
        int32_t m = oracle_first_match(rules + r0, nr, in_port, pr->src_ip, pr->dst_ip, pr->dport);
        if (m < 0 || rules[r0 + m].action == OR_DROP) { res.status = OR_DROPPED; return res; }
        uint32_t port = rules[r0 + m].action;
        uint32_t nports = port_offs[s + 1] - port_offs[s];
        if (port >= nports) { res.status = OR_DROPPED; return res; }
        int32_t peer = port_peer[port_offs[s] + port];
        if (peer < 0) { res.status = OR_DROPPED; return res; }
        if (peer & OR_HOST_BIT) {
            uint32_t q = (uint32_t)(peer & ~OR_HOST_BIT);
            res.status = (q < num_hosts && host_ip[q] == pr->dst_ip) ? OR_COMPLIANT : OR_MISDELIVERED;
            return res;
        }
        s = (uint32_t)peer >> 8;
        in_port = (uint32_t)peer & 0xFFu;
    }
    res.status = OR_LOOP;
    res.hops = (uint8_t)hop_cap;
    res.last_switch = (uint16_t)last;
    return res;
}

/* Walks probes[idx[i]] (or probes[i] when idx is NULL) into out[i]. */
void oracle_verify_probes(uint32_t num_switches, const uint32_t *rule_offs, const or_rule *rules,
                          const uint8_t *switch_region, const uint32_t *port_offs, const int32_t *port_peer,
                          uint32_t num_hosts, const uint16_t *host_switch, const uint16_t *host_port,
                          const uint32_t *host_ip, const or_probe *probes, const uint32_t *idx,
                          uint32_t count, uint32_t hop_cap, or_result *out) {
    for (uint32_t i = 0; i < count; ++i) {
        const or_probe *pr = &probes[idx ? idx[i] : i];
        out[i] = walk_one(num_switches, rule_offs, rules, switch_region, port_offs, port_peer, num_hosts,
                          host_switch, host_port, host_ip, pr, hop_cap);
    }
}

/* Multi-term node selectors (Sec. 3.3 and Sec. 4.1: placement constraints
 * are node selectors / affinities): the Kubernetes required node-affinity
 * form, a list of selector terms that are ORed, each term a list of
 * expressions that are ANDed:
 *     feasible(p) = union over p's terms t of { n : every expression of t
 *                   matches node n }.
 * Readings: a pod with no terms has no affinity and admits every node; a
 * term with no expressions matches no node (Kubernetes: an empty selector
 * term matches nothing); an In value carried by no node anywhere in the pod
 * sets UNKNOWN (the inventory check of Sec. 6.3 covers every referenced
 * label); a malformed term range or expression makes the pod BAD with an
 * empty row.  Pod p's terms are pod_terms[p] .. pod_terms[p+1]) of
 * term_offs, term t's expressions term_offs[t] .. term_offs[t+1]).  Flags
 * as oracle_eval_selectors. */
int oracle_eval_selector_terms(uint32_t num_nodes, uint32_t num_keys, const uint16_t *labels, uint32_t num_pods,
                               const uint32_t *pod_terms, uint32_t num_terms, const uint32_t *term_offs,
                               uint32_t num_exprs, const or_expr *exprs, const uint32_t *assign, uint32_t *bits,
                               uint32_t words_per_row, uint8_t *flags) {
    uint8_t *inv = build_inventory(num_nodes, num_keys, labels);
    if (!inv) return -1;
    for (uint32_t p = 0; p < num_pods; ++p) {
        uint32_t *row = bits + (size_t)p * words_per_row;
        memset(row, 0, (size_t)words_per_row * 4);
        uint32_t t0 = pod_terms[p], t1 = pod_terms[p + 1];
        int bad = t1 < t0 || t1 > num_terms;
        for (uint32_t t = t0; !bad && t < t1; ++t) {
            uint32_t lo = term_offs[t], hi = term_offs[t + 1];
            if (hi < lo || hi > num_exprs) { bad = 1; break; }
            for (uint32_t e = lo; e < hi; ++e)
                if (!expr_is_valid(&exprs[e], num_keys)) { bad = 1; break; }
        }
        if (bad) { flags[p] = OR_F_BAD; continue; }
        uint32_t count = 0;
        for (uint32_t n = 0; n < num_nodes; ++n) {
            int ok = t0 == t1;   /* no terms: no affinity */
            for (uint32_t t = t0; t < t1 && !ok; ++t) {
                uint32_t lo = term_offs[t], hi = term_offs[t + 1];
                int all = hi > lo;   /* an empty term matches nothing */
                for (uint32_t e = lo; e < hi && all; ++e)
                    all = expr_matches(&exprs[e], labels[(size_t)exprs[e].key * num_nodes + n]);
                ok = all;
            }
            if (ok) { row[n >> 5] |= 1u << (n & 31); ++count; }
        }
        int unknown = 0;
        for (uint32_t t = t0; t < t1; ++t)
            for (uint32_t e = term_offs[t]; e < term_offs[t + 1]; ++e)
                if (exprs[e].op == OR_OP_IN)
                    for (int j = 0; j < exprs[e].nvals; ++j)
                        if (!inv[(size_t)exprs[e].key * 65536u + exprs[e].vals[j]]) unknown = 1;
        uint8_t f = 0;
        if (count == 0) f |= OR_F_EMPTY;
        if (unknown) f |= OR_F_UNKNOWN;
        if (assign) {
            uint32_t a = assign[p];
            if (a < num_nodes && ((row[a >> 5] >> (a & 31)) & 1u)) f |= OR_F_ASSIGN_OK;
            if ((f & OR_F_ASSIGN_OK) && !unknown) f |= OR_F_PASS;
        }
        flags[p] = f;
    }
    free(inv);
    return 0;
}

/* ------------------------------------------------------------------------
 * Compliant reach R(s, m): empty if region(s) is not permitted by m (the
 * source itself lies on every path); otherwise the vertices visited by a
 * breadth-first search from s over CSR edges u -> v that enters v only if
 * region(v) is permitted.  Row layout as the selector bitsets.  Out-of-range
 * neighbours and regions >= 32 are never entered; an out-of-range source
 * yields an empty row.  A CSR whose offsets are malformed (some row with
 * offs[u+1] < offs[u] or offs[u+1] > num_edges) has no usable edge list, so
 * it is read as a graph with no edges.  pairs (optional) lists (mask index,
 * source index) to compute; rows are written in pair order.  Without pairs,
 * all num_masks x num_src rows are written mask-major.
 * ---------------------------------------------------------------------- */
static int vertex_allowed(const uint8_t *region, uint32_t v, uint32_t mask) {
    return region[v] < 32 && ((mask >> region[v]) & 1u);
}

static void bfs_row(uint32_t V, const uint32_t *offs, const uint32_t *cols, int has_edges, const uint8_t *region,
                    uint32_t s, uint32_t mask, uint32_t *row, uint32_t words_per_row,
                    uint32_t *queue, uint8_t *seen) {
    memset(row, 0, (size_t)words_per_row * 4);
    if (s >= V || !vertex_allowed(region, s, mask)) return;
    memset(seen, 0, V);
    uint32_t head = 0, tail = 0;
    queue[tail++] = s;
    seen[s] = 1;
    while (head < tail) {
        uint32_t u = queue[head++];
        row[u >> 5] |= 1u << (u & 31);
        if (!has_edges) continue;
        for (uint32_t e = offs[u]; e < offs[u + 1]; ++e) {
            uint32_t v = cols[e];
            if (v >= V || seen[v] || !vertex_allowed(region, v, mask)) continue;
            seen[v] = 1;
            queue[tail++] = v;
        }
    }
}

int oracle_compliant_reach(uint32_t V, const uint32_t *offs, uint32_t num_edges, const uint32_t *cols,
                           const uint8_t *region, uint32_t num_src, const uint32_t *src, uint32_t num_masks,
                           const uint32_t *masks, const uint32_t *pairs, uint32_t num_pairs, uint32_t *reach,
                           uint32_t words_per_row) {
    uint32_t *queue = (uint32_t *)malloc((size_t)(V + 1) * 4);
    uint8_t *seen = (uint8_t *)malloc((size_t)V + 1);
    if (!queue || !seen) { free(queue); free(seen); return -1; }
    int has_edges = 1;
    for (uint32_t u = 0; u < V; ++u)
        if (offs[u + 1] < offs[u] || offs[u + 1] > num_edges) has_edges = 0;
    if (pairs) {
        for (uint32_t i = 0; i < num_pairs; ++i) {
            uint32_t m = pairs[2 * i], j = pairs[2 * i + 1];
            bfs_row(V, offs, cols, has_edges, region, src[j], masks[m], reach + (size_t)i * words_per_row,
                    words_per_row, queue, seen);
        }
    } else {
        for (uint32_t m = 0; m < num_masks; ++m)
            for (uint32_t j = 0; j < num_src; ++j)
                bfs_row(V, offs, cols, has_edges, region, src[j], masks[m],
                        reach + ((size_t)m * num_src + j) * words_per_row, words_per_row, queue, seen);
    }
    free(queue);
    free(seen);
    return 0;
}

/* ------------------------------------------------------------------------
 * End-to-end composition (Sec. 4.2 hybrid coordination: pods are placed
 * first, then flows from their attachments are checked).
 *
 * Placement: the pods of group g (an intent) are placed by a seeded uniform
 * choice among the feasible nodes of row g: with c = |feasible|, pod j gets
 * the r-th feasible node in ascending order, r = draws[g*pods+j] mod c; an
 * empty row leaves the pod UNPLACED.
 * ---------------------------------------------------------------------- */
void oracle_place_pods(uint32_t num_groups, uint32_t pods_per_group, uint32_t num_nodes,
                       const uint32_t *bits, uint32_t words_per_row, const uint64_t *draws, uint32_t *assign) {
    for (uint32_t g = 0; g < num_groups; ++g) {
        const uint32_t *row = bits + (size_t)g * words_per_row;
        uint32_t c = 0;
        for (uint32_t n = 0; n < num_nodes; ++n) c += (row[n >> 5] >> (n & 31)) & 1u;
        for (uint32_t j = 0; j < pods_per_group; ++j) {
            size_t pod = (size_t)g * pods_per_group + j;
            if (c == 0) { assign[pod] = OR_UNPLACED; continue; }
            uint64_t r = draws[pod] % c;
            uint32_t seen = 0;
            for (uint32_t n = 0; n < num_nodes; ++n) {
                if (!((row[n >> 5] >> (n & 31)) & 1u)) continue;
                if (seen == r) { assign[pod] = n; break; }
                ++seen;
            }
        }
    }
}

/* Probe k of group g = k / probes_per_group is sent from the host of the
 * group's pod (k mod probes_per_group) mod pods_per_group (round robin);
 * node n is host n.  A pod without a host gives a NOSRC probe. */
void oracle_bind_probes(uint32_t num_probes, or_probe *probes, uint32_t probes_per_group,
                        uint32_t pods_per_group, const uint32_t *assign, uint32_t num_hosts,
                        const uint32_t *host_ip) {
    for (uint32_t k = 0; k < num_probes; ++k) {
        uint32_t g = k / probes_per_group;
        uint32_t pod = g * pods_per_group + (k % probes_per_group) % pods_per_group;
        uint32_t node = assign[pod];
        if (node < num_hosts) {
            probes[k].src_host = (uint16_t)node;
            probes[k].src_ip = host_ip[node];
        } else {
            probes[k].src_host = OR_NO_HOST;
            probes[k].src_ip = 0;
        }
    }
}

/* An intent passes iff every check passes (Sec. 5.5): each of its pods is on
 * a node of its feasible set, its selector references no unknown value and
 * is well formed, and every probe of its flows is COMPLIANT.
 * counts[g][0..5] = probe status histogram, counts[g][6] = pods whose
 * placement check passed, counts[g][7] = 0. */
void oracle_aggregate(uint32_t num_groups, uint32_t pods_per_group, uint32_t num_nodes,
                      const uint32_t *bits, uint32_t words_per_row, const uint8_t *group_flags,
                      const uint32_t *assign, uint32_t probes_per_group, const or_result *results,
                      uint8_t *pass, uint32_t *counts) {
    for (uint32_t g = 0; g < num_groups; ++g) {
        uint32_t *c = counts + (size_t)g * 8;
        memset(c, 0, 8 * 4);
        const uint32_t *row = bits + (size_t)g * words_per_row;
        int ok = !(group_flags[g] & (OR_F_UNKNOWN | OR_F_BAD));
        for (uint32_t j = 0; j < pods_per_group; ++j) {
            uint32_t a = assign[(size_t)g * pods_per_group + j];
            int pod_ok = a < num_nodes && ((row[a >> 5] >> (a & 31)) & 1u);
            c[6] += pod_ok;
            ok = ok && pod_ok;
        }
        for (uint32_t k = 0; k < probes_per_group; ++k) {
            uint8_t st = results[(size_t)g * probes_per_group + k].status;
            if (st < 6) c[st] += 1;
            ok = ok && st == OR_COMPLIANT;
        }
        pass[g] = (uint8_t)ok;
    }
}

/* ------------------------------------------------------------------------
 * Path constraints of a flow set (Sec. 4.2: the constraint object handed to
 * the flow scheduler names forbidden switches and must_go switches; Sec.
 * 5.3, networking intent: the realised path must include the waypoint;
 * Sec. 5.5: network checks assert that realised paths avoid forbidden
 * switches and include required waypoints).
 *
 * Policy p: forbidden switches forbid[forbid_offs[p] .. forbid_offs[p+1]),
 * required waypoints must[must_offs[p] .. must_offs[p+1]) (at most 32).
 * Probe k follows policy probe_policy[k] (or k / probes_per_policy when
 * probe_policy is NULL); a policy index >= num_policies means none.
 *
 * The walk is walk_one's with one more check at every switch visit: a
 * forbidden switch is judged exactly like a switch outside the probe's
 * jurisdictions (VIOLATION there, the walk stops).  Reading: a visit counts
 * toward the waypoints only once it has passed these checks.  hits[k] bit i
 * is set iff must[must_offs[p] + i] was visited.
 * ---------------------------------------------------------------------- */
static int in_list(const uint16_t *list, uint32_t n, uint32_t s) {
    for (uint32_t i = 0; i < n; ++i)
        if (list[i] == s) return 1;
    return 0;
}

static or_result walk_constrained(const uint32_t *rule_offs, const or_rule *rules, const uint8_t *switch_region,
                                  const uint32_t *port_offs, const int32_t *port_peer, uint32_t num_hosts,
                                  const uint16_t *host_switch, const uint16_t *host_port, const uint32_t *host_ip,
                                  const or_probe *pr, uint32_t hop_cap, const uint16_t *forbid, uint32_t nforbid,
                                  const uint16_t *must, uint32_t nmust, uint32_t *hits) {
    or_result res;
    *hits = 0;
    if (pr->src_host >= num_hosts) {
        res.status = OR_NOSRC; res.hops = 0; res.last_switch = 0xFFFF;
        return res;
    }
    uint32_t s = host_switch[pr->src_host];
    uint32_t in_port = host_port[pr->src_host];
    uint32_t last = s;
    for (uint32_t h = 0; h < hop_cap; ++h) {
        last = s;
        res.hops = (uint8_t)(h + 1);
        res.last_switch = (uint16_t)s;
        uint32_t region = switch_region[s];
        if (region >= 32 || !((pr->allowed_mask >> region) & 1u) || in_list(forbid, nforbid, s)) {
            res.status = OR_VIOLATION;
            return res;
        }
        for (uint32_t i = 0; i < nmust; ++i)
            if (must[i] == s) *hits |= 1u << i;
        uint32_t r0 = rule_offs[s], nr = rule_offs[s + 1] - r0;
        int32_t m = oracle_first_match(rules + r0, nr, in_port, pr->src_ip, pr->dst_ip, pr->dport);
        if (m < 0 || rules[r0 + m].action == OR_DROP) { res.status = OR_DROPPED; return res; }
        uint32_t port = rules[r0 + m].action;
        uint32_t nports = port_offs[s + 1] - port_offs[s];
        if (port >= nports) { res.status = OR_DROPPED; return res; }
        int32_t peer = port_peer[port_offs[s] + port];
        if (peer < 0) { res.status = OR_DROPPED; return res; }
        if (peer & OR_HOST_BIT) {
            uint32_t q = (uint32_t)(peer & ~OR_HOST_BIT);
            res.status = (q < num_hosts && host_ip[q] == pr->dst_ip) ? OR_COMPLIANT : OR_MISDELIVERED;
            return res;
        }
        s = (uint32_t)peer >> 8;
        in_port = (uint32_t)peer & 0xFFu;
    }
    res.status = OR_LOOP;
    res.hops = (uint8_t)hop_cap;
    res.last_switch = (uint16_t)last;
    return res;
}

void oracle_verify_constrained(const uint32_t *rule_offs, const or_rule *rules, const uint8_t *switch_region,
                               const uint32_t *port_offs, const int32_t *port_peer, uint32_t num_hosts,
                               const uint16_t *host_switch, const uint16_t *host_port, const uint32_t *host_ip,
                               const or_probe *probes, const uint32_t *probe_policy, uint32_t probes_per_policy,
                               uint32_t num_policies, const uint32_t *forbid_offs, const uint16_t *forbid,
                               const uint32_t *must_offs, const uint16_t *must, const uint32_t *idx, uint32_t count,
                               uint32_t hop_cap, or_result *out, uint32_t *hits) {
    for (uint32_t i = 0; i < count; ++i) {
        uint32_t k = idx ? idx[i] : i;
        uint32_t p = probe_policy ? probe_policy[k] : (probes_per_policy ? k / probes_per_policy : 0xFFFFFFFFu);
        const uint16_t *fb = NULL, *mg = NULL;
        uint32_t nf = 0, nm = 0;
        if (p < num_policies) {
            fb = forbid + forbid_offs[p];
            nf = forbid_offs[p + 1] - forbid_offs[p];
            mg = must + must_offs[p];
            nm = must_offs[p + 1] - must_offs[p];
        }
        out[i] = walk_constrained(rule_offs, rules, switch_region, port_offs, port_peer, num_hosts, host_switch,
                                  host_port, host_ip, &probes[k], hop_cap, fb, nf, mg, nm, &hits[i]);
    }
}

/* Per-intent verdict with path constraints (Sec. 5.5: an intent passes only
 * if all its checks pass).  On top of oracle_aggregate's checks, group g's
 * policy p = group_policy[g] (or g when group_policy is NULL; p >=
 * num_policies: none) must be concrete (Sec. 6.3, failure mode 2: a
 * constraint object without a concrete src/dst applies to no flow, a no-op
 * policy, and the intent is reported as not enforced) and every probe of g
 * must have visited all of p's waypoints.  counts[g][7] = probes of g that
 * missed a waypoint. */
void oracle_aggregate_constrained(uint32_t num_groups, uint32_t pods_per_group, uint32_t num_nodes,
                                  const uint32_t *bits, uint32_t words_per_row, const uint8_t *group_flags,
                                  const uint32_t *assign, uint32_t probes_per_group, const or_result *results,
                                  const uint32_t *hits, const uint32_t *group_policy, uint32_t num_policies,
                                  const uint32_t *must_offs, const uint8_t *concrete, uint8_t *pass,
                                  uint32_t *counts) {
    oracle_aggregate(num_groups, pods_per_group, num_nodes, bits, words_per_row, group_flags, assign,
                     probes_per_group, results, pass, counts);
    for (uint32_t g = 0; g < num_groups; ++g) {
        uint32_t p = group_policy ? group_policy[g] : g;
        if (p >= num_policies) continue;
        uint32_t nm = must_offs[p + 1] - must_offs[p];
        uint32_t full = nm >= 32 ? 0xFFFFFFFFu : ((1u << nm) - 1u);
        uint32_t missed = 0;
        for (uint32_t k = 0; k < probes_per_group; ++k)
            if (hits[(size_t)g * probes_per_group + k] != full) missed += 1;
        counts[(size_t)g * 8 + 7] = missed;
        if (!concrete[p] || missed) pass[g] = 0;
    }
}

/* ------------------------------------------------------------------------
 * Path scheduler (Sec. 4.2: the flow scheduling module computes paths that
 * respect the constraint object with graph algorithms -- weighted Dijkstra,
 * BFS when no weights are given -- and turns each path into per-hop flow
 * rules).
 *
 * Request r: from host src to host dst, over switches whose region the mask
 * permits and that its policy (index >= num_policies: none) does not forbid,
 * through the policy's waypoints in their listed order.  The path is the
 * concatenation of shortest segments src switch -> waypoint 1 -> ... -> dst
 * switch.  Link u --port p--> v costs w[port_offs[u] + p] (a weight of 0
 * counts as 1; all 1 when w is NULL, i.e. breadth-first hop counts).
 *
 * Readings: a shortest segment is made canonical by walking back from its
 * end and taking, at every switch v, the predecessor link (u, p) with the
 * smallest u, then the smallest p, among those on some shortest path; the
 * path is a list of visits (switch, in_port, out_port), in_port of the
 * first visit = the source host's port, out_port of the last = the
 * destination host's port.  Status: 0 OK; 1 NOSRC (a host id out of
 * range); 2 BLOCKED (an endpoint or waypoint switch is not permitted, or a
 * segment has no path); 3 TOO_LONG (more than max_len visits); 4 REPEAT (a
 * (switch, in_port) pair recurs: per-hop rules that match on the header and
 * in_port cannot realise the path).  Visits are encoded switch << 16 |
 * in_port << 8 | out_port.
 * ---------------------------------------------------------------------- */
typedef struct { uint16_t src_host, dst_host; uint32_t allowed_mask, policy, reserved; } or_path_req;

static uint32_t link_w(const uint16_t *w, uint32_t i) { return w && w[i] ? w[i] : 1u; }   /* 0 counts as 1 */

static int switch_ok(const uint8_t *region, uint32_t mask, const uint16_t *forbid, uint32_t nforbid, uint32_t s) {
    return region[s] < 32 && ((mask >> region[s]) & 1u) && !in_list(forbid, nforbid, s);
}

/* Dijkstra from a over permitted switches (simple O(S^2) selection). */
static void dijkstra(uint32_t S, const uint32_t *port_offs, const int32_t *port_peer, const uint16_t *w,
                     const uint8_t *ok, uint32_t a, uint32_t *dist, uint8_t *done) {
    for (uint32_t v = 0; v < S; ++v) { dist[v] = 0xFFFFFFFFu; done[v] = 0; }
    dist[a] = 0;
    for (;;) {
        uint32_t u = S, best = 0xFFFFFFFFu;
        for (uint32_t v = 0; v < S; ++v)
            if (!done[v] && dist[v] < best) { best = dist[v]; u = v; }
        if (u == S) return;
        done[u] = 1;
        for (uint32_t p = 0; p < port_offs[u + 1] - port_offs[u]; ++p) {
            int32_t peer = port_peer[port_offs[u] + p];
            if (peer < 0 || (peer & OR_HOST_BIT)) continue;
            uint32_t v = (uint32_t)peer >> 8;
            if (v >= S || !ok[v]) continue;
            uint32_t c = dist[u] + link_w(w, port_offs[u] + p);
            if (c < dist[v]) dist[v] = c;
        }
    }
}

void oracle_schedule_paths(uint32_t S, const uint8_t *switch_region, const uint32_t *port_offs,
                           const int32_t *port_peer, uint32_t num_hosts, const uint16_t *host_switch,
                           const uint16_t *host_port, const uint16_t *weights, uint32_t num_policies,
                           const uint32_t *forbid_offs, const uint16_t *forbid, const uint32_t *must_offs,
                           const uint16_t *must, uint32_t num_req, const or_path_req *req, uint32_t max_len,
                           uint32_t *hops, uint8_t *len, uint8_t *status) {
    uint32_t *dist = malloc((size_t)S * 4);
    uint8_t *done = malloc(S), *ok = malloc(S);
    uint32_t *seg = malloc((size_t)(S + 1) * 4 * 2);
    for (uint32_t r = 0; r < num_req; ++r) {
        uint32_t *out = hops + (size_t)r * max_len;
        len[r] = 0;
        const or_path_req *q = &req[r];
        if (q->src_host >= num_hosts || q->dst_host >= num_hosts) { status[r] = 1; continue; }
        const uint16_t *fb = NULL, *mg = NULL;
        uint32_t nf = 0, nm = 0;
        if (q->policy < num_policies) {
            fb = forbid + forbid_offs[q->policy];
            nf = forbid_offs[q->policy + 1] - forbid_offs[q->policy];
            mg = must + must_offs[q->policy];
            nm = must_offs[q->policy + 1] - must_offs[q->policy];
        }
        for (uint32_t s = 0; s < S; ++s) ok[s] = (uint8_t)switch_ok(switch_region, q->allowed_mask, fb, nf, s);
        uint32_t cur = host_switch[q->src_host], dst = host_switch[q->dst_host];
        int st = 0;
        if (!ok[cur] || !ok[dst]) st = 2;
        for (uint32_t i = 0; i < nm && !st; ++i)
            if (!ok[mg[i]]) st = 2;
        /* visits: (switch, in_port) with out_port filled when the next link is chosen */
        uint32_t n = 1, vsw[256], vin[256], vout[256];
        vsw[0] = cur; vin[0] = host_port[q->src_host]; vout[0] = 0;
        for (uint32_t i = 0; i <= nm && !st; ++i) {
            uint32_t tgt = i < nm ? mg[i] : dst;
            if (tgt == cur) continue;
            dijkstra(S, port_offs, port_peer, weights, ok, cur, dist, done);
            if (dist[tgt] == 0xFFFFFFFFu) { st = 2; break; }
            /* canonical walk back: seg holds (u, p) pairs from tgt to cur */
            uint32_t k = 0, v = tgt;
            while (v != cur) {
                uint32_t bu = S, bp = 0, bq = 0;
                for (uint32_t u = 0; u < S && bu == S; ++u) {
                    if (!ok[u] || dist[u] == 0xFFFFFFFFu) continue;
                    for (uint32_t p = 0; p < port_offs[u + 1] - port_offs[u]; ++p) {
                        int32_t peer = port_peer[port_offs[u] + p];
                        if (peer < 0 || (peer & OR_HOST_BIT) || ((uint32_t)peer >> 8) != v) continue;
                        if (dist[u] + link_w(weights, port_offs[u] + p) == dist[v]) {
                            bu = u; bp = p; bq = (uint32_t)peer & 0xFFu;
                            break;
                        }
                    }
                }
                seg[2 * k] = bu << 8 | bp;
                seg[2 * k + 1] = v << 8 | bq;
                ++k;
                v = bu;
            }
            while (k > 0 && !st) {
                --k;
                uint32_t p = seg[2 * k] & 0xFFu, v2 = seg[2 * k + 1] >> 8, q2 = seg[2 * k + 1] & 0xFFu;
                if (n >= max_len) { st = 3; break; }
                vout[n - 1] = p;
                vsw[n] = v2; vin[n] = q2; vout[n] = 0;
                ++n;
            }
            cur = tgt;
        }
        if (!st) {
            vout[n - 1] = host_port[q->dst_host];
            for (uint32_t i = 0; i < n && !st; ++i)
                for (uint32_t j = i + 1; j < n; ++j)
                    if (vsw[i] == vsw[j] && vin[i] == vin[j]) { st = 4; break; }
        }
        status[r] = (uint8_t)st;
        if (!st) {
            len[r] = (uint8_t)n;
            for (uint32_t i = 0; i < n; ++i) out[i] = vsw[i] << 16 | vin[i] << 8 | vout[i];
        }
    }
    free(dist); free(done); free(ok); free(seg);
}

/* Per-hop rules of the scheduled paths (Sec. 4.2: each path becomes per-hop
 * flow rules): visit i of an OK request becomes, at its switch, the rule
 * {priority, in_port, src /32, dst /32, any port, action out_port}, in slot
 * r * max_len + i; rule_switch of the slot = its switch, 0xFFFF for unused
 * slots. */
void oracle_compile_path_rules(uint32_t num_req, const or_path_req *req, const uint32_t *host_ip, uint32_t max_len,
                               const uint32_t *hops, const uint8_t *len, const uint8_t *status, uint16_t priority,
                               or_rule *rules, uint16_t *rule_switch) {
    for (uint32_t r = 0; r < num_req; ++r)
        for (uint32_t i = 0; i < max_len; ++i) {
            size_t k = (size_t)r * max_len + i;
            memset(&rules[k], 0, sizeof(or_rule));
            rule_switch[k] = 0xFFFF;
            if (status[r] != 0 || i >= len[r]) continue;
            uint32_t h = hops[k];
            rules[k].priority = priority;
            rules[k].in_port = (uint16_t)((h >> 8) & 0xFFu);
            rules[k].src_ip = host_ip[req[r].src_host];
            rules[k].src_len = 32;
            rules[k].dst_ip = host_ip[req[r].dst_host];
            rules[k].dst_len = 32;
            rules[k].dport_lo = 0;
            rules[k].dport_hi = 0xFFFF;
            rules[k].action = (uint16_t)(h & 0xFFu);
            rule_switch[k] = (uint16_t)(h >> 16);
        }
}
