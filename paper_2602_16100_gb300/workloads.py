"""Seeded synthetic workloads for the cross-layer privacy validator.

This module only *produces input arrays*: node label matrices, selector
expressions, switch topologies with their flow tables, probe headers, masked
graphs and the random draws used by the seeded placement.  It holds none of
the validator's arithmetic (no selector matching, no first-match, no walk, no
reachability), so both the CUDA path and the CPU oracle can consume the same
arrays without sharing any of the method.

Random numbers come from a counter-based generator: the i-th output of a
stream is the SplitMix64 output function (Steele, Lea & Flood, "Fast
splittable pseudorandom number generators", OOPSLA 2014) applied to
``key + (i + 1) * 0x9E3779B97F4A7C15``, where ``key`` is derived from the
workload seed and a stream name.  Every draw is therefore a pure function of
(seed, stream, index) and can be vectorised.

Array layouts (little endian, byte-compatible with the C structs of the
library and of the oracle):

* ``EXPR_DTYPE`` (20 B): key u16, op u8, nvals u8, vals u16[8]
* ``RULE_DTYPE`` (20 B): priority u16, in_port u16, src_ip u32, dst_ip u32,
  src_len u8, dst_len u8, dport_lo u16, dport_hi u16, action u16
* ``PROBE_DTYPE`` (16 B): src_ip u32, dst_ip u32, dport u16, src_host u16,
  allowed_mask u32
* ``RESULT_DTYPE`` (4 B): status u8, hops u8, last_switch u16

Port-peer encoding (int32): -1 = unconnected, ``HOST_BIT | h`` = host h,
otherwise ``(switch << 8) | port`` of the peer switch port.

The five workload recipes follow the configurations the validator is
benchmarked on (tiny, placement-scale, flow-verification, continuum WAN,
end-to-end cross-layer); their sizes are parameters so tests can build scaled
down instances with the same structure.
"""
from __future__ import annotations

import dataclasses
import zlib
from typing import Optional

import numpy as np

# ----------------------------------------------------------------------------
# layouts and encodings
# ----------------------------------------------------------------------------
EXPR_DTYPE = np.dtype([("key", "<u2"), ("op", "u1"), ("nvals", "u1"), ("vals", "<u2", (8,))])
RULE_DTYPE = np.dtype([("priority", "<u2"), ("in_port", "<u2"), ("src_ip", "<u4"),
                       ("dst_ip", "<u4"), ("src_len", "u1"), ("dst_len", "u1"),
                       ("dport_lo", "<u2"), ("dport_hi", "<u2"), ("action", "<u2")])
PROBE_DTYPE = np.dtype([("src_ip", "<u4"), ("dst_ip", "<u4"), ("dport", "<u2"),
                        ("src_host", "<u2"), ("allowed_mask", "<u4")])
RESULT_DTYPE = np.dtype([("status", "u1"), ("hops", "u1"), ("last_switch", "<u2")])
assert EXPR_DTYPE.itemsize == 20 and RULE_DTYPE.itemsize == 20
assert PROBE_DTYPE.itemsize == 16 and RESULT_DTYPE.itemsize == 4

ABSENT = 0xFFFF          # label value id of a key a node does not carry
OP_IN, OP_NOTIN, OP_EXISTS, OP_DOESNOTEXIST = 0, 1, 2, 3
ANY_PORT = 0xFFFF        # rule.in_port wildcard
DROP = 0xFFFF            # rule.action: drop
NO_HOST = 0xFFFF         # probe.src_host: no source (its pod was not placed)
PEER_NONE = -1
HOST_BIT = 1 << 30
UNPLACED = 0xFFFFFFFF    # assign[] value of a pod with no feasible node

ST_COMPLIANT, ST_VIOLATION, ST_DROP, ST_LOOP, ST_MISDELIVERED, ST_NOSRC = range(6)
STATUS_NAMES = ("compliant", "violation", "drop", "loop", "misdelivered", "nosrc")

F_ASSIGN_OK, F_EMPTY, F_UNKNOWN_VALUE, F_PASS, F_BAD_EXPR = 1, 2, 4, 8, 16

ROUTING_PRIORITY = 100
PASS_DPORT_LO = 49152    # end-to-end variant with passing intents: ports no ACL rule covers

_GAMMA = 0x9E3779B97F4A7C15
_M1 = 0xBF58476D1CE4E5B9
_M2 = 0x94D049BB133111EB


def words_per_row(num_bits: int) -> int:
    """Row length in u32 words for an LSB-first bitset over ``num_bits``
    items, padded to a multiple of 128 bits so rows start 16-byte aligned."""
    return max(4, ((num_bits + 127) // 128) * 4)


# ----------------------------------------------------------------------------
# counter-based random streams
# ----------------------------------------------------------------------------
def _mix64(z: np.ndarray) -> np.ndarray:
    with np.errstate(over="ignore"):
        z = (z ^ (z >> np.uint64(30))) * np.uint64(_M1)
        z = (z ^ (z >> np.uint64(27))) * np.uint64(_M2)
        return z ^ (z >> np.uint64(31))


class Stream:
    """One named counter-based random stream of a workload seed."""

    def __init__(self, seed: int, name: str):
        base = np.array([((seed * 0x100000001B3) ^ zlib.crc32(name.encode())) & 0xFFFFFFFFFFFFFFFF], dtype=np.uint64)
        self.key = _mix64(base)[0]
        self.counter = 0

    def u64(self, n: int) -> np.ndarray:
        idx = np.arange(self.counter + 1, self.counter + n + 1, dtype=np.uint64)
        self.counter += n
        with np.errstate(over="ignore"):
            return _mix64(self.key + idx * np.uint64(_GAMMA))

    def ints(self, lo: int, hi: int, n: int) -> np.ndarray:
        """n integers uniform in [lo, hi] (inclusive), as int64."""
        span = np.uint64(hi - lo + 1)
        return (self.u64(n) % span).astype(np.int64) + lo

    def floats(self, n: int) -> np.ndarray:
        return (self.u64(n) >> np.uint64(11)).astype(np.float64) * (1.0 / (1 << 53))

    def zipf(self, s: float, n_values: int, n: int) -> np.ndarray:
        """Zipf(s) over value ids 0..n_values-1 (id 0 most frequent), by
        inverse CDF over a precomputed double table."""
        w = 1.0 / np.arange(1, n_values + 1, dtype=np.float64) ** s
        cdf = np.cumsum(w) / w.sum()
        return np.minimum(np.searchsorted(cdf, self.floats(n), side="right"), n_values - 1)

    def permutation(self, n: int) -> np.ndarray:
        return np.argsort(self.u64(n), kind="stable")


# ----------------------------------------------------------------------------
# containers
# ----------------------------------------------------------------------------
# compact flow of an intent: {dst_ip, dport, reserved}
FLOW_DTYPE = np.dtype([("dst_ip", "<u4"), ("dport", "<u2"), ("reserved", "<u2")])
# path request of the scheduler: {src_host, dst_host, allowed_mask, policy, reserved}
PATH_REQ_DTYPE = np.dtype([("src_host", "<u2"), ("dst_host", "<u2"), ("allowed_mask", "<u4"), ("policy", "<u4"),
                           ("reserved", "<u4")])
NO_POLICY = 0xFFFFFFFF
PATH_OK, PATH_NOSRC, PATH_BLOCKED, PATH_TOO_LONG, PATH_REPEAT = 0, 1, 2, 3, 4


@dataclasses.dataclass
class Cluster:
    num_nodes: int
    num_keys: int
    labels: np.ndarray            # u16 [num_keys * num_nodes], key-major (SoA)


@dataclasses.dataclass
class Selectors:
    num_pods: int
    expr_offs: np.ndarray         # u32 [num_pods + 1]
    exprs: np.ndarray             # EXPR_DTYPE [num_exprs]
    assign: Optional[np.ndarray]  # u32 [num_pods] or None


@dataclasses.dataclass
class SelectorTerms:
    num_pods: int
    pod_terms: np.ndarray         # u32 [num_pods + 1]: terms of each pod (ORed)
    term_offs: np.ndarray         # u32 [num_terms + 1]: expressions of each term (ANDed)
    exprs: np.ndarray             # EXPR_DTYPE [num_exprs]
    assign: np.ndarray            # u32 [num_pods]


@dataclasses.dataclass
class Network:
    num_switches: int
    rule_offs: np.ndarray         # u32 [S + 1]
    rules: np.ndarray             # RULE_DTYPE [R]
    switch_region: np.ndarray     # u8 [S]
    port_offs: np.ndarray         # u32 [S + 1]
    port_peer: np.ndarray         # i32 [port_offs[S]]
    num_hosts: int
    host_switch: np.ndarray       # u16 [H]
    host_port: np.ndarray         # u16 [H]
    host_ip: np.ndarray           # u32 [H]
    shadowed_by: Optional[np.ndarray] = None  # i32 [R]: global index of a rule that shadows it, or -1
    adj_offs: Optional[np.ndarray] = None      # switch graph CSR (symmetric)
    adj_cols: Optional[np.ndarray] = None


@dataclasses.dataclass
class Probes:
    probes: np.ndarray            # PROBE_DTYPE [M]
    hop_cap: int


@dataclasses.dataclass
class Graph:
    num_vertices: int
    offs: np.ndarray              # u32 [V + 1]
    cols: np.ndarray              # u32 [E]
    region: np.ndarray            # u8 [V]


@dataclasses.dataclass
class ReachQuery:
    graph: Graph
    sources: np.ndarray           # u32 [num_src]
    masks: np.ndarray             # u32 [num_masks]


@dataclasses.dataclass
class EndToEnd:
    cluster: Cluster
    intents: Selectors            # one selector row per intent (assign None)
    intent_mask: np.ndarray       # u32 [I]
    pods_per_intent: int
    place_draws: np.ndarray       # u64 [I * pods_per_intent]
    network: Network
    probes: Probes                # src_host / src_ip filled by binding to placed pods
    probes_per_intent: int


@dataclasses.dataclass
class PathPolicies:
    num_policies: int
    forbid_offs: np.ndarray       # u32 [P + 1]
    forbid: np.ndarray            # u16: forbidden switches of each policy
    must_offs: np.ndarray         # u32 [P + 1]
    must: np.ndarray              # u16: required waypoints of each policy (<= 32)
    concrete: np.ndarray          # u8 [P]: 1 if the constraint names a concrete (src, dst) flow


# ----------------------------------------------------------------------------
# helpers shared by the recipes
# ----------------------------------------------------------------------------
def _csr_from_edges(n: int, edges: np.ndarray):
    """Symmetric CSR (neighbours sorted ascending) from undirected edge pairs."""
    if len(edges) == 0:
        return np.zeros(n + 1, np.uint32), np.zeros(0, np.uint32)
    a = np.concatenate([edges[:, 0], edges[:, 1]])
    b = np.concatenate([edges[:, 1], edges[:, 0]])
    order = np.lexsort((b, a))
    a, b = a[order], b[order]
    offs = np.zeros(n + 1, np.int64)
    np.add.at(offs, a + 1, 1)
    return np.cumsum(offs).astype(np.uint32), b.astype(np.uint32)


def _next_hops(num_switches: int, adj_offs: np.ndarray, adj_cols: np.ndarray) -> np.ndarray:
    """nh[s, d] = neighbour of s on a BFS shortest path to d (ties -> lowest
    neighbour id); nh[d, d] = -1.  Used only to synthesise routing rules."""
    import scipy.sparse as sp
    from scipy.sparse.csgraph import shortest_path
    n = num_switches
    m = sp.csr_matrix((np.ones(len(adj_cols)), adj_cols.astype(np.int64), adj_offs.astype(np.int64)), shape=(n, n))
    dist = shortest_path(m, method="D", unweighted=True)
    nh = np.full((n, n), -1, np.int64)
    for s in range(n):
        nb = adj_cols[adj_offs[s]:adj_offs[s + 1]].astype(np.int64)  # ascending
        if len(nb) == 0:
            continue
        good = dist[nb, :] == (dist[s, :] - 1)[None, :]     # [deg, n]
        first = np.argmax(good, axis=0)
        ok = good.any(axis=0)
        nh[s, ok] = nb[first[ok]]
        nh[s, s] = -1
    return nh


def _ports_for_graph(num_switches: int, hosts_per_switch: int, adj_offs, adj_cols):
    """Port map of a switch graph: ports 0..h-1 are hosts, then one port per
    neighbour in ascending id order.  Returns port_offs, port_peer, and a
    dict-free lookup port_of[s][neighbour] as a dense array."""
    S = num_switches
    deg = np.diff(adj_offs.astype(np.int64))
    nports = hosts_per_switch + deg
    port_offs = np.zeros(S + 1, np.int64)
    port_offs[1:] = np.cumsum(nports)
    peer = np.full(port_offs[-1], PEER_NONE, np.int64)
    port_to = {}
    for s in range(S):
        base = port_offs[s]
        for h in range(hosts_per_switch):
            peer[base + h] = HOST_BIT | (s * hosts_per_switch + h)
        for i, u in enumerate(adj_cols[adj_offs[s]:adj_offs[s + 1]]):
            port_to[(s, int(u))] = hosts_per_switch + i
    for s in range(S):
        base = port_offs[s]
        for i, u in enumerate(adj_cols[adj_offs[s]:adj_offs[s + 1]]):
            u = int(u)
            peer[base + hosts_per_switch + i] = (u << 8) | port_to[(u, s)]
    return port_offs.astype(np.uint32), peer.astype(np.int32), port_to


def _random_host_prefix(st: Stream, host_ip: np.ndarray, lens: np.ndarray) -> np.ndarray:
    """Prefix value = a random host's ip masked to the drawn length."""
    ips = host_ip[st.ints(0, len(host_ip) - 1, len(lens))].astype(np.uint64)
    mask = (np.uint64(0xFFFFFFFF) << (np.uint64(32) - lens.astype(np.uint64))) & np.uint64(0xFFFFFFFF)
    mask = np.where(lens == 0, np.uint64(0), mask)
    return (ips & mask).astype(np.uint32)


def _acl_fill(st: Stream, n: int, nports: int, host_ip: np.ndarray, *, src_len_range, dst_len_range,
              dport_width_max, p_any_in, p_drop, p_shadow, dport_max: int = 65535):
    """n ACL rules above routing priority; a fraction are shadowed copies of
    an earlier rule (narrower match, strictly lower priority).  Port ranges
    lie in [0, dport_max] (the draws are scaled into it when dport_max is
    below 65535, so the stream is consumed alike).  Returns the rule records
    and, per rule, the local index of the rule that shadows it (or -1)."""
    r = np.zeros(n, RULE_DTYPE)
    shadow_of = np.full(n, -1, np.int64)
    if n == 0:
        return r, shadow_of
    r["priority"] = st.ints(ROUTING_PRIORITY + 1, 65535, n)
    if src_len_range is None:
        r["src_len"] = 0
        r["src_ip"] = 0
    else:
        sl = st.ints(src_len_range[0], src_len_range[1], n)
        r["src_len"] = sl
        r["src_ip"] = _random_host_prefix(st, host_ip, sl)
    dl = st.ints(dst_len_range[0], dst_len_range[1], n)
    r["dst_len"] = dl
    r["dst_ip"] = _random_host_prefix(st, host_ip, dl)
    if dport_width_max is None:
        r["dport_lo"], r["dport_hi"] = 0, 65535
    else:
        lo = st.ints(0, 65535, n)
        w = st.ints(0, dport_width_max, n)
        if dport_max < 65535:
            lo = lo * (dport_max + 1) // 65536
        r["dport_lo"] = lo
        r["dport_hi"] = np.minimum(lo + w, dport_max)
    anyp = st.floats(n) < p_any_in
    r["in_port"] = np.where(anyp, ANY_PORT, st.ints(0, nports - 1, n))
    drop = st.floats(n) < p_drop
    r["action"] = np.where(drop, DROP, st.ints(0, nports - 1, n))
    # shadowed copies
    want = st.floats(n) < p_shadow
    pick = st.u64(n)
    extra = st.ints(0, 8, 2 * n).reshape(n, 2)
    shrink = st.floats(2 * n).reshape(n, 2)
    for i in np.nonzero(want)[0]:
        if i == 0:
            continue
        j = int(pick[i] % np.uint64(i))
        if r["priority"][j] <= ROUTING_PRIORITY + 1:
            continue
        c = r[j].copy()
        if src_len_range is not None:
            c["src_len"] = min(32, int(c["src_len"]) + int(extra[i, 0]))
        c["dst_len"] = min(32, int(c["dst_len"]) + int(extra[i, 1]))
        lo, hi = int(c["dport_lo"]), int(c["dport_hi"])
        lo2 = lo + int((hi - lo) * shrink[i, 0] * 0.5)
        hi2 = hi - int((hi - lo2) * shrink[i, 1] * 0.5)
        c["dport_lo"], c["dport_hi"] = lo2, max(lo2, hi2)
        c["priority"] = ROUTING_PRIORITY + 1 + int(pick[i] >> np.uint64(40)) % (int(r["priority"][j]) - ROUTING_PRIORITY - 1)
        c["action"] = r["action"][i]
        r[i] = c
        shadow_of[i] = j
    return r, shadow_of


def _assemble_tables(st: Stream, per_switch_rules, per_switch_shadow):
    """Concatenate per-switch rule lists after a seeded shuffle within each
    switch (so the loader's stable priority sort has real work to do)."""
    offs = [0]
    chunks, shadows = [], []
    for s, (r, sh) in enumerate(zip(per_switch_rules, per_switch_shadow)):
        perm = st.permutation(len(r))
        inv = np.empty_like(perm)
        inv[perm] = np.arange(len(perm))
        r2 = r[perm]
        sh2 = sh[perm]
        sh2 = np.where(sh2 >= 0, inv[np.maximum(sh2, 0)] + offs[-1], -1)
        chunks.append(r2)
        shadows.append(sh2)
        offs.append(offs[-1] + len(r2))
    return (np.array(offs, np.uint32), np.concatenate(chunks).astype(RULE_DTYPE),
            np.concatenate(shadows).astype(np.int32))


def _routing_rule(dst_ip: int, dst_len: int, action: int) -> np.ndarray:
    r = np.zeros(1, RULE_DTYPE)
    r["priority"] = ROUTING_PRIORITY
    r["in_port"] = ANY_PORT
    r["dst_ip"] = dst_ip
    r["dst_len"] = dst_len
    r["dport_lo"], r["dport_hi"] = 0, 65535
    r["action"] = action
    return r


def _ip(a, b, c, d) -> int:
    return (a << 24) | (b << 16) | (c << 8) | d


def _uniform_probes(st: Stream, host_ip: np.ndarray, m: int, mask_bits: int) -> np.ndarray:
    p = np.zeros(m, PROBE_DTYPE)
    H = len(host_ip)
    src = st.ints(0, H - 1, m)
    dst = st.ints(0, H - 1, m)
    p["src_host"] = src
    p["src_ip"] = host_ip[src]
    p["dst_ip"] = host_ip[dst]
    p["dport"] = st.ints(0, 65535, m)
    if mask_bits >= 32:
        p["allowed_mask"] = (st.u64(m) & np.uint64(0xFFFFFFFF)).astype(np.uint32)
    else:
        p["allowed_mask"] = (st.u64(m) % np.uint64(1 << mask_bits)).astype(np.uint32)
    return p


# ----------------------------------------------------------------------------
# recipe: tiny
# ----------------------------------------------------------------------------
def tiny(seed: int = 20260216, num_switches: int = 8, chords: int = 4, hosts_per_switch: int = 2,
         num_keys: int = 8, num_pods: int = 32, rules_per_switch: int = 64, num_probes: int = 1000,
         hop_cap: int = 16, num_regions: int = 4, p_absent: float = 0.0):
    """Ring of switches plus random chords; 2 hosts (= cluster nodes) per
    switch at 10.s.h.1; /16 routing by BFS next hop, /24 local delivery and a
    random dst-prefix fill; equality selectors over 8 label keys of which key
    0 is the region of the node's switch."""
    st = Stream(seed, "tiny")
    S = num_switches
    edges = {(i, (i + 1) % S) if i < (i + 1) % S else ((i + 1) % S, i) for i in range(S)}
    tries = 0
    while len(edges) < S + chords and tries < 1000:
        a, b = (int(x) for x in st.ints(0, S - 1, 2))
        tries += 1
        if a == b:
            continue
        edges.add((min(a, b), max(a, b)))
    edges = np.array(sorted(edges), np.int64)
    adj_offs, adj_cols = _csr_from_edges(S, edges)
    region = st.ints(0, num_regions - 1, S).astype(np.uint8)
    port_offs, port_peer, port_to = _ports_for_graph(S, hosts_per_switch, adj_offs, adj_cols)
    H = S * hosts_per_switch
    host_switch = (np.arange(H) // hosts_per_switch).astype(np.uint16)
    host_port = (np.arange(H) % hosts_per_switch).astype(np.uint16)
    host_ip = np.array([_ip(10, s, h, 1) for s in range(S) for h in range(hosts_per_switch)], np.uint32)
    nh = _next_hops(S, adj_offs, adj_cols)
    rules, shadows = [], []
    for s in range(S):
        nports = int(port_offs[s + 1] - port_offs[s])
        routing = [_routing_rule(_ip(10, d, 0, 0), 16, port_to[(s, int(nh[s, d]))]) for d in range(S) if d != s]
        routing += [_routing_rule(_ip(10, s, h, 0), 24, h) for h in range(hosts_per_switch)]
        routing = np.concatenate(routing)
        acl, sh = _acl_fill(st, rules_per_switch - len(routing), nports, host_ip,
                            src_len_range=None, dst_len_range=(8, 24), dport_width_max=None,
                            p_any_in=0.5, p_drop=0.2, p_shadow=0.0)
        rules.append(np.concatenate([routing, acl]))
        shadows.append(np.concatenate([np.full(len(routing), -1), np.where(sh >= 0, sh + len(routing), -1)]))
    rule_offs, all_rules, shadowed_by = _assemble_tables(st, rules, shadows)
    net = Network(S, rule_offs, all_rules, region, port_offs, port_peer, H, host_switch, host_port,
                  host_ip, shadowed_by, adj_offs, adj_cols)
    probes = Probes(_uniform_probes(st, host_ip, num_probes, num_regions), hop_cap)
    # cluster: one node per host
    N = H
    labels = st.ints(0, 15, num_keys * N).astype(np.uint16).reshape(num_keys, N)
    labels[0] = region[host_switch]
    if p_absent > 0:
        absent = st.floats(num_keys * N).reshape(num_keys, N) < p_absent
        labels[absent] = ABSENT
    cluster = Cluster(N, num_keys, labels.reshape(-1).copy())
    nexpr = st.ints(1, 3, num_pods)
    offs = np.zeros(num_pods + 1, np.uint32)
    offs[1:] = np.cumsum(nexpr)
    exprs = np.zeros(int(offs[-1]), EXPR_DTYPE)
    keyperm = st.u64(num_pods * num_keys).reshape(num_pods, num_keys)
    vals = st.ints(0, 17, int(offs[-1]))        # 16, 17 are carried by no node
    e = 0
    for p in range(num_pods):
        keys = np.argsort(keyperm[p], kind="stable")[: nexpr[p]]
        for k in keys:
            exprs[e]["key"] = k
            exprs[e]["op"] = OP_IN
            exprs[e]["nvals"] = 1
            v = int(vals[e]) if k != 0 else int(vals[e]) % (num_regions + 1)
            exprs[e]["vals"][:] = v
            e += 1
    assign = st.ints(0, N - 1, num_pods).astype(np.uint32)
    return dict(cluster=cluster, selectors=Selectors(num_pods, offs, exprs, assign), network=net, probes=probes)


# ----------------------------------------------------------------------------
# recipe: placement-scale selectors
# ----------------------------------------------------------------------------
def selector_workload(seed: int = 20260217, num_nodes: int = 5000, num_keys: int = 64,
                      num_values: int = 256, zipf_s: float = 1.1, num_pods: int = 100_000,
                      max_exprs: int = 8, p_absent: float = 0.0,
                      op_mix=(0.4, 0.3, 0.2, 0.1), p_unknown: float = 0.0,
                      with_doesnotexist: bool = False):
    """Dense label matrix with Zipf(s) value ids per key; pods with U[1,max]
    expressions on distinct keys: equality (In, 1 value) / In / NotIn / Exists
    by ``op_mix``; value sets of U[1,8] Zipf ids drawn without replacement;
    one uniform assignment per pod.  ``p_absent`` blanks labels; ``p_unknown``
    replaces a value by an id no node carries; ``with_doesnotexist`` turns
    half of the Exists into DoesNotExist (correctness variants)."""
    st = Stream(seed, "selectors")
    N, K = num_nodes, num_keys
    labels = st.zipf(zipf_s, num_values, N * K).astype(np.uint16).reshape(K, N)
    if p_absent > 0:
        absent = st.floats(N * K).reshape(K, N) < p_absent
        labels[absent] = ABSENT
    cluster = Cluster(N, K, labels.reshape(-1).copy())
    P = num_pods
    nexpr = st.ints(1, min(max_exprs, K), P)
    offs = np.zeros(P + 1, np.uint32)
    offs[1:] = np.cumsum(nexpr)
    E = int(offs[-1])
    exprs = np.zeros(E, EXPR_DTYPE)
    # distinct keys per pod: rank of per-(pod,key) random words
    pod_of = np.repeat(np.arange(P), nexpr)
    slot = np.arange(E) - offs[pod_of].astype(np.int64)
    rk = st.u64(P * K).reshape(P, K)
    keys_sorted = np.argsort(rk, axis=1, kind="stable")
    exprs["key"] = keys_sorted[pod_of, slot]
    u = st.floats(E)
    c = np.cumsum(op_mix)
    kind = np.searchsorted(c, u, side="right")          # 0 eq, 1 In, 2 NotIn, 3 Exists
    kind = np.minimum(kind, 3)
    op = np.array([OP_IN, OP_IN, OP_NOTIN, OP_EXISTS], np.uint8)[kind]
    if with_doesnotexist:
        flip = (kind == 3) & (st.floats(E) < 0.5)
        op = np.where(flip, OP_DOESNOTEXIST, op)
    exprs["op"] = op
    setsize = np.where(kind == 0, 1, st.ints(1, 8, E))
    setsize = np.where(kind == 3, 0, np.minimum(setsize, num_values))
    exprs["nvals"] = setsize
    cand = st.zipf(zipf_s, num_values, E * 32).reshape(E, 32)
    vals = np.zeros((E, 8), np.uint16)
    for e in range(E):
        n = int(setsize[e])
        if n == 0:
            continue
        _, first = np.unique(cand[e], return_index=True)
        distinct = cand[e][np.sort(first)][:n]
        if len(distinct) < n:
            rest = np.setdiff1d(np.arange(num_values), distinct)[: n - len(distinct)]
            distinct = np.concatenate([distinct, rest])
        vals[e, :n] = distinct
        vals[e, n:] = distinct[0]
    if p_unknown > 0:
        unk = (st.floats(E) < p_unknown) & (setsize > 0)
        vals[unk, 0] = num_values + 7
        for e in np.nonzero(unk)[0]:
            n = int(setsize[e])
            vals[e, n:] = vals[e, 0]
    exprs["vals"] = vals
    assign = st.ints(0, N - 1, P).astype(np.uint32)
    return dict(cluster=cluster, selectors=Selectors(P, offs, exprs, assign))


def selector_replicas(seed: int = 20260226, num_distinct: int = 10_000, num_pods: int = 100_000,
                      zipf_s: float = 1.1, **kw):
    """Pods whose selectors repeat, as the replicas of a deployment (or
    intents sharing a selector) do: ``num_distinct`` expression lists drawn
    as in selector_workload, each pod taking one of them by Zipf(s)
    popularity (list 0 the most common), written out in full per pod; one
    uniform assignment per pod."""
    d = selector_workload(seed=seed, num_pods=num_distinct, **kw)
    base = d["selectors"]
    st = Stream(seed, "replicas")
    pick = st.zipf(zipf_s, num_distinct, num_pods).astype(np.int64)   # ids 0 .. num_distinct - 1
    bo = base.expr_offs.astype(np.int64)
    n = np.diff(bo)[pick]
    offs = np.zeros(num_pods + 1, np.uint32)
    offs[1:] = np.cumsum(n)
    # expression k of pod p is expression k of its list
    src = bo[np.repeat(pick, n)] + (np.arange(int(n.sum())) - np.repeat(offs[:-1].astype(np.int64), n))
    exprs = base.exprs[src].copy()
    assign = st.ints(0, d["cluster"].num_nodes - 1, num_pods).astype(np.uint32)
    return dict(cluster=d["cluster"], selectors=Selectors(num_pods, offs, exprs, assign), pick=pick)


def selector_terms(seed: int = 20260222, num_nodes: int = 5000, num_keys: int = 64, num_values: int = 256,
                   num_pods: int = 100_000, max_terms: int = 3, max_exprs: int = 4, p_empty_term: float = 0.0,
                   **kw):
    """Pods with the node-affinity form: U[0, max_terms] selector terms each
    (ORed); every term is one pod of selector_workload's recipe (U[1,
    max_exprs] expressions on distinct keys, ANDed), or, with probability
    p_empty_term, a term without expressions.  One uniform assignment per pod."""
    st = Stream(seed, "selector-terms")
    nterm = st.ints(0, max_terms, num_pods)
    T = int(nterm.sum())
    d = selector_workload(seed=seed + 1, num_nodes=num_nodes, num_keys=num_keys, num_values=num_values,
                          num_pods=max(T, 1), max_exprs=max_exprs, **kw)
    c, sel = d["cluster"], d["selectors"]
    lens = np.diff(sel.expr_offs.astype(np.int64))[:T]
    lens = np.where(st.floats(T) < p_empty_term, 0, lens)
    keep = np.concatenate([np.arange(sel.expr_offs[t], sel.expr_offs[t] + lens[t]) for t in range(T)]) \
        if T else np.zeros(0, np.int64)
    term_offs = np.zeros(T + 1, np.uint32)
    term_offs[1:] = np.cumsum(lens)
    pod_terms = np.zeros(num_pods + 1, np.uint32)
    pod_terms[1:] = np.cumsum(nterm)
    assign = st.ints(0, num_nodes - 1, num_pods).astype(np.uint32)
    return dict(cluster=c, terms=SelectorTerms(num_pods, pod_terms, term_offs,
                                               sel.exprs[keep.astype(np.int64)].copy(), assign))


# ----------------------------------------------------------------------------
# recipe: fat-tree flow verification
# ----------------------------------------------------------------------------
def fat_tree(seed: int = 20260218, k: int = 16, rules_per_switch: int = 2000,
             num_probes: int = 10_000_000, hop_cap: int = 32, p_shadow: float = 0.05):
    """k-ary fat tree: (k/2)^2 core, k pods of k/2 aggregation and k/2 edge
    switches, k/2 hosts per edge at 10.pod.edge.(h+2).  Switch ids: core
    first, then aggregation, then edge.  Region = pod/2, core c -> c mod 8.
    Routing at priority 100 (edge: /32 local hosts and /24 per remote edge
    subnet up via aggregation (edge idx mod k/2); aggregation: /24 down per
    local edge, /24 up per remote subnet; core: /16 per pod) plus an ACL fill
    to ``rules_per_switch`` rules (src/dst prefixes /8-/32 of host
    addresses, dport ranges of width <= 1023, in_port ANY w.p. 0.75, drop
    20%), 5% of them shadowed copies."""
    st = Stream(seed, "fattree")
    h = k // 2
    n_core, n_agg, n_edge = h * h, k * h, k * h
    S = n_core + n_agg + n_edge
    core = lambda c: c
    agg = lambda p, j: n_core + p * h + j
    edge = lambda p, e: n_core + n_agg + p * h + e
    nports = np.zeros(S, np.int64)
    nports[:n_core] = k
    nports[n_core:] = k
    port_offs = np.zeros(S + 1, np.int64)
    port_offs[1:] = np.cumsum(nports)
    peer = np.full(port_offs[-1], PEER_NONE, np.int64)
    H = k * h * h
    host_switch = np.zeros(H, np.uint16)
    host_port = np.zeros(H, np.uint16)
    host_ip = np.zeros(H, np.uint32)
    hid = 0
    for p in range(k):
        for e in range(h):
            s = edge(p, e)
            for x in range(h):
                peer[port_offs[s] + x] = HOST_BIT | hid
                host_switch[hid], host_port[hid] = s, x
                host_ip[hid] = _ip(10, p, e, x + 2)
                hid += 1
            for j in range(h):
                a = agg(p, j)
                peer[port_offs[s] + h + j] = (a << 8) | e
                peer[port_offs[a] + e] = (s << 8) | (h + j)
        for j in range(h):
            a = agg(p, j)
            for c2 in range(h):
                c = j * h + c2
                peer[port_offs[a] + h + c2] = (core(c) << 8) | p
                peer[port_offs[core(c)] + p] = (a << 8) | (h + c2)
    region = np.zeros(S, np.uint8)
    region[:n_core] = np.arange(n_core) % 8
    for p in range(k):
        for j in range(h):
            region[agg(p, j)] = (p // 2) % 32
            region[edge(p, j)] = (p // 2) % 32
    rules, shadows = [], []
    for s in range(S):
        rt = []
        if s < n_core:
            for p in range(k):
                rt.append(_routing_rule(_ip(10, p, 0, 0), 16, p))
        elif s < n_core + n_agg:
            p, j = divmod(s - n_core, h)
            for e in range(h):
                rt.append(_routing_rule(_ip(10, p, e, 0), 24, e))
            for p2 in range(k):
                if p2 == p:
                    continue
                for e2 in range(h):
                    rt.append(_routing_rule(_ip(10, p2, e2, 0), 24, h + (e2 % h)))
        else:
            p, e = divmod(s - n_core - n_agg, h)
            for x in range(h):
                rt.append(_routing_rule(_ip(10, p, e, x + 2), 32, x))
            for p2 in range(k):
                for e2 in range(h):
                    if (p2, e2) == (p, e):
                        continue
                    rt.append(_routing_rule(_ip(10, p2, e2, 0), 24, h + (e2 % h)))
        rt = np.concatenate(rt)
        acl, sh = _acl_fill(st, max(0, rules_per_switch - len(rt)), int(nports[s]), host_ip,
                            src_len_range=(8, 32), dst_len_range=(8, 32), dport_width_max=1023,
                            p_any_in=0.75, p_drop=0.2, p_shadow=p_shadow)
        rules.append(np.concatenate([rt, acl]))
        shadows.append(np.concatenate([np.full(len(rt), -1), np.where(sh >= 0, sh + len(rt), -1)]))
    rule_offs, all_rules, shadowed_by = _assemble_tables(st, rules, shadows)
    net = Network(S, rule_offs, all_rules, region, port_offs.astype(np.uint32), peer.astype(np.int32),
                  H, host_switch, host_port, host_ip, shadowed_by)
    probes = Probes(_uniform_probes(st, host_ip, num_probes, 8), hop_cap)
    return dict(network=net, probes=probes)


# ----------------------------------------------------------------------------
# recipe: continuum WAN reachability
# ----------------------------------------------------------------------------
def continuum_wan(seed: int = 20260219, num_vertices: int = 4096, avg_degree: float = 6.0,
                  num_regions: int = 32, num_masks: int = 64, mask_pop=(4, 16),
                  num_sources: Optional[int] = None, kmeans_iters: int = 20):
    """Random geometric graph on U[0,1]^2 with radius giving the requested
    expected degree; components joined by their nearest cross-component pair
    (repeatedly, from the component of vertex 0); regions by Lloyd k-means
    (seeded initial centroids, ties to the lower centroid id); masks with
    U[lo,hi] distinct region bits; sources = all vertices unless limited."""
    st = Stream(seed, "wan")
    V = num_vertices
    xy = st.floats(2 * V).reshape(V, 2)
    r = np.sqrt(avg_degree / (np.pi * V))
    edges = []
    for i0 in range(0, V, 512):
        d2 = ((xy[i0:i0 + 512, None, :] - xy[None, :, :]) ** 2).sum(-1)
        ii, jj = np.nonzero(d2 < r * r)
        ii = ii + i0
        keep = ii < jj
        edges.append(np.stack([ii[keep], jj[keep]], 1))
    edges = np.concatenate(edges) if edges else np.zeros((0, 2), np.int64)
    from scipy.sparse import coo_matrix
    from scipy.sparse.csgraph import connected_components
    extra = []
    while True:
        allp = np.concatenate([edges] + ([np.array(extra)] if extra else []))
        g = coo_matrix((np.ones(len(allp)), (allp[:, 0], allp[:, 1])), shape=(V, V))
        ncomp, lab = connected_components(g, directed=False)
        if ncomp == 1:
            break
        inside = np.nonzero(lab == lab[0])[0]
        outside = np.nonzero(lab != lab[0])[0]
        best = (np.inf, -1, -1)
        for i0 in range(0, len(inside), 256):
            blk = inside[i0:i0 + 256]
            d2 = ((xy[blk, None, :] - xy[None, outside, :]) ** 2).sum(-1)
            a = np.unravel_index(np.argmin(d2), d2.shape)
            if d2[a] < best[0]:
                best = (d2[a], int(blk[a[0]]), int(outside[a[1]]))
        extra.append((min(best[1], best[2]), max(best[1], best[2])))
    allp = np.concatenate([edges] + ([np.array(extra)] if extra else []))
    offs, cols = _csr_from_edges(V, allp.astype(np.int64))
    # k-means regions
    cent = xy[st.permutation(V)[:num_regions]].copy()
    for _ in range(kmeans_iters):
        d2 = ((xy[:, None, :] - cent[None, :, :]) ** 2).sum(-1)
        lab = np.argmin(d2, axis=1)
        for c in range(num_regions):
            sel = lab == c
            if sel.any():
                cent[c] = xy[sel].mean(0)
    d2 = ((xy[:, None, :] - cent[None, :, :]) ** 2).sum(-1)
    region = np.argmin(d2, axis=1).astype(np.uint8)
    graph = Graph(V, offs, cols, region)
    masks = np.zeros(num_masks, np.uint32)
    pops = st.ints(mask_pop[0], mask_pop[1], num_masks)
    for i in range(num_masks):
        bits = st.permutation(num_regions)[: pops[i]]
        masks[i] = np.bitwise_or.reduce((np.uint64(1) << bits.astype(np.uint64))).astype(np.uint32)
    srcs = np.arange(V, dtype=np.uint32) if num_sources is None else st.ints(0, V - 1, num_sources).astype(np.uint32)
    return ReachQuery(graph, srcs, masks)


def random_digraph(seed: int, num_vertices: int, num_edges: int, num_regions: int = 8):
    """Directed random graph (for the general, non-symmetric reach path)."""
    st = Stream(seed, "digraph")
    V = num_vertices
    a = st.ints(0, V - 1, num_edges)
    b = st.ints(0, V - 1, num_edges)
    order = np.lexsort((b, a))
    a, b = a[order], b[order]
    offs = np.zeros(V + 1, np.int64)
    np.add.at(offs, a + 1, 1)
    return Graph(V, np.cumsum(offs).astype(np.uint32), b.astype(np.uint32),
                 st.ints(0, num_regions - 1, V).astype(np.uint8))


# ----------------------------------------------------------------------------
# recipe: end-to-end cross-layer
# ----------------------------------------------------------------------------
def end_to_end(seed: int = 20260220, num_switches: int = 512, avg_degree: float = 5.0,
               num_regions: int = 16, hosts_per_switch: int = 2, num_keys: int = 32,
               rules_per_switch: int = 1000, num_intents: int = 10_000, pods_per_intent: int = 4,
               probes_per_intent: int = 5000, hop_cap: int = 32, mask_pop=(2, 8), pass_share: float = 0.0):
    """Random switch graph (random spanning tree + uniform extra edges to the
    average degree), regions uniform, 2 hosts per switch (host n = cluster
    node n) at 10.(s>>8).(s&255).(h+1); /24 BFS routing to every other switch
    subnet, /32 local delivery, ACL fill as in the fat tree.  Intents: a
    region mask (U[lo,hi] regions), a selector whose first term is
    region In (the mask's regions) plus 0-3 equality/In terms on other keys
    (Zipf(1.1, 64) values), 4 pods placed by seeded choice among feasible
    nodes, and probes from the pods' hosts (round-robin) to uniform hosts.

    pass_share > 0 gives the variant in which intents can pass: the ACL
    rules' port ranges lie in [0, 49151], and a pass_share fraction of the
    intents (drawn from a stream of their own, so every other draw is that
    of the plain workload) permit every region (selector term region
    Exists) and send their flows to ports in [49152, 65535].  No ACL rule
    matches those flows, so the routing rules deliver each one along BFS
    next hops; such an intent passes when all its pods are placed."""
    st = Stream(seed, "e2e")
    S = num_switches
    perm = st.permutation(S)
    parent = st.u64(S)
    edges = set()
    for i in range(1, S):
        a, b = int(perm[i]), int(perm[int(parent[i] % np.uint64(i))])
        edges.add((min(a, b), max(a, b)))
    target = int(round(S * avg_degree / 2))
    while len(edges) < target:
        ab = st.ints(0, S - 1, 2 * (target - len(edges)) + 8).reshape(-1, 2)
        for a, b in ab:
            if a != b and len(edges) < target:
                edges.add((int(min(a, b)), int(max(a, b))))
    edges = np.array(sorted(edges), np.int64)
    adj_offs, adj_cols = _csr_from_edges(S, edges)
    region = st.ints(0, num_regions - 1, S).astype(np.uint8)
    port_offs, port_peer, port_to = _ports_for_graph(S, hosts_per_switch, adj_offs, adj_cols)
    H = S * hosts_per_switch
    host_switch = (np.arange(H) // hosts_per_switch).astype(np.uint16)
    host_port = (np.arange(H) % hosts_per_switch).astype(np.uint16)
    host_ip = np.array([_ip(10, s >> 8, s & 255, x + 1) for s in range(S) for x in range(hosts_per_switch)], np.uint32)
    nh = _next_hops(S, adj_offs, adj_cols)
    rules, shadows = [], []
    for s in range(S):
        nports = int(port_offs[s + 1] - port_offs[s])
        rt = [_routing_rule(_ip(10, d >> 8, d & 255, 0), 24, port_to[(s, int(nh[s, d]))])
              for d in range(S) if d != s and nh[s, d] >= 0]
        rt += [_routing_rule(int(host_ip[s * hosts_per_switch + x]), 32, x) for x in range(hosts_per_switch)]
        rt = np.concatenate(rt)
        acl, sh = _acl_fill(st, max(0, rules_per_switch - len(rt)), nports, host_ip,
                            src_len_range=(8, 32), dst_len_range=(8, 32), dport_width_max=1023,
                            p_any_in=0.75, p_drop=0.2, p_shadow=0.05,
                            dport_max=PASS_DPORT_LO - 1 if pass_share > 0 else 65535)
        rules.append(np.concatenate([rt, acl]))
        shadows.append(np.concatenate([np.full(len(rt), -1), np.where(sh >= 0, sh + len(rt), -1)]))
    rule_offs, all_rules, shadowed_by = _assemble_tables(st, rules, shadows)
    net = Network(S, rule_offs, all_rules, region, port_offs, port_peer, H, host_switch, host_port,
                  host_ip, shadowed_by, adj_offs, adj_cols)
    # cluster
    N, K = H, num_keys
    labels = st.zipf(1.1, 64, N * K).astype(np.uint16).reshape(K, N)
    labels[0] = region[host_switch]
    cluster = Cluster(N, K, labels.reshape(-1).copy())
    # intents
    I = num_intents
    masks = np.zeros(I, np.uint32)
    pops = st.ints(mask_pop[0], mask_pop[1], I)
    mperm = st.u64(I * num_regions).reshape(I, num_regions)
    extra_terms = st.ints(0, 3, I)
    offs = np.zeros(I + 1, np.uint32)
    offs[1:] = np.cumsum(1 + extra_terms)
    exprs = np.zeros(int(offs[-1]), EXPR_DTYPE)
    kperm = st.u64(I * (K - 1)).reshape(I, K - 1)
    tv = st.zipf(1.1, 64, int(offs[-1]) * 4).reshape(-1, 4)
    tkind = st.floats(int(offs[-1]))
    tsize = st.ints(2, 4, int(offs[-1]))
    for i in range(I):
        regs = np.argsort(mperm[i], kind="stable")[: pops[i]]
        masks[i] = int(np.bitwise_or.reduce(np.uint64(1) << regs.astype(np.uint64)))
        e = int(offs[i])
        exprs[e]["key"] = 0
        exprs[e]["op"] = OP_IN
        exprs[e]["nvals"] = len(regs)
        v = np.zeros(8, np.uint16)
        v[: len(regs)] = np.sort(regs)
        v[len(regs):] = v[0]
        exprs[e]["vals"] = v
        keys = np.argsort(kperm[i], kind="stable")[: extra_terms[i]] + 1
        for t, kk in enumerate(keys):
            e2 = e + 1 + t
            exprs[e2]["key"] = kk
            exprs[e2]["op"] = OP_IN
            if tkind[e2] < 0.7:
                vv = np.array([tv[e2, 0]])
            else:
                vv = np.unique(tv[e2, : tsize[e2]])
            exprs[e2]["nvals"] = len(vv)
            w = np.zeros(8, np.uint16)
            w[: len(vv)] = vv
            w[len(vv):] = vv[0]
            exprs[e2]["vals"] = w
    intents = Selectors(I, offs, exprs, None)
    draws = st.u64(I * pods_per_intent)
    # probes (src bound to placed pods later)
    M = I * probes_per_intent
    pr = np.zeros(M, PROBE_DTYPE)
    pr["src_host"] = NO_HOST
    pr["dst_ip"] = host_ip[st.ints(0, H - 1, M)]
    pr["dport"] = st.ints(0, 65535, M)
    if pass_share > 0:
        sp = Stream(seed, "e2e-pass")
        chosen = np.nonzero(sp.floats(I) < pass_share)[0]
        masks[chosen] = (1 << num_regions) - 1 if num_regions < 32 else 0xFFFFFFFF
        first = offs[chosen].astype(np.int64)
        exprs["op"][first] = OP_EXISTS
        exprs["nvals"][first] = 0
        exprs["vals"][first] = 0
        k = (chosen[:, None] * probes_per_intent + np.arange(probes_per_intent)[None, :]).reshape(-1)
        pr["dport"][k] = sp.ints(PASS_DPORT_LO, 65535, len(k))
    pr["allowed_mask"] = np.repeat(masks, probes_per_intent)
    return EndToEnd(cluster, intents, masks, pods_per_intent, draws, net, Probes(pr, hop_cap),
                    probes_per_intent)


def path_policies(seed: int, net: Network, num_policies: int, forbid_max: int = 2, must_max: int = 3,
                  hubs: int = 16, p_noop: float = 0.03) -> PathPolicies:
    """Path-constraint objects for a network: per policy up to forbid_max
    distinct forbidden switches drawn uniformly, U[0, must_max] waypoints
    drawn among the `hubs` switches with the most ports (the backbone that
    many paths cross), and with probability p_noop no concrete (src, dst)
    flow (the constraint applies to nothing)."""
    st = Stream(seed, "path-policies")
    S = net.num_switches
    hub = np.argsort(-np.diff(net.port_offs.astype(np.int64)), kind="stable")[: min(hubs, S)]
    want_f = st.ints(0, forbid_max, num_policies)
    nm = st.ints(0, min(must_max, len(hub)), num_policies)
    fkeys = st.u64(num_policies * max(forbid_max, 1)).reshape(num_policies, max(forbid_max, 1))
    mkeys = st.u64(num_policies * len(hub)).reshape(num_policies, len(hub))
    forbid_lists = [np.unique((fkeys[p, : want_f[p]] % np.uint64(S)).astype(np.int64)) for p in range(num_policies)]
    must_lists = [hub[np.argsort(mkeys[p], kind="stable")[: nm[p]]] for p in range(num_policies)]
    fo = np.zeros(num_policies + 1, np.uint32)
    fo[1:] = np.cumsum([len(f) for f in forbid_lists])
    mo = np.zeros(num_policies + 1, np.uint32)
    mo[1:] = np.cumsum(nm)
    forbid = np.concatenate(forbid_lists).astype(np.uint16) if num_policies else np.zeros(0, np.uint16)
    must = np.concatenate(must_lists).astype(np.uint16) if num_policies else np.zeros(0, np.uint16)
    concrete = (st.floats(num_policies) >= p_noop).astype(np.uint8)
    return PathPolicies(num_policies, fo, forbid, mo, must, concrete)


def path_requests(seed: int, net: Network, num_requests: int, num_policies: int = 0, extra_regions=(2, 8),
                  p_no_policy: float = 0.3, bad_hosts: int = 0) -> np.ndarray:
    """Scheduler requests with distinct (src, dst) host pairs: the mask
    permits the two endpoints' regions plus U[extra_regions] others; the
    policy is uniform over num_policies (or none with probability
    p_no_policy); the first bad_hosts requests name an absent host."""
    st = Stream(seed, "path-requests")
    H = net.num_hosts
    assert num_requests <= H * (H - 1)
    pairs = np.unique(st.u64(num_requests * 4) % np.uint64(H * H))
    pairs = pairs[(pairs // H) != (pairs % H)]
    pairs = pairs[st.permutation(len(pairs))][:num_requests]
    assert len(pairs) == num_requests
    req = np.zeros(num_requests, PATH_REQ_DTYPE)
    req["src_host"] = pairs // H
    req["dst_host"] = pairs % H
    reg = net.switch_region.astype(np.uint64)
    own = (np.uint64(1) << reg[net.host_switch[req["src_host"]]]) | (np.uint64(1) << reg[net.host_switch[req["dst_host"]]])
    nreg = int(reg.max()) + 1
    extra = np.zeros(num_requests, np.uint64)
    k = st.ints(extra_regions[0], extra_regions[1], num_requests)
    keys = st.u64(num_requests * nreg).reshape(num_requests, nreg)
    for r in range(num_requests):
        for g in np.argsort(keys[r], kind="stable")[: k[r]]:
            extra[r] |= np.uint64(1) << np.uint64(g)
    req["allowed_mask"] = ((own | extra) & np.uint64(0xFFFFFFFF)).astype(np.uint32)
    pol = st.ints(0, max(num_policies - 1, 0), num_requests).astype(np.uint32)
    none = (st.floats(num_requests) < p_no_policy) | (num_policies == 0)
    req["policy"] = np.where(none, NO_POLICY, pol)
    if bad_hosts:
        req["dst_host"][:bad_hosts] = 0xFFFF
    return req
