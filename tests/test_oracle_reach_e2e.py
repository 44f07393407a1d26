"""Pins for the oracle's compliant reach and end-to-end composition.

Reach is checked against brute-force simple-path enumeration on graphs of at
most 10 vertices, against connected components from a textbook union-find
(full mask on symmetric graphs), and against invariants: the source belongs
to its own row iff its region is permitted (Sec. 3.3: every vertex of a path,
the source included), symmetry on undirected graphs and monotonicity in the
mask.  Placement, probe binding and the per-intent verdict (Sec. 4.2 hybrid
coordination; Sec. 5.5 an intent passes only if all its checks pass) are
checked against closed forms and by composition.
"""
import itertools

import numpy as np
import pytest

import oracle
from paper_2602_16100_gb300 import workloads as W


def _members(row, n):
    return {i for i in range(n) if (int(row[i >> 5]) >> (i & 31)) & 1}


def _simple_path_reach(V, adj, region, s, mask):
    ok = lambda v: region[v] < 32 and (mask >> int(region[v])) & 1
    if not ok(s):
        return set()
    out = {s}

    def dfs(u, onpath):
        for v in adj[u]:
            if v < V and v not in onpath and ok(v):
                out.add(v)
                dfs(v, onpath | {v})

    dfs(s, {s})
    return out


@pytest.mark.parametrize("seed", range(6))
def test_reach_equals_simple_path_enumeration(seed):
    st = W.Stream(seed, "reach-brute")
    V = int(st.ints(2, 10, 1)[0])
    E = int(st.ints(0, 3 * V, 1)[0])
    a = st.ints(0, V - 1, E)
    b = st.ints(0, V - 1, E)
    if seed % 2 == 0:   # symmetric variant
        a, b = np.concatenate([a, b]), np.concatenate([b, a])
    order = np.lexsort((b, a))
    a, b = a[order], b[order]
    offs = np.zeros(V + 1, np.int64)
    np.add.at(offs, a + 1, 1)
    g = W.Graph(V, np.cumsum(offs).astype(np.uint32), b.astype(np.uint32), st.ints(0, 3, V).astype(np.uint8))
    masks = np.arange(16, dtype=np.uint32)
    src = np.arange(V, dtype=np.uint32)
    R = oracle.compliant_reach(g, src, masks)
    adj = [list(b[offs[u]:offs[u + 1]]) for u in range(V)] if False else \
        [list(g.cols[g.offs[u]:g.offs[u + 1]]) for u in range(V)]
    for m, s in itertools.product(range(16), range(V)):
        assert _members(R[m, s], V) == _simple_path_reach(V, adj, g.region, s, int(masks[m])), (m, s)


def _union_find_components(V, offs, cols):
    parent = list(range(V))

    def find(x):
        while parent[x] != x:
            parent[x] = parent[parent[x]]
            x = parent[x]
        return x

    for u in range(V):
        for v in cols[offs[u]:offs[u + 1]]:
            ru, rv = find(u), find(int(v))
            if ru != rv:
                parent[ru] = rv
    return [find(v) for v in range(V)]


def test_reach_invariants_on_continuum_wan_sample():
    q = W.continuum_wan(seed=3, num_vertices=600, num_masks=6, num_regions=12, mask_pop=(2, 6), num_sources=60)
    g = q.graph
    V = g.num_vertices
    full = np.array([0xFFFFFFFF], np.uint32)
    comp = _union_find_components(V, g.offs, g.cols)
    Rf = oracle.compliant_reach(g, q.sources, full)
    for j, s in enumerate(q.sources):
        assert _members(Rf[0, j], V) == {v for v in range(V) if comp[v] == comp[int(s)]}
    R = oracle.compliant_reach(g, np.arange(V, dtype=np.uint32), q.masks)
    for m in range(len(q.masks)):
        mask = int(q.masks[m])
        sets = [_members(R[m, s], V) for s in range(V)]
        for s in range(V):
            allowed = (mask >> int(g.region[s])) & 1
            assert (s in sets[s]) == bool(allowed) and (bool(sets[s]) == bool(allowed))
            for t in sets[s]:
                assert s in sets[t]                 # symmetric graph
        # monotone in the mask: adding a region only grows rows
        sup = mask | (1 << (m % 12))
        R2 = oracle.compliant_reach(g, np.arange(V, dtype=np.uint32), np.array([sup], np.uint32))
        for s in range(0, V, 7):
            assert sets[s] <= _members(R2[0, s], V)


def test_reach_pairs_and_out_of_range_inputs():
    q = W.continuum_wan(seed=4, num_vertices=200, num_masks=5)
    R = oracle.compliant_reach(q.graph, q.sources, q.masks)
    pairs = np.array([[m, s] for m in range(5) for s in range(0, 200, 13)], np.uint32)
    Rp = oracle.compliant_reach(q.graph, q.sources, q.masks, pairs=pairs)
    for i, (m, s) in enumerate(pairs):
        assert (Rp[i] == R[m, s]).all()
    # out-of-range source -> empty row; region >= 32 never entered
    g = W.Graph(3, np.array([0, 1, 2, 2], np.uint32), np.array([1, 2], np.uint32), np.array([0, 40, 0], np.uint8))
    R3 = oracle.compliant_reach(g, np.array([0, 7], np.uint32), np.array([0xFFFFFFFF], np.uint32))
    assert _members(R3[0, 0], 3) == {0} and not R3[0, 1].any()


@pytest.mark.parametrize("offs", [[0, 6, 2, 6], [0, 2, 4, 7], [1, 3, 2, 3]])
def test_reach_malformed_offsets_read_as_no_edges(offs):
    """Offsets that decrease or pass the edge count leave no usable edge
    list: every row is {s} for a permitted source (the closed form of a
    graph without edges), whatever well-formed rows the array also has."""
    cols = np.array([1, 2, 0, 2, 0, 1], np.uint32)
    region = np.array([0, 1, 0], np.uint8)
    g = W.Graph(3, np.array(offs, np.uint32), cols, region)
    masks = np.array([0xFFFFFFFF, 0b01], np.uint32)
    R = oracle.compliant_reach(g, np.arange(3, dtype=np.uint32), masks)
    for m, mask in enumerate(masks):
        for s in range(3):
            want = {s} if (int(mask) >> int(region[s])) & 1 else set()
            assert _members(R[m, s], 3) == want
    # the same arrays with well-formed offsets do have edges
    ok = oracle.compliant_reach(W.Graph(3, np.array([0, 2, 4, 6], np.uint32), cols, region),
                                np.arange(3, dtype=np.uint32), masks)
    assert _members(ok[0, 0], 3) == {0, 1, 2}


def test_placement_binding_and_verdict():
    st = W.Stream(5, "e2e-pins")
    G, N, pods = 50, 70, 4
    Wd = W.words_per_row(N)
    bits = np.zeros((G, Wd), np.uint32)
    feas = []
    for g in range(G):
        k = int(st.ints(0, N, 1)[0]) if g % 5 else (N if g % 10 else 0)
        f = sorted(set(st.ints(0, N - 1, k).tolist())) if k < N else list(range(N))
        feas.append(f)
        for n in f:
            bits[g, n >> 5] |= np.uint32(1 << (n & 31))
    draws = st.u64(G * pods)
    assign = oracle.place_pods(bits, N, pods, draws)
    for g in range(G):
        for j in range(pods):
            a = int(assign[g * pods + j])
            if not feas[g]:
                assert a == W.UNPLACED
            else:
                assert a == feas[g][int(draws[g * pods + j] % np.uint64(len(feas[g])))]
    # binding: round robin over the intent's pods
    ppg = 10
    probes = np.zeros(G * ppg, W.PROBE_DTYPE)
    host_ip = (np.arange(N, dtype=np.uint32) * 7 + 3).astype(np.uint32)
    bound = oracle.bind_probes(probes, ppg, pods, assign, host_ip)
    for k in range(G * ppg):
        a = int(assign[(k // ppg) * pods + (k % ppg) % pods])
        if a < N:
            assert bound[k]["src_host"] == a and bound[k]["src_ip"] == host_ip[a]
        else:
            assert bound[k]["src_host"] == W.NO_HOST
    # verdict: all pods OK, no unknown / bad flag, all probes compliant
    results = np.zeros(G * ppg, W.RESULT_DTYPE)
    results["status"] = W.ST_COMPLIANT
    results["status"][3 * ppg + 2] = W.ST_LOOP
    gflags = np.zeros(G, np.uint8)
    gflags[7] = W.F_UNKNOWN_VALUE
    gflags[8] = W.F_BAD_EXPR
    passed, counts = oracle.aggregate(bits, N, gflags, assign, pods, results, ppg)
    for g in range(G):
        want = bool(feas[g]) and g not in (3, 7, 8)
        assert bool(passed[g]) == want, g
        assert counts[g, :6].sum() == ppg and counts[g, 6] == (pods if feas[g] else 0) and counts[g, 7] == 0
    assert counts[3, W.ST_LOOP] == 1
