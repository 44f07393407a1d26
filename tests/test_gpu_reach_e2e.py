"""GPU parity of compliant reach and the end-to-end pipeline against the
oracle (bit-exact): random directed and symmetric graphs with ragged vertex
counts, malformed CSR reported by pv_sync, the continuum-WAN workload on
every (mask, source) row, and the end-to-end cross-layer pipeline
(selectors -> placement -> binding -> walks -> verdicts) on every output,
at full size, on the plain workload and on its variant in which intents
pass."""
import numpy as np
import pytest

import oracle
from paper_2602_16100_gb300 import binding as B
from paper_2602_16100_gb300 import workloads as W
from paper_2602_16100_gb300.validator import empty_device, flow_columns_of, to_device, to_numpy
import full_oracle as F
from gpu_util import E2E_PASS_SMALL

pytestmark = pytest.mark.gpu


def _gpu_reach(v, g, src, masks, words=None):
    dev = v.device
    words = words or W.words_per_row(g.num_vertices)
    out = v.compliant_reach(v.upload_graph(g), len(src), to_device(src.astype(np.uint32), dev), len(masks),
                            to_device(masks.astype(np.uint32), dev), words=words)
    v.sync()
    return to_numpy(out, np.uint32, (len(masks), len(src), words))


@pytest.mark.parametrize("V,E,seed", [(1, 0, 1), (37, 90, 2), (200, 900, 3), (1000, 3000, 4), (4097, 12000, 5)])
def test_random_digraphs(validator, V, E, seed):
    g = W.random_digraph(seed, V, E, num_regions=6)
    st = W.Stream(seed, "reach-test")
    src = st.ints(0, V - 1, 150).astype(np.uint32)
    masks = (st.u64(9) % np.uint64(64)).astype(np.uint32)
    masks[0] = 0xFFFFFFFF
    masks[1] = 0
    gr = _gpu_reach(validator, g, src, masks)
    orr = oracle.compliant_reach(g, src, masks)
    assert (gr == orr).all()


def test_symmetric_wan_small_all_sources(validator):
    q = W.continuum_wan(seed=7, num_vertices=700, num_masks=8, num_regions=12, mask_pop=(2, 8))
    gr = _gpu_reach(validator, q.graph, q.sources, q.masks, words=W.words_per_row(700) + 4)
    orr = oracle.compliant_reach(q.graph, q.sources, q.masks, words=W.words_per_row(700) + 4)
    assert (gr == orr).all()


def _symmetric(V, pairs, region):
    """CSR with both directions of every pair (host-side test helper)."""
    a = np.concatenate([pairs[:, 0], pairs[:, 1]]).astype(np.int64)
    b = np.concatenate([pairs[:, 1], pairs[:, 0]]).astype(np.int64)
    ab = np.unique(a * V + b)                       # sorted, no duplicate edges
    a, b = ab // V, ab % V
    offs = np.zeros(V + 1, np.int64)
    np.add.at(offs, a + 1, 1)
    return W.Graph(V, np.cumsum(offs).astype(np.uint32), b.astype(np.uint32), region.astype(np.uint8))


def _reach_both(v, g, src, masks, words=None):
    """Rows from the automatic path and from the sweeps alone, and whether
    the automatic path took the component shortcut."""
    auto = _gpu_reach(v, g, src, masks, words)
    used = B.pv_get_stat(v.ctx, B.PV_STAT_REACH_COMPONENTS)
    v.set_option(B.PV_OPT_REACH_KERNEL, 1)
    try:
        sweeps = _gpu_reach(v, g, src, masks, words)
        assert B.pv_get_stat(v.ctx, B.PV_STAT_REACH_COMPONENTS) == 0
    finally:
        v.set_option(B.PV_OPT_REACH_KERNEL, 0)
    return auto, sweeps, used


@pytest.mark.parametrize("V,E,seed", [(1, 0, 1), (37, 40, 2), (1000, 2500, 3), (4097, 9000, 4), (16384, 30000, 5)])
def test_symmetric_graphs_take_components(validator, V, E, seed):
    st = W.Stream(seed, "sym-reach")
    pairs = np.stack([st.ints(0, V - 1, E), st.ints(0, V - 1, E)], 1)
    g = _symmetric(V, pairs, st.ints(0, 7, V))
    src = st.ints(0, V - 1, 300).astype(np.uint32)
    src[:3] = [0, V - 1, V + 5]                      # ends and an out-of-range source
    masks = (st.u64(7) % np.uint64(256)).astype(np.uint32)
    masks[0], masks[1] = 0xFFFFFFFF, 0
    auto, sweeps, used = _reach_both(validator, g, src, masks)
    assert used == 1
    orr = oracle.compliant_reach(g, src, masks)
    assert (auto == orr).all() and (sweeps == orr).all()


def test_many_small_components_overflow_row_cache(validator):
    """Every source in its own or a two-vertex component: far more distinct
    components per block than row slots; plus padded rows (words_per_row
    well above ceil(V/32)) that shrink the cache."""
    V = 4096
    pairs = np.stack([np.arange(0, V, 2), np.arange(1, V, 2)], 1)[::2]
    g = _symmetric(V, pairs, np.arange(V) % 5)
    src = np.arange(V, dtype=np.uint32)[::-1].copy()
    masks = np.array([0xFFFFFFFF, 0b10110, 0b1], np.uint32)
    orr = oracle.compliant_reach(g, src, masks)
    auto, _, used = _reach_both(validator, g, src, masks)
    assert used == 1 and (auto == orr).all()
    words = W.words_per_row(V) + 1200
    auto, _, used = _reach_both(validator, g, src, masks, words)
    assert used == 1 and (auto == oracle.compliant_reach(g, src, masks, words=words)).all()


def test_asymmetric_or_high_degree_graphs_take_sweeps(validator):
    st = W.Stream(9, "asym-reach")
    V = 600
    pairs = np.stack([st.ints(0, V - 1, 1500), st.ints(0, V - 1, 1500)], 1)
    g = _symmetric(V, pairs, st.ints(0, 5, V))
    # drop one reverse edge: one direction of the first non-loop pair remains
    k = int(np.nonzero(g.cols[: g.offs[-1]] != np.repeat(np.arange(V), np.diff(g.offs)))[0][0])
    u = int(np.searchsorted(g.offs, k, side="right") - 1)
    cols = np.delete(g.cols, k)
    offs = g.offs.copy()
    offs[u + 1:] -= 1
    one_way = W.Graph(V, offs, cols, g.region)
    # a hub with more out-edges than the symmetry check scans
    hub = np.stack([np.zeros(100, np.int64), np.arange(1, 101)], 1)
    star = _symmetric(V, np.concatenate([pairs, hub]), g.region)
    src = np.arange(0, V, 3, dtype=np.uint32)
    masks = np.array([0xFFFFFFFF, 0b111, 0b101010], np.uint32)
    for graph in (one_way, star):
        auto, sweeps, used = _reach_both(validator, graph, src, masks)
        assert used == 0
        orr = oracle.compliant_reach(graph, src, masks)
        assert (auto == orr).all() and (sweeps == orr).all()


def test_malformed_csr_is_reported(validator):
    g = W.random_digraph(3, 50, 200)
    cols = g.cols.copy()
    cols[7] = 50                      # out of range neighbour: skipped, reported
    bad = W.Graph(50, g.offs, cols, g.region)
    dev = validator.device
    src = np.arange(50, dtype=np.uint32)
    masks = np.array([0xFFFFFFFF], np.uint32)
    out = validator.compliant_reach(validator.upload_graph(bad), 50, to_device(src, dev), 1, to_device(masks, dev))
    with pytest.raises(B.PVError) as e:
        validator.sync()
    assert e.value.code == B.PV_EINVAL
    validator.sync()                  # error was cleared
    # skipping the bad edge gives the oracle's answer (it never enters it either)
    got = to_numpy(out, np.uint32, (1, 50, W.words_per_row(50)))
    assert (got == oracle.compliant_reach(bad, src, masks)).all()
    with pytest.raises(B.PVError):
        B.pv_compliant_reach(validator.ctx, 0, 0, 0, 0, 0, 1, 0, 1, 0, 0, 4)


@pytest.mark.parametrize("kernel", [0, 1])
def test_overlapping_offsets_read_as_no_edges(validator, kernel):
    """Offsets that go back down let well-formed rows overlap (rows 0, 2, 4,
    ... all cover every edge), so their lengths add up to many times the
    edge count.  The call reports PV_EINVAL, writes nothing past the edge
    arrays, and gives the oracle's rows for a graph without edges, on the
    component path (kernel 0) and on the sweeps (kernel 1)."""
    V, E = 64, 300
    g0 = W.random_digraph(35, V, E)
    offs = np.where(np.arange(V + 1) % 2 == 0, 0, E).astype(np.uint32)
    bad = W.Graph(V, offs, g0.cols, g0.region)
    src = np.arange(V, dtype=np.uint32)
    masks = np.array([0xFFFFFFFF, 0b1011, 0], np.uint32)
    want = oracle.compliant_reach(bad, src, masks)
    assert (want.sum(axis=(0, 1)) != 0).any()
    dev = validator.device
    validator.set_option(B.PV_OPT_REACH_KERNEL, kernel)
    try:
        out = validator.compliant_reach(validator.upload_graph(bad), V, to_device(src, dev), len(masks),
                                        to_device(masks, dev))
        with pytest.raises(B.PVError) as e:
            validator.sync()
        assert e.value.code == B.PV_EINVAL
        validator.sync()
    finally:
        validator.set_option(B.PV_OPT_REACH_KERNEL, 0)
    got = to_numpy(out, np.uint32, want.shape)
    assert (got == want).all()


def test_continuum_wan_full_size(validator):
    """The continuum-WAN workload (4,096 sources x 64 masks) in the
    benchmark's launch configuration; every row is compared."""
    q = W.continuum_wan()
    gr = _gpu_reach(validator, q.graph, q.sources, q.masks)
    want = F.cached("continuum-wan/default", lambda: {"r": F.compliant_reach(q.graph, q.sources, q.masks)})["r"]
    assert (gr == want).all()
    assert B.pv_get_stat(validator.ctx, B.PV_STAT_REACH_COMPONENTS) == 1


def _run_e2e(v, e):
    v.load_cluster(e.cluster)
    v.load_network(e.network)
    dev, sizes = v.alloc_end_to_end(e)
    v.run_end_to_end(dev, sizes)
    I, pods, ppg = sizes["intents"], sizes["pods"], sizes["probes_per_intent"]
    # the pipeline does not return the bound records: bind them once more
    B.pv_bind_flows(v.ctx, I * ppg, dev["flows"], ppg, pods, dev["assign"], dev["masks"], dev["probes"])
    v.sync()
    words = W.words_per_row(e.cluster.num_nodes)
    return {
        "bits": to_numpy(dev["bits"], np.uint32, (I, words)),
        "flags": to_numpy(dev["flags"], np.uint8),
        "assign": to_numpy(dev["assign"], np.uint32),
        "probes": to_numpy(dev["probes"], W.PROBE_DTYPE),
        "results": to_numpy(dev["results"], W.RESULT_DTYPE),
        "pass": to_numpy(dev["pass"], np.uint8),
        "counts": to_numpy(dev["counts"], np.uint32, (I, 8)),
    }


def _oracle_e2e(e, idx_probes=None):
    c = e.cluster
    bits, flags = oracle.eval_selectors(c.num_nodes, c.num_keys, c.labels, e.intents.expr_offs, e.intents.exprs)
    assign = oracle.place_pods(bits, c.num_nodes, e.pods_per_intent, e.place_draws)
    probes = oracle.bind_probes(e.probes.probes, e.probes_per_intent, e.pods_per_intent, assign, e.network.host_ip)
    return bits, flags, assign, probes


def test_end_to_end_small(validator):
    e = W.end_to_end(seed=21, num_switches=64, num_intents=300, probes_per_intent=200, rules_per_switch=200)
    g = _run_e2e(validator, e)
    bits, flags, assign, probes = _oracle_e2e(e)
    assert (g["bits"] == bits).all() and (g["flags"] == flags).all() and (g["assign"] == assign).all()
    assert (g["probes"] == probes).all()
    res = oracle.verify_probes(e.network, probes, e.probes.hop_cap)
    assert (g["results"] == res).all()
    passed, counts = oracle.aggregate(bits, e.cluster.num_nodes, flags, assign, e.pods_per_intent, res,
                                      e.probes_per_intent)
    assert (g["pass"] == passed).all() and (g["counts"] == counts).all()


def _check_e2e_full(g, e, key, pol=None):
    """Every output of a GPU end-to-end run against the oracle pipeline
    (sharded over the host cores, cached): selector rows and flags,
    placement, bound probe records, walk results, verdicts and counts."""
    def compute():
        out = F.end_to_end(e, pol)
        out.pop("probes")                  # rebuilt below: cheap, and large to store
        return out
    want = F.cached(key, compute)
    assert (g["bits"] == want["bits"]).all() and (g["flags"] == want["flags"]).all()
    assert (g["assign"] == want["assign"]).all()
    if "probes" in g:
        probes = oracle.bind_probes(e.probes.probes, e.probes_per_intent, e.pods_per_intent, want["assign"],
                                    e.network.host_ip)
        assert (g["probes"] == probes).all()
    assert (g["results"] == want["results"]).all()
    if pol is not None:
        assert (g["hits"] == want["hits"]).all()
    assert (g["counts"] == want["counts"]).all()
    assert (g["pass"] == want["passed"]).all()
    return want


def test_end_to_end_full_size(validator):
    """The full end-to-end workload (10,000 intents, 50M probes) in the
    benchmark's launch configuration; every output is compared."""
    e = W.end_to_end()
    g = _run_e2e(validator, e)
    want = _check_e2e_full(g, e, "end-to-end/default")
    assert want["counts"][:, W.ST_COMPLIANT].sum() > 0


@pytest.mark.parametrize("size", ["small", "full"])
def test_end_to_end_with_passing_intents(validator, size):
    """The end-to-end variant in which intents can pass (a share of the
    intents permit every region and send flows on ports no ACL rule
    covers): every output matches the oracle, and at least a tenth of the
    intents pass, so the verdict's positive branch is compared too."""
    e = W.end_to_end(pass_share=0.3) if size == "full" else W.end_to_end(**E2E_PASS_SMALL)
    g = _run_e2e(validator, e)
    want = _check_e2e_full(g, e, f"end-to-end-pass/{size}")
    assert want["passed"].mean() >= 0.1
    assert (want["passed"] == 0).any()


def _pinned(a):
    import torch
    return torch.from_numpy(np.ascontiguousarray(a).view(np.uint8).reshape(-1).copy()).pin_memory()


@pytest.mark.parametrize("chunks", [1, 3, 7])
def test_end_to_end_pipelined_from_host(validator, chunks):
    """Host-buffer pipeline (probe upload of range c overlapped with the
    verification of range c-1) gives the oracle's verdicts; the device
    input buffers are zeroed first, so only the host copies can supply them."""
    import torch
    e = W.end_to_end(seed=22, num_switches=64, num_intents=301, probes_per_intent=120, rules_per_switch=200,
                     pass_share=0.3)
    validator.load_cluster(e.cluster)
    validator.load_network(e.network)
    dev, sizes = validator.alloc_end_to_end(e)
    for k in ("offs", "exprs", "draws", "masks", "dst", "dport", "flows", "probes"):
        dev[k].zero_()
    I = e.intents.num_pods
    host = {"offs": _pinned(e.intents.expr_offs.astype(np.uint32)), "exprs": _pinned(e.intents.exprs),
            "draws": _pinned(e.place_draws.astype(np.uint64)), "masks": _pinned(e.intent_mask.astype(np.uint32)),
            "dst": _pinned(flow_columns_of(e)[0]), "dport": _pinned(flow_columns_of(e)[1]),
            "pass": torch.zeros(I, dtype=torch.uint8).pin_memory(),
            "counts": torch.zeros(I * 32, dtype=torch.uint8).pin_memory()}
    stream = torch.cuda.current_stream()
    # with 3 chunks the tables are reloaded while the inputs upload
    loads = (lambda: (validator.load_cluster(e.cluster), validator.load_network(e.network))) if chunks == 3 else None
    validator.run_end_to_end_from_host(host, dev, sizes, stream, torch.cuda.Stream(), chunks, loads)
    stream.synchronize()
    validator.sync()
    bits, flags, assign, probes = _oracle_e2e(e)
    res = oracle.verify_probes(e.network, probes, e.probes.hop_cap)
    passed, counts = oracle.aggregate(bits, e.cluster.num_nodes, flags, assign, e.pods_per_intent, res,
                                      e.probes_per_intent)
    words = W.words_per_row(e.cluster.num_nodes)
    assert (to_numpy(dev["bits"], np.uint32, (I, words)) == bits).all()
    assert (to_numpy(dev["results"], W.RESULT_DTYPE) == res).all()
    assert (host["pass"].numpy() == passed).all()
    assert (host["counts"].numpy().view(np.uint32).reshape(I, 8) == counts).all()
    assert passed.any()


@pytest.mark.parametrize("loads_first,two_part", [(False, False), (False, True), (True, False), (True, True)])
def test_back_to_back_host_steps_each_with_its_own_tables(validator, loads_first, two_part):
    """Three host-buffer steps enqueued back to back with no synchronisation,
    each loading its own cluster and flow tables (in one call, or in two
    halves around the queued uploads) and verifying its own batch (batches
    A, B, A): the alternating input buffers and the loads that retire the
    replaced state only after its last use give every step the oracle's
    verdicts for its batch."""
    import torch
    kw = dict(num_switches=48, num_intents=160, probes_per_intent=90, rules_per_switch=150, pass_share=0.3)
    ea, eb = W.end_to_end(seed=31, **kw), W.end_to_end(seed=32, **kw)
    big = ea if len(ea.intents.exprs) >= len(eb.intents.exprs) else eb
    v = validator
    v.load_cluster(big.cluster)
    dev, _ = v.alloc_end_to_end(big)

    def sizes(e):
        return {"intents": e.intents.num_pods, "pods": e.pods_per_intent, "probes_per_intent": e.probes_per_intent,
                "num_exprs": len(e.intents.exprs), "hop_cap": e.probes.hop_cap}

    def host(e):
        I = e.intents.num_pods
        return {"offs": _pinned(e.intents.expr_offs.astype(np.uint32)), "exprs": _pinned(e.intents.exprs),
                "draws": _pinned(e.place_draws.astype(np.uint64)), "masks": _pinned(e.intent_mask.astype(np.uint32)),
                "dst": _pinned(flow_columns_of(e)[0]), "dport": _pinned(flow_columns_of(e)[1]), "pass": torch.zeros(I, dtype=torch.uint8).pin_memory(),
                "counts": torch.zeros(I * 32, dtype=torch.uint8).pin_memory()}

    def loads(e):
        v.load_cluster(e.cluster)
        if not two_part:
            v.load_network(e.network)
            return None
        v.begin_network(e.network)
        return v.finish_network

    stream, cs = torch.cuda.current_stream(), torch.cuda.Stream()
    steps = [(ea, host(ea)), (eb, host(eb)), (ea, host(ea))]
    for e, h in steps:
        v.run_end_to_end_from_host(h, dev, sizes(e), stream, cs, 2 if loads_first else 1, lambda e=e: loads(e),
                                   loads_first=loads_first)
    stream.synchronize()
    v.sync()
    for e, h in steps:
        bits, flags, assign, probes = _oracle_e2e(e)
        res = oracle.verify_probes(e.network, probes, e.probes.hop_cap)
        passed, counts = oracle.aggregate(bits, e.cluster.num_nodes, flags, assign, e.pods_per_intent, res,
                                          e.probes_per_intent)
        I = e.intents.num_pods
        assert (h["pass"].numpy() == passed).all()
        assert (h["counts"].numpy().view(np.uint32).reshape(I, 8) == counts).all()
    c = [h["counts"].numpy() for _, h in steps]
    assert (c[0] == c[2]).all() and not (c[0] == c[1]).all()   # the batches differ; A twice alike


def test_failed_table_load_keeps_the_loaded_tables(validator):
    """A load that fails validation leaves the previously loaded tables in
    place: walks after it give the same results as before it."""
    d = W.tiny()
    net, pr = d["network"], d["probes"].probes
    v = validator
    v.load_network(net)
    first = to_numpy(v.verify_probes(to_device(pr, v.device), len(pr), 16), W.RESULT_DTYPE)
    bad = net.rules.copy()
    bad[5]["dst_len"] = 40
    with pytest.raises(B.PVError) as e:
        B.pv_load_flow_tables(v.ctx, net.num_switches, net.rule_offs, bad, net.switch_region, net.port_offs,
                              net.port_peer, net.num_hosts, net.host_switch, net.host_port, net.host_ip)
    assert e.value.code == B.PV_EINVAL
    again = to_numpy(v.verify_probes(to_device(pr, v.device), len(pr), 16), W.RESULT_DTYPE)
    v.sync()
    assert (again == first).all()
    assert (first == oracle.verify_probes(net, pr, 16)).all()


def test_two_part_table_load(validator):
    """Between pv_load_flow_tables_begin and _end, walks use the tables
    installed before the begin; after the end, the new ones.  A second begin,
    a one-part load in between, or an end with nothing begun are refused."""
    a, b = W.tiny(seed=41)["network"], W.tiny(seed=42)["network"]
    pr = W.tiny(seed=41)["probes"].probes
    v = validator
    v.load_network(a)
    d_pr = to_device(pr, v.device)
    want_a, want_b = oracle.verify_probes(a, pr, 16), oracle.verify_probes(b, pr, 16)
    assert not (want_a == want_b).all()
    v.begin_network(b)
    try:
        mid = to_numpy(v.verify_probes(d_pr, len(pr), 16), W.RESULT_DTYPE)
        for call in (lambda: v.begin_network(b), lambda: v.load_network(b)):
            with pytest.raises(B.PVError) as e:
                call()
            assert e.value.code == B.PV_ESTATE
    finally:
        v.finish_network()
    after = to_numpy(v.verify_probes(d_pr, len(pr), 16), W.RESULT_DTYPE)
    v.sync()
    assert (mid == want_a).all()
    assert (after == want_b).all()
    with pytest.raises(B.PVError) as e:
        v.finish_network()
    assert e.value.code == B.PV_ESTATE


def test_two_part_load_with_a_bad_rule_keeps_the_tables(validator):
    """A rule field out of range is found by the device pass; the begin
    succeeds, the end reports PV_EINVAL and the installed tables stay."""
    d = W.tiny()
    net, pr = d["network"], d["probes"].probes
    v = validator
    v.load_network(net)
    bad = net.rules.copy()
    bad[5]["dst_len"] = 40
    B.pv_load_flow_tables_begin(v.ctx, net.num_switches, net.rule_offs, bad, net.switch_region, net.port_offs,
                                net.port_peer, net.num_hosts, net.host_switch, net.host_port, net.host_ip)
    with pytest.raises(B.PVError) as e:
        B.pv_load_flow_tables_end(v.ctx)
    assert e.value.code == B.PV_EINVAL
    got = to_numpy(v.verify_probes(to_device(pr, v.device), len(pr), 16), W.RESULT_DTYPE)
    v.sync()
    assert (got == oracle.verify_probes(net, pr, 16)).all()
    v.load_network(net)   # nothing left in progress


def test_flow_binding_and_fused_walk(validator):
    """pv_bind_flows builds the oracle's bound probe records from 8-byte
    flows; pv_verify_flows (binding inside the walk's first kernel) gives the
    records and results of pv_bind_flows followed by pv_verify_probes."""
    e = W.end_to_end(seed=27, num_switches=64, num_intents=120, probes_per_intent=90, rules_per_switch=150)
    v = validator
    v.load_cluster(e.cluster)
    v.load_network(e.network)
    dev, sizes = v.alloc_end_to_end(e)
    I, pods, ppg = sizes["intents"], sizes["pods"], sizes["probes_per_intent"]
    words = W.words_per_row(e.cluster.num_nodes)
    B.pv_eval_selectors(v.ctx, I, dev["offs"], sizes["num_exprs"], dev["exprs"], None, dev["bits"], words, dev["flags"])
    B.pv_place_pods(v.ctx, I, pods, dev["bits"], words, dev["draws"], dev["assign"])
    M = I * ppg
    p1 = empty_device(M * 16, v.device)
    B.pv_bind_flows(v.ctx, M, dev["flows"], ppg, pods, dev["assign"], dev["masks"], p1)
    r1 = empty_device(M * 4, v.device)
    B.pv_verify_probes(v.ctx, M, p1, sizes["hop_cap"], r1)
    p2 = empty_device(M * 16, v.device)
    r2 = empty_device(M * 4, v.device)
    B.pv_verify_flows(v.ctx, M, dev["flows"], ppg, pods, dev["assign"], dev["masks"], sizes["hop_cap"], p2, r2)
    v.sync()
    _, _, assign, probes = _oracle_e2e(e)
    assert (to_numpy(p1, W.PROBE_DTYPE) == probes).all() and (to_numpy(p2, W.PROBE_DTYPE) == probes).all()
    res = oracle.verify_probes(e.network, probes, e.probes.hop_cap)
    assert (to_numpy(r1, W.RESULT_DTYPE) == res).all() and (to_numpy(r2, W.RESULT_DTYPE) == res).all()
