"""The sharded oracle runner used by the full-size parity tests gives
exactly the single-call oracle's outputs (ranges cut at ragged sizes, more
ranges than units, one unit), and its disk cache returns what it stored
and keys on its inputs."""
import numpy as np
import pytest

import full_oracle as F
import oracle
from paper_2602_16100_gb300 import workloads as W


def test_sharded_selectors_walks_and_reach_equal_one_call():
    d = W.selector_workload(seed=3, num_nodes=333, num_keys=12, num_values=20, num_pods=1001)
    c, sel = d["cluster"], d["selectors"]
    words = W.words_per_row(c.num_nodes)
    b1, f1 = oracle.eval_selectors(c.num_nodes, c.num_keys, c.labels, sel.expr_offs, sel.exprs, sel.assign,
                                   words=words)
    b2, f2 = F.eval_selectors(c, sel, words)
    assert (b1 == b2).all() and (f1 == f2).all()
    t = W.fat_tree(seed=4, k=4, rules_per_switch=90, num_probes=3001, hop_cap=12)
    net, pr = t["network"], t["probes"].probes
    assert (F.verify_probes(net, pr, 12) == oracle.verify_probes(net, pr, 12)).all()
    assert (F.verify_probes(net, pr[:1], 12) == oracle.verify_probes(net, pr[:1], 12)).all()
    pol = W.path_policies(5, net, 31, forbid_max=2, must_max=2, hubs=6)
    r1, h1 = oracle.verify_constrained(net, pr, 12, pol, probes_per_policy=97)
    r2, h2 = F.verify_constrained(net, pr, 12, pol, 97)
    assert (r1 == r2).all() and (h1 == h2).all()
    q = W.continuum_wan(seed=6, num_vertices=300, num_masks=7, num_sources=41)
    assert (F.compliant_reach(q.graph, q.sources, q.masks) == oracle.compliant_reach(q.graph, q.sources,
                                                                                      q.masks)).all()


@pytest.mark.parametrize("with_policies", [False, True])
def test_sharded_end_to_end_equals_the_plain_pipeline(with_policies):
    e = W.end_to_end(seed=7, num_switches=40, num_intents=90, probes_per_intent=61, rules_per_switch=120,
                     pass_share=0.3)
    pol = W.path_policies(8, e.network, 90, forbid_max=1, must_max=1, hubs=4) if with_policies else None
    got = F.end_to_end(e, pol)
    c = e.cluster
    bits, flags = oracle.eval_selectors(c.num_nodes, c.num_keys, c.labels, e.intents.expr_offs, e.intents.exprs)
    assign = oracle.place_pods(bits, c.num_nodes, e.pods_per_intent, e.place_draws)
    probes = oracle.bind_probes(e.probes.probes, e.probes_per_intent, e.pods_per_intent, assign, e.network.host_ip)
    if pol is None:
        res = oracle.verify_probes(e.network, probes, e.probes.hop_cap)
        passed, counts = oracle.aggregate(bits, c.num_nodes, flags, assign, e.pods_per_intent, res,
                                          e.probes_per_intent)
    else:
        res, hits = oracle.verify_constrained(e.network, probes, e.probes.hop_cap, pol,
                                              probes_per_policy=e.probes_per_intent)
        passed, counts = oracle.aggregate_constrained(bits, c.num_nodes, flags, assign, e.pods_per_intent, res,
                                                      e.probes_per_intent, hits, pol)
        assert (got["hits"] == hits).all()
    for k, want in (("bits", bits), ("flags", flags), ("assign", assign), ("probes", probes), ("results", res),
                    ("passed", passed), ("counts", counts)):
        assert (got[k] == want).all(), k
    assert passed.any()


def test_cache_round_trip_and_keys(tmp_path, monkeypatch):
    monkeypatch.setenv("PV_ORACLE_CACHE", str(tmp_path))
    calls = []

    def compute(v):
        calls.append(v)
        return {"x": np.arange(5) * v}

    a = F.cached("k1", lambda: compute(2))
    b = F.cached("k1", lambda: compute(3))        # served from disk: not recomputed
    c = F.cached("k2", lambda: compute(3))        # another key
    assert calls == [2, 3]
    assert (a["x"] == b["x"]).all() and (c["x"] == np.arange(5) * 3).all()
    monkeypatch.setenv("PV_ORACLE_CACHE", "off")
    F.cached("k1", lambda: compute(4))
    assert calls == [2, 3, 4]
