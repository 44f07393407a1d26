"""Pins for the oracle's path-constraint checks (Sec. 4.2 constraint object
with forbidden and must_go switches; Sec. 5.3 waypoint intent; Sec. 5.5
network checks; Sec. 6.3 failure mode 2, the no-op policy).

The constrained walk is checked against a path recorded without any
constraint and judged afterwards (netbuild.trace_walk_constrained), on
hand-built worked cases and on random networks with random policies; the
verdict against closed forms over results, waypoint bits and the no-op flag.
"""
import numpy as np
import pytest

import oracle
from paper_2602_16100_gb300 import workloads as W
from netbuild import ip, make_net, probe, rule, trace_walk_constrained


def _policies(forbid_lists, must_lists, concrete=None):
    P = len(forbid_lists)
    fo = np.zeros(P + 1, np.uint32)
    fo[1:] = np.cumsum([len(f) for f in forbid_lists])
    mo = np.zeros(P + 1, np.uint32)
    mo[1:] = np.cumsum([len(m) for m in must_lists])
    cat = lambda ls: np.array([x for l in ls for x in l], np.uint16)
    cc = np.ones(P, np.uint8) if concrete is None else np.array(concrete, np.uint8)
    return W.PathPolicies(P, fo, cat(forbid_lists), mo, cat(must_lists), cc)


def _backup_switch_net(via_backup):
    """Hosts h2 on switch 2 and h4 on switch 4; switch 2 reaches switch 4
    either through the backup switch 8 or through switch 5.  Switch ids are
    dense 0..8 (0, 1, 3, 6, 7 are idle); switch 6 sits in region 1."""
    H2, H4 = ip(10, 0, 2, 1), ip(10, 0, 4, 1)
    nports = [1] * 9
    nports[2], nports[4], nports[5], nports[8] = 3, 3, 2, 2
    links = [(2, 1, 8, 0), (8, 1, 4, 1), (2, 2, 5, 0), (5, 1, 4, 2)]
    hosts = [(2, 0, H2), (4, 0, H4)]
    region = [0] * 9
    region[6] = 1
    out2 = 1 if via_backup else 2
    rules = [[] for _ in range(9)]
    rules[2] = [rule(100, H4, 32, out2), rule(100, H2, 32, 0)]
    rules[8] = [rule(100, H4, 32, 1), rule(100, H2, 32, 0)]
    rules[5] = [rule(100, H4, 32, 1), rule(100, H2, 32, 0)]
    rules[4] = [rule(100, H4, 32, 0), rule(100, H2, 32, 1 if via_backup else 2)]
    return make_net(nports, links, hosts, region, rules), H2, H4


def test_waypoint_worked_case():
    """Sec. 5.3 networking intent: traffic from host 2 to host 4 must traverse
    the backup switch (here switch 8)."""
    pol = _policies([[], [8], [5]], [[8], [8], [8, 5]])
    for via_backup in (True, False):
        net, H2, H4 = _backup_switch_net(via_backup)
        pr = np.concatenate([probe(0, H2, H4, 1)] * 3)
        res, hits = oracle.verify_constrained(net, pr, 16, pol, probe_policy=np.arange(3, dtype=np.uint32))
        if via_backup:
            # policy 0: delivered through 8; policy 1: 8 forbidden and required
            # -> violation on entering 8, the waypoint visit does not count;
            # policy 2: 5 forbidden, path avoids it, only waypoint 8 visited
            assert list(res["status"]) == [W.ST_COMPLIANT, W.ST_VIOLATION, W.ST_COMPLIANT]
            assert list(res["hops"]) == [3, 2, 3] and list(res["last_switch"]) == [4, 8, 4]
            assert list(hits) == [1, 0, 1]
        else:
            assert list(res["status"]) == [W.ST_COMPLIANT, W.ST_COMPLIANT, W.ST_VIOLATION]
            assert list(hits) == [0, 0, 0]
            assert res["last_switch"][2] == 5 and res["hops"][2] == 2
        # no policy (index out of range): the plain walk, no waypoint bits
        r0, h0 = oracle.verify_constrained(net, pr[:1], 16, pol, probe_policy=np.array([7], np.uint32))
        assert (r0 == oracle.verify_probes(net, pr[:1], 16)).all() and h0[0] == 0


@pytest.mark.parametrize("seed", range(4))
def test_constrained_walk_equals_judged_trace(seed):
    e = W.end_to_end(seed=40 + seed, num_switches=40, num_intents=24, probes_per_intent=40, rules_per_switch=90,
                     hop_cap=24)
    net = e.network
    pol = W.path_policies(seed, net, 24, forbid_max=3, must_max=4, hubs=8)
    pr = e.probes.probes.copy()
    st = W.Stream(seed, "policy-probes")
    H = net.num_hosts
    pr["src_host"] = st.ints(0, H - 1, len(pr))
    pr["src_ip"] = net.host_ip[pr["src_host"]]
    pr["src_host"][::17] = W.NO_HOST
    pr["allowed_mask"][::3] = 0xFFFFFFFF
    res, hits = oracle.verify_constrained(net, pr, 24, pol, probes_per_policy=40)
    for k in range(len(pr)):
        p = k // 40
        f = pol.forbid[pol.forbid_offs[p]:pol.forbid_offs[p + 1]]
        m = pol.must[pol.must_offs[p]:pol.must_offs[p + 1]]
        (st_, hops, last), hit = trace_walk_constrained(net, pr[k], 24, f, m)
        assert (res["status"][k], res["hops"][k], res["last_switch"][k], hits[k]) == (st_, hops, last, hit), k
    assert (hits != 0).any() and (res["status"] == W.ST_VIOLATION).any()
    # explicit per-probe policy indices give the same as the stride
    r2, h2 = oracle.verify_constrained(net, pr, 24, pol, probe_policy=np.arange(len(pr), dtype=np.uint32) // 40)
    assert (r2 == res).all() and (h2 == hits).all()


def test_constrained_verdict_closed_form():
    st = W.Stream(8, "policy-verdict")
    G, N, pods, ppg = 40, 64, 2, 6
    Wd = W.words_per_row(N)
    bits = np.full((G, Wd), 0xFFFFFFFF, np.uint32)
    bits[:, 2:] = 0
    flags = np.zeros(G, np.uint8)
    assign = st.ints(0, N - 1, G * pods).astype(np.uint32)
    results = np.zeros(G * ppg, W.RESULT_DTYPE)
    results["status"] = np.where(st.floats(G * ppg) < 0.9, W.ST_COMPLIANT, W.ST_DROP)
    must_lists = [list(range(int(x))) for x in st.ints(0, 3, G)]
    concrete = (st.floats(G) > 0.15).astype(np.uint8)
    pol = _policies([[] for _ in range(G)], must_lists, concrete)
    full = np.array([(1 << len(m)) - 1 for m in must_lists], np.uint32)
    hits = np.repeat(full, ppg)
    miss = st.floats(G * ppg) < 0.1
    hits[miss] = hits[miss] >> 1
    passed, counts = oracle.aggregate_constrained(bits, N, flags, assign, pods, results, ppg, hits, pol)
    p0, c0 = oracle.aggregate(bits, N, flags, assign, pods, results, ppg)
    missed = (hits.reshape(G, ppg) != full[:, None]).sum(1)
    assert (counts[:, :7] == c0[:, :7]).all() and (counts[:, 7] == missed).all()
    want = p0.astype(bool) & concrete.astype(bool) & (missed == 0)
    assert (passed.astype(bool) == want).all() and want.any() and not want.all()
    # a no-op policy fails the intent even when every check it names passes
    assert not passed[np.nonzero(concrete == 0)[0]].any()
    # groups mapped to no policy keep the plain verdict
    gp = np.full(G, 0xFFFFFFFF, np.uint32)
    p2, _ = oracle.aggregate_constrained(bits, N, flags, assign, pods, results, ppg, hits, pol, group_policy=gp)
    assert (p2 == p0).all()
