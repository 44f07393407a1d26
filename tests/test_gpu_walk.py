"""GPU parity of the hop-synchronous probe walk against the oracle
(bit-exact status, hops, last switch): hand-built worked cases, the tiny
ring, scaled fat trees and random graphs with every hop cap edge, and the
full flow-verification workload (k=16 fat tree, 2,000 rules per switch, 10M
probes) on a sampled subset."""
import numpy as np
import pytest

import oracle
from paper_2602_16100_gb300 import binding as B
from paper_2602_16100_gb300 import workloads as W
from paper_2602_16100_gb300.validator import empty_device, to_device, to_numpy
from gpu_util import sample
from netbuild import ip, make_net, probe, rule

pytestmark = pytest.mark.gpu


def _gpu_walk(v, net, probes, cap):
    v.load_network(net)
    out = v.verify_probes(to_device(probes, v.device), len(probes), cap)
    v.sync()
    return to_numpy(out, W.RESULT_DTYPE)


def _same(a, b):
    return (a["status"] == b["status"]).all() and (a["hops"] == b["hops"]).all() and \
        (a["last_switch"] == b["last_switch"]).all()


def test_worked_cases(validator):
    A, Bh, C = ip(10, 0, 0, 1), ip(10, 0, 2, 1), ip(10, 0, 2, 2)
    rules = [[rule(100, Bh, 24, 1), rule(100, A, 32, 0)],
             [rule(100, Bh, 24, 1), rule(100, A, 24, 0), rule(150, Bh, 32, W.DROP, lo=7, hi=7)],
             [rule(100, Bh, 32, 0), rule(100, C, 32, 2), rule(100, A, 24, 1)]]
    net = make_net([2, 2, 3], [(0, 1, 1, 0), (1, 1, 2, 1)], [(0, 0, A), (2, 0, Bh), (2, 2, C)], [0, 1, 0], rules)
    pr = np.concatenate([probe(0, A, Bh, 1), probe(0, A, Bh, 3), probe(0, A, Bh, 3, dport=7), probe(0, A, A, 1),
                         probe(0, A, C, 3), probe(W.NO_HOST, A, Bh, 3), probe(7, A, Bh, 3),
                         probe(0, A, ip(99, 0, 0, 0), 3)])
    for cap in (1, 2, 3, 16, 255):
        g = _gpu_walk(validator, net, pr, cap)
        o = oracle.verify_probes(net, pr, cap)
        assert _same(g, o), cap
    g = _gpu_walk(validator, net, pr, 16)
    assert g["status"][0] == W.ST_VIOLATION and g["last_switch"][0] == 1


def test_tiny(validator):
    d = W.tiny()
    g = _gpu_walk(validator, d["network"], d["probes"].probes, d["probes"].hop_cap)
    o = oracle.verify_probes(d["network"], d["probes"].probes, d["probes"].hop_cap)
    assert _same(g, o)


@pytest.mark.parametrize("k,rules,cap,mask_all", [(4, 100, 8, False), (4, 100, 8, True), (8, 600, 32, False),
                                                  (8, 600, 5, True), (6, 2000, 255, True)])
def test_fat_trees(validator, k, rules, cap, mask_all):
    d = W.fat_tree(seed=k * 31 + rules, k=k, rules_per_switch=rules, num_probes=20011, hop_cap=cap)
    pr = d["probes"].probes.copy()
    if mask_all:
        pr["allowed_mask"] = 0xFFFFFFFF
    g = _gpu_walk(validator, d["network"], pr, cap)
    o = oracle.verify_probes(d["network"], pr, cap)
    assert _same(g, o)
    assert len(np.unique(o["status"])) >= 3


def test_random_graph_network(validator):
    e = W.end_to_end(seed=4, num_switches=40, num_intents=20, probes_per_intent=500, rules_per_switch=150)
    pr = e.probes.probes.copy()
    H = e.network.num_hosts
    pr["src_host"] = np.arange(len(pr)) % (H + 3)            # some out-of-range hosts -> NOSRC
    ok = pr["src_host"] < H
    pr["src_ip"][ok] = e.network.host_ip[pr["src_host"][ok]]
    for cap in (1, 32):
        g = _gpu_walk(validator, e.network, pr, cap)
        o = oracle.verify_probes(e.network, pr, cap)
        assert _same(g, o)


def test_empty_and_invalid_calls(validator):
    d = W.tiny()
    validator.load_network(d["network"])
    dev = validator.device
    pr = to_device(d["probes"].probes, dev)
    out = empty_device(4 * len(d["probes"].probes), dev)
    B.pv_verify_probes(validator.ctx, 0, pr, 16, out)
    for cap in (0, 256):
        with pytest.raises(B.PVError) as e:
            B.pv_verify_probes(validator.ctx, 10, pr, cap, out)
        assert e.value.code == B.PV_EINVAL
    net = d["network"]
    bad = net.rules.copy()
    bad[3]["src_len"] = 33
    with pytest.raises(B.PVError):
        B.pv_load_flow_tables(validator.ctx, net.num_switches, net.rule_offs, bad, net.switch_region, net.port_offs,
                              net.port_peer, net.num_hosts, net.host_switch, net.host_port, net.host_ip)
    reg = net.switch_region.copy()
    reg[0] = 32
    with pytest.raises(B.PVError):
        B.pv_load_flow_tables(validator.ctx, net.num_switches, net.rule_offs, net.rules, reg, net.port_offs,
                              net.port_peer, net.num_hosts, net.host_switch, net.host_port, net.host_ip)


def test_flow_verification_full_size_sampled(validator):
    """The full flow-verification workload in the benchmark's launch
    configuration; the oracle walks a sample of probes."""
    d = W.fat_tree()
    net, P = d["network"], d["probes"]
    g = _gpu_walk(validator, net, P.probes, P.hop_cap)
    idx = sample(len(P.probes), 20000, seed=2)
    o = oracle.verify_probes(net, P.probes, P.hop_cap, idx=idx)
    assert _same(g[idx], o)
    assert (g["status"] <= W.ST_MISDELIVERED).all()
