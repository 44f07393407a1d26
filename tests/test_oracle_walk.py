"""Pins for the oracle's first-match forwarding and probe walks.

Checked against: hand cases of the OpenFlow match semantics (prefix lengths 0
and 32, inclusive port ranges, equal priorities, wildcard in_port), a
sort-then-scan formulation of first match, shadowed rules, the paper's worked
examples built as tiny topologies (Sec. 3.3 PHI/untrusted-switch example; an
EU-only flow whose only path crosses a US switch; Sec. 6.3 item 4 transit
switches), and a recursive trace that records the whole path and judges it
afterwards.
"""
import numpy as np
import pytest

import oracle
from paper_2602_16100_gb300 import workloads as W
from netbuild import first_match_sorted, ip, make_net, probe, rule, trace_walk


# ---------------------------------------------------------------------------
# first match
# ---------------------------------------------------------------------------
def test_first_match_hand_cases():
    R = np.concatenate([
        rule(10, dst_ip=ip(10, 0, 0, 0), dst_len=8, action=1),           # 0
        rule(10, dst_ip=ip(10, 1, 0, 0), dst_len=16, action=2),          # 1 same priority, later index
        rule(20, dst_ip=ip(10, 1, 2, 3), dst_len=32, action=3),          # 2 exact host
        rule(5, action=4),                                               # 3 match-all (len 0)
        rule(30, src_ip=ip(192, 168, 0, 0), src_len=16, lo=100, hi=200, action=5),  # 4
        rule(40, in_port=7, action=6),                                   # 5 in_port specific
        rule(25, dst_ip=ip(10, 1, 255, 255), dst_len=16, action=7),      # 6 non-canonical value bits
    ])
    fm = lambda ip_in, s, d, dp: oracle.first_match(R, ip_in, s, d, dp)
    assert fm(0, 0, ip(10, 1, 2, 3), 80) == 6            # /16 at 25 beats /32 at 20 (priority, not length)
    assert fm(0, 0, ip(10, 1, 2, 4), 80) == 6
    assert fm(0, 0, ip(10, 2, 0, 0), 80) == 0            # tie at 10 broken by index -> 0
    assert fm(0, 0, ip(11, 0, 0, 0), 80) == 3            # only the len-0 rule
    assert fm(0, 0, 0xFFFFFFFF, 80) == 3
    assert fm(0, ip(192, 168, 9, 9), ip(11, 0, 0, 0), 100) == 4   # range edges inclusive
    assert fm(0, ip(192, 168, 9, 9), ip(11, 0, 0, 0), 200) == 4
    assert fm(0, ip(192, 168, 9, 9), ip(11, 0, 0, 0), 99) == 3
    assert fm(0, ip(192, 168, 9, 9), ip(11, 0, 0, 0), 201) == 3
    assert fm(7, 0, 0, 0) == 5 and fm(6, 0, 0, 0) == 3
    assert oracle.first_match(R[:3], 0, 0, ip(11, 0, 0, 0), 0) == -1   # table miss
    edge = np.concatenate([rule(1, lo=0, hi=0, action=1), rule(1, lo=65535, hi=65535, action=2)])
    assert oracle.first_match(edge, 0, 0, 0, 0) == 0
    assert oracle.first_match(edge, 0, 0, 0, 65535) == 1
    assert oracle.first_match(edge, 0, 0, 0, 1) == -1
    one = rule(1, dst_ip=0x80000000, dst_len=1, action=1)
    assert oracle.first_match(one, 0, 0, 0xFFFFFFFF, 0) == 0
    assert oracle.first_match(one, 0, 0, 0x7FFFFFFF, 0) == -1


@pytest.mark.parametrize("seed", [1, 2, 3])
def test_first_match_equals_sort_then_scan(seed):
    st = W.Stream(seed, "fm-test")
    n = 300
    R = np.zeros(n, W.RULE_DTYPE)
    R["priority"] = st.ints(0, 6, n)                      # many ties
    R["in_port"] = np.where(st.floats(n) < 0.5, W.ANY_PORT, st.ints(0, 3, n))
    R["src_len"] = st.ints(0, 32, n)
    R["dst_len"] = st.ints(0, 32, n)
    R["src_ip"] = st.ints(0, 0xFFFFFFFF, n) & 0xF00000FF   # few distinct prefixes
    R["dst_ip"] = st.ints(0, 0xFFFFFFFF, n) & 0xF00000FF
    lo = st.ints(0, 65535, n)
    R["dport_lo"] = lo
    R["dport_hi"] = np.minimum(65535, lo + st.ints(0, 40000, n))
    for _ in range(400):
        h = st.ints(0, 0xFFFFFFFF, 4)
        args = (int(h[0] % 4), int(h[1]) & 0xF00000FF, int(h[2]) & 0xF00000FF, int(h[3]) % 65536)
        assert oracle.first_match(R, *args) == first_match_sorted(R, *args)


def test_shadowed_rules_never_first():
    d = W.fat_tree(seed=5, k=4, rules_per_switch=400, num_probes=10, p_shadow=0.3)
    net = d["network"]
    sh = np.nonzero(net.shadowed_by >= 0)[0]
    assert len(sh) > 50
    for g in sh:
        s = int(np.searchsorted(net.rule_offs, g, side="right") - 1)
        base = int(net.rule_offs[s])
        rs = net.rules[base:net.rule_offs[s + 1]]
        r = net.rules[g]
        in_port = 0 if int(r["in_port"]) == W.ANY_PORT else int(r["in_port"])
        m = oracle.first_match(rs, in_port, int(r["src_ip"]), int(r["dst_ip"]), int(r["dport_lo"]))
        assert m >= 0 and m != g - base
        assert int(rs[m]["priority"]) >= int(r["priority"])


# ---------------------------------------------------------------------------
# worked walks
# ---------------------------------------------------------------------------
EU, US = 0, 1
A_IP, B_IP, C_IP = ip(10, 0, 0, 1), ip(10, 0, 2, 1), ip(10, 0, 2, 2)


def _line_net(region1=US, s1_extra=()):
    """A@S0 -- S1 -- S2@B (and C on S2 port 2)."""
    rules = [
        [rule(100, B_IP, 24, 1), rule(100, A_IP, 32, 0)],
        [rule(100, B_IP, 24, 1), rule(100, A_IP, 24, 0), *s1_extra],
        [rule(100, B_IP, 32, 0), rule(100, C_IP, 32, 2), rule(100, A_IP, 24, 1)],
    ]
    return make_net([2, 2, 3], [(0, 1, 1, 0), (1, 1, 2, 1)],
                    [(0, 0, A_IP), (2, 0, B_IP), (2, 2, C_IP)], [EU, region1, EU], rules)


def _walk(net, p, cap=16):
    r = oracle.verify_probes(net, p, cap)[0]
    return int(r["status"]), int(r["hops"]), int(r["last_switch"])


def test_eu_only_flow_across_us_switch_fails():
    net = _line_net()
    assert _walk(net, probe(0, A_IP, B_IP, 1 << EU)) == (W.ST_VIOLATION, 2, 1)
    assert _walk(net, probe(0, A_IP, B_IP, (1 << EU) | (1 << US))) == (W.ST_COMPLIANT, 3, 2)
    # the same intent passes when the transit switch is relabelled EU
    assert _walk(_line_net(region1=EU), probe(0, A_IP, B_IP, 1 << EU)) == (W.ST_COMPLIANT, 3, 2)


def test_phi_traffic_avoiding_untrusted_switches():
    """Sec. 3.3 example: paths carrying PHI flows must exclude vertices
    labelled trusted=no.  Diamond S0 -> {S1 untrusted, S2 trusted} -> S3; the
    routing goes via S2, but a higher-priority rule steers dport 5432 via S1."""
    TRUSTED, UNTRUSTED = 0, 1
    rules = [
        [rule(100, B_IP, 24, 2), rule(200, B_IP, 24, 1, lo=5432, hi=5432)],
        [rule(100, B_IP, 24, 1)],
        [rule(100, B_IP, 24, 1)],
        [rule(100, B_IP, 32, 0)],
    ]
    net = make_net([3, 2, 2, 3], [(0, 1, 1, 0), (0, 2, 2, 0), (1, 1, 3, 1), (2, 1, 3, 2)],
                   [(0, 0, A_IP), (3, 0, B_IP)], [TRUSTED, UNTRUSTED, TRUSTED, TRUSTED], rules)
    only_trusted = 1 << TRUSTED
    assert _walk(net, probe(0, A_IP, B_IP, only_trusted, dport=80)) == (W.ST_COMPLIANT, 3, 3)
    assert _walk(net, probe(0, A_IP, B_IP, only_trusted, dport=5432)) == (W.ST_VIOLATION, 2, 1)


def test_loop_drop_misdelivery_and_edges():
    # ping-pong between S0 and S1
    rules = [[rule(100, B_IP, 24, 1)], [rule(100, B_IP, 24, 0)]]
    net = make_net([2, 1], [(0, 1, 1, 0)], [(0, 0, A_IP)], [EU, EU], rules)
    assert _walk(net, probe(0, A_IP, B_IP, 1), cap=5) == (W.ST_LOOP, 5, 0)
    assert _walk(net, probe(0, A_IP, B_IP, 1), cap=4) == (W.ST_LOOP, 4, 1)
    assert _walk(net, probe(0, A_IP, B_IP, 1), cap=255) == (W.ST_LOOP, 255, 0)
    # explicit drop beats routing by priority; a table miss drops
    net = _line_net(s1_extra=(rule(150, B_IP, 32, W.DROP),))
    assert _walk(net, probe(0, A_IP, B_IP, 3)) == (W.ST_DROP, 2, 1)
    assert _walk(net, probe(0, A_IP, ip(99, 0, 0, 1), 3)) == (W.ST_DROP, 1, 0)
    # region check comes before the drop: a forbidden switch that drops violates
    assert _walk(net, probe(0, A_IP, B_IP, 1 << EU)) == (W.ST_VIOLATION, 2, 1)
    # misdelivery: S1 sends C's traffic fine, but S2 delivers B's /32 rule to C's port
    net = _line_net(s1_extra=())
    net.rules[int(net.rule_offs[2])]["action"] = 2
    assert _walk(net, probe(0, A_IP, B_IP, 3)) == (W.ST_MISDELIVERED, 3, 2)
    # src == dst host
    assert _walk(_line_net(), probe(0, A_IP, A_IP, 1)) == (W.ST_COMPLIANT, 1, 0)
    # unconnected output port drops
    net = make_net([3], [], [(0, 0, A_IP)], [EU], [[rule(100, B_IP, 24, 2)]])
    assert _walk(net, probe(0, A_IP, B_IP, 1)) == (W.ST_DROP, 1, 0)
    # no source host
    assert _walk(_line_net(), probe(W.NO_HOST, A_IP, B_IP, 3)) == (W.ST_NOSRC, 0, 0xFFFF)
    assert _walk(_line_net(), probe(3, A_IP, B_IP, 3)) == (W.ST_NOSRC, 0, 0xFFFF)


def test_hop_cap_boundary_and_in_port_rules():
    net = _line_net()
    assert _walk(net, probe(0, A_IP, B_IP, 3), cap=3) == (W.ST_COMPLIANT, 3, 2)
    assert _walk(net, probe(0, A_IP, B_IP, 3), cap=2) == (W.ST_LOOP, 2, 1)
    assert _walk(net, probe(0, A_IP, B_IP, 3), cap=1) == (W.ST_LOOP, 1, 0)
    # a rule matching only traffic entering S1 from S2 (port 1) does not fire for A->B
    net = _line_net(s1_extra=(rule(300, B_IP, 24, W.DROP, in_port=1),))
    assert _walk(net, probe(0, A_IP, B_IP, 3)) == (W.ST_COMPLIANT, 3, 2)
    net = _line_net(s1_extra=(rule(300, B_IP, 24, W.DROP, in_port=0),))
    assert _walk(net, probe(0, A_IP, B_IP, 3)) == (W.ST_DROP, 2, 1)


# ---------------------------------------------------------------------------
# recursive trace on generated workloads + path invariants
# ---------------------------------------------------------------------------
def _check_against_trace(net, probes, cap, limit=None):
    res = oracle.verify_probes(net, probes, cap)
    n = len(probes) if limit is None else min(limit, len(probes))
    for i in range(n):
        want, path = trace_walk(net, probes[i], cap)
        got = tuple(int(x) for x in (res[i]["status"], res[i]["hops"], res[i]["last_switch"]))
        assert got == want, (i, got, want)
        mask = int(probes[i]["allowed_mask"])
        if got[0] == W.ST_COMPLIANT:
            assert all((mask >> int(net.switch_region[s])) & 1 for s in path)
        if got[0] == W.ST_LOOP:
            assert got[1] == cap
        assert got[1] <= cap
    return res


def test_walks_equal_recursive_trace_tiny():
    d = W.tiny()
    res = _check_against_trace(d["network"], d["probes"].probes, d["probes"].hop_cap)
    hist = np.bincount(res["status"], minlength=6)
    assert hist[W.ST_COMPLIANT] > 0 and hist[W.ST_VIOLATION] > 0 and hist[W.ST_DROP] > 0


def test_walks_equal_recursive_trace_fat_tree_and_random_graph():
    d = W.fat_tree(seed=7, k=4, rules_per_switch=120, num_probes=600, hop_cap=12)
    _check_against_trace(d["network"], d["probes"].probes, 12)
    # all-permitting masks exercise long walks
    pr = d["probes"].probes.copy()
    pr["allowed_mask"] = 0xFFFFFFFF
    res = _check_against_trace(d["network"], pr, 12)
    assert (res["status"] == W.ST_COMPLIANT).sum() > 100
    e = W.end_to_end(seed=9, num_switches=24, num_intents=8, probes_per_intent=40, rules_per_switch=80)
    pr = e.probes.probes.copy()
    pr["src_host"] = np.arange(len(pr)) % e.network.num_hosts
    pr["src_ip"] = e.network.host_ip[pr["src_host"]]
    _check_against_trace(e.network, pr, e.probes.hop_cap)


# ---------------------------------------------------------------------------
# two bounces in a row (the walk's two-switch cycle shortcut)
# ---------------------------------------------------------------------------
def _symmetric(net):
    po, pp = net.port_offs, net.port_peer
    for u in range(net.num_switches):
        for p in range(int(po[u]), int(po[u + 1])):
            peer = int(pp[p])
            if peer < 0 or peer & W.HOST_BIT:
                continue
            v, q = peer >> 8, peer & 0xFF
            if int(pp[int(po[v]) + q]) != (u << 8 | (p - int(po[u]))):
                return False
    return True


def _first_double_bounce(net, pr, cap):
    """Follow the probe's (switch, in_port) states while it is handed to
    switches (masks that permit every region); return (h, s_h, s_h+1) for the
    first visit h >= 1 at which it leaves by its in_port right after leaving
    the previous switch by that switch's in_port, with h + 1 < cap; else None."""
    hdr = (int(pr["src_ip"]), int(pr["dst_ip"]), int(pr["dport"]))
    s, p = int(net.host_switch[int(pr["src_host"])]), int(net.host_port[int(pr["src_host"])])
    prev_bounce = False
    for h in range(cap - 1):
        rs = net.rules[net.rule_offs[s]:net.rule_offs[s + 1]]
        i = first_match_sorted(rs, p, *hdr)
        if i < 0 or int(rs[i]["action"]) == W.DROP:
            return None
        port = int(rs[i]["action"])
        if port >= int(net.port_offs[s + 1] - net.port_offs[s]):
            return None
        peer = int(net.port_peer[net.port_offs[s] + port])
        if peer < 0 or peer & W.HOST_BIT:
            return None
        bounce = port == p
        if bounce and prev_bounce:
            return h, s, peer >> 8
        prev_bounce = bounce
        s, p = peer >> 8, peer & 0xFF
    return None


def test_two_bounces_in_a_row_prove_a_two_switch_cycle():
    """With symmetric cabling, a probe that leaves two switches in a row by
    the port it came in by walks back and forth between them until the hop
    cap: the full walk ends PV_LOOP with hops = cap at the switch of visit
    cap - 1, which is s_h when cap - 1 - h is even and s_h+1 otherwise.
    Checked against the oracle's full walks on every probe that shows the
    pattern, at several caps."""
    cases = []
    e = W.end_to_end(seed=9, num_switches=24, num_intents=8, probes_per_intent=40, rules_per_switch=80)
    pr = e.probes.probes.copy()
    pr["src_host"] = np.arange(len(pr)) % e.network.num_hosts
    pr["src_ip"] = e.network.host_ip[pr["src_host"]]
    cases.append((e.network, pr))
    d = W.fat_tree(seed=7, k=4, rules_per_switch=120, num_probes=600, hop_cap=12)
    cases.append((d["network"], d["probes"].probes.copy()))
    checked = 0
    for net, pr in cases:
        assert _symmetric(net)
        pr["allowed_mask"] = 0xFFFFFFFF
        for cap in (4, 7, 12, 31, 32):
            res = oracle.verify_probes(net, pr, cap)
            for k in range(len(pr)):
                hit = _first_double_bounce(net, pr[k], cap)
                if hit is None:
                    continue
                h, s0, s1 = hit
                want = (W.ST_LOOP, cap, s0 if (cap - 1 - h) % 2 == 0 else s1)
                got = tuple(int(x) for x in (res[k]["status"], res[k]["hops"], res[k]["last_switch"]))
                assert got == want, (cap, k, got, want)
                checked += 1
    assert checked > 50


def test_two_bounces_on_asymmetric_cabling_prove_nothing():
    """Port 0 of X, Y and Z leads X -> Y -> Z -> X (not back), every switch
    sends everything out of port 0: every hop after the first is a bounce,
    yet the walk has period 3, so the parity rule fails (cap 5: visit 4 is at
    Y, the rule would say Z)."""
    net = make_net([2, 1, 1], [], [(0, 1, ip(10, 0, 0, 1))], [0, 0, 0],
                   [[rule(100, 0, 0, 0)], [rule(100, 0, 0, 0)], [rule(100, 0, 0, 0)]])
    net.port_peer[net.port_offs[0]] = (1 << 8) | 0
    net.port_peer[net.port_offs[1]] = (2 << 8) | 0
    net.port_peer[net.port_offs[2]] = (0 << 8) | 0
    assert not _symmetric(net)
    pr = probe(0, ip(10, 0, 0, 1), ip(99, 0, 0, 1), 1)
    h, s0, s1 = _first_double_bounce(net, pr[0], 5)
    assert (h, s0, s1) == (2, 2, 0)
    res = oracle.verify_probes(net, pr, 5)
    assert (int(res[0]["status"]), int(res[0]["hops"]), int(res[0]["last_switch"])) == (W.ST_LOOP, 5, 1)
    assert int(res[0]["last_switch"]) != (s0 if (5 - 1 - h) % 2 == 0 else s1)
