"""Pins for the oracle's path scheduler and rule compilation (Sec. 4.2:
constraint-respecting paths from weighted Dijkstra / BFS, turned into
per-hop flow rules).

The oracle's paths are compared exactly with an independent formulation
that takes its distances from networkx's Dijkstra and applies the canonical
predecessor rule written out directly; the compiled rules close the loop:
installed ahead of each switch's table, a probe of every scheduled flow is
delivered COMPLIANT along exactly the scheduled visits, with every waypoint
entered.
"""
import numpy as np
import pytest

nx = pytest.importorskip("networkx")

import oracle
from paper_2602_16100_gb300 import workloads as W
from netbuild import ip, make_net, rule
from test_oracle_policies import _backup_switch_net, _policies


def _canonical(net, q, pol, weights, max_len):
    H, S = net.num_hosts, net.num_switches
    if q["src_host"] >= H or q["dst_host"] >= H:
        return W.PATH_NOSRC, []
    forbid, must = set(), []
    if pol is not None and q["policy"] < pol.num_policies:
        p = int(q["policy"])
        forbid = {int(x) for x in pol.forbid[pol.forbid_offs[p]:pol.forbid_offs[p + 1]]}
        must = [int(x) for x in pol.must[pol.must_offs[p]:pol.must_offs[p + 1]]]
    mask = int(q["allowed_mask"])
    ok = {s for s in range(S) if net.switch_region[s] < 32 and (mask >> int(net.switch_region[s])) & 1
          and s not in forbid}
    wt = lambda u, p: max(1, int(weights[net.port_offs[u] + p])) if weights is not None else 1
    G = nx.DiGraph()
    G.add_nodes_from(ok)
    links = {}   # v -> [(u, p, q)]
    for u in ok:
        for p in range(int(net.port_offs[u + 1] - net.port_offs[u])):
            peer = int(net.port_peer[net.port_offs[u] + p])
            if peer < 0 or peer & W.HOST_BIT or (peer >> 8) not in ok:
                continue
            v = peer >> 8
            links.setdefault(v, []).append((u, p, peer & 0xFF))
            if not G.has_edge(u, v) or G[u][v]["weight"] > wt(u, p):
                G.add_edge(u, v, weight=wt(u, p))
    src_sw, dst_sw = int(net.host_switch[q["src_host"]]), int(net.host_switch[q["dst_host"]])
    if src_sw not in ok or dst_sw not in ok or any(m not in ok for m in must):
        return W.PATH_BLOCKED, []
    visits = [[src_sw, int(net.host_port[q["src_host"]]), 0]]
    cur = src_sw
    for t in must + [dst_sw]:
        if t == cur:
            continue
        d = nx.single_source_dijkstra_path_length(G, cur)
        if t not in d:
            return W.PATH_BLOCKED, []
        back, v = [], t
        while v != cur:
            u, p, qq = min(c for c in links[v] if c[0] in d and d[c[0]] + wt(c[0], c[1]) == d[v])
            back.append((p, v, qq))
            v = u
        for p, v, qq in reversed(back):
            if len(visits) >= max_len:
                return W.PATH_TOO_LONG, []
            visits[-1][2] = p
            visits.append([v, qq, 0])
        cur = t
    visits[-1][2] = int(net.host_port[q["dst_host"]])
    states = [(s, i) for s, i, _ in visits]
    if len(set(states)) < len(states):
        return W.PATH_REPEAT, []
    return W.PATH_OK, [(s << 16) | (i << 8) | o for s, i, o in visits]


def _install(net, rules, rsw):
    """A copy of the network with the compiled rules ahead of each switch's
    own rules (slot order)."""
    tables = []
    for s in range(net.num_switches):
        mine = rules[rsw == s]
        tables.append([mine[i:i + 1] for i in range(len(mine))] +
                      [net.rules[i:i + 1] for i in range(int(net.rule_offs[s]), int(net.rule_offs[s + 1]))])
    S = net.num_switches
    rule_offs = np.zeros(S + 1, np.uint32)
    rule_offs[1:] = np.cumsum([len(t) for t in tables])
    allr = np.concatenate([np.concatenate(t) for t in tables if t])
    return W.Network(S, rule_offs, allr, net.switch_region, net.port_offs, net.port_peer, net.num_hosts,
                     net.host_switch, net.host_port, net.host_ip)


def _check_closed_loop(net, req, pol, hops, ln, st):
    rules, rsw = oracle.compile_path_rules(net, req, hops, ln, st)
    inst = _install(net, rules, rsw)
    okr = np.nonzero(st == W.PATH_OK)[0]
    pr = np.zeros(len(okr), W.PROBE_DTYPE)
    pr["src_host"] = req["src_host"][okr]
    pr["src_ip"] = net.host_ip[req["src_host"][okr]]
    pr["dst_ip"] = net.host_ip[req["dst_host"][okr]]
    pr["dport"] = np.arange(len(okr)) * 7919 % 65536
    pr["allowed_mask"] = req["allowed_mask"][okr]
    pp = req["policy"][okr].astype(np.uint32)
    polx = pol if pol is not None else _policies([[]], [[]])
    res, hits = oracle.verify_constrained(inst, pr, 255, polx, probe_policy=pp)
    assert (res["status"] == W.ST_COMPLIANT).all()
    assert (res["hops"] == ln[okr]).all()
    assert (res["last_switch"] == net.host_switch[req["dst_host"][okr]]).all()
    nm = np.array([int(polx.must_offs[p + 1] - polx.must_offs[p]) if p < polx.num_policies else 0 for p in pp])
    assert (hits == ((1 << nm) - 1)).all()


@pytest.mark.parametrize("seed,weighted,max_len", [(0, False, 64), (1, True, 64), (2, True, 12), (3, False, 255)])
def test_scheduler_equals_canonical_networkx(seed, weighted, max_len):
    e = W.end_to_end(seed=70 + seed, num_switches=60, num_intents=4, probes_per_intent=4, rules_per_switch=80)
    net = e.network
    pol = W.path_policies(seed, net, 40, forbid_max=3, must_max=3, hubs=12)
    req = W.path_requests(seed, net, 300, num_policies=40, extra_regions=(4, 12), bad_hosts=3)
    st_ = W.Stream(seed, "weights")
    weights = st_.ints(1, 20, int(net.port_offs[-1])).astype(np.uint16) if weighted else None
    if weighted:
        weights[::11] = 0                      # a weight of 0 counts as 1
    hops, ln, st = oracle.schedule_paths(net, req, pol, weights, max_len)
    for r in range(len(req)):
        want_st, want = _canonical(net, req[r], pol, weights, max_len)
        assert st[r] == want_st, r
        if want_st == W.PATH_OK:
            assert ln[r] == len(want) and list(hops[r, : ln[r]]) == want, r
    assert len(set(st.tolist())) >= 3 and (st == W.PATH_OK).sum() > 50
    _check_closed_loop(net, req, pol, hops, ln, st)


def test_waypoint_forces_the_backup_switch():
    """Sec. 5.3 networking intent, from the scheduler's side: the cheapest
    path from host 2 to host 4 goes through switch 5; with switch 8 as a
    waypoint it goes through 8; with 8 required and 5 forbidden as well, the
    same; with 8 forbidden and required, no path."""
    net, H2, H4 = _backup_switch_net(via_backup=False)
    weights = np.ones(int(net.port_offs[-1]), np.uint16)
    weights[net.port_offs[2] + 1] = 2          # switch 2 -> switch 8 costs 2: via 8 is 3, via 5 is 2
    pol = _policies([[], [], [5], [8]], [[], [8], [8], [8]])
    req = np.zeros(4, W.PATH_REQ_DTYPE)
    req["src_host"], req["dst_host"], req["allowed_mask"] = 0, 1, 1
    req["policy"] = [0, 1, 2, 3]
    hops, ln, st = oracle.schedule_paths(net, req, pol, weights)
    sw = lambda r: [int(h) >> 16 for h in hops[r, : ln[r]]]
    assert list(st) == [W.PATH_OK, W.PATH_OK, W.PATH_OK, W.PATH_BLOCKED]
    assert sw(0) == [2, 5, 4] and sw(1) == [2, 8, 4] and sw(2) == [2, 8, 4]
    # visits carry the ports: host port in, link ports, host port out
    assert hops[1, 0] == (2 << 16) | (0 << 8) | 1 and hops[1, 2] == (4 << 16) | (1 << 8) | 0
    # the requests share one (src, dst) pair, whose rules would shadow one
    # another: each is installed on its own
    for r in range(3):
        _check_closed_loop(net, req[r:r + 1], pol, hops[r:r + 1], ln[r:r + 1], st[r:r + 1])


def test_repeated_state_is_reported():
    """A waypoint behind a dead end: reaching it and coming back enters the
    junction switch twice through the same port, which header rules cannot
    realise."""
    A, B = ip(10, 0, 0, 1), ip(10, 0, 1, 1)
    # host A - s0 - s1 - s2(host B); s1 - s3 (dead end waypoint)
    nports = [2, 3, 2, 1]
    links = [(0, 1, 1, 0), (1, 1, 2, 0), (1, 2, 3, 0)]
    hosts = [(0, 0, A), (2, 1, B)]
    net = make_net(nports, links, hosts, [0, 0, 0, 0], [[rule(1)] for _ in range(4)])
    pol = _policies([[], []], [[3], [1]])
    req = np.zeros(2, W.PATH_REQ_DTYPE)
    req["src_host"], req["dst_host"], req["allowed_mask"], req["policy"] = 0, 1, 1, [0, 1]
    hops, ln, st = oracle.schedule_paths(net, req, pol)
    # via s3: s0, s1 (in 0), s3, s1 (in 2), s2 -- s1 entered through different ports: realisable
    assert st[0] == W.PATH_OK and [int(h) >> 16 for h in hops[0, : ln[0]]] == [0, 1, 3, 1, 2]
    assert st[1] == W.PATH_OK
    # a waypoint revisit through the same port: s0 -> s1 -> s0 -> s1
    net2 = make_net([2, 2, 2], [(0, 1, 1, 0), (1, 1, 2, 0)], [(0, 0, A), (2, 1, B)], [0, 0, 0],
                    [[rule(1)] for _ in range(3)])
    pol2 = _policies([[]], [[1, 0, 2]])
    req2 = req[:1].copy()
    req2["policy"] = 0
    h2, l2, s2 = oracle.schedule_paths(net2, req2, pol2)
    assert s2[0] == W.PATH_REPEAT
