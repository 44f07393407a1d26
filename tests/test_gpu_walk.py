"""GPU parity of the hop-synchronous probe walk against the oracle
(bit-exact status, hops, last switch): hand-built worked cases, the tiny
ring, scaled fat trees and random graphs with every hop cap edge, and the
full flow-verification workload (k=16 fat tree, 2,000 rules per switch, 10M
probes) on every probe."""
import numpy as np
import pytest

import oracle
from paper_2602_16100_gb300 import binding as B
from paper_2602_16100_gb300 import workloads as W
from paper_2602_16100_gb300.validator import empty_device, to_device, to_numpy
import full_oracle as F
from netbuild import ip, make_net, probe, rule

pytestmark = pytest.mark.gpu


KERNELS = [1, 2]   # linear first-match scan, indexed first match
BUCKET = 256       # destination ports per bucket of the first-match index


def _gpu_walk(v, net, probes, cap, kernel=0):
    v.load_network(net)
    v.set_option(B.PV_OPT_WALK_KERNEL, kernel)
    try:
        out = v.verify_probes(to_device(probes, v.device), len(probes), cap)
        v.sync()
    finally:
        v.set_option(B.PV_OPT_WALK_KERNEL, 0)
    return to_numpy(out, W.RESULT_DTYPE)


def _same(a, b):
    return (a["status"] == b["status"]).all() and (a["hops"] == b["hops"]).all() and \
        (a["last_switch"] == b["last_switch"]).all()


@pytest.mark.parametrize("kernel", KERNELS)
def test_worked_cases(validator, kernel):
    A, Bh, C = ip(10, 0, 0, 1), ip(10, 0, 2, 1), ip(10, 0, 2, 2)
    rules = [[rule(100, Bh, 24, 1), rule(100, A, 32, 0)],
             [rule(100, Bh, 24, 1), rule(100, A, 24, 0), rule(150, Bh, 32, W.DROP, lo=7, hi=7)],
             [rule(100, Bh, 32, 0), rule(100, C, 32, 2), rule(100, A, 24, 1)]]
    net = make_net([2, 2, 3], [(0, 1, 1, 0), (1, 1, 2, 1)], [(0, 0, A), (2, 0, Bh), (2, 2, C)], [0, 1, 0], rules)
    pr = np.concatenate([probe(0, A, Bh, 1), probe(0, A, Bh, 3), probe(0, A, Bh, 3, dport=7), probe(0, A, A, 1),
                         probe(0, A, C, 3), probe(W.NO_HOST, A, Bh, 3), probe(7, A, Bh, 3),
                         probe(0, A, ip(99, 0, 0, 0), 3)])
    for cap in (1, 2, 3, 16, 255):
        g = _gpu_walk(validator, net, pr, cap, kernel)
        o = oracle.verify_probes(net, pr, cap)
        assert _same(g, o), cap
    g = _gpu_walk(validator, net, pr, 16)
    assert g["status"][0] == W.ST_VIOLATION and g["last_switch"][0] == 1


@pytest.mark.parametrize("kernel,lane_max", [(1, 96), (2, 0), (2, 96), (2, 65535)])
def test_tiny(validator, kernel, lane_max):
    d = W.tiny()
    validator.set_option(B.PV_OPT_WALK_LANE_MAX, lane_max)
    try:
        g = _gpu_walk(validator, d["network"], d["probes"].probes, d["probes"].hop_cap, kernel)
    finally:
        validator.set_option(B.PV_OPT_WALK_LANE_MAX, 96)
    o = oracle.verify_probes(d["network"], d["probes"].probes, d["probes"].hop_cap)
    assert _same(g, o)


@pytest.mark.parametrize("k,rules,cap,mask_all", [(4, 100, 8, False), (4, 100, 8, True), (8, 600, 32, False),
                                                  (8, 600, 5, True), (6, 2000, 255, True)])
@pytest.mark.parametrize("kernel", KERNELS)
def test_fat_trees(validator, k, rules, cap, mask_all, kernel):
    d = W.fat_tree(seed=k * 31 + rules, k=k, rules_per_switch=rules, num_probes=20011, hop_cap=cap)
    pr = d["probes"].probes.copy()
    if mask_all:
        pr["allowed_mask"] = 0xFFFFFFFF
    g = _gpu_walk(validator, d["network"], pr, cap, kernel)
    o = oracle.verify_probes(d["network"], pr, cap)
    assert _same(g, o)
    assert len(np.unique(o["status"])) >= 3


@pytest.mark.parametrize("kernel", KERNELS)
def test_random_graph_network(validator, kernel):
    e = W.end_to_end(seed=4, num_switches=40, num_intents=20, probes_per_intent=500, rules_per_switch=150)
    pr = e.probes.probes.copy()
    H = e.network.num_hosts
    pr["src_host"] = np.arange(len(pr)) % (H + 3)            # some out-of-range hosts -> NOSRC
    ok = pr["src_host"] < H
    pr["src_ip"][ok] = e.network.host_ip[pr["src_host"][ok]]
    for cap in (1, 32):
        g = _gpu_walk(validator, e.network, pr, cap, kernel)
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


def _index_stress_network(seed, S=6, rules=700):
    """Ring of switches whose tables interleave destination-only runs with
    general rules: nested prefixes (/0 to /32) over a few addresses, priority
    ties, port ranges straddling the index's destination-port bucket edges,
    in_port rules with full port ranges."""
    st = W.Stream(seed, "index-stress")
    hosts_per = 2
    H = S * hosts_per
    host_ip = np.array([ip(10, s, h, 1) for s in range(S) for h in range(hosts_per)], np.uint32)
    nports = [hosts_per + 2] * S
    links = [(s, hosts_per, (s + 1) % S, hosts_per + 1) for s in range(S)]
    hosts = [(s, h, int(host_ip[s * hosts_per + h])) for s in range(S) for h in range(hosts_per)]
    tables = []
    for s in range(S):
        n = rules
        r = np.zeros(n, W.RULE_DTYPE)
        dst_only = st.floats(n) < 0.6
        # priorities in runs so destination-only rules form contiguous segments
        r["priority"] = (np.arange(n) // st.ints(1, 40, 1)[0]) % 9 + st.ints(0, 1, n)
        base = host_ip[st.ints(0, H - 1, n)].astype(np.uint64)
        base ^= (st.u64(n) & np.uint64(0x00FF00FF)) * (st.floats(n) < 0.3)
        lens = np.array([0, 8, 12, 16, 20, 24, 28, 31, 32])[st.ints(0, 8, n)]
        m = np.where(lens == 0, 0, (0xFFFFFFFF << (32 - lens)) & 0xFFFFFFFF).astype(np.uint64)
        r["dst_ip"] = (base & m).astype(np.uint32)
        r["dst_len"] = lens
        edge = st.ints(1, 255, n) * BUCKET
        lo = np.clip(edge - st.ints(0, 3, n), 0, 65535)
        hi = np.clip(edge + st.ints(-1, 900, n), 0, 65535)
        r["dport_lo"] = np.where(dst_only, 0, np.minimum(lo, hi))
        r["dport_hi"] = np.where(dst_only, 65535, np.maximum(lo, hi))
        src_rule = (~dst_only) & (st.floats(n) < 0.5)
        r["src_len"] = np.where(src_rule, st.ints(1, 32, n), 0)
        r["src_ip"] = np.where(src_rule, host_ip[st.ints(0, H - 1, n)], 0)
        inp = (~dst_only) & (st.floats(n) < 0.3)
        r["in_port"] = np.where(inp, st.ints(0, nports[s] - 1, n), W.ANY_PORT)
        full = (~dst_only) & (st.floats(n) < 0.2)                 # general rule with full port range
        r["dport_lo"] = np.where(full, 0, r["dport_lo"])
        r["dport_hi"] = np.where(full, 65535, r["dport_hi"])
        act = st.ints(0, nports[s], n)
        r["action"] = np.where(act == nports[s], W.DROP, act)
        tables.append([r[i:i + 1] for i in range(n)])
    return make_net(nports, links, hosts, st.ints(0, 3, S).astype(np.uint8), tables), host_ip


def test_long_destination_runs_split_into_segments(validator):
    """A destination-only run longer than the 4,096-rule segment limit is
    indexed as consecutive segments (first-match order kept), behind a few
    general rules; both kernels against the oracle."""
    S, hosts_per = 3, 2
    host_ip = np.array([ip(10, s, h, 1) for s in range(S) for h in range(hosts_per)], np.uint32)
    links = [(s, hosts_per, (s + 1) % S, hosts_per + 1) for s in range(S)]
    hosts = [(s, h, int(host_ip[s * hosts_per + h])) for s in range(S) for h in range(hosts_per)]
    st = W.Stream(41, "long-runs")
    tables = []
    for s in range(S):
        n_run = 4300
        t = [rule(200, int(host_ip[(s + 1) % S * hosts_per]), 32, W.DROP, lo=80, hi=80)]     # general rule first
        # /32 routes to many addresses (most unused) and the real hosts, then defaults
        addrs = (st.u64(n_run) & np.uint64(0x0003FFFF)).astype(np.uint32) | np.uint32(ip(10, 0, 0, 0))
        for i, a in enumerate(addrs):
            t.append(rule(100, int(a), 32, int(st.ints(0, hosts_per + 1, 1)[0])))
        for h in range(S * hosts_per):
            own = h // hosts_per == s
            t.append(rule(100, int(host_ip[h]), 32, h % hosts_per if own else hosts_per))
        t.append(rule(50, 0, 0, hosts_per))
        tables.append(t)
    net = make_net([hosts_per + 2] * S, links, hosts, [0] * S, tables)
    M = 6000
    pr = np.zeros(M, W.PROBE_DTYPE)
    src = st.ints(0, S * hosts_per - 1, M)
    pr["src_host"], pr["src_ip"] = src, host_ip[src]
    pick = st.floats(M)
    pr["dst_ip"] = np.where(pick < 0.5, host_ip[st.ints(0, S * hosts_per - 1, M)],
                            (st.u64(M) & np.uint64(0x0003FFFF)).astype(np.uint32) | np.uint32(ip(10, 0, 0, 0)))
    pr["dport"] = np.where(st.floats(M) < 0.3, 80, st.ints(0, 65535, M))
    pr["allowed_mask"] = 1
    validator.load_network(net)
    o = oracle.verify_probes(net, pr, 16)
    kernels = [1, 2] if B.pv_get_stat(validator.ctx, B.PV_STAT_WALK_INDEX_FITS) else [1]
    for kernel in kernels:
        assert _same(_gpu_walk(validator, net, pr, 16, kernel), o), kernel
    assert len(np.unique(o["status"])) >= 3


@pytest.mark.parametrize("seed", [1, 2, 3])
def test_index_stress_tables(validator, seed):
    net, host_ip = _index_stress_network(seed)
    st = W.Stream(seed, "index-stress-probes")
    M = 20000
    pr = np.zeros(M, W.PROBE_DTYPE)
    src = st.ints(0, net.num_hosts - 1, M)
    pr["src_host"] = src
    pr["src_ip"] = np.where(st.floats(M) < 0.8, host_ip[src], st.u64(M) & np.uint64(0xFFFFFFFF))
    pr["dst_ip"] = np.where(st.floats(M) < 0.7, host_ip[st.ints(0, net.num_hosts - 1, M)],
                            st.u64(M) & np.uint64(0xFFFFFFFF))
    edges = st.ints(0, 256, M) * BUCKET + st.ints(-2, 2, M)
    pr["dport"] = np.where(st.floats(M) < 0.5, np.clip(edges, 0, 65535), st.ints(0, 65535, M))
    pr["allowed_mask"] = 0xF
    validator.load_network(net)
    assert B.pv_get_stat(validator.ctx, B.PV_STAT_WALK_INDEX_FITS) == 1
    o = oracle.verify_probes(net, pr, 24)
    for kernel in KERNELS:
        g = _gpu_walk(validator, net, pr, 24, kernel)
        assert _same(g, o), kernel
    # indexed kernel with every batch warp-cooperative, and every batch one probe per lane
    for lane_max in (0, 65535):
        validator.set_option(B.PV_OPT_WALK_LANE_MAX, lane_max)
        try:
            g = _gpu_walk(validator, net, pr, 24, 2)
        finally:
            validator.set_option(B.PV_OPT_WALK_LANE_MAX, 96)
        assert _same(g, o), lane_max
    # every first match along the way also agrees hop by hop with the oracle's
    assert len(np.unique(o["status"])) >= 3


@pytest.mark.parametrize("tail", [0, 1, 5, 8, -1])
def test_tail_launch_agrees(validator, tail):
    """The last hops in one launch (one thread per probe, tables from L2)
    give the results of the hop-by-hop walk, from any switch-over hop, with
    and without path constraints; the live counts still add up."""
    e = W.end_to_end(seed=33, num_switches=70, num_intents=40, probes_per_intent=400, rules_per_switch=200)
    net = e.network
    pr = e.probes.probes.copy()
    st = W.Stream(33, "tail-probes")
    pr["src_host"] = st.ints(0, net.num_hosts - 1, len(pr))
    pr["src_ip"] = net.host_ip[pr["src_host"]]
    o = oracle.verify_probes(net, pr, 32)
    validator.set_option(B.PV_OPT_WALK_TAIL_HOP, tail)
    try:
        g = _gpu_walk(validator, net, pr, 32, 2)
        assert _same(g, o)
        validator.set_option(B.PV_OPT_WALK_CYCLES, 1)
        g = _gpu_walk(validator, net, pr, 32, 2)
        assert _same(g, o)
        ran = o["status"] != W.ST_NOSRC
        want = int(o["hops"][ran].astype(np.int64).sum()) - int((o["status"] == W.ST_VIOLATION).sum())
        assert B.pv_get_stat(validator.ctx, B.PV_STAT_WALK_LIVE_TOTAL) == want
        validator.set_option(B.PV_OPT_WALK_CYCLES, 0)
        from paper_2602_16100_gb300.validator import to_device as td
        pol = W.path_policies(3, net, 40, forbid_max=2, must_max=3, hubs=8)
        validator.load_policies(pol)
        out, hits = validator.verify_constrained(td(pr, validator.device), len(pr), 32, None, 400)
        validator.sync()
        oc, oh = oracle.verify_constrained(net, pr, 32, pol, probes_per_policy=400)
        assert (to_numpy(out, W.RESULT_DTYPE) == oc).all() and (to_numpy(hits, np.uint32) == oh).all()
    finally:
        validator.set_option(B.PV_OPT_WALK_TAIL_HOP, -1)
        validator.set_option(B.PV_OPT_WALK_CYCLES, 0)


def test_walk_live_total_counts_hop_entries(validator):
    """PV_STAT_WALK_LIVE_TOTAL: probes entered at a switch, summed over hops.
    A probe whose next switch (its first one included) lies outside its mask
    is judged before it enters that switch, so it counts one entry fewer
    than its result's hops."""
    d = W.fat_tree(seed=5, k=4, rules_per_switch=100, num_probes=7000, hop_cap=8)
    net, pr = d["network"], d["probes"].probes
    o = oracle.verify_probes(net, pr, 8)
    ran = o["status"] != W.ST_NOSRC
    want = int(o["hops"][ran].astype(np.int64).sum()) - int((o["status"] == W.ST_VIOLATION).sum())
    validator.set_option(B.PV_OPT_WALK_CYCLES, 1)      # every hop walked
    try:
        g = _gpu_walk(validator, net, pr, 8)
        assert _same(g, o)
        assert B.pv_get_stat(validator.ctx, B.PV_STAT_WALK_LIVE_TOTAL) == want
    finally:
        validator.set_option(B.PV_OPT_WALK_CYCLES, 0)
    g = _gpu_walk(validator, net, pr, 8)                # cycles finished early
    assert _same(g, o)
    assert B.pv_get_stat(validator.ctx, B.PV_STAT_WALK_LIVE_TOTAL) <= want


def _cycle_network():
    """Disjoint components, each a tail of t switches leading into a ring of
    R switches (every switch forwards everything to its next port), one host
    at the tail's head; one ring holds a switch of region 1.  Periods 1 (a
    switch cabled to itself) to 40, cycle entry after 0 to 20 hops."""
    nports, links, hosts, region, rules = [], [], [], [], []
    combos = [(t, R) for t in (0, 1, 3, 5, 9, 20) for R in (1, 2, 3, 5, 8, 9, 13, 40)]
    for c, (t, R) in enumerate(combos):
        base = len(nports)
        n = t + R
        for i in range(n):
            nports.append(3)                   # 0: in, 1: out, 2: host (head only)
            region.append(1 if (c % 7 == 3 and i == t + R // 2) else 0)
            rules.append([rule(100, 0, 0, 1)])  # everything out of port 1
        for i in range(n - 1):
            links.append((base + i, 1, base + i + 1, 0))
        links.append((base + n - 1, 1, base + t, 0))   # close the ring
        hosts.append((base, 2, ip(10, c, 0, 1)))
    return make_net(nports, links, hosts, region, rules), len(combos)


def test_forwarding_cycles_finish_with_the_full_walk_result(validator):
    net, C = _cycle_network()
    pr = np.concatenate([probe(h, ip(10, h, 0, 1), ip(99, 0, 0, 1), m, dport=h)
                         for h in range(C) for m in (1, 3)])
    for cap in (1, 2, 3, 4, 5, 7, 8, 9, 15, 16, 17, 31, 32, 33, 64, 100, 254, 255):
        o = oracle.verify_probes(net, pr, cap)
        for cyc in (0, 1):
            validator.set_option(B.PV_OPT_WALK_CYCLES, cyc)
            try:
                for kernel in KERNELS:
                    assert _same(_gpu_walk(validator, net, pr, cap, kernel), o), (cap, cyc, kernel)
            finally:
                validator.set_option(B.PV_OPT_WALK_CYCLES, 0)
        if cap == 255:
            assert (o["status"] == W.ST_LOOP).sum() > C and (o["status"] == W.ST_VIOLATION).any()
    # the shortcut does less work on the long cap
    validator.set_option(B.PV_OPT_WALK_CYCLES, 1)
    try:
        _gpu_walk(validator, net, pr, 255)
        full = B.pv_get_stat(validator.ctx, B.PV_STAT_WALK_LIVE_TOTAL)
    finally:
        validator.set_option(B.PV_OPT_WALK_CYCLES, 0)
    _gpu_walk(validator, net, pr, 255)
    assert B.pv_get_stat(validator.ctx, B.PV_STAT_WALK_LIVE_TOTAL) < full // 2


def _bounce_network(kinds=("pingpong", "once", "region")):
    """Components of a tail of t switches, then A, B and C: A sends
    everything to B (with kind "once", what comes back from B goes to C
    instead), B sends everything back to A (a bounce: out by the port it
    came in by), C delivers to its host.  With kind "pingpong" A bounces
    too, so the walk alternates A, B from its first bounce on; with
    "region" B lies in region 1.  The source host sits at the head switch."""
    nports, links, hosts, region, rules, comps = [], [], [], [], [], []
    for kind in kinds:
        for t in (0, 1, 2, 3, 5, 9):
            base = len(nports)
            for i in range(t):                         # tail: 0 in, 1 out, 2 host (head only)
                nports.append(3)
                region.append(0)
                rules.append([rule(100, 0, 0, 1)])
            a, b, c = base + t, base + t + 1, base + t + 2
            nports += [4, 1, 2]                        # A: 0 in, 1 to B, 2 host (head), 3 to C; B: 0; C: 0, 1 host
            region += [0, 1 if kind == "region" else 0, 0]
            ra = [rule(100, 0, 0, 1)]
            if kind == "once":
                ra = [rule(200, 0, 0, 3, in_port=1)] + ra
            rules += [ra, [rule(100, 0, 0, 0)], [rule(100, 0, 0, 1)]]
            for i in range(t - 1):
                links.append((base + i, 1, base + i + 1, 0))
            if t:
                links.append((base + t - 1, 1, a, 0))
            links += [(a, 1, b, 0), (a, 3, c, 0)]
            head = base if t else a
            src = len(hosts)
            hosts.append((head, 2, ip(10, len(comps), 0, 1)))
            hosts.append((c, 1, ip(10, len(comps), 0, 2)))
            comps.append((kind, t, src))
    return make_net(nports, links, hosts, region, rules), comps


def _bounce_probes(comps):
    pr = [probe(src, ip(10, c, 0, 1), ip(10, c, 0, 2), m, dport=c) for c, (_, _, src) in enumerate(comps)
          for m in (1, 3)]
    return np.concatenate(pr)


BOUNCE_CAPS = (1, 2, 3, 4, 5, 6, 7, 8, 9, 10, 15, 16, 17, 31, 32, 33, 100, 254, 255)


@pytest.mark.parametrize("tail", [-1, 0, 1, 3])
def test_two_switch_cycles_finish_at_the_second_bounce(validator, tail):
    """A probe that leaves two switches in a row by the port it entered
    through is in a two-switch cycle (symmetric cabling): its walk ends
    there with the full walk's result (LOOP, the hop cap, the switch of the
    last visit by parity), for every cap, both first-match kernels, any tail
    switch-over hop and with the cycle shortcuts off."""
    net, comps = _bounce_network()
    pr = _bounce_probes(comps)
    validator.set_option(B.PV_OPT_WALK_TAIL_HOP, tail)
    try:
        for cap in BOUNCE_CAPS:
            o = oracle.verify_probes(net, pr, cap)
            for cyc in (0, 1):
                validator.set_option(B.PV_OPT_WALK_CYCLES, cyc)
                for kernel in KERNELS:
                    assert _same(_gpu_walk(validator, net, pr, cap, kernel), o), (cap, cyc, kernel)
            validator.set_option(B.PV_OPT_WALK_CYCLES, 0)
            if cap == 255:
                kinds = np.repeat([k for k, _, _ in comps], 2)
                assert (o["status"][kinds == "pingpong"] == W.ST_LOOP).all()
                assert (o["status"][kinds == "once"] == W.ST_COMPLIANT).all()
        # pure ping-pong components: each probe enters its tail, A, B and A
        # again, and no further switch
        pnet, pcomps = _bounce_network(("pingpong",))
        ppr = _bounce_probes(pcomps)
        for cap in (3, 4, 8, 32, 255):
            o = oracle.verify_probes(pnet, ppr, cap)
            assert _same(_gpu_walk(validator, pnet, ppr, cap, 2), o)
            want = sum(2 * min(cap, t + 3) for _, t, _ in pcomps)
            assert B.pv_get_stat(validator.ctx, B.PV_STAT_WALK_LIVE_TOTAL) == want, cap
    finally:
        validator.set_option(B.PV_OPT_WALK_TAIL_HOP, -1)
        validator.set_option(B.PV_OPT_WALK_CYCLES, 0)


def test_bounces_on_asymmetric_cabling_are_walked_out(validator):
    """With cabling that is not symmetric two bounces in a row prove no
    two-switch cycle: X, Y and Z each send everything out of port 0, which
    leads X -> Y -> Z -> X, so every hop after the first is a bounce and the
    period is 3.  The walk must take every visit (one ping-pong component on
    symmetric links shares the tables) and still match the oracle."""
    nports = [2, 1, 1]
    rules = [[rule(100, 0, 0, 0)], [rule(100, 0, 0, 0)], [rule(100, 0, 0, 0)]]
    net0, comps = _bounce_network(("pingpong",))
    base = net0.num_switches
    nports_all = list(np.diff(net0.port_offs).astype(int)) + nports
    rules_all = [[net0.rules[j:j + 1] for j in range(int(net0.rule_offs[s]), int(net0.rule_offs[s + 1]))]
                 for s in range(base)] + rules
    links = []
    for s in range(base):
        for p in range(int(net0.port_offs[s]), int(net0.port_offs[s + 1])):
            peer = int(net0.port_peer[p])
            if peer >= 0 and not peer & W.HOST_BIT and (s, p - int(net0.port_offs[s])) < (peer >> 8, peer & 0xFF):
                links.append((s, p - int(net0.port_offs[s]), peer >> 8, peer & 0xFF))
    hosts = [(int(net0.host_switch[h]), int(net0.host_port[h]), int(net0.host_ip[h]))
             for h in range(net0.num_hosts)] + [(base, 1, ip(10, 200, 0, 1))]
    region = list(net0.switch_region) + [0, 0, 0]
    net = make_net(nports_all, links, hosts, region, rules_all)
    x, y, z = base, base + 1, base + 2
    po = net.port_offs
    net.port_peer[po[x]] = (y << 8) | 0
    net.port_peer[po[y]] = (z << 8) | 0
    net.port_peer[po[z]] = (x << 8) | 0
    pr = np.concatenate([_bounce_probes(comps),
                         probe(len(hosts) - 1, ip(10, 200, 0, 1), ip(99, 0, 0, 1), 1),
                         probe(len(hosts) - 1, ip(10, 200, 0, 1), ip(99, 0, 0, 1), 3, dport=7)])
    for cap in BOUNCE_CAPS:
        o = oracle.verify_probes(net, pr, cap)
        for kernel in KERNELS:
            assert _same(_gpu_walk(validator, net, pr, cap, kernel), o), (cap, kernel)
        if cap == 255:
            assert o["status"][-1] == W.ST_LOOP and o["last_switch"][-1] == [x, y, z][254 % 3]


@pytest.mark.parametrize("kernel", KERNELS)
def test_stalled_staging_wait_times_out_and_context_recovers(validator, kernel):
    """A staging barrier that expects bytes no copy delivers: each hop block's
    bounded wait runs out, pv_sync reports PV_ETIMEOUT, and the same context
    then walks correctly (no fault, no hang)."""
    d = W.fat_tree(seed=3, k=4, rules_per_switch=100, num_probes=5000, hop_cap=8)
    net, pr = d["network"], d["probes"].probes
    validator.load_network(net)
    dev = validator.device
    d_pr = to_device(pr, dev)
    validator.set_option(B.PV_OPT_WALK_KERNEL, kernel)
    validator.set_option(B.PV_OPT_TEST_STALL_STAGING, 1)
    try:
        validator.verify_probes(d_pr, len(pr), 8)
        with pytest.raises(B.PVError) as e:
            validator.sync()
        assert e.value.code == B.PV_ETIMEOUT
    finally:
        validator.set_option(B.PV_OPT_TEST_STALL_STAGING, 0)
        validator.set_option(B.PV_OPT_WALK_KERNEL, 0)
    g = _gpu_walk(validator, net, pr, 8, kernel)
    assert _same(g, oracle.verify_probes(net, pr, 8))


@pytest.mark.parametrize("kernel", [0] + KERNELS)
def test_flow_verification_full_size(validator, kernel):
    """The full flow-verification workload (10M probes) in the benchmark's
    launch configuration (kernel 0: the library's choice) and with each
    first-match kernel; every probe's result is compared with the oracle's."""
    d = W.fat_tree()
    net, P = d["network"], d["probes"]
    g = _gpu_walk(validator, net, P.probes, P.hop_cap, kernel)
    o = F.cached("flow-verification/default", lambda: {"r": F.verify_probes(net, P.probes, P.hop_cap)})["r"]
    assert _same(g, o)
    assert (g["status"] <= W.ST_MISDELIVERED).all()
    assert len(np.unique(o["status"])) == 5


def _scan_totals(net, probes, cap):
    """(first matches, summed scan depth) of the walk's definition: at every
    visit to a permitted switch the first match is taken by scanning the
    switch's rules in first-match order (priority descending, then input
    order); the depth is the hit's position + 1, or the rule count on a
    miss.  Every hop is walked (no cycle shortcut)."""
    per = []
    for s in range(net.num_switches):
        rs = net.rules[net.rule_offs[s]:net.rule_offs[s + 1]]
        order = sorted(range(len(rs)), key=lambda i: (-int(rs[i]["priority"]), i))
        r = rs[order]
        lens = lambda L: np.where(L == 0, 0, (0xFFFFFFFF << (32 - L.astype(np.int64))) & 0xFFFFFFFF)
        per.append((r, lens(r["src_len"]), lens(r["dst_len"])))
    n_fm = depth = 0
    for pr in probes:
        h = int(pr["src_host"])
        if h >= net.num_hosts:
            continue
        s, p = int(net.host_switch[h]), int(net.host_port[h])
        src, dst, dport, mask = int(pr["src_ip"]), int(pr["dst_ip"]), int(pr["dport"]), int(pr["allowed_mask"])
        for _ in range(cap):
            reg = int(net.switch_region[s])
            if reg >= 32 or not (mask >> reg) & 1:
                break
            r, ms, md = per[s]
            hit = (((r["in_port"] == W.ANY_PORT) | (r["in_port"] == p))
                   & ((src & ms) == (r["src_ip"].astype(np.int64) & ms))
                   & ((dst & md) == (r["dst_ip"].astype(np.int64) & md))
                   & (r["dport_lo"] <= dport) & (dport <= r["dport_hi"]))
            j = int(np.argmax(hit)) if hit.any() else -1
            n_fm += 1
            depth += j + 1 if j >= 0 else len(r)
            if j < 0 or int(r[j]["action"]) == W.DROP:
                break
            port = int(r[j]["action"])
            if port >= int(net.port_offs[s + 1] - net.port_offs[s]):
                break
            peer = int(net.port_peer[net.port_offs[s] + port])
            if peer < 0 or peer & W.HOST_BIT:
                break
            s, p = peer >> 8, peer & 0xFF
    return n_fm, depth


@pytest.mark.parametrize("kernel,tail", [(1, 0), (2, 0), (2, 3)])
def test_walk_statistics_count_first_matches_and_scan_depth(validator, kernel, tail):
    """PV_OPT_WALK_STATS: the counting kernels give the same results; their
    first-match count and ordered-scan depth equal those of the walk's
    definition recomputed here; the index never disagrees with the scan and
    tests no more candidates than the scan passes."""
    d = W.fat_tree(seed=9, k=4, rules_per_switch=120, num_probes=2500, hop_cap=8)
    net, pr = d["network"], d["probes"].probes
    o = oracle.verify_probes(net, pr, 8)
    want_fm, want_depth = _scan_totals(net, pr, 8)
    v = validator
    v.set_option(B.PV_OPT_WALK_CYCLES, 1)
    v.set_option(B.PV_OPT_WALK_TAIL_HOP, tail)
    v.set_option(B.PV_OPT_WALK_STATS, 1)
    try:
        g = _gpu_walk(v, net, pr, 8, kernel)
        stat = lambda k: B.pv_get_stat(v.ctx, k)
        fm, tests, looks = stat(B.PV_STAT_WALK_FIRST_MATCHES), stat(B.PV_STAT_WALK_RULE_TESTS), \
            stat(B.PV_STAT_WALK_INTERVAL_LOOKUPS)
        depth, bad = stat(B.PV_STAT_WALK_SCAN_DEPTH), stat(B.PV_STAT_WALK_INDEX_MISMATCHES)
    finally:
        v.set_option(B.PV_OPT_WALK_STATS, 0)
        v.set_option(B.PV_OPT_WALK_TAIL_HOP, -1)
        v.set_option(B.PV_OPT_WALK_CYCLES, 0)
    assert _same(g, o)
    assert (fm, depth, bad) == (want_fm, want_depth, 0)
    assert want_fm > 1000 and tests > 0
    if kernel == 1:
        assert looks == 0 and tests % 32 == 0 and tests >= depth
    else:
        assert looks > 0 and tests + looks <= depth
    # the default kernels leave the counters of the last statistics walk alone
    g2 = _gpu_walk(v, net, pr, 8, kernel)
    assert _same(g2, o) and B.pv_get_stat(v.ctx, B.PV_STAT_WALK_FIRST_MATCHES) == fm
