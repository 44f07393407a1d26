"""GPU parity of the path scheduler and rule compilation against the oracle
(bit-exact visits, lengths, statuses and rules), and the closed loop on the
GPU: rules installed through pv_install_path_rules, every scheduled flow's
probe walked by the constrained walk is delivered compliant along its
visits with all waypoints entered.  Random networks with and without link
weights and policies, short max_len, the backup-switch case, invalid calls,
and the end-to-end network with 10,000 requests."""
import numpy as np
import pytest

import oracle
from paper_2602_16100_gb300 import binding as B
from paper_2602_16100_gb300 import workloads as W
from paper_2602_16100_gb300.validator import empty_device, to_device, to_numpy
from test_oracle_policies import _backup_switch_net, _policies

pytestmark = pytest.mark.gpu


def _gpu_schedule(v, req, weights, max_len):
    dev = v.device
    R = len(req)
    vis = empty_device(R * max_len * 4, dev)
    ln = empty_device(R, dev)
    st = empty_device(R, dev)
    d_req = to_device(req, dev)
    d_w = None if weights is None else to_device(np.asarray(weights, np.uint16), dev)
    B.pv_schedule_paths(v.ctx, R, d_req, d_w, max_len, vis, ln, st)
    v.sync()
    return d_req, vis, ln, st


def _run(v, net, req, pol, weights, max_len):
    v.load_network(net)
    if pol is not None:
        v.load_policies(pol)
    d_req, vis, ln, st = _gpu_schedule(v, req, weights, max_len)
    R = len(req)
    g_st = to_numpy(st, np.uint8)
    g_ln = to_numpy(ln, np.uint8)
    g_vis = to_numpy(vis, np.uint32, (R, max_len))
    o_vis, o_ln, o_st = oracle.schedule_paths(net, req, pol, weights, max_len)
    assert (g_st == o_st).all()
    assert (g_ln == o_ln).all()
    for r in np.nonzero(o_st == W.PATH_OK)[0]:
        assert (g_vis[r, : o_ln[r]] == o_vis[r, : o_ln[r]]).all(), r
    # rules
    rules = empty_device(R * max_len * W.RULE_DTYPE.itemsize, v.device)
    rsw = empty_device(R * max_len * 2, v.device)
    B.pv_compile_path_rules(v.ctx, R, d_req, max_len, vis, ln, st, 65535, rules, rsw)
    v.sync()
    o_rules, o_rsw = oracle.compile_path_rules(net, req, o_vis, o_ln, o_st)
    g_rsw = to_numpy(rsw, np.uint16)
    assert (g_rsw == o_rsw).all()
    used = o_rsw != 0xFFFF
    assert (to_numpy(rules, W.RULE_DTYPE)[used] == o_rules[used]).all()
    return d_req, rules, rsw, o_ln, o_st


def _closed_loop(v, net, req, pol, rules, rsw, o_ln, o_st):
    B.pv_install_path_rules(v.ctx, len(rsw) // 2, rules, rsw)
    okr = np.nonzero(o_st == W.PATH_OK)[0]
    pr = np.zeros(len(okr), W.PROBE_DTYPE)
    pr["src_host"] = req["src_host"][okr]
    pr["src_ip"] = net.host_ip[req["src_host"][okr]]
    pr["dst_ip"] = net.host_ip[req["dst_host"][okr]]
    pr["dport"] = np.arange(len(okr)) * 7919 % 65536
    pr["allowed_mask"] = req["allowed_mask"][okr]
    pp = req["policy"][okr].astype(np.uint32)
    polx = pol if pol is not None else _policies([[]], [[]])
    v.load_policies(polx)
    dev = v.device
    out, hits = v.verify_constrained(to_device(pr, dev), len(pr), 255, to_device(pp, dev), 0)
    v.sync()
    res = to_numpy(out, W.RESULT_DTYPE)
    h = to_numpy(hits, np.uint32)
    assert (res["status"] == W.ST_COMPLIANT).all()
    assert (res["hops"] == o_ln[okr]).all()
    nm = np.array([int(polx.must_offs[p + 1] - polx.must_offs[p]) if p < polx.num_policies else 0 for p in pp])
    assert (h == ((1 << nm) - 1)).all()


@pytest.mark.parametrize("kernel", [0, 1, 2])   # automatic; links from global memory; staged
@pytest.mark.parametrize("seed,weighted,with_pol,max_len", [(0, False, False, 64), (1, True, True, 64),
                                                              (2, True, True, 10), (3, False, True, 255)])
def test_random_schedules_and_closed_loop(validator, seed, weighted, with_pol, max_len, kernel):
    e = W.end_to_end(seed=80 + seed, num_switches=90, num_intents=4, probes_per_intent=4, rules_per_switch=120)
    net = e.network
    pol = W.path_policies(seed, net, 60, forbid_max=3, must_max=3, hubs=12) if with_pol else None
    req = W.path_requests(seed, net, 400, num_policies=60 if with_pol else 0, extra_regions=(4, 12), bad_hosts=2)
    weights = None
    if weighted:
        weights = W.Stream(seed, "gpu-weights").ints(0, 30, int(net.port_offs[-1])).astype(np.uint16)
    validator.set_option(B.PV_OPT_SCHED_KERNEL, kernel)
    try:
        d_req, rules, rsw, o_ln, o_st = _run(validator, net, req, pol, weights, max_len)
    finally:
        validator.set_option(B.PV_OPT_SCHED_KERNEL, 0)
    assert (o_st == W.PATH_OK).sum() > 50
    _closed_loop(validator, net, req, pol, rules, rsw, o_ln, o_st)


def test_backup_switch_schedule(validator):
    net, H2, H4 = _backup_switch_net(via_backup=False)
    weights = np.ones(int(net.port_offs[-1]), np.uint16)
    weights[net.port_offs[2] + 1] = 2
    pol = _policies([[], [], [5], [8]], [[], [8], [8], [8]])
    req = np.zeros(4, W.PATH_REQ_DTYPE)
    req["src_host"], req["dst_host"], req["allowed_mask"] = 0, 1, 1
    req["policy"] = [0, 1, 2, 3]
    _run(validator, net, req, pol, weights, 16)


def test_invalid_schedule_calls(validator):
    d = W.tiny()
    validator.load_network(d["network"])
    req = to_device(np.zeros(2, W.PATH_REQ_DTYPE), validator.device)
    buf = empty_device(1024, validator.device)
    for max_len in (0, 256):
        with pytest.raises(B.PVError) as e:
            B.pv_schedule_paths(validator.ctx, 2, req, None, max_len, buf, buf, buf)
        assert e.value.code == B.PV_EINVAL
    with pytest.raises(B.PVError):
        B.pv_schedule_paths(validator.ctx, 2, req, None, 8, None, buf, buf)


def test_end_to_end_network_10000_requests(validator):
    e = W.end_to_end()
    net = e.network
    pol = W.path_policies(13, net, 10_000)
    req = W.path_requests(14, net, 10_000, num_policies=10_000, extra_regions=(6, 14))
    validator.load_network(net)
    validator.load_policies(pol)
    d_req, vis, ln, st = _gpu_schedule(validator, req, None, 64)
    g_st = to_numpy(st, np.uint8)
    g_ln = to_numpy(ln, np.uint8)
    g_vis = to_numpy(vis, np.uint32, (len(req), 64))
    idx = np.arange(0, len(req), 25)
    o_vis, o_ln, o_st = oracle.schedule_paths(net, req[idx], pol, None, 64)
    assert (g_st[idx] == o_st).all() and (g_ln[idx] == o_ln).all()
    for k, r in enumerate(idx):
        if o_st[k] == W.PATH_OK:
            assert (g_vis[r, : o_ln[k]] == o_vis[k, : o_ln[k]]).all()
    assert (g_st == W.PATH_OK).sum() > 1000
