"""GPU parity of the path-constraint checks against the oracle (bit-exact
status, hops, last switch and waypoint bits): the backup-switch waypoint
case, random networks and policies under both first-match kernels, hop caps
that do and do not reach the forwarding-cycle shortcut, per-probe and
strided policy indices, the constrained end-to-end verdict (with intents
that pass, fail on a missed waypoint or a forbidden switch, or fail for want
of a concrete flow), invalid calls, and the full end-to-end workload with a
policy per intent on every output."""
import numpy as np
import pytest

import oracle
from paper_2602_16100_gb300 import binding as B
from paper_2602_16100_gb300 import workloads as W
from paper_2602_16100_gb300.validator import flow_columns_of, empty_device, to_device, to_numpy
from gpu_util import E2E_CONSTRAINED, POLICIES_CONSTRAINED
from test_oracle_policies import _backup_switch_net, _policies
from netbuild import probe

pytestmark = pytest.mark.gpu


def _walk(v, net, pol, pr, cap, probe_policy=None, per=0, kernel=0):
    v.load_network(net)
    v.load_policies(pol)
    dev = v.device
    dpp = None if probe_policy is None else to_device(np.asarray(probe_policy, np.uint32), dev)
    v.set_option(B.PV_OPT_WALK_KERNEL, kernel)
    try:
        out, hits = v.verify_constrained(to_device(pr, dev), len(pr), cap, dpp, per)
        v.sync()
    finally:
        v.set_option(B.PV_OPT_WALK_KERNEL, 0)
    return to_numpy(out, W.RESULT_DTYPE), to_numpy(hits, np.uint32)


@pytest.mark.parametrize("via_backup", [True, False])
@pytest.mark.parametrize("kernel", [1, 2])
def test_backup_switch_waypoint(validator, via_backup, kernel):
    net, H2, H4 = _backup_switch_net(via_backup)
    pol = _policies([[], [8], [5]], [[8], [8], [8, 5]])
    pr = np.concatenate([probe(0, H2, H4, 1)] * 4)
    pp = np.array([0, 1, 2, 9], np.uint32)
    g, gh = _walk(validator, net, pol, pr, 16, pp, kernel=kernel)
    o, oh = oracle.verify_constrained(net, pr, 16, pol, probe_policy=pp)
    assert (g == o).all() and (gh == oh).all()


@pytest.mark.parametrize("seed,cap", [(0, 24), (1, 32), (2, 3), (3, 255)])
@pytest.mark.parametrize("kernel", [1, 2])
def test_random_policies(validator, seed, cap, kernel):
    e = W.end_to_end(seed=60 + seed, num_switches=80, num_intents=50, probes_per_intent=200, rules_per_switch=200,
                     hop_cap=cap)
    net = e.network
    pol = W.path_policies(seed, net, 50, forbid_max=3, must_max=4, hubs=10)
    pr = e.probes.probes.copy()
    st = W.Stream(seed, "gpu-policy-probes")
    H = net.num_hosts
    pr["src_host"] = st.ints(0, H - 1, len(pr))
    pr["src_ip"] = net.host_ip[pr["src_host"]]
    pr["src_host"][::23] = W.NO_HOST
    pr["allowed_mask"][::3] = 0xFFFFFFFF
    g, gh = _walk(validator, net, pol, pr, cap, per=200, kernel=kernel)
    o, oh = oracle.verify_constrained(net, pr, cap, pol, probes_per_policy=200)
    assert (g == o).all() and (gh == oh).all()
    assert (oh != 0).any() and (o["status"] == W.ST_VIOLATION).any()
    # explicit policy indices, some past the table (no constraint: the plain walk)
    pp = (np.arange(len(pr)) % 57).astype(np.uint32)
    g2, gh2 = _walk(validator, net, pol, pr, cap, pp, kernel=kernel)
    o2, oh2 = oracle.verify_constrained(net, pr, cap, pol, probe_policy=pp)
    assert (g2 == o2).all() and (gh2 == oh2).all()
    plain = pp >= 50
    assert (o2[plain] == oracle.verify_probes(net, pr[plain], cap)).all() and not oh2[plain].any()


def test_constrained_end_to_end(validator):
    e = W.end_to_end(**E2E_CONSTRAINED)
    kw = dict(POLICIES_CONSTRAINED)
    pol = W.path_policies(kw.pop("seed"), e.network, e.intents.num_pods, **kw)
    v = validator
    v.load_cluster(e.cluster)
    v.load_network(e.network)
    v.load_policies(pol)
    dev, sizes = v.alloc_end_to_end(e)
    I, pods, ppg = sizes["intents"], sizes["pods"], sizes["probes_per_intent"]
    words = W.words_per_row(e.cluster.num_nodes)
    B.pv_eval_selectors(v.ctx, I, dev["offs"], sizes["num_exprs"], dev["exprs"], None, dev["bits"], words,
                        dev["flags"])
    B.pv_place_pods(v.ctx, I, pods, dev["bits"], words, dev["draws"], dev["assign"])
    B.pv_bind_probes(v.ctx, I * ppg, dev["probes"], ppg, pods, dev["assign"])
    hits = empty_device(I * ppg * 4, v.device)
    B.pv_verify_probes_constrained(v.ctx, I * ppg, dev["probes"], sizes["hop_cap"], None, ppg, dev["results"], hits)
    B.pv_aggregate_constrained(v.ctx, I, pods, dev["bits"], words, dev["flags"], dev["assign"], ppg, dev["results"],
                               hits, None, dev["pass"], dev["counts"])
    v.sync()
    c = e.cluster
    bits, flags = oracle.eval_selectors(c.num_nodes, c.num_keys, c.labels, e.intents.expr_offs, e.intents.exprs)
    assign = oracle.place_pods(bits, c.num_nodes, pods, e.place_draws)
    probes = oracle.bind_probes(e.probes.probes, ppg, pods, assign, e.network.host_ip)
    res, oh = oracle.verify_constrained(e.network, probes, e.probes.hop_cap, pol, probes_per_policy=ppg)
    passed, counts = oracle.aggregate_constrained(bits, c.num_nodes, flags, assign, pods, res, ppg, oh, pol)
    assert (to_numpy(dev["results"], W.RESULT_DTYPE) == res).all()
    assert (to_numpy(hits, np.uint32) == oh).all()
    assert (to_numpy(dev["pass"], np.uint8)[:I] == passed).all()
    assert (to_numpy(dev["counts"], np.uint32, (I, 8)) == counts).all()
    assert counts[:, 7].any() and passed.any()


def test_invalid_policy_calls(validator):
    d = W.tiny()
    net = d["network"]
    fresh = B.pv_create(validator.device.index)
    try:
        with pytest.raises(B.PVError) as e:     # no flow tables yet
            B.pv_load_path_policies(fresh, 1, np.array([0, 0], np.uint32), np.zeros(0, np.uint16),
                                    np.array([0, 1], np.uint32), np.array([1], np.uint16), np.ones(1, np.uint8))
        assert e.value.code == B.PV_ESTATE
    finally:
        B.pv_destroy(fresh)
    validator.load_network(net)
    S = net.num_switches
    bad = [(np.array([0, 0], np.uint32), np.zeros(0, np.uint16), np.array([0, 33], np.uint32),
            np.zeros(33, np.uint16)),                                           # > 32 waypoints
           (np.array([0, 1], np.uint32), np.array([S], np.uint16), np.array([0, 0], np.uint32),
            np.zeros(0, np.uint16)),                                            # switch out of range
           (np.array([0, 2, 1], np.uint32), np.zeros(2, np.uint16), np.array([0, 0, 0], np.uint32),
            np.zeros(0, np.uint16))]                                            # decreasing offsets
    for fo, f, mo, m in bad:
        with pytest.raises(B.PVError) as e:
            B.pv_load_path_policies(validator.ctx, len(fo) - 1, fo, f, mo, m, np.ones(len(fo) - 1, np.uint8))
        assert e.value.code == B.PV_EINVAL
    pr = to_device(d["probes"].probes, validator.device)
    out = empty_device(4 * len(d["probes"].probes), validator.device)
    validator.load_policies(_policies([[1]], [[2]]))
    with pytest.raises(B.PVError):                                              # NULL waypoint output
        B.pv_verify_probes_constrained(validator.ctx, 10, pr, 16, None, 10, out, None)


@pytest.mark.parametrize("variant", ["plain", "pass"])
def test_full_size_end_to_end_policies(validator, variant):
    """The full end-to-end workload (10,000 intents, 50M probes) with one
    policy per intent, in the benchmark's launch configuration (plain), and
    its variant in which intents can pass (pass); every result, waypoint
    word, verdict and count is compared with the oracle's."""
    from test_gpu_reach_e2e import _check_e2e_full
    e = W.end_to_end(**({"pass_share": 0.3} if variant == "pass" else {}))
    pol = W.path_policies(20260221, e.network, e.intents.num_pods)
    v = validator
    v.load_cluster(e.cluster)
    v.load_network(e.network)
    v.load_policies(pol)
    dev, sizes = v.alloc_end_to_end(e, with_policies=True)
    v.run_end_to_end(dev, sizes)
    v.sync()
    I, words = sizes["intents"], W.words_per_row(e.cluster.num_nodes)
    g = {"bits": to_numpy(dev["bits"], np.uint32, (I, words)), "flags": to_numpy(dev["flags"], np.uint8),
         "assign": to_numpy(dev["assign"], np.uint32), "results": to_numpy(dev["results"], W.RESULT_DTYPE),
         "hits": to_numpy(dev["hits"], np.uint32), "pass": to_numpy(dev["pass"], np.uint8),
         "counts": to_numpy(dev["counts"], np.uint32, (I, 8))}
    want = _check_e2e_full(g, e, f"end-to-end-policies/{variant}", pol)
    assert want["hits"].any()
    if variant == "pass":
        assert want["passed"].any()


@pytest.mark.parametrize("chunks", [1, 3])
def test_constrained_pipeline_from_host(validator, chunks):
    """The host-buffer pipeline with path policies, cut into intent chunks
    (each chunk keeps its intents' policies through first_policy)."""
    import torch
    from test_gpu_reach_e2e import _pinned
    e = W.end_to_end(seed=26, num_switches=64, num_intents=203, probes_per_intent=80, rules_per_switch=200,
                     pass_share=0.3)
    pol = W.path_policies(8, e.network, 203, forbid_max=1, must_max=2, hubs=6, p_noop=0.1)
    v = validator
    v.load_cluster(e.cluster)
    v.load_network(e.network)
    v.load_policies(pol)
    dev, sizes = v.alloc_end_to_end(e, with_policies=True)
    I, pods, ppg = sizes["intents"], sizes["pods"], sizes["probes_per_intent"]
    host = {"offs": _pinned(e.intents.expr_offs.astype(np.uint32)), "exprs": _pinned(e.intents.exprs),
            "draws": _pinned(e.place_draws.astype(np.uint64)), "masks": _pinned(e.intent_mask.astype(np.uint32)),
            "dst": _pinned(flow_columns_of(e)[0]), "dport": _pinned(flow_columns_of(e)[1]),
            "pass": torch.zeros(I, dtype=torch.uint8).pin_memory(),
            "counts": torch.zeros(I * 32, dtype=torch.uint8).pin_memory()}
    stream = torch.cuda.current_stream()
    v.run_end_to_end_from_host(host, dev, sizes, stream, torch.cuda.Stream(), chunks)
    stream.synchronize()
    v.sync()
    c = e.cluster
    bits, flags = oracle.eval_selectors(c.num_nodes, c.num_keys, c.labels, e.intents.expr_offs, e.intents.exprs)
    assign = oracle.place_pods(bits, c.num_nodes, pods, e.place_draws)
    probes = oracle.bind_probes(e.probes.probes, ppg, pods, assign, e.network.host_ip)
    res, oh = oracle.verify_constrained(e.network, probes, e.probes.hop_cap, pol, probes_per_policy=ppg)
    passed, counts = oracle.aggregate_constrained(bits, c.num_nodes, flags, assign, pods, res, ppg, oh, pol)
    assert (to_numpy(dev["hits"], np.uint32) == oh).all()
    assert (host["pass"].numpy() == passed).all()
    assert (host["counts"].numpy().view(np.uint32).reshape(I, 8) == counts).all()
    assert passed.any()


@pytest.mark.parametrize("form", ["records", "columns"])
@pytest.mark.parametrize("policy_form", ["per_group", "per_probe", "per_pair_of_groups", "none"])
def test_flow_verification_direct_and_regrouped_first_hop_agree(validator, policy_form, form):
    """pv_verify_flows(_constrained) lists compact flows straight into the
    first hop's switch order when each group has one path constraint (no
    constraint, or probes_per_policy a multiple of the group size) and
    regroups them otherwise (a per-probe policy array, or a stride that cuts
    groups).  Both give the oracle's results, records and waypoint bits; a
    ragged last group (M not a multiple of the group size) is included.  The
    flows are given as 8-byte records or as the two columns of
    pv_verify_flow_columns(_constrained), read from a 2-byte offset."""
    e = W.end_to_end(seed=41, num_switches=64, num_intents=120, probes_per_intent=70, rules_per_switch=160)
    v = validator
    v.load_cluster(e.cluster)
    v.load_network(e.network)
    I, pods, ppg = e.intents.num_pods, e.pods_per_intent, e.probes_per_intent
    M = I * ppg - 33                                    # ragged last group
    pol = W.path_policies(43, e.network, 2 * I, forbid_max=1, must_max=2, hubs=6, p_noop=0.1)
    v.load_policies(pol)
    dev, sizes = v.alloc_end_to_end(e)
    words = W.words_per_row(e.cluster.num_nodes)
    B.pv_eval_selectors(v.ctx, I, dev["offs"], sizes["num_exprs"], dev["exprs"], None, dev["bits"], words,
                        dev["flags"])
    B.pv_place_pods(v.ctx, I, pods, dev["bits"], words, dev["draws"], dev["assign"])
    c = e.cluster
    bits, _ = oracle.eval_selectors(c.num_nodes, c.num_keys, c.labels, e.intents.expr_offs, e.intents.exprs)
    assign = oracle.place_pods(bits, c.num_nodes, pods, e.place_draws)
    probes = oracle.bind_probes(e.probes.probes[:M], ppg, pods, assign, e.network.host_ip)
    dp, out = empty_device(M * 16, v.device), empty_device(M * 4, v.device)
    dst = dev["dst"]
    dport = empty_device(M * 2 + 2, v.device)[2:]       # columns need only their element alignment
    dport.copy_(dev["dport"][: M * 2])
    if policy_form == "none":
        if form == "records":
            B.pv_verify_flows(v.ctx, M, dev["flows"], ppg, pods, dev["assign"], dev["masks"], sizes["hop_cap"], dp,
                              out)
        else:
            B.pv_verify_flow_columns(v.ctx, M, dst, dport, ppg, pods, dev["assign"], dev["masks"], sizes["hop_cap"],
                                     dp, out)
        v.sync()
        assert (to_numpy(out, W.RESULT_DTYPE) == oracle.verify_probes(e.network, probes, sizes["hop_cap"])).all()
        assert (to_numpy(dp, W.PROBE_DTYPE) == probes).all()
        return
    per = {"per_group": ppg, "per_probe": 0, "per_pair_of_groups": ppg // 2}[policy_form]
    pp = None
    if policy_form == "per_probe":
        pp_host = (np.arange(M) // ppg).astype(np.uint32)     # the per-group policy, given per probe
        pp = to_device(pp_host, v.device)
    hits = empty_device(M * 4, v.device)
    if form == "records":
        B.pv_verify_flows_constrained(v.ctx, M, dev["flows"], ppg, pods, dev["assign"], dev["masks"],
                                      sizes["hop_cap"], pp, per, 0, dp, out, hits)
    else:
        B.pv_verify_flow_columns_constrained(v.ctx, M, dst, dport, ppg, pods, dev["assign"], dev["masks"],
                                             sizes["hop_cap"], pp, per, 0, dp, out, hits)
    v.sync()
    if policy_form == "per_probe":
        res, oh = oracle.verify_constrained(e.network, probes, sizes["hop_cap"], pol, probe_policy=pp_host)
    else:
        res, oh = oracle.verify_constrained(e.network, probes, sizes["hop_cap"], pol, probes_per_policy=per)
    assert (to_numpy(out, W.RESULT_DTYPE) == res).all()
    assert (to_numpy(hits, np.uint32) == oh).all()
    assert (to_numpy(dp, W.PROBE_DTYPE) == probes).all()
