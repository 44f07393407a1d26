"""GPU parity of node-selector evaluation against the oracle (bit-exact):
both kernels (label-tile comparison and per-value bitset rows), ragged node
counts spanning several tiles, absent labels, hallucinated values,
DoesNotExist, malformed expressions, empty inputs, and the placement-scale
workload (100,000 pods x 5,000 nodes) on every row and flag."""
import numpy as np
import pytest
import torch

import oracle
from paper_2602_16100_gb300 import binding as B
from paper_2602_16100_gb300 import workloads as W
from paper_2602_16100_gb300.validator import empty_device, to_device, to_numpy
import full_oracle as F

pytestmark = pytest.mark.gpu


def _gpu_eval(v, cluster, sel, kernel, words=None):
    v.load_cluster(cluster)
    v.set_option(B.PV_OPT_SELECTOR_KERNEL, kernel)
    d = v.device
    words = words or W.words_per_row(cluster.num_nodes)
    d_assign = None if sel.assign is None else to_device(sel.assign.astype(np.uint32), d)
    bits, flags = v.eval_selectors(to_device(sel.expr_offs.astype(np.uint32), d), len(sel.exprs),
                                   to_device(sel.exprs, d), d_assign, sel.num_pods, words=words)
    v.sync()
    v.set_option(B.PV_OPT_SELECTOR_KERNEL, 0)
    return (to_numpy(bits, np.uint32, (sel.num_pods, words)), to_numpy(flags, np.uint8))


def _oracle_eval(cluster, sel, words=None):
    return oracle.eval_selectors(cluster.num_nodes, cluster.num_keys, cluster.labels, sel.expr_offs, sel.exprs,
                                 sel.assign, words=words)


@pytest.mark.parametrize("kernel", [1, 2])
def test_tiny_workload(validator, kernel):
    d = W.tiny()
    gb, gf = _gpu_eval(validator, d["cluster"], d["selectors"], kernel)
    ob, of = _oracle_eval(d["cluster"], d["selectors"])
    assert (gb == ob).all() and (gf == of).all()


@pytest.mark.parametrize("kernel", [1, 2])
@pytest.mark.parametrize("n,k,p_absent,p_unknown,dne", [
    (1000, 16, 0.0, 0.0, False),      # ragged: 1000 = 31.25 words
    (4097, 64, 0.1, 0.02, True),      # spans several label tiles and one extra word
    (33, 5, 0.5, 0.1, True),
    (32, 3, 0.0, 0.0, False),
    (7001, 24, 0.05, 0.0, True),
])
def test_random_workloads(validator, kernel, n, k, p_absent, p_unknown, dne):
    d = W.selector_workload(seed=n + k, num_nodes=n, num_keys=k, num_values=40, num_pods=3000,
                            p_absent=p_absent, p_unknown=p_unknown, with_doesnotexist=dne)
    gb, gf = _gpu_eval(validator, d["cluster"], d["selectors"], kernel)
    ob, of = _oracle_eval(d["cluster"], d["selectors"])
    assert (gf == of).all()
    assert (gb == ob).all()


@pytest.mark.parametrize("kernel", [1, 2])
def test_wide_rows_and_malformed_lists(validator, kernel):
    d = W.selector_workload(seed=3, num_nodes=300, num_keys=6, num_values=9, num_pods=400, p_absent=0.2)
    sel = d["selectors"]
    ex = sel.exprs.copy()
    ex[5]["key"] = 99                 # key out of range
    ex[17]["op"] = 9                  # unknown operator
    ex[40]["nvals"] = 0
    ex[41]["op"], ex[41]["nvals"] = W.OP_EXISTS, 2
    ex[60]["vals"][0] = W.ABSENT
    offs = sel.expr_offs.copy()
    bad_sel = W.Selectors(sel.num_pods, offs, ex, sel.assign)
    words = W.words_per_row(300) + 8  # caller-chosen wider rows: padding must be zero
    gb, gf = _gpu_eval(validator, d["cluster"], bad_sel, kernel, words=words)
    ob, of = _oracle_eval(d["cluster"], bad_sel, words=words)
    assert (gf == of).all() and (gb == ob).all()
    assert (of & W.F_BAD_EXPR).sum() >= 5


@pytest.mark.parametrize("kernel", [1, 2])
def test_offsets_beyond_expression_count(validator, kernel):
    d = W.selector_workload(seed=5, num_nodes=64, num_keys=4, num_values=5, num_pods=10)
    sel = d["selectors"]
    offs = sel.expr_offs.copy()
    offs[3] = offs[4] + 1             # decreasing at pod 3
    offs[-1] = len(sel.exprs)         # valid end; also try a too-large count below
    s2 = W.Selectors(sel.num_pods, offs, sel.exprs, sel.assign)
    gb, gf = _gpu_eval(validator, d["cluster"], s2, kernel)
    ob, of = _oracle_eval(d["cluster"], s2)
    assert (gf == of).all() and (gb == ob).all()


def test_empty_and_invalid_calls(validator):
    d = W.selector_workload(seed=1, num_nodes=50, num_keys=4, num_pods=4)
    validator.load_cluster(d["cluster"])
    dev = validator.device
    offs = to_device(d["selectors"].expr_offs.astype(np.uint32), dev)
    ex = to_device(d["selectors"].exprs, dev)
    bits = empty_device(4 * 4 * 4, dev)
    flags = empty_device(4, dev)
    B.pv_eval_selectors(validator.ctx, 0, offs, 0, ex, None, bits, 4, flags)   # no pods: no-op
    with pytest.raises(B.PVError) as e:
        B.pv_eval_selectors(validator.ctx, 4, offs, len(d["selectors"].exprs), ex, None, bits, 2, flags)
    assert e.value.code == B.PV_EINVAL
    with pytest.raises(B.PVError):
        B.pv_eval_selectors(validator.ctx, 4, offs, len(d["selectors"].exprs), ex, None, bits, 6, flags)
    odd = empty_device(d["selectors"].exprs.nbytes + 2, dev)[2:]   # expressions off a 4-byte boundary
    with pytest.raises(B.PVError) as e:
        B.pv_eval_selectors(validator.ctx, 4, offs, len(d["selectors"].exprs), odd, None, bits, 4, flags)
    assert e.value.code == B.PV_EINVAL
    with pytest.raises(B.PVError) as e:
        B.pv_load_cluster(validator.ctx, 0, 4, np.zeros(0, np.uint16))
    assert e.value.code == B.PV_EINVAL


@pytest.mark.parametrize("kernel", [0, 1])
def test_placement_scale_full(validator, kernel):
    """Full placement-scale workload (100,000 pods x 5,000 nodes) in the
    benchmark's launch configuration (kernel 0: the library's choice, the
    value-row kernel) and with the comparison kernel (1); every row and
    flag is compared with the oracle's."""
    d = W.selector_workload()
    c, sel = d["cluster"], d["selectors"]
    validator.load_cluster(c)
    assert B.pv_get_stat(validator.ctx, B.PV_STAT_SELECTOR_ROWS_BUILT) == 1
    words = W.words_per_row(c.num_nodes)
    gb, gf = _gpu_eval(validator, c, sel, kernel, words)
    want = F.cached("placement-scale/default", lambda: dict(zip(("bits", "flags"), F.eval_selectors(c, sel, words))))
    assert (gf == want["flags"]).all()
    assert (gb == want["bits"]).all()
    assert gf.any() and (gf & W.F_PASS).any()


@pytest.mark.parametrize("kernel", [1, 2])
@pytest.mark.parametrize("mode", [1, 2])
def test_identical_selectors_evaluated_once(validator, kernel, mode):
    """PV_OPT_SELECTOR_DEDUPE: pods sharing an expression list (Zipf
    popularity over a few hundred lists, with absent labels, unknown values,
    DoesNotExist, malformed expressions, lists that differ only in unused
    value slots, and pods whose offsets are out of range) give the oracle's
    rows and flags, each with its own placement check; with weak hashes
    (mode 2) every list collides with others and is resolved by comparison."""
    d = W.selector_replicas(seed=61, num_distinct=300, num_pods=5000, num_nodes=1500, num_keys=20, num_values=30,
                            p_absent=0.05, p_unknown=0.03, with_doesnotexist=True)
    c, s = d["cluster"], d["selectors"]
    ex = s.exprs.copy()
    st = W.Stream(62, "dedupe-edits")
    bad = st.ints(0, len(ex) - 1, 40)
    ex["nvals"][bad[:20]] = 9                      # malformed counts
    ex["op"][bad[20:]] = 7                         # unknown operators
    slack = np.nonzero((ex["op"] == W.OP_IN) & (ex["nvals"] < 8))[0][:50]
    ex["vals"][slack, 7] = 29                      # unused slots differ: still the same list
    offs = s.expr_offs.copy()
    sel = W.Selectors(s.num_pods, offs, ex, s.assign)
    ob, of = _oracle_eval(c, sel)
    v = validator
    v.set_option(B.PV_OPT_SELECTOR_DEDUPE, mode)
    try:
        gb, gf = _gpu_eval(v, c, sel, kernel)
    finally:
        v.set_option(B.PV_OPT_SELECTOR_DEDUPE, 0)
    assert (gf == of).all()
    assert (gb == ob).all()
    assert len(np.unique(d["pick"])) < 300 and s.num_pods == 5000   # lists really repeat


def test_identical_selectors_with_out_of_range_offsets(validator):
    """A pod whose expression range is malformed is its own representative
    (row empty, PV_F_BAD_EXPR), also with dedupe on."""
    d = W.selector_replicas(seed=63, num_distinct=40, num_pods=400, num_nodes=300, num_keys=8, num_values=12)
    c, s = d["cluster"], d["selectors"]
    offs = s.expr_offs.copy()
    offs[100] = offs[101] + 3                      # pod 100's range is reversed (pod 99's overlaps pod 100's list)
    sel = W.Selectors(s.num_pods, offs, s.exprs, s.assign)
    ob, of = _oracle_eval(c, sel)
    v = validator
    v.set_option(B.PV_OPT_SELECTOR_DEDUPE, 1)
    try:
        gb, gf = _gpu_eval(v, c, sel, 2)
    finally:
        v.set_option(B.PV_OPT_SELECTOR_DEDUPE, 0)
    assert (gf == of).all() and (gb == ob).all()
    assert of[100] == W.F_BAD_EXPR
