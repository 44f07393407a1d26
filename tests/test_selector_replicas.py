"""The repeated-selector workload (pods sharing expression lists, as the
replicas of one deployment do) and the oracle on it: every pod's list is a
verbatim copy of its source list, and pods with the same list get the same
row and the same flags apart from their own placement check."""
import numpy as np

import oracle
from paper_2602_16100_gb300 import workloads as W


def test_replica_lists_are_copies_of_their_source():
    d = W.selector_replicas(seed=71, num_distinct=50, num_pods=2000, num_nodes=200, num_keys=10)
    s = d["selectors"]
    base = W.selector_workload(seed=71, num_pods=50, num_nodes=200, num_keys=10)["selectors"]
    for p, k in enumerate(d["pick"]):
        mine = s.exprs[s.expr_offs[p]:s.expr_offs[p + 1]]
        src = base.exprs[base.expr_offs[k]:base.expr_offs[k + 1]]
        assert len(mine) == len(src) and (mine == src).all()
    counts = np.bincount(d["pick"], minlength=50)
    assert counts[0] == counts.max() and (counts > 0).sum() > 25   # Zipf popularity, most lists used


def test_equal_lists_give_equal_rows_in_the_oracle():
    d = W.selector_replicas(seed=72, num_distinct=30, num_pods=600, num_nodes=150, num_keys=8, p_unknown=0.05)
    c, s = d["cluster"], d["selectors"]
    bits, flags = oracle.eval_selectors(c.num_nodes, c.num_keys, c.labels, s.expr_offs, s.exprs, s.assign)
    keep = np.uint8(0xFF ^ (W.F_ASSIGN_OK | W.F_PASS))   # all flags but the placement check
    for k in np.unique(d["pick"]):
        pods = np.nonzero(d["pick"] == k)[0]
        assert (bits[pods] == bits[pods[0]]).all()
        assert ((flags[pods] & keep) == (flags[pods[0]] & keep)).all()
        for p in pods:   # the placement check is the pod's own
            a = int(s.assign[p])
            ok = bool((bits[p, a >> 5] >> (a & 31)) & 1)
            assert bool(flags[p] & W.F_ASSIGN_OK) == ok
