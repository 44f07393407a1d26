"""The GPU parity tests can catch faults in the verdict (Sec. 5.5: an
intent passes only if every one of its checks passes).

A mistake is planted in a copy of the oracle's output, on the CPU: the
verdict forced to fail, the concrete-flow flag of a policy ignored (Sec. 6.3
no-op policies), the waypoint bits ignored (Sec. 5.3 must-go switches), or
the probe statuses ignored.  Each mutant must differ from the oracle's
verdicts on the very inputs the GPU end-to-end tests use (small batches of
the variant in which intents can pass).  Those tests compare the GPU's
verdicts with the oracle's element by element, so a kernel that made any of
these mistakes would fail them."""
import numpy as np

import full_oracle as F
import oracle
from gpu_util import E2E_CONSTRAINED, E2E_PASS_SMALL, POLICIES_CONSTRAINED
from paper_2602_16100_gb300 import workloads as W


def _constrained():
    e = W.end_to_end(**E2E_CONSTRAINED)
    kw = dict(POLICIES_CONSTRAINED)
    pol = W.path_policies(kw.pop("seed"), e.network, e.intents.num_pods, **kw)
    return e, pol, F.end_to_end(e, pol)


def _verdict(e, out, pol, hits=None, results=None):
    c = e.cluster
    return oracle.aggregate_constrained(out["bits"], c.num_nodes, out["flags"], out["assign"], e.pods_per_intent,
                                        out["results"] if results is None else results, e.probes_per_intent,
                                        out["hits"] if hits is None else hits, pol)[0]


def test_unconstrained_verdicts_catch_forced_failure_and_ignored_statuses():
    e = W.end_to_end(**E2E_PASS_SMALL)
    out = F.end_to_end(e)
    passed = out["passed"]
    assert passed.mean() >= 0.1 and not passed.all()
    assert (np.zeros_like(passed) != passed).any()                    # pass forced to 0
    c = e.cluster
    all_ok = out["results"].copy()
    all_ok["status"] = W.ST_COMPLIANT                                 # probe statuses ignored
    p2, _ = oracle.aggregate(out["bits"], c.num_nodes, out["flags"], out["assign"], e.pods_per_intent, all_ok,
                             e.probes_per_intent)
    assert (p2 != passed).any()


def test_constrained_verdicts_catch_ignored_concrete_flag_and_waypoints():
    e, pol, out = _constrained()
    passed = out["passed"]
    assert passed.any() and (_verdict(e, out, pol) == passed).all()
    assert (np.zeros_like(passed) != passed).any()                    # pass forced to 0
    every = W.PathPolicies(pol.num_policies, pol.forbid_offs, pol.forbid, pol.must_offs, pol.must,
                           np.ones_like(pol.concrete))
    assert (_verdict(e, out, every) != passed).any()                  # concrete ignored
    n = np.diff(pol.must_offs.astype(np.int64))
    all_hit = np.repeat(((1 << n) - 1).astype(np.uint32), e.probes_per_intent)
    assert (_verdict(e, out, pol, hits=all_hit) != passed).any()      # missed waypoints ignored
