"""GPU parity of multi-term selectors (node-affinity form) against the
oracle, bit-exact rows and flags: random clusters with absent labels,
unknown values, DoesNotExist and empty terms; malformed term ranges; and the
placement-scale cluster with 100,000 multi-term pods on a sample."""
import numpy as np
import pytest

import oracle
from paper_2602_16100_gb300 import binding as B
from paper_2602_16100_gb300 import workloads as W
from paper_2602_16100_gb300.validator import empty_device, to_device, to_numpy
from gpu_util import sample

pytestmark = pytest.mark.gpu


def _gpu_terms(v, c, pod_terms, term_offs, exprs, assign, words=None):
    dev = v.device
    words = words or W.words_per_row(c.num_nodes)
    P = len(pod_terms) - 1
    bits = empty_device(P * words * 4, dev)
    flags = empty_device(P, dev)
    B.pv_eval_selector_terms(v.ctx, P, to_device(np.asarray(pod_terms, np.uint32), dev), len(term_offs) - 1,
                             to_device(np.asarray(term_offs, np.uint32), dev), len(exprs), to_device(exprs, dev),
                             None if assign is None else to_device(np.asarray(assign, np.uint32), dev), bits, words,
                             flags)
    v.sync()
    return to_numpy(bits, np.uint32, (P, words)), to_numpy(flags, np.uint8)


@pytest.mark.parametrize("seed,n,p_absent,p_unknown,p_empty", [(1, 41, 0.0, 0.0, 0.0), (2, 300, 0.2, 0.05, 0.1),
                                                               (3, 1000, 0.4, 0.1, 0.3), (4, 4097, 0.1, 0.02, 0.05)])
def test_random_terms(validator, seed, n, p_absent, p_unknown, p_empty):
    d = W.selector_terms(seed=seed, num_nodes=n, num_keys=7, num_values=6, num_pods=700, max_terms=4, max_exprs=4,
                         p_empty_term=p_empty, p_absent=p_absent, p_unknown=p_unknown, with_doesnotexist=True)
    c, s = d["cluster"], d["terms"]
    validator.load_cluster(c)
    for words in (None, W.words_per_row(n) + 8):
        g, gf = _gpu_terms(validator, c, s.pod_terms, s.term_offs, s.exprs, s.assign, words)
        o, of = oracle.eval_selector_terms(c.num_nodes, c.num_keys, c.labels, s.pod_terms, s.term_offs, s.exprs,
                                           s.assign, words=words)
        assert (g == o).all() and (gf == of).all()
    assert len(np.unique(of)) >= 3


def test_malformed_terms(validator):
    d = W.selector_terms(seed=9, num_nodes=100, num_keys=4, num_values=4, num_pods=4, max_terms=2, max_exprs=2)
    c = d["cluster"]
    validator.load_cluster(c)
    ex = d["terms"].exprs[:3].copy()
    bad_key = ex.copy()
    bad_key[2]["key"] = 99
    # pods: one empty term; no terms; term range past the expressions;
    # a term whose expression has an out-of-range key; pod range past the terms
    pod_terms = np.array([0, 1, 1, 2, 3, 9], np.uint32)
    term_offs = np.array([0, 0, 7, 3], np.uint32)
    for exprs in (ex, bad_key):
        g, gf = _gpu_terms(validator, c, pod_terms, term_offs, exprs, None)
        o, of = oracle.eval_selector_terms(c.num_nodes, c.num_keys, c.labels, pod_terms, term_offs, exprs)
        assert (g == o).all() and (gf == of).all()
    assert of[2] == W.F_BAD_EXPR and of[4] == W.F_BAD_EXPR


def test_placement_scale_terms_sampled(validator):
    d = W.selector_terms(num_pods=100_000)
    c, s = d["cluster"], d["terms"]
    validator.load_cluster(c)
    g, gf = _gpu_terms(validator, c, s.pod_terms, s.term_offs, s.exprs, s.assign)
    idx = sample(s.num_pods, 3000, seed=4)
    # the sampled pods as a batch of their own (terms re-packed)
    pt, to, ex = [0], [0], []
    for p in idx:
        for t in range(int(s.pod_terms[p]), int(s.pod_terms[p + 1])):
            ex.append(s.exprs[s.term_offs[t]:s.term_offs[t + 1]])
            to.append(to[-1] + int(s.term_offs[t + 1] - s.term_offs[t]))
        pt.append(len(to) - 1)
    ex = np.concatenate(ex) if ex else np.zeros(0, W.EXPR_DTYPE)
    o, of = oracle.eval_selector_terms(c.num_nodes, c.num_keys, c.labels, np.array(pt, np.uint32),
                                       np.array(to, np.uint32), ex, s.assign[idx])
    assert (g[idx] == o).all() and (gf[idx] == of).all()
