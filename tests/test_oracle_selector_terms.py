"""Pins for the oracle's multi-term selectors (Kubernetes required node
affinity: selector terms ORed, expressions within a term ANDed; Sec. 3.3 and
Sec. 4.1 placement by node selector / affinity).

Checked against a string-keyed brute force written as the definition (a node
is feasible iff some term has all its expressions satisfied), against the
single-list oracle for one-term pods, and against the union identity: a
pod's row is the OR of the rows of its terms evaluated one by one.
"""
import numpy as np
import pytest

import oracle
from paper_2602_16100_gb300 import workloads as W
from test_oracle_selectors import _members


def _brute_terms(num_nodes, num_keys, labels, pod_terms, term_offs, exprs, assign):
    lab = labels.reshape(num_keys, num_nodes)
    nodes = [{f"k{k}": f"v{int(lab[k, n])}" for k in range(num_keys) if lab[k, n] != W.ABSENT}
             for n in range(num_nodes)]
    inventory = {}
    for d in nodes:
        for k, v in d.items():
            inventory.setdefault(k, set()).add(v)

    def holds(op, key, vals, d):
        if op == W.OP_IN:
            return key in d and d[key] in vals
        if op == W.OP_NOTIN:
            return key not in d or d[key] not in vals
        if op == W.OP_EXISTS:
            return key in d
        return key not in d

    feas, flags = [], []
    for p in range(len(pod_terms) - 1):
        terms = []
        for t in range(int(pod_terms[p]), int(pod_terms[p + 1])):
            terms.append([(int(e["op"]), f"k{int(e['key'])}", {f"v{int(x)}" for x in e["vals"][: int(e["nvals"])]})
                          for e in exprs[term_offs[t]:term_offs[t + 1]]])
        if not terms:
            ok_nodes = set(range(num_nodes))
        else:
            ok_nodes = {n for n, d in enumerate(nodes)
                        if any(term and all(holds(op, k, v, d) for op, k, v in term) for term in terms)}
        unknown = any(op == W.OP_IN and not v <= inventory.get(k, set()) for term in terms for op, k, v in term)
        f = (W.F_EMPTY if not ok_nodes else 0) | (W.F_UNKNOWN_VALUE if unknown else 0)
        if int(assign[p]) in ok_nodes:
            f |= W.F_ASSIGN_OK | (0 if unknown else W.F_PASS)
        feas.append(ok_nodes)
        flags.append(f)
    return feas, flags


@pytest.mark.parametrize("seed,p_absent,p_unknown,p_empty", [(1, 0.0, 0.0, 0.0), (2, 0.2, 0.05, 0.1),
                                                             (3, 0.4, 0.1, 0.3)])
def test_terms_match_string_brute_force(seed, p_absent, p_unknown, p_empty):
    d = W.selector_terms(seed=seed, num_nodes=41, num_keys=6, num_values=5, num_pods=250, max_terms=4,
                         max_exprs=3, p_empty_term=p_empty, p_absent=p_absent, p_unknown=p_unknown,
                         with_doesnotexist=True)
    c, s = d["cluster"], d["terms"]
    bits, flags = oracle.eval_selector_terms(c.num_nodes, c.num_keys, c.labels, s.pod_terms, s.term_offs, s.exprs,
                                             s.assign)
    feas, bflags = _brute_terms(c.num_nodes, c.num_keys, c.labels, s.pod_terms, s.term_offs, s.exprs, s.assign)
    for p in range(s.num_pods):
        assert _members(bits[p], c.num_nodes) == feas[p], p
        assert int(flags[p]) == bflags[p], p
    assert (np.diff(s.pod_terms) == 0).any() and (np.diff(s.pod_terms) > 1).any()


def test_terms_union_identity_and_single_term_reduction():
    d = W.selector_terms(seed=5, num_nodes=300, num_keys=8, num_values=6, num_pods=400, max_terms=3, max_exprs=3,
                         p_absent=0.1)
    c, s = d["cluster"], d["terms"]
    bits, flags = oracle.eval_selector_terms(c.num_nodes, c.num_keys, c.labels, s.pod_terms, s.term_offs, s.exprs,
                                             s.assign)
    # each term as a one-term pod, through the single-list oracle
    tb, _ = oracle.eval_selectors(c.num_nodes, c.num_keys, c.labels, s.term_offs, s.exprs)
    for p in range(s.num_pods):
        t0, t1 = int(s.pod_terms[p]), int(s.pod_terms[p + 1])
        if t0 == t1:
            assert _members(bits[p], c.num_nodes) == set(range(c.num_nodes))
            continue
        want = np.zeros_like(bits[p])
        for t in range(t0, t1):
            want |= tb[t]
        assert (bits[p] == want).all(), p
    # one-term pods equal the single-list evaluation
    one = np.arange(len(s.term_offs), dtype=np.uint32)
    b1, f1 = oracle.eval_selector_terms(c.num_nodes, c.num_keys, c.labels, one, s.term_offs, s.exprs)
    b2, f2 = oracle.eval_selectors(c.num_nodes, c.num_keys, c.labels, s.term_offs, s.exprs)
    assert (b1 == b2).all() and (f1 == f2).all()


def test_empty_term_and_malformed_ranges():
    d = W.selector_terms(seed=6, num_nodes=50, num_keys=4, num_values=4, num_pods=3, max_terms=2, max_exprs=2)
    c = d["cluster"]
    ex = d["terms"].exprs[:2].copy()
    # pod 0: one empty term -> nothing; pod 1: no terms -> everything;
    # pod 2: term range past the expressions -> BAD
    pod_terms = np.array([0, 1, 1, 2], np.uint32)
    term_offs = np.array([0, 0, 5], np.uint32)
    bits, flags = oracle.eval_selector_terms(c.num_nodes, c.num_keys, c.labels, pod_terms, term_offs, ex)
    assert not bits[0].any() and flags[0] & W.F_EMPTY
    assert _members(bits[1], c.num_nodes) == set(range(c.num_nodes))
    assert flags[2] == W.F_BAD_EXPR and not bits[2].any()
