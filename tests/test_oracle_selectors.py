"""Pins for the oracle's selector evaluation and placement check.

The oracle is checked against things other than itself:
  * the paper's printed 5-worker label table (Sec. 5.1-5.2, Table "Worker-node
    label matrix for 5-worker cluster") with selectors whose answers are read
    off the table by eye;
  * the hallucinated-identifier failure mode (Sec. 6.3, item 3) and the
    fail-closed unenforceable intent (Sec. 5.3, intent examples table);
  * a brute force over string-keyed label dictionaries (a node either has a
    key in its dict or not; operators evaluated as Python set logic);
  * closed forms and invariants (Exists on a dense key admits every node,
    DoesNotExist admits none, feasible sets only contain nodes carrying the
    required keys, padding bits are zero).
"""
import os

import numpy as np
import pytest

import oracle
from paper_2602_16100_gb300 import workloads as W

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "worker_labels_5.txt")


def _load_worker_table():
    rows = [ln.split() for ln in open(GOLDEN) if ln.strip() and not ln.startswith("#")]
    names = [r[0] for r in rows]
    keys = ["location", "provider", "security", "zone"]
    vocab = {k: sorted({r[1 + i] for r in rows}) for i, k in enumerate(keys)}
    labels = np.zeros((len(keys), len(rows)), np.uint16)
    for i, k in enumerate(keys):
        for n, r in enumerate(rows):
            labels[i, n] = vocab[k].index(r[1 + i])
    return names, keys, vocab, labels


def _expr(key, op, vals=()):
    e = np.zeros(1, W.EXPR_DTYPE)
    e["key"], e["op"], e["nvals"] = key, op, len(vals)
    v = np.zeros(8, np.uint16)
    if vals:
        v[: len(vals)] = vals
        v[len(vals):] = vals[0]
    e["vals"] = v
    return e


def _members(row, n):
    return {i for i in range(n) if (int(row[i >> 5]) >> (i & 31)) & 1}


def test_struct_sizes_match_layouts():
    assert oracle.struct_sizes() == (W.EXPR_DTYPE.itemsize, W.RULE_DTYPE.itemsize,
                                     W.PROBE_DTYPE.itemsize, W.RESULT_DTYPE.itemsize)


def test_worker_label_table_selectors():
    names, keys, vocab, labels = _load_worker_table()
    K = {k: i for i, k in enumerate(keys)}
    val = lambda k, s: vocab[k].index(s) if s in vocab[k] else 60000 + len(s)   # unknown ids for hallucinations
    w = lambda *ns: {names.index(f"worker-{i}") for i in ns}
    cases = [
        # (expressions, expected feasible set, expect unknown)
        ([_expr(K["security"], W.OP_IN, [val("security", "high")])], w(1, 4), False),
        # Sec. 5.3 hybrid example: appointment only on high-security cloud nodes
        ([_expr(K["zone"], W.OP_IN, [val("zone", "cloud")]),
          _expr(K["security"], W.OP_IN, [val("security", "high")])], w(4), False),
        ([_expr(K["location"], W.OP_IN, [val("location", "london"), val("location", "sydney")])], w(1, 4), False),
        # keep sensitive databases off the edge zone
        ([_expr(K["zone"], W.OP_NOTIN, [val("zone", "edge")])], w(3, 4, 5), False),
        ([_expr(K["provider"], W.OP_NOTIN, [val("provider", "aws"), val("provider", "azure")])], w(5), False),
        ([_expr(K["zone"], W.OP_EXISTS)], w(1, 2, 3, 4, 5), False),
        ([_expr(K["zone"], W.OP_DOESNOTEXIST)], set(), False),
        ([_expr(K["provider"], W.OP_IN, [val("provider", "aws")]),
          _expr(K["security"], W.OP_IN, [val("security", "medium")])], w(2), False),
        # Sec. 6.3 item 3: hallucinated region value carried by no node
        ([_expr(K["location"], W.OP_IN, [val("location", "eu_region")])], set(), True),
        # an unknown value inside a larger set still fails the check
        ([_expr(K["provider"], W.OP_IN, [val("provider", "aws"), val("provider", "eu_cloud")])], w(1, 2), True),
        # NotIn with an unknown value is vacuous for that value
        ([_expr(K["provider"], W.OP_NOTIN, [val("provider", "eu_cloud")])], w(1, 2, 3, 4, 5), False),
        ([], w(1, 2, 3, 4, 5), False),
    ]
    offs = np.zeros(len(cases) + 1, np.uint32)
    offs[1:] = np.cumsum([len(c[0]) for c in cases])
    exprs = np.concatenate([e for c in cases for e in c[0]]) if offs[-1] else np.zeros(0, W.EXPR_DTYPE)
    # assign every pod to worker-4 (sydney/azure/high/cloud)
    assign = np.full(len(cases), names.index("worker-4"), np.uint32)
    bits, flags = oracle.eval_selectors(5, 4, labels.reshape(-1), offs, exprs, assign)
    for i, (_, want, unk) in enumerate(cases):
        assert _members(bits[i], 5) == want, i
        assert bool(flags[i] & W.F_EMPTY) == (not want), i
        assert bool(flags[i] & W.F_UNKNOWN_VALUE) == unk, i
        in4 = names.index("worker-4") in want
        assert bool(flags[i] & W.F_ASSIGN_OK) == in4, i
        assert bool(flags[i] & W.F_PASS) == (in4 and not unk), i
        assert not flags[i] & W.F_BAD_EXPR


def _brute(num_nodes, num_keys, labels, offs, exprs, assign):
    """String-keyed brute force: each node is a dict {"k<i>": "v<j>"} holding
    only the keys it carries."""
    lab = labels.reshape(num_keys, num_nodes)
    nodes = [{f"k{k}": f"v{int(lab[k, n])}" for k in range(num_keys) if lab[k, n] != W.ABSENT}
             for n in range(num_nodes)]
    inventory = {}
    for d in nodes:
        for k, v in d.items():
            inventory.setdefault(k, set()).add(v)
    feas, flags = [], []
    for p in range(len(offs) - 1):
        es = exprs[offs[p]:offs[p + 1]]
        sel = []
        for e in es:
            key = f"k{int(e['key'])}"
            vals = {f"v{int(x)}" for x in e["vals"][: int(e["nvals"])]}
            sel.append((int(e["op"]), key, vals))
        ok_nodes = set()
        for n, d in enumerate(nodes):
            good = True
            for op, key, vals in sel:
                if op == W.OP_IN:
                    good &= key in d and d[key] in vals
                elif op == W.OP_NOTIN:
                    good &= key not in d or d[key] not in vals
                elif op == W.OP_EXISTS:
                    good &= key in d
                else:
                    good &= key not in d
            if good:
                ok_nodes.add(n)
        unknown = any(op == W.OP_IN and not vals <= inventory.get(key, set()) for op, key, vals in sel)
        f = 0
        if not ok_nodes:
            f |= W.F_EMPTY
        if unknown:
            f |= W.F_UNKNOWN_VALUE
        if assign is not None and int(assign[p]) in ok_nodes:
            f |= W.F_ASSIGN_OK
            if not unknown:
                f |= W.F_PASS
        feas.append(ok_nodes)
        flags.append(f)
    return feas, flags


@pytest.mark.parametrize("seed,p_absent,p_unknown,dne", [
    (1, 0.0, 0.0, False), (2, 0.2, 0.05, True), (3, 0.5, 0.1, True), (4, 0.05, 0.0, False)])
def test_selectors_match_string_brute_force(seed, p_absent, p_unknown, dne):
    d = W.selector_workload(seed=seed, num_nodes=37, num_keys=6, num_values=5, num_pods=300, max_exprs=4,
                            p_absent=p_absent, p_unknown=p_unknown, with_doesnotexist=dne)
    c, s = d["cluster"], d["selectors"]
    bits, flags = oracle.eval_selectors(c.num_nodes, c.num_keys, c.labels, s.expr_offs, s.exprs, s.assign)
    feas, bflags = _brute(c.num_nodes, c.num_keys, c.labels, s.expr_offs, s.exprs, s.assign)
    for p in range(s.num_pods):
        assert _members(bits[p], c.num_nodes) == feas[p], p
        assert int(flags[p]) == bflags[p], p


def test_selector_invariants_and_closed_forms():
    d = W.selector_workload(seed=11, num_nodes=1000, num_keys=16, num_pods=3000, p_absent=0.1)
    c, s = d["cluster"], d["selectors"]
    lab = c.labels.reshape(c.num_keys, c.num_nodes)
    bits, flags = oracle.eval_selectors(c.num_nodes, c.num_keys, c.labels, s.expr_offs, s.exprs, s.assign)
    Wd = bits.shape[1]
    # padding bits beyond num_nodes are zero
    allbits = np.unpackbits(bits.view(np.uint8), axis=1, bitorder="little")
    assert not allbits[:, c.num_nodes:].any()
    for p in range(0, s.num_pods, 7):
        mem = allbits[p, : c.num_nodes].astype(bool)
        for e in s.exprs[s.expr_offs[p]:s.expr_offs[p + 1]]:
            col = lab[int(e["key"])]
            if int(e["op"]) in (W.OP_IN, W.OP_EXISTS):
                assert not (mem & (col == W.ABSENT)).any()         # carries every required key
            if int(e["op"]) == W.OP_IN and int(e["nvals"]) == 1:
                assert not (mem & (col != e["vals"][0])).any()      # equality: exact value
    # dense key: Exists = all nodes, DoesNotExist = none; empty list = all
    d2 = W.selector_workload(seed=12, num_nodes=77, num_keys=3, num_pods=1)
    c2 = d2["cluster"]
    offs = np.array([0, 1, 2, 2], np.uint32)
    ex = np.concatenate([_expr(1, W.OP_EXISTS), _expr(2, W.OP_DOESNOTEXIST)])
    b2, f2 = oracle.eval_selectors(c2.num_nodes, c2.num_keys, c2.labels, offs, ex)
    assert _members(b2[0], 77) == set(range(77))
    assert _members(b2[1], 77) == set() and f2[1] & W.F_EMPTY
    assert _members(b2[2], 77) == set(range(77))
    assert Wd == W.words_per_row(c.num_nodes)


def test_malformed_expressions_fail_closed():
    labels = np.zeros((2, 10), np.uint16).reshape(-1)
    bad = [
        _expr(2, W.OP_IN, [0]),                 # key out of range
        _expr(0, 7, [0]),                       # unknown operator
        _expr(0, W.OP_IN, []),                  # In without values
        _expr(0, W.OP_EXISTS, [1]),             # Exists with values
        _expr(0, W.OP_NOTIN, [W.ABSENT]),       # the absent sentinel is not a value
    ]
    e9 = _expr(0, W.OP_IN, [0]); e9["nvals"] = 9
    bad.append(e9)
    exprs = np.concatenate(bad + [_expr(0, W.OP_IN, [0])])
    offs = np.arange(len(exprs) + 1, dtype=np.uint32)        # one expression per pod
    # last pod: a good expression -> feasible = all nodes
    bits, flags = oracle.eval_selectors(10, 2, labels, offs, exprs, np.zeros(len(offs) - 1, np.uint32))
    for p in range(len(bad)):
        assert flags[p] == W.F_BAD_EXPR and not bits[p].any(), p
    assert flags[-1] == W.F_ASSIGN_OK | W.F_PASS
    # non-monotone offsets / offsets beyond the expression count
    offs2 = np.array([0, 1, 0, 50], np.uint32)
    b3, f3 = oracle.eval_selectors(10, 2, labels, offs2, exprs[-1:].copy())
    assert f3[1] == W.F_BAD_EXPR and f3[2] == W.F_BAD_EXPR and f3[0] == 0
