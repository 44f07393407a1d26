"""The unchanged CPU oracle over every output of a full-size workload.

Test infrastructure.  Each function cuts its units (pods, probes, masks)
into disjoint contiguous ranges and runs the single-threaded oracle on each
range from a pool of host threads (the oracle's C calls release the GIL
and share no state, so the ranges run in parallel on all host cores); the
pieces are concatenated in order, so the result is exactly that of one
oracle call over everything.

Results are cached on disk under $PV_ORACLE_CACHE (default
~/.cache/pv_oracle; "off" disables the cache), keyed by the caller's
workload key and a hash of the oracle's source, its binding, the workload
generator and this file, so a cached value is only ever reused for the
same inputs and the same oracle.  Nothing here computes any part of the
method; no value comes from the GPU path.
"""
from __future__ import annotations

import concurrent.futures as cf
import hashlib
import os
from typing import Callable, Dict

import numpy as np

import oracle

_ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
_HASHED = ("oracle/pv_oracle.c", "oracle/__init__.py", "paper_2602_16100_gb300/workloads.py", "tests/full_oracle.py")


def threads() -> int:
    return max(1, os.cpu_count() or 1)


def _ranges(n: int, parts: int):
    cuts = np.linspace(0, n, max(1, min(parts, n)) + 1).astype(np.int64)
    return [(int(a), int(b)) for a, b in zip(cuts[:-1], cuts[1:]) if b > a]


def _map(fn, ranges):
    with cf.ThreadPoolExecutor(max_workers=threads()) as ex:
        return list(ex.map(lambda r: fn(*r), ranges))


# ----------------------------------------------------------------------------
# disk cache
# ----------------------------------------------------------------------------
def _cache_dir():
    d = os.environ.get("PV_ORACLE_CACHE", "")
    if d.lower() == "off":
        return None
    return d or os.path.join(os.path.expanduser("~"), ".cache", "pv_oracle")


def _digest(key: str) -> str:
    h = hashlib.sha256(key.encode())
    for rel in _HASHED:
        with open(os.path.join(_ROOT, rel), "rb") as f:
            h.update(f.read())
    return h.hexdigest()[:32]


def cached(key: str, compute: Callable[[], Dict[str, np.ndarray]]) -> Dict[str, np.ndarray]:
    """compute() once per (key, oracle and generator sources); later calls
    load the stored arrays.  A cache that cannot be read or written is
    skipped (the value is then computed)."""
    d = _cache_dir()
    path = os.path.join(d, _digest(key) + ".npz") if d else None
    if path and os.path.exists(path):
        try:
            with np.load(path) as z:
                return {k: z[k] for k in z.files}
        except Exception:
            pass
    out = compute()
    if path:
        try:
            os.makedirs(d, exist_ok=True)
            tmp = f"{path}.tmp{os.getpid()}.npz"
            np.savez(tmp, **out)
            os.replace(tmp, path)
        except Exception:
            pass
    return out


# ----------------------------------------------------------------------------
# sharded oracle calls
# ----------------------------------------------------------------------------
def eval_selectors(cluster, sel, words, assign=None):
    """All rows and flags of oracle.eval_selectors, by ranges of pods."""
    offs = sel.expr_offs.astype(np.int64)
    assert (np.diff(offs) >= 0).all() and offs[0] == 0, "well-formed expression offsets only"
    P = len(offs) - 1
    a = sel.assign if assign is None else assign

    def one(lo, hi):
        o = (offs[lo:hi + 1] - offs[lo]).astype(np.uint32)
        ex = sel.exprs[offs[lo]:offs[hi]]
        return oracle.eval_selectors(cluster.num_nodes, cluster.num_keys, cluster.labels, o, ex,
                                     None if a is None else a[lo:hi], words=words)

    parts = _map(one, _ranges(P, 4 * threads()))
    return np.concatenate([p[0] for p in parts]), np.concatenate([p[1] for p in parts])


def verify_probes(net, probes, hop_cap):
    """Every result of oracle.verify_probes, by ranges of probes."""
    out = np.zeros(len(probes), oracle._RESULT)

    def one(lo, hi):
        out[lo:hi] = oracle.verify_probes(net, probes, hop_cap, idx=np.arange(lo, hi, dtype=np.uint32))

    _map(one, _ranges(len(probes), 8 * threads()))
    return out


def verify_constrained(net, probes, hop_cap, pol, probes_per_policy):
    """Every result and waypoint word of oracle.verify_constrained."""
    out = np.zeros(len(probes), oracle._RESULT)
    hits = np.zeros(len(probes), np.uint32)

    def one(lo, hi):
        r, h = oracle.verify_constrained(net, probes, hop_cap, pol, probes_per_policy=probes_per_policy,
                                         idx=np.arange(lo, hi, dtype=np.uint32))
        out[lo:hi], hits[lo:hi] = r, h

    _map(one, _ranges(len(probes), 8 * threads()))
    return out, hits


def compliant_reach(graph, sources, masks, words=None):
    """Every row of oracle.compliant_reach, by ranges of masks."""
    masks = np.asarray(masks, np.uint32)
    parts = _map(lambda lo, hi: oracle.compliant_reach(graph, sources, masks[lo:hi], words=words),
                 _ranges(len(masks), len(masks)))
    return np.concatenate(parts)


def end_to_end(e, pol=None):
    """The whole oracle pipeline of an end-to-end batch: selector rows and
    flags, placement, bound probe records, walk results (and waypoint
    words), verdicts and per-intent counts."""
    c = e.cluster
    words = oracle.words_per_row(c.num_nodes)
    bits, flags = eval_selectors(c, e.intents, words)
    assign = oracle.place_pods(bits, c.num_nodes, e.pods_per_intent, e.place_draws)
    probes = oracle.bind_probes(e.probes.probes, e.probes_per_intent, e.pods_per_intent, assign, e.network.host_ip)
    out = {"bits": bits, "flags": flags, "assign": assign, "probes": probes}
    if pol is None:
        res = verify_probes(e.network, probes, e.probes.hop_cap)
        passed, counts = oracle.aggregate(bits, c.num_nodes, flags, assign, e.pods_per_intent, res,
                                          e.probes_per_intent)
    else:
        res, hits = verify_constrained(e.network, probes, e.probes.hop_cap, pol, e.probes_per_intent)
        passed, counts = oracle.aggregate_constrained(bits, c.num_nodes, flags, assign, e.pods_per_intent, res,
                                                      e.probes_per_intent, hits, pol)
        out["hits"] = hits
    out.update(results=res, passed=passed, counts=counts)
    return out
