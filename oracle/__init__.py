"""CPU oracle of the cross-layer privacy validator (test infrastructure).

Only the test suite, the package smoke check and the benchmark's CPU-baseline
leg may import this package.  The product path (the CUDA library and its
binding) never imports, links or executes anything here.

The arithmetic lives in ``pv_oracle.c`` (plain single-threaded C, compiled
with gcc by :func:`build`); this module only marshals numpy arrays.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
from typing import Optional

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "pv_oracle.c")
_LIB = os.path.join(_HERE, "liboracle.so")
_lib = None

# record layouts (byte-compatible with the structs in pv_oracle.c)
_RESULT = np.dtype([("status", "u1"), ("hops", "u1"), ("last_switch", "<u2")])


def build(force: bool = False) -> str:
    """Compile the oracle shared library if it is missing or stale."""
    if force or not os.path.exists(_LIB) or os.path.getmtime(_LIB) < os.path.getmtime(_SRC):
        tmp = _LIB + f".tmp{os.getpid()}"
        subprocess.check_call(["gcc", "-O2", "-std=c11", "-shared", "-fPIC", "-o", tmp, _SRC])
        os.replace(tmp, _LIB)
    return _LIB


def _load():
    global _lib
    if _lib is None:
        build()
        _lib = ctypes.CDLL(_LIB)
        _lib.oracle_first_match.restype = ctypes.c_int32
        _lib.oracle_eval_selectors.restype = ctypes.c_int
        _lib.oracle_eval_selector_terms.restype = ctypes.c_int
        _lib.oracle_compliant_reach.restype = ctypes.c_int
    return _lib


def _p(a: Optional[np.ndarray]):
    if a is None:
        return None
    assert a.flags["C_CONTIGUOUS"]
    return ctypes.c_void_p(a.ctypes.data)


def struct_sizes():
    out = np.zeros(4, np.uint32)
    _load().oracle_struct_sizes(_p(out))
    return tuple(int(x) for x in out)


def words_per_row(num_bits: int) -> int:
    return max(4, ((num_bits + 127) // 128) * 4)


# ----------------------------------------------------------------------------
def eval_selectors(num_nodes, num_keys, labels, expr_offs, exprs, assign=None, words=None):
    """Feasible-node bitsets and per-pod flags (see pv_oracle.c)."""
    lib = _load()
    labels = np.ascontiguousarray(labels, np.uint16)
    offs = np.ascontiguousarray(expr_offs, np.uint32)
    exprs = np.ascontiguousarray(exprs)
    P = len(offs) - 1
    W = words or words_per_row(num_nodes)
    bits = np.zeros((P, W), np.uint32)
    flags = np.zeros(P, np.uint8)
    a = None if assign is None else np.ascontiguousarray(assign, np.uint32)
    rc = lib.oracle_eval_selectors(ctypes.c_uint32(num_nodes), ctypes.c_uint32(num_keys), _p(labels),
                                   ctypes.c_uint32(P), _p(offs), ctypes.c_uint32(len(exprs)), _p(exprs),
                                   _p(a), _p(bits), ctypes.c_uint32(W), _p(flags))
    if rc != 0:
        raise MemoryError("oracle inventory allocation failed")
    return bits, flags


def eval_selector_terms(num_nodes, num_keys, labels, pod_terms, term_offs, exprs, assign=None, words=None):
    """Multi-term selectors: returns (bits [P, W] uint32, flags [P] uint8)."""
    lib = _load()
    W = words or words_per_row(num_nodes)
    labels = np.ascontiguousarray(labels, np.uint16)
    pt = np.ascontiguousarray(pod_terms, np.uint32)
    to = np.ascontiguousarray(term_offs, np.uint32)
    exprs = np.ascontiguousarray(exprs)
    P = len(pt) - 1
    bits = np.zeros((P, W), np.uint32)
    flags = np.zeros(P, np.uint8)
    asg = None if assign is None else np.ascontiguousarray(assign, np.uint32)
    rc = lib.oracle_eval_selector_terms(ctypes.c_uint32(num_nodes), ctypes.c_uint32(num_keys), _p(labels),
                                        ctypes.c_uint32(P), _p(pt), ctypes.c_uint32(len(to) - 1), _p(to),
                                        ctypes.c_uint32(len(exprs)), _p(exprs), _p(asg), _p(bits),
                                        ctypes.c_uint32(W), _p(flags))
    if rc != 0:
        raise MemoryError("oracle inventory allocation failed")
    return bits, flags


def first_match(rules, in_port, src, dst, dport) -> int:
    rules = np.ascontiguousarray(rules)
    return int(_load().oracle_first_match(_p(rules), ctypes.c_uint32(len(rules)), ctypes.c_uint32(in_port),
                                          ctypes.c_uint32(src), ctypes.c_uint32(dst), ctypes.c_uint32(dport)))


def verify_probes(net, probes, hop_cap, idx=None):
    """Walk the probes (all, or probes[idx]) and return RESULT records."""
    lib = _load()
    probes = np.ascontiguousarray(probes)
    ix = None if idx is None else np.ascontiguousarray(idx, np.uint32)
    n = len(probes) if ix is None else len(ix)
    out = np.zeros(n, _RESULT)
    arr = [np.ascontiguousarray(x) for x in (net.rule_offs.astype(np.uint32), net.rules,
                                             net.switch_region.astype(np.uint8), net.port_offs.astype(np.uint32),
                                             net.port_peer.astype(np.int32), net.host_switch.astype(np.uint16),
                                             net.host_port.astype(np.uint16), net.host_ip.astype(np.uint32))]
    lib.oracle_verify_probes(ctypes.c_uint32(net.num_switches), _p(arr[0]), _p(arr[1]), _p(arr[2]), _p(arr[3]),
                             _p(arr[4]), ctypes.c_uint32(net.num_hosts), _p(arr[5]), _p(arr[6]), _p(arr[7]),
                             _p(probes), _p(ix), ctypes.c_uint32(n), ctypes.c_uint32(hop_cap), _p(out))
    return out


def compliant_reach(graph, sources, masks, pairs=None, words=None):
    """Reach rows [num_masks, num_src, W] (or [num_pairs, W] for pairs)."""
    lib = _load()
    V = graph.num_vertices
    W = words or words_per_row(V)
    offs = np.ascontiguousarray(graph.offs, np.uint32)
    cols = np.ascontiguousarray(graph.cols, np.uint32)
    region = np.ascontiguousarray(graph.region, np.uint8)
    src = np.ascontiguousarray(sources, np.uint32)
    msk = np.ascontiguousarray(masks, np.uint32)
    if pairs is None:
        out = np.zeros((len(msk), len(src), W), np.uint32)
        pr, npairs = None, 0
    else:
        pr = np.ascontiguousarray(pairs, np.uint32).reshape(-1, 2)
        npairs = len(pr)
        out = np.zeros((npairs, W), np.uint32)
    rc = lib.oracle_compliant_reach(ctypes.c_uint32(V), _p(offs), ctypes.c_uint32(len(cols)), _p(cols), _p(region),
                                    ctypes.c_uint32(len(src)),
                                    _p(src), ctypes.c_uint32(len(msk)), _p(msk), _p(pr), ctypes.c_uint32(npairs),
                                    _p(out), ctypes.c_uint32(W))
    if rc != 0:
        raise MemoryError("oracle reach allocation failed")
    return out


def place_pods(bits, num_nodes, pods_per_group, draws):
    bits = np.ascontiguousarray(bits, np.uint32)
    G, W = bits.shape
    draws = np.ascontiguousarray(draws, np.uint64)
    assign = np.zeros(G * pods_per_group, np.uint32)
    _load().oracle_place_pods(ctypes.c_uint32(G), ctypes.c_uint32(pods_per_group), ctypes.c_uint32(num_nodes),
                              _p(bits), ctypes.c_uint32(W), _p(draws), _p(assign))
    return assign


def bind_probes(probes, probes_per_group, pods_per_group, assign, host_ip):
    """Returns a bound copy of the probe array."""
    out = np.ascontiguousarray(probes).copy()
    assign = np.ascontiguousarray(assign, np.uint32)
    hip = np.ascontiguousarray(host_ip, np.uint32)
    _load().oracle_bind_probes(ctypes.c_uint32(len(out)), _p(out), ctypes.c_uint32(probes_per_group),
                               ctypes.c_uint32(pods_per_group), _p(assign), ctypes.c_uint32(len(hip)), _p(hip))
    return out


def aggregate(bits, num_nodes, group_flags, assign, pods_per_group, results, probes_per_group):
    bits = np.ascontiguousarray(bits, np.uint32)
    G, W = bits.shape
    gf = np.ascontiguousarray(group_flags, np.uint8)
    assign = np.ascontiguousarray(assign, np.uint32)
    results = np.ascontiguousarray(results)
    passed = np.zeros(G, np.uint8)
    counts = np.zeros((G, 8), np.uint32)
    _load().oracle_aggregate(ctypes.c_uint32(G), ctypes.c_uint32(pods_per_group), ctypes.c_uint32(num_nodes),
                             _p(bits), ctypes.c_uint32(W), _p(gf), _p(assign), ctypes.c_uint32(probes_per_group),
                             _p(results), _p(passed), _p(counts))
    return passed, counts


def _policy_arrays(pol):
    return [np.ascontiguousarray(x) for x in (pol.forbid_offs.astype(np.uint32), pol.forbid.astype(np.uint16),
                                              pol.must_offs.astype(np.uint32), pol.must.astype(np.uint16),
                                              pol.concrete.astype(np.uint8))]


def verify_constrained(net, probes, hop_cap, pol, probe_policy=None, probes_per_policy=0, idx=None):
    """Walk with path constraints; returns (RESULT records, waypoint hit bits)."""
    lib = _load()
    probes = np.ascontiguousarray(probes)
    ix = None if idx is None else np.ascontiguousarray(idx, np.uint32)
    n = len(probes) if ix is None else len(ix)
    out = np.zeros(n, _RESULT)
    hits = np.zeros(n, np.uint32)
    arr = [np.ascontiguousarray(x) for x in (net.rule_offs.astype(np.uint32), net.rules,
                                             net.switch_region.astype(np.uint8), net.port_offs.astype(np.uint32),
                                             net.port_peer.astype(np.int32), net.host_switch.astype(np.uint16),
                                             net.host_port.astype(np.uint16), net.host_ip.astype(np.uint32))]
    pp = None if probe_policy is None else np.ascontiguousarray(probe_policy, np.uint32)
    fo, fb, mo, mg, _ = _policy_arrays(pol)
    lib.oracle_verify_constrained(_p(arr[0]), _p(arr[1]), _p(arr[2]), _p(arr[3]), _p(arr[4]),
                                  ctypes.c_uint32(net.num_hosts), _p(arr[5]), _p(arr[6]), _p(arr[7]), _p(probes),
                                  _p(pp), ctypes.c_uint32(probes_per_policy), ctypes.c_uint32(pol.num_policies),
                                  _p(fo), _p(fb), _p(mo), _p(mg), _p(ix), ctypes.c_uint32(n),
                                  ctypes.c_uint32(hop_cap), _p(out), _p(hits))
    return out, hits


def aggregate_constrained(bits, num_nodes, group_flags, assign, pods_per_group, results, probes_per_group, hits,
                          pol, group_policy=None):
    bits = np.ascontiguousarray(bits, np.uint32)
    G, W = bits.shape
    gf = np.ascontiguousarray(group_flags, np.uint8)
    assign = np.ascontiguousarray(assign, np.uint32)
    results = np.ascontiguousarray(results)
    hits = np.ascontiguousarray(hits, np.uint32)
    gp = None if group_policy is None else np.ascontiguousarray(group_policy, np.uint32)
    _, _, mo, _, cc = _policy_arrays(pol)
    passed = np.zeros(G, np.uint8)
    counts = np.zeros((G, 8), np.uint32)
    _load().oracle_aggregate_constrained(ctypes.c_uint32(G), ctypes.c_uint32(pods_per_group),
                                         ctypes.c_uint32(num_nodes), _p(bits), ctypes.c_uint32(W), _p(gf),
                                         _p(assign), ctypes.c_uint32(probes_per_group), _p(results), _p(hits),
                                         _p(gp), ctypes.c_uint32(pol.num_policies), _p(mo), _p(cc), _p(passed),
                                         _p(counts))
    return passed, counts


def schedule_paths(net, requests, pol=None, weights=None, max_len=64):
    """Scheduled paths: (visits [R, max_len] u32, lengths [R] u8, status [R] u8)."""
    assert 1 <= max_len <= 255
    lib = _load()
    req = np.ascontiguousarray(requests)
    R = len(req)
    hops = np.zeros((R, max_len), np.uint32)
    ln = np.zeros(R, np.uint8)
    st = np.zeros(R, np.uint8)
    arr = [np.ascontiguousarray(x) for x in (net.switch_region.astype(np.uint8), net.port_offs.astype(np.uint32),
                                             net.port_peer.astype(np.int32), net.host_switch.astype(np.uint16),
                                             net.host_port.astype(np.uint16))]
    w = None if weights is None else np.ascontiguousarray(weights, np.uint16)
    if pol is None:
        P, fo, fb, mo, mg = 0, None, None, None, None
    else:
        P = pol.num_policies
        fo, fb, mo, mg, _ = _policy_arrays(pol)
    lib.oracle_schedule_paths(ctypes.c_uint32(net.num_switches), _p(arr[0]), _p(arr[1]), _p(arr[2]),
                              ctypes.c_uint32(net.num_hosts), _p(arr[3]), _p(arr[4]), _p(w), ctypes.c_uint32(P),
                              _p(fo), _p(fb), _p(mo), _p(mg), ctypes.c_uint32(R), _p(req), ctypes.c_uint32(max_len),
                              _p(hops), _p(ln), _p(st))
    return hops, ln, st


def compile_path_rules(net, requests, hops, lengths, status, priority=65535):
    """Per-hop rules: (rules [R * max_len] RULE records, rule_switch [R * max_len] u16)."""
    req = np.ascontiguousarray(requests)
    R, L = hops.shape
    rules = np.zeros(R * L, net.rules.dtype)
    rsw = np.zeros(R * L, np.uint16)
    hip = np.ascontiguousarray(net.host_ip, np.uint32)
    _load().oracle_compile_path_rules(ctypes.c_uint32(R), _p(req), _p(hip), ctypes.c_uint32(L),
                                      _p(np.ascontiguousarray(hops, np.uint32)),
                                      _p(np.ascontiguousarray(lengths, np.uint8)),
                                      _p(np.ascontiguousarray(status, np.uint8)), ctypes.c_uint16(priority),
                                      _p(rules), _p(rsw))
    return rules, rsw
