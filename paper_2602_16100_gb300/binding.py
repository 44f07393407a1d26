"""Thin Python binding of libpv.so (include/pv.h), same names as the C ABI.

Argument marshalling only: device arguments accept a torch tensor (its
``data_ptr()``) or a raw integer address; host arrays are numpy arrays;
streams accept a ``torch.cuda.Stream``, a raw ``cudaStream_t`` integer or
None (legacy default stream).  Every call returns the C status code; a
non-zero status raises :class:`PVError` carrying ``pv_last_error``.

There is no fallback of any kind: if libpv.so is missing or cannot be loaded
every call raises.
"""
from __future__ import annotations

import ctypes
import os
from typing import Optional

import numpy as np

from . import build as _build

PV_OK, PV_EINVAL, PV_ENOMEM, PV_ECUDA, PV_ESTATE, PV_ETIMEOUT, PV_ENOTIMPL = range(7)
PV_OPT_SELECTOR_KERNEL, PV_OPT_WALK_KERNEL, PV_OPT_WALK_LANE_MAX, PV_OPT_TEST_STALL_STAGING = 1, 2, 3, 4
PV_STAT_SELECTOR_ROWS_BUILT, PV_STAT_SCRATCH_BYTES, PV_STAT_WALK_INDEX_FITS, PV_STAT_WALK_INDEX_BYTES = 1, 2, 3, 4
PV_STAT_WALK_LIVE_TOTAL, PV_STAT_REACH_COMPONENTS = 5, 6
PV_OPT_REACH_KERNEL, PV_OPT_WALK_CYCLES, PV_OPT_WALK_TAIL_HOP = 5, 6, 7
PV_OPT_WALK_STATS, PV_OPT_SELECTOR_DEDUPE, PV_OPT_SCHED_KERNEL = 8, 9, 10
(PV_STAT_WALK_FIRST_MATCHES, PV_STAT_WALK_RULE_TESTS, PV_STAT_WALK_INTERVAL_LOOKUPS, PV_STAT_WALK_SCAN_DEPTH,
 PV_STAT_WALK_INDEX_MISMATCHES) = 7, 8, 9, 10, 11

#: every entry point declared in include/pv.h
SYMBOLS = ("pv_create", "pv_destroy", "pv_last_error", "pv_sync", "pv_version", "pv_load_cluster",
           "pv_eval_selectors", "pv_load_flow_tables", "pv_verify_probes", "pv_compliant_reach",
           "pv_place_pods", "pv_bind_probes", "pv_aggregate_intents", "pv_set_option", "pv_get_stat",
           "pv_profile_enable", "pv_profile_collect", "pv_profile_read", "pv_compliant_reach_noalloc",
           "pv_load_path_policies", "pv_verify_probes_constrained", "pv_aggregate_constrained",
           "pv_eval_selector_terms", "pv_schedule_paths", "pv_compile_path_rules", "pv_install_path_rules",
           "pv_bind_flows", "pv_verify_flows", "pv_verify_flows_constrained", "pv_verify_flow_columns",
           "pv_verify_flow_columns_constrained", "pv_load_flow_tables_begin",
           "pv_load_flow_tables_end")

#: kernel groups timed by the library profiler (PV_K_* in include/pv.h)
PV_K_NAMES = ("selector", "place", "bind", "walk_init", "walk_regroup", "walk_hop", "aggregate", "reach", "schedule")

_lib = None


class PVError(RuntimeError):
    def __init__(self, code: int, msg: str):
        super().__init__(f"libpv error {code}: {msg}")
        self.code = code


def library_path() -> str:
    return _build.LIB


def load_library(path: Optional[str] = None):
    """Load libpv.so (ctypes).  Raises if it is missing; never falls back."""
    global _lib
    if _lib is not None and path is None:
        return _lib
    p = path or _build.LIB
    if not os.path.exists(p):
        raise RuntimeError(f"libpv.so not built ({p}); run paper_2602_16100_gb300.build.build_library()")
    lib = ctypes.CDLL(p)
    u32, i32, i64, vp = ctypes.c_uint32, ctypes.c_int32, ctypes.c_int64, ctypes.c_void_p
    sig = {
        "pv_create": (ctypes.c_int, [ctypes.POINTER(vp), ctypes.c_int]),
        "pv_destroy": (None, [vp]),
        "pv_last_error": (ctypes.c_char_p, [vp]),
        "pv_sync": (ctypes.c_int, [vp, vp]),
        "pv_version": (ctypes.c_int, []),
        "pv_load_cluster": (ctypes.c_int, [vp, u32, u32, vp]),
        "pv_eval_selectors": (ctypes.c_int, [vp, u32, vp, u32, vp, vp, vp, u32, vp, vp]),
        "pv_load_flow_tables": (ctypes.c_int, [vp, u32, vp, vp, vp, vp, vp, u32, vp, vp, vp]),
        "pv_load_flow_tables_begin": (ctypes.c_int, [vp, u32, vp, vp, vp, vp, vp, u32, vp, vp, vp]),
        "pv_load_flow_tables_end": (ctypes.c_int, [vp]),
        "pv_verify_probes": (ctypes.c_int, [vp, u32, vp, u32, vp, vp]),
        "pv_compliant_reach": (ctypes.c_int, [vp, u32, vp, u32, vp, vp, u32, vp, u32, vp, vp, u32, vp]),
        "pv_place_pods": (ctypes.c_int, [vp, u32, u32, vp, u32, vp, vp, vp]),
        "pv_bind_probes": (ctypes.c_int, [vp, u32, vp, u32, u32, vp, vp]),
        "pv_bind_flows": (ctypes.c_int, [vp, u32, vp, u32, u32, vp, vp, vp, vp]),
        "pv_verify_flows": (ctypes.c_int, [vp, u32, vp, u32, u32, vp, vp, u32, vp, vp, vp]),
        "pv_verify_flows_constrained": (ctypes.c_int, [vp, u32, vp, u32, u32, vp, vp, u32, vp, u32, u32, vp, vp, vp,
                                                       vp]),
        "pv_verify_flow_columns": (ctypes.c_int, [vp, u32, vp, vp, u32, u32, vp, vp, u32, vp, vp, vp]),
        "pv_verify_flow_columns_constrained": (ctypes.c_int, [vp, u32, vp, vp, u32, u32, vp, vp, u32, vp, u32, u32,
                                                              vp, vp, vp, vp]),
        "pv_aggregate_intents": (ctypes.c_int, [vp, u32, u32, vp, u32, vp, vp, u32, vp, vp, vp, vp]),
        "pv_set_option": (ctypes.c_int, [vp, ctypes.c_int, i64]),
        "pv_get_stat": (ctypes.c_int, [vp, ctypes.c_int, ctypes.POINTER(i64)]),
        "pv_profile_enable": (ctypes.c_int, [vp, ctypes.c_int]),
        "pv_profile_collect": (ctypes.c_int, [vp, vp]),
        "pv_profile_read": (ctypes.c_int, [vp, ctypes.c_int, ctypes.POINTER(ctypes.c_double),
                                           ctypes.POINTER(ctypes.c_uint64)]),
        "pv_compliant_reach_noalloc": (ctypes.c_int, [u32, vp, u32, vp, vp, u32, vp, u32, vp, vp, u32, vp]),
        "pv_load_path_policies": (ctypes.c_int, [vp, u32, vp, vp, vp, vp, vp]),
        "pv_eval_selector_terms": (ctypes.c_int, [vp, u32, vp, u32, vp, u32, vp, vp, vp, u32, vp, vp]),
        "pv_schedule_paths": (ctypes.c_int, [vp, u32, vp, vp, u32, vp, vp, vp, vp]),
        "pv_compile_path_rules": (ctypes.c_int, [vp, u32, vp, u32, vp, vp, vp, ctypes.c_uint16, vp, vp, vp]),
        "pv_install_path_rules": (ctypes.c_int, [vp, u32, vp, vp]),
        "pv_verify_probes_constrained": (ctypes.c_int, [vp, u32, vp, u32, vp, u32, u32, vp, vp, vp]),
        "pv_aggregate_constrained": (ctypes.c_int, [vp, u32, u32, vp, u32, vp, vp, u32, vp, vp, vp, u32, vp, vp,
                                                    vp]),
    }
    for name, (res, args) in sig.items():
        f = getattr(lib, name)
        f.restype = res
        f.argtypes = args
    if path is None:
        _lib = lib
    return lib


# ----------------------------------------------------------------------------
# marshalling helpers
# ----------------------------------------------------------------------------
def _dev(x) -> Optional[int]:
    if x is None:
        return None
    if isinstance(x, int):
        return x
    if hasattr(x, "data_ptr"):
        if not x.is_cuda:
            raise ValueError("expected a CUDA tensor for a device argument")
        if not x.is_contiguous():
            raise ValueError("device arguments must be contiguous")
        return x.data_ptr()
    raise TypeError(f"cannot pass {type(x)!r} as a device pointer")


def _host(a) -> Optional[int]:
    if a is None:
        return None
    if not isinstance(a, np.ndarray) or not a.flags["C_CONTIGUOUS"]:
        raise ValueError("host arguments must be C-contiguous numpy arrays")
    return a.ctypes.data


def _stream(s) -> Optional[int]:
    if s is None or s == 0:
        return None
    if isinstance(s, int):
        return s
    return s.cuda_stream


def _check(ctx, rc: int) -> int:
    if rc != PV_OK:
        msg = load_library().pv_last_error(ctx)
        raise PVError(rc, msg.decode() if msg else "")
    return rc


# ----------------------------------------------------------------------------
# C ABI, one function per entry point
# ----------------------------------------------------------------------------
def pv_version() -> int:
    return load_library().pv_version()


def pv_create(cuda_device: int = 0):
    ctx = ctypes.c_void_p()
    rc = load_library().pv_create(ctypes.byref(ctx), cuda_device)
    if rc != PV_OK:
        raise PVError(rc, f"pv_create(device={cuda_device}) failed")
    return ctx


def pv_destroy(ctx) -> None:
    load_library().pv_destroy(ctx)
    _TABLE_LOADS.pop(ctx.value, None)


def pv_last_error(ctx) -> str:
    m = load_library().pv_last_error(ctx)
    return m.decode() if m else ""


def pv_sync(ctx, stream=None) -> int:
    return _check(ctx, load_library().pv_sync(ctx, _stream(stream)))


def pv_set_option(ctx, option: int, value: int) -> int:
    return _check(ctx, load_library().pv_set_option(ctx, option, value))


def pv_get_stat(ctx, stat: int) -> int:
    v = ctypes.c_int64()
    _check(ctx, load_library().pv_get_stat(ctx, stat, ctypes.byref(v)))
    return v.value


def pv_profile_enable(ctx, on: bool) -> int:
    return _check(ctx, load_library().pv_profile_enable(ctx, 1 if on else 0))


def pv_profile_collect(ctx, stream=None) -> int:
    return _check(ctx, load_library().pv_profile_collect(ctx, _stream(stream)))


def pv_profile_read(ctx, group: int):
    """(total device milliseconds, kernel launches) of one kernel group."""
    ms, n = ctypes.c_double(), ctypes.c_uint64()
    _check(ctx, load_library().pv_profile_read(ctx, group, ctypes.byref(ms), ctypes.byref(n)))
    return ms.value, n.value


def pv_load_cluster(ctx, num_nodes: int, num_keys: int, labels: np.ndarray) -> int:
    labels = np.ascontiguousarray(labels, np.uint16)
    return _check(ctx, load_library().pv_load_cluster(ctx, num_nodes, num_keys, _host(labels)))


def pv_eval_selectors(ctx, num_pods, d_expr_offs, num_exprs, d_exprs, d_assign, d_bits, words_per_row, d_flags,
                      stream=None) -> int:
    return _check(ctx, load_library().pv_eval_selectors(ctx, num_pods, _dev(d_expr_offs), num_exprs, _dev(d_exprs),
                                                        _dev(d_assign), _dev(d_bits), words_per_row, _dev(d_flags),
                                                        _stream(stream)))


def _table_arrays(rule_offs, rules, switch_region, port_offs, port_peer, host_switch, host_port, host_ip):
    return [np.ascontiguousarray(rule_offs, np.uint32), np.ascontiguousarray(rules),
            np.ascontiguousarray(switch_region, np.uint8), np.ascontiguousarray(port_offs, np.uint32),
            np.ascontiguousarray(port_peer, np.int32), np.ascontiguousarray(host_switch, np.uint16),
            np.ascontiguousarray(host_port, np.uint16), np.ascontiguousarray(host_ip, np.uint32)]


def pv_load_flow_tables(ctx, num_switches, rule_offs, rules, switch_region, port_offs, port_peer, num_hosts,
                        host_switch, host_port, host_ip) -> int:
    a = _table_arrays(rule_offs, rules, switch_region, port_offs, port_peer, host_switch, host_port, host_ip)
    return _check(ctx, load_library().pv_load_flow_tables(ctx, num_switches, _host(a[0]), _host(a[1]), _host(a[2]),
                                                          _host(a[3]), _host(a[4]), num_hosts, _host(a[5]),
                                                          _host(a[6]), _host(a[7])))


#: host arrays of a two-part table load, kept alive until its end (by context)
_TABLE_LOADS = {}


def pv_load_flow_tables_begin(ctx, num_switches, rule_offs, rules, switch_region, port_offs, port_peer, num_hosts,
                              host_switch, host_port, host_ip) -> int:
    a = _table_arrays(rule_offs, rules, switch_region, port_offs, port_peer, host_switch, host_port, host_ip)
    rc = _check(ctx, load_library().pv_load_flow_tables_begin(ctx, num_switches, _host(a[0]), _host(a[1]),
                                                              _host(a[2]), _host(a[3]), _host(a[4]), num_hosts,
                                                              _host(a[5]), _host(a[6]), _host(a[7])))
    _TABLE_LOADS[ctx.value] = a
    return rc


def pv_load_flow_tables_end(ctx) -> int:
    try:
        return _check(ctx, load_library().pv_load_flow_tables_end(ctx))
    finally:
        _TABLE_LOADS.pop(ctx.value, None)


def pv_verify_probes(ctx, num_probes, d_probes, hop_cap, d_out, stream=None) -> int:
    return _check(ctx, load_library().pv_verify_probes(ctx, num_probes, _dev(d_probes), hop_cap, _dev(d_out),
                                                       _stream(stream)))


def pv_eval_selector_terms(ctx, num_pods, d_pod_terms, num_terms, d_term_offs, num_exprs, d_exprs, d_assign, d_bits,
                           words_per_row, d_flags, stream=None) -> int:
    return _check(ctx, load_library().pv_eval_selector_terms(ctx, num_pods, _dev(d_pod_terms), num_terms,
                                                             _dev(d_term_offs), num_exprs, _dev(d_exprs),
                                                             _dev(d_assign), _dev(d_bits), words_per_row,
                                                             _dev(d_flags), _stream(stream)))


def pv_schedule_paths(ctx, num_requests, d_requests, d_link_weights, max_len, d_visits, d_len, d_status,
                      stream=None) -> int:
    return _check(ctx, load_library().pv_schedule_paths(ctx, num_requests, _dev(d_requests), _dev(d_link_weights),
                                                        max_len, _dev(d_visits), _dev(d_len), _dev(d_status),
                                                        _stream(stream)))


def pv_compile_path_rules(ctx, num_requests, d_requests, max_len, d_visits, d_len, d_status, priority, d_rules,
                          d_rule_switch, stream=None) -> int:
    return _check(ctx, load_library().pv_compile_path_rules(ctx, num_requests, _dev(d_requests), max_len,
                                                            _dev(d_visits), _dev(d_len), _dev(d_status), priority,
                                                            _dev(d_rules), _dev(d_rule_switch), _stream(stream)))


def pv_install_path_rules(ctx, num_slots, d_rules, d_rule_switch) -> int:
    return _check(ctx, load_library().pv_install_path_rules(ctx, num_slots, _dev(d_rules), _dev(d_rule_switch)))


def pv_load_path_policies(ctx, num_policies, forbid_offs, forbid, must_offs, must, concrete) -> int:
    a = [np.ascontiguousarray(forbid_offs, np.uint32), np.ascontiguousarray(forbid, np.uint16),
         np.ascontiguousarray(must_offs, np.uint32), np.ascontiguousarray(must, np.uint16),
         np.ascontiguousarray(concrete, np.uint8)]
    return _check(ctx, load_library().pv_load_path_policies(ctx, num_policies, *[_host(x) for x in a]))


def pv_verify_probes_constrained(ctx, num_probes, d_probes, hop_cap, d_probe_policy, probes_per_policy, d_out,
                                 d_waypoints, stream=None, first_policy=0) -> int:
    return _check(ctx, load_library().pv_verify_probes_constrained(ctx, num_probes, _dev(d_probes), hop_cap,
                                                                   _dev(d_probe_policy), probes_per_policy,
                                                                   first_policy, _dev(d_out), _dev(d_waypoints),
                                                                   _stream(stream)))


def pv_aggregate_constrained(ctx, num_groups, pods_per_group, d_bits, words_per_row, d_group_flags, d_assign,
                             probes_per_group, d_results, d_waypoints, d_group_policy, d_pass, d_counts,
                             stream=None, first_policy=0) -> int:
    return _check(ctx, load_library().pv_aggregate_constrained(ctx, num_groups, pods_per_group, _dev(d_bits),
                                                               words_per_row, _dev(d_group_flags), _dev(d_assign),
                                                               probes_per_group, _dev(d_results),
                                                               _dev(d_waypoints), _dev(d_group_policy),
                                                               first_policy, _dev(d_pass), _dev(d_counts),
                                                               _stream(stream)))


def pv_compliant_reach(ctx, V, d_offs, num_edges, d_cols, d_region, num_src, d_src, num_masks, d_masks, d_reach,
                       words_per_row, stream=None) -> int:
    return _check(ctx, load_library().pv_compliant_reach(ctx, V, _dev(d_offs), num_edges, _dev(d_cols),
                                                         _dev(d_region), num_src, _dev(d_src), num_masks,
                                                         _dev(d_masks), _dev(d_reach), words_per_row,
                                                         _stream(stream)))


def pv_place_pods(ctx, num_groups, pods_per_group, d_bits, words_per_row, d_draws, d_assign, stream=None) -> int:
    return _check(ctx, load_library().pv_place_pods(ctx, num_groups, pods_per_group, _dev(d_bits), words_per_row,
                                                    _dev(d_draws), _dev(d_assign), _stream(stream)))


def pv_bind_probes(ctx, num_probes, d_probes, probes_per_group, pods_per_group, d_assign, stream=None) -> int:
    return _check(ctx, load_library().pv_bind_probes(ctx, num_probes, _dev(d_probes), probes_per_group,
                                                     pods_per_group, _dev(d_assign), _stream(stream)))


def pv_bind_flows(ctx, num_probes, d_flows, probes_per_group, pods_per_group, d_assign, d_group_mask, d_probes,
                  stream=None) -> int:
    return _check(ctx, load_library().pv_bind_flows(ctx, num_probes, _dev(d_flows), probes_per_group,
                                                    pods_per_group, _dev(d_assign), _dev(d_group_mask),
                                                    _dev(d_probes), _stream(stream)))


def pv_verify_flows(ctx, num_probes, d_flows, probes_per_group, pods_per_group, d_assign, d_group_mask, hop_cap,
                    d_probes, d_out, stream=None) -> int:
    return _check(ctx, load_library().pv_verify_flows(ctx, num_probes, _dev(d_flows), probes_per_group,
                                                      pods_per_group, _dev(d_assign), _dev(d_group_mask), hop_cap,
                                                      _dev(d_probes), _dev(d_out), _stream(stream)))


def pv_verify_flows_constrained(ctx, num_probes, d_flows, probes_per_group, pods_per_group, d_assign, d_group_mask,
                                hop_cap, d_probe_policy, probes_per_policy, first_policy, d_probes, d_out,
                                d_waypoints, stream=None) -> int:
    return _check(ctx, load_library().pv_verify_flows_constrained(
        ctx, num_probes, _dev(d_flows), probes_per_group, pods_per_group, _dev(d_assign), _dev(d_group_mask),
        hop_cap, _dev(d_probe_policy), probes_per_policy, first_policy, _dev(d_probes), _dev(d_out),
        _dev(d_waypoints), _stream(stream)))


def pv_verify_flow_columns(ctx, num_probes, d_dst_ip, d_dport, probes_per_group, pods_per_group, d_assign,
                           d_group_mask, hop_cap, d_probes, d_out, stream=None) -> int:
    return _check(ctx, load_library().pv_verify_flow_columns(
        ctx, num_probes, _dev(d_dst_ip), _dev(d_dport), probes_per_group, pods_per_group, _dev(d_assign),
        _dev(d_group_mask), hop_cap, _dev(d_probes), _dev(d_out), _stream(stream)))


def pv_verify_flow_columns_constrained(ctx, num_probes, d_dst_ip, d_dport, probes_per_group, pods_per_group,
                                       d_assign, d_group_mask, hop_cap, d_probe_policy, probes_per_policy,
                                       first_policy, d_probes, d_out, d_waypoints, stream=None) -> int:
    return _check(ctx, load_library().pv_verify_flow_columns_constrained(
        ctx, num_probes, _dev(d_dst_ip), _dev(d_dport), probes_per_group, pods_per_group, _dev(d_assign),
        _dev(d_group_mask), hop_cap, _dev(d_probe_policy), probes_per_policy, first_policy, _dev(d_probes),
        _dev(d_out), _dev(d_waypoints), _stream(stream)))


def pv_aggregate_intents(ctx, num_groups, pods_per_group, d_bits, words_per_row, d_group_flags, d_assign,
                         probes_per_group, d_results, d_pass, d_counts, stream=None) -> int:
    return _check(ctx, load_library().pv_aggregate_intents(ctx, num_groups, pods_per_group, _dev(d_bits),
                                                           words_per_row, _dev(d_group_flags), _dev(d_assign),
                                                           probes_per_group, _dev(d_results), _dev(d_pass),
                                                           _dev(d_counts), _stream(stream)))


def pv_compliant_reach_noalloc(V, d_offs, num_edges, d_cols, d_region, num_src, d_src, num_masks, d_masks, d_reach,
                               words_per_row, stream=None) -> int:
    """Compliant reach without any device allocation (no context): for callers
    whose device memory is owned by another allocator or a fixed budget, or
    that cannot absorb cudaMalloc/cudaFree synchronisation.  Works in a static
    ~1.2 MB device array shared by all calls (V <= 16384, num_edges <=
    262144).  Returns the C status; a non-zero status raises PVError."""
    rc = load_library().pv_compliant_reach_noalloc(V, _dev(d_offs), num_edges, _dev(d_cols), _dev(d_region), num_src,
                                                   _dev(d_src), num_masks, _dev(d_masks), _dev(d_reach),
                                                   words_per_row, _stream(stream))
    if rc != PV_OK:
        raise PVError(rc, "pv_compliant_reach_noalloc rejected its arguments or failed")
    return rc
