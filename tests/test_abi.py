"""CPU checks of the C-ABI boundary: the library builds for sm_103a, loads,
exports every entry point include/pv.h declares, and its struct layouts match
the workload arrays byte for byte.  No compute call is made here."""
import ctypes
import os
import re
import subprocess

import numpy as np
import pytest

from paper_2602_16100_gb300 import binding as B
from paper_2602_16100_gb300 import build as BUILD
from paper_2602_16100_gb300 import workloads as W

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "pv.h")


def _declared():
    text = open(HEADER).read()
    return set(re.findall(r"^\s*(?:int|void|const char \*)\s*(pv_\w+)\s*\(", text, re.M))


@pytest.fixture(scope="module")
def lib():
    BUILD.build_library()
    return ctypes.CDLL(BUILD.LIB)


def test_every_declared_symbol_is_exported(lib):
    decl = _declared()
    assert len(decl) >= 15
    for name in decl:
        assert hasattr(lib, name), name
    assert decl == set(B.SYMBOLS)
    out = subprocess.run(["nm", "-D", "--defined-only", BUILD.LIB], capture_output=True, text=True).stdout
    exported = set(re.findall(r"\bT (pv_\w+)", out))
    assert decl <= exported


def test_binding_loads_and_reports_version(lib):
    assert B.pv_version() == 100


def test_struct_layouts_match_header(tmp_path):
    src = tmp_path / "layout.c"
    src.write_text(r'''
#include <stddef.h>
#include <stdio.h>
#include "pv.h"
int main(void) {
  printf("%zu %zu %zu %zu\n", sizeof(pv_expr), sizeof(pv_rule), sizeof(pv_probe), sizeof(pv_result));
  printf("%zu %zu %zu\n", offsetof(pv_expr, op), offsetof(pv_expr, nvals), offsetof(pv_expr, vals));
  printf("%zu %zu %zu %zu %zu %zu %zu %zu\n", offsetof(pv_rule, in_port), offsetof(pv_rule, src_ip),
         offsetof(pv_rule, dst_ip), offsetof(pv_rule, src_len), offsetof(pv_rule, dst_len),
         offsetof(pv_rule, dport_lo), offsetof(pv_rule, dport_hi), offsetof(pv_rule, action));
  printf("%zu %zu %zu %zu\n", offsetof(pv_probe, dst_ip), offsetof(pv_probe, dport),
         offsetof(pv_probe, src_host), offsetof(pv_probe, allowed_mask));
  printf("%zu %zu\n", offsetof(pv_result, hops), offsetof(pv_result, last_switch));
  return 0;
}
''')
    exe = tmp_path / "layout"
    subprocess.check_call(["gcc", "-I", os.path.join(ROOT, "include"), str(src), "-o", str(exe)])
    lines = subprocess.check_output([str(exe)], text=True).split("\n")
    sizes = [int(x) for x in lines[0].split()]
    assert sizes == [W.EXPR_DTYPE.itemsize, W.RULE_DTYPE.itemsize, W.PROBE_DTYPE.itemsize, W.RESULT_DTYPE.itemsize]
    f = W.EXPR_DTYPE.fields
    assert [int(x) for x in lines[1].split()] == [f["op"][1], f["nvals"][1], f["vals"][1]]
    f = W.RULE_DTYPE.fields
    names = ["in_port", "src_ip", "dst_ip", "src_len", "dst_len", "dport_lo", "dport_hi", "action"]
    assert [int(x) for x in lines[2].split()] == [f[n][1] for n in names]
    f = W.PROBE_DTYPE.fields
    assert [int(x) for x in lines[3].split()] == [f[n][1] for n in ["dst_ip", "dport", "src_host", "allowed_mask"]]
    f = W.RESULT_DTYPE.fields
    assert [int(x) for x in lines[4].split()] == [f["hops"][1], f["last_switch"][1]]


def test_constants_match_header():
    text = open(HEADER).read()
    def define(name):
        return int(re.search(rf"#define {name} \(?(-?0x[0-9A-Fa-f]+|-?\d+)", text).group(1), 0)
    assert define("PV_ABSENT") == W.ABSENT
    assert define("PV_ANY_PORT") == W.ANY_PORT and define("PV_DROP") == W.DROP
    assert define("PV_NO_HOST") == W.NO_HOST and define("PV_PEER_HOST") == W.HOST_BIT
    assert define("PV_UNPLACED") == W.UNPLACED


def test_create_without_gpu_fails_cleanly():
    import torch
    if torch.cuda.is_available():
        pytest.skip("a GPU is present")
    with pytest.raises(B.PVError) as e:
        B.pv_create(0)
    assert e.value.code == B.PV_ECUDA


def test_missing_library_raises(tmp_path):
    with pytest.raises(RuntimeError):
        B.load_library(str(tmp_path / "nope.so"))


def test_path_request_layout_matches_header(tmp_path):
    src = tmp_path / "req.c"
    src.write_text(r'''
#include <stddef.h>
#include <stdio.h>
#include "pv.h"
int main(void) {
  printf("%zu %zu %zu\n", sizeof(pv_flow), offsetof(pv_flow, dport), offsetof(pv_flow, reserved));
  printf("%zu %zu %zu %zu %zu\n", sizeof(pv_path_req), offsetof(pv_path_req, dst_host),
         offsetof(pv_path_req, allowed_mask), offsetof(pv_path_req, policy), offsetof(pv_path_req, reserved));
  printf("%d %d %d %d %d\n", PV_PATH_OK, PV_PATH_NOSRC, PV_PATH_BLOCKED, PV_PATH_TOO_LONG, PV_PATH_REPEAT);
  return 0;
}
''')
    exe = tmp_path / "req"
    subprocess.check_call(["gcc", "-I", os.path.join(ROOT, "include"), str(src), "-o", str(exe)])
    lines = subprocess.check_output([str(exe)], text=True).split("\n")
    ff = W.FLOW_DTYPE.fields
    assert [int(x) for x in lines[0].split()] == [W.FLOW_DTYPE.itemsize, ff["dport"][1], ff["reserved"][1]]
    lines = lines[1:]
    f = W.PATH_REQ_DTYPE.fields
    assert [int(x) for x in lines[0].split()] == [W.PATH_REQ_DTYPE.itemsize, f["dst_host"][1], f["allowed_mask"][1],
                                                  f["policy"][1], f["reserved"][1]]
    assert [int(x) for x in lines[1].split()] == [W.PATH_OK, W.PATH_NOSRC, W.PATH_BLOCKED, W.PATH_TOO_LONG,
                                                  W.PATH_REPEAT]


def test_two_part_table_load_keeps_its_host_arrays_until_the_end(monkeypatch):
    """The binding keeps the arrays it hands to pv_load_flow_tables_begin
    (converted copies included) alive until pv_load_flow_tables_end or
    pv_destroy, and drops them afterwards, whether the end succeeds or not
    (a fake library stands in for libpv: no GPU is needed)."""
    seen = {}

    class Fake:
        def __init__(self):
            self.end_rc = B.PV_OK

        def pv_load_flow_tables_begin(self, ctx, S, *ptrs):
            seen["ptrs"] = ptrs
            return B.PV_OK

        def pv_load_flow_tables_end(self, ctx):
            return self.end_rc

        def pv_destroy(self, ctx):
            pass

        def pv_last_error(self, ctx):
            return b"fake failure"

    fake = Fake()
    monkeypatch.setattr(B, "load_library", lambda path=None: fake)
    ctx = ctypes.c_void_p(0x1234)
    net = W.tiny()["network"]
    offs = net.rule_offs.astype(np.int64)   # converted to u32 by the binding: a temporary it must keep
    args = (net.num_switches, offs, net.rules, net.switch_region, net.port_offs, net.port_peer, net.num_hosts,
            net.host_switch, net.host_port, net.host_ip)
    B.pv_load_flow_tables_begin(ctx, *args)
    kept = B._TABLE_LOADS[ctx.value]
    assert kept[0].dtype == np.uint32 and kept[0].ctypes.data == seen["ptrs"][0]
    assert (kept[0] == net.rule_offs).all()
    B.pv_load_flow_tables_end(ctx)
    assert ctx.value not in B._TABLE_LOADS

    fake.end_rc = B.PV_EINVAL
    B.pv_load_flow_tables_begin(ctx, *args)
    with pytest.raises(B.PVError) as e:
        B.pv_load_flow_tables_end(ctx)
    assert e.value.code == B.PV_EINVAL and ctx.value not in B._TABLE_LOADS

    B.pv_load_flow_tables_begin(ctx, *args)
    B.pv_destroy(ctx)
    assert ctx.value not in B._TABLE_LOADS
