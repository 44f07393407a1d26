"""GPU check of the compliant-reach entry point that allocates nothing.

Some callers cannot allocate device memory: their device memory belongs to
another framework's pool or is held to a fixed budget, or they cannot absorb
the device-wide synchronisation that cudaMalloc / cudaFree may imply.  For
them the library offers pv_compliant_reach_noalloc, which needs no context and
works in one static device array.  This test calls it through the C ABI twice
in a row (on different inputs, so the second call must not see leftovers of
the first) and compares each result with the regular pv_compliant_reach
bit for bit and with the CPU oracle, gives the oracle's rows for a CSR with
overlapping rows (malformed offsets: no edges) without writing past its
array, and checks that oversized inputs are refused.  The file is named to
be collected last.
"""
import numpy as np
import pytest

import oracle
from paper_2602_16100_gb300 import binding as B
from paper_2602_16100_gb300 import workloads as W
from paper_2602_16100_gb300.validator import empty_device, to_device, to_numpy

pytestmark = pytest.mark.gpu


def _inputs(v, g, src, masks):
    d = v.device
    return dict(V=g.num_vertices, offs=to_device(g.offs.astype(np.uint32), d), E=len(g.cols),
                cols=to_device(g.cols.astype(np.uint32), d), region=to_device(g.region.astype(np.uint8), d),
                src=to_device(src.astype(np.uint32), d), masks=to_device(masks.astype(np.uint32), d),
                words=W.words_per_row(g.num_vertices), ns=len(src), nm=len(masks))


def _regular(v, x):
    out = empty_device(x["nm"] * x["ns"] * x["words"] * 4, v.device)
    B.pv_compliant_reach(v.ctx, x["V"], x["offs"], x["E"], x["cols"], x["region"], x["ns"], x["src"], x["nm"],
                         x["masks"], out, x["words"])
    v.sync()
    return to_numpy(out, np.uint32)


def _noalloc(v, x):
    out = empty_device(x["nm"] * x["ns"] * x["words"] * 4, v.device)
    B.pv_compliant_reach_noalloc(x["V"], x["offs"], x["E"], x["cols"], x["region"], x["ns"], x["src"], x["nm"],
                                 x["masks"], out, x["words"])
    v.sync()
    return to_numpy(out, np.uint32)


def test_noalloc_reach_matches_regular_call_twice(validator):
    first = W.continuum_wan(seed=31, num_vertices=3000, num_masks=7, num_regions=16, mask_pop=(3, 10),
                            num_sources=200)
    second = W.random_digraph(32, 1500, 9000, num_regions=6)
    st = W.Stream(33, "noalloc")
    src2 = st.ints(0, 1499, 130).astype(np.uint32)
    masks2 = (st.u64(5) % np.uint64(64)).astype(np.uint32)
    for g, src, masks in ((first.graph, first.sources, first.masks), (second, src2, masks2)):
        x = _inputs(validator, g, src, masks)
        want = _regular(validator, x)
        got = _noalloc(validator, x)
        assert (got == want).all()
        assert want.any()
        assert (got == oracle.compliant_reach(g, src, masks).reshape(-1)).all()


def test_noalloc_reach_overlapping_offsets_read_as_no_edges(validator):
    V, E = 64, 300
    g0 = W.random_digraph(36, V, E)
    offs = np.where(np.arange(V + 1) % 2 == 0, 0, E).astype(np.uint32)   # rows overlap; total >> E
    bad = W.Graph(V, offs, g0.cols, g0.region)
    src = np.arange(V, dtype=np.uint32)
    masks = np.array([0xFFFFFFFF, 0b1011], np.uint32)
    got = _noalloc(validator, _inputs(validator, bad, src, masks))
    assert (got == oracle.compliant_reach(bad, src, masks).reshape(-1)).all()
    # the next call on a well-formed graph is not affected
    x = _inputs(validator, g0, src, masks)
    assert (_noalloc(validator, x) == oracle.compliant_reach(g0, src, masks).reshape(-1)).all()


def test_noalloc_reach_rejects_oversized_inputs(validator):
    g = W.random_digraph(34, 64, 200)
    x = _inputs(validator, g, np.arange(8, dtype=np.uint32), np.array([0xFFFFFFFF], np.uint32))
    out = empty_device(64 * 4 * 8, validator.device)
    for V, E in ((16385, x["E"]), (x["V"], 262145)):
        with pytest.raises(B.PVError) as err:
            B.pv_compliant_reach_noalloc(V, x["offs"], E, x["cols"], x["region"], x["ns"], x["src"], x["nm"],
                                         x["masks"], out, W.words_per_row(V))
        assert err.value.code == B.PV_EINVAL
