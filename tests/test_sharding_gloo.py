"""The multi-rank path on CPU: intent-range sharding is exact (gloo ranks
each run the oracle pipeline on their own range; the concatenation equals
the unsharded run), the ranges partition the batch, and the host-side
reductions the benchmark uses behave: the max over ranks of the timed
region, and the sums over ranks of the per-status counters and verdict
counts, which equal the unsharded run's (a batch in which intents pass)."""
import os
import socket

import numpy as np
import pytest
import torch.multiprocessing as mp

import oracle
from paper_2602_16100_gb300 import sharding as SH
from paper_2602_16100_gb300 import workloads as W


def _batch():
    return W.end_to_end(seed=31, num_switches=48, num_intents=37, probes_per_intent=40, rules_per_switch=120,
                        hop_cap=16, pass_share=0.3)


def _pipeline(e):
    c = e.cluster
    bits, flags = oracle.eval_selectors(c.num_nodes, c.num_keys, c.labels, e.intents.expr_offs, e.intents.exprs)
    assign = oracle.place_pods(bits, c.num_nodes, e.pods_per_intent, e.place_draws)
    probes = oracle.bind_probes(e.probes.probes, e.probes_per_intent, e.pods_per_intent, assign, e.network.host_ip)
    res = oracle.verify_probes(e.network, probes, e.probes.hop_cap)
    passed, counts = oracle.aggregate(bits, c.num_nodes, flags, assign, e.pods_per_intent, res, e.probes_per_intent)
    return {"bits": bits, "flags": flags, "assign": assign, "probes": probes, "results": res, "pass": passed,
            "counts": counts}


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, outdir):
    import torch.distributed as dist
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world),
                      LOCAL_RANK=str(rank))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        r, w, _ = SH.world_info()
        assert (r, w) == (rank, world)
        part = _pipeline(SH.shard_end_to_end(_batch(), r, w))
        np.savez(os.path.join(outdir, f"rank{r}.npz"), **part)
        m = SH.max_over_ranks(10.0 + r, dist)
        s = SH.sum_over_ranks(int(part["pass"].sum()), dist)
        np.save(os.path.join(outdir, f"agg{r}.npy"), np.array([m, s], np.float64))
        # per-status histogram of the rank's probes, the per-intent counter
        # columns and the verdict count, summed over ranks
        local = np.concatenate([np.bincount(part["results"]["status"], minlength=6),
                                part["counts"].astype(np.int64).sum(axis=0), [int(part["pass"].sum())]])
        np.save(os.path.join(outdir, f"sums{r}.npy"), SH.sum_vector_over_ranks(local, dist))
        dist.barrier()
    finally:
        dist.destroy_process_group()


@pytest.mark.parametrize("world", [2, 3])
def test_sharded_pipeline_equals_unsharded(tmp_path, world):
    mp.start_processes(_rank_main, args=(world, _free_port(), str(tmp_path)), nprocs=world, join=True,
                       start_method="spawn")
    whole = _pipeline(_batch())
    parts = [dict(np.load(tmp_path / f"rank{r}.npz")) for r in range(world)]
    for k in ("bits", "flags", "assign", "probes", "results", "pass", "counts"):
        got = np.concatenate([p[k] for p in parts])
        assert (got == whole[k]).all(), k
    want = np.concatenate([np.bincount(whole["results"]["status"], minlength=6),
                           whole["counts"].astype(np.int64).sum(axis=0), [int(whole["pass"].sum())]])
    assert whole["pass"].sum() > 0
    for r in range(world):
        m, s = np.load(tmp_path / f"agg{r}.npy")
        assert m == 10.0 + world - 1 and s == int(whole["pass"].sum())
        assert (np.load(tmp_path / f"sums{r}.npy") == want).all()


def test_shard_ranges_partition():
    for n in (0, 1, 5, 37, 10_000):
        for world in (1, 2, 3, 8):
            cov = []
            for r in range(world):
                lo, hi = SH.shard_range(n, r, world)
                assert 0 <= lo <= hi <= n
                cov += list(range(lo, hi))
            assert cov == list(range(n))
            lens = [SH.shard_range(n, r, world)[1] - SH.shard_range(n, r, world)[0] for r in range(world)]
            assert max(lens) - min(lens) <= 1
    with pytest.raises(ValueError):
        SH.shard_range(4, 2, 2)
    assert len({SH.shard_seed(7, r) for r in range(8)}) == 8 and SH.shard_seed(7, 0) == 7


def test_single_process_reductions_are_identity():
    assert SH.max_over_ranks(3.5) == 3.5 and SH.sum_over_ranks(4) == 4
    assert (SH.sum_vector_over_ranks([1, 2, 3]) == [1, 2, 3]).all()
