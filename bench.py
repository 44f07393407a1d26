#!/usr/bin/env python3
"""Benchmark of the GB300 privacy-intent validator.

Default workload: the end-to-end cross-layer configuration (10,000 intents on
1,024 nodes x 32 label keys attached to a 512-switch random graph with 1,000
rules per switch; per intent a node-selector conjunction, a region mask, 4
pods placed by seeded choice among feasible nodes and 5,000 probes; 50M
probes, hop cap 32).  One step = selector rows -> placement -> probe binding
-> hop-synchronous walks -> per-intent verdicts, all in libpv's kernels.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]
                  [--workload e2e|e2e_policies|placement|placement_terms|placement_replicas|flow|wan|schedule]
                  [--no-extra-configs] [--no-cpu-baseline]

Prints one JSON line (rank 0).  `value` is device-timed throughput with the
inputs resident in HBM (CUDA events on the launching stream, K steps after W
warm-ups, max over ranks); `e2e` is the same metric through the public API
from pinned host buffers (loads, host->device copies, the step and the
device->host read of the verdicts inside the timed region).  `kernels` and
`roofline` come from a second pass of the same K steps under the library's
CUDA-event profiler, so its events stay out of the timed region.  With the
default workload, `configs` holds the other configurations of the metric
(placement-scale, flow-verification, continuum WAN), each measured the same
way on its own device-resident batch with its own roofline and CPU baseline
(`--no-extra-configs` leaves them out).  Under torchrun each rank processes
its own shard (seed offset by rank): weak scaling, no collective on the data
path; after the timed regions the per-status counters and verdict counts are
summed over ranks (`summed_over_ranks`).  `--impl reference` times the CPU
oracle on a bounded sample of the same workload.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import statistics
import subprocess
import sys
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

from paper_2602_16100_gb300 import workloads as W  # noqa: E402

METRIC = "probe-hop verifications/s and pod×node selector evals/s; % of HBM peak"
HBM_FALLBACK_GBS = 6800.0


# ----------------------------------------------------------------------------
# environment helpers
# ----------------------------------------------------------------------------
def hbm_peak():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(p) as f:
            return float(json.load(f)["hbm_gbs"]), "measured"
    except Exception:
        return HBM_FALLBACK_GBS, "fallback"


class ClockSampler:
    """nvidia-smi clock / throttle-reason samples during the timed region."""
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index):
        self.gpu_index = gpu_index
        self.proc = None

    def __enter__(self):
        try:
            cmd = ["nvidia-smi", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits", "-lms", "200"]
            if self.gpu_index is not None:
                cmd += ["-i", str(self.gpu_index)]
            self.proc = subprocess.Popen(cmd, stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except Exception:
            self.proc = None
        return self

    def __exit__(self, *exc):
        self.result = None
        if self.proc is None:
            return
        time.sleep(0.25)
        self.proc.terminate()
        try:
            out, _ = self.proc.communicate(timeout=5)
        except Exception:
            self.proc.kill()
            out = ""
        sm, mx, reasons = [], [], set()
        names = ("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap")
        for line in out.strip().splitlines():
            f = [x.strip() for x in line.split(",")]
            if len(f) < 9:
                continue
            try:
                sm.append(float(f[1]))
                mx.append(float(f[2]))
            except ValueError:
                continue
            for n, val in zip(names, f[5:9]):
                if val.lower().startswith("active"):
                    reasons.add(n)
        if sm:
            self.result = {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(mx), "reasons": sorted(reasons),
                           "samples": len(sm)}


def source_hash(*names):
    h = hashlib.sha256()
    for n in names:
        with open(os.path.join(ROOT, "paper_2602_16100_gb300", "csrc", n), "rb") as f:
            h.update(f.read())
    return h.hexdigest()[:16]


def committed_traffic(kernel: str, src_hash: str):
    """DRAM bytes per unit from the committed ncu summary, if it was taken on
    the current kernel source (else None)."""
    p = os.path.join(ROOT, "profiles", "traffic.json")
    try:
        with open(p) as f:
            d = json.load(f)[kernel]
        return float(d["dram_bytes_per_unit"]) if d.get("source_hash") == src_hash else None
    except Exception:
        return None


def walk_statistics(v):
    """Counters of the last walk run with PV_OPT_WALK_STATS: first matches,
    index rule tests and interval lookups (the work the indexed kernels do),
    the depth a scan in first-match order reaches (the work a linear scan
    does), and index/scan disagreements (0)."""
    from paper_2602_16100_gb300 import binding as B
    g = lambda k: int(B.pv_get_stat(v.ctx, k))
    fm = g(B.PV_STAT_WALK_FIRST_MATCHES)
    d = {"first_matches": fm, "index_rule_tests": g(B.PV_STAT_WALK_RULE_TESTS),
         "interval_lookups": g(B.PV_STAT_WALK_INTERVAL_LOOKUPS), "scan_depth": g(B.PV_STAT_WALK_SCAN_DEPTH),
         "index_mismatches": g(B.PV_STAT_WALK_INDEX_MISMATCHES)}
    n = max(fm, 1)
    d.update({"index_rule_tests_per_first_match": d["index_rule_tests"] / n,
              "interval_lookups_per_first_match": d["interval_lookups"] / n,
              "scan_rules_per_first_match": d["scan_depth"] / n})
    return d


def _walk_entries(v):
    """Probe-hop entries the hop kernel processed in the last walk (the sum
    over hops of the live probes; a probe judged at a hand-off is counted in
    its result's hops but never entered at the next switch)."""
    from paper_2602_16100_gb300 import binding as B
    return int(B.pv_get_stat(v.ctx, B.PV_STAT_WALK_LIVE_TOTAL))


# ----------------------------------------------------------------------------
# workloads
# ----------------------------------------------------------------------------
INPUT_KEYS = ("offs", "exprs", "draws", "masks", "dst", "dport")   # host-buffer step inputs


class EndToEndBench:
    name = "end-to-end cross-layer"
    unit = "probe-hop verifications/s"
    walks = True

    def __init__(self, seed, intents=None, policies=False):
        self.e = W.end_to_end(seed=20260220 + seed, **({"num_intents": intents} if intents else {}))
        # path constraints (forbidden switches, waypoints), one policy per intent
        self.pol = W.path_policies(20260221 + seed, self.e.network, self.e.intents.num_pods) if policies else None
        if policies:
            self.name = "end-to-end cross-layer with path constraints"

    def config(self):
        e = self.e
        return {"workload": self.name, "intents": e.intents.num_pods, "nodes": e.cluster.num_nodes,
                "label_keys": e.cluster.num_keys, "switches": e.network.num_switches,
                "rules_per_switch": int(np.diff(e.network.rule_offs).max()), "pods_per_intent": e.pods_per_intent,
                "probes": len(e.probes.probes), "hop_cap": e.probes.hop_cap,
                "l2": "inputs larger than L2 (300 MB of flow columns in, a 16-byte walk record built per listed flow, 200 MB of results per step)",
                **({"path_policies": self.pol.num_policies, "forbidden_switches": len(self.pol.forbid),
                    "waypoints": len(self.pol.must)} if self.pol is not None else {})}

    def setup(self, v):
        self.v = v
        v.load_cluster(self.e.cluster)
        v.load_network(self.e.network)
        if self.pol is not None:
            v.load_policies(self.pol)
        self.dev, self.sizes = v.alloc_end_to_end(self.e, with_policies=self.pol is not None)

    def step(self, stream):
        self.v.run_end_to_end(self.dev, self.sizes, stream)

    def measure_units(self):
        import torch
        res = self.dev["results"].view(-1, 4)
        self.probe_hops = int(res[:, 1].to(torch.int64).sum().item())
        self.selector_evals = self.e.intents.num_pods * self.e.cluster.num_nodes
        self.status_hist = torch.bincount(res[:, 0].to(torch.int64), minlength=6).tolist()
        self.pass_count = int(self.dev["pass"][: self.e.intents.num_pods].to(torch.int64).sum().item())
        self.hop_entries = _walk_entries(self.v)
        return self.probe_hops

    def extra(self, secs_per_step):
        return {"selector_evals_per_s": self.selector_evals / secs_per_step,
                "probe_hops_per_step": self.probe_hops, "hop_kernel_entries_per_step": self.hop_entries,
                "status_histogram": dict(zip(W.STATUS_NAMES, self.status_hist)),
                "intents_passed": self.pass_count}

    def counters(self):
        return (list(W.STATUS_NAMES) + ["probe_hops", "intents_passed"],
                list(self.status_hist) + [self.probe_hops, self.pass_count])

    def release(self):
        """Drop the batch's device and pinned host buffers."""
        for k in ("dev", "host"):
            if hasattr(self, k):
                delattr(self, k)

    def algorithmic_bytes(self, group):
        e = self.e
        I = e.intents.num_pods
        M = len(e.probes.probes)
        if group == "walk_hop":         # per hop entry: 16 B probe record read + 4 B result / state written
            return 20 * self.hop_entries
        if group == "walk_regroup":     # per hop entry: 8 B state read + 8 B state written
            return 16 * self.hop_entries
        if group == "selector":
            return I * W.words_per_row(e.cluster.num_nodes) * 4 + len(e.intents.exprs) * 20 + I * 5
        if group == "bind":
            return M * 16 * 2
        if group == "aggregate":
            return M * 4 + I * 33
        if group == "walk_init":
            return M * 16
        return 0

    def traffic_unit(self, group):
        return self.hop_entries if group in ("walk_hop", "walk_regroup") else None

    # host-buffer end-to-end step through the public API
    def setup_e2e(self, v, chunks=1):
        import torch
        e = self.e
        pin = lambda a: torch.from_numpy(np.ascontiguousarray(a).view(np.uint8).reshape(-1).copy()).pin_memory()
        from paper_2602_16100_gb300.validator import flow_columns_of
        dst, dport = flow_columns_of(e)
        self.host = {"offs": pin(e.intents.expr_offs.astype(np.uint32)), "exprs": pin(e.intents.exprs),
                     "draws": pin(e.place_draws.astype(np.uint64)), "masks": pin(e.intent_mask.astype(np.uint32)),
                     "dst": pin(dst), "dport": pin(dport),
                     "pass": torch.empty(e.intents.num_pods, dtype=torch.uint8).pin_memory(),
                     "counts": torch.empty(e.intents.num_pods * 32, dtype=torch.uint8).pin_memory()}
        self.copy_stream = torch.cuda.Stream()
        self.chunks = chunks
        self.loads_first = getattr(self, "loads_first", True)
        net = e.network
        self.h2d = (sum(self.host[k].numel() for k in INPUT_KEYS)
                    + e.cluster.labels.nbytes + net.rule_offs.nbytes + net.rules.nbytes + net.switch_region.nbytes
                    + net.port_offs.nbytes + net.port_peer.nbytes + net.host_switch.nbytes + net.host_port.nbytes
                    + net.host_ip.nbytes)
        self.d2h = self.host["pass"].numel() + self.host["counts"].numel()

    def step_e2e(self, v, stream):
        """Every input from host memory: intents (selectors, placement draws,
        masks) and their flows copied (8 B per flow), the cluster labels and
        flow tables loaded meanwhile (the table load in two halves around
        the queued uploads), verification of `chunks` intent ranges as their
        flows arrive, verdicts and counters copied back."""
        e = self.e

        def loads():
            v.load_cluster(e.cluster)
            if self.pol is not None:   # checked against the installed tables: the same network every step
                v.load_policies(self.pol)
            v.begin_network(e.network)
            return v.finish_network

        v.run_end_to_end_from_host(self.host, self.dev, self.sizes, stream, self.copy_stream, self.chunks, loads,
                                   self.loads_first)

    def e2e_phases(self, v, stream, reps=3):
        """Each part of the host-buffer step alone (diagnostic, after the
        timed region): the two table loads, the input upload, the device
        pipeline on resident inputs."""
        import torch
        e = self.e
        torch.cuda.synchronize()
        t0 = time.perf_counter()
        for _ in range(reps):
            v.load_cluster(e.cluster)
            v.load_network(e.network)
            if self.pol is not None:
                v.load_policies(self.pol)
        torch.cuda.synchronize()
        load = (time.perf_counter() - t0) / reps
        t0 = time.perf_counter()
        for _ in range(reps):
            with torch.cuda.stream(self.copy_stream):
                for k in INPUT_KEYS:
                    self.dev[k][: self.host[k].numel()].copy_(self.host[k], non_blocking=True)
        torch.cuda.synchronize()
        upload = (time.perf_counter() - t0) / reps
        t0 = time.perf_counter()
        for _ in range(reps):
            self.v.run_end_to_end(self.dev, self.sizes, stream)
        torch.cuda.synchronize()
        dev = (time.perf_counter() - t0) / reps
        up_bytes = sum(self.host[k].numel() for k in INPUT_KEYS)
        return {"load_tables_ms": load * 1e3, "upload_inputs_ms": upload * 1e3,
                "upload_gbs": up_bytes / upload / 1e9, "device_pipeline_ms": dev * 1e3}

    # oracle on a bounded sample: the first n intents, whole pipeline
    def oracle_sample(self, n_intents):
        import oracle
        e = self.e
        c = e.cluster
        ppg, pods = e.probes_per_intent, e.pods_per_intent
        offs = e.intents.expr_offs[: n_intents + 1].astype(np.uint32)
        exprs = e.intents.exprs[: int(offs[-1])]
        t0 = time.perf_counter()
        bits, flags = oracle.eval_selectors(c.num_nodes, c.num_keys, c.labels, offs, exprs)
        assign = oracle.place_pods(bits, c.num_nodes, pods, e.place_draws[: n_intents * pods])
        probes = oracle.bind_probes(e.probes.probes[: n_intents * ppg], ppg, pods, assign, e.network.host_ip)
        if self.pol is None:
            res = oracle.verify_probes(e.network, probes, e.probes.hop_cap)
            oracle.aggregate(bits, c.num_nodes, flags, assign, pods, res, ppg)
        else:
            res, hits = oracle.verify_constrained(e.network, probes, e.probes.hop_cap, self.pol, probes_per_policy=ppg)
            oracle.aggregate_constrained(bits, c.num_nodes, flags, assign, pods, res, ppg, hits, self.pol)
        dt = time.perf_counter() - t0
        units = int(res["hops"].astype(np.int64).sum())
        return units, dt, f"first {n_intents} intents ({n_intents * ppg} probes), whole pipeline"

    oracle_start = 2

    def oracle_max(self):
        return self.e.intents.num_pods


class PlacementBench:
    name = "placement-scale"
    unit = "pod×node selector evals/s"

    def __init__(self, seed):
        d = W.selector_workload(seed=20260217 + seed)
        self.c, self.s = d["cluster"], d["selectors"]

    def config(self):
        return {"workload": self.name, "nodes": self.c.num_nodes, "label_keys": self.c.num_keys,
                "pods": self.s.num_pods, "expressions": len(self.s.exprs),
                "l2": "output bitsets (64 MB) rewritten each step; labels and value rows L2-resident"}

    def setup(self, v):
        from paper_2602_16100_gb300.validator import to_device, empty_device
        self.v = v
        v.load_cluster(self.c)
        d = v.device
        self.words = W.words_per_row(self.c.num_nodes)
        self.d_offs = to_device(self.s.expr_offs.astype(np.uint32), d)
        self.d_exprs = to_device(self.s.exprs, d)
        self.d_assign = to_device(self.s.assign.astype(np.uint32), d)
        self.d_bits = empty_device(self.s.num_pods * self.words * 4, d)
        self.d_flags = empty_device(self.s.num_pods, d)

    def step(self, stream):
        self.v.eval_selectors(self.d_offs, len(self.s.exprs), self.d_exprs, self.d_assign, self.s.num_pods,
                              words=self.words, d_bits=self.d_bits, d_flags=self.d_flags, stream=stream)

    def measure_units(self):
        return self.s.num_pods * self.c.num_nodes

    def extra(self, secs_per_step):
        return {}

    def algorithmic_bytes(self, group):
        if group != "selector":
            return 0
        P = self.s.num_pods
        return P * self.words * 4 + len(self.s.exprs) * 20 + P * 4 * 2 + P + self.c.labels.nbytes

    def traffic_unit(self, group):
        return self.s.num_pods if group == "selector" else None

    def oracle_sample(self, n):
        import oracle
        idx = np.arange(n)
        offs = self.s.expr_offs[: n + 1].astype(np.uint32)
        ex = self.s.exprs[: int(offs[-1])]
        t0 = time.perf_counter()
        oracle.eval_selectors(self.c.num_nodes, self.c.num_keys, self.c.labels, offs, ex, self.s.assign[idx])
        dt = time.perf_counter() - t0
        return n * self.c.num_nodes, dt, f"first {n} pods"

    oracle_start = 500

    def oracle_max(self):
        return self.s.num_pods


class ReplicasBench(PlacementBench):
    """Placement scale with repeated selectors (100,000 pods drawing their
    expression lists from 10,000 by Zipf popularity, as replicas of
    deployments do), evaluated with PV_OPT_SELECTOR_DEDUPE; the same step
    without it is reported beside."""
    name = "placement-scale, repeated selectors"

    def __init__(self, seed):
        d = W.selector_replicas(seed=20260226 + seed)
        self.c, self.s = d["cluster"], d["selectors"]
        self.distinct = int(len(np.unique(d["pick"])))

    def config(self):
        return {**super().config(), "distinct_lists": self.distinct, "dedupe": True}

    def setup(self, v):
        from paper_2602_16100_gb300 import binding as B
        super().setup(v)
        B.pv_set_option(v.ctx, B.PV_OPT_SELECTOR_DEDUPE, 1)

    def extra(self, secs_per_step):
        import torch
        from paper_2602_16100_gb300 import binding as B
        B.pv_set_option(self.v.ctx, B.PV_OPT_SELECTOR_DEDUPE, 0)
        stream = torch.cuda.current_stream()
        for _ in range(3):
            self.step(stream)
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record(stream)
        for _ in range(10):
            self.step(stream)
        b.record(stream)
        torch.cuda.synchronize()
        B.pv_set_option(self.v.ctx, B.PV_OPT_SELECTOR_DEDUPE, 1)
        return {"ms_per_step_without_dedupe": a.elapsed_time(b) / 10}


class PlacementTermsBench:
    name = "placement-scale, multi-term node affinity"
    unit = "pod×node selector evals/s"

    def __init__(self, seed):
        d = W.selector_terms(seed=20260222 + seed)
        self.c, self.t = d["cluster"], d["terms"]

    def config(self):
        return {"workload": self.name, "nodes": self.c.num_nodes, "label_keys": self.c.num_keys,
                "pods": self.t.num_pods, "terms": len(self.t.term_offs) - 1, "expressions": len(self.t.exprs),
                "l2": "output bitsets (64 MB) rewritten each step; labels and value rows L2-resident"}

    def setup(self, v):
        from paper_2602_16100_gb300.validator import to_device, empty_device
        self.v = v
        v.load_cluster(self.c)
        d = v.device
        self.words = W.words_per_row(self.c.num_nodes)
        self.d_pt = to_device(self.t.pod_terms.astype(np.uint32), d)
        self.d_to = to_device(self.t.term_offs.astype(np.uint32), d)
        self.d_exprs = to_device(self.t.exprs, d)
        self.d_assign = to_device(self.t.assign.astype(np.uint32), d)
        self.d_bits = empty_device(self.t.num_pods * self.words * 4, d)
        self.d_flags = empty_device(self.t.num_pods, d)

    def step(self, stream):
        from paper_2602_16100_gb300 import binding as B
        B.pv_eval_selector_terms(self.v.ctx, self.t.num_pods, self.d_pt, len(self.t.term_offs) - 1, self.d_to,
                                 len(self.t.exprs), self.d_exprs, self.d_assign, self.d_bits, self.words,
                                 self.d_flags, stream)

    def measure_units(self):
        return self.t.num_pods * self.c.num_nodes

    def extra(self, secs_per_step):
        return {}

    def algorithmic_bytes(self, group):
        if group != "selector":
            return 0
        P, T = self.t.num_pods, len(self.t.term_offs) - 1
        return P * self.words * 4 + len(self.t.exprs) * 20 + T * 4 + P * 4 * 2 + P + self.c.labels.nbytes

    def traffic_unit(self, group):
        return self.t.num_pods if group == "selector" else None

    def oracle_sample(self, n):
        import oracle
        pt = self.t.pod_terms[: n + 1].astype(np.uint32)
        to = self.t.term_offs[: int(pt[-1]) + 1].astype(np.uint32)
        ex = self.t.exprs[: int(to[-1])]
        t0 = time.perf_counter()
        oracle.eval_selector_terms(self.c.num_nodes, self.c.num_keys, self.c.labels, pt, to, ex, self.t.assign[:n])
        dt = time.perf_counter() - t0
        return n * self.c.num_nodes, dt, f"first {n} pods"

    oracle_start = 500

    def oracle_max(self):
        return self.t.num_pods


class ScheduleBench:
    name = "path scheduling on the end-to-end network"
    unit = "scheduled paths/s"
    max_len = 64

    def __init__(self, seed):
        e = W.end_to_end(seed=20260220 + seed, num_intents=8, probes_per_intent=1)
        self.net = e.network
        self.pol = W.path_policies(20260223 + seed, self.net, 10_000)
        self.req = W.path_requests(20260224 + seed, self.net, 10_000, num_policies=10_000, extra_regions=(6, 14))
        self.weights = W.Stream(20260225 + seed, "link-weights").ints(1, 16, int(self.net.port_offs[-1])).astype(
            np.uint16)

    def config(self):
        return {"workload": self.name, "switches": self.net.num_switches, "requests": len(self.req),
                "path_policies": self.pol.num_policies, "waypoints": len(self.pol.must),
                "forbidden_switches": len(self.pol.forbid), "max_len": self.max_len, "weights": "U[1,16] per link",
                "l2": "working set L2-resident (small graph); every step recomputes all paths and rules"}

    def setup(self, v):
        from paper_2602_16100_gb300.validator import to_device, empty_device
        self.v = v
        v.load_network(self.net)
        v.load_policies(self.pol)
        d = v.device
        R, L = len(self.req), self.max_len
        self.d_req = to_device(self.req, d)
        self.d_w = to_device(self.weights, d)
        self.d_vis = empty_device(R * L * 4, d)
        self.d_len = empty_device(R, d)
        self.d_st = empty_device(R, d)
        self.d_rules = empty_device(R * L * W.RULE_DTYPE.itemsize, d)
        self.d_rsw = empty_device(R * L * 2, d)

    def step(self, stream):
        from paper_2602_16100_gb300 import binding as B
        R, L = len(self.req), self.max_len
        B.pv_schedule_paths(self.v.ctx, R, self.d_req, self.d_w, L, self.d_vis, self.d_len, self.d_st, stream)
        B.pv_compile_path_rules(self.v.ctx, R, self.d_req, L, self.d_vis, self.d_len, self.d_st, 65535,
                                self.d_rules, self.d_rsw, stream)

    def measure_units(self):
        import torch
        st = self.d_st.to(torch.int64)
        self.hist = torch.bincount(st, minlength=5).tolist()
        self.mean_len = float(self.d_len.to(torch.float64).sum().item()) / max(1, self.hist[0])
        return len(self.req)

    def extra(self, secs_per_step):
        return {"status_histogram": dict(zip(("ok", "nosrc", "blocked", "too_long", "repeat"), self.hist)),
                "mean_visits_of_ok_paths": self.mean_len}

    def algorithmic_bytes(self, group):
        if group != "schedule":
            return 0
        R, L = len(self.req), self.max_len
        # requests in, visits / lengths / statuses out, rules and their switches out
        return R * (16 + 2) + int(self.hist[0] * self.mean_len) * 4 + R * L * (W.RULE_DTYPE.itemsize + 2)

    def traffic_unit(self, group):
        return None

    def oracle_sample(self, n):
        import oracle
        t0 = time.perf_counter()
        hops, ln, st = oracle.schedule_paths(self.net, self.req[:n], self.pol, self.weights, self.max_len)
        oracle.compile_path_rules(self.net, self.req[:n], hops, ln, st)
        return n, time.perf_counter() - t0, f"first {n} requests"

    oracle_start = 50

    def oracle_max(self):
        return len(self.req)


class FlowBench:
    name = "flow-verification"
    unit = "probe-hop verifications/s"
    walks = True

    def __init__(self, seed):
        d = W.fat_tree(seed=20260218 + seed)
        self.net, self.p = d["network"], d["probes"]

    def config(self):
        return {"workload": self.name, "switches": self.net.num_switches, "hosts": self.net.num_hosts,
                "rules_per_switch": int(np.diff(self.net.rule_offs).max()), "probes": len(self.p.probes),
                "hop_cap": self.p.hop_cap, "l2": "inputs larger than L2 (160 MB probes, 40 MB results)"}

    def setup(self, v):
        from paper_2602_16100_gb300.validator import to_device, empty_device
        self.v = v
        v.load_network(self.net)
        self.d_probes = to_device(self.p.probes, v.device)
        self.d_out = empty_device(len(self.p.probes) * 4, v.device)

    def step(self, stream):
        self.v.verify_probes(self.d_probes, len(self.p.probes), self.p.hop_cap, d_out=self.d_out, stream=stream)

    def measure_units(self):
        import torch
        res = self.d_out.view(-1, 4)
        self.probe_hops = int(res[:, 1].to(torch.int64).sum().item())
        self.hist = torch.bincount(res[:, 0].to(torch.int64), minlength=6).tolist()
        self.hop_entries = _walk_entries(self.v)
        return self.probe_hops

    def extra(self, secs_per_step):
        return {"probe_hops_per_step": self.probe_hops, "hop_kernel_entries_per_step": self.hop_entries,
                "status_histogram": dict(zip(W.STATUS_NAMES, self.hist))}

    def counters(self):
        return list(W.STATUS_NAMES) + ["probe_hops"], list(self.hist) + [self.probe_hops]

    def release(self):
        for k in ("d_probes", "d_out"):
            if hasattr(self, k):
                delattr(self, k)

    def algorithmic_bytes(self, group):
        return {"walk_hop": 20, "walk_regroup": 16}.get(group, 0) * self.hop_entries + \
            (len(self.p.probes) * 16 if group == "walk_init" else 0)

    def traffic_unit(self, group):
        return self.hop_entries if group in ("walk_hop", "walk_regroup") else None

    def oracle_sample(self, n):
        import oracle
        idx = np.arange(n, dtype=np.uint32)
        t0 = time.perf_counter()
        r = oracle.verify_probes(self.net, self.p.probes, self.p.hop_cap, idx=idx)
        dt = time.perf_counter() - t0
        return int(r["hops"].astype(np.int64).sum()), dt, f"first {n} probes"

    oracle_start = 2000

    def oracle_max(self):
        return len(self.p.probes)


class WanBench:
    name = "continuum WAN"
    unit = "compliant-reach (mask, source) rows/s"

    def __init__(self, seed):
        self.q = W.continuum_wan(seed=20260219 + seed)

    def config(self):
        g = self.q.graph
        return {"workload": self.name, "vertices": g.num_vertices, "edges": len(g.cols),
                "masks": len(self.q.masks), "sources": len(self.q.sources),
                "l2": "output rows (128 MB) rewritten each step"}

    def setup(self, v):
        from paper_2602_16100_gb300.validator import to_device, empty_device
        self.v = v
        d = v.device
        self.g = v.upload_graph(self.q.graph)
        self.d_src = to_device(self.q.sources.astype(np.uint32), d)
        self.d_masks = to_device(self.q.masks.astype(np.uint32), d)
        self.words = W.words_per_row(self.q.graph.num_vertices)
        self.d_out = empty_device(len(self.q.masks) * len(self.q.sources) * self.words * 4, d)

    def step(self, stream):
        self.v.compliant_reach(self.g, len(self.q.sources), self.d_src, len(self.q.masks), self.d_masks,
                               words=self.words, d_reach=self.d_out, stream=stream)

    def measure_units(self):
        return len(self.q.masks) * len(self.q.sources)

    def extra(self, secs_per_step):
        return {}

    def algorithmic_bytes(self, group):
        if group != "reach":
            return 0
        return len(self.q.masks) * len(self.q.sources) * self.words * 4 + len(self.q.graph.cols) * 4

    def traffic_unit(self, group):
        return len(self.q.masks) * len(self.q.sources) if group == "reach" else None

    def oracle_sample(self, n):
        import oracle
        m = len(self.q.masks)
        pairs = np.stack([np.arange(n) % m, np.arange(n) // m], 1).astype(np.uint32)
        t0 = time.perf_counter()
        oracle.compliant_reach(self.q.graph, self.q.sources, self.q.masks, pairs=pairs)
        return n, time.perf_counter() - t0, f"first {n} (mask, source) rows"

    oracle_start = 256

    def oracle_max(self):
        return len(self.q.masks) * len(self.q.sources)


WORKLOADS = {"e2e": EndToEndBench, "placement_terms": PlacementTermsBench, "schedule": ScheduleBench,
             "e2e_policies": lambda seed, **kw: EndToEndBench(seed, policies=True, **kw), "placement": PlacementBench, "flow": FlowBench, "wan": WanBench,
             "placement_replicas": ReplicasBench}
SOURCES = {"schedule": ("k_sched.cu",), "walk_hop": ("k_walk.cu",), "walk_regroup": ("k_walk.cu",), "selector": ("k_selector.cu",),
           "reach": ("k_reach.cu",)}


def timed_oracle(wl, target_s=12.0, cap_s=40.0):
    """Grow the sample until one run takes >= target_s seconds of CPU."""
    n = min(wl.oracle_start, wl.oracle_max())
    while True:
        units, dt, desc = wl.oracle_sample(n)
        if dt >= target_s or dt * 2 > cap_s or n >= wl.oracle_max():
            return units, dt, desc, n
        n = min(wl.oracle_max(), int(n * max(1.5, min(8.0, target_s / max(dt, 1e-3)))))


def cpu_model() -> str:
    """The host CPU's model name (x86: /proc/cpuinfo; Arm: lscpu)."""
    try:
        with open("/proc/cpuinfo") as f:
            for line in f:
                if line.lower().startswith("model name"):
                    return line.split(":", 1)[1].strip()
    except OSError:
        pass
    try:
        out = subprocess.run(["lscpu"], capture_output=True, text=True, timeout=10).stdout
        for line in out.splitlines():
            if line.strip().lower().startswith("model name"):
                return line.split(":", 1)[1].strip()
    except Exception:
        pass
    import platform
    return platform.processor() or platform.machine()


def cpu_baseline(wl, target_s):
    """The oracle, single-threaded as written, on a bounded sample."""
    u, dt, desc, _ = timed_oracle(wl, target_s=target_s, cap_s=max(40.0, 3 * target_s))
    return {"value": u / dt, "unit": wl.unit, "cores": 1, "host_cores": os.cpu_count(), "cpu_model": cpu_model(),
            "kind": "oracle", "sample": desc, "seconds": dt}


# ----------------------------------------------------------------------------
# arms
# ----------------------------------------------------------------------------
def run_reference(args):
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return 0
    wl = WORKLOADS[args.workload](0)
    # size one step to a few seconds of single-threaded CPU work (this also
    # serves as warm-up), then time K steps on that sample
    _, _, desc, n = timed_oracle(wl, target_s=3.0, cap_s=20.0)
    for _ in range(max(0, args.warmup - 1)):
        wl.oracle_sample(max(1, n // 8))
    tot_units, tot_s = 0, 0.0
    for _ in range(args.steps):
        u, d, desc = wl.oracle_sample(n)
        tot_units += u
        tot_s += d
    value = tot_units / tot_s
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": wl.unit, "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * tot_s / args.steps,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "u32",
            "data": "synthetic", "config": wl.config(),
            "cpu_baseline": {"value": value, "unit": wl.unit, "cores": 1, "host_cores": os.cpu_count(),
                             "cpu_model": cpu_model(), "kind": "oracle", "sample": desc},
            "e2e": {"value": value, "unit": wl.unit, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)
    return 0


def measure(wl, v, args, stream, barrier, dist, gpu_index):
    """One workload on the device: W warm-up steps, K steps timed with CUDA
    events on the launching stream (clocks sampled meanwhile), the same K
    steps once more under the library's CUDA-event profiler (per kernel
    group), and for walks one diagnostic step with the counting kernels.
    Returns the timing, the kernel groups and the dominant group's roofline."""
    import torch
    from paper_2602_16100_gb300 import binding as B
    from paper_2602_16100_gb300 import sharding as SH
    wl.setup(v)
    for _ in range(max(args.warmup, 1)):
        wl.step(stream)
    v.sync(stream)
    units = wl.measure_units()
    barrier()
    start, stop = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with ClockSampler(gpu_index) as clk:
        start.record(stream)
        for _ in range(args.steps):
            wl.step(stream)
        stop.record(stream)
        barrier()
    ms = start.elapsed_time(stop)
    v.sync(stream)
    # per-kernel-group breakdown: the same steps once more, bracketed by the
    # library's CUDA-event profiler (kept out of the timed region above)
    B.pv_profile_enable(v.ctx, True)
    p0, p1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    p0.record(stream)
    for _ in range(args.steps):
        wl.step(stream)
    p1.record(stream)
    B.pv_profile_collect(v.ctx, stream)
    barrier()
    B.pv_profile_enable(v.ctx, False)
    prof_ms = p0.elapsed_time(p1)
    v.sync(stream)
    # first-match statistics of one more step, run with the library's
    # counting kernels (a diagnostic pass, outside both timed regions)
    walk_stats = None
    if getattr(wl, "walks", False):
        B.pv_set_option(v.ctx, B.PV_OPT_WALK_STATS, 1)
        wl.step(stream)
        v.sync(stream)
        B.pv_set_option(v.ctx, B.PV_OPT_WALK_STATS, 0)
        walk_stats = walk_statistics(v)
    ms = SH.max_over_ranks(ms, dist, "cuda")
    secs_per_step = ms / 1e3 / args.steps
    kernels, launches = {}, 0
    for gi, name in enumerate(B.PV_K_NAMES):
        kms, n = B.pv_profile_read(v.ctx, gi)
        if n:
            kernels[name] = {"ms_per_step": kms / args.steps, "launches_per_step": n / args.steps,
                             "share_of_step": kms / prof_ms}
            launches += n
    dom = max(kernels, key=lambda k: kernels[k]["ms_per_step"]) if kernels else None
    peak, peak_kind = hbm_peak()
    roofline = None
    if dom:
        kd = kernels[dom]
        n_launch = kd["launches_per_step"]
        bytes_per_launch = wl.algorithmic_bytes(dom) / max(n_launch, 1)
        avg_launch_s = kd["ms_per_step"] / 1e3 / max(n_launch, 1)
        achieved = bytes_per_launch / avg_launch_s / 1e9 if avg_launch_s > 0 else 0.0
        tr_unit = committed_traffic(dom, source_hash(*SOURCES.get(dom, ("k_walk.cu",))))
        u = wl.traffic_unit(dom)
        traffic = tr_unit * u / max(n_launch, 1) if (tr_unit is not None and u) else None
        roofline = {"kernel": dom, "bound": "hbm", "achieved": achieved, "peak": peak, "unit": "GB/s",
                    "frac": achieved / peak, "peak_source": peak_kind, "traffic": traffic,
                    "algorithmic_bytes_per_launch": bytes_per_launch, "avg_launch_ms": avg_launch_s * 1e3}
    if walk_stats:
        walk_stats = dict(walk_stats)
        walk_stats["rule_tests_per_s"] = (walk_stats["index_rule_tests"] + walk_stats["interval_lookups"]) / \
            secs_per_step
        walk_stats["scan_equivalent_rules_per_s"] = walk_stats["scan_depth"] / secs_per_step
    return {"units": units, "ms": ms, "secs_per_step": secs_per_step, "kernels": kernels, "launches": launches,
            "roofline": roofline, "clocks": clk.result, "walk_statistics": walk_stats}


def sum_counters(wl, dist):
    """The per-status histogram, probe-hop count and verdict count of a
    rank's batch summed over all ranks (host bookkeeping after the timed
    regions; one all-reduce of a few integers)."""
    from paper_2602_16100_gb300 import sharding as SH
    if not hasattr(wl, "counters"):
        return {}
    names, vals = wl.counters()
    tot = SH.sum_vector_over_ranks(vals, dist, "cuda")
    return {"summed_over_ranks": dict(zip(names, (int(x) for x in tot)))}


EXTRA_CONFIGS = ("placement", "flow", "wan")   # measured beside the end-to-end headline


def run_ours(args):
    import torch
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    dist = None
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl")
    torch.cuda.set_device(local)
    from paper_2602_16100_gb300 import build
    from paper_2602_16100_gb300 import sharding as SH
    from paper_2602_16100_gb300.validator import Validator
    if rank == 0 or world == 1:
        build.build_library()
    if dist:
        dist.barrier()
    # weak scaling: every rank verifies its own batch of the same shape (the
    # units are independent; no collective on the data path)
    wl = WORKLOADS[args.workload](SH.shard_seed(0, rank), **({"intents": args.intents} if args.intents else {}))
    v = Validator(local)
    stream = torch.cuda.current_stream()

    def barrier():
        torch.cuda.synchronize()
        if dist:
            dist.barrier()
        torch.cuda.synchronize()

    vis = os.environ.get("CUDA_VISIBLE_DEVICES")
    gpu_index = vis.split(",")[local] if vis else local
    m = measure(wl, v, args, stream, barrier, dist, gpu_index)
    secs_per_step = m["secs_per_step"]
    value = m["units"] * world / secs_per_step
    sums = sum_counters(wl, dist)

    # end-to-end through the public API from pinned host buffers
    e2e = None
    if hasattr(wl, "setup_e2e"):
        wl.loads_first = args.e2e_loads_first
        wl.setup_e2e(v, args.e2e_chunks)
        for _ in range(max(args.warmup, 1)):
            wl.step_e2e(v, stream)
        barrier()
        t0 = time.perf_counter()
        for _ in range(args.steps):
            wl.step_e2e(v, stream)
        barrier()
        e_s = (time.perf_counter() - t0) / args.steps
        e_s = SH.max_over_ranks(e_s, dist, "cuda")
        e2e = {"value": m["units"] * world / e_s, "unit": wl.unit, "h2d_bytes_per_step": int(wl.h2d),
               "d2h_bytes_per_step": int(wl.d2h), "ms_per_step": e_s * 1e3, "upload_chunks": args.e2e_chunks,
               "loads": ("before the uploads" if args.e2e_loads_first
                         else "uploads of the tables queued first, the rest of the load while the inputs arrive")}
        if hasattr(wl, "e2e_phases"):
            e2e["phases"] = wl.e2e_phases(v, stream)
        wl.release()

    baseline_s = 12.0
    cpu = cpu_baseline(wl, baseline_s) if rank == 0 and world == 1 and not args.no_cpu_baseline else None

    # the other configurations of the metric, each timed the same way on its
    # own batch (one device-resident step each; the headline stays the
    # end-to-end line)
    configs = {}
    if args.workload == "e2e" and not args.no_extra_configs:
        for name in EXTRA_CONFIGS:
            xw = WORKLOADS[name](SH.shard_seed(0, rank))
            xm = measure(xw, v, args, stream, barrier, dist, gpu_index)
            entry = {"value": xm["units"] * world / xm["secs_per_step"], "unit": xw.unit,
                     "ms_per_step": xm["ms"] / args.steps, "config": xw.config(), "roofline": xm["roofline"],
                     "kernels": xm["kernels"], "gpu_launches": xm["launches"], "clocks": xm["clocks"],
                     **xw.extra(xm["secs_per_step"]), **sum_counters(xw, dist)}
            if xm["walk_statistics"]:
                entry["walk_statistics"] = xm["walk_statistics"]
            if rank == 0 and world == 1 and not args.no_cpu_baseline:
                entry["cpu_baseline"] = cpu_baseline(xw, 6.0)
            configs[xw.name] = entry
            if hasattr(xw, "release"):
                xw.release()

    if rank == 0:
        line = {"metric": METRIC, "value": value, "unit": wl.unit, "n_gpus": world, "steps": args.steps,
                "warmup": args.warmup, "ms_per_step": m["ms"] / args.steps, "higher_is_better": True,
                "scaling": "weak", "vs_baseline": None, "dtype": "u32", "data": "synthetic",
                "config": {**wl.config(), "parallelism": f"independent shards x{world}"},
                "roofline": m["roofline"], "cpu_baseline": cpu, "e2e": e2e, "gpu_launches": m["launches"],
                "clocks": m["clocks"], "kernels": m["kernels"], **wl.extra(secs_per_step), **sums}
        if m["walk_statistics"]:
            line["walk_statistics"] = m["walk_statistics"]
        if configs:
            line["configs"] = configs
        print(json.dumps(line), flush=True)
    v.close()
    if dist:
        dist.destroy_process_group()
    return 0


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=10)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", choices=("ours", "reference"), default="ours")
    ap.add_argument("--workload", choices=tuple(WORKLOADS), default="e2e")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-extra-configs", action="store_true",
                    help="end-to-end only: leave out the placement, flow-verification and WAN entries of `configs`")
    ap.add_argument("--e2e-chunks", type=int, default=1,
                    help="intent ranges whose probe upload overlaps verification in the host-buffer step")
    ap.add_argument("--e2e-loads-first", action="store_true",
                    help="host-buffer step: finish the table loads before queueing the input uploads "
                         "(default: the second half of the table load runs while the inputs arrive)")
    ap.add_argument("--intents", type=int, default=None,
                    help="end-to-end only: fewer intents (a smaller case for profiling, not a bench line)")
    args = ap.parse_args()
    if args.intents and not args.workload.startswith("e2e"):
        ap.error("--intents applies to the end-to-end workload only")
    if args.warmup < 3:
        print("note: warmup raised to 3", file=sys.stderr)
        args.warmup = 3
    return run_reference(args) if args.impl == "reference" else run_ours(args)


if __name__ == "__main__":
    sys.exit(main())
