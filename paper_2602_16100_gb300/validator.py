"""User-facing wrapper over the C ABI: owns a pv_ctx, moves numpy arrays to
device byte tensors and back, and chains the end-to-end pipeline.

Every computation runs in libpv's CUDA kernels; this module only allocates
torch device buffers, copies, and calls the binding.
"""
from __future__ import annotations

from typing import Optional

import numpy as np
import torch

from . import binding as B
from . import workloads as W


def to_device(a: np.ndarray, device) -> torch.Tensor:
    """Byte tensor on `device` holding the bytes of the numpy array."""
    a = np.ascontiguousarray(a)
    return torch.from_numpy(a.view(np.uint8).reshape(-1).copy()).to(device)


def empty_device(nbytes: int, device) -> torch.Tensor:
    """Uninitialised device byte buffer (torch allocations are 512-byte
    aligned, which the 16-byte alignment rules of the C ABI need)."""
    return torch.empty(max(1, int(nbytes)), dtype=torch.uint8, device=device)


def to_numpy(t: torch.Tensor, dtype, shape=None) -> np.ndarray:
    a = t.detach().cpu().numpy().view(dtype)
    return a.reshape(shape) if shape is not None else a


def flows_of(e: W.EndToEnd) -> np.ndarray:
    """The compact flows {dst_ip, dport} of an end-to-end workload's probes."""
    f = np.zeros(len(e.probes.probes), W.FLOW_DTYPE)
    f["dst_ip"] = e.probes.probes["dst_ip"]
    f["dport"] = e.probes.probes["dport"]
    return f


def flow_columns_of(e: W.EndToEnd) -> tuple:
    """The same flows as two columns: destination addresses (uint32) and
    destination ports (uint16), 6 bytes per flow."""
    pr = e.probes.probes
    return np.ascontiguousarray(pr["dst_ip"], np.uint32), np.ascontiguousarray(pr["dport"], np.uint16)


class Validator:
    """One GPU validator context (not thread-safe)."""

    def __init__(self, device: int = 0):
        self.device = torch.device("cuda", device)
        torch.cuda.set_device(self.device)
        self.ctx = B.pv_create(device)
        self.num_nodes = 0
        self.num_hosts = 0

    def close(self):
        if self.ctx is not None:
            B.pv_destroy(self.ctx)
            self.ctx = None

    def __enter__(self):
        return self

    def __exit__(self, *exc):
        self.close()

    # -- options -------------------------------------------------------------
    def set_option(self, option: int, value: int):
        B.pv_set_option(self.ctx, option, value)

    def sync(self, stream=None):
        B.pv_sync(self.ctx, stream)

    # -- loads (host arrays) -------------------------------------------------
    def load_cluster(self, cluster: W.Cluster):
        B.pv_load_cluster(self.ctx, cluster.num_nodes, cluster.num_keys, cluster.labels)
        self.num_nodes = cluster.num_nodes

    def load_network(self, net: W.Network):
        B.pv_load_flow_tables(self.ctx, net.num_switches, net.rule_offs, net.rules, net.switch_region,
                              net.port_offs, net.port_peer, net.num_hosts, net.host_switch, net.host_port,
                              net.host_ip)
        self.num_hosts = net.num_hosts

    def begin_network(self, net: W.Network):
        """First half of a table load: host checks, the uploads and the first
        device passes queued; evaluation keeps the installed tables until
        finish_network installs these."""
        B.pv_load_flow_tables_begin(self.ctx, net.num_switches, net.rule_offs, net.rules, net.switch_region,
                                    net.port_offs, net.port_peer, net.num_hosts, net.host_switch, net.host_port,
                                    net.host_ip)
        self._pending_hosts = net.num_hosts

    def finish_network(self):
        """Second half of a table load begun by begin_network."""
        B.pv_load_flow_tables_end(self.ctx)
        self.num_hosts = self._pending_hosts

    # -- evaluation (device tensors) -----------------------------------------
    def eval_selectors(self, d_offs, num_exprs, d_exprs, d_assign, num_pods, words=None, d_bits=None,
                       d_flags=None, stream=None):
        words = words or W.words_per_row(self.num_nodes)
        if d_bits is None:
            d_bits = empty_device(num_pods * words * 4, self.device)
        if d_flags is None:
            d_flags = empty_device(num_pods, self.device)
        B.pv_eval_selectors(self.ctx, num_pods, d_offs, num_exprs, d_exprs, d_assign, d_bits, words, d_flags, stream)
        return d_bits, d_flags

    def verify_probes(self, d_probes, num_probes, hop_cap, d_out=None, stream=None):
        if d_out is None:
            d_out = empty_device(num_probes * 4, self.device)
        B.pv_verify_probes(self.ctx, num_probes, d_probes, hop_cap, d_out, stream)
        return d_out

    def load_policies(self, pol: W.PathPolicies):
        B.pv_load_path_policies(self.ctx, pol.num_policies, pol.forbid_offs, pol.forbid, pol.must_offs, pol.must,
                                pol.concrete)

    def verify_constrained(self, d_probes, num_probes, hop_cap, d_probe_policy=None, probes_per_policy=0,
                           d_out=None, d_waypoints=None, stream=None):
        """Walk under the loaded path constraints; returns (results, waypoint bits)."""
        if d_out is None:
            d_out = empty_device(num_probes * 4, self.device)
        if d_waypoints is None:
            d_waypoints = empty_device(num_probes * 4, self.device)
        B.pv_verify_probes_constrained(self.ctx, num_probes, d_probes, hop_cap, d_probe_policy, probes_per_policy,
                                       d_out, d_waypoints, stream)
        return d_out, d_waypoints

    def compliant_reach(self, graph_dev, num_src, d_src, num_masks, d_masks, words=None, d_reach=None,
                        stream=None):
        V, d_offs, E, d_cols, d_region = graph_dev
        words = words or W.words_per_row(V)
        if d_reach is None:
            d_reach = empty_device(num_masks * num_src * words * 4, self.device)
        B.pv_compliant_reach(self.ctx, V, d_offs, E, d_cols, d_region, num_src, d_src, num_masks, d_masks, d_reach,
                             words, stream)
        return d_reach

    def upload_graph(self, g: W.Graph):
        return (g.num_vertices, to_device(g.offs.astype(np.uint32), self.device), len(g.cols),
                to_device(g.cols.astype(np.uint32), self.device), to_device(g.region.astype(np.uint8), self.device))

    # -- end-to-end ------------------------------------------------------------
    def run_end_to_end(self, dev: dict, e2e_sizes: dict, stream=None) -> dict:
        """Selector rows -> seeded placement -> probe binding -> walks ->
        per-intent verdict, all on the device.  ``dev`` holds the device
        inputs (offs, exprs, draws, probes) and output buffers."""
        I, pods, ppg = e2e_sizes["intents"], e2e_sizes["pods"], e2e_sizes["probes_per_intent"]
        words = W.words_per_row(self.num_nodes)
        M = I * ppg
        B.pv_eval_selectors(self.ctx, I, dev["offs"], e2e_sizes["num_exprs"], dev["exprs"], None, dev["bits"], words,
                            dev["flags"], stream)
        B.pv_place_pods(self.ctx, I, pods, dev["bits"], words, dev["draws"], dev["assign"], stream)
        self._walk_and_verdict(dev, e2e_sizes, 0, I, stream)
        return dev

    def _walk_and_verdict(self, dev, e2e_sizes, lo, hi, stream):
        """Binding, walks and verdicts of intents [lo, hi) (one fused call
        binds the flows and walks them); under the loaded path policies
        (policy i for intent i) when ``dev`` holds a "hits" buffer."""
        ppg, pods, n = e2e_sizes["probes_per_intent"], e2e_sizes["pods"], hi - lo
        words = W.words_per_row(self.num_nodes)
        results = dev["results"][lo * ppg * 4:]
        dst, dport, masks = dev["dst"][lo * ppg * 4:], dev["dport"][lo * ppg * 2:], dev["masks"][lo * 4:]
        bits, flags, assign = dev["bits"][lo * words * 4:], dev["flags"][lo:], dev["assign"][lo * pods * 4:]
        cap = e2e_sizes["hop_cap"]
        if "hits" in dev:
            hits = dev["hits"][lo * ppg * 4:]
            B.pv_verify_flow_columns_constrained(self.ctx, n * ppg, dst, dport, ppg, pods, assign, masks, cap, None,
                                                 ppg, lo, None, results, hits, stream)
            B.pv_aggregate_constrained(self.ctx, n, pods, bits, words, flags, assign, ppg, results, hits, None,
                                       dev["pass"][lo:], dev["counts"][lo * 32:], stream, first_policy=lo)
        else:
            B.pv_verify_flow_columns(self.ctx, n * ppg, dst, dport, ppg, pods, assign, masks, cap, None, results,
                                     stream)
            B.pv_aggregate_intents(self.ctx, n, pods, bits, words, flags, assign, ppg, results, dev["pass"][lo:],
                                   dev["counts"][lo * 32:], stream)

    _INPUTS = ("offs", "exprs", "draws", "masks", "dst", "dport")

    def run_end_to_end_from_host(self, host: dict, dev: dict, e2e_sizes: dict, stream, copy_stream,
                                 chunks: int = 1, loads=None, loads_first: bool = False) -> dict:
        """The end-to-end pipeline on inputs in pinned HOST memory.  Every
        input upload is enqueued on `copy_stream`, the flows cut into
        `chunks` intent ranges (independent units), and range c is verified
        on `stream` as soon as its flows have arrived.  ``loads()``, if given
        (the cluster and table loads), runs before any upload is queued, so
        its copies go first on the host-to-device link; if it returns a
        callable (the second half of a two-part table load, which waits on
        the host for the load's first device passes), that runs once every
        upload is queued, while the inputs arrive, or at once with
        `loads_first`.  The evaluation calls wait for the loads' device work
        on the device.  The per-intent verdicts and counters come back into
        ``host["pass"]`` and ``host["counts"]`` on `stream` (not
        synchronised).

        ``host`` holds pinned byte tensors "offs", "exprs", "draws", "masks",
        "dst", "dport" (inputs, as alloc_end_to_end lays them out: the flows
        as two columns, 6 bytes each, the probe records are built on the
        device) and "pass", "counts" (outputs);
        ``dev`` the device buffers of alloc_end_to_end.

        Consecutive calls alternate between two sets of device input buffers,
        so a call's uploads wait only for the call two back (the last one to
        read that set), not for the previous call's kernels: the uploads of
        one batch overlap the verification of the one before."""
        I, pods, ppg = e2e_sizes["intents"], e2e_sizes["pods"], e2e_sizes["probes_per_intent"]
        words = W.words_per_row(self.num_nodes)
        ctx = self.ctx
        chunks = max(1, min(int(chunks), max(1, I // 4)))
        # range edges on multiples of 4 intents (keeps every slice 16-byte aligned)
        edges = [0] + [((I * c) // chunks) & ~3 for c in range(1, chunks)] + [I]
        ranges = [(lo, hi) for lo, hi in zip(edges[:-1], edges[1:]) if hi > lo]
        finish = loads() if loads is not None else None
        if callable(finish) and loads_first:
            finish()
            finish = None
        if "_inputs" not in dev:   # the second input set, and each set's last reader
            dev["_inputs"] = [{k: dev[k] for k in self._INPUTS},
                              {k: torch.empty_like(dev[k]) for k in self._INPUTS}]
            dev["_read"] = [None, None]
            dev["_slot"] = [0]
        k_slot = dev["_slot"][0]
        dev["_slot"][0] ^= 1
        read = dev["_read"]
        dev = {**dev, **dev["_inputs"][k_slot]}
        # the kernels that last read this input set must be done with it
        ready = []
        with torch.cuda.stream(copy_stream):
            if read[k_slot] is not None:
                copy_stream.wait_event(read[k_slot])
            for k in ("offs", "exprs", "draws", "masks"):
                n = host[k].numel()
                dev[k][:n].copy_(host[k], non_blocking=True)
            for lo, hi in ranges:   # flows of intents [lo, hi)
                for k, b in (("dst", 4), ("dport", 2)):
                    dev[k][lo * ppg * b:hi * ppg * b].copy_(host[k][lo * ppg * b:hi * ppg * b], non_blocking=True)
                ev = torch.cuda.Event()
                ev.record(copy_stream)
                ready.append(ev)
        if callable(finish):
            finish()
        for (lo, hi), ev in zip(ranges, ready):
            n = hi - lo
            stream.wait_event(ev)
            bits = dev["bits"][lo * words * 4:]
            flags = dev["flags"][lo:]
            assign = dev["assign"][lo * pods * 4:]
            B.pv_eval_selectors(ctx, n, dev["offs"][lo * 4:], e2e_sizes["num_exprs"], dev["exprs"], None, bits,
                                words, flags, stream)
            B.pv_place_pods(ctx, n, pods, bits, words, dev["draws"][lo * pods * 8:], assign, stream)
            self._walk_and_verdict(dev, e2e_sizes, lo, hi, stream)
        done = torch.cuda.Event()
        done.record(stream)
        read[k_slot] = done
        with torch.cuda.stream(stream):
            host["pass"].copy_(dev["pass"][: host["pass"].numel()], non_blocking=True)
            host["counts"].copy_(dev["counts"][: host["counts"].numel()], non_blocking=True)
        return host

    def alloc_end_to_end(self, e: W.EndToEnd, with_policies: bool = False) -> tuple:
        """Device buffers for an end-to-end workload (inputs uploaded); with
        with_policies, a waypoint-bit buffer that makes the pipeline check the
        loaded path policies (policy i for intent i)."""
        I, pods, ppg = e.intents.num_pods, e.pods_per_intent, e.probes_per_intent
        words = W.words_per_row(e.cluster.num_nodes)
        M = I * ppg
        d = self.device
        dev = {
            "offs": to_device(e.intents.expr_offs.astype(np.uint32), d),
            "exprs": to_device(e.intents.exprs, d),
            "draws": to_device(e.place_draws.astype(np.uint64), d),
            "probes": to_device(e.probes.probes, d),
            "flows": to_device(flows_of(e), d),
            "dst": to_device(flow_columns_of(e)[0], d),
            "dport": to_device(flow_columns_of(e)[1], d),
            "masks": to_device(e.intent_mask.astype(np.uint32), d),
            "bits": empty_device(I * words * 4, d),
            "flags": empty_device(I, d),
            "assign": empty_device(I * pods * 4, d),
            "results": empty_device(M * 4, d),
            "pass": empty_device(I, d),
            "counts": empty_device(I * 8 * 4, d),
        }
        if with_policies:
            dev["hits"] = empty_device(M * 4, d)
        sizes = {"intents": I, "pods": pods, "probes_per_intent": ppg, "num_exprs": len(e.intents.exprs),
                 "hop_cap": e.probes.hop_cap}
        return dev, sizes
