"""Helpers for the GPU parity tests (no method arithmetic)."""
import numpy as np

from paper_2602_16100_gb300 import workloads as W


def sub_selectors(sel: W.Selectors, idx: np.ndarray):
    """CSR of the pods in idx (for oracle evaluation of sampled rows)."""
    offs = sel.expr_offs.astype(np.int64)
    counts = offs[idx + 1] - offs[idx]
    new_offs = np.zeros(len(idx) + 1, np.uint32)
    new_offs[1:] = np.cumsum(counts)
    parts = [sel.exprs[offs[i]:offs[i + 1]] for i in idx]
    exprs = np.concatenate(parts) if parts else np.zeros(0, W.EXPR_DTYPE)
    assign = None if sel.assign is None else sel.assign[idx]
    return new_offs, exprs, assign


def sample(n: int, k: int, seed: int = 0) -> np.ndarray:
    """k distinct sorted indices in [0, n), always including both ends."""
    st = W.Stream(seed, "sample")
    if k >= n:
        return np.arange(n)
    s = np.unique(np.concatenate([[0, n - 1], (st.u64(k) % np.uint64(n)).astype(np.int64)]))
    return s


# Small end-to-end batches of the GPU parity tests, shared with the CPU test
# that shows their expected verdicts tell planted faults apart.
E2E_PASS_SMALL = dict(seed=21, num_switches=64, num_intents=300, probes_per_intent=200, rules_per_switch=200,
                      pass_share=0.3)
E2E_CONSTRAINED = dict(seed=25, num_switches=64, num_intents=300, probes_per_intent=100, rules_per_switch=200,
                       pass_share=0.3)
POLICIES_CONSTRAINED = dict(seed=7, forbid_max=1, must_max=2, hubs=6, p_noop=0.3)
