"""Helpers of the GPU-vs-oracle step comparisons.

Comparison rules (the method's own tolerances):
  * logits / hidden states: max |gpu - oracle| <= tol * max|oracle row|, tol = 1e-4 for
    fp32 models and 2e-2 for bf16 models;
  * discrete results (argmax, top-k, tree tokens, accepted path, emitted tokens) are
    bit-exact, except where the oracle's own margin between the two candidates is
    below 1e-2 of the row's max |value| (a near-tie): there the GPU's choice must be
    valid under the oracle's values (within the tolerance of the best one) and the
    case is counted as flagged.
"""
from __future__ import annotations

import numpy as np

NEAR_TIE = 1e-2


def tol_of(cfg) -> float:
    return 1e-4 if cfg["dtype"] == "fp32" else 2e-2


def rel_rows(a: np.ndarray, ref: np.ndarray) -> float:
    a = np.asarray(a, np.float64)
    ref = np.asarray(ref, np.float64)
    den = np.maximum(np.max(np.abs(ref), axis=-1, keepdims=True), 1e-30)
    return float(np.max(np.abs(a - ref) / den))


def check_choice(gpu_idx: int, z: np.ndarray, ref_idx: int, rank_vals=None) -> bool:
    """True if gpu_idx equals the oracle's choice, or if the oracle's choice is within a
    near-tie of it (the case is then flagged by the caller).  Raises on a real miss."""
    if gpu_idx == ref_idx:
        return False
    scale = np.max(np.abs(z))
    if abs(z[ref_idx] - z[gpu_idx]) <= NEAR_TIE * scale:
        return True
    raise AssertionError(f"choice {gpu_idx} (oracle value {z[gpu_idx]:.6g}) vs oracle {ref_idx} "
                         f"({z[ref_idx]:.6g}): margin {(z[ref_idx] - z[gpu_idx]) / scale:.3g} of row max")


def check_topk(gpu_idx, z: np.ndarray, k: int) -> int:
    """GPU top-k list against the oracle's values; returns the number of flagged ranks."""
    from oracle import chimera_oracle as co
    ref = co.topk_desc(z, k)
    flags = 0
    for r in range(k):
        flags += int(check_choice(int(gpu_idx[r]), z, int(ref[r])))
    assert len(set(int(i) for i in gpu_idx[:k])) == k
    return flags
