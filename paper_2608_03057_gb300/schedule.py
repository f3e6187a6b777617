"""Host-side bookkeeping of a TASQ bit schedule (no device work).

The schedule is the bit-allocation map of App. F.1: one operating precision
b in 2..8 per (layer, stage), stored as uint8 [L][S].  Stages are contiguous
partitions of the denoising trajectory, stage 0 holding the noisiest steps
(Sec. 3.2, stage-wise sharing; App. D.1 convention).
"""
from __future__ import annotations

import numpy as np


def stage_of_step(step: int, n_steps: int, n_stages: int) -> int:
    """Contiguous partition: stage = floor(step * S / T)."""
    if not (0 <= step < n_steps) or n_stages < 1 or n_stages > n_steps:
        raise ValueError("need 0 <= step < n_steps and 1 <= n_stages <= n_steps")
    return (step * n_stages) // n_steps


def effective_bits(table: np.ndarray, layer_ops) -> np.ndarray:
    """Average operating weight precision of each stage, weighted by each
    layer's multiply-add count ("Eff. W" of the quality-compute table)."""
    t = np.asarray(table, np.float64)
    w = np.asarray(layer_ops, np.float64)
    return (t * w[:, None]).sum(0) / w.sum()


def rel_bitops(eff_w_bits: float, a_bits: int) -> float:
    """Compute cost relative to static W8A8: (W bits x A bits) / 64."""
    return float(eff_w_bits) * float(a_bits) / 64.0
