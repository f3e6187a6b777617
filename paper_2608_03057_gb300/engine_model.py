"""Cycle model of the paper's bit-serial Temporal-Precision Engine (host only).

The engine multiplies an L-plane weight tile by an R-plane activation tile as
L x R binary passes, EXEC(W_i, A_j, shift i + j) = popcount(W_i AND A_j)
<< (i + j), and differs between schedules only in how often it fetches a
plane (Algorithm "Bit-plane schedules"):

  naive                  for i: for j: fetch W_i, fetch A_j, EXEC   2 L R fetches
  weight-stationary      for i: fetch W_i; for j: fetch A_j, EXEC   L + L R fetches
  activation-stationary  fetch A_1..A_R; for i: fetch W_i;          L + R fetches
                         for j: EXEC

(the last one is the paper's engine: per stage, L = L_s is one register write
and only the top L_s stored weight planes are streamed; Sec. 3.3, App. F.2).

`walk` runs a schedule's loop nest on one tile of integer codes, counting the
fetches and passes it actually makes, and returns the exact integer product, so
the fetch counts and bit-exactness are properties of the loops, not of the
formulas above.

Two cost regimes are printed in the paper, and the model reproduces both:
  * a fetch-bound single tile (Table "Bit-plane dataflows", R = 4, L in
    {3, 4, 8}): cycles = FETCH_CYCLES x fetches + OVERHEAD[schedule];
  * the compute-bound network setting (Table "Measured four-tile GEMM cost",
    A4, W1..W8 and the mixed {1, 2, 3, 4} schedule): cycles = PASS_CYCLES x
    L x R per tile, additive over tiles (a precision switch costs 0 cycles).
The paper prints the cycle counts but not these constants: they are the exact
least-squares fit to the printed tables (every printed count is reproduced to
the cycle), recomputed from the tables by tests/golden/fit_engine_cycles.py.

The GPU path does not run on this engine (its tensor pipe has a fixed operand
precision); the model only reports what the paper's engine would spend on a
schedule, next to Rel. BitOPs.
"""
from __future__ import annotations

from typing import Dict, Iterable, List, Sequence, Tuple

import numpy as np

SCHEDULES = ("naive", "weight_stationary", "activation_stationary")

# Fit to Table "Bit-plane dataflows" (fetch-bound single tile): one plane fetch
# costs 570 cycles; the fixed part is 173 cycles for the two re-fetching loops
# and 323 for the activation-stationary one.
FETCH_CYCLES = 570
OVERHEAD = {"naive": 173, "weight_stationary": 173, "activation_stationary": 323}
# Fit to Table "Measured four-tile GEMM cost" (compute-bound): 33 cycles per
# binary pass, so a W-bit x A4 tile costs 132 W cycles.
PASS_CYCLES = 33


def planes(codes: np.ndarray, n_planes: int, top: int = 8) -> List[np.ndarray]:
    """Bit planes of unsigned codes: plane p (0 = least significant) of the
    `n_planes` most significant of `top` planes, returned from the lowest
    selected plane up, each with its weight exponent."""
    codes = np.asarray(codes, np.int64)
    first = top - n_planes
    return [((codes >> p) & 1) for p in range(first, top)]


def walk(schedule: str, w_codes: np.ndarray, a_codes: np.ndarray, L: int, R: int,
         w_top: int = 8, a_top: int = None) -> Tuple[int, int, int]:
    """Run one tile of `schedule` on unsigned codes (w_codes, a_codes: 1-D of
    equal length).  The weight operand is its top L of w_top planes (the
    truncated operating weight of Eq. hw_multi_lsb), the activation operand all
    R planes.  Returns (integer product, plane fetches, binary passes)."""
    if schedule not in SCHEDULES:
        raise ValueError(schedule)
    a_top = R if a_top is None else a_top
    Wp = planes(w_codes, L, w_top)
    Ap = planes(a_codes, R, a_top)
    w0, a0 = w_top - L, a_top - R  # exponent of the lowest selected plane
    fetches = passes = 0
    acc = 0

    def exec_pass(wi, aj, shift):
        nonlocal acc, passes
        passes += 1
        acc += int(np.sum(wi & aj)) << shift

    if schedule == "naive":
        for i in range(L):
            for j in range(R):
                fetches += 2  # W_i and A_j, refetched every pass
                exec_pass(Wp[i], Ap[j], w0 + i + a0 + j)
    elif schedule == "weight_stationary":
        for i in range(L):
            fetches += 1  # W_i held while the activation planes stream past
            for j in range(R):
                fetches += 1
                exec_pass(Wp[i], Ap[j], w0 + i + a0 + j)
    else:
        fetches += R  # every activation plane stays on chip for the tile
        for i in range(L):
            fetches += 1  # each selected weight plane is streamed once
            for j in range(R):
                exec_pass(Wp[i], Ap[j], w0 + i + a0 + j)
    return acc, fetches, passes


def fetch_count(schedule: str, L: int, R: int) -> int:
    """Plane fetches of one tile, by walking the schedule's loop nest."""
    z = np.zeros(1, np.int64)
    return walk(schedule, z, z, L, R, w_top=max(L, 8), a_top=R)[1]


def fetch_bound_cycles(schedule: str, L: int, R: int = 4) -> int:
    """Cycles of one fetch-bound tile (Table "Bit-plane dataflows" regime)."""
    return FETCH_CYCLES * fetch_count(schedule, L, R) + OVERHEAD[schedule]


def compute_bound_cycles(w_bits: Sequence[int], a_bits: int = 4) -> int:
    """Cycles of a sequence of compute-bound tiles, one per entry of w_bits
    (Table "Measured four-tile GEMM cost" regime): PASS_CYCLES x W x A each,
    and nothing for switching precision between tiles."""
    return int(sum(PASS_CYCLES * int(w) * int(a_bits) for w in w_bits))


def schedule_cost(table: np.ndarray, layer_ops: Iterable[float], a_bits: int = 8) -> Dict[str, float]:
    """What the paper's engine would spend on a bit schedule [L][S], relative
    to running every (layer, stage) at 8 bits: each layer-stage weighs its
    multiply-adds (layer_ops) times the cost of one tile at its precision b.

      compute_bound            sum ops x b x A / sum ops x 8 x A
      fetch_bound_<schedule>   sum ops x cycles(b) / sum ops x cycles(8)
                               (per-tile fetch-bound cycles at R = a_bits)
    """
    t = np.asarray(table, np.int64)
    w = np.asarray(list(layer_ops), np.float64)[:, None] * np.ones((1, t.shape[1]))
    out = {"compute_bound": float((w * compute_cost_grid(t, a_bits)).sum()
                                  / (w * compute_bound_cycles([8], a_bits)).sum())}
    for sch in SCHEDULES:
        cyc = np.vectorize(lambda b: fetch_bound_cycles(sch, int(b), a_bits))(t)
        out[f"fetch_bound_{sch}"] = float((w * cyc).sum() / (w * fetch_bound_cycles(sch, 8, a_bits)).sum())
    return out


def compute_cost_grid(table: np.ndarray, a_bits: int) -> np.ndarray:
    return PASS_CYCLES * np.asarray(table, np.int64) * int(a_bits)
