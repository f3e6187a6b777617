"""Pins of the cycle model of the paper's bit-serial engine (host only).

The model walks the three loop nests of Algorithm "Bit-plane schedules"; these
tests check it against what the paper prints: the plane-fetch models of Table
"Bit-plane dataflows" (2LR, L+LR, L+R; 64/40/12 at L = 8, R = 4), every cycle
count of that table, the 528 W linear law and the mixed {1, 2, 3, 4} schedule
(1,320 cycles, no switching overhead) of Table "Measured four-tile GEMM cost",
the 3.2-5.1x reduction quoted in Sec. 3.3, and bit-exactness of every schedule
against the integer product of the truncated weight (Eq. hw_multi_lsb).
"""
import importlib.util
import os

import numpy as np
import pytest

from paper_2608_03057_gb300 import engine_model as E
from paper_2608_03057_gb300 import schedule, workloads

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")


def _fit_module():
    spec = importlib.util.spec_from_file_location("fit_engine_cycles", os.path.join(GOLDEN, "fit_engine_cycles.py"))
    m = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(m)
    return m


def _constants():
    out = {}
    for line in open(os.path.join(GOLDEN, "engine_cycle_constants.txt")):
        if line.strip() and not line.startswith("#"):
            k, v = line.split()
            out[k] = int(v)
    return out


def test_constants_match_the_fit_of_the_printed_tables():
    c = _constants()
    assert (c["fetch_cycles"], c["pass_cycles"]) == (E.FETCH_CYCLES, E.PASS_CYCLES)
    for s in E.SCHEDULES:
        assert c[f"overhead_{s}"] == E.OVERHEAD[s]
    # the committed constants are what the script computes from the paper's numbers
    f_cyc, over, p = _fit_module().fit()
    assert (f_cyc, p) == (E.FETCH_CYCLES, E.PASS_CYCLES) and over == E.OVERHEAD


@pytest.mark.parametrize("L", range(1, 9))
@pytest.mark.parametrize("R", [1, 2, 4, 8])
def test_fetch_counts_are_the_printed_models(L, R):
    assert E.fetch_count("naive", L, R) == 2 * L * R
    assert E.fetch_count("weight_stationary", L, R) == L + L * R
    assert E.fetch_count("activation_stationary", L, R) == L + R


def test_fetch_counts_at_l8_r4():
    assert [E.fetch_count(s, 8, 4) for s in E.SCHEDULES] == [64, 40, 12]


def test_fetch_bound_cycles_reproduce_the_table():
    fetch, _ = _fit_module().read_table()
    assert len(fetch) == 9
    for sch, L, R, _, cycles in fetch:
        assert E.fetch_bound_cycles(sch, L, R) == cycles, (sch, L)


def test_reduction_over_the_naive_loop():
    # "3.2-5.1x fewer cycles than the naive loop" across L = 3, 4, 8
    r = [E.fetch_bound_cycles("naive", L) / E.fetch_bound_cycles("activation_stationary", L) for L in (3, 4, 8)]
    assert round(min(r), 1) == 3.2 and round(max(r), 1) == 5.1


def test_compute_bound_law_and_mixed_schedule():
    _, compute = _fit_module().read_table()
    for label, w_bits, a_bits, cycles in compute:
        assert E.compute_bound_cycles(w_bits, a_bits) == cycles, label
    static = {w: E.compute_bound_cycles([w] * 4, 4) for w in (1, 2, 3, 4, 6, 8)}
    assert all(static[w] == 528 * w for w in static)  # linear in W at A4
    mixed = E.compute_bound_cycles([1, 2, 3, 4], 4)
    assert mixed == 1320
    # no switching overhead: the mixed run costs the mean of the static runs it mixes
    assert mixed == sum(static[w] for w in (1, 2, 3, 4)) // 4


@pytest.mark.parametrize("schedule_name", E.SCHEDULES)
@pytest.mark.parametrize("L", [8, 6, 3, 1])
def test_every_schedule_is_bit_exact(schedule_name, L):
    """Each loop nest returns sum_k Q_x[k] * trunc_L(Q_w[k]) exactly, with
    trunc_L keeping the top L of the 8 stored planes (the operating weight on
    the stored grid, Eq. hw_multi_lsb), and makes L x R passes."""
    K = 97
    R = 4
    qw = workloads.uniform_codes((K,), 41, 0, 127).astype(np.int64) * 2 + 1  # odd codes up to 255
    qx = workloads.uniform_codes((K,), 42, 0, 15).astype(np.int64)  # A4 codes
    acc, fetches, passes = E.walk(schedule_name, qw, qx, L, R)
    k = 8 - L
    want = int(np.dot((qw >> k) << k, qx))
    assert acc == want
    assert passes == L * R
    assert fetches == E.fetch_count(schedule_name, L, R)


def test_schedule_cost_of_the_benchmark_schedules():
    """All 8 bits costs 1; in the compute-bound regime the relative cost at A8
    equals Rel. BitOPs = Eff. W x 8 / 64; fetch-bound costs fall more slowly
    than b (the R activation fetches and the fixed part do not shrink)."""
    for name in ("pixart", "sana", "sdxl"):
        layers = workloads.inventory(name)
        ops = [l.ops for l in layers]
        table = workloads.schedule_for(name, len(layers))
        c8 = E.schedule_cost(np.full_like(table, 8), ops)
        assert all(abs(v - 1.0) < 1e-12 for v in c8.values())
        c = E.schedule_cost(table, ops)
        eff = float((schedule.effective_bits(table, ops)).mean())
        assert abs(c["compute_bound"] - schedule.rel_bitops(eff, 8)) < 1e-12
        assert c["compute_bound"] < c["fetch_bound_activation_stationary"] < 1.0
