#!/usr/bin/env python3
"""Fits the cycle constants of the bit-serial engine model to the paper's
printed cycle counts (tests/golden/engine_cycles_paper.txt) and writes them to
tests/golden/engine_cycle_constants.txt.

Fetch-bound tiles: cycles = f x fetches + c[schedule], with fetches from the
table's own fetch model (2LR, L+LR, L+R); least squares over the nine printed
counts, one shared f and one intercept per schedule.  Compute-bound tiles:
cycles = p x sum over tiles of W x A; least squares over the seven printed
counts.  Both fits are exact on the printed numbers (zero residual), which the
script checks before writing.

Run: python tests/golden/fit_engine_cycles.py
"""
from __future__ import annotations

import os

import numpy as np

HERE = os.path.dirname(os.path.abspath(__file__))
SRC = os.path.join(HERE, "engine_cycles_paper.txt")
OUT = os.path.join(HERE, "engine_cycle_constants.txt")
SCHEDULES = ("naive", "weight_stationary", "activation_stationary")
FETCH_MODEL = {"2LR": lambda L, R: 2 * L * R, "L+LR": lambda L, R: L + L * R, "L+R": lambda L, R: L + R}


def read_table(path=SRC):
    fetch, compute = [], []
    for line in open(path):
        f = line.split()
        if not f or f[0].startswith("#"):
            continue
        if f[0] == "fetchbound":
            fetch.append((f[1], int(f[2]), int(f[3]), f[4], int(f[5])))
        elif f[0] == "computebound":
            compute.append((f[1], [int(v) for v in f[2].split(",")], int(f[3]), int(f[4])))
    return fetch, compute


def fit(path=SRC):
    fetch, compute = read_table(path)
    A = np.zeros((len(fetch), 1 + len(SCHEDULES)))
    y = np.zeros(len(fetch))
    for r, (sch, L, R, model, cyc) in enumerate(fetch):
        A[r, 0] = FETCH_MODEL[model](L, R)
        A[r, 1 + SCHEDULES.index(sch)] = 1.0
        y[r] = cyc
    sol = np.linalg.lstsq(A, y, rcond=None)[0]
    f_cyc = int(round(sol[0]))
    over = {s: int(round(sol[1 + i])) for i, s in enumerate(SCHEDULES)}
    assert np.allclose(A @ np.array([f_cyc] + [over[s] for s in SCHEDULES]), y), "fetch-bound fit is not exact"
    B = np.array([[sum(w * a for w in ws)] for _, ws, a, _ in compute], np.float64)
    z = np.array([c for *_, c in compute], np.float64)
    p = int(round(np.linalg.lstsq(B, z, rcond=None)[0][0]))
    assert np.allclose(B[:, 0] * p, z), "compute-bound fit is not exact"
    return f_cyc, over, p


def main():
    f_cyc, over, p = fit()
    with open(OUT, "w") as fh:
        fh.write("# Written by tests/golden/fit_engine_cycles.py from engine_cycles_paper.txt (the paper's\n"
                 "# printed cycle counts); exact least-squares fit, zero residual.\n")
        fh.write(f"fetch_cycles {f_cyc}\n")
        for s in SCHEDULES:
            fh.write(f"overhead_{s} {over[s]}\n")
        fh.write(f"pass_cycles {p}\n")
    print(open(OUT).read(), end="")


if __name__ == "__main__":
    main()
