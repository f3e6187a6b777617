"""Measures the tensor-core MMA kinds this GPU offers for integer-valued
operands (tasq_probe_mma, a diagnostic with no counterpart in the paper):

  * rate: cycles per tcgen05.mma (M = 128, N = 128 / 192 / 256) of kind::f16,
    the operand type of the exact route, against kind::f8f6f4 with e4m3 or
    e5m2 operands (twice the K per instruction), every SM issuing at once;
  * exactness: long fp32 accumulations of integer products in each kind,
    against the exact integer result, on patterns chosen to expose a reduced-
    precision accumulation: extreme codes, partial sums up to just below 2^24,
    large and small products in one instruction, cancelling signs, and random
    A4 activation codes times truncated weights (5-bit for e4m3; for e5m2 the
    b <= 4 weights mask_b(s_w) = 16 t, |t| <= 8, that the 8-bit route feeds it).

Run: python -m paper_2608_03057_gb300.mma_probe  (prints one JSON object)
"""
from __future__ import annotations

import json

import numpy as np

from . import tasq, workloads

KINDS = {0: "f16", 1: "e4m3 (kind::f8f6f4)", 2: "e5m2 (kind::f8f6f4)"}
# repetitions of a row for the exactness runs: the longest reaches just below 2^24
EXACT_REPS = {0: (1, 64, 511), 1: (1, 64, 511), 2: (1, 16, 127)}


def patterns(kind: int, n: int, seed: int = 3):
    """Integer operand rows: A [128][E], B [n][E] with E = 64 (f16) or 128 (8-bit)
    elements per 128-byte row."""
    E = 64 if kind == 0 else 128
    h = E // 2
    rng = workloads.rng(seed)
    if kind == 2:
        # values with at most three significant bits: A4 codes, b <= 4 weights
        a_types = [np.full(E, 8), np.full(E, 1), np.r_[np.full(h, 8), np.full(h, 1)],
                   np.tile([8, -8], h), np.r_[np.full(E - 1, -8), [1]]]
        A = np.stack([a_types[i % len(a_types)] if i < 96 else rng.integers(-8, 8, E) for i in range(128)])
        b_types = [np.full(E, 112), np.full(E, 1), np.tile([112, -112], h), np.r_[np.full(E - 2, -128), [1, -1]],
                   np.full(E, -128)]
        B = np.stack([b_types[i % len(b_types)] if i < n // 2 else 16 * rng.integers(-8, 8, E) for i in range(n)])
        return A.astype(np.int64), B.astype(np.int64)
    a_types = [np.full(E, 16), np.full(E, 1), np.r_[np.full(h, 16), np.full(h, 1)],
               np.tile([16, -16], h), np.r_[np.full(E - 1, -16), [1]]]
    A = np.stack([a_types[i % len(a_types)] if i < 96 else rng.integers(-8, 8, E) for i in range(128)])
    b_types = [np.full(E, 15), np.full(E, 1), np.tile([15, -15], h), np.r_[np.full(E - 2, 16), [1, -1]],
               np.full(E, -16)]
    B = np.stack([b_types[i % len(b_types)] if i < n // 2 else rng.integers(-16, 16, E) for i in range(n)])
    return A.astype(np.int64), B.astype(np.int64)


def encode(vals: np.ndarray, kind: int) -> np.ndarray:
    """Byte image of integer values as fp16 (kind 0), e4m3 (kind 1) or e5m2 (kind 2)."""
    import torch
    t = torch.from_numpy(vals.astype(np.float32))
    if kind == 0:
        return t.to(torch.float16).view(torch.uint8).numpy().reshape(vals.shape[0], -1)
    enc = t.to(torch.float8_e4m3fn if kind == 1 else torch.float8_e5m2)
    assert bool((enc.float() == t).all()), f"value not exact in {KINDS[kind]}"
    return enc.view(torch.uint8).numpy().reshape(vals.shape[0], -1)


def run_probe(kind: int, n: int, reps: int, A: np.ndarray, B: np.ndarray, ctas: int = 1):
    import torch
    da = torch.from_numpy(np.ascontiguousarray(encode(A, kind))).cuda()
    db = torch.from_numpy(np.ascontiguousarray(encode(B, kind))).cuda()
    dd = torch.zeros((128, n), dtype=torch.float32, device="cuda")
    cyc = torch.zeros((ctas,), dtype=torch.int64, device="cuda")
    tasq.tasq_probe_mma(kind, n, reps, da, db, dd, cyc, ctas)
    torch.cuda.synchronize()
    return dd.cpu().numpy(), cyc.cpu().numpy()


def exactness(kind: int, n: int = 256, reps=None):
    """Largest |D| reached and mismatches against the exact integer result."""
    reps = EXACT_REPS[kind] if reps is None else reps
    A, B = patterns(kind, n)
    ref1 = A @ B.T
    out = []
    for r in reps:
        d, cyc = run_probe(kind, n, r, A, B)
        assert cyc[0] != 0, "probe wait timed out"
        ref = ref1 * r
        got = d.astype(np.float64)
        bad = got != ref
        out.append({"reps": r, "K": r * A.shape[1], "max_abs": int(np.abs(ref).max()), "mismatches": int(bad.sum()),
                    "elements": int(bad.size)})
    return out


def rate(kind: int, n: int, sms: int, reps: int = 256, clock_mhz: float = None):
    A, B = patterns(kind, n)
    run_probe(kind, n, 8, A, B, sms)  # warm-up
    _, cyc = run_probe(kind, n, reps, A, B, sms)
    per_mma = float(np.median(cyc)) / (4 * reps)
    k = 16 if kind == 0 else 32
    out = {"kind": KINDS[kind], "N": n, "K_per_mma": k, "cycles_per_mma": per_mma}
    if clock_mhz:
        out["tflops_all_sms"] = 2 * 128 * n * k * sms / (per_mma / (clock_mhz * 1e6)) / 1e12
    return out


def run(clock_mhz: float = None) -> dict:
    import torch
    sms = torch.cuda.get_device_properties(0).multi_processor_count
    res = {"rates": [rate(kind, n, sms, clock_mhz=clock_mhz) for kind in (0, 1, 2) for n in (128, 192, 256)],
           "exactness": {KINDS[k]: exactness(k) for k in (0, 1, 2)},
           "sms": sms, "clock_mhz_assumed": clock_mhz}
    return res


if __name__ == "__main__":
    import torch
    mhz = None
    try:
        import subprocess
        mhz = float(subprocess.run(["nvidia-smi", "-i", "0", "--query-gpu=clocks.max.sm", "--format=csv,noheader,nounits"],
                                   capture_output=True, text=True).stdout.split()[0])
    except Exception:
        pass
    print(json.dumps(run(mhz)))
