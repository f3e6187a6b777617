"""One masked contraction shape, timed (and a fixed launch sequence to profile).

Packs seeded uniform weight codes in [-127, 127], draws activation codes
uniform over the range of n-bit codes, and runs tasq_masked_gemm at one b: a
few eager calls, then a CUDA graph of back-to-back calls timed with CUDA events.
With --act-bits 4 the codes come in the fp16 + e5m2 format, so b <= 4 takes the
8-bit-float route.  Prints one JSON object.

Run: python -m paper_2608_03057_gb300.one_gemm --M 4096 --N 4096 --K 4096 --b 4 --act-bits 4
"""
from __future__ import annotations

import argparse
import json

import numpy as np

from . import tasq


def main(argv=None):
    ap = argparse.ArgumentParser()
    ap.add_argument("--M", type=int, default=4096)
    ap.add_argument("--N", type=int, default=4096)
    ap.add_argument("--K", type=int, default=4096)
    ap.add_argument("--b", type=int, default=8)
    ap.add_argument("--act-bits", type=int, default=8, help="activation code bits (<= 4: fp16 + e5m2 codes)")
    ap.add_argument("--eager", type=int, default=3, help="eager calls before the timed graph")
    ap.add_argument("--reps", type=int, default=20, help="calls in the timed graph (0: no graph)")
    ap.add_argument("--seed", type=int, default=0)
    args = ap.parse_args(argv)
    import torch
    M, N, K, n = args.M, args.N, args.K, args.act_bits
    ctx = tasq.tasq_create(torch.cuda.current_device())
    tasq.tasq_set_schedule(ctx, np.array([[args.b]], np.uint8), 1, 1)
    g = torch.Generator(device="cuda")
    g.manual_seed(args.seed)
    sw = torch.randint(-127, 128, (N, K), generator=g, device="cuda", dtype=torch.int8)
    cw = torch.rand((N,), generator=g, device="cuda") * 1e-3 + 1e-4
    pk = torch.empty((tasq.tasq_packed_bytes(tasq.TASQ_LINEAR, N, K),), dtype=torch.uint8, device="cuda")
    tasq.tasq_pack_weights(ctx, tasq.TASQ_LINEAR, sw, cw, None, N, K, 0, pk)
    half = 1 << (n - 1)
    s = torch.randint(-half, half, (M, K), generator=g, device="cuda", dtype=torch.int8)
    f8 = n <= 4
    fmt = tasq.TASQ_CODES_F16_E5M2 if f8 else tasq.TASQ_CODES_F16
    codes = torch.empty(((3 if f8 else 2) * M * K,), dtype=torch.uint8, device="cuda")
    codes[:2 * M * K].view(torch.float16).copy_(s.view(-1).to(torch.float16))
    if f8:
        codes[2 * M * K:].view(torch.float8_e5m2).copy_(s.view(-1).to(torch.float8_e5m2))
    al = torch.rand((M,), generator=g, device="cuda") * 1e-2 + 1e-3
    zc = torch.full((M,), 0.5, device="cuda")
    y = torch.empty((M, N), dtype=torch.int16, device="cuda")
    call = lambda: tasq.tasq_masked_gemm(ctx, 0, 0, codes, fmt, al, zc, M, pk, N, K, y)
    for _ in range(args.eager):
        call()
    torch.cuda.synchronize()
    out = {"M": M, "N": N, "K": K, "b": args.b, "act_bits": n, "code_format": "fp16+e5m2" if f8 else "fp16"}
    if args.reps:
        gr = torch.cuda.CUDAGraph()
        with torch.cuda.graph(gr, capture_error_mode="thread_local"):
            for _ in range(args.reps):
                call()
        gr.replay()
        torch.cuda.synchronize()
        best = float("inf")
        for _ in range(3):
            t0, t1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            t0.record()
            gr.replay()
            t1.record()
            torch.cuda.synchronize()
            best = min(best, t0.elapsed_time(t1) * 1e3 / args.reps)
        out.update({"us_per_call": best, "tops": 2.0 * M * N * K / (best * 1e-6) / 1e12})
    assert tasq.tasq_device_status(ctx) == tasq.TASQ_OK
    tasq.tasq_destroy(ctx)
    print(json.dumps(out))


if __name__ == "__main__":
    main()
