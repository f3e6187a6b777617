"""Timeline of the tensor-core contraction kernel, for kernel development.

Builds a second copy of the library with -DTASQ_TRACE (per-CTA event times and
per-K-block clock stamps of CTA 0's producer, MMA, converter and epilogue
warps; see the TQ/TE macros in csrc/gemm_tc.cu) into _build/trace/, runs each
given M x N x K linear layer a few times with L2 flushed in between, and prints
where the time goes.  The traced kernels are slower than the product build (the
stamps are global stores); read the cycle counts for their proportions.

    python -m paper_2608_03057_gb300.trace_tc 4096x3456x1152 4096x1152x1152

Needs a GPU.  Not used by the tests or the benchmark.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import sys

import numpy as np

from . import build as B

OUT = os.path.join(B.HERE, "_build", "trace")
EVENTS = ["entry", "setup", "released", "landed", "mma0", "mmaN", "acc0", "accN", "epi", "prod", "exit"]


def build_traced() -> str:
    os.makedirs(OUT, exist_ok=True)
    objs, procs = [], []
    for s in B.SOURCES:
        o = os.path.join(OUT, s.replace(".cu", ".o"))
        objs.append(o)
        procs.append(subprocess.Popen([B.nvcc()] + B._flags(["-DTASQ_TRACE"]) + ["-c", os.path.join(B.CSRC, s),
                                                                                  "-o", o]))
    if not all(p.wait() == 0 for p in procs):
        raise RuntimeError("nvcc failed for the traced build")
    lib = os.path.join(OUT, "libtasq_trace.so")
    subprocess.run([B.nvcc()] + B.ARCH + ["-shared", "-o", lib] + objs, check=True)
    return lib


def _series(name, v):
    v = [int(x) for x in v]
    med = int(np.median(v)) if v else 0
    print(f"  {name:34s} median {med:6d}  {v[:24]}")


def trace_linear(tasq, L, torch, ctx, M, N, K, reps=8):
    g = torch.Generator(device="cuda")
    g.manual_seed(0)
    w = torch.randn(N, K, device="cuda", generator=g) * 0.02
    sw = torch.empty(N, K, dtype=torch.int8, device="cuda")
    cw = torch.empty(N, device="cuda")
    al = torch.empty(N, device="cuda")
    tasq.tasq_quant_weights(ctx, w, tasq.TASQ_F32, N, K, sw, cw, al)
    packed = torch.empty(tasq.tasq_packed_bytes(tasq.TASQ_LINEAR, N, K), dtype=torch.uint8, device="cuda")
    tasq.tasq_pack_weights(ctx, tasq.TASQ_LINEAR, sw, cw, torch.zeros(N, device="cuda"), N, K, 0, packed)
    tasq.tasq_set_schedule(ctx, np.full((1, 1), 8, np.uint8), 1, 1)
    x = (torch.randn(M, K, device="cuda", generator=g)).to(torch.bfloat16)
    codes = torch.empty(M, K, dtype=torch.float16, device="cuda")
    a = torch.empty(M, device="cuda")
    z = torch.empty(M, device="cuda")
    tasq.tasq_quant_act(ctx, x, tasq.TASQ_BF16, M, K, 8, tasq.TASQ_SYMRANGE, tasq.TASQ_PER_TOKEN, codes,
                        tasq.TASQ_CODES_F16, a, z)
    y = torch.empty(M, N, dtype=torch.bfloat16, device="cuda")
    flush = torch.empty(256 << 20, dtype=torch.uint8, device="cuda")
    times = []
    for _ in range(reps):
        flush.zero_()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record()
        tasq.tasq_masked_gemm(ctx, 0, 0, codes, tasq.TASQ_CODES_F16, a, z, M, packed, N, K, y)
        e1.record()
        torch.cuda.synchronize()
        times.append(e0.elapsed_time(e1) * 1e3)
    del flush
    plan = tasq.tasq_plan_tc(tasq.TASQ_LINEAR, M, N, K, 0, 0, 0, 0,
                             torch.cuda.get_device_properties(0).multi_processor_count)
    ev = np.zeros((512, 12, 2), np.uint64)
    assert L.tasq_debug_events(ev.ctypes.data, ev.nbytes) == 0
    nct = min(plan["grid"], ev.shape[0])  # the stamps of earlier, larger launches stay beyond this
    e = ev[:nct].astype(np.int64)
    t0 = e[:, 0, 0].min()
    print(f"== {M} x {N} x {K}: {np.median(times):.2f} us per launch (min {min(times):.2f}), "
          f"{2 * M * N * K / np.median(times) / 1e6:.1f} TOPS; {plan['tile_tokens']}-token tiles, "
          f"{plan['tiles_ch'] * plan['tiles_tok']} tiles, {plan['splits']} slice(s), {nct} CTAs")
    for i, n in enumerate(EVENTS):
        col = e[:, i, 0]
        col = col[col > 0]
        if col.size:
            rel = (col - t0) / 1e3
            print(f"  {n:9s} min {rel.min():7.2f}  median {np.median(rel):7.2f}  max {rel.max():7.2f} us")
    tr = np.zeros((4, 256, 8), np.uint64)
    assert L.tasq_debug_trace(tr.ctypes.data, tr.nbytes) == 0
    tr = tr.astype(np.int64)
    # K blocks of CTA 0 in this launch (stamps beyond them are left from earlier launches)
    kt = -(-K // 128)
    works = plan["tiles_ch"] * plan["tiles_tok"] * plan["splits"]
    nit = min(-(-works // plan["grid"]) * -(-kt // plan["splits"]), tr.shape[1])
    start = tr[1, :nit, 0]
    print(f"  CTA 0: {nit} K blocks (cycles)")
    _series("K-block period (MMA thread)", np.diff(start))
    _series("MMA wait for stage + weights", tr[1, :nit, 1] - tr[1, :nit, 0])
    _series("MMA issue of the block", tr[1, :nit, 2] - tr[1, :nit, 1])
    _series("converter wait for weight tile", tr[2, :nit, 1] - tr[2, :nit, 0])
    _series("converter mask + widen", tr[2, :nit, 2] - tr[2, :nit, 1])
    _series("converter wait for its slot", tr[2, :nit, 3] - tr[2, :nit, 2])
    _series("converter store + signal", tr[2, :nit, 5] - tr[2, :nit, 3])
    _series("MMA sees weights after signal", [tr[1, i, 1] - tr[2, i, 5] for i in range(nit)])
    nu = min(nit * (2 if plan["tile_tokens"] == 256 else 1), tr.shape[1])  # activation stages per K block
    _series("producer wait for a free stage", tr[0, :nu, 1] - tr[0, :nu, 0])
    print()


def main(argv):
    shapes = [tuple(int(v) for v in s.split("x")) for s in argv] or [
        (4096, 3456, 1152), (4096, 1152, 1152), (4096, 1152, 4608), (300, 1152, 1152)]
    lib = build_traced()
    from . import tasq
    tasq.LIB_PATH = lib
    L = tasq.lib()
    for name in ("tasq_debug_events", "tasq_debug_trace", "tasq_debug_fin"):
        f = getattr(L, name)
        f.argtypes = [ctypes.c_void_p, ctypes.c_size_t]
        f.restype = ctypes.c_int
    import torch
    ctx = tasq.tasq_create(0)
    try:
        for M, N, K in shapes:
            trace_linear(tasq, L, torch, ctx, M, N, K)
    finally:
        tasq.tasq_destroy(ctx)


if __name__ == "__main__":
    main(sys.argv[1:])
