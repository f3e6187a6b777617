#!/usr/bin/env python3
"""Benchmark of the TASQ masked-W8A8 path on GB300.

One step = one denoising step of a synthetic backbone: for every quantized
layer, activation quantization (per token; per tensor for a 3x3 conv) and the
masked contraction at that layer's operating precision for the step's stage,
read from the device-resident bit table.  The whole step is captured once as
a CUDA graph; the stage comes from a device int written before each replay,
so a stage switch is a 4-byte write and never a weight copy.

Default workload: the PixArt-Sigma-shaped DiT at 1024 px (224 layers, 4096
image tokens, 300 text tokens, 20 stages, learned-style schedule).  The JSON
line reports throughput in int8-equivalent TOPS (2*M*N*K per layer call,
independent of b), ms per step, the same step under the all-8-bit schedule,
the roofline of the dominant kernel (from a replay of the step's launch
sequence with only its contractions), an end-to-end figure through the C ABI
with host buffers, and the CPU oracle's throughput on a bounded sample.  The
other workloads (SANA-1.6B, SDXL-Turbo, the single 256x1152x1152 layer) are
measured the same way in the same run, under "per_workload".

--impl reference times the CPU oracle (the reference arm of this repository)
on a bounded sample of the same workload, on the host cores.
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import numpy as np

METRIC = "masked W8A8 GEMM TOPS and % int8 tensor peak vs effective bits b; ms/denoise step"

# DRAM bytes (read + write) per masked-contraction launch of one workload, from one
# `ncu --metrics dram__bytes_read.sum,dram__bytes_write.sum` capture of the
# contraction kernel.  It describes only the kernel sources it was measured on,
# identified by their SHA-256; after any change to them the field reads null until
# the capture is repeated.
TRAFFIC = {"pixart": {"bytes_per_launch": 15386843,
                      "sources_sha256": "d16ec13a0670875b9b251ee9d216646ab80f59dbf378476f7fdc700d0ada32ac"}}
KERNEL_SOURCES = ("gemm_tc.cu", "tc_ptx.cuh", "tasq_internal.cuh")


def kernel_sources_sha256() -> str:
    import hashlib
    h = hashlib.sha256()
    here = os.path.join(os.path.dirname(os.path.abspath(__file__)), "paper_2608_03057_gb300", "csrc")
    for f in KERNEL_SOURCES:
        with open(os.path.join(here, f), "rb") as fh:
            h.update(fh.read())
    return h.hexdigest()


def measured_traffic(workload: str):
    """DRAM bytes per contraction launch from the recorded ncu capture of this
    workload, or None when there is none or the kernel sources have changed since."""
    tr = TRAFFIC.get(workload)
    return tr["bytes_per_launch"] if tr and tr["sources_sha256"] == kernel_sources_sha256() else None


UNIT = "TOPS"
# Units of the step (layers that read one input: one quantization, one contraction call).
GROUPINGS = {
    "text": "every layer that reads the text tokens (the key and value projections of all cross-attention "
            "blocks) in one unit per shape, first in the step: one quantization and one contraction launch "
            "with the member list in device memory, each layer at its own b",
    "pairs": "a cross-attention's key and value projections read one input: one quantization and one grouped "
             "contraction, each layer at its own b",
    "none": "every layer its own quantization and contraction",
}
WORKLOAD_NAMES = {
    "pixart": "pixart_sigma_1024px_denoise_step",
    "pixart_a4": "pixart_sigma_1024px_denoise_step_a4_w4a4_budget",
    "pixart_lr": "pixart_sigma_1024px_denoise_step_with_rank32_lowrank_branch",
    "sana": "sana_1600m_1024px_denoise_step",
    "sdxl": "sdxl_turbo_512px_denoise_step",
    "single": "single_linear_256x1152x1152",
}


def parse_args():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=100)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--workload", choices=list(WORKLOAD_NAMES), default="pixart")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--e2e-copy-streams", type=int, default=1,
                    help="copy streams per direction in the end-to-end step (layers take them in turn)")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--cpu-seconds", type=float, default=12.0, help="CPU oracle sample budget")
    ap.add_argument("--seed", type=int, default=0)
    ap.add_argument("--blocks", type=int, default=0, help="keep only the first N transformer blocks (small cases)")
    ap.add_argument("--no-all8", action="store_true", help="skip the all-8-bit schedule comparison")
    ap.add_argument("--no-sweep", action="store_true", help="skip the GEMM sweep and the stage-switch test")
    ap.add_argument("--no-per-workload", action="store_true",
                    help="time only --workload, not the other workloads of the suite")
    ap.add_argument("--grouping", choices=list(GROUPINGS), default="text",
                    help="which layers share one quantization and one contraction launch")
    return ap.parse_args()


def load_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        d = json.load(open(p))
        return dict(hbm=d.get("hbm_gbs", 6800.0), bf16=d.get("bf16_tflops", 1900.0),
                    bf16_sus=d.get("bf16_tflops_sustained", 1700.0), src="measured")
    return dict(hbm=6800.0, bf16=1900.0, bf16_sus=1700.0, src="fallback")


# ------------------------------------------------------------------ clocks --
class ClockSampler:
    """nvidia-smi sampling of SM clock and throttle reasons during a region."""
    Q = ("index,clocks.sm,clocks.max.sm,power.draw,utilization.gpu,clocks_event_reasons.active,"
         "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index: int):
        self.index = index
        self.proc = None
        self.out = None

    def start(self):
        try:
            self.proc = subprocess.Popen(["nvidia-smi", "-i", str(self.index), f"--query-gpu={self.Q}",
                                          "--format=csv,noheader,nounits", "-lms", "50"],
                                         stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except OSError:
            self.proc = None
        time.sleep(0.3)

    def stop(self):
        if not self.proc:
            return None
        time.sleep(0.1)
        self.proc.terminate()
        try:
            out, _ = self.proc.communicate(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
            out, _ = self.proc.communicate()
        rows = []
        for line in out.strip().splitlines():
            f = [x.strip() for x in line.split(",")]
            if len(f) < 10:
                continue
            try:
                rows.append(dict(sm=float(f[1]), smax=float(f[2]), util=float(f[4]), hw=f[6], hwt=f[7], swt=f[8],
                                 swp=f[9]))
            except ValueError:
                continue
        if not rows:
            return None
        load = [r for r in rows if r["util"] >= 50] or rows
        reasons = set()
        for r in load:
            for key, name in (("hw", "hw_slowdown"), ("hwt", "hw_thermal_slowdown"), ("swt", "sw_thermal_slowdown"),
                              ("swp", "sw_power_cap")):
                if r[key].lower().startswith("active"):
                    reasons.add(name)
        return {"sm_mhz": statistics.median(r["sm"] for r in load), "sm_max_mhz": max(r["smax"] for r in load),
                "reasons": sorted(reasons), "samples": len(load)}


# --------------------------------------------------------------- workload --
class Step:
    """Device-resident workload of one denoising step and its launch sequence.

    The step runs unit by unit: a unit is the layers that read one input.  With
    grouping "text" (the default) every layer that reads the text tokens -- the key
    and value projections of all cross-attention blocks -- is in one unit per shape,
    first in the step, contracted by tasq_masked_gemm_shared_input; with "pairs" each
    cross-attention's key and value projections form a unit (tasq_masked_gemm_grouped);
    every other layer is a unit alone.  A unit's input is quantized once and
    contracted by one call, at each member layer's own precision from the bit table.
    Every layer keeps its own row of the table."""

    def __init__(self, torch, tasq, workloads, name: str, seed: int, blocks: int = 0, grouping="text"):
        self.torch, self.tasq = torch, tasq
        self.layers = workloads.inventory(name)
        self.table = workloads.schedule_for(name, len(self.layers))
        # activation precision; at n <= 4 the codes also come as e5m2 bytes, so that
        # linear contractions at b <= 4 run on the 8-bit-float tensor-core kind
        self.act_bits = workloads.ACT_BITS.get(name, 8)
        self.code_fmt = tasq.TASQ_CODES_F16_E5M2 if self.act_bits <= 4 else tasq.TASQ_CODES_F16
        # 16-bit low-rank branch beside every linear layer: one call per layer
        self.rank = workloads.LOWRANK.get(name, 0)
        if self.rank:
            grouping = "none"
        self.grouping = grouping
        if blocks:
            keep = len(workloads.inventory_blocks(name, blocks))
            self.layers, self.table = self.layers[:keep], np.ascontiguousarray(self.table[:keep])
        if grouping == "text":
            self.units = workloads.shared_input_units(self.layers)
        elif grouping == "pairs":
            self.units = workloads.input_groups(self.layers)
        else:
            self.units = [[i] for i in range(len(self.layers))]
        # units contracted with the member list in device memory
        self.d_layers = [torch.tensor(unit, dtype=torch.int32, device="cuda") if grouping == "text" and len(unit) > 1
                         else None for unit in self.units]
        self.S = self.table.shape[1]
        self.ctx = tasq.tasq_create(torch.cuda.current_device())
        tasq.tasq_set_schedule(self.ctx, self.table, len(self.layers), self.S)
        dev = "cuda"
        self.packed, self.x, self.y = [], [], []
        max_mk = max(l.M * (l.Cin if l.Cin else l.K) for l in self.layers)
        max_m = max(l.M for l in self.layers)
        self.codes = torch.empty((max_mk * (3 if self.act_bits <= 4 else 2) // 2,), dtype=torch.float16, device=dev)
        self.alpha = torch.empty((max_m,), dtype=torch.float32, device=dev)
        self.zc = torch.empty((max_m,), dtype=torch.float32, device=dev)
        self.l1, self.l2 = [], []
        if self.rank:
            self.u = torch.empty((max_m, 64), dtype=torch.int16, device=dev)  # u' rows of 64 fp16
        for unit in self.units:
            l = self.layers[unit[0]]
            N = sum(self.layers[i].N for i in unit)
            # each member's weights and bias from its own seed, stacked along N
            w = torch.cat([workloads.device_normal((self.layers[i].N, l.K), seed * 100003 + 2 * i + 1, 0.02)
                           for i in unit])
            bias = torch.cat([workloads.device_normal((self.layers[i].N,), seed * 100003 + 2 * i + 2, 0.02)
                              for i in unit])
            sw = torch.empty((N, l.K), dtype=torch.int8, device=dev)
            cw = torch.empty((N,), dtype=torch.float32, device=dev)
            tasq.tasq_quant_weights(self.ctx, w, tasq.TASQ_F32, N, l.K, sw, cw)
            kind = tasq.TASQ_CONV3X3 if l.kind == workloads.CONV3X3 else tasq.TASQ_LINEAR
            pk = torch.empty((tasq.tasq_packed_bytes(kind, N, l.K),), dtype=torch.uint8, device=dev)
            tasq.tasq_pack_weights(self.ctx, kind, sw, cw, bias, N, l.K, l.Cin, pk)
            self.packed.append(pk)
            xs = (l.B, l.H, l.W, l.Cin) if l.kind == workloads.CONV3X3 else (l.M, l.K)
            self.x.append(workloads.device_normal(xs, seed * 100003 + 1000003 + unit[0], 1.0, torch.bfloat16))
            self.y.append(torch.empty((l.M, N), dtype=torch.int16, device=dev))
            if self.rank and l.kind != workloads.CONV3X3:
                # the branch's factors (bf16 bits): l2 [rank][K] and l1 [N][rank]
                i = unit[0]
                self.l2.append(workloads.device_normal((self.rank, l.K), seed * 100003 + 3000003 + i, 0.05,
                                                       torch.bfloat16).view(torch.int16))
                self.l1.append(workloads.device_normal((N, self.rank), seed * 100003 + 4000003 + i, 0.05,
                                                       torch.bfloat16).view(torch.int16))
            else:
                self.l1.append(None)
                self.l2.append(None)
            del w, sw, cw, bias
        self.d_stage = torch.zeros((4,), dtype=torch.int32, device=dev)
        tasq.tasq_set_stage_device(self.ctx, self.d_stage)
        torch.cuda.synchronize()
        self.ops = sum(l.ops for l in self.layers)
        self.gemm_ops = [l.ops for l in self.layers]
        self.conv = workloads.CONV3X3

    def launch(self, parts=("quant", "gemm")):
        """Enqueue one step on the current stream (stage read from d_stage).
        parts: which kernels of each unit to enqueue (the quantization, the
        contraction, or both, in the step's order)."""
        for u in range(len(self.units)):
            self.launch_unit(u, parts)

    def launch_unit(self, u, parts=("quant", "gemm")):
        """Enqueue unit u (one quantization + one masked contraction) on the current stream."""
        t = self.tasq
        unit = self.units[u]
        l = self.layers[unit[0]]
        N = self.y[u].shape[1]
        conv = l.kind == self.conv
        if "quant" in parts:
            gran = t.TASQ_PER_TENSOR if conv else t.TASQ_PER_TOKEN
            t.tasq_quant_act(self.ctx, self.x[u], t.TASQ_BF16, l.M, l.Cin if conv else l.K, self.act_bits,
                             t.TASQ_SYMRANGE, gran, self.codes, self.code_fmt, self.alpha, self.zc)
        if "gemm" in parts:
            if conv:
                t.tasq_masked_conv3x3(self.ctx, unit[0], -1, self.codes, self.code_fmt, self.alpha, self.zc, l.B,
                                      l.H, l.W, l.Cin, self.packed[u], N, self.y[u], None)
            elif self.l1[u] is not None:
                # the low-rank branch: its down-projection of this input, then the layer
                t.tasq_lowrank_down(self.ctx, self.x[u], t.TASQ_BF16, l.M, l.K, self.l2[u], self.rank, self.alpha,
                                    self.u)
                t.tasq_masked_gemm_lr(self.ctx, unit[0], -1, self.codes, self.code_fmt, self.alpha, self.zc, l.M,
                                      self.packed[u], N, l.K, self.u, self.l1[u], self.rank, self.y[u], None)
            elif self.d_layers[u] is not None:
                t.tasq_masked_gemm_shared_input(self.ctx, self.d_layers[u], len(unit), -1, self.codes, self.code_fmt,
                                                self.alpha, self.zc, l.M, self.packed[u], N, l.K, self.y[u], None)
            elif len(unit) == 1:
                t.tasq_masked_gemm(self.ctx, unit[0], -1, self.codes, self.code_fmt, self.alpha, self.zc, l.M,
                                   self.packed[u], N, l.K, self.y[u], None)
            else:
                t.tasq_masked_gemm_grouped(self.ctx, unit, -1, self.codes, self.code_fmt, self.alpha, self.zc,
                                           l.M, self.packed[u], N, l.K, self.y[u], None)

    def launches_per_step(self):
        """Kernels the library enqueues for one step, counted by the library itself
        (one eager launch of the step, outside any timed region)."""
        if not hasattr(self, "_launches"):
            before = self.tasq.tasq_kernel_count(self.ctx)
            self.launch()
            self.torch.cuda.synchronize()
            self._launches = self.tasq.tasq_kernel_count(self.ctx) - before
        return self._launches

    def _unit_shapes(self):
        for u, unit in enumerate(self.units):
            l = self.layers[unit[0]]
            yield l, (l.Cin if l.Cin else l.K), self.y[u].shape[1]

    def act_bytes(self):
        """Algorithmic HBM bytes of activation quantization per step: bf16 in,
        one byte per code out (an int8 code; the tensor-core route holds it in
        fp16, which doubles the bytes actually written), 8 bytes of scales per
        token (per-tensor: per tensor)."""
        return sum(l.M * k_in * 3 + 8 * l.M for l, k_in, _ in self._unit_shapes())

    def gemm_bytes(self):
        """Algorithmic HBM bytes of the contractions per step: int8 activation codes
        (M K), int8 weights (N K), bf16 output (2 M N), per-token scales (8 M) and
        per-channel scale, bias and the seven row sums (4 N (2 + 7))."""
        return sum(l.M * k_in + N * l.K + 2 * l.M * N + 8 * l.M + 36 * N for l, k_in, N in self._unit_shapes())

    def close(self):
        self.tasq.tasq_destroy(self.ctx)


def capture(torch, step, parts=("quant", "gemm")):
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, capture_error_mode="thread_local"):
        step.launch(parts)
    return g


def f8_op_share(tasq, step, steps, stage_of, num_sms):
    """Share of a step's int8-equivalent ops that run on the 8-bit-float route,
    over the stages of `steps` timed replays: linear units with e5m2 codes whose
    members are all at b <= 4, in unsplit launches (the route's conditions)."""
    if step.code_fmt != tasq.TASQ_CODES_F16_E5M2:
        return 0.0
    f8 = tot = 0.0
    for k in range(steps):
        s = stage_of(k)
        for u, unit in enumerate(step.units):
            l = step.layers[unit[0]]
            ops = sum(step.layers[i].ops for i in unit)
            tot += ops
            if l.kind == step.conv or any(int(step.table[i, s]) > 4 for i in unit):
                continue
            plan = tasq.tasq_plan_tc(tasq.TASQ_LINEAR, l.M, step.y[u].shape[1], l.K, 0, 0, 0, 0, num_sms)
            if plan["splits"] == 1 or step.d_layers[u] is not None:  # (member lists in device memory: unsplit)
                f8 += ops
    return f8 / tot if tot else 0.0


def timed_replays(torch, g, step, steps, stage_of):
    s = torch.cuda.current_stream()
    t0 = torch.cuda.Event(enable_timing=True)
    t1 = torch.cuda.Event(enable_timing=True)
    torch.cuda.synchronize()
    t0.record(s)
    for k in range(steps):
        step.d_stage.fill_(stage_of(k))
        g.replay()
    t1.record(s)
    torch.cuda.synchronize()
    return t0.elapsed_time(t1) / steps


# ------------------------------------------------------------------ sweep --
def run_sweep(torch, tasq, workloads, shapes=None, reps=10, seed=0):
    """GEMM sweep: M x (K = N) x b = 2..8 on seeded uniform codes in [-127, 127];
    TOPS (2*M*N*K per call, independent of b) per point.  Also the stage-switch
    cost: 1000 back-to-back calls alternating the stage every call versus 1000
    calls at one stage."""
    ctx = tasq.tasq_create(torch.cuda.current_device())
    table = workloads.schedule_for("sweep", 1)  # stages 0..6 <-> b = 2..8, stage 7 = 8
    tasq.tasq_set_schedule(ctx, table, 1, table.shape[1])
    out = []
    switch = None
    shapes = shapes or list(workloads.sweep_shapes())
    for si, (M, KN) in enumerate(shapes):
        N = K = KN
        g = torch.Generator(device="cuda")
        g.manual_seed(seed * 1000 + si)
        sw = torch.randint(-127, 128, (N, K), generator=g, device="cuda", dtype=torch.int8)
        cw = torch.rand((N,), generator=g, device="cuda") * 1e-3 + 1e-4
        pk = torch.empty((tasq.tasq_packed_bytes(tasq.TASQ_LINEAR, N, K),), dtype=torch.uint8, device="cuda")
        tasq.tasq_pack_weights(ctx, tasq.TASQ_LINEAR, sw, cw, None, N, K, 0, pk)
        codes = torch.randint(-127, 128, (M, K), generator=g, device="cuda", dtype=torch.int8).to(torch.float16)
        al = torch.rand((M,), generator=g, device="cuda") * 1e-2 + 1e-3
        zc = torch.full((M,), 0.5, device="cuda")
        y = torch.empty((M, N), dtype=torch.int16, device="cuda")
        row = {"M": M, "K": K, "N": N, "tops_by_b": {}}
        for b in range(2, 9):
            stage = b - 2
            tasq.tasq_masked_gemm(ctx, 0, stage, codes, tasq.TASQ_CODES_F16, al, zc, M, pk, N, K, y)
            gr = torch.cuda.CUDAGraph()
            with torch.cuda.graph(gr, capture_error_mode="thread_local"):
                for _ in range(reps):
                    tasq.tasq_masked_gemm(ctx, 0, stage, codes, tasq.TASQ_CODES_F16, al, zc, M, pk, N, K, y)
            gr.replay()
            torch.cuda.synchronize()
            t0, t1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            t0.record()
            gr.replay()
            t1.record()
            torch.cuda.synchronize()
            us = t0.elapsed_time(t1) * 1e3 / reps
            row["tops_by_b"][b] = 2.0 * M * N * K / (us * 1e-6) / 1e12
        out.append(row)
        if (M, KN) == (4096, 4096):
            # stage switch: alternate b = 2 / 8 every call, and b = 5 / 5 (same
            # precision, different stage) every call, against one fixed stage
            def timed(stages):
                gr = torch.cuda.CUDAGraph()
                with torch.cuda.graph(gr, capture_error_mode="thread_local"):
                    for st in stages:
                        tasq.tasq_masked_gemm(ctx, 0, st, codes, tasq.TASQ_CODES_F16, al, zc, M, pk, N, K, y)
                gr.replay()
                torch.cuda.synchronize()
                t0, t1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                t0.record()
                gr.replay()
                t1.record()
                torch.cuda.synchronize()
                return t0.elapsed_time(t1) * 1e3 / len(stages)
            n = 1000
            fixed8 = timed([6] * n)
            alt = timed([0 if i % 2 == 0 else 6 for i in range(n)])
            fixed2 = timed([0] * n)
            same_b = timed([6 if i % 2 == 0 else 7 for i in range(n)])  # stages 6 and 7 both hold b = 8
            switch = {"shape": [M, N, K], "calls": n, "us_per_call_fixed_b8": fixed8, "us_per_call_fixed_b2": fixed2,
                      "us_per_call_alternating_b2_b8": alt, "us_per_call_alternating_stages_same_b8": same_b,
                      "switch_overhead_us": same_b - fixed8}
        del sw, cw, pk, codes, al, zc, y
    tasq.tasq_destroy(ctx)
    return out, switch


def run_sweep_a4(torch, tasq, workloads, shapes=((4096, 4096), (16384, 4096), (4096, 1152)), reps=10, seed=0):
    """The shape sweep with 4-bit activation codes (uniform in [-8, 7]) in the dual
    fp16 + e5m2 storage: b <= 4 runs the K loop on the e5m2 tensor-core kind, b >= 5
    on the fp16 codes.  TOPS (2 M N K per call) per b."""
    ctx = tasq.tasq_create(torch.cuda.current_device())
    table = workloads.schedule_for("sweep", 1)  # stages 0..6 <-> b = 2..8
    tasq.tasq_set_schedule(ctx, table, 1, table.shape[1])
    F8 = tasq.TASQ_CODES_F16_E5M2
    out = []
    for si, (M, KN) in enumerate(shapes):
        N = K = KN
        g = torch.Generator(device="cuda")
        g.manual_seed(seed * 1000 + 300 + si)
        sw = torch.randint(-127, 128, (N, K), generator=g, device="cuda", dtype=torch.int8)
        cw = torch.rand((N,), generator=g, device="cuda") * 1e-3 + 1e-4
        pk = torch.empty((tasq.tasq_packed_bytes(tasq.TASQ_LINEAR, N, K),), dtype=torch.uint8, device="cuda")
        tasq.tasq_pack_weights(ctx, tasq.TASQ_LINEAR, sw, cw, None, N, K, 0, pk)
        s = torch.randint(-8, 8, (M, K), generator=g, device="cuda", dtype=torch.int8)
        codes = torch.empty((3 * M * K,), dtype=torch.uint8, device="cuda")
        codes[:2 * M * K].view(torch.float16).copy_(s.view(-1).to(torch.float16))
        codes[2 * M * K:].view(torch.float8_e5m2).copy_(s.view(-1).to(torch.float8_e5m2))
        al = torch.rand((M,), generator=g, device="cuda") * 1e-2 + 1e-3
        zc = torch.full((M,), 0.5, device="cuda")
        y = torch.empty((M, N), dtype=torch.int16, device="cuda")
        row = {"M": M, "K": K, "N": N, "act_bits": 4, "tops_by_b": {}}
        for b in range(2, 9):
            stage = b - 2
            call = lambda: tasq.tasq_masked_gemm(ctx, 0, stage, codes, F8, al, zc, M, pk, N, K, y)
            call()
            gr = torch.cuda.CUDAGraph()
            with torch.cuda.graph(gr, capture_error_mode="thread_local"):
                for _ in range(reps):
                    call()
            gr.replay()
            torch.cuda.synchronize()
            t0, t1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            t0.record()
            gr.replay()
            t1.record()
            torch.cuda.synchronize()
            us = t0.elapsed_time(t1) * 1e3 / reps
            row["tops_by_b"][b] = 2.0 * M * N * K / (us * 1e-6) / 1e12
        out.append(row)
        del sw, cw, pk, s, codes, al, zc, y
    assert tasq.tasq_device_status(ctx) == tasq.TASQ_OK
    tasq.tasq_destroy(ctx)
    return out


def int8_tensor_peak(torch, n=8192, reps=20):
    """Measured int8 tensor-core peak of this GPU from the library int8 GEMM
    (torch._int_mm, cuBLASLt s8 x s8 -> s32) on n^3: 2 n^3 / t in TOPS."""
    try:
        a = torch.randint(-127, 128, (n, n), dtype=torch.int8, device="cuda")
        b = torch.randint(-127, 128, (n, n), dtype=torch.int8, device="cuda")
        for _ in range(3):
            torch._int_mm(a, b)
        torch.cuda.synchronize()
        t0, t1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        t0.record()
        for _ in range(reps):
            torch._int_mm(a, b)
        t1.record()
        torch.cuda.synchronize()
        ms = t0.elapsed_time(t1) / reps
        del a, b
        return {"tops": 2.0 * n ** 3 / (ms * 1e-3) / 1e12, "shape": [n, n, n],
                "source": "torch._int_mm (cuBLASLt int8 GEMM), CUDA events, 20 back-to-back calls"}
    except (RuntimeError, AttributeError) as exc:  # no int8 GEMM in this torch build
        return {"tops": None, "source": f"unavailable: {exc}"}


def s8_route_tops(torch, tasq, workloads, n=4096, reps=10):
    """The library's own int8 route (warp-level mma.sync s8, TASQ_CODES_S8) on an
    n^3 masked contraction at b = 8, for comparison with the tensor-core route."""
    ctx = tasq.tasq_create(torch.cuda.current_device())
    table = workloads.schedule_for("sweep", 1)
    tasq.tasq_set_schedule(ctx, table, 1, table.shape[1])
    g = torch.Generator(device="cuda")
    g.manual_seed(7)
    sw = torch.randint(-127, 128, (n, n), generator=g, device="cuda", dtype=torch.int8)
    cw = torch.rand((n,), generator=g, device="cuda") * 1e-3 + 1e-4
    pk = torch.empty((tasq.tasq_packed_bytes(tasq.TASQ_LINEAR, n, n),), dtype=torch.uint8, device="cuda")
    tasq.tasq_pack_weights(ctx, tasq.TASQ_LINEAR, sw, cw, None, n, n, 0, pk)
    codes = torch.randint(-127, 128, (n, n), generator=g, device="cuda", dtype=torch.int8)
    al = torch.rand((n,), generator=g, device="cuda") * 1e-2 + 1e-3
    zc = torch.full((n,), 0.5, device="cuda")
    y = torch.empty((n, n), dtype=torch.int16, device="cuda")
    call = lambda: tasq.tasq_masked_gemm(ctx, 0, 6, codes, tasq.TASQ_CODES_S8, al, zc, n, pk, n, n, y)
    call()
    torch.cuda.synchronize()
    t0, t1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    t0.record()
    for _ in range(reps):
        call()
    t1.record()
    torch.cuda.synchronize()
    ms = t0.elapsed_time(t1) / reps
    tasq.tasq_destroy(ctx)
    return {"shape": [n, n, n], "b": 8, "tops": 2.0 * n ** 3 / (ms * 1e-3) / 1e12}


def run_small_m_weight_bytes(torch, tasq, shapes=((300, 1152, 1152), (300, 2304, 1152), (77, 1280, 2048),
                                                  (256, 1280, 1280)), layers=128, seed=0):
    """How much of a small-M contraction's time is reading its weights from HBM:
    each shape (b = 3, 64-token tiles) as a CUDA graph of `layers` back-to-back
    calls, either all on one packed layer (its weights stay in L2) or each on a
    different packed layer of the same shape (`layers` x N x K bytes, more than
    L2 holds, so every call reads its weights from HBM); the activation codes are
    the same buffer in both.  A layout that streams only the selected weight
    planes (e.g. hi/lo-nibble planes, half the bytes at b <= 4) could save at
    most half of the difference per call."""
    ctx = tasq.tasq_create(torch.cuda.current_device())
    tasq.tasq_set_schedule(ctx, np.array([[3]] * layers, np.uint8), layers, 1)
    out = []
    for si, (M, N, K) in enumerate(shapes):
        g = torch.Generator(device="cuda")
        g.manual_seed(seed * 1000 + 700 + si)
        nbytes = tasq.tasq_packed_bytes(tasq.TASQ_LINEAR, N, K)
        pks = []
        for _ in range(layers):
            sw = torch.randint(-127, 128, (N, K), generator=g, device="cuda", dtype=torch.int8)
            cw = torch.rand((N,), generator=g, device="cuda") * 1e-3 + 1e-4
            pk = torch.empty((nbytes,), dtype=torch.uint8, device="cuda")
            tasq.tasq_pack_weights(ctx, tasq.TASQ_LINEAR, sw, cw, None, N, K, 0, pk)
            pks.append(pk)
            del sw, cw
        codes = torch.randint(-127, 128, (M, K), generator=g, device="cuda", dtype=torch.int8).to(torch.float16)
        al = torch.rand((M,), generator=g, device="cuda") * 1e-2 + 1e-3
        zc = torch.full((M,), 0.5, device="cuda")
        y = torch.empty((M, N), dtype=torch.int16, device="cuda")

        def graph_us(which):
            def seq():
                for i in range(layers):
                    j = which(i)
                    tasq.tasq_masked_gemm(ctx, j, 0, codes, tasq.TASQ_CODES_F16, al, zc, M, pks[j], N, K, y)
            seq()
            gr = torch.cuda.CUDAGraph()
            with torch.cuda.graph(gr, capture_error_mode="thread_local"):
                seq()
            best = None
            for _ in range(4):
                gr.replay()
                torch.cuda.synchronize()
                t0, t1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                t0.record()
                gr.replay()
                t1.record()
                torch.cuda.synchronize()
                us = t0.elapsed_time(t1) * 1e3 / layers
                best = us if best is None else min(best, us)
            return best

        warm = graph_us(lambda i: 0)
        cold = graph_us(lambda i: i)
        out.append({"M": M, "N": N, "K": K, "b": 3, "weight_bytes": N * K, "us_weights_in_l2": warm,
                    "us_weights_from_hbm": cold, "max_saving_us_half_weight_bytes": max(0.0, cold - warm) / 2})
        del pks, codes, al, zc, y
    tasq.tasq_destroy(ctx)
    return out


def run_zero_point(torch, tasq, workloads, shapes=((4096, 1152, 1152), (4096, 3456, 1152), (300, 1152, 1152)),
                   reps=20, seed=0):
    """Asymmetric weights (App. A.1.1 on each channel's [min, max], a real zero
    point per channel) against the symmetric reading on the same layer shapes:
    per-call time of the activation quantization (with / without the per-token
    code sums) and of the contraction (four-term / two-term epilogue), CUDA
    graphs of `reps` back-to-back calls, b = 5."""
    ctx = tasq.tasq_create(torch.cuda.current_device())
    table = workloads.schedule_for("sweep", 1)  # stage 3 <-> b = 5
    tasq.tasq_set_schedule(ctx, table, 1, table.shape[1])
    stage = 3

    def graph_us(fn):
        fn()
        gr = torch.cuda.CUDAGraph()
        with torch.cuda.graph(gr, capture_error_mode="thread_local"):
            for _ in range(reps):
                fn()
        gr.replay()
        torch.cuda.synchronize()
        t0, t1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        t0.record()
        gr.replay()
        t1.record()
        torch.cuda.synchronize()
        return t0.elapsed_time(t1) * 1e3 / reps

    out = []
    for si, (M, N, K) in enumerate(shapes):
        g = torch.Generator(device="cuda")
        g.manual_seed(seed * 1000 + 500 + si)
        w = torch.randn((N, K), generator=g, device="cuda") * 0.02
        w[::2] += 0.02  # skewed channels
        x = torch.randn((M, K), generator=g, device="cuda").to(torch.bfloat16)
        sw = torch.empty((N, K), dtype=torch.int8, device="cuda")
        cw = torch.empty((N,), device="cuda")
        zcw = torch.empty((N,), device="cuda")
        nbytes = tasq.tasq_packed_bytes(tasq.TASQ_LINEAR, N, K)
        pk_sym = torch.empty((nbytes,), dtype=torch.uint8, device="cuda")
        pk_zp = torch.empty((nbytes,), dtype=torch.uint8, device="cuda")
        tasq.tasq_quant_weights(ctx, w, tasq.TASQ_F32, N, K, sw, cw)
        tasq.tasq_pack_weights(ctx, tasq.TASQ_LINEAR, sw, cw, None, N, K, 0, pk_sym)
        tasq.tasq_quant_weights_asym(ctx, w, tasq.TASQ_F32, N, K, sw, cw, zcw)
        tasq.tasq_pack_weights_zp(ctx, tasq.TASQ_LINEAR, sw, cw, zcw, None, N, K, 0, pk_zp)
        codes = torch.empty((M, K), dtype=torch.float16, device="cuda")
        al = torch.empty((M,), device="cuda")
        zc = torch.empty((M,), device="cuda")
        sums = torch.empty((M,), dtype=torch.int32, device="cuda")
        y = torch.empty((M, N), dtype=torch.int16, device="cuda")
        q_sym = graph_us(lambda: tasq.tasq_quant_act(ctx, x, tasq.TASQ_BF16, M, K, 8, tasq.TASQ_SYMRANGE,
                                                     tasq.TASQ_PER_TOKEN, codes, tasq.TASQ_CODES_F16, al, zc))
        q_zp = graph_us(lambda: tasq.tasq_quant_act_sums(ctx, x, tasq.TASQ_BF16, M, K, 8, tasq.TASQ_SYMRANGE,
                                                         tasq.TASQ_PER_TOKEN, codes, tasq.TASQ_CODES_F16, al, zc, sums))
        g_sym = graph_us(lambda: tasq.tasq_masked_gemm(ctx, 0, stage, codes, tasq.TASQ_CODES_F16, al, zc, M, pk_sym,
                                                       N, K, y))
        g_zp = graph_us(lambda: tasq.tasq_masked_gemm_zp(ctx, 0, stage, codes, tasq.TASQ_CODES_F16, al, zc, sums, M,
                                                         pk_zp, N, K, y))
        out.append({"M": M, "N": N, "K": K, "b": 5, "quant_us_symmetric": q_sym, "quant_us_with_code_sums": q_zp,
                    "contraction_us_symmetric": g_sym, "contraction_us_zero_point": g_zp,
                    "contraction_tops_zero_point": 2.0 * M * N * K / (g_zp * 1e-6) / 1e12})
        del w, x, sw, cw, zcw, pk_sym, pk_zp, codes, al, zc, sums, y
    tasq.tasq_destroy(ctx)
    return out


# ------------------------------------------------------------ CPU oracle --
def oracle_sample(workload: str, budget_s: float, rows: int = 32, seed: int = 0, max_layers=None, threads=0):
    """Time the CPU oracle (act quant, int32 contraction, row sums, fp32
    epilogue) on `rows` token rows of successive layers of the workload until
    the budget is spent, on `threads` OpenMP threads (0: every core).
    Returns (ops, seconds, layers_done, rows, threads)."""
    from oracle import oracle
    from paper_2608_03057_gb300 import workloads

    layers = workloads.inventory(workload)
    table = workloads.schedule_for(workload, len(layers))
    oracle.build()
    oracle.set_threads(threads)
    ops = 0
    spent = 0.0
    done = 0
    for i, l in enumerate(layers):
        if (max_layers is not None and done >= max_layers) or spent >= budget_s:
            break
        w = workloads.normal((l.N, l.K), seed + 2 * i + 1, 0.02)
        wq = oracle.quant_weight(w)
        b = int(table[i, 0])
        if l.kind == workloads.CONV3X3:
            # `rows` 3x3 images: 9 output pixels each with 4 (corner), 6 (edge) or 9 valid taps
            x = workloads.normal((rows, 3, 3, l.Cin), seed + 7 * i + 3)
            t0 = time.perf_counter()
            s_x, a, z = oracle.quant_act(x.reshape(1, -1), 8, oracle.SYMRANGE, oracle.PER_TOKEN)
            acc, rs = oracle.conv3x3(s_x.reshape(rows, 3, 3, l.Cin), wq["s"], b)
            oracle.epilogue_f32(acc, a, z, rs, wq["c"], None, per_tensor=True, rs_per_row=True)
            spent += time.perf_counter() - t0
            ops += 2 * rows * (4 * 4 + 4 * 6 + 9) * l.Cin * l.N
        else:
            x = workloads.normal((rows, l.K), seed + 7 * i + 3)
            t0 = time.perf_counter()
            oracle.linear_layer(x, wq["s"], wq["c"], None, b)
            spent += time.perf_counter() - t0
            ops += 2 * rows * l.N * l.K
        done += 1
    return ops, spent, done, rows, oracle.threads()


def run_reference(args):
    if dist_env()[1] != 0:  # under torchrun only rank 0 times the oracle
        return 0
    # warm-up samples, then K timed samples of one layer-row block each
    per_step = max(0.5, min(5.0, 60.0 / max(1, args.steps + args.warmup)))
    for _ in range(args.warmup):
        oracle_sample(args.workload, per_step / 4, seed=args.seed)
    ops = secs = 0.0
    layers_done = 0
    threads = 1
    rows = 32
    for k in range(args.steps):
        o, s, d, rows, threads = oracle_sample(args.workload, per_step, seed=args.seed + k)
        ops += o
        secs += s
        layers_done += d
    value = ops / secs / 1e12
    sample = (f"{rows} token rows x the first layers of the {WORKLOAD_NAMES[args.workload]} inventory per step "
              f"({layers_done} layer calls in {args.steps} steps, ~{per_step:.1f} s each); act quant + int32 "
              f"contraction + fp32 epilogue")
    line = {"metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": secs * 1e3 / args.steps, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "int8", "data": "synthetic",
            "config": {"workload": WORKLOAD_NAMES[args.workload], "sample": "bounded CPU sample"},
            "impl": "reference",
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": threads, "kind": "oracle", "sample": sample},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)
    return 0


# ------------------------------------------------- replicas over N GPUs --
def dist_env():
    """(world, rank, local_rank) from the launcher's environment (1, 0, 0 alone)."""
    return (int(os.environ.get("WORLD_SIZE", "1")), int(os.environ.get("RANK", "0")),
            int(os.environ.get("LOCAL_RANK", "0")))


def max_over_ranks(torch, dist, value: float, device) -> float:
    """The largest of every rank's `value` (each rank calls it; no-op alone)."""
    if dist is None:
        return value
    t = torch.tensor([value], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_tops(ops_per_rank: float, world: int, ms: float) -> float:
    """Whole-job throughput: every rank runs an independent replica of the step
    (weak scaling), so the job does world x the ops in the slowest rank's time."""
    return world * ops_per_rank / (ms * 1e-3) / 1e12


# ------------------------------------------------------------------- main --
# Denoising steps of the trajectory each workload's stages partition (stage of
# step t = floor(t S / T), stage 0 the noisiest): 20 for the DiTs, 4 for the
# distilled UNet; the single layer runs its 4 stages once each.
TRAJECTORY_STEPS = {"pixart": 20, "pixart_a4": 20, "pixart_lr": 20, "sana": 20, "sdxl": 4, "single": 4}


def stage_map(name: str, S: int):
    from paper_2608_03057_gb300 import schedule
    T = max(TRAJECTORY_STEPS[name], S)
    return lambda k: schedule.stage_of_step(k % T, T, S)


def e2e_measure(torch, tasq, step, n_steps, stage_of, copy_streams=1):
    """The step end to end through the C ABI with host buffers: each unit's input
    is copied in from pinned host memory on one stream and its output copied out on
    another, the units run in order on the compute stream, so the copies of other
    units overlap the kernels.  Everything is captured into one graph."""
    L = len(step.units)
    xh = [x.cpu().pin_memory() for x in step.x]
    yh = [torch.empty(y.shape, dtype=y.dtype, pin_memory=True) for y in step.y]
    nc = max(1, copy_streams)
    sh = [torch.cuda.Stream() for _ in range(nc)]
    sd = [torch.cuda.Stream() for _ in range(nc)]
    evx = [torch.cuda.Event() for _ in range(L)]
    evy = [torch.cuda.Event() for _ in range(L)]
    fork = torch.cuda.Event()
    joins = [torch.cuda.Event() for _ in range(2 * nc)]

    def e2e_step():
        # the stream the kernels go to: under graph capture the capture stream, so
        # that the copy streams fork from it and join it again and every copy is a
        # node of the captured step
        s = torch.cuda.current_stream()
        fork.record(s)
        for c in sh + sd:
            c.wait_event(fork)
        for i in range(L):
            with torch.cuda.stream(sh[i % nc]):
                step.x[i].copy_(xh[i], non_blocking=True)
                evx[i].record(sh[i % nc])
            s.wait_event(evx[i])
            step.launch_unit(i)
            evy[i].record(s)
            with torch.cuda.stream(sd[i % nc]):
                sd[i % nc].wait_event(evy[i])
                yh[i].copy_(step.y[i], non_blocking=True)
        for c, j in zip(sh + sd, joins):
            j.record(c)
            s.wait_event(j)

    def copies_only(h2d, d2h):
        # the step's own copies on the same streams, without its kernels: the time the
        # host link alone needs for them, measured beside the end-to-end figure
        s = torch.cuda.current_stream()
        fork.record(s)
        for c in sh + sd:
            c.wait_event(fork)
        for i in range(L):
            if h2d:
                with torch.cuda.stream(sh[i % nc]):
                    step.x[i].copy_(xh[i], non_blocking=True)
            if d2h:
                with torch.cuda.stream(sd[i % nc]):
                    yh[i].copy_(step.y[i], non_blocking=True)
        for c, j in zip(sh + sd, joins):
            j.record(c)
            s.wait_event(j)

    def graph_of(fn):
        fn()
        torch.cuda.synchronize()
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, capture_error_mode="thread_local"):
            fn()
        for k in range(3):  # the first replays of a new graph upload it and touch every pinned page
            g.replay()
        torch.cuda.synchronize()
        return g

    bi = int(sum(x.numel() * x.element_size() for x in xh))
    bo = int(sum(y.numel() * y.element_size() for y in yh))
    ge = graph_of(e2e_step)
    ms = timed_replays(torch, ge, step, n_steps, stage_of)
    link = {}
    for key, h2d, d2h in (("h2d_only", True, False), ("d2h_only", False, True), ("both", True, True)):
        gc = graph_of(lambda: copies_only(h2d, d2h))
        link[key + "_ms"] = timed_replays(torch, gc, step, 3, stage_of)
        del gc
    link["h2d_gbs"] = bi / link["h2d_only_ms"] / 1e6
    link["d2h_gbs"] = bo / link["d2h_only_ms"] / 1e6
    link["both_gbs"] = (bi + bo) / link["both_ms"] / 1e6
    out = {"ms_per_step": ms, "copy_streams_per_direction": nc,
           "h2d_bytes_per_step": bi, "d2h_bytes_per_step": bo,
           # the same copies with no kernels, timed right after the end-to-end replays
           "copies_only": link}
    del xh, yh, ge
    return out


def measure_workload(torch, tasq, workloads, name, args, peaks, steps, dist=None, world=1, clocks=None,
                     e2e=True, all8=True):
    """Time one workload's denoising step (CUDA graph of the whole step, the stage
    from a device int), then the same launch sequence with only its contractions
    and with only its quantizations, the all-8-bit schedule on the same graph, and
    the end-to-end step.  Returns the figures and the Step (closed by the caller)."""
    from paper_2608_03057_gb300 import engine_model, schedule
    step = Step(torch, tasq, workloads, name, args.seed,
                args.blocks if name in ("pixart", "pixart_a4", "pixart_lr", "sana") else 0, args.grouping)
    S = step.S
    stage_of = stage_map(name, S)
    for k in range(2):  # eager launches first: they set kernel attributes outside any capture
        step.d_stage.fill_(stage_of(k))
        step.launch()
    torch.cuda.synchronize()
    assert tasq.tasq_device_status(step.ctx) == tasq.TASQ_OK
    g = capture(torch, step)
    g_gemm = capture(torch, step, parts=("gemm",))
    g_quant = capture(torch, step, parts=("quant",))
    for k in range(max(3, args.warmup)):
        step.d_stage.fill_(stage_of(k))
        g.replay()
    torch.cuda.synchronize()
    if clocks:
        clocks.start()
    if dist:
        dist.barrier()
    ms = timed_replays(torch, g, step, steps, stage_of)
    clk = clocks.stop() if clocks else None
    status = tasq.tasq_device_status(step.ctx)
    if status != tasq.TASQ_OK:
        raise SystemExit(f"device status {status} after the timed region ({name})")
    ms = max_over_ranks(torch, dist, ms, "cuda")
    # the same launch sequence with one kind of kernel left out: each launch still
    # overlaps the previous one's tail (programmatic dependent launch), as in the step
    ms_gemm = timed_replays(torch, g_gemm, step, steps, stage_of)
    ms_quant = timed_replays(torch, g_quant, step, steps, stage_of)
    L = len(step.layers)
    ms8 = None
    if all8:  # the all-8-bit schedule on the same captured graph (the table is re-read on the device)
        tasq.tasq_set_schedule(step.ctx, workloads.schedule_constant(L, S, 8), L, S)
        ms8 = timed_replays(torch, g, step, steps, stage_of)
        tasq.tasq_set_schedule(step.ctx, step.table, L, S)
    # at 4-bit activations linear layers run the K loop on the e5m2 kind for b <= 4: the
    # same graph replayed with every (layer, stage) at one b shows the step time against b
    ms_by_b = None
    if step.act_bits <= 4:
        ms_by_b = {}
        for bb in (2, 4, 5, 6, 8):
            tasq.tasq_set_schedule(step.ctx, workloads.schedule_constant(L, S, bb), L, S)
            ms_by_b[bb] = timed_replays(torch, g, step, steps, stage_of)
        tasq.tasq_set_schedule(step.ctx, step.table, L, S)
    assert tasq.tasq_device_status(step.ctx) == tasq.TASQ_OK
    e2e_out = None
    if e2e:
        e2e_out = e2e_measure(torch, tasq, step, max(5, steps // 10), stage_of, args.e2e_copy_streams)
        e2e_out["ms_per_step"] = max_over_ranks(torch, dist, e2e_out["ms_per_step"], "cuda")
        e2e_out = {"value": job_tops(step.ops, world, e2e_out["ms_per_step"]), "unit": UNIT, **e2e_out}
    del g, g_gemm, g_quant

    achieved = step.ops / (ms_gemm * 1e-3) / 1e12
    # ops on the 8-bit-float route (4-bit codes, b <= 4) run at twice the bf16 rate (the
    # nominal fp8 : bf16 ratio, and the probe's equal cycles per MMA for twice the K): the
    # peak is the ops-weighted harmonic mean of the two rates
    phi = f8_op_share(tasq, step, steps, stage_of, torch.cuda.get_device_properties(0).multi_processor_count)
    peak = peaks["bf16"] / ((1.0 - phi) + phi / 2.0)
    traffic = measured_traffic(name)
    U = len(step.units)
    roofline = {"bound": "tensor", "achieved": achieved, "peak": peak, "unit": "TFLOP/s", "frac": achieved / peak,
                "traffic": traffic, "algorithmic_bytes_per_launch": step.gemm_bytes() / U,
                "kernel": "gemm_tc_kernel",
                "peak_source": f"{peaks['src']} bf16 burst (cuBLAS); the fp16 tcgen05 MMA runs at the bf16 rate, "
                               "and the contraction-only replay lasts well under a second"
                               + (f"; {phi:.3f} of the ops on the 8-bit-float route at twice that rate "
                                  "(ops-weighted harmonic mean)" if phi else ""),
                "f8_op_share": phi,
                "timing": "CUDA events around replays of the step's launch sequence with only its contractions "
                          f"({steps} replays, {U} calls each, every launch overlapping the previous one's tail "
                          "as in the step); achieved = int8-equivalent ops per step / that time"}
    if traffic is not None:
        roofline["traffic_note"] = ("mean DRAM bytes per contraction launch (ncu); inputs just written by the "
                                    "quantization can stay in L2, so traffic may sit below the algorithmic bytes")
    act_b = step.act_bytes()
    bits = step.table.astype(np.float64)
    ops_w = np.array(step.gemm_ops, np.float64)
    eff_w = float((bits * ops_w[:, None]).sum() / (ops_w.sum() * S))
    out = {
        "workload": WORKLOAD_NAMES[name], "layers": L, "contraction_calls": U, "stages": S, "ms_per_step": ms,
        "value": job_tops(step.ops, world, ms), "unit": UNIT, "ms_per_step_all8": ms8,
        "act_bits": step.act_bits, "ms_per_step_constant_b": ms_by_b,
        "effective_w_bits": eff_w, "rel_bitops": schedule.rel_bitops(eff_w, step.act_bits),
        "engine_model_rel_cost": engine_model.schedule_cost(step.table, step.gemm_ops, step.act_bits),
        "roofline": roofline,
        "roofline_quant_act": {"bound": "hbm", "bytes_per_step": act_b, "achieved": act_b / (ms_quant * 1e-3) / 1e9,
                               "peak": peaks["hbm"], "unit": "GB/s",
                               "frac": act_b / (ms_quant * 1e-3) / 1e9 / peaks["hbm"], "ms_per_step": ms_quant,
                               "bytes": "bf16 in, one byte per code out, 8 B of scales per group"},
        "step_breakdown_ms": {"contractions_only": ms_gemm, "quantizations_only": ms_quant, "timed_step": ms},
        "e2e": e2e_out, "clocks": clk,
    }
    return out, step


def clk_mhz(clk):
    """The median SM clock sampled during the timed region, else the maximum SM clock."""
    if clk and clk.get("sm_mhz"):
        return float(clk["sm_mhz"])
    return 2070.0


def main():
    args = parse_args()
    if args.impl == "reference":
        return run_reference(args)

    import torch

    from paper_2608_03057_gb300 import tasq, workloads

    world, rank, local = dist_env()
    torch.cuda.set_device(local)
    dist = None
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl")
    peaks = load_peaks()

    clocks = ClockSampler(local) if rank == 0 else None
    head, step = measure_workload(torch, tasq, workloads, args.workload, args, peaks, args.steps, dist, world, clocks,
                                  e2e=not args.no_e2e, all8=not args.no_all8)
    launches = step.launches_per_step()
    step.close()
    del step
    torch.cuda.empty_cache()

    # the other workloads of the benchmark suite, each a full step of its own
    per_workload = {}
    if not args.no_per_workload:
        for name in WORKLOAD_NAMES:
            if name == args.workload:
                continue
            r, st = measure_workload(torch, tasq, workloads, name, args, peaks, max(10, min(args.steps, 50)), dist,
                                     world, None, e2e=not args.no_e2e, all8=not args.no_all8)
            st.close()
            del st
            torch.cuda.empty_cache()
            per_workload[name] = r

    sweep = switch = zp = i8 = small_m = mma_kinds = sweep_a4 = None
    if not args.no_sweep:
        sweep, switch = run_sweep(torch, tasq, workloads, seed=args.seed)
        sweep_a4 = run_sweep_a4(torch, tasq, workloads, seed=args.seed)
        zp = run_zero_point(torch, tasq, workloads, seed=args.seed)
        small_m = run_small_m_weight_bytes(torch, tasq, seed=args.seed)
        from paper_2608_03057_gb300 import mma_probe
        mma_kinds = mma_probe.run(clk_mhz(head["clocks"]))
        # int8 GEMMs measured on this GPU, for context: the library int8 GEMM and this
        # library's own mma.sync s8 route (sm_103a has no tcgen05 int8 kind)
        i8 = {"cublaslt_int8_gemm": int8_tensor_peak(torch), "mma_sync_s8_route": s8_route_tops(torch, tasq, workloads),
              "note": "context only; the contraction runs on the fp16 tcgen05 kind, whose peak is the "
                      "measured bf16 cuBLAS rate"}

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        o, s, d, rows, threads = oracle_sample(args.workload, args.cpu_seconds, seed=args.seed)
        cpu = {"value": o / s / 1e12, "unit": UNIT, "cores": threads, "kind": "oracle",
               "sample": f"{rows} token rows of each of the first {d} layers of the step ({s:.1f} s)"}
        o1, s1, d1, rows1, _ = oracle_sample(args.workload, min(8.0, args.cpu_seconds), seed=args.seed, threads=1)
        cpu["single_thread"] = {"value": o1 / s1 / 1e12, "cores": 1,
                                "sample": f"{rows1} token rows of each of the first {d1} layers ({s1:.1f} s)"}

    if rank == 0:
        route_peak = {"tflops": peaks["bf16"], "source": f"{peaks['src']} bf16 cuBLAS burst",
                      "step_frac": head["value"] / peaks["bf16"],
                      "contractions_frac": head["roofline"]["frac"]}
        line = {
            "metric": METRIC, "value": head["value"], "unit": UNIT, "n_gpus": world, "steps": args.steps,
            "warmup": max(3, args.warmup), "ms_per_step": head["ms_per_step"], "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f16-exact-int8", "data": "synthetic",
            "config": {"workload": head["workload"], "layers": head["layers"],
                       "contraction_calls": head["contraction_calls"], "stages": head["stages"],
                       "shared_inputs": GROUPINGS[args.grouping],
                       "schedule": "seeded learned-style per-(layer, stage) bits",
                       "effective_w_bits": head["effective_w_bits"], "rel_bitops": head["rel_bitops"],
                       "route": "tcgen05 fp16 MMA, exact int32",
                       "activations": "bf16 in HBM, per-token int8 codes held as fp16",
                       "l2": "inputs larger than L2 (per-step activations and weights exceed 129 MB)",
                       "graph": "whole step captured once; stage from a device int",
                       "parallelism": f"replicas x{world}" if world > 1 else "single GPU"},
            "ms_per_step_all8": head["ms_per_step_all8"],
            "roofline": head["roofline"],
            "roofline_quant_act": head["roofline_quant_act"],
            "step_breakdown_ms": head["step_breakdown_ms"],
            "engine_model_rel_cost": head["engine_model_rel_cost"],
            "e2e": head["e2e"],
            "gpu_launches": launches * args.steps,
            "cpu_baseline": cpu,
            "clocks": head["clocks"],
            "route_peak": route_peak,
            "per_workload": per_workload,
            "sweep_tops_by_b": sweep,
            "sweep_a4_tops_by_b": sweep_a4,
            "stage_switch": switch,
            "asym_weights": zp,
            "small_m_weight_bytes": small_m,
            "mma_kinds": mma_kinds,
            "int8_gemm_context": i8,
        }
        print(json.dumps(line), flush=True)
    if dist:
        dist.barrier()
        dist.destroy_process_group()
    return 0


if __name__ == "__main__":
    sys.exit(main())
