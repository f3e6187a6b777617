"""Test helpers: run one masked layer through the C ABI on cuda:0 from numpy
inputs and bring every intermediate back to the host for comparison with the
oracle.  Allocation and copies use torch; every step of the path runs in the
library's kernels."""
from __future__ import annotations

import numpy as np

from paper_2608_03057_gb300 import tasq


def torch():
    import torch as t
    return t


def dev(a, dtype=None):
    t = torch()
    x = t.from_numpy(np.ascontiguousarray(a)).cuda()
    return x if dtype is None else x.to(dtype)


def to_bf16(a):
    """fp32 numpy -> torch bf16 on the GPU (round to nearest even) and its exact fp32 value on the host."""
    t = torch()
    x = t.from_numpy(np.ascontiguousarray(a, np.float32)).to(t.bfloat16)
    return x.cuda(), x.float().numpy()


def empty(shape, dtype):
    t = torch()
    return t.empty(shape, dtype=dtype, device="cuda")


class Ctx:
    def __init__(self):
        self.h = tasq.tasq_create(0)

    def close(self):
        tasq.tasq_destroy(self.h)


def quant_weights(ctx, w_dev, dtype, N, K):
    t = torch()
    sw = empty((N, K), t.int8)
    cw = empty((N,), t.float32)
    al = empty((N,), t.float32)
    tasq.tasq_quant_weights(ctx.h, w_dev, dtype, N, K, sw, cw, al)
    return sw, cw, al


def quant_weights_asym(ctx, w_dev, dtype, N, K):
    t = torch()
    sw = empty((N, K), t.int8)
    cw = empty((N,), t.float32)
    zcw = empty((N,), t.float32)
    al = empty((N,), t.float32)
    tasq.tasq_quant_weights_asym(ctx.h, w_dev, dtype, N, K, sw, cw, zcw, al)
    return sw, cw, zcw, al


def pack_zp(ctx, sw, cw, zcw, bias, N, K, kind=tasq.TASQ_LINEAR, Cin=0):
    t = torch()
    packed = empty((tasq.tasq_packed_bytes(kind, N, K),), t.uint8)
    tasq.tasq_pack_weights_zp(ctx.h, kind, sw, cw, zcw, bias, N, K, Cin, packed)
    return packed


def quant_act_sums(ctx, x_dev, dtype, M, K, n_bits=8, mode=tasq.TASQ_SYMRANGE, code_fmt=tasq.TASQ_CODES_S8,
                   gran=tasq.TASQ_PER_TOKEN):
    t = torch()
    codes = empty((M, K), t.int8 if code_fmt == tasq.TASQ_CODES_S8 else t.float16)
    g = 1 if gran == tasq.TASQ_PER_TENSOR else M
    alpha = empty((max(g, 1),), t.float32)
    zc = empty((max(g, 1),), t.float32)
    sums = empty((max(M, 1),), t.int32)
    tasq.tasq_quant_act_sums(ctx.h, x_dev, dtype, M, K, n_bits, mode, gran, codes, code_fmt, alpha, zc, sums)
    return codes, alpha, zc, sums


def gemm_zp(ctx, layer, stage, codes, code_fmt, alpha, zc, sums, M, packed, N, K, want_acc=True):
    t = torch()
    y = empty((M, N), t.int16)
    acc = empty((M, N), t.int32) if want_acc else None
    tasq.tasq_masked_gemm_zp(ctx.h, layer, stage, codes, code_fmt, alpha, zc, sums, M, packed, N, K, y, acc)
    return y, acc


def pack(ctx, kind, sw, cw, bias, N, K, Cin=0):
    t = torch()
    nbytes = tasq.tasq_packed_bytes(kind, N, K)
    packed = empty((nbytes,), t.uint8)
    tasq.tasq_pack_weights(ctx.h, kind, sw, cw, bias, N, K, Cin, packed)
    return packed


def quant_act(ctx, x_dev, dtype, M, K, n_bits=8, mode=tasq.TASQ_SYMRANGE, gran=tasq.TASQ_PER_TOKEN,
              code_fmt=tasq.TASQ_CODES_S8):
    t = torch()
    codes = empty((M, K), t.int8 if code_fmt == tasq.TASQ_CODES_S8 else t.float16)
    g = 1 if gran == tasq.TASQ_PER_TENSOR else M
    alpha = empty((max(g, 1),), t.float32)
    zc = empty((max(g, 1),), t.float32)
    tasq.tasq_quant_act(ctx.h, x_dev, dtype, M, K, n_bits, mode, gran, codes, code_fmt, alpha, zc)
    return codes, alpha, zc


def codes_to_int8(codes):
    t = torch()
    if codes.dtype == t.float16:
        f = codes.float()
        assert bool((f == f.round()).all())
        return f.to(t.int8).cpu().numpy()
    return codes.cpu().numpy()


def gemm(ctx, layer, stage, codes, code_fmt, alpha, zc, M, packed, N, K, want_acc=True):
    t = torch()
    y = empty((M, N), t.int16)
    acc = empty((M, N), t.int32) if want_acc else None
    tasq.tasq_masked_gemm(ctx.h, layer, stage, codes, code_fmt, alpha, zc, M, packed, N, K, y, acc)
    return y, acc


def conv(ctx, layer, stage, codes, code_fmt, alpha, zc, B, H, W, Cin, packed, Cout, want_acc=True):
    t = torch()
    y = empty((B * H * W, Cout), t.int16)
    acc = empty((B * H * W, Cout), t.int32) if want_acc else None
    tasq.tasq_masked_conv3x3(ctx.h, layer, stage, codes, code_fmt, alpha, zc, B, H, W, Cin, packed, Cout, y, acc)
    return y, acc


def bf16_bits_host(y_dev):
    return y_dev.cpu().numpy().view(np.uint16)


def packed_header(packed):
    """(chunk_kb[0..8], off_rs, off_ts) read back from a packed buffer."""
    raw = packed[:256].cpu().numpy()
    ints = raw.view(np.int32)
    chunk = ints[5:14].copy()
    i64 = raw[56:104].view(np.int64)  # off_w, off_cw, off_bias, off_rs, off_ts, total
    return chunk, dict(off_w=int(i64[0]), off_cw=int(i64[1]), off_bias=int(i64[2]), off_rs=int(i64[3]),
                       off_ts=int(i64[4]), total=int(i64[5]))


def assert_bf16_close(y_gpu_bits, y_ref_bits, atol=1e-2, rtol=1e-3):
    """|gpu - ref| <= atol + rtol * |ref| element by element on the bf16 values;
    returns the number of bit-identical elements."""
    g = (y_gpu_bits.astype(np.uint32) << 16).view(np.float32).astype(np.float64)
    r = (y_ref_bits.astype(np.uint32) << 16).view(np.float32).astype(np.float64)
    bad = np.abs(g - r) > atol + rtol * np.abs(r)
    assert not bad.any(), f"{bad.sum()} of {bad.size} bf16 outputs outside tolerance; first at {np.argwhere(bad)[:5]}"
    return int((y_gpu_bits == y_ref_bits).sum())
