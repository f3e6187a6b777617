"""ctypes front end of the TASQ CPU oracle (oracle/tasq_oracle.c).

TEST INFRASTRUCTURE ONLY: tests/, __graft_entry__.smoke() and bench.py's CPU
baseline leg may import this module; the product path (the package
paper_2608_03057_gb300) never does.  The C source is compiled with plain gcc
(-O2 -ffp-contract=off, OpenMP over output rows) on first use or by
__graft_entry__.build().

Each wrapper names the passage of the paper (TASQ, arXiv 2608.03057) that the C
function restates; see the C file for the fp32 operation orders.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "tasq_oracle.c")
_BUILD = os.path.join(_HERE, "_build")
_SO = os.path.join(_BUILD, "libtasq_oracle.so")
_LOCK = threading.Lock()
_LIB = None

SYMRANGE = 0
ASYM = 1
PER_TOKEN = 0
PER_TENSOR = 1


def build(force: bool = False) -> str:
    """Compile the oracle with gcc into oracle/_build/libtasq_oracle.so."""
    os.makedirs(_BUILD, exist_ok=True)
    if not force and os.path.exists(_SO) and os.path.getmtime(_SO) >= os.path.getmtime(_SRC):
        return _SO
    tmp = _SO + f".{os.getpid()}.tmp"
    cmd = ["gcc", "-O2", "-std=c11", "-ffp-contract=off", "-fno-fast-math", "-fopenmp", "-fPIC", "-shared",
           _SRC, "-o", tmp, "-lm"]
    subprocess.run(cmd, check=True)
    os.replace(tmp, _SO)
    return _SO


def _lib():
    global _LIB
    with _LOCK:
        if _LIB is None:
            build()
            lib = ctypes.CDLL(_SO)
            P = ctypes.c_void_p
            i32, i64, f32 = ctypes.c_int, ctypes.c_int64, ctypes.c_float
            lib.oq_f32_to_bf16.argtypes = [P, i64, P]
            lib.oq_quant_weight.argtypes = [P, i32, i32, i32, i32, P, P, P, P, P]
            lib.oq_quant_act.argtypes = [P, i32, i32, i32, i32, i32, P, P, P]
            lib.oq_mask.argtypes = [i32, i32]
            lib.oq_mask.restype = i32
            lib.oq_mask_weights.argtypes = [P, i64, i32, P]
            lib.oq_gemm.argtypes = [P, i32, P, i32, i32, i32, P]
            lib.oq_gemm.restype = i64
            lib.oq_row_sums.argtypes = [P, i32, i32, i32, P]
            lib.oq_epilogue_f32.argtypes = [P, i32, i32, P, P, i32, P, i64, P, P, P, P]
            lib.oq_linear_def_f64.argtypes = [P, P, P, i32, P, P, P, i32, i32, i32, P]
            lib.oq_conv3x3.argtypes = [P, i32, i32, i32, i32, P, i32, i32, P, P]
            lib.oq_conv3x3_def_f64.argtypes = [P, f32, f32, i32, i32, i32, i32, P, P, P, i32, i32, P]
            lib.oq_weight_zero_offsets.argtypes = [P, i32, i32, P]
            lib.oq_code_sums.argtypes = [P, i32, i32, P]
            lib.oq_epilogue_zp_f32.argtypes = [P, i32, i32, i32, P, P, P, P, P, P, P, P, P]
            lib.oq_linear_zp_def_f64.argtypes = [P, P, P, i32, P, P, P, P, i32, i32, i32, P]
            lib.oq_conv3x3_code_sums.argtypes = [P, i32, i32, i32, i32, P, P]
            lib.oq_set_threads.argtypes = [i32]
            lib.oq_threads.restype = i32
            lib.oq_conv_epilogue_zp_f32.argtypes = [P, i64, i32, f32, f32, P, P, P, P, P, P, P, P]
            lib.oq_conv3x3_zp_def_f64.argtypes = [P, f32, f32, i32, i32, i32, i32, P, P, P, P, i32, i32, P]
            _LIB = lib
    return _LIB


def _p(a):
    return None if a is None else ctypes.c_void_p(a.ctypes.data)


def _c(a, dtype):
    return np.ascontiguousarray(a, dtype=dtype)


def set_threads(n: int) -> None:
    """Threads of the oracle's OpenMP loops (n <= 0: every processor)."""
    _lib().oq_set_threads(int(n))


def threads() -> int:
    return int(_lib().oq_threads())


def f32_to_bf16_bits(y):
    """fp32 -> bf16 bit patterns (uint16), round to nearest even."""
    y = _c(y, np.float32)
    out = np.empty(y.shape, np.uint16)
    _lib().oq_f32_to_bf16(_p(y), y.size, _p(out))
    return out


def bf16_bits_to_f32(b):
    return (np.asarray(b, np.uint16).astype(np.uint32) << 16).view(np.float32)


def quant_weight(w, n_bits=8, mode=SYMRANGE):
    """App. A.1.1, per output channel.  Returns dict(q, s, alpha, z, c, zcw);
    zcw = RN(2^(n-1) - z) is the weight zero offset of Eq. weight_dequant on the
    stored signed code (0 for the symmetric range)."""
    w = _c(w, np.float32)
    N, K = w.shape
    q = np.empty((N, K), np.int32)
    s = np.empty((N, K), np.int8)
    alpha = np.empty(N, np.float32)
    z = np.empty(N, np.float32)
    c = np.empty(N, np.float32)
    _lib().oq_quant_weight(_p(w), N, K, n_bits, mode, _p(q), _p(s) if n_bits <= 8 else None, _p(alpha), _p(z), _p(c))
    zcw = np.empty(N, np.float32)
    _lib().oq_weight_zero_offsets(_p(z), N, n_bits, _p(zcw))
    return dict(q=q, s=s if n_bits <= 8 else None, alpha=alpha, z=z, c=c, zcw=zcw)


def quant_act(x, n_bits=8, mode=SYMRANGE, gran=PER_TOKEN):
    """App. A.1.2.  Returns (s int8 [M,K], alpha, zc) with len(alpha) = M or 1."""
    x = _c(x, np.float32)
    M, K = x.shape
    s = np.empty((M, K), np.int8)
    g = 1 if gran == PER_TENSOR else M
    alpha = np.empty(g, np.float32)
    zc = np.empty(g, np.float32)
    _lib().oq_quant_act(_p(x), M, K, n_bits, mode, gran, _p(s), _p(alpha), _p(zc))
    return s, alpha, zc


def mask(v, b):
    """Eq. hw_rightshift on the stored signed code (vectorised through C)."""
    v = _c(v, np.int8)
    out = np.empty(v.shape, np.int8)
    _lib().oq_mask_weights(_p(v), v.size, int(b), _p(out))
    return out


def mask_scalar(v, b):
    return int(_lib().oq_mask(int(v), int(b)))


def gemm(s_x, s_w, b):
    """acc = s_x . mask_b(s_w)^T in int32 (Eq. qalora on codes); raises on int32 overflow."""
    s_x = _c(s_x, np.int8)
    s_w = _c(s_w, np.int8)
    M, K = s_x.shape
    N, K2 = s_w.shape
    assert K == K2
    acc = np.empty((M, N), np.int32)
    ov = _lib().oq_gemm(_p(s_x), M, _p(s_w), N, K, int(b), _p(acc))
    if ov:
        raise OverflowError(f"{ov} accumulators exceed int32")
    return acc


def row_sums(s_w, b):
    s_w = _c(s_w, np.int8)
    N, K = s_w.shape
    rs = np.empty(N, np.int32)
    _lib().oq_row_sums(_p(s_w), N, K, int(b), _p(rs))
    return rs


def epilogue_f32(acc, alpha, zc, rs, c_w, bias=None, per_tensor=False, rs_per_row=False):
    """Dequant epilogue in the kernel's fp32 order.  Returns (y_f32, y_bf16_bits)."""
    acc = _c(acc, np.int32)
    M, N = acc.shape
    alpha = _c(alpha, np.float32)
    zc = _c(zc, np.float32)
    rs = _c(rs, np.int32)
    c_w = _c(c_w, np.float32)
    bias = None if bias is None else _c(bias, np.float32)
    y = np.empty((M, N), np.float32)
    yb = np.empty((M, N), np.uint16)
    _lib().oq_epilogue_f32(_p(acc), M, N, _p(alpha), _p(zc), int(per_tensor), _p(rs), N if rs_per_row else 0,
                           _p(c_w), _p(bias), _p(y), _p(yb))
    return y, yb


def code_sums(s_x):
    """sx[m] = sum_k s_x[m][k], int32."""
    s_x = _c(s_x, np.int8)
    M, K = s_x.shape
    sx = np.empty(M, np.int32)
    _lib().oq_code_sums(_p(s_x), M, K, _p(sx))
    return sx


def epilogue_zp_f32(acc, alpha, zc, sx, rs, c_w, zcw, bias, K):
    """Four-term dequant epilogue (asymmetric weights, per token) in the kernel's
    fp32 order.  Returns (y_f32, y_bf16_bits)."""
    acc = _c(acc, np.int32)
    M, N = acc.shape
    args = [_c(alpha, np.float32), _c(zc, np.float32), _c(sx, np.int32), _c(rs, np.int32), _c(c_w, np.float32),
            _c(zcw, np.float32)]
    bias = None if bias is None else _c(bias, np.float32)
    y = np.empty((M, N), np.float32)
    yb = np.empty((M, N), np.uint16)
    _lib().oq_epilogue_zp_f32(_p(acc), M, N, int(K), *[_p(a) for a in args], _p(bias), _p(y), _p(yb))
    return y, yb


def linear_zp_def_f64(s_x, alpha, zc, s_w, c_w, z, bias, b):
    """The dequantized linear layer with asymmetric weights (zero point z per
    channel) by definition, fp64."""
    s_x = _c(s_x, np.int8)
    s_w = _c(s_w, np.int8)
    M, K = s_x.shape
    N = s_w.shape[0]
    bias = None if bias is None else _c(bias, np.float32)
    y = np.empty((M, N), np.float64)
    _lib().oq_linear_zp_def_f64(_p(s_x), _p(_c(alpha, np.float32)), _p(_c(zc, np.float32)), M, _p(s_w),
                                _p(_c(c_w, np.float32)), _p(_c(z, np.float32)), _p(bias), N, K, int(b), _p(y))
    return y


def linear_def_f64(s_x, alpha, zc, s_w, c_w, bias, b):
    """The dequantized linear layer by definition, fp64."""
    s_x = _c(s_x, np.int8)
    s_w = _c(s_w, np.int8)
    M, K = s_x.shape
    N = s_w.shape[0]
    alpha = _c(alpha, np.float32)
    zc = _c(zc, np.float32)
    c_w = _c(c_w, np.float32)
    bias = None if bias is None else _c(bias, np.float32)
    y = np.empty((M, N), np.float64)
    _lib().oq_linear_def_f64(_p(s_x), _p(alpha), _p(zc), M, _p(s_w), _p(c_w), _p(bias), N, K, int(b), _p(y))
    return y


def conv3x3(s_x_nhwc, s_w, b):
    """3x3/s1/p1 conv on codes.  s_w is [Cout, 9*Cin] (kh, kw, cin).  Returns (acc, rs) [P, Cout]."""
    s_x = _c(s_x_nhwc, np.int8)
    B, H, W, Cin = s_x.shape
    s_w = _c(s_w, np.int8).reshape(s_w.shape[0], -1)
    Cout = s_w.shape[0]
    assert s_w.shape[1] == 9 * Cin
    P = B * H * W
    acc = np.empty((P, Cout), np.int32)
    rs = np.empty((P, Cout), np.int32)
    _lib().oq_conv3x3(_p(s_x), B, H, W, Cin, _p(s_w), Cout, int(b), _p(acc), _p(rs))
    return acc, rs


def conv3x3_def_f64(s_x_nhwc, alpha, zc, s_w, c_w, bias, b):
    s_x = _c(s_x_nhwc, np.int8)
    B, H, W, Cin = s_x.shape
    s_w = _c(s_w, np.int8).reshape(s_w.shape[0], -1)
    Cout = s_w.shape[0]
    c_w = _c(c_w, np.float32)
    bias = None if bias is None else _c(bias, np.float32)
    y = np.empty((B * H * W, Cout), np.float64)
    _lib().oq_conv3x3_def_f64(_p(s_x), float(alpha), float(zc), B, H, W, Cin, _p(s_w), _p(c_w), _p(bias), Cout,
                              int(b), _p(y))
    return y


def linear_layer(x, w_s, c_w, bias, b, n_bits=8, mode=SYMRANGE):
    """Whole masked linear layer: act quant -> int32 GEMM -> fp32-order epilogue."""
    s_x, alpha, zc = quant_act(x, n_bits, mode, PER_TOKEN)
    acc = gemm(s_x, w_s, b)
    rs = row_sums(w_s, b)
    y, yb = epilogue_f32(acc, alpha, zc, rs, c_w, bias)
    return dict(s_x=s_x, alpha=alpha, zc=zc, acc=acc, rs=rs, y=y, y_bf16=yb)


def conv3x3_code_sums(s_x_nhwc):
    """Per output pixel: (sxw, Kv) = (sum of the in-bounds taps' input codes, Cin x in-bounds taps)."""
    s_x = _c(s_x_nhwc, np.int8)
    B, H, W, Cin = s_x.shape
    P = B * H * W
    sxw = np.empty(P, np.int32)
    kv = np.empty(P, np.int32)
    _lib().oq_conv3x3_code_sums(_p(s_x), B, H, W, Cin, _p(sxw), _p(kv))
    return sxw, kv


def conv_epilogue_zp_f32(acc, alpha, zc, sxw, kv, rs, c_w, zcw, bias):
    """Four-term conv epilogue (asymmetric weights, one activation scale) in the
    kernel's fp32 order.  acc, rs: [P, N].  Returns (y_f32, y_bf16_bits)."""
    acc = _c(acc, np.int32)
    P, N = acc.shape
    bias = None if bias is None else _c(bias, np.float32)
    y = np.empty((P, N), np.float32)
    yb = np.empty((P, N), np.uint16)
    _lib().oq_conv_epilogue_zp_f32(_p(acc), P, N, float(np.float32(alpha)), float(np.float32(zc)),
                                   _p(_c(sxw, np.int32)), _p(_c(kv, np.int32)), _p(_c(rs, np.int32)),
                                   _p(_c(c_w, np.float32)), _p(_c(zcw, np.float32)), _p(bias), _p(y), _p(yb))
    return y, yb


def conv3x3_zp_def_f64(s_x_nhwc, alpha, zc, s_w, c_w, z, bias, b):
    s_x = _c(s_x_nhwc, np.int8)
    B, H, W, Cin = s_x.shape
    s_w = _c(s_w, np.int8).reshape(s_w.shape[0], -1)
    Cout = s_w.shape[0]
    bias = None if bias is None else _c(bias, np.float32)
    y = np.empty((B * H * W, Cout), np.float64)
    _lib().oq_conv3x3_zp_def_f64(_p(s_x), float(alpha), float(zc), B, H, W, Cin, _p(s_w), _p(_c(c_w, np.float32)),
                                 _p(_c(z, np.float32)), _p(bias), Cout, int(b), _p(y))
    return y


# ------------------------------------------------ 16-bit low-rank branch --
# The frozen SVD low-rank branch that the paper's SVDQuant+TASQ pipelines keep
# beside the masked int8 weights (rank 32 for the 4-bit setting, 16 for the
# 6-bit one; the training-setting passage of the appendix): the layer computes
# y = Q(x) Q_b(R)^T + (x l2^T) l1^T, the branch on 16-bit (bf16) numbers.
# Readings: x enters the branch rounded to bf16; the branch's value is the exact
# sum, added to the dequantized main branch before the output's bf16 rounding.
# Plain numpy: fp64 matrix products of bf16 values.

def bf16_round(x):
    """fp32 values rounded to the nearest bf16 (ties to even), as fp32."""
    return bf16_bits_to_f32(f32_to_bf16_bits(np.asarray(x, np.float32)))


def lowrank_down(x, l2_bits):
    """u = sum_k bf16(x[m][k]) * l2[j][k] (fp64): x [M][K] fp32, l2 [r][K] bf16 bits."""
    return bf16_round(x).astype(np.float64) @ bf16_bits_to_f32(l2_bits).astype(np.float64).T


def lowrank_up(u, l1_bits):
    """lr[m][n] = sum_j u[m][j] * l1[n][j] (fp64), l1 [N][r] bf16 bits."""
    return np.asarray(u, np.float64) @ bf16_bits_to_f32(l1_bits).astype(np.float64).T


def linear_lowrank_def_f64(s_x, alpha, zc, s_w, c_w, bias, b, lr):
    """The dequantized masked linear layer plus its low-rank branch, fp64."""
    return linear_def_f64(s_x, alpha, zc, s_w, c_w, bias, b) + np.asarray(lr, np.float64)
