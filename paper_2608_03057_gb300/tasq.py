"""Thin Python binding of libtasq.so (include/tasq.h): same names, argument
marshalling only.  Every step of the path runs in the library's CUDA kernels.

Pointer arguments accept a torch tensor (its data_ptr()), a plain int address,
or None (NULL).  Stream arguments accept None (torch's current stream on the
current device), a torch.cuda.Stream, or a raw cudaStream_t int.  A non-zero
return code raises TasqError carrying the code and tasq_last_error() text.

The library must have been built (paper_2608_03057_gb300/build.py, or
__graft_entry__.build()); loading fails loudly otherwise -- there is no CPU
fallback.
"""
from __future__ import annotations

import ctypes
import os
import threading

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "_lib", "libtasq.so")

# enums of include/tasq.h
TASQ_OK, TASQ_ERR_INVALID_ARG, TASQ_ERR_UNSUPPORTED, TASQ_ERR_CUDA, TASQ_ERR_DEVICE_TIMEOUT, TASQ_ERR_DEVICE = range(6)
TASQ_LINEAR, TASQ_CONV3X3 = 0, 1
TASQ_F32, TASQ_BF16 = 0, 1
TASQ_SYMRANGE, TASQ_ASYM = 0, 1
TASQ_PER_TOKEN, TASQ_PER_TENSOR = 0, 1
TASQ_CODES_S8, TASQ_CODES_F16, TASQ_CODES_F16_E5M2 = 0, 1, 2
TASQ_ROUTE_AUTO, TASQ_ROUTE_TC, TASQ_ROUTE_MMA_S8 = 0, 1, 2

_lock = threading.Lock()
_lib = None


class tasq_tc_plan(ctypes.Structure):
    """The tasq_tc_plan struct of include/tasq.h."""
    _fields_ = [("tile_channels", ctypes.c_int), ("tile_tokens", ctypes.c_int), ("acc_buffers", ctypes.c_int),
                ("tiles_ch", ctypes.c_int), ("tiles_tok", ctypes.c_longlong), ("box_rows", ctypes.c_int),
                ("box_cols", ctypes.c_int), ("splits", ctypes.c_int), ("grid", ctypes.c_int),
                ("reduce_grid", ctypes.c_int), ("kernels", ctypes.c_int)]


class TasqError(RuntimeError):
    def __init__(self, code: int, msg: str):
        super().__init__(f"tasq error {code}: {msg}")
        self.code = code


def lib():
    """Load libtasq.so once; raise if it has not been built."""
    global _lib
    with _lock:
        if _lib is None:
            if not os.path.exists(LIB_PATH):
                raise RuntimeError(f"{LIB_PATH} is missing: build it with paper_2608_03057_gb300/build.py "
                                   "(the CUDA library is the only implementation; there is no fallback)")
            L = ctypes.CDLL(LIB_PATH)
            P, I, U64, SZ = ctypes.c_void_p, ctypes.c_int, ctypes.c_uint64, ctypes.c_size_t
            sigs = {
                "tasq_version": ([], I),
                "tasq_create": ([ctypes.POINTER(P), I], I),
                "tasq_destroy": ([P], None),
                "tasq_last_error": ([P], ctypes.c_char_p),
                "tasq_device_status": ([P, ctypes.POINTER(I)], I),
                "tasq_kernel_count": ([P, ctypes.POINTER(ctypes.c_ulonglong)], I),
                "tasq_set_route": ([P, I], I),
                "tasq_set_timeout_ns": ([P, U64], I),
                "tasq_selftest_timeout": ([P, U64, P], I),
                "tasq_selftest_quotients": ([P, P, I, P, I, P, P], I),
                "tasq_quant_weights": ([P, P, I, I, I, P, P, P, P], I),
                "tasq_quant_weights_asym": ([P, P, I, I, I, P, P, P, P, P], I),
                "tasq_packed_bytes": ([I, I, I], SZ),
                "tasq_pack_weights": ([P, I, P, P, P, I, I, I, P, P], I),
                "tasq_pack_weights_zp": ([P, I, P, P, P, P, I, I, I, P, P], I),
                "tasq_set_schedule": ([P, P, I, I], I),
                "tasq_set_stage_device": ([P, P], I),
                "tasq_quant_act": ([P, P, I, I, I, I, I, I, P, I, P, P, P], I),
                "tasq_quant_act_sums": ([P, P, I, I, I, I, I, I, P, I, P, P, P, P], I),
                "tasq_masked_gemm": ([P, I, I, P, I, P, P, I, P, I, I, P, P, P], I),
                "tasq_masked_gemm_zp": ([P, I, I, P, I, P, P, P, I, P, I, I, P, P, P], I),
                "tasq_masked_gemm_lr": ([P, I, I, P, I, P, P, I, P, I, I, P, P, I, P, P, P], I),
                "tasq_lowrank_down": ([P, P, I, I, I, P, I, P, P, P], I),
                "tasq_masked_gemm_grouped": ([P, P, I, I, P, I, P, P, I, P, I, I, P, P, P], I),
                "tasq_masked_gemm_shared_input": ([P, P, I, I, P, I, P, P, I, P, I, I, P, P, P], I),
                "tasq_masked_conv3x3": ([P, I, I, P, I, P, P, I, I, I, I, P, I, P, P, P], I),
                "tasq_masked_conv3x3_zp": ([P, I, I, P, I, P, P, P, I, I, I, I, P, I, P, P, P], I),
                "tasq_quant_act_tensor_noalloc": ([P, I, I, I, I, I, P, I, P, P, P], I),
                "tasq_plan_tc": ([I, I, I, I, I, I, I, I, I, ctypes.POINTER(tasq_tc_plan)], I),
                "tasq_probe_mma": ([I, I, I, P, P, P, P, I, P], I),
            }
            for name, (args, res) in sigs.items():
                f = getattr(L, name)
                f.argtypes = args
                f.restype = res
            _lib = L
    return _lib


def _ptr(t):
    if t is None:
        return None
    if isinstance(t, int):
        return t
    if hasattr(t, "data_ptr"):
        return t.data_ptr()
    if hasattr(t, "ctypes"):  # numpy array (host pointer)
        return t.ctypes.data
    raise TypeError(f"cannot pass {type(t)} as a pointer")


def _stream(s):
    if s is None:
        import torch
        return torch.cuda.current_stream().cuda_stream
    if isinstance(s, int):
        return s
    return s.cuda_stream


def _check(ctx, rc):
    if rc != TASQ_OK:
        raise TasqError(rc, tasq_last_error(ctx))


def tasq_version() -> int:
    return lib().tasq_version()


def tasq_create(device: int = 0):
    h = ctypes.c_void_p()
    rc = lib().tasq_create(ctypes.byref(h), int(device))
    if rc != TASQ_OK:
        raise TasqError(rc, tasq_last_error(None))
    return h


def tasq_destroy(ctx) -> None:
    lib().tasq_destroy(ctx)


def tasq_last_error(ctx) -> str:
    s = lib().tasq_last_error(ctx)
    return s.decode() if s else ""


def tasq_device_status(ctx) -> int:
    v = ctypes.c_int()
    _check(ctx, lib().tasq_device_status(ctx, ctypes.byref(v)))
    return v.value


def tasq_kernel_count(ctx) -> int:
    v = ctypes.c_ulonglong()
    _check(ctx, lib().tasq_kernel_count(ctx, ctypes.byref(v)))
    return v.value


def tasq_set_route(ctx, route: int) -> None:
    _check(ctx, lib().tasq_set_route(ctx, int(route)))


def tasq_set_timeout_ns(ctx, ns: int) -> None:
    _check(ctx, lib().tasq_set_timeout_ns(ctx, int(ns)))


def tasq_selftest_timeout(ctx, timeout_ns: int, stream=None) -> None:
    _check(ctx, lib().tasq_selftest_timeout(ctx, int(timeout_ns), _stream(stream)))


def tasq_selftest_quotients(ctx, x, nx, a, na, mismatches, stream=None) -> None:
    _check(ctx, lib().tasq_selftest_quotients(ctx, _ptr(x), int(nx), _ptr(a), int(na), _ptr(mismatches),
                                              _stream(stream)))


def tasq_quant_weights(ctx, w, dtype, N, K, sw, cw, alpha=None, stream=None) -> None:
    _check(ctx, lib().tasq_quant_weights(ctx, _ptr(w), int(dtype), int(N), int(K), _ptr(sw), _ptr(cw), _ptr(alpha),
                                         _stream(stream)))


def tasq_quant_weights_asym(ctx, w, dtype, N, K, sw, cw, zcw, alpha=None, stream=None) -> None:
    _check(ctx, lib().tasq_quant_weights_asym(ctx, _ptr(w), int(dtype), int(N), int(K), _ptr(sw), _ptr(cw), _ptr(zcw),
                                              _ptr(alpha), _stream(stream)))


def tasq_packed_bytes(kind, N, K) -> int:
    return int(lib().tasq_packed_bytes(int(kind), int(N), int(K)))


def tasq_pack_weights(ctx, kind, sw, cw, bias, N, K, Cin, packed, stream=None) -> None:
    _check(ctx, lib().tasq_pack_weights(ctx, int(kind), _ptr(sw), _ptr(cw), _ptr(bias), int(N), int(K), int(Cin),
                                        _ptr(packed), _stream(stream)))


def tasq_pack_weights_zp(ctx, kind, sw, cw, zcw, bias, N, K, Cin, packed, stream=None) -> None:
    _check(ctx, lib().tasq_pack_weights_zp(ctx, int(kind), _ptr(sw), _ptr(cw), _ptr(zcw), _ptr(bias), int(N), int(K),
                                           int(Cin), _ptr(packed), _stream(stream)))


def tasq_set_schedule(ctx, h_bits, L, S) -> None:
    """h_bits: a C-contiguous uint8 numpy array [L][S] (host memory)."""
    _check(ctx, lib().tasq_set_schedule(ctx, _ptr(h_bits), int(L), int(S)))


def tasq_set_stage_device(ctx, d_stage) -> None:
    _check(ctx, lib().tasq_set_stage_device(ctx, _ptr(d_stage)))


def tasq_quant_act(ctx, x, dtype, M, K, n_bits, mode, gran, codes, code_fmt, alpha, zc, stream=None) -> None:
    _check(ctx, lib().tasq_quant_act(ctx, _ptr(x), int(dtype), int(M), int(K), int(n_bits), int(mode), int(gran),
                                     _ptr(codes), int(code_fmt), _ptr(alpha), _ptr(zc), _stream(stream)))


def tasq_quant_act_sums(ctx, x, dtype, M, K, n_bits, mode, gran, codes, code_fmt, alpha, zc, code_sums,
                        stream=None) -> None:
    _check(ctx, lib().tasq_quant_act_sums(ctx, _ptr(x), int(dtype), int(M), int(K), int(n_bits), int(mode), int(gran),
                                          _ptr(codes), int(code_fmt), _ptr(alpha), _ptr(zc), _ptr(code_sums),
                                          _stream(stream)))


def tasq_masked_gemm_zp(ctx, layer, stage, codes, code_fmt, alpha, zc, code_sums, M, packed, N, K, y, acc=None,
                        stream=None) -> None:
    _check(ctx, lib().tasq_masked_gemm_zp(ctx, int(layer), int(stage), _ptr(codes), int(code_fmt), _ptr(alpha),
                                          _ptr(zc), _ptr(code_sums), int(M), _ptr(packed), int(N), int(K), _ptr(y),
                                          _ptr(acc), _stream(stream)))


def tasq_lowrank_down(ctx, x, dtype, M, K, l2, rank, alpha, u, stream=None) -> None:
    _check(ctx, lib().tasq_lowrank_down(ctx, _ptr(x), int(dtype), int(M), int(K), _ptr(l2), int(rank), _ptr(alpha),
                                        _ptr(u), _stream(stream)))


def tasq_masked_gemm_lr(ctx, layer, stage, codes, code_fmt, alpha, zc, M, packed, N, K, u, l1, rank, y, acc=None,
                        stream=None) -> None:
    _check(ctx, lib().tasq_masked_gemm_lr(ctx, int(layer), int(stage), _ptr(codes), int(code_fmt), _ptr(alpha),
                                          _ptr(zc), int(M), _ptr(packed), int(N), int(K), _ptr(u), _ptr(l1), int(rank),
                                          _ptr(y), _ptr(acc), _stream(stream)))


def tasq_masked_gemm(ctx, layer, stage, codes, code_fmt, alpha, zc, M, packed, N, K, y, acc=None, stream=None) -> None:
    _check(ctx, lib().tasq_masked_gemm(ctx, int(layer), int(stage), _ptr(codes), int(code_fmt), _ptr(alpha), _ptr(zc),
                                       int(M), _ptr(packed), int(N), int(K), _ptr(y), _ptr(acc), _stream(stream)))


def tasq_masked_gemm_grouped(ctx, layers, stage, codes, code_fmt, alpha, zc, M, packed, N, K, y, acc=None,
                             stream=None) -> None:
    """layers: the member layer indices (a sequence of 1..4 ints)."""
    h = (ctypes.c_int32 * len(layers))(*[int(v) for v in layers])
    _check(ctx, lib().tasq_masked_gemm_grouped(ctx, h, len(layers), int(stage), _ptr(codes), int(code_fmt), _ptr(alpha),
                                               _ptr(zc), int(M), _ptr(packed), int(N), int(K), _ptr(y), _ptr(acc),
                                               _stream(stream)))


def tasq_masked_gemm_shared_input(ctx, d_layers, n_layers, stage, codes, code_fmt, alpha, zc, M, packed, N, K, y,
                                  acc=None, stream=None) -> None:
    """d_layers: device int32 array of the n_layers member layer indices."""
    _check(ctx, lib().tasq_masked_gemm_shared_input(ctx, _ptr(d_layers), int(n_layers), int(stage), _ptr(codes),
                                                    int(code_fmt), _ptr(alpha), _ptr(zc), int(M), _ptr(packed), int(N),
                                                    int(K), _ptr(y), _ptr(acc), _stream(stream)))


def tasq_masked_conv3x3(ctx, layer, stage, codes, code_fmt, alpha, zc, B, H, W, Cin, packed, Cout, y, acc=None,
                        stream=None) -> None:
    _check(ctx, lib().tasq_masked_conv3x3(ctx, int(layer), int(stage), _ptr(codes), int(code_fmt), _ptr(alpha),
                                          _ptr(zc), int(B), int(H), int(W), int(Cin), _ptr(packed), int(Cout), _ptr(y),
                                          _ptr(acc), _stream(stream)))


def tasq_masked_conv3x3_zp(ctx, layer, stage, codes, code_fmt, alpha, zc, code_sums, B, H, W, Cin, packed, Cout, y,
                           acc=None, stream=None) -> None:
    _check(ctx, lib().tasq_masked_conv3x3_zp(ctx, int(layer), int(stage), _ptr(codes), int(code_fmt), _ptr(alpha),
                                             _ptr(zc), _ptr(code_sums), int(B), int(H), int(W), int(Cin), _ptr(packed),
                                             int(Cout), _ptr(y), _ptr(acc), _stream(stream)))


def tasq_quant_act_tensor_noalloc(x, dtype, M, K, n_bits, mode, codes, code_fmt, alpha, zc, stream=None) -> None:
    """Per-tensor activation quantization that allocates nothing (no context)."""
    _check(None, lib().tasq_quant_act_tensor_noalloc(_ptr(x), int(dtype), int(M), int(K), int(n_bits), int(mode),
                                                     _ptr(codes), int(code_fmt), _ptr(alpha), _ptr(zc),
                                                     _stream(stream)))


def tasq_plan_tc(kind, M, N, K, B, H, W, Cin, num_sms) -> dict:
    """Launch plan of the tensor-core route for one contraction shape (host only:
    no context, no GPU).  Returns the tasq_tc_plan fields as a dict."""
    out = tasq_tc_plan()
    _check(None, lib().tasq_plan_tc(int(kind), int(M), int(N), int(K), int(B), int(H), int(W), int(Cin), int(num_sms),
                                    ctypes.byref(out)))
    return {name: getattr(out, name) for name, _ in tasq_tc_plan._fields_}


def tasq_probe_mma(kind, n, reps, a, b, d, cycles, ctas, stream=None) -> None:
    """Tensor-core MMA kind probe (diagnostic; see include/tasq.h)."""
    _check(None, lib().tasq_probe_mma(int(kind), int(n), int(reps), _ptr(a), _ptr(b), _ptr(d), _ptr(cycles), int(ctas),
                                      _stream(stream)))
