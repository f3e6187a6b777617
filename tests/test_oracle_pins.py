"""Pins of the CPU oracle against what the paper and the mathematics fix.

Each test checks the oracle through a route that is independent of the
oracle's own formula: a different equation of the paper for the same
quantity, a closed form, a brute-force bit-plane evaluation (the paper's
bit-serial engine, Algorithm "Bit-plane schedules"), or a library routine in
a special case.  A plausible mistake in the oracle (a dropped term, a wrong
sign, a transposed operand, a wrong rounding) fails at least one of them.
"""
import math
import os

import numpy as np
import pytest

from paper_2608_03057_gb300 import schedule, workloads

ALL_CODES = np.arange(-128, 128, dtype=np.int64).astype(np.int8)


# ---------------------------------------------------------------- LSB mask --

def test_mask_b8_is_identity(oracle):
    # b = b_max keeps every plane: the operating weight is the stored weight.
    assert np.array_equal(oracle.mask(ALL_CODES, 8), ALL_CODES)


@pytest.mark.parametrize("b", range(2, 9))
def test_mask_grid_and_idempotent(oracle, b):
    m = oracle.mask(ALL_CODES, b).astype(np.int64)
    k = 8 - b
    # the value stays on the stored 8-bit grid and is a multiple of 2^k there
    assert np.all((m + 128) % (1 << k) == 0)
    # truncation only removes magnitude from the unsigned code
    assert np.all(m <= ALL_CODES.astype(np.int64)) and np.all(ALL_CODES - m < (1 << k))
    # idempotent, and chains of truncation compose to the smaller precision
    assert np.array_equal(oracle.mask(m.astype(np.int8), b), m.astype(np.int8))
    for b2 in range(2, 9):
        assert np.array_equal(oracle.mask(oracle.mask(ALL_CODES, b), b2), oracle.mask(ALL_CODES, min(b, b2)))
    # exactly 2^b distinct operating values
    assert len(np.unique(m)) == 1 << b


def _recursive_lsb_removal(Q, k, n=8):
    """Eq. lsb_extraction + Eq. lsb_masking with M = 0 applied to the k least
    significant planes one after another: at level j the (n-j)-bit code is
    Q_{n-j} = floor(Q / 2^j), its LSB is Q_{n-j} - 2 Q_{n-j-1}, and removing it
    subtracts 2^j * LSB on the stored grid."""
    out = Q
    for j in range(k):
        q_hi = Q // (1 << j)
        q_lo = Q // (1 << (j + 1))
        lsb = q_hi - 2 * q_lo
        assert lsb in (0, 1)
        out = out - (1 << j) * lsb
    return out


@pytest.mark.parametrize("b", range(2, 9))
def test_mask_equals_recursive_lsb_masking(oracle, b):
    for s in range(-128, 128):
        Q = s + 128
        want = _recursive_lsb_removal(Q, 8 - b) - 128
        assert oracle.mask_scalar(s, b) == want
        # Eq. hw_multi_lsb: the dropped block is the sum of the low bit-planes
        lsb_k = sum((1 << p) * ((Q >> p) & 1) for p in range(8 - b))
        assert Q - lsb_k - 128 == want


# ------------------------------------------------------------ quantizers --

def test_truncquant_lsb_is_a_bit():
    # Eq. truncquant on a normalized weight W in [0,1): Q_{n-1} = floor(Q_n / 2)
    # is the direct (n-1)-bit quantization, and Eq. lsb_extraction is 0 or 1.
    W = np.arange(0, 4096) / 4096.0
    for n in range(2, 9):
        Qn = np.floor(W * 2 ** n)
        Qn1 = np.floor(Qn / 2)
        assert np.array_equal(Qn1, np.floor(W * 2 ** (n - 1)))
        lsb = Qn - 2 * Qn1
        assert set(np.unique(lsb)) <= {0.0, 1.0}


@pytest.mark.parametrize("mode", [0, 1])
def test_weight_quant_nests_under_truncation(oracle, mode):
    # The 2^n (not 2^n - 1) denominator of Eq. weight_scale makes the b-bit
    # code equal the truncated 8-bit code (Eq. hw_rightshift), in fp32 too.
    w = workloads.normal((64, 257), seed=11, std=0.02)
    w[3] += 0.05  # an all-positive row for the asymmetric mode
    q8 = oracle.quant_weight(w, 8, mode)["q"]
    for k in range(1, 7):
        qb = oracle.quant_weight(w, 8 - k, mode)["q"]
        assert np.array_equal(q8 >> k, qb), k


def test_weight_quant_matches_truncquant_on_a_dyadic_grid(oracle):
    # With max|w| = 1 every step below is exact, so the symmetric-range
    # quantizer must equal Eq. truncquant on W = (w - min) / (max - min).
    j = np.arange(-1024, 1025)
    w = (j / 1024.0).astype(np.float32)[None, :]
    d = oracle.quant_weight(w, 8, 0)
    W = (j + 1024) / 2048.0
    want = np.minimum(np.floor(W * 256), 255)
    assert np.array_equal(d["q"][0], want)
    assert d["alpha"][0] == np.float32(1 / 128) and d["z"][0] == 128.0


def test_weight_quant_closed_form(oracle):
    w = workloads.normal((32, 1152), seed=1, std=0.02)
    d = oracle.quant_weight(w, 8, 0)
    amax = np.abs(w).max(1)
    assert np.array_equal(d["alpha"], (amax / 128).astype(np.float32))
    assert np.all(d["z"] == 128.0)
    assert np.array_equal(d["s"].astype(np.int32), d["q"] - 128)
    # floor: alpha (Q - z) lies in (w - alpha, w], except the clamped top code
    rec = d["alpha"][:, None].astype(np.float64) * (d["q"] - 128)
    err = w.astype(np.float64) - rec
    top = d["q"] == 255
    a = np.broadcast_to(d["alpha"][:, None].astype(np.float64), w.shape)
    # slack: w/alpha + z is rounded to fp32 (ulp <= 2^-15 below 256) before the floor
    slack = 2.0 ** -14 * a
    assert np.all((err[~top] > -slack[~top]) & (err[~top] < a[~top] + slack[~top]))
    assert np.all(np.abs(err[top]) <= a[top] + slack[top])
    # the channel minimum maps to code 0, the maximum to 2^n - 1 (Eq. weight_quant clamp)
    for n in range(32):
        assert d["q"][n, np.argmax(np.abs(w[n]))] in (0, 255)
    # Eq. weight_dequant scale: 2^n / (2^n - 1) * alpha
    np.testing.assert_allclose(d["c"], d["alpha"].astype(np.float64) * 256 / 255, rtol=2e-7)


def test_weight_quant_degenerate_row(oracle):
    w = np.zeros((2, 16), np.float32)
    w[1] = 0.5
    d = oracle.quant_weight(w, 8, 0)
    assert np.all(d["s"][0] == 0) and d["alpha"][0] == 1.0
    da = oracle.quant_weight(w, 8, 1)
    # asymmetric degenerate row dequantizes back to its constant value
    assert np.allclose(da["alpha"][1] * (da["q"][1] - da["z"][1]), 0.5)


def test_act_quant_round_half_even(oracle):
    # min = 0, max = 255 gives alpha = 1, z = 0: codes are rint(x) with ties to even.
    x = np.array([[0.0, 255.0, 2.5, 3.5, 0.5, 1.5, 254.5, 100.49999]], np.float32)
    s, alpha, zc = oracle.quant_act(x, 8, 1, 0)
    assert alpha[0] == 1.0 and zc[0] == 128.0
    assert list(s[0].astype(int) + 128) == [0, 255, 2, 4, 0, 2, 254, 100]


@pytest.mark.parametrize("mode", [0, 1])
@pytest.mark.parametrize("n_bits", [8, 4])
def test_act_quant_closed_form(oracle, mode, n_bits):
    x = workloads.normal((64, 1152), seed=0)
    x[5] = np.abs(x[5]) + 0.1  # a row that does not straddle zero
    s, alpha, zc = oracle.quant_act(x, n_bits, mode, 0)
    half = 1 << (n_bits - 1)
    Q = s.astype(np.int64) + half
    assert Q.min() >= 0 and Q.max() <= 2 ** n_bits - 1
    lo = x.min(1) if mode else -np.abs(x).max(1)
    hi = x.max(1) if mode else np.abs(x).max(1)
    np.testing.assert_allclose(alpha, (hi.astype(np.float64) - lo) / (2 ** n_bits - 1), rtol=1e-6)
    z = half - zc.astype(np.float64)
    np.testing.assert_allclose(z, -lo / alpha.astype(np.float64), rtol=1e-6, atol=1e-5)
    # round to nearest: |x - alpha (Q - z)| <= alpha / 2 (plus fp32 slack)
    rec = alpha[:, None].astype(np.float64) * (Q - z[:, None])
    assert np.all(np.abs(x - rec) <= alpha[:, None] * (0.5 + 1e-4))
    # the range ends land on the extreme codes
    if mode:
        assert np.all(Q[np.arange(64), x.argmin(1)] == 0)
        assert np.all(Q[np.arange(64), x.argmax(1)] == 2 ** n_bits - 1)


def test_act_quant_per_tensor_equals_single_row(oracle):
    x = workloads.normal((7, 33), seed=3)
    s_t, a_t, z_t = oracle.quant_act(x, 8, 0, 1)
    s_r, a_r, z_r = oracle.quant_act(x.reshape(1, -1), 8, 0, 0)
    assert np.array_equal(s_t.reshape(-1), s_r.reshape(-1)) and a_t[0] == a_r[0] and z_t[0] == z_r[0]


# ------------------------------------------------------------ contraction --

def _engine_bitserial(Qx, Qw, a_bits=8, w_planes=range(8)):
    """The bit-serial schedule of the paper's engine on unsigned codes:
    sum over weight planes i and activation planes j of
    2^(i+j) * popcount(W_i AND A_j)."""
    total = 0
    for i in w_planes:
        Wi = [(q >> i) & 1 for q in Qw]
        for j in range(a_bits):
            Aj = [(q >> j) & 1 for q in Qx]
            total += (1 << (i + j)) * sum(wi & aj for wi, aj in zip(Wi, Aj))
    return total


@pytest.mark.parametrize("b", [8, 6, 5, 3, 2])
def test_gemm_equals_bitserial_engine(oracle, b):
    M, N, K = 3, 4, 37
    s_x = workloads.uniform_codes((M, K), seed=5, lo=-128, hi=127)
    s_w = workloads.uniform_codes((N, K), seed=6, lo=-128, hi=127)
    acc = oracle.gemm(s_x, s_w, b)
    k = 8 - b
    for m in range(M):
        for n in range(N):
            Qx = [int(v) + 128 for v in s_x[m]]
            Qw8 = [int(v) + 128 for v in s_w[n]]
            # the engine streams only the top b stored planes (App. F.2)
            E = _engine_bitserial(Qx, Qw8, 8, range(k, 8))
            wm = [((q >> k) << k) for q in Qw8]  # operating code on the stored grid
            # E = sum (s_x + 128)(w' + 128) with w' the signed operating weight
            want = E - 128 * sum(int(v) for v in s_x[m]) - 128 * sum(q - 128 for q in wm) - 128 * 128 * K
            assert acc[m, n] == want


def test_gemm_signed_planes_brute_force(oracle):
    # Two's-complement plane decomposition of the masked weight (plane 7 weighs -128).
    M, N, K = 4, 5, 50
    s_x = workloads.uniform_codes((M, K), seed=8, lo=-128, hi=127).astype(np.int64)
    s_w = workloads.uniform_codes((N, K), seed=9, lo=-128, hi=127)
    for b in (8, 4):
        wm = oracle.mask(s_w, b).astype(np.int64) & 0xFF
        acc = oracle.gemm(s_x.astype(np.int8), s_w, b)
        for m in range(M):
            for n in range(N):
                tot = 0
                for p in range(8):
                    plane = (wm[n] >> p) & 1
                    weight = -(1 << p) if p == 7 else (1 << p)
                    tot += weight * int(np.dot(plane, s_x[m]))
                assert acc[m, n] == tot


def test_gemm_closed_forms(oracle):
    K = 1024
    a = np.full((2, K), -128, np.int8)
    w = np.full((3, K), -128, np.int8)
    assert np.all(oracle.gemm(a, w, 8) == 16384 * K)
    assert np.all(oracle.gemm(a, w, 2) == 16384 * K)  # -128 survives every mask
    one = np.ones((2, K), np.int8)
    w7 = np.full((3, K), 127, np.int8)
    for b in range(2, 9):
        assert np.all(oracle.gemm(one, w7, b) == K * (127 & ~((1 << (8 - b)) - 1)))
    # operand order: acc[m][n] pairs row m of s_x with row n of s_w
    x = np.zeros((2, 4), np.int8)
    x[1, 2] = 1
    ww = np.zeros((3, 4), np.int8)
    ww[2, 2] = 64
    acc = oracle.gemm(x, ww, 8)
    assert acc[1, 2] == 64 and acc.sum() == 64


def test_gemm_int32_overflow_is_reported(oracle):
    K = 131073  # 16384 * K > 2^31 - 1
    a = np.full((1, K), -128, np.int8)
    with pytest.raises(OverflowError):
        oracle.gemm(a, a, 8)


# --------------------------------------------------------------- epilogue --

@pytest.mark.parametrize("mode", [0, 1])
@pytest.mark.parametrize("b", [8, 5, 3])
def test_epilogue_f32_matches_definition(oracle, mode, b):
    M, N, K = 48, 40, 1152
    x = workloads.normal((M, K), seed=21)
    w = workloads.normal((N, K), seed=22, std=0.02)
    bias = workloads.normal((N,), seed=23, std=0.02)
    wq = oracle.quant_weight(w, 8, 0)
    s_x, alpha, zc = oracle.quant_act(x, 8, mode, 0)
    acc = oracle.gemm(s_x, wq["s"], b)
    rs = oracle.row_sums(wq["s"], b)
    y32, ybf = oracle.epilogue_f32(acc, alpha, zc, rs, wq["c"], bias)
    y64 = oracle.linear_def_f64(s_x, alpha, zc, wq["s"], wq["c"], bias, b)
    # the factored fp32 sequence is the definition up to a few fp32 roundings
    scale = np.abs(alpha)[:, None] * np.abs(wq["c"])[None, :] * (np.abs(acc) + np.abs(zc)[:, None] * np.abs(rs)[None, :])
    assert np.all(np.abs(y32 - y64) <= 8 * 2.0 ** -24 * (scale + np.abs(y64)) + 1e-9)
    # bf16 output is within half a bf16 ulp of the definition, plus that slack
    yb = oracle.bf16_bits_to_f32(ybf).astype(np.float64)
    ulp = 2.0 ** (np.floor(np.log2(np.maximum(np.abs(y64), 1e-30))) - 7)
    assert np.all(np.abs(yb - y64) <= 0.5 * ulp + 8 * 2.0 ** -24 * (scale + np.abs(y64)) + 1e-9)


def test_epilogue_real_domain_error_is_quantization_sized(oracle):
    # End to end at b = 8 the dequantized layer approximates x @ w^T + bias.
    M, N, K = 16, 24, 512
    x = workloads.normal((M, K), seed=31)
    w = workloads.normal((N, K), seed=32, std=0.02)
    out = oracle.linear_layer(x, oracle.quant_weight(w)["s"], oracle.quant_weight(w)["c"], None, 8)
    ref = x.astype(np.float64) @ w.astype(np.float64).T
    rel = np.linalg.norm(out["y"] - ref) / np.linalg.norm(ref)
    assert rel < 0.02


# ------------------------------------------- asymmetric weights (zero point) --

def test_asym_weight_quant_closed_form(oracle):
    # App. A.1.1 on each channel's true [min, max]: alpha = (max - min) / 2^n,
    # z = -min / alpha (real valued), Q = clamp(floor(w / alpha + z), 0, 2^n - 1).
    w = workloads.normal((24, 1152), seed=41, std=0.02)
    w[::3] += 0.03  # skewed channels: min and max of different magnitude
    d = oracle.quant_weight(w, 8, 1)
    lo, hi = w.min(1), w.max(1)
    assert np.array_equal(d["alpha"], ((hi - lo).astype(np.float32) / np.float32(256)).astype(np.float32))
    assert np.array_equal(d["z"], (-lo / d["alpha"]).astype(np.float32))
    assert np.array_equal(d["zcw"], (np.float32(128) - d["z"]).astype(np.float32))
    # the channel minimum is code 0 and the maximum the top code (clamped from 2^n)
    assert np.all(d["q"][np.arange(24), np.argmin(w, 1)] == 0)
    assert np.all(d["q"][np.arange(24), np.argmax(w, 1)] == 255)
    # floor quantizer: alpha (Q - z) lies in (w - alpha, w] up to the fp32 rounding of
    # w / alpha + z (ulp <= 2^-15 below 256), except at the clamped top code
    rec = d["alpha"][:, None].astype(np.float64) * (d["q"] - d["z"][:, None].astype(np.float64))
    err = w.astype(np.float64) - rec
    a = np.broadcast_to(d["alpha"][:, None].astype(np.float64), w.shape)
    top = d["q"] == 255
    slack = 2.0 ** -14 * a
    assert np.all((err[~top] > -slack[~top]) & (err[~top] < a[~top] + slack[~top]))
    assert np.all(np.abs(err[top]) <= a[top] + slack[top])


def test_asym_weight_quant_on_a_symmetric_channel_is_the_symmetric_one(oracle):
    # a channel whose minimum is exactly -max: both readings give z = 128, zcw = 0
    w = workloads.normal((6, 300), seed=42, std=0.02)
    for n in range(6):
        w[n, 7] = -np.abs(w[n]).max()
        w[n, 9] = -w[n, 7]
    ds, da = oracle.quant_weight(w, 8, 0), oracle.quant_weight(w, 8, 1)
    assert np.array_equal(ds["q"], da["q"]) and np.all(da["z"] == 128.0) and np.all(da["zcw"] == 0.0)


def test_code_sums(oracle):
    s_x = workloads.uniform_codes((9, 1000), seed=43)
    assert np.array_equal(oracle.code_sums(s_x), s_x.astype(np.int64).sum(1))


def test_epilogue_zp_with_zero_offsets_is_the_symmetric_epilogue(oracle):
    M, N, K = 20, 36, 640
    s_x, alpha, zc = oracle.quant_act(workloads.normal((M, K), seed=44), 8, 1, 0)
    wq = oracle.quant_weight(workloads.normal((N, K), seed=45, std=0.02), 8, 0)
    acc = oracle.gemm(s_x, wq["s"], 5)
    rs = oracle.row_sums(wq["s"], 5)
    bias = workloads.normal((N,), seed=46, std=0.02)
    y0, yb0 = oracle.epilogue_f32(acc, alpha, zc, rs, wq["c"], bias)
    y1, yb1 = oracle.epilogue_zp_f32(acc, alpha, zc, oracle.code_sums(s_x), rs, wq["c"], wq["zcw"], bias, K)
    assert np.all(wq["zcw"] == 0.0)
    assert np.array_equal(y0.view(np.uint32), y1.view(np.uint32)) and np.array_equal(yb0, yb1)


@pytest.mark.parametrize("mode", [0, 1])
@pytest.mark.parametrize("b", [8, 5, 3, 2])
def test_epilogue_zp_matches_definition(oracle, mode, b):
    # The factored four-term fp32 sequence against the element-by-element fp64
    # definition with the quantizer's own zero point: a dropped term, a wrong sign
    # or a wrong zero offset is off by far more than fp32 rounding.
    M, N, K = 40, 48, 1152
    x = workloads.normal((M, K), seed=47)
    w = workloads.normal((N, K), seed=48, std=0.02)
    w[::2] += 0.02
    bias = workloads.normal((N,), seed=49, std=0.02)
    wq = oracle.quant_weight(w, 8, 1)
    s_x, alpha, zc = oracle.quant_act(x, 8, mode, 0)
    acc = oracle.gemm(s_x, wq["s"], b)
    rs = oracle.row_sums(wq["s"], b)
    sx = oracle.code_sums(s_x)
    y32, ybf = oracle.epilogue_zp_f32(acc, alpha, zc, sx, rs, wq["c"], wq["zcw"], bias, K)
    y64 = oracle.linear_zp_def_f64(s_x, alpha, zc, wq["s"], wq["c"], wq["z"], bias, b)
    terms = (np.abs(acc) + np.abs(zc)[:, None] * np.abs(rs)[None, :] + np.abs(wq["zcw"])[None, :] * np.abs(sx)[:, None]
             + K * np.abs(zc)[:, None] * np.abs(wq["zcw"])[None, :])
    scale = np.abs(alpha)[:, None] * np.abs(wq["c"])[None, :] * terms
    assert np.all(np.abs(y32 - y64) <= 16 * 2.0 ** -24 * (scale + np.abs(y64)) + 1e-9)
    # and the zero-offset terms are not negligible here (the check has teeth)
    dropped = np.abs(alpha)[:, None] * np.abs(wq["c"])[None, :] * np.abs(
        wq["zcw"][None, :] * sx[:, None] + K * zc[:, None] * wq["zcw"][None, :])
    assert np.median(dropped) > 1e3 * np.median(16 * 2.0 ** -24 * (scale + np.abs(y64)))


def test_asym_weights_fit_skewed_channels_better(oracle):
    # The reason for a weight zero point: on channels whose values are not centred
    # at 0 the asymmetric grid is finer (here about half the step), so the weight
    # grid alpha (Q - z) is closer to w and the dequantized layer closer to x w^T.
    # (Both layers also carry the 2^n / (2^n - 1) factor of Eq. weight_dequant, a
    # common 0.4 % scale that the comparison of weight grids leaves out.)
    M, N, K = 16, 32, 512
    x = workloads.normal((M, K), seed=50)
    w = workloads.normal((N, K), seed=51, std=0.02) + 0.05
    ref = x.astype(np.float64) @ w.astype(np.float64).T
    s_x, alpha, zc = oracle.quant_act(x, 8, 1, 0)
    grid_err, layer_err = [], []
    for mode in (0, 1):
        wq = oracle.quant_weight(w, 8, mode)
        grid = wq["alpha"][:, None].astype(np.float64) * (wq["q"] - wq["z"][:, None].astype(np.float64))
        grid_err.append(np.sqrt(np.mean((grid - w) ** 2)))
        y = oracle.linear_zp_def_f64(s_x, alpha, zc, wq["s"], wq["c"], wq["z"], None, 8)
        layer_err.append(np.linalg.norm(y - ref) / np.linalg.norm(ref))
    assert grid_err[1] < 0.7 * grid_err[0], grid_err
    assert layer_err[1] < layer_err[0], layer_err


def test_bf16_rounding_ties_to_even(oracle):
    # 1 + 2^-8 is halfway between bf16 neighbours 1 and 1 + 2^-7: ties go to even (1.0)
    v = np.array([1.0 + 2 ** -8, 1.0 + 3 * 2 ** -8, -(1.0 + 2 ** -8), 1.0 + 2 ** -8 + 2 ** -20], np.float32)
    got = oracle.bf16_bits_to_f32(oracle.f32_to_bf16_bits(v))
    assert list(got) == [1.0, 1.0 + 2 ** -6, -1.0, 1.0 + 2 ** -7]


# ------------------------------------------------------------------- conv --

def test_conv_definition_matches_torch_conv2d(oracle):
    torch = pytest.importorskip("torch")
    B, H, W, Cin, Cout = 2, 5, 6, 8, 7
    x = workloads.normal((B, H, W, Cin), seed=41)
    w = workloads.normal((Cout, 9 * Cin), seed=42, std=0.05)
    bias = workloads.normal((Cout,), seed=43, std=0.02)
    wq = oracle.quant_weight(w)
    s_x, alpha, zc = oracle.quant_act(x.reshape(1, -1), 8, 1, 0)
    s_x = s_x.reshape(B, H, W, Cin)
    for b in (8, 4):
        y64 = oracle.conv3x3_def_f64(s_x, alpha[0], zc[0], wq["s"], wq["c"], bias, b)
        xh = torch.tensor(alpha[0], dtype=torch.float64) * (torch.tensor(s_x, dtype=torch.float64) + float(zc[0]))
        wh = torch.tensor(wq["c"], dtype=torch.float64)[:, None] * torch.tensor(oracle.mask(wq["s"], b), dtype=torch.float64)
        wh = wh.reshape(Cout, 3, 3, Cin).permute(0, 3, 1, 2)
        ref = torch.nn.functional.conv2d(xh.permute(0, 3, 1, 2), wh, torch.tensor(bias, dtype=torch.float64), padding=1)
        ref = ref.permute(0, 2, 3, 1).reshape(-1, Cout).numpy()
        np.testing.assert_allclose(y64, ref, rtol=1e-12, atol=1e-12)
        # codes + border-aware row sums + fp32 epilogue reproduce the definition
        acc, rs = oracle.conv3x3(s_x, wq["s"], b)
        y32, _ = oracle.epilogue_f32(acc, alpha, zc, rs, wq["c"], bias, per_tensor=True, rs_per_row=True)
        np.testing.assert_allclose(y32, y64, rtol=1e-5, atol=1e-6)


def test_conv_1x1_image_is_center_tap_linear(oracle):
    Cin, Cout = 16, 5
    s_x = workloads.uniform_codes((3, 1, 1, Cin), seed=51, lo=-128, hi=127)
    s_w = workloads.uniform_codes((Cout, 9 * Cin), seed=52, lo=-128, hi=127)
    acc, rs = oracle.conv3x3(s_x, s_w, 6)
    center = s_w.reshape(Cout, 9, Cin)[:, 4, :]
    assert np.array_equal(acc, oracle.gemm(s_x.reshape(3, Cin), center, 6))
    assert np.array_equal(rs, np.broadcast_to(oracle.row_sums(center, 6), (3, Cout)))


def test_conv_interior_pixel_is_full_im2col_row(oracle):
    B, H, W, Cin, Cout = 1, 4, 4, 8, 3
    s_x = workloads.uniform_codes((B, H, W, Cin), seed=53, lo=-128, hi=127)
    s_w = workloads.uniform_codes((Cout, 9 * Cin), seed=54, lo=-128, hi=127)
    acc, rs = oracle.conv3x3(s_x, s_w, 5)
    h, w = 2, 1
    patch = np.concatenate([s_x[0, h + dh, w + dw] for dh in (-1, 0, 1) for dw in (-1, 0, 1)])[None]
    assert np.array_equal(acc[h * W + w], oracle.gemm(patch, s_w, 5)[0])
    assert np.array_equal(rs[h * W + w], oracle.row_sums(s_w, 5))


def test_conv_zp_definition_matches_torch_conv2d(oracle):
    # asymmetric weights in a 3x3 conv: the fp64 definition equals torch's conv2d on
    # dequantized operands (padding zero in the real domain), and the code-domain
    # four-term epilogue with windowed code sums reproduces it
    torch = pytest.importorskip("torch")
    B, H, W, Cin, Cout = 2, 5, 6, 8, 7
    x = workloads.normal((B, H, W, Cin), seed=61)
    w = workloads.normal((Cout, 9 * Cin), seed=62, std=0.05)
    w[::2] += 0.05
    bias = workloads.normal((Cout,), seed=63, std=0.02)
    wq = oracle.quant_weight(w, 8, oracle.ASYM)
    s_x, alpha, zc = oracle.quant_act(x.reshape(1, -1), 8, 1, 0)
    s_x = s_x.reshape(B, H, W, Cin)
    sxw, kv = oracle.conv3x3_code_sums(s_x)
    for b in (8, 4, 2):
        y64 = oracle.conv3x3_zp_def_f64(s_x, alpha[0], zc[0], wq["s"], wq["c"], wq["z"], bias, b)
        xh = torch.tensor(alpha[0], dtype=torch.float64) * (torch.tensor(s_x, dtype=torch.float64) + float(zc[0]))
        qb = torch.tensor(oracle.mask(wq["s"], b), dtype=torch.float64) + 128.0
        wh = torch.tensor(wq["c"], dtype=torch.float64)[:, None] * (qb - torch.tensor(wq["z"], dtype=torch.float64)[:, None])
        wh = wh.reshape(Cout, 3, 3, Cin).permute(0, 3, 1, 2)
        ref = torch.nn.functional.conv2d(xh.permute(0, 3, 1, 2), wh, torch.tensor(bias, dtype=torch.float64), padding=1)
        ref = ref.permute(0, 2, 3, 1).reshape(-1, Cout).numpy()
        np.testing.assert_allclose(y64, ref, rtol=1e-12, atol=1e-12)
        acc, rs = oracle.conv3x3(s_x, wq["s"], b)
        y32, _ = oracle.conv_epilogue_zp_f32(acc, alpha[0], zc[0], sxw, kv, rs, wq["c"], wq["zcw"], bias)
        np.testing.assert_allclose(y32, y64, rtol=1e-5, atol=1e-5)


def test_conv_code_sums_interior_and_corner(oracle):
    B, H, W, Cin = 1, 4, 5, 16
    s_x = workloads.uniform_codes((B, H, W, Cin), seed=64, lo=-128, hi=127)
    sxw, kv = oracle.conv3x3_code_sums(s_x)
    px = s_x.astype(np.int64).sum(3)[0]  # per-pixel sums [H, W]
    assert sxw[2 * W + 2] == px[1:4, 1:4].sum() and kv[2 * W + 2] == 9 * Cin  # interior
    assert sxw[0] == px[0:2, 0:2].sum() and kv[0] == 4 * Cin                  # corner
    assert sxw[W - 2] == px[0:2, W - 3:W].sum() and kv[W - 2] == 6 * Cin      # top edge


def test_conv_epilogue_zp_with_zero_offsets_is_the_symmetric_epilogue(oracle):
    B, H, W, Cin, Cout = 1, 3, 4, 16, 8
    s_x = workloads.uniform_codes((B, H, W, Cin), seed=65, lo=-128, hi=127)
    wq = oracle.quant_weight(workloads.normal((Cout, 9 * Cin), seed=66, std=0.02), 8, 0)
    acc, rs = oracle.conv3x3(s_x, wq["s"], 6)
    sxw, kv = oracle.conv3x3_code_sums(s_x)
    alpha, zc = np.float32(0.01), np.float32(0.5)
    y0, _ = oracle.epilogue_f32(acc, np.array([alpha]), np.array([zc]), rs, wq["c"], None, per_tensor=True,
                                rs_per_row=True)
    y1, _ = oracle.conv_epilogue_zp_f32(acc, alpha, zc, sxw, kv, rs, wq["c"], wq["zcw"], None)
    assert np.array_equal(y0.view(np.uint32), y1.view(np.uint32))


# --------------------------------------------------------------- schedule --

def _golden_rows(name):
    here = os.path.join(os.path.dirname(__file__), "golden", name)
    for line in open(here):
        line = line.split("#")[0].strip()
        if line:
            parts = line.split()
            yield int(parts[0]), float(parts[1]), float(parts[2])


def test_rel_bitops_reproduces_paper_table():
    rows = list(_golden_rows("rel_bitops_table.txt"))
    assert len(rows) >= 6
    for a_bits, eff_w, rel in rows:
        assert round(schedule.rel_bitops(eff_w, a_bits) + 1e-9, 2) == rel


def test_stage_partition_is_contiguous():
    # 20 steps in 4 stages: 5 consecutive steps each, stage 0 first (noisiest)
    st = [schedule.stage_of_step(t, 20, 4) for t in range(20)]
    assert st == sorted(st) and [st.count(s) for s in range(4)] == [5, 5, 5, 5] and st[0] == 0
    # SDXL-Turbo: four steps, each its own stage
    assert [schedule.stage_of_step(t, 4, 4) for t in range(4)] == [0, 1, 2, 3]
    # uneven split still covers every stage in order
    st = [schedule.stage_of_step(t, 7, 3) for t in range(7)]
    assert st == sorted(st) and set(st) == {0, 1, 2}


def test_effective_bits_weights_by_ops():
    tab = np.array([[8, 4], [2, 4]], np.uint8)
    eb = schedule.effective_bits(tab, [3, 1])
    assert eb[0] == pytest.approx((8 * 3 + 2) / 4) and eb[1] == 4.0


# ------------------------------------------------ 16-bit low-rank branch --

def test_lowrank_down_identity_rows_select_columns(oracle):
    # l2 = the first 16 rows of the identity: u = bf16(x[:, :16]) exactly (one product per sum)
    rng = np.random.default_rng(5)
    x = rng.standard_normal((7, 48)).astype(np.float32)
    l2 = np.zeros((16, 48), np.float32)
    l2[np.arange(16), np.arange(16)] = 1.0
    u = oracle.lowrank_down(x, oracle.f32_to_bf16_bits(l2))
    assert np.array_equal(u, oracle.bf16_round(x[:, :16]).astype(np.float64))
    # a permutation of the rank rows permutes the columns of u
    perm = rng.permutation(16)
    u2 = oracle.lowrank_down(x, oracle.f32_to_bf16_bits(l2[perm]))
    assert np.array_equal(u2, u[:, perm])


def test_lowrank_branch_equals_the_product_of_its_factors(oracle):
    # small integers: every bf16 value and every sum is exact, so
    # (x l2^T) l1^T must equal x (l1 l2)^T computed in int64
    rng = np.random.default_rng(6)
    M, K, N, r = 9, 64, 24, 32
    x = rng.integers(-2, 3, (M, K))
    l2 = rng.integers(-1, 2, (r, K))
    l1 = rng.integers(-3, 4, (N, r))
    u = oracle.lowrank_down(x.astype(np.float32), oracle.f32_to_bf16_bits(l2.astype(np.float32)))
    lr = oracle.lowrank_up(u, oracle.f32_to_bf16_bits(l1.astype(np.float32)))
    assert np.array_equal(lr, (x @ (l1 @ l2).T).astype(np.float64))
    assert np.array_equal(u, (x @ l2.T).astype(np.float64))


def test_lowrank_layer_adds_the_branch_to_the_dequantized_layer(oracle):
    # with a zero branch the layer is the plain masked layer; a constant branch shifts every output
    rng = np.random.default_rng(7)
    s_x = rng.integers(-128, 128, (5, 32)).astype(np.int8)
    s_w = rng.integers(-128, 128, (6, 32)).astype(np.int8)
    alpha = rng.uniform(0.01, 0.02, 5).astype(np.float32)
    zc = rng.uniform(-1, 1, 5).astype(np.float32)
    c_w = rng.uniform(1e-3, 2e-3, 6).astype(np.float32)
    bias = rng.uniform(-0.1, 0.1, 6).astype(np.float32)
    y0 = oracle.linear_def_f64(s_x, alpha, zc, s_w, c_w, bias, 5)
    assert np.array_equal(oracle.linear_lowrank_def_f64(s_x, alpha, zc, s_w, c_w, bias, 5, np.zeros((5, 6))), y0)
    y1 = oracle.linear_lowrank_def_f64(s_x, alpha, zc, s_w, c_w, bias, 5, np.full((5, 6), 0.25))
    assert np.allclose(y1 - y0, 0.25, rtol=0, atol=1e-12)
