"""GPU parity: every step of the path, called through the C ABI, against the
CPU oracle on the same seeded inputs.

Bar: int8 codes, int32 accumulators, row sums and the packed certificate are
bit-exact; bf16 outputs are within |d| <= 1e-2 + 1e-3 |ref| of the oracle's
fp32-order epilogue (and are expected to be bit-identical, since both sides
round every fp32 operation to nearest even in the same order).
"""
import numpy as np
import pytest

from paper_2608_03057_gb300 import tasq, workloads
from tests import gpu_layer as G
from tests import gpu_layer as GL

pytestmark = pytest.mark.gpu

ROUTES = [pytest.param(tasq.TASQ_CODES_S8, id="mma_s8"), pytest.param(tasq.TASQ_CODES_F16, id="tc")]


@pytest.fixture(scope="module")
def ctx():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    c = G.Ctx()
    yield c
    assert tasq.tasq_device_status(c.h) == tasq.TASQ_OK
    c.close()


# ------------------------------------------------------------ quantizers --

@pytest.mark.parametrize("dtype", [tasq.TASQ_F32, tasq.TASQ_BF16])
def test_quant_weights_bitexact(ctx, oracle, dtype):
    torch = G.torch()
    N, K = 136, 1168
    w = workloads.normal((N, K), seed=1, std=0.02)
    w[5] = 0.0  # degenerate channel
    if dtype == tasq.TASQ_BF16:
        wd, w = G.to_bf16(w)
    else:
        wd = G.dev(w)
    sw, cw, al = G.quant_weights(ctx, wd, dtype, N, K)
    ref = oracle.quant_weight(w, 8, oracle.SYMRANGE)
    assert np.array_equal(sw.cpu().numpy(), ref["s"])
    assert np.array_equal(cw.cpu().numpy(), ref["c"])
    assert np.array_equal(al.cpu().numpy(), ref["alpha"])


def _near_boundary_rows(x, r0, n_bits, mode, nrows=8):
    """Rows whose values sit within a few ulps of the rounding boundaries
    x / alpha + z = k + 1/2 (scale and offset computed as the quantizer does,
    in fp32), so that any shortcut in the division or the rounding shows up."""
    K = x.shape[1]
    qmax = np.float32((1 << n_bits) - 1)
    f = np.float32
    for i in range(nrows):
        A = f(0.37 + 0.61 * i)
        row = x[r0 + i]
        row[0], row[1] = A, -A if mode == tasq.TASQ_SYMRANGE else -f(0.5) * A
        lo, hi = (-A, A) if mode == tasq.TASQ_SYMRANGE else (row[1], A)
        alpha = f(f(hi - lo) / qmax)
        z = f(f(-lo) / alpha)
        k = np.arange(K - 2) % int(qmax)
        base = ((k + f(0.5) - z).astype(np.float32) * alpha).astype(np.float32)
        steps = (np.arange(K - 2) % 7) - 3
        v = base.copy()
        for _ in range(3):
            v = np.where(steps > 0, np.nextafter(v, np.float32(np.inf)), np.where(steps < 0, np.nextafter(v, np.float32(-np.inf)), v))
            steps = steps - np.sign(steps)
        row[2:] = np.clip(v, lo, hi)


@pytest.mark.parametrize("code_fmt", [tasq.TASQ_CODES_S8, tasq.TASQ_CODES_F16])
@pytest.mark.parametrize("mode", [tasq.TASQ_SYMRANGE, tasq.TASQ_ASYM])
@pytest.mark.parametrize("n_bits", [8, 4])
@pytest.mark.parametrize("dtype", [tasq.TASQ_F32, tasq.TASQ_BF16])
def test_quant_act_per_token_bitexact(ctx, oracle, code_fmt, mode, n_bits, dtype):
    M, K = 203, 1152
    x = workloads.normal((M, K), seed=0)
    x[7] = 0.0          # constant row
    x[9] = np.abs(x[9]) + 0.5  # one-signed row
    x[11, :] = 3.0
    x[11, 5] = 2.5      # exact ties of the rounding
    _near_boundary_rows(x, 13, n_bits, mode)
    x[21] = 1000.0 + workloads.uniform((K,), seed=4, lo=0.0, hi=1.0)  # far from zero: large quotients, small range
    if dtype == tasq.TASQ_BF16:
        xd, x = G.to_bf16(x)
    else:
        xd = G.dev(x)
    codes, alpha, zc = G.quant_act(ctx, xd, dtype, M, K, n_bits, mode, tasq.TASQ_PER_TOKEN, code_fmt)
    s, a, z = oracle.quant_act(x, n_bits, mode, oracle.PER_TOKEN)
    assert np.array_equal(G.codes_to_int8(codes), s)
    assert np.array_equal(alpha.cpu().numpy(), a)
    assert np.array_equal(zc.cpu().numpy(), z)


@pytest.mark.parametrize("mode", [tasq.TASQ_SYMRANGE, tasq.TASQ_ASYM])
@pytest.mark.parametrize("code_fmt", [tasq.TASQ_CODES_S8, tasq.TASQ_CODES_F16])
def test_quant_act_per_tensor_bitexact(ctx, oracle, mode, code_fmt):
    B, H, W, C = 1, 64, 64, 320
    x = workloads.normal((B, H, W, C), seed=2)
    codes, alpha, zc = G.quant_act(ctx, G.dev(x), tasq.TASQ_F32, B * H * W, C, 8, mode, tasq.TASQ_PER_TENSOR, code_fmt)
    s, a, z = oracle.quant_act(x.reshape(1, -1), 8, mode, oracle.PER_TOKEN)
    assert np.array_equal(G.codes_to_int8(codes).reshape(-1), s.reshape(-1))
    assert alpha.cpu().numpy()[0] == a[0] and zc.cpu().numpy()[0] == z[0]


# ------------------------------------------------------------------ pack --

def _expected_chunk(masked_abs_blocks, limit=1 << 17):
    """Longest window length (in 64-wide K blocks) all of whose windows stay
    within the limit, minimized over channels."""
    best = None
    for row in masked_abs_blocks:
        KB = len(row)
        c = KB
        for L in range(1, KB + 1):
            if max(row[i:i + L].sum() for i in range(KB - L + 1)) > limit:
                c = L - 1
                break
        best = c if best is None else min(best, c)
    return max(best, 1)


@pytest.mark.parametrize("kind", [tasq.TASQ_LINEAR, tasq.TASQ_CONV3X3])
def test_pack_row_sums_and_certificate(ctx, oracle, kind):
    torch = G.torch()
    if kind == tasq.TASQ_LINEAR:
        N, K, Cin = 72, 4096, 0
    else:
        N, Cin = 48, 320
        K = 9 * Cin
    s_w = workloads.uniform_codes((N, K), seed=3, lo=-128, hi=127)
    cw = workloads.uniform((N,), 4, 1e-4, 1e-3)
    packed = G.pack(ctx, kind, G.dev(s_w), G.dev(cw), None, N, K, Cin)
    torch.cuda.synchronize()
    chunk, off = G.packed_header(packed)
    raw = packed.cpu().numpy()
    assert np.array_equal(raw[off["off_w"]:off["off_w"] + N * K].view(np.int8).reshape(N, K), s_w)
    rs = raw[off["off_rs"]:off["off_rs"] + 4 * 7 * N].view(np.int32).reshape(7, N)
    for b in range(2, 9):
        masked = oracle.mask(s_w, b).astype(np.int64)
        assert np.array_equal(rs[b - 2], oracle.row_sums(s_w, b)), b
        KB = (K + 63) // 64
        blocks = np.abs(np.pad(masked, ((0, 0), (0, KB * 64 - K)))).reshape(N, KB, 64).sum(2)
        assert chunk[b] == _expected_chunk(blocks), b
        if kind == tasq.TASQ_CONV3X3:
            ts = raw[off["off_ts"]:off["off_ts"] + 4 * 7 * N * 9].view(np.int32).reshape(7, N, 9)
            assert np.array_equal(ts[b - 2], masked.reshape(N, 9, Cin).sum(2)), b


# ---------------------------------------------------------- linear layer --

def _setup_linear(ctx, oracle, M, N, K, bits, seed=0, x_std=1.0, w_std=0.02, dtype=tasq.TASQ_F32, code_fmt=None,
                  mode=tasq.TASQ_SYMRANGE):
    w = workloads.normal((N, K), seed + 1, w_std)
    bias = workloads.normal((N,), seed + 2, 0.02)
    x = workloads.normal((M, K), seed, x_std)
    if dtype == tasq.TASQ_BF16:
        xd, x = G.to_bf16(x)
    else:
        xd = G.dev(x)
    sw, cw, _ = G.quant_weights(ctx, G.dev(w), tasq.TASQ_F32, N, K)
    packed = G.pack(ctx, tasq.TASQ_LINEAR, sw, cw, G.dev(bias), N, K)
    tasq.tasq_set_schedule(ctx.h, np.asarray([bits], np.uint8), 1, len(bits))
    codes, alpha, zc = G.quant_act(ctx, xd, dtype, M, K, 8, mode, tasq.TASQ_PER_TOKEN, code_fmt)
    wq = oracle.quant_weight(w)
    s_x, a_ref, z_ref = oracle.quant_act(x, 8, mode, oracle.PER_TOKEN)
    return dict(packed=packed, codes=codes, alpha=alpha, zc=zc, wq=wq, s_x=s_x, a=a_ref, z=z_ref, bias=bias)


def _check_layer(oracle, st, b, y, acc, rows=None):
    s_x, a, z = st["s_x"], st["a"], st["z"]
    if rows is not None:
        s_x, a, z = s_x[rows], a[rows], z[rows]
    ref_acc = oracle.gemm(s_x, st["wq"]["s"], b)
    got_acc = acc.cpu().numpy() if rows is None else acc.cpu().numpy()[rows]
    assert np.array_equal(got_acc, ref_acc), f"b={b}: {(got_acc != ref_acc).sum()} int32 mismatches"
    rs = oracle.row_sums(st["wq"]["s"], b)
    _, yb = oracle.epilogue_f32(ref_acc, a, z, rs, st["wq"]["c"], st["bias"])
    got_y = G.bf16_bits_host(y) if rows is None else G.bf16_bits_host(y)[rows]
    same = G.assert_bf16_close(got_y, yb)
    assert same == yb.size, f"b={b}: {yb.size - same} bf16 outputs differ in the last bit"


@pytest.mark.parametrize("code_fmt", ROUTES)
def test_single_linear_all_stages(ctx, oracle, code_fmt):
    """256 tokens x 1152 -> 1152, stages at b = 8, 6, 4, 3 on one shared buffer."""
    M, N, K = 256, 1152, 1152
    st = _setup_linear(ctx, oracle, M, N, K, [8, 6, 4, 3], code_fmt=code_fmt)
    for stage, b in enumerate([8, 6, 4, 3]):
        y, acc = G.gemm(ctx, 0, stage, st["codes"], code_fmt, st["alpha"], st["zc"], M, st["packed"], N, K)
        _check_layer(oracle, st, b, y, acc)


@pytest.mark.parametrize("code_fmt", ROUTES)
@pytest.mark.parametrize("M,N,K", [(1, 8, 16), (77, 24, 48), (300, 136, 1168), (129, 264, 2240), (513, 72, 64)])
def test_ragged_shapes(ctx, oracle, code_fmt, M, N, K):
    bits = [2, 5, 7, 8]
    st = _setup_linear(ctx, oracle, M, N, K, bits, seed=M + N, code_fmt=code_fmt, mode=tasq.TASQ_ASYM)
    for stage, b in enumerate(bits):
        y, acc = G.gemm(ctx, 0, stage, st["codes"], code_fmt, st["alpha"], st["zc"], M, st["packed"], N, K)
        _check_layer(oracle, st, b, y, acc)


@pytest.mark.parametrize("code_fmt", ROUTES)
def test_wide_tiles_ragged_full(ctx, oracle, code_fmt):
    """A launch whose 256-token tiles fit one wave of CTAs (the wide, single-
    accumulator configuration of the tensor-core route), with a ragged last
    token tile and a ragged last channel tile, checked in full."""
    M, N, K = 4000, 1096, 384
    bits = [8, 3]
    st = _setup_linear(ctx, oracle, M, N, K, bits, seed=7, code_fmt=code_fmt)
    for stage, b in enumerate(bits):
        y, acc = G.gemm(ctx, 0, stage, st["codes"], code_fmt, st["alpha"], st["zc"], M, st["packed"], N, K)
        _check_layer(oracle, st, b, y, acc)


@pytest.mark.parametrize("code_fmt", ROUTES)
@pytest.mark.parametrize("M,N,K", [(300, 1152, 1168), (77, 640, 2048), (64, 128, 4096)])
def test_split_k_repeated_launches(ctx, oracle, code_fmt, M, N, K):
    """Few tiles and a long K (ragged last K block): where the tensor-core route
    cuts K into slices, their exact partial sums are added by a second kernel.
    Each stage runs twice on the same context (shared split scratch) and must
    give identical, exact results."""
    bits = [8, 3]
    st = _setup_linear(ctx, oracle, M, N, K, bits, seed=M + 3, code_fmt=code_fmt)
    for stage, b in enumerate(bits):
        outs = []
        for _ in range(2):
            y, acc = G.gemm(ctx, 0, stage, st["codes"], code_fmt, st["alpha"], st["zc"], M, st["packed"], N, K)
            _check_layer(oracle, st, b, y, acc)
            outs.append(G.bf16_bits_host(y))
        assert np.array_equal(outs[0], outs[1])
    assert tasq.tasq_device_status(ctx.h) == tasq.TASQ_OK


@pytest.mark.parametrize("kind,shape", [
    (tasq.TASQ_LINEAR, (4096, 3456, 1152)),   # 192-token tiles, persistent
    (tasq.TASQ_LINEAR, (4000, 1096, 384)),    # 256-token tiles
    (tasq.TASQ_LINEAR, (300, 2304, 1152)),    # 64-token tiles
    (tasq.TASQ_LINEAR, (64, 1152, 4608)),     # 64-token tiles, split K
    (tasq.TASQ_CONV3X3, (1, 64, 64, 640, 640)),
    (tasq.TASQ_CONV3X3, (2, 6, 6, 64, 128)),
])
def test_launches_follow_the_plan(ctx, kind, shape):
    """The contraction enqueues the kernels tasq_plan_tc reports for its shape
    on this GPU's SM count (two where K is split), and leaves no device error."""
    torch = G.torch()
    sms = torch.cuda.get_device_properties(0).multi_processor_count
    F16 = tasq.TASQ_CODES_F16
    if kind == tasq.TASQ_LINEAR:
        M, N, K = shape
        plan = tasq.tasq_plan_tc(kind, M, N, K, 0, 0, 0, 0, sms)
        Cin = 0
    else:
        B, H, W, Cin, N = shape
        M, K = B * H * W, 9 * Cin
        plan = tasq.tasq_plan_tc(kind, 0, N, 0, B, H, W, Cin, sms)
    assert plan["kernels"] >= 1 and plan["grid"] <= sms
    w = workloads.normal((N, K), 31, 0.02)
    sw, cw, _ = G.quant_weights(ctx, G.dev(w), tasq.TASQ_F32, N, K)
    packed = G.pack(ctx, kind, sw, cw, G.dev(np.zeros(N, np.float32)), N, K, Cin)
    tasq.tasq_set_schedule(ctx.h, np.array([[6]], np.uint8), 1, 1)
    gran = tasq.TASQ_PER_TENSOR if kind == tasq.TASQ_CONV3X3 else tasq.TASQ_PER_TOKEN
    k_in = Cin if Cin else K
    codes, alpha, zc = G.quant_act(ctx, G.dev(workloads.normal((M, k_in), 32)), tasq.TASQ_F32, M, k_in, gran=gran,
                                   code_fmt=F16)
    before = tasq.tasq_kernel_count(ctx.h)
    if kind == tasq.TASQ_LINEAR:
        G.gemm(ctx, 0, 0, codes, F16, alpha, zc, M, packed, N, K, want_acc=False)
    else:
        G.conv(ctx, 0, 0, codes, F16, alpha, zc, B, H, W, Cin, packed, N, want_acc=False)
    assert tasq.tasq_kernel_count(ctx.h) - before == plan["kernels"]
    assert tasq.tasq_device_status(ctx.h) == tasq.TASQ_OK


@pytest.mark.parametrize("graph", [False, True])
def test_two_layer_chain_reads_the_previous_output(ctx, oracle, graph):
    """Layer 2 quantizes layer 1's bf16 output, so every kernel depends on the one
    before it: the quantization may start (and prefetch its input into L2) while the
    first contraction drains, and the second contraction runs its weight pipeline
    before its dependency wait.  Eager and captured in a CUDA graph, the chain must
    give the oracle's result on the first layer's actual output."""
    torch = G.torch()
    M, K1, N1, N2 = 1000, 1152, 1152, 2304
    x1 = workloads.normal((M, K1), 91)
    w1 = workloads.normal((N1, K1), 92, 0.03)
    w2 = workloads.normal((N2, N1), 93, 0.03)
    b1 = workloads.normal((N1,), 94, 0.02)
    b2 = workloads.normal((N2,), 95, 0.02)
    sw1, cw1, _ = G.quant_weights(ctx, G.dev(w1), tasq.TASQ_F32, N1, K1)
    sw2, cw2, _ = G.quant_weights(ctx, G.dev(w2), tasq.TASQ_F32, N2, N1)
    p1 = G.pack(ctx, tasq.TASQ_LINEAR, sw1, cw1, G.dev(b1), N1, K1)
    p2 = G.pack(ctx, tasq.TASQ_LINEAR, sw2, cw2, G.dev(b2), N2, N1)
    tasq.tasq_set_schedule(ctx.h, np.array([[5, 8], [3, 6]], np.uint8), 2, 2)
    x1d, x1h = G.to_bf16(x1)
    F16 = tasq.TASQ_CODES_F16
    c1, c2 = G.empty((M, K1), torch.float16), G.empty((M, N1), torch.float16)
    a1, z1, a2, z2 = (G.empty((M,), torch.float32) for _ in range(4))
    y1, y2 = G.empty((M, N1), torch.int16), G.empty((M, N2), torch.int16)

    def chain(stage):
        tasq.tasq_quant_act(ctx.h, x1d, tasq.TASQ_BF16, M, K1, 8, tasq.TASQ_SYMRANGE, tasq.TASQ_PER_TOKEN, c1, F16,
                            a1, z1)
        tasq.tasq_masked_gemm(ctx.h, 0, stage, c1, F16, a1, z1, M, p1, N1, K1, y1, None)
        tasq.tasq_quant_act(ctx.h, y1, tasq.TASQ_BF16, M, N1, 8, tasq.TASQ_SYMRANGE, tasq.TASQ_PER_TOKEN, c2, F16,
                            a2, z2)
        tasq.tasq_masked_gemm(ctx.h, 1, stage, c2, F16, a2, z2, M, p2, N2, N1, y2, None)

    wq1, wq2 = oracle.quant_weight(w1), oracle.quant_weight(w2)
    for stage in (0, 1):
        y1.fill_(0)
        y2.fill_(0)
        if graph:
            chain(stage)  # first launches set kernel attributes outside the capture
            torch.cuda.synchronize()
            y1.fill_(0)
            y2.fill_(0)
            s = torch.cuda.Stream()
            s.wait_stream(torch.cuda.current_stream())
            g = torch.cuda.CUDAGraph()
            with torch.cuda.stream(s), torch.cuda.graph(g, stream=s):
                chain(stage)
            g.replay()
        else:
            chain(stage)
        torch.cuda.synchronize()
        b1_, b2_ = [(5, 8), (3, 6)][0][stage], [(5, 8), (3, 6)][1][stage]
        s_x1, ar1, zr1 = oracle.quant_act(x1h)
        acc1 = oracle.gemm(s_x1, wq1["s"], b1_)
        _, yb1 = oracle.epilogue_f32(acc1, ar1, zr1, oracle.row_sums(wq1["s"], b1_), wq1["c"], b1)
        assert np.array_equal(G.bf16_bits_host(y1), yb1)
        # layer 2 from the GPU's layer-1 output (bit-identical to the oracle's)
        x2h = oracle.bf16_bits_to_f32(yb1)
        s_x2, ar2, zr2 = oracle.quant_act(x2h)
        acc2 = oracle.gemm(s_x2, wq2["s"], b2_)
        _, yb2 = oracle.epilogue_f32(acc2, ar2, zr2, oracle.row_sums(wq2["s"], b2_), wq2["c"], b2)
        assert np.array_equal(G.bf16_bits_host(y2), yb2)
    assert tasq.tasq_device_status(ctx.h) == tasq.TASQ_OK


@pytest.mark.parametrize("code_fmt", ROUTES)
def test_output_without_acc(ctx, oracle, code_fmt):
    M, N, K = 200, 128, 256
    st = _setup_linear(ctx, oracle, M, N, K, [6], code_fmt=code_fmt)
    y0, acc = G.gemm(ctx, 0, 0, st["codes"], code_fmt, st["alpha"], st["zc"], M, st["packed"], N, K)
    y1, _ = G.gemm(ctx, 0, 0, st["codes"], code_fmt, st["alpha"], st["zc"], M, st["packed"], N, K, want_acc=False)
    assert np.array_equal(G.bf16_bits_host(y0), G.bf16_bits_host(y1))


@pytest.mark.parametrize("code_fmt", ROUTES)
def test_empty_batch_is_a_noop(ctx, code_fmt):
    torch = G.torch()
    N, K = 64, 64
    sw = torch.zeros((N, K), dtype=torch.int8, device="cuda")
    cw = torch.ones((N,), dtype=torch.float32, device="cuda")
    packed = G.pack(ctx, tasq.TASQ_LINEAR, sw, cw, None, N, K)
    tasq.tasq_set_schedule(ctx.h, np.array([[8]], np.uint8), 1, 1)
    one = torch.zeros((16,), dtype=torch.float32, device="cuda")
    tasq.tasq_masked_gemm(ctx.h, 0, 0, one, code_fmt, one, one, 0, packed, N, K, one, None)
    assert tasq.tasq_device_status(ctx.h) == tasq.TASQ_OK


@pytest.mark.parametrize("code_fmt", ROUTES)
def test_extreme_codes_exact(ctx, oracle, code_fmt):
    """All activation and weight codes at -128 (|acc| = 16384 K) and
    alternating-sign rows: the accumulators must stay exact."""
    torch = G.torch()
    M, N, K = 130, 136, 1024
    s_w = np.full((N, K), -128, np.int8)
    s_w[1::2, 1::2] = 127
    s_x = np.full((M, K), -128, np.int8)
    s_x[1::3, ::2] = 127
    cw = np.full((N,), 1e-6, np.float32)
    packed = G.pack(ctx, tasq.TASQ_LINEAR, G.dev(s_w), G.dev(cw), None, N, K)
    tasq.tasq_set_schedule(ctx.h, np.array([[8, 2, 5]], np.uint8), 1, 3)
    codes = G.dev(s_x) if code_fmt == tasq.TASQ_CODES_S8 else G.dev(s_x.astype(np.float16))
    alpha = G.dev(np.full((M,), 1e-3, np.float32))
    zc = G.dev(np.full((M,), 0.5, np.float32))
    for stage, b in enumerate([8, 2, 5]):
        y, acc = G.gemm(ctx, 0, stage, codes, code_fmt, alpha, zc, M, packed, N, K)
        assert np.array_equal(acc.cpu().numpy(), oracle.gemm(s_x, s_w, b)), b


@pytest.mark.parametrize("code_fmt", ROUTES)
def test_uniform_codes_long_k_exact(ctx, oracle, code_fmt):
    """Uniform [-127, 127] codes with K = 4096: sums of |w| exceed the fp32
    exact range, so the tensor-core route must drain in certified chunks."""
    M, N, K = 256, 256, 4096
    s_x = workloads.uniform_codes((M, K), seed=61)
    s_w = workloads.uniform_codes((N, K), seed=62)
    cw = workloads.uniform((N,), 63, 1e-4, 2e-4)
    packed = G.pack(ctx, tasq.TASQ_LINEAR, G.dev(s_w), G.dev(cw), None, N, K)
    tasq.tasq_set_schedule(ctx.h, np.array([[8, 7, 4, 2]], np.uint8), 1, 4)
    codes = G.dev(s_x) if code_fmt == tasq.TASQ_CODES_S8 else G.dev(s_x.astype(np.float16))
    alpha = G.dev(workloads.uniform((M,), 64, 1e-3, 2e-3))
    zc = G.dev(np.full((M,), 0.5, np.float32))
    for stage, b in enumerate([8, 7, 4, 2]):
        y, acc = G.gemm(ctx, 0, stage, codes, code_fmt, alpha, zc, M, packed, N, K)
        assert np.array_equal(acc.cpu().numpy(), oracle.gemm(s_x, s_w, b)), b


@pytest.mark.parametrize("code_fmt", ROUTES)
def test_stage_from_device_int(ctx, oracle, code_fmt):
    torch = G.torch()
    M, N, K = 128, 256, 512
    bits = [3, 8, 5]
    st = _setup_linear(ctx, oracle, M, N, K, bits, code_fmt=code_fmt)
    d_stage = torch.zeros((4,), dtype=torch.int32, device="cuda")
    tasq.tasq_set_stage_device(ctx.h, d_stage)
    try:
        for stage, b in enumerate(bits):
            d_stage.fill_(stage)
            y, acc = G.gemm(ctx, 0, -1, st["codes"], code_fmt, st["alpha"], st["zc"], M, st["packed"], N, K)
            _check_layer(oracle, st, b, y, acc)
        d_stage.fill_(7)  # out of range: recorded on the device, nothing written
        G.gemm(ctx, 0, -1, st["codes"], code_fmt, st["alpha"], st["zc"], M, st["packed"], N, K)
        assert tasq.tasq_device_status(ctx.h) == tasq.TASQ_ERR_DEVICE
        assert tasq.tasq_device_status(ctx.h) == tasq.TASQ_OK
    finally:
        tasq.tasq_set_stage_device(ctx.h, None)


@pytest.mark.parametrize("code_fmt", ROUTES)
@pytest.mark.parametrize("M,N,K", [(4096, 3456, 1152), (4096, 1152, 4608), (4096, 1152, 1152), (1200, 2240, 2240),
                                   (77, 1280, 2048), (4096, 6720, 2240), (4096, 11200, 2240), (4096, 2240, 5600),
                                   (256, 1280, 5120), (256, 10240, 1280), (1024, 640, 640), (16384, 4096, 4096)])
def test_full_size_sampled_rows(ctx, oracle, code_fmt, M, N, K):
    """Full-size layer shapes of the backbones, checked on sampled token rows
    (the oracle computes those rows one by one)."""
    bits = [3, 8]
    st = _setup_linear(ctx, oracle, M, N, K, bits, seed=K, dtype=tasq.TASQ_BF16, code_fmt=code_fmt)
    rows = np.unique(np.concatenate([np.arange(0, M, max(1, M // 40)), [M - 1]]))
    for stage, b in enumerate(bits):
        y, acc = G.gemm(ctx, 0, stage, st["codes"], code_fmt, st["alpha"], st["zc"], M, st["packed"], N, K)
        _check_layer(oracle, st, b, y, acc, rows=rows)


# ---------------------------------------------- asymmetric weights (zp) --

@pytest.mark.parametrize("dtype", [tasq.TASQ_F32, tasq.TASQ_BF16])
def test_quant_weights_asym_bitexact(ctx, oracle, dtype):
    N, K = 136, 1168
    w = workloads.normal((N, K), seed=71, std=0.02)
    w[::3] += 0.03  # skewed channels
    w[5] = 0.25     # constant channel: alpha = 1, z = -min
    if dtype == tasq.TASQ_BF16:
        wd, w = G.to_bf16(w)
    else:
        wd = G.dev(w)
    sw, cw, zcw, al = G.quant_weights_asym(ctx, wd, dtype, N, K)
    ref = oracle.quant_weight(w, 8, oracle.ASYM)
    assert np.array_equal(sw.cpu().numpy(), ref["s"])
    assert np.array_equal(cw.cpu().numpy(), ref["c"])
    assert np.array_equal(zcw.cpu().numpy(), ref["zcw"])
    assert np.array_equal(al.cpu().numpy(), ref["alpha"])


@pytest.mark.parametrize("code_fmt", [tasq.TASQ_CODES_S8, tasq.TASQ_CODES_F16])
@pytest.mark.parametrize("mode", [tasq.TASQ_SYMRANGE, tasq.TASQ_ASYM])
@pytest.mark.parametrize("M,K", [(70, 1152), (33, 8192)])
def test_quant_act_code_sums_bitexact(ctx, oracle, code_fmt, mode, M, K):
    """Per-token codes with their sums, from the one-pass (rows in registers)
    and the two-pass (K = 8192) kernels."""
    x = workloads.normal((M, K), seed=72)
    x[3] += 2.0
    codes, alpha, zc, sums = G.quant_act_sums(ctx, G.dev(x), tasq.TASQ_F32, M, K, 8, mode, code_fmt)
    s_x, a_ref, z_ref = oracle.quant_act(x, 8, mode, oracle.PER_TOKEN)
    assert np.array_equal(G.codes_to_int8(codes), s_x)
    assert np.array_equal(alpha.cpu().numpy(), a_ref) and np.array_equal(zc.cpu().numpy(), z_ref)
    assert np.array_equal(sums.cpu().numpy(), oracle.code_sums(s_x))


def _setup_linear_zp(ctx, oracle, M, N, K, bits, seed, code_fmt, mode=tasq.TASQ_SYMRANGE, dtype=tasq.TASQ_F32):
    w = workloads.normal((N, K), seed + 1, 0.02)
    w[::2] += 0.02  # half the channels skewed: their zero offsets are far from 0
    bias = workloads.normal((N,), seed + 2, 0.02)
    x = workloads.normal((M, K), seed, 1.0)
    if dtype == tasq.TASQ_BF16:
        xd, x = G.to_bf16(x)
    else:
        xd = G.dev(x)
    sw, cw, zcw, _ = G.quant_weights_asym(ctx, G.dev(w), tasq.TASQ_F32, N, K)
    packed = G.pack_zp(ctx, sw, cw, zcw, G.dev(bias), N, K)
    tasq.tasq_set_schedule(ctx.h, np.asarray([bits], np.uint8), 1, len(bits))
    codes, alpha, zc, sums = G.quant_act_sums(ctx, xd, dtype, M, K, 8, mode, code_fmt)
    wq = oracle.quant_weight(w, 8, oracle.ASYM)
    s_x, a_ref, z_ref = oracle.quant_act(x, 8, mode, oracle.PER_TOKEN)
    return dict(packed=packed, codes=codes, alpha=alpha, zc=zc, sums=sums, wq=wq, s_x=s_x, a=a_ref, z=z_ref,
                bias=bias, K=K)


def _check_layer_zp(oracle, st, b, y, acc, rows=None):
    s_x, a, z = st["s_x"], st["a"], st["z"]
    if rows is not None:
        s_x, a, z = s_x[rows], a[rows], z[rows]
    ref_acc = oracle.gemm(s_x, st["wq"]["s"], b)
    got_acc = acc.cpu().numpy() if rows is None else acc.cpu().numpy()[rows]
    assert np.array_equal(got_acc, ref_acc), f"b={b}: {(got_acc != ref_acc).sum()} int32 mismatches"
    rs = oracle.row_sums(st["wq"]["s"], b)
    _, yb = oracle.epilogue_zp_f32(ref_acc, a, z, oracle.code_sums(s_x), rs, st["wq"]["c"], st["wq"]["zcw"],
                                   st["bias"], st["K"])
    got_y = G.bf16_bits_host(y) if rows is None else G.bf16_bits_host(y)[rows]
    same = G.assert_bf16_close(got_y, yb)
    assert same == yb.size, f"b={b}: {yb.size - same} bf16 outputs differ in the last bit"


@pytest.mark.parametrize("code_fmt", ROUTES)
@pytest.mark.parametrize("M,N,K", [(256, 1152, 1152), (300, 136, 1168), (64, 128, 4096), (4000, 1096, 384),
                                   (1, 8, 16)])
def test_zp_linear_parity(ctx, oracle, code_fmt, M, N, K):
    """Four-term epilogue (asymmetric weights) on every tile configuration of
    the tensor-core route (192-, 256- and 64-token tiles, split K) and on the
    mma.sync route: exact int32 sums and bit-exact bf16 outputs."""
    bits = [8, 5, 3, 2]
    st = _setup_linear_zp(ctx, oracle, M, N, K, bits, seed=M + 5, code_fmt=code_fmt, mode=tasq.TASQ_ASYM)
    for stage, b in enumerate(bits):
        y, acc = G.gemm_zp(ctx, 0, stage, st["codes"], code_fmt, st["alpha"], st["zc"], st["sums"], M, st["packed"],
                           N, K)
        _check_layer_zp(oracle, st, b, y, acc)


@pytest.mark.parametrize("code_fmt", ROUTES)
@pytest.mark.parametrize("zero_point", [False, True])
def test_a4_activations(ctx, oracle, code_fmt, zero_point):
    """4-bit activations (App. A.1.2 with n = 4: codes in [-8, 7], zc = 8 - z)
    through the same contraction, with symmetric or asymmetric weights."""
    M, N, K = 300, 264, 1152
    bits = [8, 4, 2]
    x = workloads.normal((M, K), 81)
    w = workloads.normal((N, K), 82, 0.02)
    w[::2] += 0.02
    bias = workloads.normal((N,), 83, 0.02)
    if zero_point:
        sw, cw, zcw, _ = G.quant_weights_asym(ctx, G.dev(w), tasq.TASQ_F32, N, K)
        packed = G.pack_zp(ctx, sw, cw, zcw, G.dev(bias), N, K)
        wq = oracle.quant_weight(w, 8, oracle.ASYM)
    else:
        sw, cw, _ = G.quant_weights(ctx, G.dev(w), tasq.TASQ_F32, N, K)
        packed = G.pack(ctx, tasq.TASQ_LINEAR, sw, cw, G.dev(bias), N, K)
        wq = oracle.quant_weight(w, 8, oracle.SYMRANGE)
    tasq.tasq_set_schedule(ctx.h, np.asarray([bits], np.uint8), 1, len(bits))
    codes, alpha, zc, sums = G.quant_act_sums(ctx, G.dev(x), tasq.TASQ_F32, M, K, 4, tasq.TASQ_ASYM, code_fmt)
    s_x, a_ref, z_ref = oracle.quant_act(x, 4, oracle.ASYM, oracle.PER_TOKEN)
    assert np.array_equal(G.codes_to_int8(codes), s_x) and s_x.min() >= -8 and s_x.max() <= 7
    for stage, b in enumerate(bits):
        if zero_point:
            y, acc = G.gemm_zp(ctx, 0, stage, codes, code_fmt, alpha, zc, sums, M, packed, N, K)
        else:
            y, acc = G.gemm(ctx, 0, stage, codes, code_fmt, alpha, zc, M, packed, N, K)
        ref_acc = oracle.gemm(s_x, wq["s"], b)
        assert np.array_equal(acc.cpu().numpy(), ref_acc)
        rs = oracle.row_sums(wq["s"], b)
        if zero_point:
            _, yb = oracle.epilogue_zp_f32(ref_acc, a_ref, z_ref, oracle.code_sums(s_x), rs, wq["c"], wq["zcw"],
                                           bias, K)
        else:
            _, yb = oracle.epilogue_f32(ref_acc, a_ref, z_ref, rs, wq["c"], bias)
        assert G.assert_bf16_close(G.bf16_bits_host(y), yb) == yb.size


@pytest.mark.parametrize("code_fmt", ROUTES)
def test_zp_full_size_sampled_rows(ctx, oracle, code_fmt):
    M, N, K = 4096, 3456, 1152
    bits = [4, 8]
    st = _setup_linear_zp(ctx, oracle, M, N, K, bits, seed=9, code_fmt=code_fmt, dtype=tasq.TASQ_BF16)
    rows = np.unique(np.concatenate([np.arange(0, M, max(1, M // 40)), [M - 1]]))
    for stage, b in enumerate(bits):
        y, acc = G.gemm_zp(ctx, 0, stage, st["codes"], code_fmt, st["alpha"], st["zc"], st["sums"], M, st["packed"],
                           N, K)
        _check_layer_zp(oracle, st, b, y, acc, rows=rows)


@pytest.mark.parametrize("code_fmt", ROUTES)
def test_zp_call_on_a_symmetric_pack_equals_the_plain_call(ctx, oracle, code_fmt):
    # a symmetric pack stores zcw = 0: the four-term epilogue gives the two-term result
    M, N, K = 200, 264, 640
    st = _setup_linear(ctx, oracle, M, N, K, [6], code_fmt=code_fmt)
    _, _, _, sums = G.quant_act_sums(ctx, G.dev(workloads.normal((M, K), 0, 1.0)), tasq.TASQ_F32, M, K, 8,
                                     tasq.TASQ_SYMRANGE, code_fmt)
    y0, _ = G.gemm(ctx, 0, 0, st["codes"], code_fmt, st["alpha"], st["zc"], M, st["packed"], N, K)
    y1, _ = G.gemm_zp(ctx, 0, 0, st["codes"], code_fmt, st["alpha"], st["zc"], sums, M, st["packed"], N, K)
    assert np.array_equal(G.bf16_bits_host(y0), G.bf16_bits_host(y1))


@pytest.mark.parametrize("code_fmt", ROUTES)
def test_zp_pack_without_code_sums_is_caught_on_device(ctx, oracle, code_fmt):
    torch = G.torch()
    M, N, K = 128, 128, 256
    st = _setup_linear_zp(ctx, oracle, M, N, K, [8], seed=3, code_fmt=code_fmt)
    y = torch.full((M, N), 0x1234, dtype=torch.int16, device="cuda")
    tasq.tasq_masked_gemm(ctx.h, 0, 0, st["codes"], code_fmt, st["alpha"], st["zc"], M, st["packed"], N, K, y, None)
    assert tasq.tasq_device_status(ctx.h) == tasq.TASQ_ERR_DEVICE
    assert bool((y == 0x1234).all())  # nothing written
    assert tasq.tasq_device_status(ctx.h) == tasq.TASQ_OK


# ------------------------------------------------------------------ conv --

def _run_conv(ctx, oracle, B, H, W, Cin, Cout, bits, code_fmt, seed=0, rows=None):
    torch = G.torch()
    K = 9 * Cin
    x = workloads.normal((B, H, W, Cin), seed)
    w = workloads.normal((Cout, K), seed + 1, 0.02)
    bias = workloads.normal((Cout,), seed + 2, 0.02)
    sw, cw, _ = G.quant_weights(ctx, G.dev(w), tasq.TASQ_F32, Cout, K)
    packed = G.pack(ctx, tasq.TASQ_CONV3X3, sw, cw, G.dev(bias), Cout, K, Cin)
    tasq.tasq_set_schedule(ctx.h, np.asarray([bits], np.uint8), 1, len(bits))
    codes, alpha, zc = G.quant_act(ctx, G.dev(x), tasq.TASQ_F32, B * H * W, Cin, 8, tasq.TASQ_SYMRANGE,
                                   tasq.TASQ_PER_TENSOR, code_fmt)
    wq = oracle.quant_weight(w)
    s_x, a, z = oracle.quant_act(x.reshape(1, -1), 8, 0, 0)
    s_x = s_x.reshape(B, H, W, Cin)
    assert np.array_equal(G.codes_to_int8(codes).reshape(B, H, W, Cin), s_x)
    for stage, b in enumerate(bits):
        y, acc = G.conv(ctx, 0, stage, codes, code_fmt, alpha, zc, B, H, W, Cin, packed, Cout)
        if rows is None:
            ref_acc, rs = oracle.conv3x3(s_x, wq["s"], b)
            got_acc, got_y = acc.cpu().numpy(), G.bf16_bits_host(y)
        else:
            ref_acc, rs = _conv_rows(oracle, s_x, wq["s"], b, rows)
            got_acc, got_y = acc.cpu().numpy()[rows], G.bf16_bits_host(y)[rows]
        assert np.array_equal(got_acc, ref_acc), f"b={b}: {(got_acc != ref_acc).sum()} int32 mismatches"
        _, yb = oracle.epilogue_f32(ref_acc, a, z, rs, wq["c"], bias, per_tensor=True, rs_per_row=True)
        same = G.assert_bf16_close(got_y, yb)
        assert same == yb.size


def _run_conv_zp(ctx, oracle, B, H, W, Cin, Cout, bits, code_fmt, seed=0, rows=None):
    """3x3 conv with asymmetric weights (zero offsets) and per-pixel code sums."""
    K = 9 * Cin
    x = workloads.normal((B, H, W, Cin), seed)
    w = workloads.normal((Cout, K), seed + 1, 0.02)
    w[::2] += 0.02
    bias = workloads.normal((Cout,), seed + 2, 0.02)
    sw, cw, zcw, _ = G.quant_weights_asym(ctx, G.dev(w), tasq.TASQ_F32, Cout, K)
    packed = G.pack_zp(ctx, sw, cw, zcw, G.dev(bias), Cout, K, kind=tasq.TASQ_CONV3X3, Cin=Cin)
    tasq.tasq_set_schedule(ctx.h, np.asarray([bits], np.uint8), 1, len(bits))
    codes, alpha, zc, sums = G.quant_act_sums(ctx, G.dev(x), tasq.TASQ_F32, B * H * W, Cin, 8, tasq.TASQ_ASYM,
                                              code_fmt, gran=tasq.TASQ_PER_TENSOR)
    wq = oracle.quant_weight(w, 8, oracle.ASYM)
    s_x, a, z = oracle.quant_act(x.reshape(1, -1), 8, oracle.ASYM, 0)
    s_x = s_x.reshape(B, H, W, Cin)
    assert np.array_equal(G.codes_to_int8(codes).reshape(B, H, W, Cin), s_x)
    assert np.array_equal(sums.cpu().numpy(), s_x.astype(np.int64).sum(3).reshape(-1))
    sxw, kv = oracle.conv3x3_code_sums(s_x)
    for stage, b in enumerate(bits):
        y = G.empty((B * H * W, Cout), G.torch().int16)
        acc = G.empty((B * H * W, Cout), G.torch().int32)
        tasq.tasq_masked_conv3x3_zp(ctx.h, 0, stage, codes, code_fmt, alpha, zc, sums, B, H, W, Cin, packed, Cout,
                                    y, acc)
        if rows is None:
            ref_acc, rs = oracle.conv3x3(s_x, wq["s"], b)
            got_acc, got_y, sx_r, kv_r = acc.cpu().numpy(), G.bf16_bits_host(y), sxw, kv
        else:
            ref_acc, rs = _conv_rows(oracle, s_x, wq["s"], b, rows)
            got_acc, got_y, sx_r, kv_r = acc.cpu().numpy()[rows], G.bf16_bits_host(y)[rows], sxw[rows], kv[rows]
        assert np.array_equal(got_acc, ref_acc), f"b={b}: {(got_acc != ref_acc).sum()} int32 mismatches"
        _, yb = oracle.conv_epilogue_zp_f32(ref_acc, a[0], z[0], sx_r, kv_r, rs, wq["c"], wq["zcw"], bias)
        same = G.assert_bf16_close(got_y, yb)
        assert same == yb.size, f"b={b}: {yb.size - same} bf16 outputs differ in the last bit"


@pytest.mark.parametrize("code_fmt", ROUTES)
@pytest.mark.parametrize("B,H,W,Cin,Cout", [(1, 8, 8, 64, 16), (2, 5, 7, 64, 24), (1, 1, 1, 128, 8),
                                            (2, 16, 16, 64, 256), (1, 4, 4, 1280, 128)])
def test_conv_zp_small_full(ctx, oracle, code_fmt, B, H, W, Cin, Cout):
    """Asymmetric-weight convs checked in full: borders and corners (windowed code
    sums over in-bounds taps only), a 1x1 image, several tile configurations and a
    long K (9 * 1280, split K)."""
    _run_conv_zp(ctx, oracle, B, H, W, Cin, Cout, [8, 5, 2], code_fmt, seed=B * 7 + H)


@pytest.mark.parametrize("code_fmt", ROUTES)
def test_conv_zp_full_size_sampled(ctx, oracle, code_fmt):
    B, C, HW = 1, 320, 64
    P = B * HW * HW
    rows = np.unique(np.concatenate([np.arange(0, P, 97), [0, HW - 1, P - HW, P - 1]]))
    _run_conv_zp(ctx, oracle, B, HW, HW, C, C, [4, 8], code_fmt, seed=5, rows=rows)


def _conv_rows(oracle, s_x, s_w, b, rows):
    """Oracle conv restricted to output pixels `rows`: each pixel's 3x3
    neighbourhood is cut out (zero code padding outside the image) and run
    through the oracle conv on a 3x3 image, whose centre pixel is the wanted one."""
    B, H, W, Cin = s_x.shape
    acc_out, rs_out = [], []
    for p in rows:
        bb, h, w = p // (H * W), (p // W) % H, p % W
        patch = np.zeros((1, 3, 3, Cin), np.int8)
        valid = np.zeros((3, 3), bool)
        for dh in range(3):
            for dw in range(3):
                ih, iw = h + dh - 1, w + dw - 1
                if 0 <= ih < H and 0 <= iw < W:
                    patch[0, dh, dw] = s_x[bb, ih, iw]
                    valid[dh, dw] = True
        acc, _ = oracle.conv3x3(patch, s_w, b)
        acc_out.append(acc[4])
        m = oracle.mask(s_w, b).astype(np.int64).reshape(s_w.shape[0], 3, 3, Cin).sum(3)
        rs_out.append((m * valid[None]).sum((1, 2)).astype(np.int32))
    return np.stack(acc_out), np.stack(rs_out)


@pytest.mark.parametrize("code_fmt", ROUTES)
@pytest.mark.parametrize("B,H,W,Cin,Cout", [(1, 8, 8, 64, 16), (2, 5, 7, 64, 24), (1, 1, 1, 128, 8), (1, 3, 1, 64, 136),
                                            (1, 9, 13, 192, 40), (2, 16, 16, 64, 256)])
def test_conv_small_full(ctx, oracle, code_fmt, B, H, W, Cin, Cout):
    _run_conv(ctx, oracle, B, H, W, Cin, Cout, [8, 4, 6], code_fmt)


@pytest.mark.parametrize("B,H,W,Cin,Cout", [(1, 8, 8, 32, 16), (2, 5, 7, 16, 24), (1, 1, 1, 48, 8)])
def test_conv_narrow_channels(ctx, oracle, B, H, W, Cin, Cout):
    """Cin % 16 == 0 but not % 64: the int8 route runs it; the tensor-core
    route (whose 64-wide K blocks must not straddle a tap) refuses it."""
    _run_conv(ctx, oracle, B, H, W, Cin, Cout, [8, 4, 6], tasq.TASQ_CODES_S8)
    with pytest.raises(tasq.TasqError) as e:
        _run_conv(ctx, oracle, B, H, W, Cin, Cout, [8], tasq.TASQ_CODES_F16)
    assert e.value.code == tasq.TASQ_ERR_UNSUPPORTED


@pytest.mark.parametrize("code_fmt", ROUTES)
@pytest.mark.parametrize("C,HW,Cout", [(320, 64, 320), (640, 32, 640), (1280, 16, 1280), (64, 64, 1024)])
def test_conv_full_size_sampled(ctx, oracle, code_fmt, C, HW, Cout):
    """Full-size convolutions on sampled output pixels (borders included); the
    64-channel, 1024-output case runs the wide single-tile configuration."""
    rng = workloads.rng(C)
    P = HW * HW
    border = [0, HW - 1, HW * (HW - 1), P - 1, HW // 2, HW * (HW // 2)]
    rows = np.unique(np.concatenate([border, rng.integers(0, P, 24)]))
    _run_conv(ctx, oracle, 1, HW, HW, C, Cout, [5, 8], code_fmt, seed=C, rows=rows)


# ------------------------------------------------------ failure handling --

def test_invalid_arguments_launch_nothing(ctx):
    torch = G.torch()
    buf = torch.zeros((1 << 16,), dtype=torch.uint8, device="cuda")
    with pytest.raises(tasq.TasqError) as e:
        tasq.tasq_set_schedule(ctx.h, np.array([[9]], np.uint8), 1, 1)
    assert e.value.code == tasq.TASQ_ERR_INVALID_ARG
    tasq.tasq_set_schedule(ctx.h, np.array([[8, 4]], np.uint8), 1, 2)
    cases = [
        dict(layer=1, stage=0, K=64, N=64, code=tasq.TASQ_ERR_INVALID_ARG),
        dict(layer=0, stage=2, K=64, N=64, code=tasq.TASQ_ERR_INVALID_ARG),
        dict(layer=0, stage=-1, K=64, N=64, code=tasq.TASQ_ERR_INVALID_ARG),
        dict(layer=0, stage=0, K=40, N=64, code=tasq.TASQ_ERR_UNSUPPORTED),
        dict(layer=0, stage=0, K=64, N=60, code=tasq.TASQ_ERR_UNSUPPORTED),
    ]
    for c in cases:
        with pytest.raises(tasq.TasqError) as e:
            tasq.tasq_masked_gemm(ctx.h, c["layer"], c["stage"], buf, tasq.TASQ_CODES_S8, buf, buf, 16, buf, c["N"],
                                  c["K"], buf, None)
        assert e.value.code == c["code"], c
    with pytest.raises(tasq.TasqError) as e:  # misaligned output pointer
        tasq.tasq_masked_gemm(ctx.h, 0, 0, buf, tasq.TASQ_CODES_S8, buf, buf, 16, buf, 64, 64, buf.data_ptr() + 2, None)
    assert e.value.code == tasq.TASQ_ERR_UNSUPPORTED
    with pytest.raises(tasq.TasqError) as e:  # route and code storage disagree
        tasq.tasq_set_route(ctx.h, tasq.TASQ_ROUTE_TC)
        tasq.tasq_masked_gemm(ctx.h, 0, 0, buf, tasq.TASQ_CODES_S8, buf, buf, 16, buf, 64, 64, buf, None)
    tasq.tasq_set_route(ctx.h, tasq.TASQ_ROUTE_AUTO)
    assert e.value.code == tasq.TASQ_ERR_UNSUPPORTED
    assert tasq.tasq_device_status(ctx.h) == tasq.TASQ_OK


def test_packed_buffer_mismatch_is_caught_on_device(ctx, oracle):
    torch = G.torch()
    N, K = 64, 128
    sw = torch.zeros((N, K), dtype=torch.int8, device="cuda")
    cw = torch.ones((N,), dtype=torch.float32, device="cuda")
    packed = G.pack(ctx, tasq.TASQ_LINEAR, sw, cw, None, N, K)
    tasq.tasq_set_schedule(ctx.h, np.array([[8]], np.uint8), 1, 1)
    codes = torch.zeros((16, 64), dtype=torch.int8, device="cuda")
    al = torch.ones((16,), dtype=torch.float32, device="cuda")
    y = torch.zeros((16, 64), dtype=torch.int16, device="cuda")
    tasq.tasq_masked_gemm(ctx.h, 0, 0, codes, tasq.TASQ_CODES_S8, al, al, 16, packed, 64, 64, y, None)  # K mismatch
    assert tasq.tasq_device_status(ctx.h) == tasq.TASQ_ERR_DEVICE


def test_device_wait_timeout_is_reported_and_context_survives(ctx, oracle):
    tasq.tasq_selftest_timeout(ctx.h, 50_000_000)  # 50 ms wait on a barrier nothing arrives at
    assert tasq.tasq_device_status(ctx.h) == tasq.TASQ_ERR_DEVICE_TIMEOUT
    assert tasq.tasq_device_status(ctx.h) == tasq.TASQ_OK
    # the context still computes correctly afterwards
    M, N, K = 64, 64, 128
    st = _setup_linear(ctx, oracle, M, N, K, [7], code_fmt=tasq.TASQ_CODES_S8)
    y, acc = G.gemm(ctx, 0, 0, st["codes"], tasq.TASQ_CODES_S8, st["alpha"], st["zc"], M, st["packed"], N, K)
    _check_layer(oracle, st, 7, y, acc)


def test_quotient_routine_matches_ieee_division(ctx):
    """The activation quantizer's x / alpha (reciprocal once per group, two
    exact remainder corrections) equals IEEE round-to-nearest division for
    every finite bf16 dividend against divisors spanning the normal range."""
    torch = G.torch()
    bits = np.arange(1 << 16, dtype=np.uint32)
    xs = (bits << 16).view(np.float32)
    e = (bits >> 7) & 0xFF
    xs = xs[(e > 30) & (e < 225)]  # normal dividends, quotients stay normal
    rng = workloads.rng(5)
    a = np.concatenate([np.exp2(rng.uniform(-30, 30, 2000)), 2.0 ** np.arange(-30, 31),
                        rng.uniform(1e-3, 5e-2, 1000)]).astype(np.float32)
    mism = torch.zeros((1,), dtype=torch.int64, device="cuda")
    tasq.tasq_selftest_quotients(ctx.h, G.dev(xs), xs.size, G.dev(a), a.size, mism)
    torch.cuda.synchronize()
    assert int(mism.item()) == 0



def test_quotient_routine_matches_ieee_division_fp32(ctx):
    """The same quotient routine on fp32 dividends (the per-token quantizer of an
    fp32 input divides fp32 values): 10^8 seeded random bit patterns with
    exponents that keep every quotient normal, against the same divisor set as
    the bf16 test above.  Zero mismatches expected."""
    torch = G.torch()
    rng = workloads.rng(5)
    a = np.concatenate([np.exp2(rng.uniform(-30, 30, 2000)), 2.0 ** np.arange(-30, 31),
                        rng.uniform(1e-3, 5e-2, 1000)]).astype(np.float32)
    ad = G.dev(a)
    gen = torch.Generator(device="cuda")
    gen.manual_seed(12)
    mism = torch.zeros((1,), dtype=torch.int64, device="cuda")
    total = 0
    while total < 100_000_000:
        bits = torch.randint(-(2 ** 31), 2 ** 31 - 1, (30_000_000,), dtype=torch.int32, generator=gen, device="cuda")
        e = (bits >> 23) & 0xFF
        xs = bits[(e > 30) & (e < 225)].view(torch.float32).contiguous()
        tasq.tasq_selftest_quotients(ctx.h, xs, xs.numel(), ad, a.size, mism)
        total += xs.numel()
        del bits, e, xs
    torch.cuda.synchronize()
    assert total >= 100_000_000
    assert int(mism.item()) == 0


# --------------------------------------- the sweep's shapes, uniform codes --

SWEEP = [(M, KN) for M in (1024, 4096, 16384) for KN in (1152, 2240, 4096)]


@pytest.mark.parametrize("M,KN", SWEEP)
def test_sweep_shapes_uniform_codes(ctx, oracle, M, KN):
    """The shape sweep at its own shapes: codes uniform in [-127, 127] for
    activations and weights (sums of |w| far past one fp32-exact chunk), every
    b = 2..8, on the tensor-core route.  The output is checked on sampled token
    rows plus the last row, for the call without the int32 debug output (the
    call the benchmark times) and, with it, the int32 accumulators as well.
    M = 1024, K = N = 4096 runs the 256-token single-accumulator tiles over
    several certified chunks."""
    torch = G.torch()
    N = K = KN
    F16 = tasq.TASQ_CODES_F16
    seed = 1000 + M + KN
    s_x = workloads.uniform_codes((M, K), seed)
    s_w = workloads.uniform_codes((N, K), seed + 1)
    cw = workloads.uniform((N,), seed + 2, 1e-4, 2e-4)
    bias = workloads.normal((N,), seed + 3, 0.02)
    alpha = workloads.uniform((M,), seed + 4, 1e-3, 2e-3)
    zc = workloads.uniform((M,), seed + 5, -0.5, 0.5)
    packed = G.pack(ctx, tasq.TASQ_LINEAR, G.dev(s_w), G.dev(cw), G.dev(bias), N, K)
    bits = list(range(2, 9))
    tasq.tasq_set_schedule(ctx.h, np.array([bits], np.uint8), 1, len(bits))
    codes = G.dev(s_x).to(torch.float16)
    ad, zd = G.dev(alpha), G.dev(zc)
    sms = torch.cuda.get_device_properties(0).multi_processor_count
    plan = tasq.tasq_plan_tc(tasq.TASQ_LINEAR, M, N, K, 0, 0, 0, 0, sms)
    chunk_kb, _ = G.packed_header(packed)
    KT = (K + 127) // 128
    nchunks = {b: -(-KT // max(1, min(KT, int(chunk_kb[b]) // 2))) for b in bits}
    if (M, KN) == (1024, 4096) and sms >= 128:
        assert plan["tile_tokens"] == 256 and plan["acc_buffers"] == 1, plan
        assert nchunks[8] > 1, nchunks
    rows = np.unique(np.concatenate([np.arange(0, M, max(1, M // 40)), [M - 1]]))
    rows_d = torch.from_numpy(rows).cuda()
    y_prod = G.empty((M, N), torch.int16)
    for stage, b in enumerate(bits):
        tasq.tasq_masked_gemm(ctx.h, 0, stage, codes, F16, ad, zd, M, packed, N, K, y_prod, None)
        y_dbg, acc = G.gemm(ctx, 0, stage, codes, F16, ad, zd, M, packed, N, K)
        ref_acc = oracle.gemm(s_x[rows], s_w, b)
        got_acc = acc.index_select(0, rows_d).cpu().numpy()
        assert np.array_equal(got_acc, ref_acc), f"b={b}: {(got_acc != ref_acc).sum()} int32 mismatches"
        _, yb = oracle.epilogue_f32(ref_acc, alpha[rows], zc[rows], oracle.row_sums(s_w, b), cw, bias)
        for y in (y_prod, y_dbg):
            got = G.bf16_bits_host(y.index_select(0, rows_d))
            assert G.assert_bf16_close(got, yb) == yb.size, f"b={b}: bf16 outputs differ in the last bit"
        del y_dbg, acc
    assert tasq.tasq_device_status(ctx.h) == tasq.TASQ_OK


# ------------------------- the product call (no int32 output) vs the oracle --

@pytest.mark.parametrize("code_fmt", ROUTES)
@pytest.mark.parametrize("M,N,K,full", [
    (4096, 3456, 1152, False),  # 192-token tiles, two accumulators, persistent
    (4000, 1096, 384, True),    # 256-token tiles, one accumulator, ragged tiles
    (300, 1152, 1152, True),    # 64-token tiles, K split over slices
    (77, 640, 2048, True),      # 64-token tiles, split K, ragged tokens
    (1024, 4096, 4096, False),  # 256-token tiles over several certified chunks (N(0, 0.02) weights: one chunk)
])
def test_product_call_matches_oracle(ctx, oracle, code_fmt, M, N, K, full):
    """tasq_masked_gemm with d_acc = NULL -- the call a network makes -- against
    the oracle's bf16 output (not against the GPU's own debug call), one shape
    per tile configuration of the tensor-core route."""
    torch = G.torch()
    bits = [8, 4, 2]
    st = _setup_linear(ctx, oracle, M, N, K, bits, seed=M + K + 17, dtype=tasq.TASQ_BF16, code_fmt=code_fmt)
    rows = np.arange(M) if full else np.unique(np.concatenate([np.arange(0, M, max(1, M // 48)), [M - 1]]))
    rows_d = torch.from_numpy(rows).cuda()
    for stage, b in enumerate(bits):
        y, _ = G.gemm(ctx, 0, stage, st["codes"], code_fmt, st["alpha"], st["zc"], M, st["packed"], N, K,
                      want_acc=False)
        ref_acc = oracle.gemm(st["s_x"][rows], st["wq"]["s"], b)
        _, yb = oracle.epilogue_f32(ref_acc, st["a"][rows], st["z"][rows], oracle.row_sums(st["wq"]["s"], b),
                                    st["wq"]["c"], st["bias"])
        got = G.bf16_bits_host(y.index_select(0, rows_d))
        assert G.assert_bf16_close(got, yb) == yb.size, f"b={b}"
    assert tasq.tasq_device_status(ctx.h) == tasq.TASQ_OK


@pytest.mark.parametrize("code_fmt", ROUTES)
def test_conv_product_call_matches_oracle(ctx, oracle, code_fmt):
    """tasq_masked_conv3x3 with d_acc = NULL against the oracle's bf16 output
    (full check, border pixels included)."""
    B, H, W, Cin, Cout = 1, 12, 20, 64, 136
    x = workloads.normal((B, H, W, Cin), 301)
    w = workloads.normal((Cout, 9 * Cin), 302, 0.03)
    bias = workloads.normal((Cout,), 303, 0.02)
    sw, cw, _ = G.quant_weights(ctx, G.dev(w), tasq.TASQ_F32, Cout, 9 * Cin)
    packed = G.pack(ctx, tasq.TASQ_CONV3X3, sw, cw, G.dev(bias), Cout, 9 * Cin, Cin)
    tasq.tasq_set_schedule(ctx.h, np.array([[7, 3]], np.uint8), 1, 2)
    M = B * H * W
    codes, alpha, zc = G.quant_act(ctx, G.dev(x), tasq.TASQ_F32, M, Cin, 8, tasq.TASQ_SYMRANGE,
                                   tasq.TASQ_PER_TENSOR, code_fmt)
    wq = oracle.quant_weight(w)
    s_x, a, z = oracle.quant_act(x.reshape(1, -1), 8, oracle.SYMRANGE, oracle.PER_TOKEN)
    for stage, b in enumerate([7, 3]):
        y, _ = G.conv(ctx, 0, stage, codes, code_fmt, alpha, zc, B, H, W, Cin, packed, Cout, want_acc=False)
        acc, rs = oracle.conv3x3(s_x.reshape(B, H, W, Cin), wq["s"], b)
        _, yb = oracle.epilogue_f32(acc, a, z, rs, wq["c"], bias, per_tensor=True, rs_per_row=True)
        assert G.assert_bf16_close(G.bf16_bits_host(y), yb) == yb.size, f"b={b}"


# -------------------------------- a captured graph follows the bit table --

def test_graph_replay_follows_schedule_updates(ctx, oracle):
    """A CUDA graph captured once keeps reading the context's bit table: after a
    same-size tasq_set_schedule its replay runs the new bits; after a smaller
    schedule that no longer holds the captured stage, the replay records
    TASQ_ERR_DEVICE and writes nothing."""
    torch = G.torch()
    M, N, K = 256, 384, 640
    st = _setup_linear(ctx, oracle, M, N, K, [8, 6], seed=77, code_fmt=tasq.TASQ_CODES_F16)
    F16 = tasq.TASQ_CODES_F16
    y = G.empty((M, N), torch.int16)

    def call():
        tasq.tasq_masked_gemm(ctx.h, 0, 1, st["codes"], F16, st["alpha"], st["zc"], M, st["packed"], N, K, y, None)

    call()
    torch.cuda.synchronize()
    s = torch.cuda.Stream()
    s.wait_stream(torch.cuda.current_stream())
    g = torch.cuda.CUDAGraph()
    with torch.cuda.stream(s), torch.cuda.graph(g, stream=s):
        call()

    def expect(b):
        ref_acc = oracle.gemm(st["s_x"], st["wq"]["s"], b)
        _, yb = oracle.epilogue_f32(ref_acc, st["a"], st["z"], oracle.row_sums(st["wq"]["s"], b), st["wq"]["c"],
                                    st["bias"])
        return yb

    for table, b in (([[8, 6]], 6), ([[5, 3]], 3), ([[2, 7]], 7)):
        tasq.tasq_set_schedule(ctx.h, np.array(table, np.uint8), 1, 2)
        y.fill_(0)
        g.replay()
        torch.cuda.synchronize()
        assert np.array_equal(G.bf16_bits_host(y), expect(b)), table
    assert tasq.tasq_device_status(ctx.h) == tasq.TASQ_OK
    # one stage only: the captured stage 1 is now out of range
    tasq.tasq_set_schedule(ctx.h, np.array([[4]], np.uint8), 1, 1)
    y.fill_(0)
    g.replay()
    assert tasq.tasq_device_status(ctx.h) == tasq.TASQ_ERR_DEVICE
    assert not bool(y.any())


# --------------------------------------------- grouped contraction call --

@pytest.mark.parametrize("code_fmt", ROUTES)
@pytest.mark.parametrize("M,Ng,K,G", [(300, 1152, 1152, 2), (77, 1280, 2048, 2), (513, 136, 1168, 3),
                                      (129, 264, 2240, 4)])
def test_grouped_members_match_single_layers(ctx, oracle, code_fmt, M, Ng, K, G):
    """One grouped launch over G layers that share their activations (weights
    packed once, concatenated along N) equals, member by member, the oracle's
    single layer at that member's own b.  Members straddle 128-channel tiles
    (Ng = 136, 264) and two shapes split K on the tensor-core route."""
    N = G * Ng
    w = workloads.normal((N, K), 400 + M, 0.02)
    bias = workloads.normal((N,), 401 + M, 0.02)
    x = workloads.normal((M, K), 402 + M)
    sw, cw, _ = GL.quant_weights(ctx, GL.dev(w), tasq.TASQ_F32, N, K)
    packed = GL.pack(ctx, tasq.TASQ_LINEAR, sw, cw, GL.dev(bias), N, K)
    table = np.array([[8, 3], [2, 7], [5, 5], [6, 4]], np.uint8)
    tasq.tasq_set_schedule(ctx.h, table, 4, 2)
    layers = [2, 0, 3, 1][:G]
    codes, alpha, zc = GL.quant_act(ctx, GL.dev(x), tasq.TASQ_F32, M, K, 8, tasq.TASQ_SYMRANGE,
                                    tasq.TASQ_PER_TOKEN, code_fmt)
    wq = oracle.quant_weight(w)
    s_x, a, z = oracle.quant_act(x)
    for stage in range(2):
        for want_acc in (True, False):
            y = GL.empty((M, N), GL.torch().int16)
            acc = GL.empty((M, N), GL.torch().int32) if want_acc else None
            tasq.tasq_masked_gemm_grouped(ctx.h, layers, stage, codes, code_fmt, alpha, zc, M, packed, N, K, y, acc)
            yh = GL.bf16_bits_host(y)
            acch = acc.cpu().numpy() if want_acc else None
            for g, layer in enumerate(layers):
                b = int(table[layer, stage])
                sl = slice(g * Ng, (g + 1) * Ng)
                ref = oracle.gemm(s_x, wq["s"][sl], b)
                if want_acc:
                    assert np.array_equal(acch[:, sl], ref), (g, b)
                _, yb = oracle.epilogue_f32(ref, a, z, oracle.row_sums(wq["s"][sl], b), wq["c"][sl], bias[sl])
                assert GL.assert_bf16_close(yh[:, sl], yb) == yb.size, (g, b)
    assert tasq.tasq_device_status(ctx.h) == tasq.TASQ_OK


def test_grouped_call_rejects_bad_groups(ctx):
    torch = GL.torch()
    buf = torch.zeros((1 << 16,), dtype=torch.uint8, device="cuda")
    tasq.tasq_set_schedule(ctx.h, np.array([[8], [4]], np.uint8), 2, 1)
    F16 = tasq.TASQ_CODES_F16
    for layers, N, code in (([0, 1, 0, 1, 0], 80, tasq.TASQ_ERR_INVALID_ARG),  # more than 4 members
                            ([0, 2], 64, tasq.TASQ_ERR_INVALID_ARG),           # no layer 2
                            ([0, 1, 1], 64, tasq.TASQ_ERR_UNSUPPORTED),        # 64 channels do not split in 3
                            ([0, 1], 40, tasq.TASQ_ERR_UNSUPPORTED)):          # 20-channel members
        with pytest.raises(tasq.TasqError) as e:
            tasq.tasq_masked_gemm_grouped(ctx.h, layers, 0, buf, F16, buf, buf, 16, buf, N, 64, buf, None)
        assert e.value.code == code, layers
    assert tasq.tasq_device_status(ctx.h) == tasq.TASQ_OK


# ------------------------------- e5m2 codes: the K loop on the 8-bit-float MMA kind --

F8 = tasq.TASQ_CODES_F16_E5M2


def _e5m2_part(codes, M, K):
    """The e5m2 copy that follows the M x K fp16 codes, decoded on the host."""
    torch = G.torch()
    raw = codes.view(torch.uint8)[2 * M * K:3 * M * K].cpu()
    return raw.view(torch.float8_e5m2).float().numpy().reshape(M, K)


@pytest.mark.parametrize("n_bits", [2, 3, 4])
@pytest.mark.parametrize("gran", [tasq.TASQ_PER_TOKEN, tasq.TASQ_PER_TENSOR])
@pytest.mark.parametrize("dtype", [tasq.TASQ_F32, tasq.TASQ_BF16])
def test_quant_act_e5m2_copy_bitexact(ctx, oracle, n_bits, gran, dtype):
    """TASQ_CODES_F16_E5M2: the fp16 codes equal the oracle's codes, and the e5m2
    copy after them holds the same integers, element for element."""
    torch = G.torch()
    M, K = 333, 1152 if gran == tasq.TASQ_PER_TOKEN else 640
    x = workloads.normal((M, K), 71 + n_bits)
    x[5, 7] = 9.0
    if dtype == tasq.TASQ_BF16:
        xd, x = G.to_bf16(x)
    else:
        xd = G.dev(x)
    codes = G.empty((3 * M * K // 2,), torch.float16)  # 3 M K bytes
    g = 1 if gran == tasq.TASQ_PER_TENSOR else M
    alpha, zc = G.empty((g,), torch.float32), G.empty((g,), torch.float32)
    tasq.tasq_quant_act(ctx.h, xd, dtype, M, K, n_bits, tasq.TASQ_SYMRANGE, gran, codes, F8, alpha, zc)
    torch.cuda.synchronize()
    if gran == tasq.TASQ_PER_TOKEN:
        s, a, z = oracle.quant_act(x, n_bits, oracle.SYMRANGE, oracle.PER_TOKEN)
    else:
        s, a, z = oracle.quant_act(x.reshape(1, -1), n_bits, oracle.SYMRANGE, oracle.PER_TOKEN)
        s = s.reshape(M, K)
    f16 = codes[:M * K].float().cpu().numpy().reshape(M, K)
    assert np.array_equal(f16, s.astype(np.float32))
    assert np.array_equal(_e5m2_part(codes, M, K), s.astype(np.float32))
    assert np.array_equal(alpha.cpu().numpy(), a) and np.array_equal(zc.cpu().numpy(), z)


def test_e5m2_codes_need_four_bits_or_fewer(ctx):
    torch = G.torch()
    buf = torch.zeros((1 << 16,), dtype=torch.uint8, device="cuda")
    with pytest.raises(tasq.TasqError) as e:
        tasq.tasq_quant_act(ctx.h, buf, tasq.TASQ_F32, 16, 64, 5, tasq.TASQ_SYMRANGE, tasq.TASQ_PER_TOKEN, buf, F8,
                            buf, buf)
    assert e.value.code == tasq.TASQ_ERR_UNSUPPORTED


def _setup_f8(ctx, oracle, M, N, K, bits, seed, n_bits=4, uniform_w=False):
    w = workloads.normal((N, K), seed + 1, 0.02)
    bias = workloads.normal((N,), seed + 2, 0.02)
    x = workloads.normal((M, K), seed)
    if uniform_w:
        s_w = workloads.uniform_codes((N, K), seed + 3)
        cw = workloads.uniform((N,), seed + 4, 1e-4, 2e-4)
        packed = G.pack(ctx, tasq.TASQ_LINEAR, G.dev(s_w), G.dev(cw), G.dev(bias), N, K)
        wq = dict(s=s_w, c=cw)
    else:
        sw, cw, _ = G.quant_weights(ctx, G.dev(w), tasq.TASQ_F32, N, K)
        packed = G.pack(ctx, tasq.TASQ_LINEAR, sw, cw, G.dev(bias), N, K)
        wq = oracle.quant_weight(w)
    tasq.tasq_set_schedule(ctx.h, np.array([bits], np.uint8), 1, len(bits))
    torch = G.torch()
    codes = G.empty((3 * M * K // 2,), torch.float16)
    alpha, zc = G.empty((M,), torch.float32), G.empty((M,), torch.float32)
    tasq.tasq_quant_act(ctx.h, G.dev(x), tasq.TASQ_F32, M, K, n_bits, tasq.TASQ_SYMRANGE, tasq.TASQ_PER_TOKEN, codes,
                        F8, alpha, zc)
    s_x, a, z = oracle.quant_act(x, n_bits, oracle.SYMRANGE, oracle.PER_TOKEN)
    return dict(packed=packed, codes=codes, alpha=alpha, zc=zc, wq=wq, s_x=s_x, a=a, z=z, bias=bias)


@pytest.mark.parametrize("M,N,K,full", [
    (256, 1152, 1152, True),    # 64-token tiles
    (4000, 1096, 384, True),    # 256-token tiles, one accumulator: two activation stages per 256-code block
    (4096, 3456, 1152, False),  # 192-token tiles, two accumulators
    (77, 640, 2048, True),      # 64-token tiles, split K
    (513, 72, 64, True),        # K shorter than one block
    (300, 136, 1168, True),     # ragged last K block
])
@pytest.mark.parametrize("n_bits", [3, 4])
def test_f8_route_every_b(ctx, oracle, M, N, K, full, n_bits):
    """Codes in the dual format: at b <= 4 the K loop runs on the e5m2 MMA kind
    (unsplit launches), at b = 5..8 on the fp16 codes; every b gives the oracle's
    exact int32 accumulators and bf16 outputs, with and without the int32 output."""
    torch = G.torch()
    bits = list(range(2, 9))
    st = _setup_f8(ctx, oracle, M, N, K, bits, seed=M + N + n_bits, n_bits=n_bits)
    rows = np.arange(M) if full else np.unique(np.concatenate([np.arange(0, M, max(1, M // 48)), [M - 1]]))
    rows_d = torch.from_numpy(rows).cuda()
    y_prod = G.empty((M, N), torch.int16)
    for stage, b in enumerate(bits):
        tasq.tasq_masked_gemm(ctx.h, 0, stage, st["codes"], F8, st["alpha"], st["zc"], M, st["packed"], N, K, y_prod,
                              None)
        y, acc = G.gemm(ctx, 0, stage, st["codes"], F8, st["alpha"], st["zc"], M, st["packed"], N, K)
        ref = oracle.gemm(st["s_x"][rows], st["wq"]["s"], b)
        got = acc.index_select(0, rows_d).cpu().numpy()
        assert np.array_equal(got, ref), f"b={b}: {(got != ref).sum()} int32 mismatches"
        _, yb = oracle.epilogue_f32(ref, st["a"][rows], st["z"][rows], oracle.row_sums(st["wq"]["s"], b),
                                    st["wq"]["c"], st["bias"])
        for yy in (y, y_prod):
            assert G.assert_bf16_close(G.bf16_bits_host(yy.index_select(0, rows_d)), yb) == yb.size, b
    assert tasq.tasq_device_status(ctx.h) == tasq.TASQ_OK


def test_f8_route_uniform_codes(ctx, oracle):
    """Uniform weight codes in [-127, 127] and K = 4096 at M = 1024 (single-
    accumulator tiles), on either path."""
    torch = G.torch()
    M, N, K = 1024, 4096, 4096
    bits = [2, 4, 5, 8]
    st = _setup_f8(ctx, oracle, M, N, K, bits, seed=91, uniform_w=True)
    rows = np.unique(np.concatenate([np.arange(0, M, 37), [M - 1]]))
    rows_d = torch.from_numpy(rows).cuda()
    for stage, b in enumerate(bits):
        y, acc = G.gemm(ctx, 0, stage, st["codes"], F8, st["alpha"], st["zc"], M, st["packed"], N, K)
        ref = oracle.gemm(st["s_x"][rows], st["wq"]["s"], b)
        assert np.array_equal(acc.index_select(0, rows_d).cpu().numpy(), ref), b


def test_f8_codes_lengthen_the_exact_chunk(ctx, oracle):
    """Codes of magnitude <= 8 (the e5m2 format) let an exact fp32 chunk run 16
    times as far as the run certified for 8-bit codes.  Odd extreme operands
    (weight codes +127 / -125, activation code 7 on the positive rows; -8 on
    the others) over K = 40960 make the positive rows' products odd and the row
    totals ~2^25, so a chunk one doubling too long would round its fp32 partial
    sum; at b = 8 (fp16 codes) and b = 4 (e5m2 kind, a multiple of 16 per
    product) the int32 accumulators must equal the oracle's."""
    torch = G.torch()
    M, N, K = 640, 1152, 40960  # 90 tiles of 64 tokens: one unsplit wave
    col = torch.where(torch.arange(N, device="cuda") % 2 == 0, 127, -125).to(torch.int8)
    s_w = col[:, None].expand(N, K).contiguous()
    cw = torch.full((N,), 1e-4, device="cuda")
    packed = G.pack(ctx, tasq.TASQ_LINEAR, s_w, cw, None, N, K)
    sign = torch.where(torch.arange(M, device="cuda") % 3 == 0, -1.0, 1.0)
    x = sign[:, None].expand(M, K).contiguous()
    bits = [8, 4]
    tasq.tasq_set_schedule(ctx.h, np.array([bits], np.uint8), 1, len(bits))
    codes = G.empty((3 * M * K // 2,), torch.float16)
    alpha, zc = G.empty((M,), torch.float32), G.empty((M,), torch.float32)
    tasq.tasq_quant_act(ctx.h, x, tasq.TASQ_F32, M, K, 4, tasq.TASQ_SYMRANGE, tasq.TASQ_PER_TOKEN, codes, F8,
                        alpha, zc)
    rows = np.array([0, 1, 2, 300, M - 1])
    s_x, _, _ = oracle.quant_act(np.where(rows % 3 == 0, -1.0, 1.0)[:, None] * np.ones((1, K)), 4, oracle.SYMRANGE,
                                 oracle.PER_TOKEN)
    assert np.array_equal(codes[:M * K].view(M, K)[torch.from_numpy(rows).cuda()].cpu().numpy(), s_x)
    assert (s_x[rows % 3 != 0] == 7).all()  # odd codes on the positive rows
    s_w_host = np.where(np.arange(N) % 2 == 0, 127, -125).astype(np.int8)[:, None] * np.ones((1, K), np.int8)
    for stage, b in enumerate(bits):
        _, acc = G.gemm(ctx, 0, stage, codes, F8, alpha, zc, M, packed, N, K)
        ref = oracle.gemm(s_x, s_w_host, b)
        assert np.abs(ref).max() > 2 ** 24
        got = acc.index_select(0, torch.from_numpy(rows).cuda()).cpu().numpy()
        assert np.array_equal(got, ref), f"b={b}: {(got != ref).sum()} mismatches"
    assert tasq.tasq_device_status(ctx.h) == tasq.TASQ_OK


def test_f8_route_grouped_members_choose_the_path_together(ctx, oracle):
    """A grouped call runs on the e5m2 kind only when every member's b is <= 4;
    either way each member equals the oracle's single layer at its b."""
    torch = G.torch()
    M, Ng, K = 300, 1152, 1152
    N = 2 * Ng
    w = workloads.normal((N, K), 501, 0.02)
    bias = workloads.normal((N,), 502, 0.02)
    x = workloads.normal((M, K), 503)
    sw, cw, _ = G.quant_weights(ctx, G.dev(w), tasq.TASQ_F32, N, K)
    packed = G.pack(ctx, tasq.TASQ_LINEAR, sw, cw, G.dev(bias), N, K)
    table = np.array([[3, 4], [2, 7]], np.uint8)  # stage 0: (3, 2) e5m2; stage 1: (4, 7) fp16
    tasq.tasq_set_schedule(ctx.h, table, 2, 2)
    codes = G.empty((3 * M * K // 2,), torch.float16)
    alpha, zc = G.empty((M,), torch.float32), G.empty((M,), torch.float32)
    tasq.tasq_quant_act(ctx.h, G.dev(x), tasq.TASQ_F32, M, K, 4, tasq.TASQ_SYMRANGE, tasq.TASQ_PER_TOKEN, codes, F8,
                        alpha, zc)
    wq = oracle.quant_weight(w)
    s_x, a, z = oracle.quant_act(x, 4, oracle.SYMRANGE, oracle.PER_TOKEN)
    for stage in range(2):
        y = G.empty((M, N), torch.int16)
        acc = G.empty((M, N), torch.int32)
        tasq.tasq_masked_gemm_grouped(ctx.h, [0, 1], stage, codes, F8, alpha, zc, M, packed, N, K, y, acc)
        yh, acch = G.bf16_bits_host(y), acc.cpu().numpy()
        for g in range(2):
            b = int(table[g, stage])
            sl = slice(g * Ng, (g + 1) * Ng)
            ref = oracle.gemm(s_x, wq["s"][sl], b)
            assert np.array_equal(acch[:, sl], ref), (stage, g)
            _, yb = oracle.epilogue_f32(ref, a, z, oracle.row_sums(wq["s"][sl], b), wq["c"][sl], bias[sl])
            assert G.assert_bf16_close(yh[:, sl], yb) == yb.size


# ------------------------- members listed in device memory (one shared input) --

@pytest.mark.parametrize("code_fmt,n_bits", [(tasq.TASQ_CODES_F16, 8), (F8, 4)], ids=["f16", "e5m2"])
@pytest.mark.parametrize("M,Ng,K,L", [(300, 128, 256, 56), (77, 136, 256, 9), (33, 8, 128, 256),
                                      (200, 64, 1152, 40), (129, 1152, 384, 3)])
def test_shared_input_members_match_single_layers(ctx, oracle, code_fmt, n_bits, M, Ng, K, L):
    """tasq_masked_gemm_shared_input: L layers (up to 256) that read one input, listed
    in device memory in a shuffled order, contracted by one launch; each member equals
    the oracle's single layer at its own b.  Stage 0 draws every b from 2..8 (fp16
    route), stage 1 from 2..4 (the e5m2 kind when the codes come as e5m2), and the
    stage is also read from the device int.  Members straddle 128-channel tiles
    (Ng = 8, 64, 136) or span several (Ng = 1152)."""
    torch = G.torch()
    N = L * Ng
    w = workloads.normal((N, K), 700 + L, 0.02)
    bias = workloads.normal((N,), 701 + L, 0.02)
    x = workloads.normal((M, K), 702 + L)
    sw, cw, _ = G.quant_weights(ctx, G.dev(w), tasq.TASQ_F32, N, K)
    packed = G.pack(ctx, tasq.TASQ_LINEAR, sw, cw, G.dev(bias), N, K)
    r = workloads.rng(703 + L)
    n_table = L + 5  # the table holds layers that are not members too
    table = np.stack([r.integers(2, 9, n_table), r.integers(2, 5, n_table)], 1).astype(np.uint8)
    tasq.tasq_set_schedule(ctx.h, table, n_table, 2)
    layers = r.permutation(n_table)[:L].astype(np.int32)
    d_layers = G.dev(layers)
    f8 = code_fmt == F8
    codes = G.empty(((3 if f8 else 2) * M * K // 2,), torch.float16)
    alpha, zc = G.empty((M,), torch.float32), G.empty((M,), torch.float32)
    tasq.tasq_quant_act(ctx.h, G.dev(x), tasq.TASQ_F32, M, K, n_bits, tasq.TASQ_SYMRANGE, tasq.TASQ_PER_TOKEN, codes,
                        code_fmt, alpha, zc)
    wq = oracle.quant_weight(w)
    s_x, a, z = oracle.quant_act(x, n_bits, oracle.SYMRANGE, oracle.PER_TOKEN)
    d_stage = torch.zeros((4,), dtype=torch.int32, device="cuda")
    tasq.tasq_set_stage_device(ctx.h, d_stage)
    try:
        for stage, call_stage in ((0, 0), (1, 1), (1, -1)):
            d_stage.fill_(stage)
            y = G.empty((M, N), torch.int16)
            acc = G.empty((M, N), torch.int32)
            tasq.tasq_masked_gemm_shared_input(ctx.h, d_layers, L, call_stage, codes, code_fmt, alpha, zc, M, packed,
                                               N, K, y, acc)
            yh, acch = G.bf16_bits_host(y), acc.cpu().numpy()
            for g, layer in enumerate(layers):
                b = int(table[layer, stage])
                sl = slice(g * Ng, (g + 1) * Ng)
                ref = oracle.gemm(s_x, wq["s"][sl], b)
                assert np.array_equal(acch[:, sl], ref), (stage, g, b)
                _, yb = oracle.epilogue_f32(ref, a, z, oracle.row_sums(wq["s"][sl], b), wq["c"][sl], bias[sl])
                assert G.assert_bf16_close(yh[:, sl], yb) == yb.size, (stage, g, b)
    finally:
        tasq.tasq_set_stage_device(ctx.h, None)
    assert tasq.tasq_device_status(ctx.h) == tasq.TASQ_OK


@pytest.mark.parametrize("M,Ng,K,L", [(300, 1152, 1152, 56), (77, 1280, 2048, 120)], ids=["pixart_text", "sdxl_text"])
def test_shared_input_full_size_sampled_rows(ctx, oracle, M, Ng, K, L):
    """The text units at the sizes the bench runs them (every cross-attention key and value
    projection of PixArt-Sigma's 28 blocks, of SDXL-Turbo's 60 width-1280 blocks) in the
    same launch: sampled token rows (the first, the last and six in between) of every
    member's output against the oracle's single layer at that member's b."""
    torch = G.torch()
    N = L * Ng
    wd = workloads.device_normal((N, K), 730 + L, 0.02)
    sw, cw, _ = G.quant_weights(ctx, wd, tasq.TASQ_F32, N, K)
    del wd
    bias = workloads.normal((N,), 731 + L, 0.02)
    packed = G.pack(ctx, tasq.TASQ_LINEAR, sw, cw, G.dev(bias), N, K)
    swh, cwh = sw.cpu().numpy(), cw.cpu().numpy()
    r = workloads.rng(732 + L)
    table = r.integers(2, 9, (L, 1)).astype(np.uint8)
    tasq.tasq_set_schedule(ctx.h, table, L, 1)
    d_layers = G.dev(np.arange(L, dtype=np.int32))
    x = workloads.normal((M, K), 733 + L)
    codes, alpha, zc = G.quant_act(ctx, G.dev(x), tasq.TASQ_F32, M, K, 8, tasq.TASQ_SYMRANGE, tasq.TASQ_PER_TOKEN,
                                   tasq.TASQ_CODES_F16)
    y = G.empty((M, N), torch.int16)
    tasq.tasq_masked_gemm_shared_input(ctx.h, d_layers, L, 0, codes, tasq.TASQ_CODES_F16, alpha, zc, M, packed, N, K,
                                       y, None)
    rows = np.unique(np.concatenate([[0, M - 1], r.integers(0, M, 6)]))
    yh = G.bf16_bits_host(y)[rows]
    s_x, a, z = oracle.quant_act(x)
    for g in range(L):
        b = int(table[g, 0])
        sl = slice(g * Ng, (g + 1) * Ng)
        ref = oracle.gemm(s_x[rows], swh[sl], b)
        _, yb = oracle.epilogue_f32(ref, a[rows], z[rows], oracle.row_sums(swh[sl], b), cwh[sl], bias[sl])
        assert np.array_equal(yh[:, sl], yb), (g, b)
    assert tasq.tasq_device_status(ctx.h) == tasq.TASQ_OK


def test_shared_input_in_a_graph_and_bad_members(ctx, oracle):
    """The member list is read at every replay of a captured call (a later change
    of the list or of the bit table shows in the next replay); a layer index outside
    the table is found on the device, recorded as TASQ_ERR_DEVICE, and no output is
    written.  Host-side checks: the member count, the channel split, the code format
    and a NULL list."""
    torch = G.torch()
    M, Ng, K, L = 64, 128, 256, 6
    N = L * Ng
    w = workloads.normal((N, K), 711, 0.02)
    x = workloads.normal((M, K), 712)
    sw, cw, _ = G.quant_weights(ctx, G.dev(w), tasq.TASQ_F32, N, K)
    packed = G.pack(ctx, tasq.TASQ_LINEAR, sw, cw, None, N, K)
    table = np.array([[2 + i % 7] for i in range(8)], np.uint8)
    tasq.tasq_set_schedule(ctx.h, table, 8, 1)
    codes, alpha, zc = G.quant_act(ctx, G.dev(x), tasq.TASQ_F32, M, K, 8, tasq.TASQ_SYMRANGE, tasq.TASQ_PER_TOKEN,
                                   tasq.TASQ_CODES_F16)
    wq = oracle.quant_weight(w)
    s_x, a, z = oracle.quant_act(x)
    d_layers = G.dev(np.arange(L, dtype=np.int32))
    y = G.empty((M, N), torch.int16)

    def call():
        tasq.tasq_masked_gemm_shared_input(ctx.h, d_layers, L, 0, codes, tasq.TASQ_CODES_F16, alpha, zc, M, packed, N,
                                           K, y, None)

    call()
    torch.cuda.synchronize()
    s = torch.cuda.Stream()
    s.wait_stream(torch.cuda.current_stream())
    g = torch.cuda.CUDAGraph()
    with torch.cuda.stream(s), torch.cuda.graph(g, stream=s):
        call()

    def check(layers):
        yh = G.bf16_bits_host(y)
        for m, layer in enumerate(layers):
            b = int(table[layer, 0])
            sl = slice(m * Ng, (m + 1) * Ng)
            ref = oracle.gemm(s_x, wq["s"][sl], b)
            _, yb = oracle.epilogue_f32(ref, a, z, oracle.row_sums(wq["s"][sl], b), wq["c"][sl])
            assert np.array_equal(yh[:, sl], yb), (m, layer, b)

    for layers in ([0, 1, 2, 3, 4, 5], [7, 6, 5, 4, 3, 2]):
        d_layers.copy_(torch.tensor(layers, dtype=torch.int32))
        y.fill_(0)
        g.replay()
        torch.cuda.synchronize()
        check(layers)
    assert tasq.tasq_device_status(ctx.h) == tasq.TASQ_OK
    d_layers.copy_(torch.tensor([0, 1, 2, 8, 4, 5], dtype=torch.int32))  # layer 8: not in the table
    y.fill_(0)
    g.replay()
    torch.cuda.synchronize()
    assert tasq.tasq_device_status(ctx.h) == tasq.TASQ_ERR_DEVICE
    assert not bool(y.any())
    buf = torch.zeros((1 << 16,), dtype=torch.uint8, device="cuda")
    big = G.dev(np.zeros(300, np.int32))
    for dl, n, NN, fmt, code in ((big, 257, 257 * 8, tasq.TASQ_CODES_F16, tasq.TASQ_ERR_INVALID_ARG),  # > 256
                                 (big, 0, 64, tasq.TASQ_CODES_F16, tasq.TASQ_ERR_INVALID_ARG),          # none
                                 (big, 3, 64, tasq.TASQ_CODES_F16, tasq.TASQ_ERR_UNSUPPORTED),          # 64 / 3
                                 (big, 2, 64, tasq.TASQ_CODES_S8, tasq.TASQ_ERR_UNSUPPORTED),           # int8 codes
                                 (None, 2, 64, tasq.TASQ_CODES_F16, tasq.TASQ_ERR_INVALID_ARG)):        # no list
        with pytest.raises(tasq.TasqError) as e:
            tasq.tasq_masked_gemm_shared_input(ctx.h, dl, n, 0, buf, fmt, buf, buf, 16, buf, NN, 64, buf, None)
        assert e.value.code == code, (n, NN, fmt)
    assert tasq.tasq_device_status(ctx.h) == tasq.TASQ_OK


def test_e5m2_codes_in_a_convolution_use_the_fp16_codes(ctx, oracle):
    """A 3x3 convolution given dual-format codes reads their fp16 part."""
    torch = G.torch()
    B, H, W, Cin, Cout = 1, 8, 8, 64, 16
    x = workloads.normal((B, H, W, Cin), 511)
    w = workloads.normal((Cout, 9 * Cin), 512, 0.03)
    sw, cw, _ = G.quant_weights(ctx, G.dev(w), tasq.TASQ_F32, Cout, 9 * Cin)
    packed = G.pack(ctx, tasq.TASQ_CONV3X3, sw, cw, None, Cout, 9 * Cin, Cin)
    tasq.tasq_set_schedule(ctx.h, np.array([[4]], np.uint8), 1, 1)
    M = B * H * W
    codes = G.empty((3 * M * Cin // 2,), torch.float16)
    alpha, zc = G.empty((1,), torch.float32), G.empty((1,), torch.float32)
    tasq.tasq_quant_act(ctx.h, G.dev(x), tasq.TASQ_F32, M, Cin, 4, tasq.TASQ_SYMRANGE, tasq.TASQ_PER_TENSOR, codes,
                        F8, alpha, zc)
    y, acc = G.conv(ctx, 0, 0, codes, F8, alpha, zc, B, H, W, Cin, packed, Cout)
    wq = oracle.quant_weight(w)
    s_x, a, z = oracle.quant_act(x.reshape(1, -1), 4, oracle.SYMRANGE, oracle.PER_TOKEN)
    ref, rs = oracle.conv3x3(s_x.reshape(B, H, W, Cin), wq["s"], 4)
    assert np.array_equal(acc.cpu().numpy(), ref)


# ------------------------------------------------ 16-bit low-rank branch --

def _bf16_bits(a):
    torch = G.torch()
    return torch.from_numpy(np.asarray(a, np.float32)).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)


def _dev_bits(bits):
    torch = G.torch()
    return torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).cuda()


def _ulp(v, mant):
    """Spacing of a float format with `mant` stored mantissa bits at |v|."""
    e = np.floor(np.log2(np.maximum(np.abs(v), 2.0 ** -60)))
    return 2.0 ** (e - mant)


def _down_sums(oracle, x, l2_bits):
    """sum_k |bf16(x) l2| per (row, rank): the fp32 accumulation's error scale."""
    return np.abs(oracle.bf16_round(x).astype(np.float64)) @ np.abs(
        oracle.bf16_bits_to_f32(l2_bits).astype(np.float64)).T


@pytest.mark.parametrize("M,K,r,dtype", [(300, 1152, 32, tasq.TASQ_BF16), (4096, 1152, 16, tasq.TASQ_F32),
                                         (77, 2048, 32, tasq.TASQ_F32), (17, 16, 16, tasq.TASQ_BF16),
                                         (33, 48, 32, tasq.TASQ_F32), (4096, 1152, 32, tasq.TASQ_BF16),
                                         (200, 4608, 16, tasq.TASQ_BF16)])
def test_lowrank_down_parity(ctx, oracle, M, K, r, dtype):
    """u' = fp16((bf16(x) . l2^T) / alpha) in rows of 64 fp16 against the oracle's
    u / alpha, within the fp32 accumulation (K 2^-23 sum |x_b l2|) and one fp16
    rounding; columns past the rank are zero.  bf16 x takes the tensor-core kernel
    (128 rows per CTA, ragged M, K shorter than one 64-wide stage, several trips
    round the stage ring), fp32 x the warp-MMA kernel (ragged M, K shorter than
    its sixteen slices)."""
    torch = G.torch()
    x = workloads.normal((M, K), 801 + M)
    l2 = _bf16_bits(workloads.normal((r, K), 802 + K, 0.05))
    alpha = workloads.uniform((M,), 805 + M, 0.005, 0.02).astype(np.float32)
    if dtype == tasq.TASQ_BF16:
        xd, x = G.to_bf16(x)
    else:
        xd = G.dev(x)
    u = G.empty((M, 64), torch.int16)
    tasq.tasq_lowrank_down(ctx.h, xd, dtype, M, K, _dev_bits(l2), r, G.dev(alpha), u)
    got = u.cpu().numpy().view(np.float16).astype(np.float64)
    ref = oracle.lowrank_down(x, l2) / alpha[:, None].astype(np.float64)
    tol = K * 2.0 ** -23 * _down_sums(oracle, x, l2) / alpha[:, None] + _ulp(np.abs(ref) + 1e-30, 10) * 1.01
    assert np.all(np.abs(got[:, :r] - ref) <= tol)
    assert not got[:, r:].any()
    assert tasq.tasq_device_status(ctx.h) == tasq.TASQ_OK


@pytest.mark.parametrize("M,N,K,r,full,act_bits", [
    (256, 1152, 1152, 32, True, 8),    # 64-token tiles
    (4000, 1096, 384, 16, True, 8),    # 256-token tiles (two stages per block), ragged channel tile
    (4096, 3456, 1152, 32, False, 8),  # 192-token tiles, two accumulators
    (77, 640, 2048, 32, True, 8),      # a shape the plan would split along K: kept whole
    (4096, 1152, 4608, 32, False, 4),  # e5m2 codes, 8-bit-float route at b <= 4
    (300, 512, 1168, 16, True, 4),     # e5m2 codes, ragged last K block
])
def test_masked_gemm_lr_parity(ctx, oracle, M, N, K, r, full, act_bits):
    """The layer with its low-rank branch against the fp64 definition (masked
    layer plus (x_b l2^T) l1^T), at every b: within one bf16 ulp, the fp32
    epilogue chain, and the branch's 16-bit roundings (u' and l1 / c_w in fp16:
    2^-10 of each product) and fp32 accumulations."""
    torch = G.torch()
    bits = [8, 5, 4, 2]
    if act_bits <= 4:
        st = _setup_f8(ctx, oracle, M, N, K, bits, seed=M + N + r, n_bits=act_bits)
        x = workloads.normal((M, K), M + N + r)  # the input _setup_f8 quantized
        fmt = F8
    else:
        w = workloads.normal((N, K), M + 11, 0.02)
        bias = workloads.normal((N,), M + 12, 0.02)
        x = workloads.normal((M, K), M + 13)
        sw, cw, _ = G.quant_weights(ctx, G.dev(w), tasq.TASQ_F32, N, K)
        packed = G.pack(ctx, tasq.TASQ_LINEAR, sw, cw, G.dev(bias), N, K)
        tasq.tasq_set_schedule(ctx.h, np.array([bits], np.uint8), 1, len(bits))
        codes = G.empty((M, K), torch.float16)
        alpha, zc = G.empty((M,), torch.float32), G.empty((M,), torch.float32)
        tasq.tasq_quant_act(ctx.h, G.dev(x), tasq.TASQ_F32, M, K, 8, tasq.TASQ_SYMRANGE, tasq.TASQ_PER_TOKEN, codes,
                            tasq.TASQ_CODES_F16, alpha, zc)
        s_x, a, z = oracle.quant_act(x, 8, oracle.SYMRANGE, oracle.PER_TOKEN)
        st = dict(packed=packed, codes=codes, alpha=alpha, zc=zc, wq=oracle.quant_weight(w), s_x=s_x, a=a, z=z,
                  bias=bias)
        fmt = tasq.TASQ_CODES_F16
    l2 = _bf16_bits(workloads.normal((r, K), 803 + K, 0.05))
    l1 = _bf16_bits(workloads.normal((N, r), 804 + N, 0.05))
    u = G.empty((M, 64), torch.int16)
    tasq.tasq_lowrank_down(ctx.h, G.dev(x), tasq.TASQ_F32, M, K, _dev_bits(l2), r, st["alpha"], u)
    rows = np.arange(M) if full else np.unique(np.concatenate([np.arange(0, M, max(1, M // 40)), [M - 1]]))
    rows_d = torch.from_numpy(rows).cuda()
    u_ref = oracle.lowrank_down(x[rows], l2)
    lr = oracle.lowrank_up(u_ref, l1)
    l1a = np.abs(oracle.bf16_bits_to_f32(l1).astype(np.float64))
    branch_err = (2.0 ** -9 * np.abs(u_ref) + K * 2.0 ** -22 * _down_sums(oracle, x[rows], l2)) @ l1a.T
    scale = np.abs(st["a"][rows].astype(np.float64)[:, None] * st["wq"]["c"].astype(np.float64)[None, :])
    for stage, b in enumerate(bits):
        y = G.empty((M, N), torch.int16)
        tasq.tasq_masked_gemm_lr(ctx.h, 0, stage, st["codes"], fmt, st["alpha"], st["zc"], M, st["packed"], N, K, u,
                                 _dev_bits(l1), r, y, None)
        s_w = st["wq"]["s"]
        ydef = oracle.linear_lowrank_def_f64(st["s_x"][rows], st["a"][rows], st["z"][rows], s_w, st["wq"]["c"],
                                            st["bias"], b, lr)
        acc = oracle.gemm(st["s_x"][rows], s_w, b).astype(np.float64)
        rs = oracle.row_sums(s_w, b).astype(np.float64)
        chain = 2.0 ** -18 * (scale * (np.abs(acc) + np.abs(st["z"][rows, None] * rs[None, :])) + np.abs(lr)
                              + np.abs(st["bias"])[None, :])
        got = oracle.bf16_bits_to_f32(G.bf16_bits_host(y.index_select(0, rows_d))).astype(np.float64)
        tol = _ulp(np.maximum(np.abs(ydef), np.abs(got)), 7) + chain + branch_err
        bad = np.abs(got - ydef) > tol
        assert not bad.any(), (b, bad.sum(), np.abs(got - ydef)[bad][:5], tol[bad][:5])
    assert tasq.tasq_device_status(ctx.h) == tasq.TASQ_OK


def test_lowrank_bad_arguments(ctx):
    torch = G.torch()
    buf = torch.zeros((1 << 16,), dtype=torch.uint8, device="cuda")
    tasq.tasq_set_schedule(ctx.h, np.array([[8]], np.uint8), 1, 1)
    for rank in (8, 64):
        with pytest.raises(tasq.TasqError) as e:
            tasq.tasq_lowrank_down(ctx.h, buf, tasq.TASQ_F32, 16, 64, buf, rank, buf, buf)
        assert e.value.code == tasq.TASQ_ERR_INVALID_ARG
    with pytest.raises(tasq.TasqError) as e:  # K not a multiple of 16
        tasq.tasq_lowrank_down(ctx.h, buf, tasq.TASQ_BF16, 16, 40, buf, 16, buf, buf)
    assert e.value.code == tasq.TASQ_ERR_UNSUPPORTED
    with pytest.raises(tasq.TasqError) as e:  # u must be 16-byte aligned
        tasq.tasq_lowrank_down(ctx.h, buf, tasq.TASQ_BF16, 16, 64, buf, 16, buf, buf.data_ptr() + 8)
    assert e.value.code == tasq.TASQ_ERR_UNSUPPORTED
    with pytest.raises(tasq.TasqError) as e:  # int8 codes: the mma.sync s8 route has no low-rank block
        tasq.tasq_masked_gemm_lr(ctx.h, 0, 0, buf, tasq.TASQ_CODES_S8, buf, buf, 16, buf, 64, 64, buf, buf, 16, buf)
    assert e.value.code == tasq.TASQ_ERR_UNSUPPORTED
    with pytest.raises(tasq.TasqError) as e:  # rank outside 16 / 32
        tasq.tasq_masked_gemm_lr(ctx.h, 0, 0, buf, tasq.TASQ_CODES_F16, buf, buf, 16, buf, 64, 64, buf, buf, 24, buf)
    assert e.value.code == tasq.TASQ_ERR_INVALID_ARG
    with pytest.raises(tasq.TasqError) as e:  # no int32 accumulators with the branch
        tasq.tasq_masked_gemm_lr(ctx.h, 0, 0, buf, tasq.TASQ_CODES_F16, buf, buf, 16, buf, 64, 64, buf, buf, 16, buf,
                                 buf)
    assert e.value.code == tasq.TASQ_ERR_INVALID_ARG
    assert tasq.tasq_device_status(ctx.h) == tasq.TASQ_OK
