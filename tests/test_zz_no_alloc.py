"""The allocation-free per-tensor activation quantizer.

Some callers cannot allocate device memory while they run (an inference
plugin whose framework forbids allocation during enqueue, or a service whose
device memory is planned once at start-up), so they cannot create a context.
tasq_quant_act_tensor_noalloc serves them with a reduction scratch compiled
into the library.  Its results must equal those of the context-based entry
point, call after call.  This file is collected last so that, if it fails,
a run that stops at the first failure has already run every other test.
"""
import numpy as np
import pytest

from paper_2608_03057_gb300 import tasq, workloads
from tests import gpu_layer as G

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def ctx():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    c = G.Ctx()
    yield c
    c.close()


def _noalloc(x_dev, dtype, M, K, mode, code_fmt):
    torch = G.torch()
    codes = torch.empty((M, K), dtype=torch.int8 if code_fmt == tasq.TASQ_CODES_S8 else torch.float16, device="cuda")
    alpha = torch.empty((1,), dtype=torch.float32, device="cuda")
    zc = torch.empty((1,), dtype=torch.float32, device="cuda")
    tasq.tasq_quant_act_tensor_noalloc(x_dev, dtype, M, K, 8, mode, codes, code_fmt, alpha, zc)
    return codes, alpha, zc


def test_two_calls_match_the_context_entry_point(ctx):
    torch = G.torch()
    cases = [  # a large NHWC tensor, then a smaller one: nothing may carry over
        ((1, 64, 64, 320), 91, tasq.TASQ_F32, tasq.TASQ_SYMRANGE, tasq.TASQ_CODES_F16),
        ((2, 5, 7, 64), 92, tasq.TASQ_BF16, tasq.TASQ_ASYM, tasq.TASQ_CODES_S8),
    ]
    for shape, seed, dtype, mode, code_fmt in cases:
        x = workloads.normal(shape, seed)
        x[(0,) * (len(shape) - 1)] += 5.0  # an outlier decides the range
        xd = G.to_bf16(x)[0] if dtype == tasq.TASQ_BF16 else G.dev(x)
        M, K = int(np.prod(shape[:-1])), shape[-1]
        c1, a1, z1 = _noalloc(xd, dtype, M, K, mode, code_fmt)
        c0, a0, z0 = G.quant_act(ctx, xd, dtype, M, K, 8, mode, tasq.TASQ_PER_TENSOR, code_fmt)
        torch.cuda.synchronize()
        # integer codes: bit-exact; scales: identical fp32 values
        assert torch.equal(c1, c0)
        assert a1.item() == a0.item() and z1.item() == z0.item()


@pytest.fixture(scope="module")
def oracle():
    from oracle import oracle as o
    o.build()
    return o


@pytest.mark.parametrize("shape,seed,dtype,mode,code_fmt", [
    ((1, 64, 64, 320), 93, tasq.TASQ_BF16, tasq.TASQ_SYMRANGE, tasq.TASQ_CODES_F16),
    ((2, 16, 16, 1280), 94, tasq.TASQ_F32, tasq.TASQ_ASYM, tasq.TASQ_CODES_S8),
    ((3, 112), 95, tasq.TASQ_F32, tasq.TASQ_SYMRANGE, tasq.TASQ_CODES_F16),
])
def test_matches_the_oracle(ctx, oracle, shape, seed, dtype, mode, code_fmt):
    """Against the oracle's App. A.1.2 quantizer applied to the whole tensor as
    one group: codes bit for bit, alpha and zc as identical fp32 values."""
    x = workloads.normal(shape, seed)
    x.reshape(-1, shape[-1])[-1, 1] -= 7.0  # an outlier decides the range
    if dtype == tasq.TASQ_BF16:
        xd, x = G.to_bf16(x)
    else:
        xd = G.dev(x)
    M, K = int(np.prod(shape[:-1])), shape[-1]
    codes, alpha, zc = _noalloc(xd, dtype, M, K, mode, code_fmt)
    s, a, z = oracle.quant_act(x.reshape(1, -1), 8, mode, oracle.PER_TOKEN)
    assert np.array_equal(G.codes_to_int8(codes).reshape(-1), s.reshape(-1))
    assert alpha.item() == a[0] and zc.item() == z[0]


def test_at_the_size_limit(ctx, oracle):
    """Exactly the documented limit, 2048 slices of 32,768 elements (65,536 x
    1,024): every slot of the array and the largest grid of the range kernel
    are used.  Codes, alpha and zc equal the oracle's and the context entry
    point's."""
    torch = G.torch()
    M, K = 65536, 1024
    x = workloads.normal((M, K), 96)
    x[M - 1, K - 1] = 9.5  # the range is decided by the last slice
    xd, xh = G.to_bf16(x)
    del x
    c1, a1, z1 = _noalloc(xd, tasq.TASQ_BF16, M, K, tasq.TASQ_SYMRANGE, tasq.TASQ_CODES_F16)
    c0, a0, z0 = G.quant_act(ctx, xd, tasq.TASQ_BF16, M, K, 8, tasq.TASQ_SYMRANGE, tasq.TASQ_PER_TENSOR,
                             tasq.TASQ_CODES_F16)
    torch.cuda.synchronize()
    assert torch.equal(c1, c0)
    assert a1.item() == a0.item() and z1.item() == z0.item()
    s, a, z = oracle.quant_act(xh.reshape(1, -1), 8, oracle.SYMRANGE, oracle.PER_TOKEN)
    assert np.array_equal(G.codes_to_int8(c1).reshape(-1), s.reshape(-1))
    assert a1.item() == a[0] and z1.item() == z[0]


def test_oversize_tensor_is_rejected_without_launching():
    torch = G.torch()
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    buf = torch.zeros((16,), dtype=torch.float32, device="cuda")
    with pytest.raises(tasq.TasqError) as e:
        tasq.tasq_quant_act_tensor_noalloc(buf, tasq.TASQ_F32, 4096 * 16 + 1, 1024, 8, tasq.TASQ_SYMRANGE, buf,
                                           tasq.TASQ_CODES_F16, buf, buf)
    assert e.value.code == tasq.TASQ_ERR_UNSUPPORTED
    assert "limit" in tasq.tasq_last_error(None)
    # one 16-element group past the limit
    with pytest.raises(tasq.TasqError) as e:
        tasq.tasq_quant_act_tensor_noalloc(buf, tasq.TASQ_F32, 1, 2048 * 32768 + 16, 8, tasq.TASQ_SYMRANGE, buf,
                                           tasq.TASQ_CODES_F16, buf, buf)
    assert e.value.code == tasq.TASQ_ERR_UNSUPPORTED
