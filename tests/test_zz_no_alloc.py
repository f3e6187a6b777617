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
