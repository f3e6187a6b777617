"""The tensor-core MMA kinds for integer-valued operands (tasq_probe_mma).

The exact route holds int8 codes in fp16 and relies on the fp32 accumulator of
tcgen05 kind::f16 adding integer products exactly while partial sums stay
below 2^24.  The 8-bit route for b <= 4 weights and 4-bit activations holds the
codes in e5m2 (kind::f8f6f4, twice the K per instruction) and relies on the same
property; e4m3 (integers of magnitude <= 16) is checked too.  Each kind is
checked here against the exact integer result on adversarial patterns (extreme
codes, partial sums up to just below 2^24, large and small products in one
instruction, cancelling signs, random A4 codes), and the cycles per MMA of each
kind are measured.
"""
import numpy as np
import pytest

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def probe():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    from paper_2608_03057_gb300 import mma_probe
    return mma_probe


@pytest.mark.parametrize("kind", [0, 1, 2])
def test_integer_products_accumulate_exactly(probe, kind):
    for r in probe.exactness(kind, n=256):
        assert r["mismatches"] == 0, r
    # the longest accumulation reaches 2^23 - 2^14 (fp16, 64 elements per row),
    # 2^24 - 2^15 (e4m3, 128 elements per row) or 2^24 - 2^17 (e5m2: 127 x 128 x 8 x 128)
    assert r["max_abs"] >= {0: (1 << 23) - (1 << 14), 1: (1 << 24) - (1 << 15), 2: (1 << 24) - (1 << 17)}[kind]


def test_rates_of_the_kinds(probe):
    import torch
    sms = torch.cuda.get_device_properties(0).multi_processor_count
    for n in (128, 256):
        # at least the dense rate of M = 128 x N x 16 (f16) per N / 2 cycles, within 25 %;
        # the 8-bit kinds do twice the K in the same instruction count
        for kind in (0, 1, 2):
            r = probe.rate(kind, n, sms, reps=64)
            assert 0 < r["cycles_per_mma"] < 1.25 * n / 2, r


def test_probe_rejects_bad_arguments(probe):
    import torch
    from paper_2608_03057_gb300 import tasq
    buf = torch.zeros((1 << 16,), dtype=torch.uint8, device="cuda")
    for kind, n, reps in ((3, 128, 1), (-1, 128, 1), (0, 8, 1), (1, 264, 1), (0, 128, 0)):
        with pytest.raises(tasq.TasqError) as e:
            tasq.tasq_probe_mma(kind, n, reps, buf, buf, buf, buf, 1)
        assert e.value.code == tasq.TASQ_ERR_INVALID_ARG
