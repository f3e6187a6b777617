"""CPU checks of the C ABI: the library builds, loads without a GPU, exports
every entry point include/tasq.h declares, and the binding's enums match the
header.  No compute call is made here (there is no GPU in this container)."""
import ctypes
import os
import re
import subprocess

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "tasq.h")


def _declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(tasq_\w+)\s*\(", text)))


@pytest.fixture(scope="module")
def built_lib():
    from paper_2608_03057_gb300 import build
    return build.build()


def test_header_declares_the_boundary():
    names = _declared_functions()
    for required in ("tasq_pack_weights", "tasq_set_schedule", "tasq_quant_act", "tasq_masked_gemm",
                     "tasq_masked_conv3x3", "tasq_quant_weights", "tasq_device_status"):
        assert required in names


def test_library_exports_every_declared_symbol(built_lib):
    out = subprocess.run(["nm", "-D", "--defined-only", built_lib], capture_output=True, text=True, check=True).stdout
    exported = set(re.findall(r"\bT (tasq_\w+)", out))
    declared = set(_declared_functions())
    assert declared <= exported, declared - exported
    lib = ctypes.CDLL(built_lib)
    for name in declared:
        assert hasattr(lib, name)


def test_binding_enums_match_header():
    from paper_2608_03057_gb300 import tasq
    text = open(HEADER).read()
    for name, value in re.findall(r"\b(TASQ_[A-Z0-9_]+)\s*=\s*(\d+)", text):
        assert getattr(tasq, name) == int(value), name
    assert tasq.tasq_version() == int(re.search(r"TASQ_ABI_VERSION (\d+)", text).group(1))


def test_binding_names_match_header():
    from paper_2608_03057_gb300 import tasq
    for name in _declared_functions():
        assert callable(getattr(tasq, name)), name


def test_packed_bytes_layout(built_lib):
    from paper_2608_03057_gb300 import tasq
    n, k = 1152, 1152
    b = tasq.tasq_packed_bytes(tasq.TASQ_LINEAR, n, k)
    # 1 KB header, int8 weights, scale, bias, 7 row-sum vectors, weight zero offsets, 256-byte aligned
    assert b % 256 == 0 and b >= 1024 + n * k + 4 * n * 2 + 7 * 4 * n + 4 * n
    c = tasq.tasq_packed_bytes(tasq.TASQ_CONV3X3, 320, 9 * 320)
    assert c >= 1024 + 320 * 2880 + 7 * 4 * 320 * 10
    assert tasq.tasq_packed_bytes(tasq.TASQ_CONV3X3, 320, 100) == 0  # K not 9*Cin
    assert tasq.tasq_packed_bytes(7, 8, 16) == 0


def test_create_without_gpu_fails_cleanly(built_lib):
    torch = pytest.importorskip("torch")
    if torch.cuda.is_available():
        pytest.skip("a GPU is present")
    from paper_2608_03057_gb300 import tasq
    with pytest.raises(tasq.TasqError) as e:
        tasq.tasq_create(0)
    assert e.value.code in (tasq.TASQ_ERR_CUDA, tasq.TASQ_ERR_INVALID_ARG)
    assert tasq.tasq_last_error(None)


def test_null_context_is_rejected(built_lib):
    from paper_2608_03057_gb300 import tasq
    L = tasq.lib()
    assert L.tasq_set_route(None, 0) == tasq.TASQ_ERR_INVALID_ARG
    assert L.tasq_masked_gemm(None, 0, 0, None, 0, None, None, 1, None, 8, 16, None, None, None) == tasq.TASQ_ERR_INVALID_ARG
