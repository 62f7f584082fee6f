"""Host-side checks of the C ABI that need no GPU: the library builds, loads
and exports every function include/isam.h declares, and argument errors are
reported before any CUDA call is made."""
import ctypes

import pytest

from paper_1810_09958_gb300 import build, isam


@pytest.fixture(scope="module")
def lib():
    build.build()
    return isam.load()


def test_exports_every_declared_symbol(lib):
    names = isam.declared_functions()
    assert {"isam_gemm", "isam_gru_forward", "isam_dwsep_conv", "isam_sync",
            "isam_set_stream", "isam_last_error_string", "isam_shutdown"} <= set(names)
    for n in names:
        assert hasattr(lib, n), n


def test_version(lib):
    assert lib.isam_version() == 100


def test_gemm_rejects_bad_sizes_without_cuda(lib):
    p = ctypes.c_void_p(16)
    assert lib.isam_gemm(0, 4, 4, 0, 0, 1.0, p, p, 0.0, p) == isam.ISAM_ERR_INVALID_ARG
    assert b"sizes" in lib.isam_last_error_string()
    assert lib.isam_gemm(4, 4, 4, 2, 0, 1.0, p, p, 0.0, p) == isam.ISAM_ERR_INVALID_ARG
    assert lib.isam_gemm(4, 4, 4, 0, 0, 1.0, None, p, 0.0, p) == isam.ISAM_ERR_INVALID_ARG


def test_gemm_rejects_unaligned_without_cuda(lib):
    p = ctypes.c_void_p(16)
    # K = 12 is not a multiple of 8 for a K-major A: row pitch not 16-byte aligned.
    assert lib.isam_gemm(16, 16, 12, 0, 0, 1.0, p, p, 0.0, p) == isam.ISAM_ERR_UNSUPPORTED
    # Misaligned base pointer.
    q = ctypes.c_void_p(18)
    assert lib.isam_gemm(16, 16, 16, 0, 0, 1.0, q, p, 0.0, p) == isam.ISAM_ERR_UNSUPPORTED


def test_gru_and_dwsep_reject_bad_args_without_cuda(lib):
    p = ctypes.c_void_p(16)
    assert lib.isam_gru_forward(0, 1, 128, p, p, p, p, None, p) == isam.ISAM_ERR_INVALID_ARG
    assert lib.isam_gru_forward(1, 1, 128, None, p, p, p, None, p) == isam.ISAM_ERR_INVALID_ARG
    assert lib.isam_gru_forward_reset_before(1, 0, 128, p, p, p, p, None, p) == isam.ISAM_ERR_INVALID_ARG
    assert lib.isam_gru_forward_reset_before(1, 1, 128, p, p, None, p, None, p) == isam.ISAM_ERR_INVALID_ARG
    assert lib.isam_gru_forward_stack(0, 1, 1, 128, 0, p, p, p, p, None, p) == isam.ISAM_ERR_INVALID_ARG
    assert lib.isam_gru_forward_stack(2, 1, 1, 128, 2, p, p, p, p, None, p) == isam.ISAM_ERR_INVALID_ARG
    assert lib.isam_gru_forward_stack(2, 1, 1, 128, 0, p, p, p, None, None, p) == isam.ISAM_ERR_INVALID_ARG
    assert lib.isam_dwsep_conv(1, 0, 4, 16, 16, p, p, p, p) == isam.ISAM_ERR_INVALID_ARG
    assert lib.isam_dwsep_conv(1, 4, 4, 16, 16, p, None, p, p) == isam.ISAM_ERR_INVALID_ARG
    assert lib.isam_dwsep_plan_info(0, 16, 16, p) == isam.ISAM_ERR_INVALID_ARG
    assert lib.isam_dwsep_plan_info(4, 16, 16, None) == isam.ISAM_ERR_INVALID_ARG


def test_binding_has_no_fallback(monkeypatch, tmp_path):
    """The binding raises when the library is missing instead of computing
    anything elsewhere."""
    monkeypatch.setattr(isam, "_lib", None)
    monkeypatch.setattr(isam, "LIB_PATH", str(tmp_path / "missing.so"))
    with pytest.raises(ImportError):
        isam.load()


def test_grouped_rejects_bad_count_without_cuda(lib):
    p = ctypes.c_void_p(16)
    assert lib.isam_gemm_grouped(0, p, p, p, p, p, p, p, p, p, p) == isam.ISAM_ERR_INVALID_ARG
    assert lib.isam_gemm_grouped(65, p, p, p, p, p, p, p, p, p, p) == isam.ISAM_ERR_INVALID_ARG
    assert lib.isam_gemm_grouped(2, None, p, p, p, p, p, p, p, p, p) == isam.ISAM_ERR_INVALID_ARG


def test_product_path_never_references_the_oracle():
    """The library and its binding are independent of the oracle: no source
    under the package, its CUDA directory or the public header imports, loads
    or names it (synth.py, the input generators both sides share, only says
    so in its docstring)."""
    import os
    import re
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    pkg = os.path.join(root, "paper_1810_09958_gb300")
    files = [os.path.join(pkg, f) for f in os.listdir(pkg) if f.endswith(".py") and f != "synth.py"]
    csrc = os.path.join(pkg, "csrc")
    files += [os.path.join(csrc, f) for f in os.listdir(csrc) if f.endswith((".cu", ".cuh", ".h", ".cpp"))]
    files += [os.path.join(root, "include", f) for f in os.listdir(os.path.join(root, "include"))]
    pattern = re.compile(r"oracle", re.IGNORECASE)
    for path in files:
        with open(path) as f:
            assert not pattern.search(f.read()), path
    with open(os.path.join(pkg, "synth.py")) as f:
        src = f.read()
    assert not re.search(r"^\s*(import|from)\s+oracle", src, re.MULTILINE)
