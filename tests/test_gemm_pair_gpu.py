"""The CTA-pair GEMM (256 x 256 tiles, tcgen05 cta_group::2) on the GPU
against the fp64 oracle.  isam_gemm takes this path for K-major A, N % 4 == 0
and at least one 256 x 256 tile per SM pair; integer-valued inputs must match
bit for bit, others within the GEMM tolerance 5e-3."""
import numpy as np
import pytest

import oracle
from paper_1810_09958_gb300 import isam, synth
from gpu_util import Guarded, dev_bf16, nmax_err

pytestmark = pytest.mark.gpu
TOL = 5e-3


@pytest.fixture(scope="module", autouse=True)
def _lib():
    import torch
    from paper_1810_09958_gb300 import build
    build.build()
    isam.load()
    torch.cuda.set_device(0)
    yield
    isam.sync()


def run_gemm(M, N, K, tA, tB, alpha, beta, A, B, C0=None, fill=None):
    init = C0 if C0 is not None else (np.full(M * N, fill, np.float32) if fill is not None else None)
    out = Guarded(M * N, init=init)
    isam.gemm(M, N, K, tA, tB, alpha, dev_bf16(A), dev_bf16(B), beta, out.t)
    isam.sync()
    assert out.guards_intact(), "write outside C"
    return out.numpy().reshape(M, N)


def test_pair_plan_chosen_for_large_k_major_problems():
    p = isam.gemm_plan(8192, 8192, 8192, 0, 0, 1.0)
    assert (p["tile_m"], p["cta_pair"], p["BN"], p["split"]) == (256, 2, 256, 1)
    assert p["grid"] % 2 == 0
    assert isam.gemm_plan(8192, 8192, 8192, 0, 1, 0.0)["cta_pair"] == 2
    # MN-major A, N not a multiple of 4, or too few 256 x 256 tiles: one-SM tiles.
    assert isam.gemm_plan(8192, 8192, 8192, 1, 0, 0.0)["cta_pair"] == 1
    assert isam.gemm_plan(4096, 4098, 1024, 0, 1, 0.0)["cta_pair"] == 1
    assert isam.gemm_plan(512, 512, 512, 0, 0, 0.0)["cta_pair"] == 1


@pytest.mark.parametrize("tB", [0, 1], ids=["NN", "NT"])
def test_pair_integer_bit_exact_ragged(tB):
    """10 x 9 tiles of 256 with a partial tile in M, N and K (K = 9.1 k-blocks)."""
    M, N, K = 2344, 2088, 584
    assert isam.gemm_plan(M, N, K, 0, tB, -1.0)["cta_pair"] == 2
    A, B, C0 = synth.gemm_operands(M, N, K, 0, tB, seed=301 + tB, dist="int4", beta_c=True)
    got = run_gemm(M, N, K, 0, tB, 2.0, -1.0, A, B, C0=C0)
    ref = oracle.gemm(M, N, K, 0, tB, 2.0, A, B, -1.0, C0)
    assert np.array_equal(got.astype(np.float64), ref)


@pytest.mark.parametrize("tB", [0, 1], ids=["NN", "NT"])
def test_pair_uniform_parity(tB):
    M, N, K = 2560, 2304, 1000
    assert isam.gemm_plan(M, N, K, 0, tB, 0.5)["cta_pair"] == 2
    A, B, C0 = synth.gemm_operands(M, N, K, 0, tB, seed=311 + tB, beta_c=True)
    got = run_gemm(M, N, K, 0, tB, 1.25, 0.5, A, B, C0=C0)
    ref = oracle.gemm(M, N, K, 0, tB, 1.25, A, B, 0.5, C0)
    assert nmax_err(got, ref) <= TOL


def test_pair_beta_zero_does_not_read_c():
    M, N, K = 2304, 2304, 256
    A, B, _ = synth.gemm_operands(M, N, K, 0, 0, seed=321)
    got = run_gemm(M, N, K, 0, 0, 1.0, 0.0, A, B, fill=np.nan)
    assert np.isfinite(got).all()
    assert nmax_err(got, oracle.gemm(M, N, K, 0, 0, 1.0, A, B)) <= TOL


def test_pair_matches_one_sm_tiles_on_integers(monkeypatch):
    """Both tilings of an integer problem give the exact result."""
    M, N, K = 2560, 2048, 320
    A, B, _ = synth.gemm_operands(M, N, K, 0, 0, seed=331, dist="int4")
    pair = run_gemm(M, N, K, 0, 0, 1.0, 0.0, A, B)
    monkeypatch.setenv("ISAM_NO_PAIR", "1")
    assert isam.gemm_plan(M, N, K, 0, 0, 0.0)["cta_pair"] == 1
    one = run_gemm(M, N, K, 0, 0, 1.0, 0.0, A, B)
    assert np.array_equal(pair, one)


def test_pair_repeat_calls_identical():
    M, N, K = 2304, 2560, 768
    A, B, _ = synth.gemm_operands(M, N, K, 0, 1, seed=341)
    a = run_gemm(M, N, K, 0, 1, 1.0, 0.0, A, B)
    b = run_gemm(M, N, K, 0, 1, 1.0, 0.0, A, B)
    assert np.array_equal(a, b)
