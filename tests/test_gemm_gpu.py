"""GEMM parity on the GPU through the C ABI (isam_gemm) against the fp64 oracle.

Tolerance: normalised max error max|gpu - ref| / (max|ref| + 1e-6) <= 5e-3;
integer-valued inputs must match bit for bit (every product and partial sum
is exact in fp32, whatever the reduction order or split)."""
import os

import numpy as np
import pytest

import oracle
from paper_1810_09958_gb300 import isam, synth
from gpu_util import Guarded, dev_bf16, nmax_err

pytestmark = pytest.mark.gpu
TOL = 5e-3

SKINNY_MK = [(1760, 1760), (2560, 2560), (4096, 4096), (7680, 2560)]
SKINNY_N = [16, 32, 64, 128]


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
    Ad, Bd = dev_bf16(A), dev_bf16(B)
    out = Guarded(M * N, init=C0 if C0 is not None else (np.full(M * N, fill, np.float32) if fill is not None else None))
    isam.gemm(M, N, K, tA, tB, alpha, Ad, Bd, beta, out.t)
    isam.sync()
    assert out.guards_intact(), "write outside C"
    return out.numpy().reshape(M, N)


def test_gemm_512_cube_nn():
    M = N = K = 512
    A, B, _ = synth.gemm_operands(M, N, K, 0, 0, seed=synth.stream_seed(synth.BASE_SEED, 0))
    got = run_gemm(M, N, K, 0, 0, 1.0, 0.0, A, B)
    ref = oracle.gemm(M, N, K, 0, 0, 1.0, A, B)
    assert nmax_err(got, ref) <= TOL


@pytest.mark.parametrize("tA", [0, 1], ids=["NN", "TN"])
@pytest.mark.parametrize("MK", SKINNY_MK, ids=lambda v: f"{v[0]}x{v[1]}")
def test_gemm_skinny_sweep(MK, tA):
    M, K = MK
    for N in SKINNY_N:
        A, B, _ = synth.gemm_operands(M, N, K, tA, 0, seed=synth.stream_seed(synth.BASE_SEED, 1, M, K, N, tA))
        got = run_gemm(M, N, K, tA, 0, 1.0, 0.0, A, B)
        ref = oracle.gemm(M, N, K, tA, 0, 1.0, A, B)
        err = nmax_err(got, ref)
        assert err <= TOL, (M, N, K, tA, err, isam.gemm_plan(M, N, K, tA, 0))


def test_gemm_8192_cube_beta1_sampled_rows():
    M = N = K = 8192
    A, B, C0 = synth.gemm_operands(M, N, K, 0, 0, seed=synth.stream_seed(synth.BASE_SEED, 2),
                                   dist="normal002", beta_c=True)
    got = run_gemm(M, N, K, 0, 0, 1.0, 1.0, A, B, C0=C0)
    rng = np.random.default_rng(2)
    rows = np.unique(np.concatenate([[0, 127, 128, M - 1], rng.integers(0, M, 92)]))
    ref = oracle.gemm(M, N, K, 0, 0, 1.0, A, B, 1.0, C0, rows=rows)
    assert nmax_err(got[rows], ref) <= TOL


FORCED = [(16, 1), (32, 2), (64, 4), (128, 8), (256, 1), (128, 1), (64, 2), (16, 8), (128, 2), (128, 4)]


@pytest.mark.parametrize("tA,tB", [(0, 0), (1, 0), (0, 1), (1, 1)], ids=["NN", "TN", "NT", "TT"])
@pytest.mark.parametrize("tile", FORCED, ids=lambda t: f"BN{t[0]}s{t[1]}")
def test_gemm_integer_bit_exact_all_tiles(tA, tB, tile, monkeypatch):
    """Ragged M, N and K (several tiles plus a partial one in every dimension)."""
    M, N, K = 328, 200, 584   # 2.56 M-tiles, K = 9.1 k-blocks, N ragged for every BN
    if tile[1] > (K + 63) // 64:
        pytest.skip("split larger than the k-block count")
    monkeypatch.setenv("ISAM_FORCE_TILE", f"{tile[0]},{tile[1]},0")
    A, B, C0 = synth.gemm_operands(M, N, K, tA, tB, seed=77 + tA + 2 * tB, dist="int4", beta_c=True)
    got = run_gemm(M, N, K, tA, tB, 2.0, -1.0, A, B, C0=C0)
    ref = oracle.gemm(M, N, K, tA, tB, 2.0, A, B, -1.0, C0)
    assert np.array_equal(got.astype(np.float64), ref)
    plan = isam.gemm_plan(M, N, K, tA, tB, -1.0)
    assert (plan["BN"], plan["split"]) == tile


@pytest.mark.parametrize("shape", [(8, 8, 8), (1, 8, 8), (8, 8, 16), (129, 24, 40), (64, 264, 8),
                                   (1000, 16, 72), (136, 8, 4104)])
@pytest.mark.parametrize("tA", [0, 1])
def test_gemm_small_and_ragged(shape, tA):
    M, N, K = shape
    if tA and M % 8:
        M = (M + 7) // 8 * 8
    A, B, C0 = synth.gemm_operands(M, N, K, tA, 0, seed=M * 7 + N * 3 + K, beta_c=True)
    got = run_gemm(M, N, K, tA, 0, 1.5, -0.5, A, B, C0=C0)
    ref = oracle.gemm(M, N, K, tA, 0, 1.5, A, B, -0.5, C0)
    assert nmax_err(got, ref) <= TOL


@pytest.mark.parametrize("tA", [0, 1], ids=["NT", "TT"])
def test_gemm_odd_n_c_rows_not_16_byte_aligned(tA):
    """N = 13 and 77 with K-major B (transB = 1): a row of C is not 16-byte
    aligned, so C moves by plain stores; integer inputs must match exactly."""
    for (M, N, K) in [(200, 13, 136), (136, 77, 520)]:
        A, B, C0 = synth.gemm_operands(M, N, K, tA, 1, seed=M + N + K + tA, dist="int4", beta_c=True)
        got = run_gemm(M, N, K, tA, 1, 2.0, -1.0, A, B, C0=C0)
        ref = oracle.gemm(M, N, K, tA, 1, 2.0, A, B, -1.0, C0)
        assert np.array_equal(got.astype(np.float64), ref), (M, N, K)


def test_gemm_beta_zero_does_not_read_c():
    M, N, K = 384, 128, 256
    A, B, _ = synth.gemm_operands(M, N, K, 0, 0, seed=5)
    got = run_gemm(M, N, K, 0, 0, 1.0, 0.0, A, B, fill=np.nan)
    assert np.isfinite(got).all()
    assert nmax_err(got, oracle.gemm(M, N, K, 0, 0, 1.0, A, B)) <= TOL


@pytest.mark.parametrize("split", [2, 4, 8])
def test_gemm_split_k_several_tiles_per_cluster(split, monkeypatch):
    """128-column split tiles (partial rows pushed through the per-warp
    transpose) with more tiles than resident clusters, so every cluster runs
    several tiles and reuses its reduction slots; ragged M, N and K, integer
    data exact."""
    monkeypatch.setenv("ISAM_FORCE_TILE", f"128,{split},0")
    M, N, K = 5000, 136, 520
    A, B, C0 = synth.gemm_operands(M, N, K, 0, 0, seed=300 + split, dist="int4", beta_c=True)
    got = run_gemm(M, N, K, 0, 0, 2.0, -1.0, A, B, C0=C0)
    ref = oracle.gemm(M, N, K, 0, 0, 2.0, A, B, -1.0, C0)
    assert np.array_equal(got.astype(np.float64), ref)
    plan = isam.gemm_plan(M, N, K, 0, 0, -1.0)
    assert (plan["BN"], plan["split"]) == (128, split)
    assert plan["grid"] // split < 40 * 2  # fewer resident clusters than tiles


def test_gemm_split_k_deterministic(monkeypatch):
    monkeypatch.setenv("ISAM_FORCE_TILE", "64,8,0")
    M, N, K = 1760, 64, 1760
    A, B, _ = synth.gemm_operands(M, N, K, 0, 0, seed=9)
    a = run_gemm(M, N, K, 0, 0, 1.0, 0.0, A, B)
    b = run_gemm(M, N, K, 0, 0, 1.0, 0.0, A, B)
    assert np.array_equal(a, b)


def test_gemm_on_side_stream():
    import torch
    M, N, K = 512, 64, 512
    A, B, _ = synth.gemm_operands(M, N, K, 1, 0, seed=10)
    s = torch.cuda.Stream()
    Ad, Bd = dev_bf16(A), dev_bf16(B)
    C = torch.zeros(M * N, dtype=torch.float32, device="cuda")
    torch.cuda.synchronize()
    with torch.cuda.stream(s):
        isam.gemm(M, N, K, 1, 0, 1.0, Ad, Bd, 0.0, C)
    isam.sync()
    s.synchronize()
    ref = oracle.gemm(M, N, K, 1, 0, 1.0, A, B)
    assert nmax_err(C.cpu().numpy().reshape(M, N), ref) <= TOL


def test_gemm_rejects_mismatched_tensor():
    import torch
    A = torch.zeros(64, dtype=torch.float32, device="cuda")
    with pytest.raises(ValueError):
        isam.gemm(8, 8, 8, 0, 0, 1.0, A, A, 0.0, A)
