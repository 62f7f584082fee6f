"""isam_gemm_grouped on the GPU: every problem of a group against the fp64
oracle (tolerance as isam_gemm: normalised max error <= 5e-3; integer inputs
bit-exact), mixed layouts and widths in one launch."""
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


def run_group(specs, dist="uniform", seed0=500):
    """specs: list of (M, N, K, tA, tB, alpha, beta). Returns [(got, ref)]."""
    probs, keep = [], []
    for i, (M, N, K, tA, tB, alpha, beta) in enumerate(specs):
        A, B, C0 = synth.gemm_operands(M, N, K, tA, tB, seed=seed0 + i, dist=dist, beta_c=True)
        out = Guarded(M * N, init=C0)
        probs.append((M, N, K, tA, tB, alpha, dev_bf16(A), dev_bf16(B), beta, out.t))
        keep.append((A, B, C0, out))
    isam.gemm_grouped(probs)
    isam.sync()
    res = []
    for (M, N, K, tA, tB, alpha, beta), (A, B, C0, out) in zip(specs, keep):
        assert out.guards_intact()
        ref = oracle.gemm(M, N, K, tA, tB, alpha, A, B, beta, C0)
        res.append((out.numpy().reshape(M, N), ref))
    return res


def test_grouped_skinny_sweep_matches_oracle():
    specs = [(M, N, K, tA, 0, 1.0, 0.0) for tA in (0, 1)
             for (M, K) in [(1760, 1760), (2560, 2560), (4096, 4096), (7680, 2560)] for N in (16, 32, 64, 128)]
    for (got, ref), spec in zip(run_group(specs), specs):
        assert nmax_err(got, ref) <= TOL, spec


def test_grouped_integer_bit_exact_mixed_layouts():
    specs = [(328, 200, 584, 0, 0, 2.0, -1.0), (200, 13, 136, 0, 1, 1.0, 0.5), (136, 48, 72, 1, 0, 1.0, 0.0),
             (64, 160, 264, 1, 1, -1.0, 1.0), (1, 8, 8, 0, 0, 1.0, 0.0), (257, 129, 1000, 0, 1, 1.0, -2.0)]
    for (got, ref), spec in zip(run_group(specs, dist="int4"), specs):
        assert np.array_equal(got.astype(np.float64), ref), spec


def test_grouped_64_problems_mixed():
    """The largest group: 64 problems of varied shape, layout, alpha and beta."""
    specs = []
    for i in range(64):
        M = 64 + 40 * (i % 7) + (i % 3)
        N = 8 * (1 + i % 20)
        K = 16 * (1 + (i * 5) % 23)
        tA, tB = i % 2, (i // 2) % 2
        if tA and M % 8:
            M += 8 - M % 8
        specs.append((M, N, K, tA, tB, 1.0 + 0.25 * (i % 3), 0.5 * (i % 2)))
    for (got, ref), spec in zip(run_group(specs, seed0=900), specs):
        assert nmax_err(got, ref) <= TOL, spec


def test_grouped_single_problem_and_beta():
    specs = [(512, 96, 512, 1, 0, 1.5, -0.5)]
    (got, ref), = run_group(specs)
    assert nmax_err(got, ref) <= TOL


def test_grouped_names_the_bad_problem():
    import torch
    z = torch.zeros(96, dtype=torch.bfloat16, device="cuda")
    c = torch.zeros(96, dtype=torch.float32, device="cuda")
    # Problem 1 has K = 12: a K-major A row pitch of 24 bytes is not 16-byte aligned.
    with pytest.raises(isam.IsamError) as e:
        isam.gemm_grouped([(8, 8, 8, 0, 0, 1.0, z[:64], z[:64], 0.0, c[:64]),
                           (8, 8, 12, 0, 0, 1.0, z, z, 0.0, c[:64])])
    assert e.value.code == isam.ISAM_ERR_UNSUPPORTED
    assert "problem 1" in str(e.value)


def dev_u8(bits):
    import torch
    return torch.from_numpy(np.ascontiguousarray(bits).reshape(-1)).to("cuda")


def run_group_fp8(specs, dist="uniform", seed0=700):
    """specs: (M, N, K, alpha, beta); E4M3 A (M x K) and B (N x K)."""
    probs, keep = [], []
    for i, (M, N, K, alpha, beta) in enumerate(specs):
        if dist == "int":
            A = synth.e4m3_integers(seed0 + 3 * i, (M, K), -4, 4)
            B = synth.e4m3_integers(seed0 + 3 * i + 1, (N, K), -4, 4)
            C0 = synth.integers(seed0 + 3 * i + 2, M * N, -8, 8).astype(np.float32).reshape(M, N)
        else:
            A = synth.e4m3_uniform(seed0 + 3 * i, (M, K))
            B = synth.e4m3_uniform(seed0 + 3 * i + 1, (N, K))
            C0 = synth.f32_uniform(seed0 + 3 * i + 2, (M, N))
        out = Guarded(M * N, init=C0)
        probs.append((M, N, K, alpha, dev_u8(A), dev_u8(B), beta, out.t))
        keep.append((A, B, C0, out))
    isam.GroupedGemmFp8(probs)()
    isam.sync()
    res = []
    for (M, N, K, alpha, beta), (A, B, C0, out) in zip(specs, keep):
        assert out.guards_intact()
        res.append((out.numpy().reshape(M, N), oracle.gemm_fp8(M, N, K, alpha, A, B, beta, C0)))
    return res


def test_grouped_fp8_skinny_shapes():
    specs = [(M, N, K, 1.0, 0.0) for (M, K) in [(1760, 1760), (2560, 2560), (4096, 4096), (7680, 2560)]
             for N in (16, 32, 64, 128)]
    for (got, ref), spec in zip(run_group_fp8(specs), specs):
        assert nmax_err(got, ref) <= TOL, spec


def test_grouped_fp8_integer_bit_exact_ragged():
    specs = [(328, 200, 1168, 2.0, -1.0), (200, 13, 144, 1.0, 0.5), (136, 48, 80, 1.0, 0.0),
             (1, 8, 16, 1.0, 0.0), (257, 129, 1008, 1.0, -2.0)]
    for (got, ref), spec in zip(run_group_fp8(specs, dist="int"), specs):
        assert np.array_equal(got.astype(np.float64), ref), spec


# 256-row tiles (two 128-row panels sharing each B block) forced on every
# problem taller than one panel: last tiles whose second panel is partial,
# a single row, or wholly below the matrix; all four layouts; beta and plain
# stores (N % 4 != 0).
TALL_SPECS = [(328, 200, 584, 0, 0, 2.0, -1.0), (200, 13, 136, 0, 1, 1.0, 0.5), (136, 48, 72, 1, 0, 1.0, 0.0),
              (384, 160, 264, 1, 1, -1.0, 1.0), (257, 129, 1000, 0, 1, 1.0, -2.0), (640, 16, 2560, 0, 0, 1.0, 0.0),
              (512, 64, 128, 1, 0, 1.0, 0.0), (1, 8, 8, 0, 0, 1.0, 0.0)]


def test_grouped_tall_tiles_integer_bit_exact(monkeypatch):
    monkeypatch.setenv("ISAM_GROUP_PANELS", "2")
    for (got, ref), spec in zip(run_group(TALL_SPECS, dist="int4", seed0=1300), TALL_SPECS):
        assert np.array_equal(got.astype(np.float64), ref), spec


def test_grouped_tall_tiles_uniform(monkeypatch):
    monkeypatch.setenv("ISAM_GROUP_PANELS", "2")
    for (got, ref), spec in zip(run_group(TALL_SPECS, seed0=1400), TALL_SPECS):
        assert nmax_err(got, ref) <= TOL, spec


def test_grouped_one_panel_tiles_on_the_sweep(monkeypatch):
    """The skinny sweep with every tile 128 rows high (the heavy problems
    take 256-row tiles by default)."""
    monkeypatch.setenv("ISAM_GROUP_PANELS", "1")
    specs = [(M, N, K, tA, 0, 1.0, 0.0) for tA in (0, 1)
             for (M, K) in [(2560, 2560), (4096, 4096)] for N in (16, 128)]
    for (got, ref), spec in zip(run_group(specs, seed0=1500), specs):
        assert nmax_err(got, ref) <= TOL, spec


def test_grouped_fp8_tall_tiles_integer_bit_exact(monkeypatch):
    monkeypatch.setenv("ISAM_GROUP_PANELS", "2")
    specs = [(328, 200, 1168, 2.0, -1.0), (200, 13, 144, 1.0, 0.5), (384, 48, 80, 1.0, 0.0),
             (257, 129, 1008, 1.0, -2.0), (1, 8, 16, 1.0, 0.0)]
    for (got, ref), spec in zip(run_group_fp8(specs, dist="int", seed0=1600), specs):
        assert np.array_equal(got.astype(np.float64), ref), spec
