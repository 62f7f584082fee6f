"""isam_gemm_fp8 on the GPU against the fp64 oracle over the same E4M3 bytes
(tolerance as isam_gemm: normalised max error <= 5e-3; integer inputs, exact in
E4M3, must match bit for bit)."""
import numpy as np
import pytest

import oracle
from paper_1810_09958_gb300 import isam, synth
from gpu_util import Guarded, nmax_err

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


def dev_u8(bits):
    import torch
    return torch.from_numpy(np.ascontiguousarray(bits).reshape(-1)).to("cuda")


def run(M, N, K, alpha, beta, A8, B8, C0=None):
    out = Guarded(M * N, init=C0)
    isam.gemm_fp8(M, N, K, alpha, dev_u8(A8), dev_u8(B8), beta, out.t)
    isam.sync()
    assert out.guards_intact(), "write outside C"
    return out.numpy().reshape(M, N)


@pytest.mark.parametrize("MK", [(1760, 1760), (2560, 2560), (4096, 4096), (7680, 2560)], ids=lambda v: f"{v[0]}x{v[1]}")
def test_fp8_skinny_sweep(MK):
    M, K = MK
    for N in (16, 32, 64, 128):
        A8 = synth.e4m3_uniform(synth.stream_seed(synth.BASE_SEED, 7, M, K, N, 1), (M, K))
        B8 = synth.e4m3_uniform(synth.stream_seed(synth.BASE_SEED, 7, M, K, N, 2), (N, K))
        got = run(M, N, K, 1.0, 0.0, A8, B8)
        ref = oracle.gemm_fp8(M, N, K, 1.0, A8, B8)
        assert nmax_err(got, ref) <= TOL, (M, N, K, isam.gemm_plan(M, N, K, 0, 1))


FORCED = [(16, 1), (32, 2), (64, 4), (128, 8), (256, 1), (128, 1), (16, 8)]


@pytest.mark.parametrize("tile", FORCED, ids=lambda t: f"BN{t[0]}s{t[1]}")
def test_fp8_integer_bit_exact_all_tiles(tile, monkeypatch):
    """Ragged M, N and K (several tiles plus a partial one in every dimension)."""
    M, N, K = 328, 200, 1168   # K = 9.1 atoms of 128
    if tile[1] > (K + 127) // 128:
        pytest.skip("split larger than the atom count")
    monkeypatch.setenv("ISAM_FORCE_TILE", f"{tile[0]},{tile[1]},0")
    A8 = synth.e4m3_integers(61, (M, K), -4, 4)
    B8 = synth.e4m3_integers(62, (N, K), -4, 4)
    C0 = synth.integers(63, M * N, -8, 8).astype(np.float32).reshape(M, N)
    got = run(M, N, K, 2.0, -1.0, A8, B8, C0)
    ref = oracle.gemm_fp8(M, N, K, 2.0, A8, B8, -1.0, C0)
    assert np.array_equal(got.astype(np.float64), ref)


@pytest.mark.parametrize("shape", [(1, 16, 16), (129, 24, 48), (1024, 1024, 1024), (1000, 8, 4112)])
def test_fp8_small_large_and_ragged(shape):
    M, N, K = shape
    A8 = synth.e4m3_uniform(M + 3 * N + K, (M, K), -2.0, 2.0)
    B8 = synth.e4m3_uniform(M + 5 * N + K, (N, K), -2.0, 2.0)
    C0 = synth.f32_uniform(M * N + 1, (M, N))
    got = run(M, N, K, 1.5, 0.5, A8, B8, C0)
    ref = oracle.gemm_fp8(M, N, K, 1.5, A8, B8, 0.5, C0)
    assert nmax_err(got, ref) <= TOL


def test_fp8_rejects_unsupported():
    import torch
    z = torch.zeros(4096, dtype=torch.uint8, device="cuda")
    c = torch.zeros(4096, dtype=torch.float32, device="cuda")
    import ctypes
    p = lambda t: ctypes.c_void_p(t.data_ptr())
    lib = isam.load()
    assert lib.isam_gemm_fp8(16, 16, 24, 1.0, p(z), p(z), 0.0, p(c)) == isam.ISAM_ERR_UNSUPPORTED
    assert lib.isam_gemm_fp8(0, 16, 16, 1.0, p(z), p(z), 0.0, p(c)) == isam.ISAM_ERR_INVALID_ARG
