"""isam_gemm_mxfp8 / isam_gemm_grouped_mxfp8 (block-scaled E4M3, one E8M0
scale per 32 K elements, passed atom-major with NaN bytes in the padding past
K, which the library must ignore) on the GPU against the fp64 oracle
(oracle.gemm_mxfp8): unit scales reproduce the grouped E4M3 GEMM bit for bit;
integer operands with power-of-two scales are exact; uniform operands with
random scales are within the GEMM tolerance (5e-3)."""
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


def dev_u8(a):
    import torch
    return torch.from_numpy(np.ascontiguousarray(a, dtype=np.uint8).reshape(-1)).to("cuda")


def atom_major(S, K, pad=255):
    """[rows][ceil(K/32)] scale bytes (the oracle's layout) rearranged into the
    library's [ceil(K/128)][rows][4]; the bytes of blocks past ceil(K/32) are
    `pad` (255 is an E8M0 NaN, which the library must ignore there)."""
    rows, kb = S.shape
    na = (K + 127) // 128
    out = np.full((na, rows, 4), pad, np.uint8)
    for a in range(na):
        for t in range(4):
            if 4 * a + t < kb:
                out[a, :, t] = S[:, 4 * a + t]
    return out


def dev_scales(S, K):
    return dev_u8(atom_major(S, K))


def operands(M, N, K, seed, dist):
    kb = (K + 31) // 32
    if dist == "int":
        A = synth.e4m3_integers(seed, (M, K), -3, 3)
        B = synth.e4m3_integers(seed + 1, (N, K), -3, 3)
        SA = synth.integers(seed + 2, M * kb, 125, 129).astype(np.uint8).reshape(M, kb)
        SB = synth.integers(seed + 3, N * kb, 125, 129).astype(np.uint8).reshape(N, kb)
        C0 = synth.integers(seed + 4, M * N, -8, 8).astype(np.float32).reshape(M, N)
    else:
        A = synth.e4m3_uniform(seed, (M, K))
        B = synth.e4m3_uniform(seed + 1, (N, K))
        SA = synth.integers(seed + 2, M * kb, 118, 136).astype(np.uint8).reshape(M, kb)
        SB = synth.integers(seed + 3, N * kb, 118, 136).astype(np.uint8).reshape(N, kb)
        C0 = synth.f32_uniform(seed + 4, (M, N))
    return A, SA, B, SB, C0


def run_mx(M, N, K, alpha, beta, A, SA, B, SB, C0):
    out = Guarded(M * N, init=C0)
    isam.gemm_mxfp8(M, N, K, alpha, dev_u8(A), dev_scales(SA, K), dev_u8(B), dev_scales(SB, K), beta, out.t)
    isam.sync()
    assert out.guards_intact()
    return out.numpy().reshape(M, N)


SHAPES = [(128, 128, 128), (256, 32, 512), (200, 13, 144), (1, 8, 16), (328, 200, 1168), (513, 64, 1040),
          (1760, 16, 1760), (384, 128, 4096)]


@pytest.mark.parametrize("M,N,K", SHAPES)
def test_unit_scales_equal_the_e4m3_gemm(M, N, K):
    """Scale byte 127 (2^0) everywhere: the block-scaled instruction must give
    exactly the unscaled E4M3 GEMM's result, summed in the same order (the
    grouped E4M3 kernel: one CTA per tile, K atoms in order, no split-K)."""
    import torch
    A, _, B, _, C0 = operands(M, N, K, 3000 + M + K, "uniform")
    kb = (K + 31) // 32
    one_a = np.full((M, kb), 127, np.uint8)
    one_b = np.full((N, kb), 127, np.uint8)
    got = run_mx(M, N, K, 1.0, 0.0, A, one_a, B, one_b, C0)
    ref = Guarded(M * N, init=C0)
    isam.GroupedGemmFp8([(M, N, K, 1.0, dev_u8(A), dev_u8(B), 0.0, ref.t)])()
    isam.sync()
    assert np.array_equal(got, ref.numpy().reshape(M, N))


@pytest.mark.parametrize("M,N,K", SHAPES)
def test_integer_operands_power_of_two_scales_exact(M, N, K):
    """Integers in [-3, 3] with scales 2^-2 .. 2^2 (different for every row
    and 32-element block of A and of B): every product and partial sum is a
    multiple of 2^-4 below 2^20, so the result equals the oracle exactly;
    alpha = 2, beta = -1 with an integer C."""
    A, SA, B, SB, C0 = operands(M, N, K, 3100 + M + K, "int")
    got = run_mx(M, N, K, 2.0, -1.0, A, SA, B, SB, C0)
    ref = oracle.gemm_mxfp8(M, N, K, 2.0, A, SA, B, SB, -1.0, C0)
    assert np.array_equal(got.astype(np.float64), ref)


@pytest.mark.parametrize("M,N,K", [(1760, 16, 1760), (2560, 64, 2560), (4096, 128, 4096), (300, 40, 1008)])
def test_uniform_operands_random_scales(M, N, K):
    A, SA, B, SB, C0 = operands(M, N, K, 3200 + M + K, "uniform")
    got = run_mx(M, N, K, 1.0, 0.0, A, SA, B, SB, C0)
    ref = oracle.gemm_mxfp8(M, N, K, 1.0, A, SA, B, SB)
    assert nmax_err(got, ref) <= TOL


def test_scale_changes_only_its_block():
    """Raising one scale byte of A (row 5, block 3) by one step doubles that
    block's contribution to row 5 and leaves every other row bit for bit."""
    M, N, K = 256, 48, 512
    A, SA, B, SB, C0 = operands(M, N, K, 3300, "int")
    base = run_mx(M, N, K, 1.0, 0.0, A, SA, B, SB, C0)
    SA2 = SA.copy()
    SA2[5, 3] += 1
    bumped = run_mx(M, N, K, 1.0, 0.0, A, SA2, B, SB, C0)
    assert np.array_equal(np.delete(bumped, 5, axis=0), np.delete(base, 5, axis=0))
    ref = oracle.gemm_mxfp8(M, N, K, 1.0, A, SA2, B, SB)
    assert np.array_equal(bumped.astype(np.float64), ref)


def test_nan_scale_poisons_only_its_row():
    """E8M0 byte 255 is NaN: row 2 of C becomes NaN, every other row stays
    finite (the oracle's reading of the format)."""
    M, N, K = 130, 24, 96
    A, SA, B, SB, C0 = operands(M, N, K, 3400, "int")
    SA = SA.copy()
    SA[2, 1] = 255
    got = run_mx(M, N, K, 1.0, 0.0, A, SA, B, SB, C0)
    assert np.isnan(got[2]).all()
    assert np.isfinite(np.delete(got, 2, axis=0)).all()


def test_grouped_mixed_problems():
    """The skinny shapes and ragged ones in one grouped launch, alpha and beta
    per problem, plain stores where N % 4 != 0; integer data exact."""
    specs = [(1760, 16, 1760, 1.0, 0.0), (2560, 32, 2560, 1.0, 0.0), (200, 13, 144, 2.0, -1.0),
             (328, 200, 1168, 1.0, 0.5), (1, 8, 16, 1.0, 0.0), (4096, 64, 1024, 0.5, 1.0)]
    probs, keep = [], []
    for i, (M, N, K, alpha, beta) in enumerate(specs):
        A, SA, B, SB, C0 = operands(M, N, K, 3500 + 7 * i, "int")
        out = Guarded(M * N, init=C0)
        probs.append((M, N, K, alpha, dev_u8(A), dev_scales(SA, K), dev_u8(B), dev_scales(SB, K), beta, out.t))
        keep.append((A, SA, B, SB, C0, out))
    isam.GroupedGemmMxfp8(probs)()
    isam.sync()
    for (M, N, K, alpha, beta), (A, SA, B, SB, C0, out) in zip(specs, keep):
        assert out.guards_intact()
        ref = oracle.gemm_mxfp8(M, N, K, alpha, A, SA, B, SB, beta, C0)
        assert np.array_equal(out.numpy().reshape(M, N).astype(np.float64), ref), (M, N, K)


def test_argument_errors():
    import torch
    z = torch.zeros(4096, dtype=torch.uint8, device="cuda")
    c = torch.zeros(256, dtype=torch.float32, device="cuda")
    lib = isam.load()
    p = lambda t: isam._ptr(t)
    # K not a multiple of 16: the rows are not 16-byte aligned
    assert lib.isam_gemm_mxfp8(8, 8, 24, 1.0, p(z), p(z), p(z), p(z), 0.0, p(c)) == isam.ISAM_ERR_UNSUPPORTED
    assert lib.isam_gemm_mxfp8(0, 8, 32, 1.0, p(z), p(z), p(z), p(z), 0.0, p(c)) == isam.ISAM_ERR_INVALID_ARG
    assert lib.isam_gemm_mxfp8(8, 8, 32, 1.0, p(z), None, p(z), p(z), 0.0, p(c)) == isam.ISAM_ERR_INVALID_ARG
    assert lib.isam_gemm_mxfp8(8, 8, 32, 1.0, p(z[1:]), p(z), p(z), p(z), 0.0, p(c)) == isam.ISAM_ERR_UNSUPPORTED
    # scale arrays hold 4-byte words
    assert lib.isam_gemm_mxfp8(8, 8, 32, 1.0, p(z), p(z[2:]), p(z), p(z), 0.0, p(c)) == isam.ISAM_ERR_UNSUPPORTED


def test_atom_major_layout_helper():
    """The rearrangement the tests use: byte t of word (a, row) is block 4a + t."""
    S = np.arange(3 * 5, dtype=np.uint8).reshape(3, 5)  # 3 rows, K = 160 -> 5 blocks, 2 atoms
    out = atom_major(S, 160)
    assert out.shape == (2, 3, 4)
    assert np.array_equal(out[0], S[:, 0:4]) and np.array_equal(out[1, :, 0], S[:, 4])
    assert (out[1, :, 1:] == 255).all()
