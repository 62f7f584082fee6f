"""Separable depthwise convolution parity on the GPU through the C ABI
(isam_dwsep_conv) against the fp64 oracle.  Tolerance: normalised max error
<= 5e-3; integer-valued inputs (depthwise sums exactly representable in bf16)
must match bit for bit."""
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


def run_dwsep(x, dw, pw):
    N, H, W, Cin = x.shape
    Cout = pw.shape[1]
    out = Guarded(N * H * W * Cout)
    isam.dwsep_conv(N, H, W, Cin, Cout, dev_bf16(x), dev_bf16(dw), dev_bf16(pw), out.t)
    isam.sync()
    assert out.guards_intact(), "write outside out"
    return out.numpy().reshape(N, H, W, Cout)


def test_dwsep_benchmark_layer_full_oracle():
    """N = 32, 56 x 56, 128 -> 256 channels (the benchmark layer)."""
    N, H, W, Cin, Cout = 32, 56, 56, 128, 256
    x, dw, pw = synth.dwsep_operands(N, H, W, Cin, Cout, seed=synth.stream_seed(synth.BASE_SEED, 4))
    got = run_dwsep(x, dw, pw)
    ref = oracle.dwsep(x, dw, pw)
    assert nmax_err(got, ref) <= TOL


@pytest.mark.parametrize("shape", [(1, 1, 1, 16, 32), (1, 5, 7, 16, 16), (2, 9, 8, 32, 48),
                                   (3, 4, 33, 64, 96), (2, 13, 11, 128, 256), (1, 3, 130, 48, 16),
                                   (1, 7, 19, 256, 64), (4, 2, 3, 80, 144),
                                   # one-row tiles (65 <= W <= 128), exactly 128 pixels, full
                                   # 2 x 64 tiles, many small images (tiles of several images
                                   # per CTA), a 48-channel input (12 lanes per pixel)
                                   (2, 6, 100, 32, 32), (1, 4, 128, 64, 128), (2, 10, 64, 128, 256),
                                   (200, 3, 40, 64, 64), (3, 8, 24, 48, 80)])
def test_dwsep_shapes(shape):
    N, H, W, Cin, Cout = shape
    x, dw, pw = synth.dwsep_operands(N, H, W, Cin, Cout, seed=sum(shape) * 31 + Cin)
    got = run_dwsep(x, dw, pw)
    ref = oracle.dwsep(x, dw, pw)
    assert nmax_err(got, ref) <= TOL, shape


def test_dwsep_integer_bit_exact():
    N, H, W, Cin, Cout = 3, 10, 17, 64, 96
    x = synth.bf16_integers(1, (N, H, W, Cin), -3, 3)
    dw = synth.bf16_integers(2, (3, 3, Cin), -2, 2)
    pw = synth.bf16_integers(3, (Cin, Cout), -2, 2)
    got = run_dwsep(x, dw, pw)
    ref = oracle.dwsep(x, dw, pw)
    assert np.array_equal(got.astype(np.float64), ref)


def test_dwsep_ones_window_boundary_pattern():
    """All-ones window on a constant image with an identity pointwise stage:
    9c inside, 6c on edges, 4c in corners."""
    N, H, W, C = 2, 6, 9, 32
    c = 1.5
    x = synth.to_bf16_bits(np.full((N, H, W, C), c))
    dw = synth.to_bf16_bits(np.ones((3, 3, C)))
    pw = synth.to_bf16_bits(np.eye(C))
    got = run_dwsep(x, dw, pw)
    rows = np.array([2] + [3] * (H - 2) + [2])
    cols = np.array([2] + [3] * (W - 2) + [2])
    want = c * np.outer(rows, cols)
    for k in range(C):
        assert np.array_equal(got[0, :, :, k].astype(np.float64), want)


def test_dwsep_benchmark_layer_plan():
    """The benchmark layer runs as one launch of the row-ring kernel, two
    image rows (112 pixels) per tile."""
    assert isam.dwsep_plan(56, 128, 256) == {"kernel": 0, "rows_per_tile": 2, "blocks": 1, "block_cout": 256}


# (N, H, W, Cin, Cout) with the plan the shared-memory budget gives: wide
# layers whose resident pointwise weights do not fit in one launch run as
# several output-channel blocks, each block's columns written with the
# layer's full row pitch (unwritten outputs would keep the canary value).
BLOCKED = [
    ((2, 5, 8, 256, 256), (0, 6, 2, 128)),     # row ring, 6 rows per tile, 2 blocks
    ((1, 6, 56, 192, 256), (0, 1, 2, 128)),    # row ring, one row per tile, 2 blocks
    ((1, 4, 56, 256, 256), (1, 0, 4, 64)),     # per-pixel kernel, 4 blocks
    ((1, 3, 130, 256, 256), (1, 0, 4, 64)),    # wider than one MMA block
    ((2, 3, 130, 208, 80), (1, 0, 2, 48)),     # 48-wide blocks (a 16-column TMEM tail)
    ((2, 4, 130, 144, 208), (1, 0, 2, 112)),
    # the row ring with idle producer threads (52 and 36 channel groups do
    # not divide the producers; the threads past the last whole segment only
    # join the barriers)
    ((2, 3, 11, 208, 80), (0, 5, 1, 80)),
    ((2, 4, 33, 144, 208), (0, 1, 1, 208)),
    ((3, 2, 1, 256, 256), (0, 15, 2, 128)),    # one-pixel-wide images
]


@pytest.mark.parametrize("shape,plan", BLOCKED, ids=[str(s[0]) for s in BLOCKED])
def test_dwsep_channel_blocks(shape, plan):
    N, H, W, Cin, Cout = shape
    got_plan = isam.dwsep_plan(W, Cin, Cout)
    assert (got_plan["kernel"], got_plan["rows_per_tile"], got_plan["blocks"], got_plan["block_cout"]) == plan
    x, dw, pw = synth.dwsep_operands(N, H, W, Cin, Cout, seed=sum(shape) * 17 + Cout)
    got = run_dwsep(x, dw, pw)
    ref = oracle.dwsep(x, dw, pw)
    assert nmax_err(got, ref) <= TOL, shape


def test_dwsep_channel_blocks_integer_bit_exact():
    """256 -> 256 channels in two blocks of 128: exact on integer data."""
    N, H, W, Cin, Cout = 2, 5, 8, 256, 256
    assert isam.dwsep_plan(W, Cin, Cout)["blocks"] == 2
    x = synth.bf16_integers(11, (N, H, W, Cin), -3, 3)
    dw = synth.bf16_integers(12, (3, 3, Cin), -2, 2)
    pw = synth.bf16_integers(13, (Cin, Cout), -2, 2)
    got = run_dwsep(x, dw, pw)
    ref = oracle.dwsep(x, dw, pw)
    assert np.array_equal(got.astype(np.float64), ref)


def test_dwsep_unsupported_rejected():
    import ctypes
    import torch
    z = torch.zeros(1 << 16, dtype=torch.bfloat16, device="cuda")
    f = torch.zeros(1 << 16, dtype=torch.float32, device="cuda")
    lib = isam.load()
    p = lambda t: ctypes.c_void_p(t.data_ptr())
    assert lib.isam_dwsep_conv(1, 4, 4, 24, 16, p(z), p(z), p(z), p(f)) == isam.ISAM_ERR_UNSUPPORTED
    assert lib.isam_dwsep_conv(1, 4, 4, 16, 272, p(z), p(z), p(z), p(f)) == isam.ISAM_ERR_UNSUPPORTED
    assert lib.isam_dwsep_conv(1, 4, 4, 272, 16, p(z), p(z), p(z), p(f)) == isam.ISAM_ERR_UNSUPPORTED
    out = (ctypes.c_int * 4)()
    assert lib.isam_dwsep_plan_info(4, 16, 8, out) == isam.ISAM_ERR_UNSUPPORTED


def test_dwsep_plan_on_the_device_matches_the_host_plan():
    for (W, cin, cout) in [(56, 128, 256), (56, 256, 256), (8, 256, 256), (130, 48, 16)]:
        assert isam.dwsep_plan(W, cin, cout) == isam.dwsep_plan(W, cin, cout, smem_optin=232448)


# ---- the depthwise factor alone (isam_depthwise_conv3x3) and the unfused
# schedule: depthwise to memory, then the pointwise factor through isam_gemm

def run_depthwise(x, dw):
    import torch
    N, H, W, C = x.shape
    y = torch.full((N * H * W * C + 2 * 64,), float("nan"), dtype=torch.bfloat16, device="cuda")
    yv = y[64:64 + N * H * W * C]
    isam.depthwise_conv3x3(N, H, W, C, dev_bf16(x), dev_bf16(dw), yv)
    isam.sync()
    guard = y.float().cpu().numpy()
    assert np.isnan(guard[:64]).all() and np.isnan(guard[-64:]).all(), "write outside y"
    return yv, yv.float().cpu().numpy().reshape(N, H, W, C)


def identity_pw(C):
    return synth.to_bf16_bits(np.eye(C))


@pytest.mark.parametrize("shape", [(1, 1, 1, 8), (2, 5, 7, 16), (1, 9, 130, 24), (3, 4, 33, 64), (2, 13, 11, 128),
                                   (32, 56, 56, 128)])
def test_depthwise_alone_matches_oracle(shape):
    """The oracle's separable layer with an identity pointwise factor is the
    depthwise sum itself (each output channel picks one input channel, exactly
    in fp64); the kernel sums in fp32 and rounds once to bf16 (8 significant
    bits), so each element is within 2^-8 of its own magnitude and the
    normalised error is at most 2^-8 (plus fp32 summation, far below)."""
    N, H, W, C = shape
    x, dw, _ = synth.dwsep_operands(N, H, W, C, C, seed=sum(shape) * 17 + C)
    _, got = run_depthwise(x, dw)
    ref = oracle.dwsep(x, dw, identity_pw(C))
    assert nmax_err(got, ref) <= 2.0 ** -8 + 1e-6, shape


def test_depthwise_alone_integer_exact():
    """Integer data whose window sums fit bf16's 8-bit significand: exact."""
    N, H, W, C = 2, 6, 9, 32
    x = synth.to_bf16_bits(synth.integers(601, N * H * W * C, -3, 3).reshape(N, H, W, C))
    dw = synth.to_bf16_bits(synth.integers(602, 9 * C, -2, 2).reshape(3, 3, C))
    _, got = run_depthwise(x, dw)
    ref = oracle.dwsep(x, dw, identity_pw(C))
    assert np.array_equal(got.astype(np.float64), ref)


def test_unfused_schedule_matches_oracle_and_fused_layer():
    """Depthwise to memory, then isam_gemm(M = N*H*W, N = Cout, K = Cin,
    A = y, B = pw_w): the separable layer within the tolerance, and equal to
    the fused kernel up to summation order (both feed bf16 depthwise sums to
    fp32-accumulating tensor cores)."""
    import torch
    N, H, W, Cin, Cout = 4, 14, 14, 128, 256
    x, dw, pw = synth.dwsep_operands(N, H, W, Cin, Cout, seed=611)
    yv, _ = run_depthwise(x, dw)
    M = N * H * W
    out = Guarded(M * Cout)
    isam.gemm(M, Cout, Cin, 0, 0, 1.0, yv, dev_bf16(pw), 0.0, out.t)
    isam.sync()
    assert out.guards_intact()
    unfused = out.numpy().reshape(N, H, W, Cout)
    ref = oracle.dwsep(x, dw, pw)
    assert nmax_err(unfused, ref) <= TOL
    fused = run_dwsep(x, dw, pw)
    assert nmax_err(unfused, fused) <= 1e-5


def test_depthwise_rejects_bad_arguments():
    import torch
    lib = isam.load()
    z = torch.zeros(4096, dtype=torch.bfloat16, device="cuda")
    p = isam._ptr
    assert lib.isam_depthwise_conv3x3(1, 2, 2, 12, p(z), p(z), p(z)) == isam.ISAM_ERR_UNSUPPORTED  # C % 8
    assert lib.isam_depthwise_conv3x3(1, 2, 2, 16, p(z[1:]), p(z), p(z)) == isam.ISAM_ERR_UNSUPPORTED
    assert lib.isam_depthwise_conv3x3(0, 2, 2, 16, p(z), p(z), p(z)) == isam.ISAM_ERR_INVALID_ARG
    assert lib.isam_depthwise_conv3x3(1, 2, 2, 16, None, p(z), p(z)) == isam.ISAM_ERR_INVALID_ARG
