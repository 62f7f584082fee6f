"""Pins the fp64 oracle to facts that do not come from the oracle itself:
brute force on tiny inputs, exact integer arithmetic, identity and permutation
matrices, closed forms of the GRU recurrence, the boundary pattern of the 3x3
window, and independent library routines (numpy / torch float64).

Each pin is chosen so that a plausible slip in the oracle (a dropped term, a
swapped index or operand, a wrong sign, a bias in the wrong place) fails it.
"""
import math

import numpy as np
import pytest

from paper_1810_09958_gb300 import synth


def f64(bits):
    return synth.bf16_bits_to_f64(bits)


def opA(A, M, K, transA):
    a = f64(A)
    return a.reshape(K, M).T if transA else a.reshape(M, K)


def opB(B, K, N, transB):
    b = f64(B)
    return b.reshape(N, K).T if transB else b.reshape(K, N)


# --------------------------------------------------------------------------
# GEMM (Listing 1 / Listing 4)
# --------------------------------------------------------------------------
@pytest.mark.parametrize("transA", [0, 1])
@pytest.mark.parametrize("transB", [0, 1])
def test_gemm_bruteforce_tiny(oracle_lib, transA, transB):
    rng = np.random.default_rng(7)
    for trial in range(6):
        M, N, K = (int(v) for v in rng.integers(1, 34, size=3))
        A, B, C = synth.gemm_operands(M, N, K, transA, transB, seed=100 + trial, beta_c=True)
        alpha, beta = 1.5, -0.75
        got = oracle_lib.gemm(M, N, K, transA, transB, alpha, A, B, beta, C)
        a, b = opA(A, M, K, transA), opB(B, K, N, transB)
        for i in range(M):
            for j in range(N):
                s = 0.0
                for k in range(K):
                    s += float(a[i, k]) * float(b[k, j])
                want = alpha * s + beta * float(C[i, j])
                assert got[i, j] == want, (M, N, K, i, j)


def test_gemm_integer_exact(oracle_lib):
    for transA in (0, 1):
        M, N, K = 37, 19, 301
        A, B, C = synth.gemm_operands(M, N, K, transA, 0, seed=11, dist="int4", beta_c=True)
        ai = opA(A, M, K, transA).astype(np.int64)
        bi = opB(B, K, N, 0).astype(np.int64)
        got = oracle_lib.gemm(M, N, K, transA, 0, 1.0, A, B)
        assert np.array_equal(got, (ai @ bi).astype(np.float64))
        # alpha = 2, beta = -1 closed form on integers.
        got2 = oracle_lib.gemm(M, N, K, transA, 0, 2.0, A, B, -1.0, C)
        want2 = 2 * (ai @ bi) - C.astype(np.int64)
        assert np.array_equal(got2, want2.astype(np.float64))


def test_gemm_identity_and_permutation(oracle_lib):
    M, K = 23, 40
    A, _, _ = synth.gemm_operands(M, K, K, 0, 0, seed=5)
    eye = synth.to_bf16_bits(np.eye(K))
    got = oracle_lib.gemm(M, K, K, 0, 0, 1.0, A, eye)
    assert np.array_equal(got, f64(A).reshape(M, K))
    perm = np.random.default_rng(3).permutation(K)
    P = np.zeros((K, K))
    P[perm, np.arange(K)] = 1.0          # column j of A @ P is column perm[j] of A
    got = oracle_lib.gemm(M, K, K, 0, 0, 1.0, A, synth.to_bf16_bits(P))
    assert np.array_equal(got, f64(A).reshape(M, K)[:, perm])
    # Same through the transposed-A path: I @ A^T stored K x M.
    At = np.ascontiguousarray(A.reshape(M, K).T)
    got = oracle_lib.gemm(M, K, K, 1, 0, 1.0, At, eye)
    assert np.array_equal(got, f64(A).reshape(M, K))
    # Left identity through transB: A = I_M @ A with A read as B^T.
    eyeM = synth.to_bf16_bits(np.eye(M))
    got = oracle_lib.gemm(M, K, M, 0, 1, 1.0, eyeM, At)
    assert np.array_equal(got, f64(A).reshape(M, K))


def test_gemm_beta_zero_ignores_c(oracle_lib):
    M, N, K = 8, 9, 10
    A, B, _ = synth.gemm_operands(M, N, K, 0, 0, seed=9)
    Cnan = np.full((M, N), np.nan, dtype=np.float32)
    got = oracle_lib.gemm(M, N, K, 0, 0, 1.0, A, B, 0.0, Cnan)
    assert np.isfinite(got).all()


def test_gemm_vs_numpy_float64(oracle_lib):
    for transA, transB in ((0, 0), (1, 0), (0, 1)):
        M, N, K = 130, 70, 257
        A, B, C = synth.gemm_operands(M, N, K, transA, transB, seed=21, beta_c=True)
        got = oracle_lib.gemm(M, N, K, transA, transB, 0.5, A, B, 2.0, C)
        want = 0.5 * (opA(A, M, K, transA) @ opB(B, K, N, transB)) + 2.0 * C.astype(np.float64)
        assert np.max(np.abs(got - want)) <= 1e-12 * np.max(np.abs(want))


def test_gemm_rows_subset_matches_full(oracle_lib):
    M, N, K = 50, 33, 64
    A, B, C = synth.gemm_operands(M, N, K, 1, 0, seed=31, beta_c=True)
    full = oracle_lib.gemm(M, N, K, 1, 0, 1.0, A, B, 1.0, C)
    rows = np.array([49, 0, 17, 17, 3])
    sub = oracle_lib.gemm(M, N, K, 1, 0, 1.0, A, B, 1.0, C, rows=rows)
    assert np.array_equal(sub, full[rows])


def test_gemm_rejects_bad_args(oracle_lib):
    A = np.zeros(4, np.uint16)
    with pytest.raises(ValueError):
        oracle_lib.gemm(2, 2, 2, 0, 0, 1.0, A, A, 1.0, None)   # beta != 0 needs C


# --------------------------------------------------------------------------
# GRU (Section 3.6 recurrent scheduling; Section 5.1.2)
# --------------------------------------------------------------------------
def sig(v):
    return 1.0 / (1.0 + np.exp(-v))


def test_gru_zero_weights_closed_form(oracle_lib):
    """W = U = 0: r, z, n are constants from the biases and
    h_t = n + z**t * (h0 - n) (geometric decay towards n)."""
    T, batch, H = 9, 3, 16
    zero = np.zeros((3 * H, H), np.uint16)
    x = synth.bf16_normal(1, (T, batch, H))
    b = synth.f32_uniform(2, (6 * H,), -2.0, 2.0)
    h0 = synth.f32_uniform(3, (batch, H))
    got = oracle_lib.gru_forward(x, zero, zero, b, h0)
    bd = b.astype(np.float64)
    r = sig(bd[0:H] + bd[3 * H:4 * H])
    z = sig(bd[H:2 * H] + bd[4 * H:5 * H])
    n = np.tanh(bd[2 * H:3 * H] + r * bd[5 * H:6 * H])
    for t in range(T):
        want = n[None, :] + z[None, :] ** (t + 1) * (h0.astype(np.float64) - n[None, :])
        np.testing.assert_allclose(got[t], want, rtol=0, atol=1e-14)


def test_gru_saturated_update_gate_keeps_h0(oracle_lib):
    """b_z = +30 drives z to 1 - 9.4e-14, so h_t stays at h0."""
    T, batch, H = 12, 2, 32
    x, W, U, b, _ = synth.gru_operands(T, batch, H, seed=4)
    b = b.copy()
    b[H:2 * H] = 30.0
    h0 = synth.f32_uniform(5, (batch, H))
    got = oracle_lib.gru_forward(x, W, U, b, h0)
    for t in range(T):
        np.testing.assert_allclose(got[t], h0.astype(np.float64), rtol=0, atol=1e-11)


def test_gru_closed_update_gate_follows_candidate(oracle_lib):
    """b_z = -30 drives z to ~1e-13, so h_t is the candidate alone: h_t = n_t
    with n_t = tanh(W_n x_t + b_in + r_t * (U_n h_{t-1} + b_hn)) and
    r_t = sigmoid(W_r x_t + b_ir + U_r h_{t-1} + b_hr), evaluated step by step
    in float64 numpy (the one-step formula, no update-gate term)."""
    T, batch, H = 6, 3, 24
    x, W, U, b, _ = synth.gru_operands(T, batch, H, seed=14)
    b = b.copy()
    b[H:2 * H] = -30.0
    h0 = synth.f32_uniform(15, (batch, H))
    got = oracle_lib.gru_forward(x, W, U, b, h0)
    Wf, Uf, xf, bb = f64(W), f64(U), f64(x), b.astype(np.float64)
    h = h0.astype(np.float64)
    for t in range(T):
        gx = xf[t] @ Wf.T + bb[:3 * H]
        gh = h @ Uf.T + bb[3 * H:]
        r = sig(gx[:, :H] + gh[:, :H])
        h = np.tanh(gx[:, 2 * H:] + r * gh[:, 2 * H:])
        np.testing.assert_allclose(got[t], h, rtol=0, atol=1e-11)


def test_gru_matches_torch_float64(oracle_lib):
    """torch.nn.GRU uses the same (r, z, n) order with the reset gate applied
    after the recurrent product, so it is an independent implementation."""
    torch = pytest.importorskip("torch")
    T, batch, H = 7, 4, 24
    x, W, U, b, _ = synth.gru_operands(T, batch, H, seed=8)
    h0 = synth.f32_uniform(9, (batch, H))
    got = oracle_lib.gru_forward(x, W, U, b, h0)
    gru = torch.nn.GRU(H, H, num_layers=1, bias=True).double()
    with torch.no_grad():
        gru.weight_ih_l0.copy_(torch.from_numpy(f64(W)))
        gru.weight_hh_l0.copy_(torch.from_numpy(f64(U)))
        gru.bias_ih_l0.copy_(torch.from_numpy(b[:3 * H].astype(np.float64)))
        gru.bias_hh_l0.copy_(torch.from_numpy(b[3 * H:].astype(np.float64)))
        out, hT = gru(torch.from_numpy(f64(x)), torch.from_numpy(h0.astype(np.float64))[None])
    np.testing.assert_allclose(got, out.numpy(), rtol=0, atol=1e-12)
    np.testing.assert_allclose(got[-1], hT[0].numpy(), rtol=0, atol=1e-12)


def test_gru_single_step_from_zero_state(oracle_lib):
    """T = 1 and h0 = 0: the recurrent product vanishes, so h_1 = (1 - z) n with
    every gate a function of W x + biases alone (one GEMM, numpy's)."""
    T, batch, H = 1, 5, 16
    x, W, U, b, h0 = synth.gru_operands(T, batch, H, seed=12)
    got = oracle_lib.gru_forward(x, W, U, b, h0)
    gx = f64(x[0]) @ f64(W).T + b[:3 * H].astype(np.float64)
    bh = b[3 * H:].astype(np.float64)
    r = sig(gx[:, :H] + bh[:H])
    z = sig(gx[:, H:2 * H] + bh[H:2 * H])
    n = np.tanh(gx[:, 2 * H:] + r * bh[2 * H:])
    np.testing.assert_allclose(got[0], (1 - z) * n, rtol=0, atol=1e-14)


def test_gru_batch_rows_independent(oracle_lib):
    T, batch, H = 5, 6, 16
    x, W, U, b, _ = synth.gru_operands(T, batch, H, seed=14)
    h0 = synth.f32_uniform(15, (batch, H))
    full = oracle_lib.gru_forward(x, W, U, b, h0)
    sel = [4, 1]
    sub = oracle_lib.gru_forward(np.ascontiguousarray(x[:, sel]), W, U, b, h0[sel])
    assert np.array_equal(sub, full[:, sel])


# --------------------------------------------------------------------------
# Separable depthwise convolution (Listing 3, factorisation of Section 2.3)
# --------------------------------------------------------------------------
def test_dwsep_literal_listing_loop(oracle_lib):
    """The unfactored 8-deep loop of Listing 3 (s = 1, c = 1, zero border of
    one pixel), brute force on a tiny case, equals the factored oracle."""
    N, H, W, Cin, Cout = 2, 4, 5, 3, 4
    x, dw, pw = synth.dwsep_operands(N, H, W, Cin, Cout, seed=17)
    X, D, P = f64(x), f64(dw), f64(pw)
    want = np.zeros((N, H, W, Cout))
    for b in range(N):
        for i in range(H):
            for j in range(W):
                for k in range(Cout):
                    for di in range(3):
                        for dj in range(3):
                            for q in range(Cin):
                                for r in range(1):
                                    ii, jj = i + di - 1, j + dj - 1
                                    if 0 <= ii < H and 0 <= jj < W:
                                        want[b, i, j, k] += X[b, ii, jj, q] * D[di, dj, q] * P[q + r, k]
    got = oracle_lib.dwsep(x, dw, pw)
    np.testing.assert_allclose(got, want, rtol=1e-13, atol=1e-15)


def test_dwsep_delta_kernel_is_pointwise_gemm(oracle_lib):
    N, H, W, Cin, Cout = 2, 6, 7, 16, 24
    x, _, pw = synth.dwsep_operands(N, H, W, Cin, Cout, seed=19)
    D = np.zeros((3, 3, Cin))
    D[1, 1, :] = 1.0
    got = oracle_lib.dwsep(x, synth.to_bf16_bits(D), pw)
    want = f64(x).reshape(-1, Cin) @ f64(pw)
    np.testing.assert_allclose(got.reshape(-1, Cout), want, rtol=1e-13, atol=1e-15)


def test_dwsep_ones_window_boundary_pattern(oracle_lib):
    """All-ones 3x3 window on a constant image, identity pointwise: 9c inside,
    6c on edges, 4c in corners (exact)."""
    N, H, W, C = 1, 5, 6, 8
    c = 1.5
    x = synth.to_bf16_bits(np.full((N, H, W, C), c))
    D = synth.to_bf16_bits(np.ones((3, 3, C)))
    P = synth.to_bf16_bits(np.eye(C))
    got = oracle_lib.dwsep(x, D, P)[0, :, :, 0]
    rows = np.array([2] + [3] * (H - 2) + [2])
    cols = np.array([2] + [3] * (W - 2) + [2])
    assert np.array_equal(got, c * np.outer(rows, cols))


def test_dwsep_integer_exact(oracle_lib):
    N, H, W, Cin, Cout = 1, 7, 9, 16, 8
    x = synth.bf16_integers(31, (N, H, W, Cin), -3, 3)
    dw = synth.bf16_integers(32, (3, 3, Cin), -2, 2)
    pw = synth.bf16_integers(33, (Cin, Cout), -2, 2)
    X = np.pad(f64(x).astype(np.int64), ((0, 0), (1, 1), (1, 1), (0, 0)))
    D = f64(dw).astype(np.int64)
    Y = np.zeros((N, H, W, Cin), np.int64)
    for di in range(3):
        for dj in range(3):
            Y += X[:, di:di + H, dj:dj + W, :] * D[di, dj]
    want = (Y.reshape(-1, Cin) @ f64(pw).astype(np.int64)).reshape(N, H, W, Cout)
    assert np.array_equal(oracle_lib.dwsep(x, dw, pw), want.astype(np.float64))


def test_dwsep_matches_torch_conv_float64(oracle_lib):
    torch = pytest.importorskip("torch")
    F = torch.nn.functional
    N, H, W, Cin, Cout = 2, 9, 8, 16, 32
    x, dw, pw = synth.dwsep_operands(N, H, W, Cin, Cout, seed=41)
    xt = torch.from_numpy(f64(x)).permute(0, 3, 1, 2)                  # NCHW
    wd = torch.from_numpy(f64(dw)).permute(2, 0, 1).unsqueeze(1)       # [Cin,1,3,3]
    wp = torch.from_numpy(f64(pw)).t().reshape(Cout, Cin, 1, 1)
    y = F.conv2d(F.conv2d(xt, wd, padding=1, groups=Cin), wp)
    want = y.permute(0, 2, 3, 1).numpy()
    np.testing.assert_allclose(oracle_lib.dwsep(x, dw, pw), want, rtol=0, atol=1e-12)


# --------------------------------------------------------------------------
# Input generator sanity (it feeds both sides)
# --------------------------------------------------------------------------
def test_splitmix64_reference_values():
    """First outputs of SplitMix64 seeded with 0 (published reference values
    of the generator as defined by Steele, Lea and Flood / Vigna)."""
    z = synth.splitmix64(0, 0, 3)
    assert [int(v) for v in z] == [0xE220A8397B1DCDAF, 0x6E789E6AA1B965F4, 0x06C45D188009454F]


def test_bf16_rounding_is_nearest_even():
    vals = np.array([1.0, 1.0 + 2 ** -8, 1.0 + 3 * 2 ** -8, -2.5, 1.0 + 2 ** -9], dtype=np.float32)
    bits = synth.to_bf16_bits(vals)
    back = synth.bf16_bits_to_f32(bits)
    assert back.tolist() == [1.0, 1.0, 1.0 + 2 ** -6, -2.5, 1.0]


def test_torch_generator_matches_numpy():
    torch = pytest.importorskip("torch")
    n = 100_003
    seed = synth.stream_seed(synth.BASE_SEED, 1, 7)
    a = synth.bf16_uniform(seed, (n,))
    b = synth.bf16_uniform_torch(seed, n, "cpu").view(torch.int16).numpy().view(np.uint16)
    assert np.array_equal(a, b)
    c = synth.f32_uniform(seed, (n,))
    d = synth.f32_uniform_torch(seed, n, "cpu").numpy()
    assert np.array_equal(c, d)
    e = synth.bf16_normal(seed, (n,)).astype(np.int32)
    f = synth.bf16_normal_torch(seed, n, "cpu").view(torch.int16).numpy().view(np.uint16).astype(np.int32)
    assert np.mean(e == f) > 0.999


def test_uniform_at_matches_stream():
    seed = synth.stream_seed(synth.BASE_SEED, 9)
    full = synth.uniform(seed, 5000)
    idx = np.array([[0, 4999, 17], [2500, 3, 3]])
    assert np.array_equal(synth.uniform_at(seed, idx), full[idx])


# --------------------------------------------------------------------------- E4M3 (8-bit) GEMM

def test_e4m3_decode_known_values(oracle_lib):
    """Values fixed by the OCP E4M3 definition (bias 7, 3 mantissa bits, no
    infinities, S.1111.111 is NaN)."""
    known = {0x00: 0.0, 0x01: 2.0 ** -9, 0x07: 7 * 2.0 ** -9, 0x08: 2.0 ** -6, 0x38: 1.0, 0x3C: 1.5,
             0x40: 2.0, 0x7E: 448.0, 0xB8: -1.0, 0xFE: -448.0, 0x30: 0.5, 0x48: 4.0, 0x59: 18.0}
    for byte, v in known.items():
        assert oracle_lib.e4m3(byte) == v, hex(byte)
    assert math.isnan(oracle_lib.e4m3(0x7F)) and math.isnan(oracle_lib.e4m3(0xFF))


def test_e4m3_decode_matches_float32_construction(oracle_lib):
    """Every normal code equals the float32 with the same sign, exponent
    (rebiased 7 -> 127) and mantissa (shifted to the top); subnormals m * 2^-9."""
    import struct
    for byte in range(256):
        s, e, m = byte >> 7, (byte >> 3) & 15, byte & 7
        if e == 15 and m == 7:
            continue
        if e == 0:
            v = m * 2.0 ** -9
        else:
            v = struct.unpack("<f", struct.pack("<I", (e - 7 + 127) << 23 | m << 20))[0]
        assert oracle_lib.e4m3(byte) == (-v if s else v), hex(byte)


def test_e4m3_gemm_integer_exact_and_alpha_beta(oracle_lib):
    """Integer inputs (exact in E4M3) against int64 matmul, with alpha = 2,
    beta = -1: every product and partial sum is an exact integer."""
    rng = np.random.default_rng(8)
    M, N, K = 9, 7, 48
    Ai = rng.integers(-4, 5, (M, K))
    Bi = rng.integers(-4, 5, (N, K))
    Ci = rng.integers(-8, 9, (M, N)).astype(np.float32)
    A8, B8 = synth.to_e4m3_bits(Ai.astype(float)), synth.to_e4m3_bits(Bi.astype(float))
    got = oracle_lib.gemm_fp8(M, N, K, 2.0, A8, B8, -1.0, Ci)
    assert np.array_equal(got, 2.0 * (Ai @ Bi.T) - Ci)


def test_e4m3_rounding_of_inputs(oracle_lib):
    """The input generator rounds to nearest with ties to the even code and
    saturates at 448; every finite code round-trips."""
    assert list(synth.to_e4m3_bits(np.array([1.0625, 1.1875, 1000.0, -1.0, 2.0 ** -10]))) == [
        0x38, 0x3A, 0x7E, 0xB8, 0x00]
    codes = np.array([c for c in range(256) if (c & 0x7F) != 0x7F and c != 0x80], dtype=np.uint8)
    vals = np.array([oracle_lib.e4m3(c) for c in codes])
    assert np.array_equal(synth.to_e4m3_bits(vals), codes)


# --------------------------------------------------------------------------- MX block-scaled E4M3 GEMM

def test_e8m0_decode_known_values(oracle_lib):
    """Values fixed by the OCP MX E8M0 scale format: 2^(e - 127), 255 is NaN."""
    known = {127: 1.0, 128: 2.0, 126: 0.5, 0: 2.0 ** -127, 254: 2.0 ** 127, 137: 1024.0}
    for byte, v in known.items():
        assert oracle_lib.e8m0(byte) == v, byte
    assert math.isnan(oracle_lib.e8m0(255))


def _scales(seed, rows, kb, lo, hi):
    return synth.integers(seed, rows * kb, lo, hi).astype(np.uint8).reshape(rows, kb)


def test_mxfp8_unit_scales_are_the_e4m3_gemm(oracle_lib):
    """Every scale 2^0 (byte 127): exactly the unscaled E4M3 GEMM, with a
    ragged last block (K = 80: blocks of 32, 32, 16)."""
    M, N, K = 11, 6, 80
    A = synth.e4m3_uniform(41, (M, K))
    B = synth.e4m3_uniform(42, (N, K))
    C0 = synth.f32_uniform(43, (M, N))
    ones_a = np.full((M, 3), 127, np.uint8)
    ones_b = np.full((N, 3), 127, np.uint8)
    got = oracle_lib.gemm_mxfp8(M, N, K, 1.5, A, ones_a, B, ones_b, -0.5, C0)
    assert np.array_equal(got, oracle_lib.gemm_fp8(M, N, K, 1.5, A, B, -0.5, C0))


def test_mxfp8_is_the_sum_of_scaled_block_products(oracle_lib):
    """With integer E4M3 data and power-of-two scales every term is exact, so
    the block-scaled GEMM equals the sum over K blocks of
    diag(2^(SA-127)) (A_blk B_blk^T) diag(2^(SB-127)), each block product
    taken by the (separately pinned) unscaled E4M3 GEMM."""
    M, N, K = 9, 7, 112  # blocks of 32, 32, 32, 16
    kb = (K + 31) // 32
    A = synth.e4m3_integers(51, (M, K), -6, 6)
    B = synth.e4m3_integers(52, (N, K), -6, 6)
    SA = _scales(53, M, kb, 120, 134)
    SB = _scales(54, N, kb, 121, 133)
    got = oracle_lib.gemm_mxfp8(M, N, K, 1.0, A, SA, B, SB)
    want = np.zeros((M, N))
    for blk in range(kb):
        k0, k1 = 32 * blk, min(K, 32 * blk + 32)
        part = oracle_lib.gemm_fp8(M, N, k1 - k0, 1.0, np.ascontiguousarray(A[:, k0:k1]),
                                   np.ascontiguousarray(B[:, k0:k1]))
        sa = np.ldexp(1.0, SA[:, blk].astype(int) - 127)
        sb = np.ldexp(1.0, SB[:, blk].astype(int) - 127)
        want += sa[:, None] * part * sb[None, :]
    assert np.array_equal(got, want)
    # A scale one step up doubles exactly that block's share of its row.
    SA2 = SA.copy()
    SA2[4, 1] += 1
    got2 = oracle_lib.gemm_mxfp8(M, N, K, 1.0, A, SA2, B, SB)
    part1 = oracle_lib.gemm_fp8(M, N, 32, 1.0, np.ascontiguousarray(A[:, 32:64]), np.ascontiguousarray(B[:, 32:64]))
    delta = np.ldexp(1.0, int(SA[4, 1]) - 127) * part1[4] * np.ldexp(1.0, SB[:, 1].astype(int) - 127)
    assert np.array_equal(got2[4] - got[4], delta)
    assert np.array_equal(np.delete(got2, 4, axis=0), np.delete(got, 4, axis=0))


def test_mxfp8_nan_scale_poisons_only_its_row(oracle_lib):
    M, N, K = 5, 4, 64
    A = synth.e4m3_integers(61, (M, K), -3, 3)
    B = synth.e4m3_integers(62, (N, K), -3, 3)
    SA = np.full((M, 2), 127, np.uint8)
    SB = np.full((N, 2), 127, np.uint8)
    SA[2, 0] = 255
    got = oracle_lib.gemm_mxfp8(M, N, K, 1.0, A, SA, B, SB)
    assert np.isnan(got[2]).all() and np.isfinite(np.delete(got, 2, axis=0)).all()


# --------------------------------------------------------------------------- GRU, reset before the product

def _gru_rb_python(x, W, U, b, h0):
    """The reset-before equations in plain Python floats (tiny shapes)."""
    T, B, H = x.shape
    out = np.zeros((T, B, H))
    for s in range(B):
        h = [float(v) for v in h0[s]]
        for t in range(T):
            xt = x[t, s]
            gx = [sum(W[g, k] * xt[k] for k in range(H)) + b[g] for g in range(3 * H)]
            sig = lambda v: 1.0 / (1.0 + math.exp(-v))
            r = [sig(gx[j] + sum(U[j, k] * h[k] for k in range(H)) + b[3 * H + j]) for j in range(H)]
            z = [sig(gx[H + j] + sum(U[H + j, k] * h[k] for k in range(H)) + b[4 * H + j]) for j in range(H)]
            rh = [r[k] * h[k] for k in range(H)]
            n = [math.tanh(gx[2 * H + j] + sum(U[2 * H + j, k] * rh[k] for k in range(H)) + b[5 * H + j])
                 for j in range(H)]
            h = [(1 - z[j]) * n[j] + z[j] * h[j] for j in range(H)]
            out[t, s] = h
    return out


def test_gru_reset_before_matches_python_loops(oracle_lib):
    T, B, H = 3, 2, 4
    x, W, U, b, _ = synth.gru_operands(T, B, H, seed=41)
    h0 = synth.f32_uniform(42, (B, H))
    got = oracle_lib.gru_forward(x, W, U, b, h0, reset_before=True)
    ref = _gru_rb_python(f64(x), f64(W), f64(U), b.astype(np.float64), h0.astype(np.float64))
    assert np.max(np.abs(got - ref)) < 1e-12


def test_gru_reset_before_zero_weights_closed_form(oracle_lib):
    """W = U = 0: constant gates, n = tanh(b_in + b_hn), h_t = n (1 - z^t) + z^t h0."""
    T, B, H = 6, 3, 8
    x = synth.bf16_normal(43, (T, B, H))
    Z = np.zeros((3 * H, H), dtype=np.uint16)
    b = synth.f32_uniform(44, 6 * H, -0.5, 0.5).astype(np.float32)
    h0 = synth.f32_uniform(45, (B, H))
    got = oracle_lib.gru_forward(x, Z, Z, b, h0, reset_before=True)
    bb = b.astype(np.float64)
    z = 1 / (1 + np.exp(-(bb[H:2 * H] + bb[4 * H:5 * H])))
    n = np.tanh(bb[2 * H:3 * H] + bb[5 * H:])
    for t in range(T):
        assert np.max(np.abs(got[t] - (n * (1 - z ** (t + 1)) + z ** (t + 1) * h0))) < 1e-12


def test_gru_reset_before_saturated_reset_gate(oracle_lib):
    """r = 1 (b_ir = +30): U_n (r h) = r (U_n h), so both GRU forms agree; r = 0
    (b_ir = -30) with b_hn = 0: U_n no longer matters, and the form equals the
    reset-after one with the n rows of U zeroed."""
    T, B, H = 4, 3, 16
    x, W, U, b, _ = synth.gru_operands(T, B, H, seed=46)
    h0 = synth.f32_uniform(47, (B, H))
    b1 = b.copy()
    b1[:H] = 30.0
    a = oracle_lib.gru_forward(x, W, U, b1, h0, reset_before=True)
    c = oracle_lib.gru_forward(x, W, U, b1, h0)
    assert np.max(np.abs(a - c)) < 1e-10
    b0 = b.copy()
    b0[:H] = -30.0
    b0[5 * H:] = 0.0
    U0 = U.copy()
    U0[2 * H:] = 0
    a = oracle_lib.gru_forward(x, W, U, b0, h0, reset_before=True)
    c = oracle_lib.gru_forward(x, W, U0, b0, h0)
    assert np.max(np.abs(a - c)) < 1e-10


# ---- stacked GRU (layer l > 0 reads layer l - 1's states)

def _stack_operands(L, T, B, H, seed):
    x, _, _, _, _ = synth.gru_operands(T, B, H, seed=seed)
    W = np.stack([synth.gru_operands(1, 1, H, seed=seed + 10 * l + 1)[1] for l in range(L)])
    U = np.stack([synth.gru_operands(1, 1, H, seed=seed + 10 * l + 2)[2] for l in range(L)])
    b = np.stack([synth.gru_operands(1, 1, H, seed=seed + 10 * l + 3)[3] for l in range(L)])
    h0 = synth.f32_uniform(seed + 7, (L, B, H))
    return x, W, U, b, h0


@pytest.mark.parametrize("reset_before", [False, True])
def test_gru_stack_one_layer_is_the_single_layer_gru(oracle_lib, reset_before):
    T, B, H = 5, 3, 16
    x, W, U, b, h0 = _stack_operands(1, T, B, H, seed=50)
    got = oracle_lib.gru_stack(x, W, U, b, h0, reset_before=reset_before)
    ref = oracle_lib.gru_forward(x, W[0], U[0], b[0], h0[0], reset_before=reset_before)
    assert np.max(np.abs(got[0] - ref)) < 1e-12


def test_gru_stack_matches_torch_float64(oracle_lib):
    """torch.nn.GRU(num_layers=3) feeds each layer's output sequence to the
    next layer, with per-layer initial states: an independent implementation
    of the same stack (reset gate after the recurrent product)."""
    torch = pytest.importorskip("torch")
    L, T, B, H = 3, 6, 4, 20
    x, W, U, b, h0 = _stack_operands(L, T, B, H, seed=60)
    got = oracle_lib.gru_stack(x, W, U, b, h0)
    gru = torch.nn.GRU(H, H, num_layers=L, bias=True).double()
    with torch.no_grad():
        for l in range(L):
            getattr(gru, f"weight_ih_l{l}").copy_(torch.from_numpy(f64(W[l])))
            getattr(gru, f"weight_hh_l{l}").copy_(torch.from_numpy(f64(U[l])))
            getattr(gru, f"bias_ih_l{l}").copy_(torch.from_numpy(b[l, :3 * H].astype(np.float64)))
            getattr(gru, f"bias_hh_l{l}").copy_(torch.from_numpy(b[l, 3 * H:].astype(np.float64)))
        out, hT = gru(torch.from_numpy(f64(x)), torch.from_numpy(h0.astype(np.float64)))
    np.testing.assert_allclose(got[-1], out.numpy(), rtol=0, atol=1e-12)
    for l in range(L):
        np.testing.assert_allclose(got[l, -1], hT[l].numpy(), rtol=0, atol=1e-12)


def test_gru_stack_reset_before_matches_python_loops(oracle_lib):
    L, T, B, H = 2, 3, 2, 4
    x, W, U, b, h0 = _stack_operands(L, T, B, H, seed=70)
    got = oracle_lib.gru_stack(x, W, U, b, h0, reset_before=True)
    inp = f64(x)
    for l in range(L):
        ref = _gru_rb_python(inp, f64(W[l]), f64(U[l]), b[l].astype(np.float64),
                             h0[l].astype(np.float64))
        assert np.max(np.abs(got[l] - ref)) < 1e-12
        inp = ref


@pytest.mark.parametrize("reset_before", [False, True])
def test_gru_stack_lower_layers_ignore_upper_weights(oracle_lib, reset_before):
    """Layer l depends on layers 0..l only: changing the top layer's weights
    leaves every lower layer's states bit for bit unchanged, and changes the
    top layer's."""
    L, T, B, H = 3, 4, 2, 12
    x, W, U, b, h0 = _stack_operands(L, T, B, H, seed=80)
    a = oracle_lib.gru_stack(x, W, U, b, h0, reset_before=reset_before)
    W2, U2 = W.copy(), U.copy()
    W2[-1] = W[0]
    U2[-1] = U[1]
    c = oracle_lib.gru_stack(x, W2, U2, b, h0, reset_before=reset_before)
    assert np.array_equal(a[:-1], c[:-1])
    assert np.max(np.abs(a[-1] - c[-1])) > 1e-3


# ---- reset-before candidate: where the reset gate sits relative to U_n

def _masked_reset(b, H, mask):
    """b with b_ir = +30 on the units where mask is 1 and -30 elsewhere."""
    b = b.copy()
    b[:H] = np.where(mask, 30.0, -30.0).astype(np.float32)
    return b


def _masked_reset_case(seed, T=4, B=3, H=16):
    """Operands whose reset gate is a fixed 0/1 mask per unit: the r rows of W
    and U are zero, so r_j = sigmoid(b_ir_j + b_hr_j) with b_ir = +-30."""
    x, W, U, b, _ = synth.gru_operands(T, B, H, seed=seed)
    h0 = synth.f32_uniform(seed + 1, (B, H))
    W = W.copy()
    U = U.copy()
    W[:H] = 0
    U[:H] = 0
    mask = (np.arange(H) % 3 != 1)          # mixed pattern, both values present
    return x, W, U, b, h0, mask


def _masked_reset_expected(oracle_gru, x, W, U, b, h0, mask, H):
    """With r = mask, U_n (r * h) = (U_n with the columns of the masked-off
    units zeroed) h, which the reset-after form computes exactly when its own
    reset gate is 1 everywhere (b_ir = +30, r = 1 to 1e-13)."""
    Um = U.copy()
    Um[2 * H:, ~mask] = 0
    b1 = _masked_reset(b, H, np.ones(H, dtype=bool))
    return oracle_gru(x, W, Um, b1, h0)


def test_gru_reset_before_masked_reset_gate(oracle_lib):
    """A per-unit 0/1 reset gate selects COLUMNS of U_n in the reset-before
    form (r multiplies h before the product), never rows of the product:
    the slips r * (U_n h) + b_hn and r * (U_n h + b_hn) both fail here."""
    T, B, H = 4, 3, 16
    x, W, U, b, h0, mask = _masked_reset_case(90, T, B, H)
    got = oracle_lib.gru_forward(x, W, U, _masked_reset(b, H, mask), h0, reset_before=True)
    want = _masked_reset_expected(oracle_lib.gru_forward, x, W, U, b, h0, mask, H)
    assert np.max(np.abs(got - want)) < 1e-10
    # the row-selecting reading gives a clearly different answer on these inputs
    Ur = U.copy()
    Ur[2 * H:][~mask] = 0
    wrong = oracle_lib.gru_forward(x, W, Ur, _masked_reset(b, H, np.ones(H, dtype=bool)), h0)
    assert np.max(np.abs(wrong - want)) > 1e-3


@pytest.mark.parametrize("layers", [1, 2])
def test_gru_stack_reset_before_masked_reset_gate(oracle_lib, layers):
    """The same pin through the stacked oracle's reset-before branch: every
    layer's reset gate is a mask, so each layer equals the reset-after stack
    with its U_n columns zeroed."""
    T, B, H = 4, 3, 16
    x, W1, U1, b1, h01, mask = _masked_reset_case(91, T, B, H)
    Ws, Us, bs, bref, Uref = [], [], [], [], []
    for l in range(layers):
        _, Wl, Ul, bl, _, _ = _masked_reset_case(92 + 5 * l, T, B, H)
        Ws.append(Wl)
        Us.append(Ul)
        bs.append(_masked_reset(bl, H, mask))
        bref.append(_masked_reset(bl, H, np.ones(H, dtype=bool)))
        Um = Ul.copy()
        Um[2 * H:, ~mask] = 0
        Uref.append(Um)
    h0 = synth.f32_uniform(93, (layers, B, H))
    got = oracle_lib.gru_stack(x, np.stack(Ws), np.stack(Us), np.stack(bs), h0, reset_before=True)
    want = oracle_lib.gru_stack(x, np.stack(Ws), np.stack(Uref), np.stack(bref), h0)
    assert np.max(np.abs(got - want)) < 1e-10


def _build_mutant(tmp_path, replacements):
    """Compiles a copy of the oracle's C source with the given text edits (a
    planted mistake) into a library of its own under tmp_path."""
    import ctypes
    import os
    import subprocess
    import oracle
    src = open(os.path.join(os.path.dirname(oracle.__file__), "isam_oracle.c")).read()
    for old, new in replacements:
        assert src.count(old) == 1, old
        src = src.replace(old, new)
    c = tmp_path / "mutant.c"
    c.write_text(src)
    so = tmp_path / "libmutant.so"
    subprocess.run(["gcc", "-O1", "-std=c11", "-fPIC", "-shared", "-fopenmp", "-ffp-contract=off",
                    "-o", str(so), str(c), "-lm"], check=True)
    lib = ctypes.CDLL(str(so))
    P, i = ctypes.c_void_p, ctypes.c_int
    lib.oracle_gru_forward.argtypes = [i, i, i, P, P, P, P, P, P]
    lib.oracle_gru_forward_reset_before.argtypes = [i, i, i, P, P, P, P, P, P]
    lib.oracle_gru_stack.argtypes = [i, i, i, i, i, P, P, P, P, P, P]
    return lib


def _call_gru(fn, x, W, U, b, h0):
    import ctypes
    T, B, H = x.shape
    out = np.empty((T, B, H))
    arrs = [np.ascontiguousarray(a) for a in (x, W, U, b.astype(np.float32), h0.astype(np.float32))]
    ptr = [a.ctypes.data_as(ctypes.c_void_p) for a in arrs]
    assert fn(T, B, H, *ptr, out.ctypes.data_as(ctypes.c_void_p)) == 0
    return out


def test_masked_reset_pin_catches_a_planted_slip(tmp_path, oracle_lib):
    """Plants r * (U_n h) + b_hn into a copy of the reset-before oracle (CPU
    only).  The copy still passes the saturated-gate pins (r = 1, and r = 0
    with b_hn = 0), and the masked-reset pin fails it."""
    mut = _build_mutant(tmp_path, [
        ("rh[j] = r * h[j];", "rh[j] = r;"),
        ("for (int k = 0; k < H; ++k) an += bf(un[k]) * rh[k];",
         "for (int k = 0; k < H; ++k) an += bf(un[k]) * h[k];"),
        ("const double n = tanh(gx[2 * H + j] + an + (double)b[G + 2 * H + j]);",
         "const double n = tanh(gx[2 * H + j] + rh[j] * an + (double)b[G + 2 * H + j]);"),
    ])
    T, B, H = 4, 3, 16
    # r = 1 everywhere: the slip agrees with the true form
    x, W, U, b, _ = synth.gru_operands(T, B, H, seed=46)
    h0 = synth.f32_uniform(47, (B, H))
    b1 = b.copy()
    b1[:H] = 30.0
    np.testing.assert_allclose(_call_gru(mut.oracle_gru_forward_reset_before, x, W, U, b1, h0),
                               oracle_lib.gru_forward(x, W, U, b1, h0, reset_before=True), rtol=0, atol=1e-10)
    # the masked reset gate separates them
    x, W, U, b, h0, mask = _masked_reset_case(90, T, B, H)
    got = _call_gru(mut.oracle_gru_forward_reset_before, x, W, U, _masked_reset(b, H, mask), h0)
    want = _masked_reset_expected(oracle_lib.gru_forward, x, W, U, b, h0, mask, H)
    assert np.max(np.abs(got - want)) > 1e-3


def test_masked_reset_pin_catches_a_planted_slip_in_the_stack(tmp_path, oracle_lib):
    """The same slip planted in the stacked oracle's layer loop."""
    import ctypes
    mut = _build_mutant(tmp_path, [
        ("rh[j] = reset_before ? r * h[j] : h[j];", "rh[j] = h[j];"),
        ("const double n = reset_before ? tanh(gx[2 * H + j] + gh[2 * H + j])",
         "const double n = reset_before ? tanh(gx[2 * H + j] + r * (gh[2 * H + j] - (double)b[G + 2 * H + j])"
         " + (double)b[G + 2 * H + j])"),
    ])
    T, B, H = 4, 3, 16
    x, W, U, b, h0, mask = _masked_reset_case(91, T, B, H)
    bm = _masked_reset(b, H, mask)
    out = np.empty((1, T, B, H))
    arrs = [np.ascontiguousarray(a) for a in (x, W[None], U[None], bm[None], h0[None].astype(np.float32))]
    ptr = [a.ctypes.data_as(ctypes.c_void_p) for a in arrs]
    assert mut.oracle_gru_stack(1, T, B, H, 1, *ptr, out.ctypes.data_as(ctypes.c_void_p)) == 0
    want = _masked_reset_expected(oracle_lib.gru_forward, x, W, U, b, h0, mask, H)
    assert np.max(np.abs(out[0] - want)) > 1e-3
    good = oracle_lib.gru_stack(x, W[None], U[None], bm[None], h0[None], reset_before=True)
    assert np.max(np.abs(good[0] - want)) < 1e-10
