"""GRU forward parity on the GPU through the C ABI (isam_gru_forward and
isam_gru_forward_reset_before) against the fp64 oracle.  Tolerance: normalised
max error over every step's hidden state (all of h_out) <= 1e-2."""
import os
import subprocess
import sys
import textwrap

import numpy as np
import pytest

import oracle
from paper_1810_09958_gb300 import isam, synth
from gpu_util import Guarded, dev_bf16, nmax_err

pytestmark = pytest.mark.gpu
TOL = 1e-2
ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module", autouse=True)
def _lib():
    import torch
    from paper_1810_09958_gb300 import build
    build.build()
    isam.load()
    torch.cuda.set_device(0)
    yield
    isam.sync()


def run_gru(x, W, U, b, h0, reset_before=False):
    import torch
    T, batch, H = x.shape
    out = Guarded(T * batch * H)
    h0d = None if h0 is None else torch.from_numpy(np.ascontiguousarray(h0, np.float32)).cuda()
    isam.gru_forward(T, batch, H, dev_bf16(x), dev_bf16(W), dev_bf16(U),
                     torch.from_numpy(b).cuda(), h0d, out.t, reset_before=reset_before)
    isam.sync()
    assert out.guards_intact(), "write outside h_out"
    return out.numpy().reshape(T, batch, H)


def test_gru_benchmark_shape_full_oracle():
    """hidden = input = 1024, batch 32, 128 steps, h0 = 0 (the GRU benchmark shape)."""
    T, batch, H = 128, 32, 1024
    x, W, U, b, h0 = synth.gru_operands(T, batch, H, seed=synth.stream_seed(synth.BASE_SEED, 3))
    got = run_gru(x, W, U, b, h0)
    ref = oracle.gru_forward(x, W, U, b, h0)
    err = nmax_err(got, ref)
    assert err <= TOL, err
    assert nmax_err(got[-1], ref[-1]) <= TOL


@pytest.mark.parametrize("T,batch,H", [(1, 1, 64), (5, 3, 64), (7, 17, 192), (9, 32, 128),
                                       (20, 32, 512), (3, 31, 320), (16, 8, 1024),
                                       # 3, 7 and 13 K atoms per CTA (4, 2 and 1 K splits)
                                       (6, 32, 768), (4, 5, 896), (3, 2, 832)])
def test_gru_shapes_with_initial_state(T, batch, H):
    x, W, U, b, _ = synth.gru_operands(T, batch, H, seed=T * 1000 + batch * 10 + H)
    h0 = synth.f32_uniform(T + batch + H, (batch, H))
    got = run_gru(x, W, U, b, h0)
    ref = oracle.gru_forward(x, W, U, b, h0)
    assert nmax_err(got, ref) <= TOL


def test_gru_null_h0_means_zeros():
    T, batch, H = 4, 5, 128
    x, W, U, b, _ = synth.gru_operands(T, batch, H, seed=44)
    got = run_gru(x, W, U, b, None)
    ref = oracle.gru_forward(x, W, U, b, None)
    assert nmax_err(got, ref) <= TOL


def test_gru_zero_weights_closed_form():
    """W = U = 0: h_t = n + z**t (h0 - n) with r, z, n set by the biases alone."""
    T, batch, H = 6, 4, 128
    zero = np.zeros((3 * H, H), np.uint16)
    x = synth.bf16_normal(1, (T, batch, H))
    b = synth.f32_uniform(2, (6 * H,), -2.0, 2.0)
    h0 = synth.f32_uniform(3, (batch, H))
    got = run_gru(x, zero, zero, b, h0)
    ref = oracle.gru_forward(x, zero, zero, b, h0)
    assert np.max(np.abs(got - ref)) <= 1e-5


def test_gru_saturated_update_gate_keeps_state():
    T, batch, H = 10, 6, 256
    x, W, U, b, _ = synth.gru_operands(T, batch, H, seed=7)
    b = b.copy()
    b[H:2 * H] = 30.0
    h0 = synth.f32_uniform(8, (batch, H))
    got = run_gru(x, W, U, b, h0)
    assert np.max(np.abs(got - h0[None])) <= 1e-6


def test_gru_repeat_calls_identical():
    T, batch, H = 12, 32, 256
    x, W, U, b, h0 = synth.gru_operands(T, batch, H, seed=12)
    a = run_gru(x, W, U, b, h0)
    c = run_gru(x, W, U, b, h0)
    assert np.array_equal(a, c)


def test_gru_unsupported_shapes_rejected():
    import torch
    z = torch.zeros(4096, dtype=torch.bfloat16, device="cuda")
    f = torch.zeros(4096, dtype=torch.float32, device="cuda")
    lib = isam.load()
    import ctypes
    p = lambda t: ctypes.c_void_p(t.data_ptr())
    assert lib.isam_gru_forward(1, 257, 64, p(z), p(z), p(z), p(f), None, p(f)) == isam.ISAM_ERR_UNSUPPORTED
    assert lib.isam_gru_forward(1, 1, 80, p(z), p(z), p(z), p(f), None, p(f)) == isam.ISAM_ERR_UNSUPPORTED
    assert lib.isam_gru_forward(1, 1, 1056, p(z), p(z), p(z), p(f), None, p(f)) == isam.ISAM_ERR_UNSUPPORTED


@pytest.mark.parametrize("reset_before", [False, True])
def test_gru_missing_participant_times_out_cleanly(reset_before):
    """One CTA never signals the step counter (a flag nothing sets): every
    bounded wait runs out, the kernel returns, isam_sync reports
    ISAM_ERR_TIMEOUT, and the context stays usable for a correct call."""
    rb = bool(reset_before)
    code = textwrap.dedent(f"""
        import sys, numpy as np, torch
        sys.path.insert(0, {ROOT!r}); sys.path.insert(0, {os.path.join(ROOT, 'tests')!r})
        import os
        from paper_1810_09958_gb300 import isam, synth
        import oracle
        from gpu_util import dev_bf16, nmax_err
        torch.cuda.set_device(0)
        T, batch, H = 4, 8, 128
        x, W, U, b, h0 = synth.gru_operands(T, batch, H, seed=3)
        args = [dev_bf16(x), dev_bf16(W), dev_bf16(U), torch.from_numpy(b).cuda(), None]
        out = torch.zeros(T * batch * H, device="cuda")
        os.environ["ISAM_DEBUG_GRU_SKIP_CTA"] = "0"
        isam.gru_forward(T, batch, H, *args, out, reset_before={rb!r})
        rc = isam.load().isam_sync()
        assert rc == isam.ISAM_ERR_TIMEOUT, rc
        del os.environ["ISAM_DEBUG_GRU_SKIP_CTA"]
        isam.gru_forward(T, batch, H, *args, out, reset_before={rb!r})
        isam.sync()
        ref = oracle.gru_forward(x, W, U, b, None, reset_before={rb!r})
        assert nmax_err(out.cpu().numpy().reshape(T, batch, H), ref) <= 1e-2
        print("TIMEOUT_OK")
    """)
    env = dict(os.environ, ISAM_WAIT_TIMEOUT_MS="300")
    r = subprocess.run([sys.executable, "-c", code], env=env, capture_output=True, text=True,
                       timeout=300)
    assert r.returncode == 0 and "TIMEOUT_OK" in r.stdout, r.stdout + r.stderr


# ---- reset gate applied before the candidate's recurrent product:
# n = tanh(W_n x + b_in + U_n (r * h_{t-1}) + b_hn).

def test_gru_reset_before_benchmark_shape_full_oracle():
    T, batch, H = 128, 32, 1024
    x, W, U, b, h0 = synth.gru_operands(T, batch, H, seed=synth.stream_seed(synth.BASE_SEED, 3))
    got = run_gru(x, W, U, b, h0, reset_before=True)
    ref = oracle.gru_forward(x, W, U, b, h0, reset_before=True)
    assert nmax_err(got, ref) <= TOL
    assert nmax_err(got[-1], ref[-1]) <= TOL
    # the two forms really differ at this shape (the test would not see a mix-up otherwise)
    other = oracle.gru_forward(x, W, U, b, h0)
    assert nmax_err(other, ref) > 10 * TOL


@pytest.mark.parametrize("T,batch,H", [(1, 1, 64), (5, 3, 64), (7, 17, 192), (9, 32, 128),
                                       (3, 31, 320), (16, 8, 1024), (6, 32, 768), (4, 5, 896),
                                       (3, 2, 832)])
def test_gru_reset_before_shapes_with_initial_state(T, batch, H):
    x, W, U, b, _ = synth.gru_operands(T, batch, H, seed=T * 1000 + batch * 10 + H + 1)
    h0 = synth.f32_uniform(T + batch + H + 1, (batch, H))
    got = run_gru(x, W, U, b, h0, reset_before=True)
    ref = oracle.gru_forward(x, W, U, b, h0, reset_before=True)
    assert nmax_err(got, ref) <= TOL


def test_gru_reset_before_open_reset_gate_matches_reset_after():
    """A reset gate saturated at 1 (b_ir = 30) makes both forms the same
    function; the two kernels then see the same bf16 operands and the same
    summation order, so their outputs agree to fp32 rounding of the gates."""
    T, batch, H = 8, 32, 512
    x, W, U, b, h0 = synth.gru_operands(T, batch, H, seed=21)
    b = b.copy()
    b[:H] = 30.0
    rb = run_gru(x, W, U, b, h0, reset_before=True)
    ra = run_gru(x, W, U, b, h0)
    assert nmax_err(rb, ra) <= 1e-4
    assert nmax_err(rb, oracle.gru_forward(x, W, U, b, h0, reset_before=True)) <= TOL


def test_gru_reset_before_zero_weights_closed_form():
    T, batch, H = 6, 4, 128
    zero = np.zeros((3 * H, H), np.uint16)
    x = synth.bf16_normal(1, (T, batch, H))
    b = synth.f32_uniform(2, (6 * H,), -2.0, 2.0)
    h0 = synth.f32_uniform(3, (batch, H))
    got = run_gru(x, zero, zero, b, h0, reset_before=True)
    ref = oracle.gru_forward(x, zero, zero, b, h0, reset_before=True)
    assert np.max(np.abs(got - ref)) <= 1e-5


def test_gru_reset_before_repeat_and_interleaved_calls_identical():
    """Both forms share the exchange workspace: interleaving them changes nothing."""
    T, batch, H = 12, 32, 256
    x, W, U, b, h0 = synth.gru_operands(T, batch, H, seed=13)
    a = run_gru(x, W, U, b, h0, reset_before=True)
    m = run_gru(x, W, U, b, h0)
    c = run_gru(x, W, U, b, h0, reset_before=True)
    d = run_gru(x, W, U, b, h0)
    assert np.array_equal(a, c) and np.array_equal(m, d)


# ---- batches wider than 32: the recurrence runs with a padded batch of 64 or
# 128 (the MMA's N), in chunks of that many rows.

@pytest.mark.parametrize("T,batch,H,rb", [(6, 33, 1024, False), (5, 64, 1024, False), (4, 100, 1024, True),
                                          (6, 128, 1024, False), (3, 200, 1024, False), (3, 256, 1024, True),
                                          (5, 96, 896, False), (4, 70, 448, True), (3, 129, 256, False),
                                          (2, 256, 64, False)])
def test_gru_wide_batch(T, batch, H, rb):
    x, W, U, b, _ = synth.gru_operands(T, batch, H, seed=T * 31 + batch * 7 + H)
    h0 = synth.f32_uniform(batch + H + 5, (batch, H))
    got = run_gru(x, W, U, b, h0, reset_before=rb)
    ref = oracle.gru_forward(x, W, U, b, h0, reset_before=rb)
    assert nmax_err(got, ref) <= TOL, nmax_err(got, ref)


def test_gru_wide_batch_rows_independent_of_chunking():
    """Rows are independent sequences: the first 32 rows of a batch of 160
    (chunks of 128 padded rows) match the same rows run as a batch of 32.
    Not bit for bit: the input projection's GEMM takes another tile plan at
    M = 960 than at M = 192 (another fp32 summation order), and bf16 rounding
    of h carries that over the steps; rows mixing across the chunk would show
    errors of order 1."""
    T, batch, H = 6, 160, 1024
    x, W, U, b, _ = synth.gru_operands(T, batch, H, seed=515)
    h0 = synth.f32_uniform(516, (batch, H))
    wide = run_gru(x, W, U, b, h0)
    narrow = run_gru(np.ascontiguousarray(x[:, :32]), W, U, b, np.ascontiguousarray(h0[:32]))
    assert nmax_err(wide[:, :32], narrow) <= 1e-3
    ref = oracle.gru_forward(x, W, U, b, h0)
    assert nmax_err(wide, ref) <= TOL


# ---- hidden a multiple of 32 but not of 64: one CTA per group of 32 units,
# the last 64-wide K atom half outside the matrix (zero-filled on both sides).

@pytest.mark.parametrize("T,batch,H,rb", [(5, 3, 32, False), (4, 17, 96, False), (6, 32, 160, True),
                                          (3, 8, 480, False), (4, 50, 224, False), (3, 5, 800, True),
                                          (3, 6, 864, False), (3, 7, 992, True), (3, 40, 928, False)])
def test_gru_hidden_odd_multiple_of_32(T, batch, H, rb):
    x, W, U, b, _ = synth.gru_operands(T, batch, H, seed=T * 17 + batch + H * 3)
    h0 = synth.f32_uniform(H + batch, (batch, H))
    got = run_gru(x, W, U, b, h0, reset_before=rb)
    ref = oracle.gru_forward(x, W, U, b, h0, reset_before=rb)
    assert nmax_err(got, ref) <= TOL, nmax_err(got, ref)


# ---- K ranges that end past the matrix: hidden 480 and 576-896 (other than
# multiples of 128) run 2 K splits, 928-992 run 4, each CTA holding
# ceil(atoms / splits) whole atoms; the last CTA's range ends in zeros read by
# the tensor maps (at 960 with 4 splits its last atom lies wholly outside U).

@pytest.mark.parametrize("T,batch,H,rb", [(3, 5, 960, False), (3, 32, 960, True), (4, 9, 576, False),
                                          (3, 70, 960, False), (4, 12, 704, True)])
def test_gru_uneven_k_splits(T, batch, H, rb):
    x, W, U, b, _ = synth.gru_operands(T, batch, H, seed=T * 29 + batch + H * 5)
    h0 = synth.f32_uniform(H + batch + 1, (batch, H))
    got = run_gru(x, W, U, b, h0, reset_before=rb)
    ref = oracle.gru_forward(x, W, U, b, h0, reset_before=rb)
    assert nmax_err(got, ref) <= TOL, nmax_err(got, ref)


def test_gru_plan_on_the_device_matches_the_host_plan():
    """isam_gru_plan_info (this device's limits) equals isam_gru_plan_for with
    the limits the host-side planner tests assume (152 SMs, 232448 bytes)."""
    import torch
    sms = torch.cuda.get_device_properties(0).multi_processor_count
    for (layers, batch, H, rb) in [(1, 32, 1024, False), (2, 32, 1024, False), (2, 32, 1024, True),
                                   (1, 200, 960, False), (3, 8, 864, True)]:
        assert isam.gru_plan(layers, batch, H, rb) == isam.gru_plan(layers, batch, H, rb, num_sms=sms,
                                                                     smem_optin=232448)
