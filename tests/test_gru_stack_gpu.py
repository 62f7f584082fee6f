"""Stacked GRU (isam_gru_forward_stack) on the GPU against the fp64 oracle's
stacked GRU.  Tolerance: normalised max error over every layer's states
<= 1e-2 (the GRU bar); the oracle feeds each layer the unrounded states of
the layer below, the GPU their bf16 rounding (as for the recurrent product)."""
import ctypes

import numpy as np
import pytest

import oracle
from paper_1810_09958_gb300 import isam, synth
from gpu_util import Guarded, dev_bf16, nmax_err

pytestmark = pytest.mark.gpu
TOL = 1e-2


@pytest.fixture(scope="module", autouse=True)
def _lib():
    import torch
    from paper_1810_09958_gb300 import build
    build.build()
    isam.load()
    torch.cuda.set_device(0)
    yield
    isam.sync()


def f32dev(a):
    import torch
    return torch.from_numpy(np.ascontiguousarray(a, np.float32).reshape(-1)).cuda()


def run_stack(x, W, U, b, h0, reset_before=False):
    T, batch, H = x.shape
    L = W.shape[0]
    out = Guarded(L * T * batch * H)
    isam.gru_forward_stack(L, T, batch, H, dev_bf16(x), dev_bf16(W), dev_bf16(U), f32dev(b),
                           None if h0 is None else f32dev(h0), out.t, reset_before=reset_before)
    isam.sync()
    assert out.guards_intact(), "write outside h_out"
    return out.numpy().reshape(L, T, batch, H)


def run_single(x, W, U, b, h0, reset_before=False):
    T, batch, H = x.shape
    out = Guarded(T * batch * H)
    isam.gru_forward(T, batch, H, dev_bf16(x), dev_bf16(W), dev_bf16(U), f32dev(b),
                     None if h0 is None else f32dev(h0), out.t, reset_before=reset_before)
    isam.sync()
    return out.numpy().reshape(T, batch, H)


@pytest.mark.parametrize("reset_before", [False, True])
def test_gru_stack_two_layers_benchmark_shape(reset_before):
    """Two layers at hidden 1024, batch 32, 128 steps."""
    L, T, batch, H = 2, 128, 32, 1024
    x, W, U, b, h0 = synth.gru_stack_operands(L, T, batch, H, seed=synth.stream_seed(synth.BASE_SEED, 5))
    got = run_stack(x, W, U, b, h0, reset_before)
    ref = oracle.gru_stack(x, W, U, b, h0, reset_before=reset_before)
    for l in range(L):
        assert nmax_err(got[l], ref[l]) <= TOL, (l, nmax_err(got[l], ref[l]))


@pytest.mark.parametrize("L,T,batch,H,rb", [
    (2, 5, 3, 64, False), (3, 7, 17, 192, False), (2, 9, 32, 128, True), (3, 4, 5, 896, False),
    (2, 3, 2, 448, True), (4, 6, 32, 256, False), (2, 16, 8, 1024, True), (2, 3, 31, 320, False),
    (3, 5, 9, 768, True), (2, 1, 1, 512, False)])
def test_gru_stack_shapes(L, T, batch, H, rb):
    x, W, U, b, h0 = synth.gru_stack_operands(L, T, batch, H, seed=L * 7919 + T * 131 + batch * 17 + H)
    got = run_stack(x, W, U, b, h0, rb)
    ref = oracle.gru_stack(x, W, U, b, h0, reset_before=rb)
    for l in range(L):
        assert nmax_err(got[l], ref[l]) <= TOL, (l, nmax_err(got[l], ref[l]))


def test_gru_stack_null_h0_means_zeros():
    L, T, batch, H = 2, 4, 6, 256
    x, W, U, b, _ = synth.gru_stack_operands(L, T, batch, H, seed=91)
    got = run_stack(x, W, U, b, None)
    ref = oracle.gru_stack(x, W, U, b, None)
    assert nmax_err(got, ref) <= TOL


@pytest.mark.parametrize("reset_before", [False, True])
def test_gru_stack_first_layer_is_the_single_layer_call(reset_before):
    """Layer 0 runs the same kernel as isam_gru_forward, the next layer's
    product going to separate accumulator columns: its states are identical
    bit for bit; one layer is isam_gru_forward itself."""
    L, T, batch, H = 3, 10, 32, 512
    x, W, U, b, h0 = synth.gru_stack_operands(L, T, batch, H, seed=92)
    got = run_stack(x, W, U, b, h0, reset_before)
    one = run_single(x, W[0], U[0], b[0], h0[0], reset_before)
    assert np.array_equal(got[0], one)
    got1 = run_stack(x, W[:1], U[:1], b[:1], h0[:1], reset_before)
    assert np.array_equal(got1[0], one)


def test_gru_stack_repeat_calls_identical():
    L, T, batch, H = 3, 12, 32, 1024
    x, W, U, b, h0 = synth.gru_stack_operands(L, T, batch, H, seed=93)
    a = run_stack(x, W, U, b, h0)
    c = run_stack(x, W, U, b, h0)
    assert np.array_equal(a, c)


def test_gru_stack_unsupported_shapes_rejected():
    import torch
    z = torch.zeros(1 << 22, dtype=torch.bfloat16, device="cuda")
    f = torch.zeros(1 << 22, dtype=torch.float32, device="cuda")
    lib = isam.load()
    p = lambda t: ctypes.c_void_p(t.data_ptr())
    assert lib.isam_gru_forward_stack(2, 1, 1, 80, 0, p(z), p(z), p(z), p(f), None, p(f)) == \
        isam.ISAM_ERR_UNSUPPORTED
    assert lib.isam_gru_forward_stack(2, 1, 257, 128, 0, p(z), p(z), p(z), p(f), None, p(f)) == \
        isam.ISAM_ERR_UNSUPPORTED
    o = torch.zeros(832, dtype=torch.float32, device="cuda")
    assert lib.isam_gru_forward_stack(1, 1, 1, 832, 0, p(z), p(z), p(z), p(f), None, p(o)) == isam.ISAM_OK
    isam.sync()


@pytest.mark.parametrize("L", [2, 3])
def test_gru_stack_pairs_and_per_layer_chain_agree(L, monkeypatch):
    """At hidden 1024 (reset gate after the product) layers run in pairs in one
    kernel; ISAM_NO_WAVE=1 selects the per-layer chain.  Both match the
    oracle, and layer 0 is the same computation in both (identical)."""
    T, batch, H = 20, 32, 1024
    x, W, U, b, h0 = synth.gru_stack_operands(L, T, batch, H, seed=94 + L)
    pairs = run_stack(x, W, U, b, h0)
    monkeypatch.setenv("ISAM_NO_WAVE", "1")
    chain = run_stack(x, W, U, b, h0)
    ref = oracle.gru_stack(x, W, U, b, h0)
    for l in range(L):
        assert nmax_err(pairs[l], ref[l]) <= TOL
        assert nmax_err(chain[l], ref[l]) <= TOL
    assert np.array_equal(pairs[0], chain[0])


def test_gru_stack_pair_kernel_missing_participant_times_out_cleanly():
    """One CTA of the two-layer kernel never signals the round counter (a flag
    nothing sets): every bounded wait runs out, the kernel returns, isam_sync
    reports ISAM_ERR_TIMEOUT, and a correct call works afterwards."""
    import os
    import subprocess
    import sys
    import textwrap
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    code = textwrap.dedent(f"""
        import os, sys, numpy as np, torch
        sys.path.insert(0, {root!r}); sys.path.insert(0, {os.path.join(root, 'tests')!r})
        from paper_1810_09958_gb300 import isam, synth
        import oracle
        from gpu_util import dev_bf16, nmax_err
        torch.cuda.set_device(0)
        L, T, batch, H = 2, 4, 8, 256
        x, W, U, b, h0 = synth.gru_stack_operands(L, T, batch, H, seed=97)
        args = [dev_bf16(x), dev_bf16(W), dev_bf16(U), torch.from_numpy(b.reshape(-1)).cuda(), None]
        out = torch.zeros(L * T * batch * H, device="cuda")
        os.environ["ISAM_DEBUG_GRU_SKIP_CTA"] = "0"
        isam.gru_forward_stack(L, T, batch, H, *args, out)
        rc = isam.load().isam_sync()
        assert rc == isam.ISAM_ERR_TIMEOUT, rc
        del os.environ["ISAM_DEBUG_GRU_SKIP_CTA"]
        isam.gru_forward_stack(L, T, batch, H, *args, out)
        isam.sync()
        ref = oracle.gru_stack(x, W, U, b, None)
        assert nmax_err(out.cpu().numpy().reshape(L, T, batch, H), ref) <= 1e-2
        print("TIMEOUT_OK")
    """)
    env = dict(os.environ, ISAM_WAIT_TIMEOUT_MS="300")
    r = subprocess.run([sys.executable, "-c", code], env=env, capture_output=True, text=True, timeout=300)
    assert r.returncode == 0 and "TIMEOUT_OK" in r.stdout, r.stdout + r.stderr


@pytest.mark.parametrize("L,T,batch,H,rb", [(2, 5, 48, 1024, False), (3, 4, 130, 512, True), (2, 3, 256, 256, False)])
def test_gru_stack_wide_batch(L, T, batch, H, rb):
    """Batches wider than 32: each layer projects the bf16 states below with
    the GEMM and runs its recurrence in chunks of padded rows."""
    x, W, U, b, h0 = synth.gru_stack_operands(L, T, batch, H, seed=L * 13 + batch + H)
    got = run_stack(x, W, U, b, h0, rb)
    ref = oracle.gru_stack(x, W, U, b, h0, reset_before=rb)
    for l in range(L):
        assert nmax_err(got[l], ref[l]) <= TOL, (l, nmax_err(got[l], ref[l]))


@pytest.mark.parametrize("L,T,batch,H,rb", [(2, 4, 9, 96, False), (3, 3, 32, 352, True),
                                            # per-layer chain with uneven K ranges: 2 splits
                                            # (480, 832) and 4 splits (960, 992)
                                            (2, 3, 7, 480, False), (2, 3, 5, 832, True),
                                            (2, 3, 6, 960, False), (2, 2, 32, 992, True)])
def test_gru_stack_hidden_odd_multiple_of_32(L, T, batch, H, rb):
    x, W, U, b, h0 = synth.gru_stack_operands(L, T, batch, H, seed=L + T + batch + H)
    got = run_stack(x, W, U, b, h0, rb)
    ref = oracle.gru_stack(x, W, U, b, h0, reset_before=rb)
    for l in range(L):
        assert nmax_err(got[l], ref[l]) <= TOL, (l, nmax_err(got[l], ref[l]))
