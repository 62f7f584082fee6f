"""The allocation-free GRU entry point (isam_gru_forward_noalloc), called
through the C ABI and checked against the regular isam_gru_forward on the same
inputs, on two calls in a row.

It exists for callers that cannot let a library call cudaMalloc (device
memory reserved up front by a framework's caching allocator, or a request path
where an allocation's device-wide synchronisation is not allowed); its
workspaces live in a fixed 8 MiB array inside the library.  This file is
collected last so that a run stopping at the first failure has already run
every other test."""
import ctypes

import numpy as np
import pytest

from paper_1810_09958_gb300 import isam, synth
from gpu_util import Guarded, dev_bf16, nmax_err

pytestmark = pytest.mark.gpu
TOL = 1e-2   # the GRU parity tolerance used by the other GRU tests


def _ptr(t):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


@pytest.fixture(scope="module")
def lib():
    import torch
    from paper_1810_09958_gb300 import build
    build.build()
    torch.cuda.set_device(0)
    return isam.load()


@pytest.mark.parametrize("T,batch,H", [(128, 32, 1024), (9, 5, 192), (6, 7, 96), (5, 32, 960)])
def test_noalloc_matches_regular_entry_twice(lib, T, batch, H):
    import torch
    x, W, U, b, _ = synth.gru_operands(T, batch, H, seed=9000 + H)
    h0 = synth.f32_uniform(9001 + H, (batch, H))
    xd, Wd, Ud = dev_bf16(x), dev_bf16(W), dev_bf16(U)
    bd = torch.from_numpy(b).cuda()
    h0d = torch.from_numpy(h0).cuda()
    stream = ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)

    ref = Guarded(T * batch * H)
    assert lib.isam_set_stream(stream) == 0
    assert lib.isam_gru_forward(T, batch, H, _ptr(xd), _ptr(Wd), _ptr(Ud), _ptr(bd), _ptr(h0d),
                                _ptr(ref.t)) == 0
    assert lib.isam_sync() == 0
    want = ref.numpy()

    for call in range(2):
        out = Guarded(T * batch * H, init=np.full(T * batch * H, np.nan, np.float32))
        rc = lib.isam_gru_forward_noalloc(T, batch, H, _ptr(xd), _ptr(Wd), _ptr(Ud), _ptr(bd),
                                          _ptr(h0d), _ptr(out.t))
        assert rc == 0, lib.isam_last_error_string()
        torch.cuda.synchronize()
        assert out.guards_intact()
        got = out.numpy()
        assert np.isfinite(got).all()
        assert nmax_err(got, want) <= TOL, (call, nmax_err(got, want))


def test_noalloc_rejects_sizes_beyond_limits(lib):
    import torch
    z = torch.zeros(1 << 16, dtype=torch.bfloat16, device="cuda")
    f = torch.zeros(1 << 16, dtype=torch.float32, device="cuda")
    p = _ptr
    assert lib.isam_gru_forward_noalloc(4, 33, 64, p(z), p(z), p(z), p(f), None, p(f)) == 2
    assert b"batch <= 32" in lib.isam_last_error_string()
    assert lib.isam_gru_forward_noalloc(4, 8, 2048, p(z), p(z), p(z), p(f), None, p(f)) == 2
    assert lib.isam_gru_forward_noalloc(0, 8, 64, p(z), p(z), p(z), p(f), None, p(f)) == 1
