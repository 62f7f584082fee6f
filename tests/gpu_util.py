"""Helpers for the GPU parity tests (inputs from synth, expected values from
the oracle; nothing here computes the method)."""
import numpy as np

from paper_1810_09958_gb300 import synth

GUARD = 64          # fp32 canary words on each side of an output (16-byte aligned)
CANARY = -7.0e30


def nmax_err(got, ref):
    """max |got - ref| / (max |ref| + 1e-6), the parity metric."""
    got = np.asarray(got, dtype=np.float64)
    ref = np.asarray(ref, dtype=np.float64)
    return float(np.max(np.abs(got - ref)) / (np.max(np.abs(ref)) + 1e-6))


def dev_bf16(bits):
    import torch
    return synth.as_torch_bf16(bits).cuda()


class Guarded:
    """An fp32 device output with canary words on both sides."""

    def __init__(self, n, init=None):
        import torch
        self.n = n
        self.buf = torch.full((n + 2 * GUARD,), CANARY, dtype=torch.float32, device="cuda")
        self.t = self.buf[GUARD:GUARD + n]
        if init is not None:
            self.t.copy_(torch.from_numpy(np.ascontiguousarray(init, dtype=np.float32).reshape(-1)))

    def numpy(self):
        return self.t.cpu().numpy()

    def guards_intact(self):
        b = self.buf.cpu().numpy()
        return bool(np.all(b[:GUARD] == CANARY) and np.all(b[GUARD + self.n:] == CANARY))
