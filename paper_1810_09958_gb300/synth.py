"""Seeded synthetic inputs shared by the CUDA path's tests/bench and the oracle.

This module only draws numbers: it holds none of the method's arithmetic and
imports nothing else from this package, so the oracle and the CUDA path can
both take their inputs from it without sharing any compute code.

Generator: SplitMix64 (Steele, Lea and Flood, "Fast splittable pseudorandom
number generators", OOPSLA 2014), used counter-based: draw ``i`` of stream
``seed`` is ``mix64(seed + (i + 1) * 0x9E3779B97F4A7C15)``.  Uniforms take the
top 53 bits; normals use the Box-Muller transform on consecutive draw pairs.
Values are rounded to float32 (numpy, round-to-nearest-even) and then to
bfloat16 with round-to-nearest-even on the float32 bit pattern.  Every array
that feeds the library as bf16 is returned as its uint16 bit pattern, so both
sides see bit-identical operands.

Workload recipes (shapes and distributions of the paper's benchmarks, Section
5.1: DeepBench-sized GEMMs, a GRU over 128 steps, and the separable depthwise
convolution of Listing 3) live at the bottom of this file.
"""
from __future__ import annotations

import math

import numpy as np

_GOLDEN = np.uint64(0x9E3779B97F4A7C15)
_M1 = np.uint64(0xBF58476D1CE4E5B9)
_M2 = np.uint64(0x94D049BB133111EB)
_CHUNK = 1 << 22


def _mix64(z: np.ndarray) -> np.ndarray:
    z = (z ^ (z >> np.uint64(30))) * _M1
    z = (z ^ (z >> np.uint64(27))) * _M2
    return z ^ (z >> np.uint64(31))


def splitmix64(seed: int, start: int, count: int) -> np.ndarray:
    """Draws ``start .. start+count-1`` of the SplitMix64 stream ``seed``."""
    with np.errstate(over="ignore"):
        idx = np.arange(start + 1, start + count + 1, dtype=np.uint64)
        return _mix64(np.uint64(seed & 0xFFFFFFFFFFFFFFFF) + idx * _GOLDEN)


def uniform(seed: int, n: int, lo: float = -1.0, hi: float = 1.0) -> np.ndarray:
    """``n`` float64 values uniform in [lo, hi)."""
    out = np.empty(n, dtype=np.float64)
    for s in range(0, n, _CHUNK):
        c = min(_CHUNK, n - s)
        z = splitmix64(seed, s, c)
        u = (z >> np.uint64(11)).astype(np.float64) * (1.0 / 9007199254740992.0)
        out[s:s + c] = lo + (hi - lo) * u
    return out


def uniform_at(seed: int, idx: np.ndarray, lo: float = -1.0, hi: float = 1.0) -> np.ndarray:
    """Draws number ``idx`` (any shape of non-negative indices) of the stream, as
    uniform() would return them: uniform(seed, n)[idx] == uniform_at(seed, idx)."""
    with np.errstate(over="ignore"):
        z = _mix64(np.uint64(seed & 0xFFFFFFFFFFFFFFFF) +
                   (np.asarray(idx, dtype=np.uint64) + np.uint64(1)) * _GOLDEN)
    u = (z >> np.uint64(11)).astype(np.float64) * (1.0 / 9007199254740992.0)
    return lo + (hi - lo) * u


def normal(seed: int, n: int, mean: float = 0.0, std: float = 1.0) -> np.ndarray:
    """``n`` float64 normal values; value i uses draws 2i and 2i+1 (Box-Muller)."""
    out = np.empty(n, dtype=np.float64)
    for s in range(0, n, _CHUNK):
        c = min(_CHUNK, n - s)
        z = splitmix64(seed, 2 * s, 2 * c)
        u = ((z >> np.uint64(11)).astype(np.float64) + 1.0) * (1.0 / 9007199254740992.0)
        u1, u2 = u[0::2], u[1::2]
        out[s:s + c] = mean + std * np.sqrt(-2.0 * np.log(u1)) * np.cos(2.0 * math.pi * u2)
    return out


def integers(seed: int, n: int, lo: int, hi: int) -> np.ndarray:
    """``n`` float64 integer values uniform in [lo, hi] (inclusive)."""
    z = splitmix64(seed, 0, n)
    span = np.uint64(hi - lo + 1)
    return (z % span).astype(np.int64).astype(np.float64) + lo


def to_bf16_bits(x: np.ndarray) -> np.ndarray:
    """Rounds finite values to bfloat16 (round-to-nearest-even); uint16 bits."""
    f = np.ascontiguousarray(x, dtype=np.float32)
    b = f.view(np.uint32)
    b = (b + (np.uint32(0x7FFF) + ((b >> np.uint32(16)) & np.uint32(1)))) >> np.uint32(16)
    return b.astype(np.uint16).reshape(np.shape(x))


def bf16_bits_to_f32(bits: np.ndarray) -> np.ndarray:
    """Widens bf16 bit patterns to float32 exactly."""
    return (bits.astype(np.uint32) << np.uint32(16)).view(np.float32)


def bf16_bits_to_f64(bits: np.ndarray) -> np.ndarray:
    """Widens bf16 bit patterns to float64 exactly."""
    return bf16_bits_to_f32(bits).astype(np.float64)


def as_torch_bf16(bits: np.ndarray):
    """A CPU torch bfloat16 tensor with exactly these bit patterns."""
    import torch
    return torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).view(torch.bfloat16)


def _e4m3_positive():
    """Positive finite OCP E4M3 codes 0x00..0x7E and their values, ascending."""
    codes = np.arange(0x7F, dtype=np.int64)
    e, m = codes >> 3, codes & 7
    vals = np.where(e == 0, (m / 8.0) * 2.0 ** -6, (1.0 + m / 8.0) * np.exp2(e - 7.0))
    return codes, vals


_E4M3_CODES, _E4M3_VALS = _e4m3_positive()


def to_e4m3_bits(x: np.ndarray) -> np.ndarray:
    """float -> E4M3 byte, round to nearest (ties to the even code), magnitudes
    above 448 saturate to 448; zero encodes as 0x00."""
    x = np.asarray(x, dtype=np.float64)
    a = np.minimum(np.abs(x), 448.0)
    idx = np.clip(np.searchsorted(_E4M3_VALS, a), 1, len(_E4M3_VALS) - 1)
    lo, hi = _E4M3_VALS[idx - 1], _E4M3_VALS[idx]
    up = (a - lo > hi - a) | ((a - lo == hi - a) & ((_E4M3_CODES[idx] & 1) == 0))
    code = np.where(up, _E4M3_CODES[idx], _E4M3_CODES[idx - 1])
    code = np.where(a == 0.0, 0, code)
    sign = np.where(np.signbit(x) & (code != 0), 0x80, 0)
    return (code | sign).astype(np.uint8)


def e4m3_bits_to_f64(bits: np.ndarray) -> np.ndarray:
    """E4M3 byte -> float64 (finite codes; NaN codes give NaN)."""
    b = np.asarray(bits, dtype=np.int64)
    mag = _E4M3_VALS[np.minimum(b & 0x7F, 0x7E)]
    mag = np.where((b & 0x7F) == 0x7F, np.nan, mag)
    return np.where(b & 0x80, -mag, mag)


def e4m3_uniform(seed: int, shape, lo=-1.0, hi=1.0) -> np.ndarray:
    n = int(np.prod(shape))
    return to_e4m3_bits(uniform(seed, n, lo, hi)).reshape(shape)


def e4m3_integers(seed: int, shape, lo: int, hi: int) -> np.ndarray:
    """Integers in [lo, hi] (exact in E4M3 for |v| <= 16)."""
    n = int(np.prod(shape))
    return to_e4m3_bits(integers(seed, n, lo, hi).astype(np.float64)).reshape(shape)


def e4m3_uniform_torch(seed: int, n: int, device, lo=-1.0, hi=1.0):
    """Device-side E4M3 bytes (torch.uint8) for large benchmark operands: the
    same uniform stream rounded to E4M3 by torch's float8 cast."""
    import torch
    f = f32_uniform_torch(seed, n, device, lo, hi)
    return f.to(torch.float8_e4m3fn).view(torch.uint8)


def bf16_uniform(seed: int, shape, lo=-1.0, hi=1.0) -> np.ndarray:
    n = int(np.prod(shape))
    return to_bf16_bits(uniform(seed, n, lo, hi)).reshape(shape)


def bf16_normal(seed: int, shape, mean=0.0, std=1.0) -> np.ndarray:
    n = int(np.prod(shape))
    return to_bf16_bits(normal(seed, n, mean, std)).reshape(shape)


def bf16_integers(seed: int, shape, lo: int, hi: int) -> np.ndarray:
    n = int(np.prod(shape))
    return to_bf16_bits(integers(seed, n, lo, hi)).reshape(shape)


def f32_uniform(seed: int, shape, lo=-1.0, hi=1.0) -> np.ndarray:
    n = int(np.prod(shape))
    return uniform(seed, n, lo, hi).astype(np.float32).reshape(shape)


# ---------------------------------------------------------------------------
# The same streams drawn with torch on any device (used to fill large device
# buffers quickly).  Uniform draws are bit-identical to uniform()/bf16_uniform();
# torch int64 arithmetic wraps modulo 2**64 like the uint64 version and right
# shifts are made logical by masking.
# ---------------------------------------------------------------------------
def _to_i64(v: int) -> int:
    v &= 0xFFFFFFFFFFFFFFFF
    return v - (1 << 64) if v >= (1 << 63) else v


def _lshr(z, s: int):
    return (z >> s) & ((1 << (64 - s)) - 1)


def splitmix64_torch(seed: int, start: int, count: int, device):
    import torch
    idx = torch.arange(start + 1, start + count + 1, dtype=torch.int64, device=device)
    z = idx * _to_i64(0x9E3779B97F4A7C15) + _to_i64(seed)
    z = (z ^ _lshr(z, 30)) * _to_i64(0xBF58476D1CE4E5B9)
    z = (z ^ _lshr(z, 27)) * _to_i64(0x94D049BB133111EB)
    return z ^ _lshr(z, 31)


def bf16_uniform_torch(seed: int, n: int, device, lo=-1.0, hi=1.0):
    """A flat torch.bfloat16 tensor on ``device``, bit-identical to bf16_uniform(seed, (n,))."""
    import torch
    out = torch.empty(n, dtype=torch.bfloat16, device=device)
    chunk = 1 << 24
    for s in range(0, n, chunk):
        c = min(chunk, n - s)
        z = splitmix64_torch(seed, s, c, device)
        u = _lshr(z, 11).to(torch.float64) * (1.0 / 9007199254740992.0)
        out[s:s + c] = (lo + (hi - lo) * u).to(torch.float32).to(torch.bfloat16)
    return out


def bf16_normal_torch(seed: int, n: int, device, mean=0.0, std=1.0):
    """A flat torch.bfloat16 tensor of normal draws from the same stream as
    normal() (device libm may differ from numpy's in the last bit of a rare
    value; used only to fill timing inputs)."""
    import torch
    out = torch.empty(n, dtype=torch.bfloat16, device=device)
    chunk = 1 << 23
    for s in range(0, n, chunk):
        c = min(chunk, n - s)
        z = splitmix64_torch(seed, 2 * s, 2 * c, device)
        u = (_lshr(z, 11).to(torch.float64) + 1.0) * (1.0 / 9007199254740992.0)
        v = mean + std * torch.sqrt(-2.0 * torch.log(u[0::2])) * torch.cos(2.0 * math.pi * u[1::2])
        out[s:s + c] = v.to(torch.float32).to(torch.bfloat16)
    return out


def f32_uniform_torch(seed: int, n: int, device, lo=-1.0, hi=1.0):
    import torch
    out = torch.empty(n, dtype=torch.float32, device=device)
    chunk = 1 << 24
    for s in range(0, n, chunk):
        c = min(chunk, n - s)
        z = splitmix64_torch(seed, s, c, device)
        u = _lshr(z, 11).to(torch.float64) * (1.0 / 9007199254740992.0)
        out[s:s + c] = (lo + (hi - lo) * u).to(torch.float32)
    return out


# ---------------------------------------------------------------------------
# Workload recipes.  Seeds are derived from a base seed and a stream tag so that
# the operands of one problem never share a stream.
# ---------------------------------------------------------------------------
BASE_SEED = 0x15A4


def stream_seed(base: int, *tags: int) -> int:
    h = np.uint64(base & 0xFFFFFFFFFFFFFFFF)
    with np.errstate(over="ignore"):
        for t in tags:
            h = _mix64(h + np.uint64(t & 0xFFFFFFFFFFFFFFFF) * _GOLDEN + _GOLDEN)
    return int(h)


def gemm_operands(M, N, K, transA, transB, seed, dist="uniform", beta_c=False):
    """A, B as bf16 bits in their stored layouts, plus fp32 C_in when beta_c.

    dist 'uniform': U[-1,1]; 'normal002': N(0,1)*0.02; 'int4': integers in
    [-4,4] (every product and partial sum exact in fp32 for K <= 2**19).
    A is stored M x K (transA=0) or K x M (transA=1); B is stored K x N
    (transB=0) or N x K (transB=1); row-major, packed.
    """
    a_shape = (K, M) if transA else (M, K)
    b_shape = (N, K) if transB else (K, N)
    sa, sb, sc = (stream_seed(seed, i) for i in (1, 2, 3))
    if dist == "uniform":
        A, B = bf16_uniform(sa, a_shape), bf16_uniform(sb, b_shape)
    elif dist == "normal002":
        A, B = bf16_normal(sa, a_shape, 0.0, 0.02), bf16_normal(sb, b_shape, 0.0, 0.02)
    elif dist == "int4":
        A, B = bf16_integers(sa, a_shape, -4, 4), bf16_integers(sb, b_shape, -4, 4)
    else:
        raise ValueError(dist)
    C = None
    if beta_c:
        if dist == "int4":
            C = integers(sc, M * N, -8, 8).astype(np.float32).reshape(M, N)
        else:
            C = f32_uniform(sc, (M, N))
    return A, B, C


def gru_operands(T, batch, hidden, seed):
    """x [T,batch,hidden] bf16 N(0,1); W,U [3H,H] bf16 U(+-1/sqrt(H));
    b fp32 [6H] U(+-0.1) (input biases then recurrent biases); h0 zeros."""
    H = hidden
    s = 1.0 / math.sqrt(H)
    x = bf16_normal(stream_seed(seed, 11), (T, batch, H))
    W = bf16_uniform(stream_seed(seed, 12), (3 * H, H), -s, s)
    U = bf16_uniform(stream_seed(seed, 13), (3 * H, H), -s, s)
    b = f32_uniform(stream_seed(seed, 14), (6 * H,), -0.1, 0.1)
    h0 = np.zeros((batch, H), dtype=np.float32)
    return x, W, U, b, h0


def gru_stack_operands(layers, T, batch, hidden, seed):
    """A stack of GRU layers drawn as gru_operands per layer: x [T,batch,H];
    W, U [layers,3H,H]; b [layers,6H]; h0 [layers,batch,H] U(-1,1)."""
    x = gru_operands(T, batch, hidden, seed)[0]
    per = [gru_operands(1, 1, hidden, stream_seed(seed, 100 + l)) for l in range(layers)]
    W = np.stack([q[1] for q in per])
    U = np.stack([q[2] for q in per])
    b = np.stack([q[3] for q in per])
    h0 = f32_uniform(stream_seed(seed, 99), (layers, batch, hidden))
    return x, W, U, b, h0


def dwsep_operands(N, H, W, Cin, Cout, seed):
    """x NHWC bf16 N(0,1); dw_w [3,3,Cin] bf16 U(+-1/3) (fan-in 9);
    pw_w [Cin,Cout] bf16 U(+-1/sqrt(Cin))."""
    x = bf16_normal(stream_seed(seed, 21), (N, H, W, Cin))
    dw = bf16_uniform(stream_seed(seed, 22), (3, 3, Cin), -1.0 / 3.0, 1.0 / 3.0)
    s = 1.0 / math.sqrt(Cin)
    pw = bf16_uniform(stream_seed(seed, 23), (Cin, Cout), -s, s)
    return x, dw, pw
