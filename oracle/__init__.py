"""fp64 CPU oracle for the GEMM / GRU / separable-depthwise hot path.

TEST INFRASTRUCTURE ONLY: imported by ``tests/``, ``__graft_entry__.smoke()``
and the CPU-baseline leg of ``bench.py``; never by the library.  It shares no
code with the CUDA path.  The arithmetic is in ``isam_oracle.c`` (plain C,
double precision, OpenMP over independent outputs); this module builds it
with gcc and wraps it with ctypes.

Every function takes bf16 operands as numpy uint16 bit patterns (see
``paper_1810_09958_gb300.synth``), fp32 operands as float32 arrays, and returns
float64 arrays.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "isam_oracle.c")
_LIB_PATH = os.path.join(_HERE, "liboracle.so")
_lock = threading.Lock()
_lib = None


def build(force: bool = False) -> str:
    """Compiles isam_oracle.c into liboracle.so (gcc, OpenMP, no FP contraction)."""
    if (not force and os.path.exists(_LIB_PATH)
            and os.path.getmtime(_LIB_PATH) >= os.path.getmtime(_SRC)):
        return _LIB_PATH
    tmp = _LIB_PATH + f".tmp{os.getpid()}"
    cmd = ["gcc", "-O2", "-std=c11", "-fPIC", "-shared", "-fopenmp",
           "-ffp-contract=off", "-fno-fast-math", "-o", tmp, _SRC, "-lm"]
    subprocess.run(cmd, check=True)
    os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def _load():
    global _lib
    with _lock:
        if _lib is None:
            build()
            lib = ctypes.CDLL(_LIB_PATH)
            P = ctypes.c_void_p
            i, d = ctypes.c_int, ctypes.c_double
            lib.oracle_gemm_rows.argtypes = [i, i, i, i, i, d, P, P, d, P, i, P, P]
            lib.oracle_gemm.argtypes = [i, i, i, i, i, d, P, P, d, P, P]
            lib.oracle_gru_forward.argtypes = [i, i, i, P, P, P, P, P, P]
            lib.oracle_dwsep.argtypes = [i, i, i, i, i, P, P, P, P]
            lib.oracle_num_threads.argtypes = []
            lib.oracle_e4m3.argtypes = [ctypes.c_uint8]
            lib.oracle_e4m3.restype = ctypes.c_double
            lib.oracle_gemm_fp8.argtypes = [i, i, i, d, P, P, d, P, P]
            lib.oracle_gru_forward_reset_before.argtypes = [i, i, i, P, P, P, P, P, P]
            lib.oracle_gru_forward_reset_before.restype = ctypes.c_int
            lib.oracle_gemm_fp8.restype = ctypes.c_int
            lib.oracle_e8m0.argtypes = [ctypes.c_uint8]
            lib.oracle_e8m0.restype = ctypes.c_double
            lib.oracle_gemm_mxfp8.argtypes = [i, i, i, d, P, P, P, P, d, P, P]
            lib.oracle_gemm_mxfp8.restype = ctypes.c_int
            lib.oracle_gru_stack.argtypes = [i, i, i, i, i, P, P, P, P, P, P]
            lib.oracle_gru_stack.restype = ctypes.c_int
            for f in (lib.oracle_gemm_rows, lib.oracle_gemm, lib.oracle_gru_forward,
                      lib.oracle_dwsep, lib.oracle_num_threads):
                f.restype = ctypes.c_int
            _lib = lib
    return _lib


def _p(a):
    return None if a is None else a.ctypes.data_as(ctypes.c_void_p)


def _u16(a):
    a = np.ascontiguousarray(a)
    assert a.dtype == np.uint16, a.dtype
    return a


def num_threads() -> int:
    return _load().oracle_num_threads()


def gemm(M, N, K, transA, transB, alpha, A, B, beta=0.0, C_in=None, rows=None):
    """C = alpha * opA @ opB + beta * C_in (Listing 1); returns [len(rows) or M, N] float64."""
    A, B = _u16(A), _u16(B)
    assert A.size == M * K and B.size == K * N
    if C_in is not None:
        C_in = np.ascontiguousarray(C_in, dtype=np.float32)
        assert C_in.size == M * N
    if rows is not None:
        rows = np.ascontiguousarray(rows, dtype=np.int32)
        out = np.empty((rows.size, N), dtype=np.float64)
        rc = _load().oracle_gemm_rows(M, N, K, int(transA), int(transB), float(alpha),
                                      _p(A), _p(B), float(beta), _p(C_in), rows.size,
                                      _p(rows), _p(out))
    else:
        out = np.empty((M, N), dtype=np.float64)
        rc = _load().oracle_gemm(M, N, K, int(transA), int(transB), float(alpha),
                                 _p(A), _p(B), float(beta), _p(C_in), _p(out))
    if rc != 0:
        raise ValueError("oracle_gemm: invalid argument")
    return out


def e4m3(byte: int) -> float:
    """The value of one E4M3 byte (exact)."""
    return _load().oracle_e4m3(int(byte) & 0xFF)


def gemm_fp8(M, N, K, alpha, A, B, beta=0.0, C_in=None):
    """C = alpha * A @ B^T + beta * C_in, A (M x K) and B (N x K) E4M3 bytes;
    returns [M, N] float64."""
    A = np.ascontiguousarray(A, dtype=np.uint8)
    B = np.ascontiguousarray(B, dtype=np.uint8)
    assert A.size == M * K and B.size == N * K
    if C_in is not None:
        C_in = np.ascontiguousarray(C_in, dtype=np.float32)
        assert C_in.size == M * N
    out = np.empty((M, N), dtype=np.float64)
    rc = _load().oracle_gemm_fp8(M, N, K, float(alpha), _p(A), _p(B), float(beta), _p(C_in), _p(out))
    if rc != 0:
        raise ValueError("oracle_gemm_fp8: invalid argument")
    return out


def e8m0(byte: int) -> float:
    """The value of one OCP MX E8M0 scale byte: 2^(byte - 127), NaN for 255."""
    return _load().oracle_e8m0(int(byte) & 0xFF)


def gemm_mxfp8(M, N, K, alpha, A, SA, B, SB, beta=0.0, C_in=None):
    """Block-scaled E4M3 GEMM (OCP MX): C = alpha * (SA . A) @ (SB . B)^T +
    beta * C_in, A (M x K) and B (N x K) E4M3 bytes, SA (M x ceil(K/32)) and
    SB (N x ceil(K/32)) E8M0 scale bytes, one per 32 consecutive K elements;
    returns [M, N] float64."""
    kb = (K + 31) // 32
    A = np.ascontiguousarray(A, dtype=np.uint8)
    B = np.ascontiguousarray(B, dtype=np.uint8)
    SA = np.ascontiguousarray(SA, dtype=np.uint8)
    SB = np.ascontiguousarray(SB, dtype=np.uint8)
    assert A.size == M * K and B.size == N * K and SA.size == M * kb and SB.size == N * kb
    if C_in is not None:
        C_in = np.ascontiguousarray(C_in, dtype=np.float32)
        assert C_in.size == M * N
    out = np.empty((M, N), dtype=np.float64)
    rc = _load().oracle_gemm_mxfp8(M, N, K, float(alpha), _p(A), _p(SA), _p(B), _p(SB), float(beta), _p(C_in),
                                   _p(out))
    if rc != 0:
        raise ValueError("oracle_gemm_mxfp8: invalid argument")
    return out


def gru_forward(x, W, U, b, h0=None, reset_before=False):
    """All T hidden states [T, batch, H] float64 of the GRU (r, z, n gate order);
    reset_before: the candidate's recurrent input is U_n (r * h)."""
    x, W, U = _u16(x), _u16(W), _u16(U)
    T, batch, H = x.shape
    assert W.shape == (3 * H, H) and U.shape == (3 * H, H)
    b = np.ascontiguousarray(b, dtype=np.float32)
    assert b.size == 6 * H
    if h0 is not None:
        h0 = np.ascontiguousarray(h0, dtype=np.float32)
        assert h0.size == batch * H
    out = np.empty((T, batch, H), dtype=np.float64)
    fn = _load().oracle_gru_forward_reset_before if reset_before else _load().oracle_gru_forward
    rc = fn(T, batch, H, _p(x), _p(W), _p(U), _p(b), _p(h0), _p(out))
    if rc != 0:
        raise ValueError("oracle_gru_forward: invalid argument")
    return out


def gru_stack(x, W, U, b, h0=None, reset_before=False):
    """Every layer's hidden states [layers, T, batch, H] float64 of a stacked
    GRU: W, U [layers, 3H, H] bf16 bits, b [layers, 6H], h0 [layers, batch, H]
    or None; layer l > 0 reads layer l - 1's states unrounded."""
    x, W, U = _u16(x), _u16(W), _u16(U)
    T, batch, H = x.shape
    L = W.shape[0]
    assert W.shape == (L, 3 * H, H) and U.shape == (L, 3 * H, H)
    b = np.ascontiguousarray(b, dtype=np.float32)
    assert b.size == L * 6 * H
    if h0 is not None:
        h0 = np.ascontiguousarray(h0, dtype=np.float32)
        assert h0.size == L * batch * H
    out = np.empty((L, T, batch, H), dtype=np.float64)
    rc = _load().oracle_gru_stack(L, T, batch, H, int(bool(reset_before)), _p(x), _p(W), _p(U),
                                  _p(b), _p(h0), _p(out))
    if rc != 0:
        raise ValueError("oracle_gru_stack: invalid argument")
    return out


def dwsep(x, dw, pw):
    """Separable depthwise conv (3x3, stride 1, pad 1, then 1x1); NHWC float64."""
    x, dw, pw = _u16(x), _u16(dw), _u16(pw)
    N, H, W, Cin = x.shape
    Cout = pw.shape[1]
    assert dw.shape == (3, 3, Cin) and pw.shape == (Cin, Cout)
    out = np.empty((N, H, W, Cout), dtype=np.float64)
    rc = _load().oracle_dwsep(N, H, W, Cin, Cout, _p(x), _p(dw), _p(pw), _p(out))
    if rc != 0:
        raise ValueError("oracle_dwsep: invalid argument")
    return out
