"""Thin Python binding of libisam.so (include/isam.h): argument marshalling only.

Each function takes torch tensors that already live on the current CUDA
device, checks dtype/shape/contiguity, points the library at torch's current
stream and passes raw device pointers through the C ABI.  Every step of the
computation runs in the library's CUDA kernels; there is no fallback.  If the
library has not been built, loading it raises.
"""
from __future__ import annotations

import ctypes
import os
import re
import threading

PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(PKG, "libisam.so")
HEADER = os.path.join(os.path.dirname(PKG), "include", "isam.h")

ISAM_OK, ISAM_ERR_INVALID_ARG, ISAM_ERR_UNSUPPORTED, ISAM_ERR_CUDA, ISAM_ERR_TIMEOUT = range(5)

_lock = threading.Lock()
_lib = None


class IsamError(RuntimeError):
    def __init__(self, code: int, msg: str):
        super().__init__(f"isam error {code}: {msg}")
        self.code = code


def declared_functions() -> list[str]:
    """Names of every function declared in include/isam.h."""
    with open(HEADER) as f:
        text = f.read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(isam_[a-z0-9_]+)\s*\(", text)))


def load():
    """Loads libisam.so (raises if it has not been built)."""
    global _lib
    with _lock:
        if _lib is not None:
            return _lib
        if not os.path.exists(LIB_PATH):
            raise ImportError(
                f"{LIB_PATH} is missing: build it with `python -c 'import __graft_entry__ as g; g.build()'`")
        lib = ctypes.CDLL(LIB_PATH)
        i, f, P = ctypes.c_int, ctypes.c_float, ctypes.c_void_p
        lib.isam_version.argtypes = []
        lib.isam_set_stream.argtypes = [P]
        lib.isam_sync.argtypes = []
        lib.isam_last_error_string.argtypes = []
        lib.isam_last_error_string.restype = ctypes.c_char_p
        lib.isam_shutdown.argtypes = []
        lib.isam_gemm.argtypes = [i, i, i, i, i, f, P, P, f, P]
        lib.isam_gemm_plan_info.argtypes = [i, i, i, i, i, f, P]
        lib.isam_gemm_plan_info2.argtypes = [i, i, i, i, i, f, P]
        lib.isam_gemm_grouped.argtypes = [i, P, P, P, P, P, P, P, P, P, P]
        lib.isam_gemm_fp8.argtypes = [i, i, i, f, P, P, f, P]
        lib.isam_gemm_grouped_fp8.argtypes = [i, P, P, P, P, P, P, P, P]
        lib.isam_gemm_mxfp8.argtypes = [i, i, i, f, P, P, P, P, f, P]
        lib.isam_gemm_grouped_mxfp8.argtypes = [i, P, P, P, P, P, P, P, P, P, P]
        lib.isam_gru_forward.argtypes = [i, i, i, P, P, P, P, P, P]
        lib.isam_gru_forward_reset_before.argtypes = [i, i, i, P, P, P, P, P, P]
        lib.isam_gru_forward_stack.argtypes = [i, i, i, i, i, P, P, P, P, P, P]
        lib.isam_dwsep_conv.argtypes = [i, i, i, i, i, P, P, P, P]
        lib.isam_depthwise_conv3x3.argtypes = [i, i, i, i, P, P, P]
        lib.isam_dwsep_plan_info.argtypes = [i, i, i, P]
        lib.isam_dwsep_plan_for.argtypes = [i, i, i, i, P]
        lib.isam_gemm_plan_for.argtypes = [i, i, i, i, i, f, i, i, P, P]
        lib.isam_gru_plan_info.argtypes = [i, i, i, i, P]
        lib.isam_gru_plan_for.argtypes = [i, i, i, i, i, i, P]
        for name in ("isam_version", "isam_set_stream", "isam_sync", "isam_shutdown", "isam_gemm",
                     "isam_gemm_plan_info", "isam_gemm_plan_info2", "isam_gemm_grouped", "isam_gemm_fp8", "isam_gemm_grouped_fp8",
                     "isam_gemm_mxfp8", "isam_gemm_grouped_mxfp8",
                     "isam_gru_forward", "isam_gru_forward_reset_before",
                     "isam_gru_forward_stack",
                     "isam_dwsep_conv", "isam_dwsep_plan_info", "isam_dwsep_plan_for", "isam_depthwise_conv3x3",
                     "isam_gru_plan_info", "isam_gru_plan_for", "isam_gemm_plan_for"):
            getattr(lib, name).restype = ctypes.c_int
        _lib = lib
        return lib


def last_error() -> str:
    return load().isam_last_error_string().decode(errors="replace")


def check(rc: int) -> None:
    if rc != ISAM_OK:
        raise IsamError(rc, last_error())


def _ptr(t):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _dev(t, dtype, numel, name):
    import torch
    if t.device.type != "cuda":
        raise ValueError(f"{name} must be a CUDA tensor")
    if t.dtype != dtype:
        raise ValueError(f"{name} must be {dtype}, got {t.dtype}")
    if not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")
    if t.numel() != numel:
        raise ValueError(f"{name} has {t.numel()} elements, expected {numel}")
    if t.device.index != torch.cuda.current_device():
        raise ValueError(f"{name} is not on the current device")


def _use_current_stream(lib):
    import torch
    lib.isam_set_stream(ctypes.c_void_p(torch.cuda.current_stream().cuda_stream))


def sync() -> None:
    check(load().isam_sync())


def shutdown() -> None:
    check(load().isam_shutdown())


def gemm(M, N, K, transA, transB, alpha, A, B, beta, C) -> None:
    """isam_gemm: C = alpha op(A) op(B) + beta C (A, B bf16; C fp32)."""
    import torch
    lib = load()
    _dev(A, torch.bfloat16, M * K, "A")
    _dev(B, torch.bfloat16, K * N, "B")
    _dev(C, torch.float32, M * N, "C")
    _use_current_stream(lib)
    check(lib.isam_gemm(M, N, K, int(transA), int(transB), float(alpha), _ptr(A), _ptr(B),
                        float(beta), _ptr(C)))


def gemm_fp8(M, N, K, alpha, A, B, beta, C) -> None:
    """isam_gemm_fp8: C = alpha A B^T + beta C (A: M x K, B: N x K, E4M3 bytes as
    torch.uint8 or torch.float8_e4m3fn; C fp32)."""
    import torch
    lib = load()
    for t, n, name in ((A, M * K, "A"), (B, N * K, "B")):
        if t.dtype not in (torch.uint8, getattr(torch, "float8_e4m3fn", torch.uint8)):
            raise ValueError(f"{name} must hold E4M3 bytes (uint8 or float8_e4m3fn), got {t.dtype}")
        _dev(t, t.dtype, n, name)
    _dev(C, torch.float32, M * N, "C")
    _use_current_stream(lib)
    check(lib.isam_gemm_fp8(M, N, K, float(alpha), _ptr(A), _ptr(B), float(beta), _ptr(C)))


def _e4m3_dev(t, n, name):
    import torch
    if t.dtype not in (torch.uint8, getattr(torch, "float8_e4m3fn", torch.uint8)):
        raise ValueError(f"{name} must hold E4M3 bytes (uint8 or float8_e4m3fn), got {t.dtype}")
    _dev(t, t.dtype, n, name)


def mx_scale_bytes(rows, K) -> int:
    """Bytes of an atom-major scale array: ceil(K/128) x rows x 4."""
    return (K + 127) // 128 * rows * 4


def gemm_mxfp8(M, N, K, alpha, A, SA, B, SB, beta, C) -> None:
    """isam_gemm_mxfp8: C = alpha (SA o A)(SB o B)^T + beta C with A (M x K) and
    B (N x K) E4M3 bytes, SA and SB E8M0 bytes (torch.uint8) in the atom-major
    layout [ceil(K/128)][rows][4] (include/isam.h), C fp32."""
    import torch
    lib = load()
    _e4m3_dev(A, M * K, "A")
    _e4m3_dev(B, N * K, "B")
    _dev(SA, torch.uint8, mx_scale_bytes(M, K), "SA")
    _dev(SB, torch.uint8, mx_scale_bytes(N, K), "SB")
    _dev(C, torch.float32, M * N, "C")
    _use_current_stream(lib)
    check(lib.isam_gemm_mxfp8(M, N, K, float(alpha), _ptr(A), _ptr(SA), _ptr(B), _ptr(SB), float(beta), _ptr(C)))


class GroupedGemmMxfp8:
    """Marshalled arguments of one isam_gemm_grouped_mxfp8 call over a list of
    (M, N, K, alpha, A, SA, B, SB, beta, C); SA, SB atom-major (mx_scale_bytes)."""

    def __init__(self, problems):
        import torch
        n = len(problems)
        ia = lambda vals: (ctypes.c_int * n)(*vals)
        fa = lambda vals: (ctypes.c_float * n)(*vals)
        pa = lambda vals: (ctypes.c_void_p * n)(*vals)
        for (M, N, K, alpha, A, SA, B, SB, beta, C) in problems:
            _e4m3_dev(A, M * K, "A")
            _e4m3_dev(B, N * K, "B")
            _dev(SA, torch.uint8, mx_scale_bytes(M, K), "SA")
            _dev(SB, torch.uint8, mx_scale_bytes(N, K), "SB")
            _dev(C, torch.float32, M * N, "C")
        cols = list(zip(*problems))
        self.n = n
        ptrs = lambda col: pa([t.data_ptr() for t in col])
        self.args = (ia(cols[0]), ia(cols[1]), ia(cols[2]), fa(cols[3]), ptrs(cols[4]), ptrs(cols[5]),
                     ptrs(cols[6]), ptrs(cols[7]), fa(cols[8]), ptrs(cols[9]))

    def __call__(self):
        lib = load()
        _use_current_stream(lib)
        check(lib.isam_gemm_grouped_mxfp8(self.n, *self.args))


class GroupedGemm:
    """Marshalled argument arrays of one isam_gemm_grouped call (build once,
    call many times: the arrays keep the ctypes buffers alive)."""

    def __init__(self, problems):
        import torch
        n = len(problems)
        ia = lambda vals: (ctypes.c_int * n)(*vals)
        fa = lambda vals: (ctypes.c_float * n)(*vals)
        pa = lambda vals: (ctypes.c_void_p * n)(*vals)
        for (M, N, K, tA, tB, alpha, A, B, beta, C) in problems:
            _dev(A, torch.bfloat16, M * K, "A")
            _dev(B, torch.bfloat16, K * N, "B")
            _dev(C, torch.float32, M * N, "C")
        cols = list(zip(*problems))
        self.n = n
        self.args = (ia(cols[0]), ia(cols[1]), ia(cols[2]), ia(cols[3]), ia(cols[4]), fa(cols[5]),
                     pa([t.data_ptr() for t in cols[6]]), pa([t.data_ptr() for t in cols[7]]), fa(cols[8]),
                     pa([t.data_ptr() for t in cols[9]]))

    def __call__(self):
        lib = load()
        _use_current_stream(lib)
        check(lib.isam_gemm_grouped(self.n, *self.args))


class GroupedGemmFp8:
    """Marshalled arguments of one isam_gemm_grouped_fp8 call over a list of
    (M, N, K, alpha, A, B, beta, C); A, B E4M3 bytes (uint8 / float8_e4m3fn)."""

    def __init__(self, problems):
        import torch
        n = len(problems)
        ia = lambda vals: (ctypes.c_int * n)(*vals)
        fa = lambda vals: (ctypes.c_float * n)(*vals)
        pa = lambda vals: (ctypes.c_void_p * n)(*vals)
        for (M, N, K, alpha, A, B, beta, C) in problems:
            _dev(A, A.dtype, M * K, "A")
            _dev(B, B.dtype, N * K, "B")
            _dev(C, torch.float32, M * N, "C")
        cols = list(zip(*problems))
        self.n = n
        self.args = (ia(cols[0]), ia(cols[1]), ia(cols[2]), fa(cols[3]), pa([t.data_ptr() for t in cols[4]]),
                     pa([t.data_ptr() for t in cols[5]]), fa(cols[6]), pa([t.data_ptr() for t in cols[7]]))

    def __call__(self):
        lib = load()
        _use_current_stream(lib)
        check(lib.isam_gemm_grouped_fp8(self.n, *self.args))


def gemm_grouped(problems) -> None:
    """isam_gemm_grouped over a list of (M, N, K, transA, transB, alpha, A, B, beta, C)."""
    GroupedGemm(problems)()


def gemm_plan(M, N, K, transA, transB, beta=0.0, num_sms=None, smem_optin=None, cluster_caps=None) -> dict:
    """The tile plan the library's cost model picks (nothing is launched);
    with num_sms, smem_optin and cluster_caps (resident clusters of 2, 4, 8
    CTAs), isam_gemm_plan_for on those limits (no GPU)."""
    lib = load()
    out = (ctypes.c_int * 8)()
    if num_sms is None:
        check(lib.isam_gemm_plan_info2(M, N, K, int(transA), int(transB), float(beta), out))
    else:
        caps = (ctypes.c_int * 3)(*cluster_caps)
        check(lib.isam_gemm_plan_for(M, N, K, int(transA), int(transB), float(beta), num_sms, smem_optin, caps, out))
    return dict(zip(("BN", "split", "stages", "group_m", "grid", "smem", "tile_m", "cta_pair"), list(out)))


def gru_forward(T, batch, hidden, x, W, U, b, h0, h_out, reset_before=False) -> None:
    """isam_gru_forward, or isam_gru_forward_reset_before with reset_before
    (x, W, U bf16; b, h0, h_out fp32; h0 may be None)."""
    import torch
    lib = load()
    H = hidden
    _dev(x, torch.bfloat16, T * batch * H, "x")
    _dev(W, torch.bfloat16, 3 * H * H, "W")
    _dev(U, torch.bfloat16, 3 * H * H, "U")
    _dev(b, torch.float32, 6 * H, "b")
    if h0 is not None:
        _dev(h0, torch.float32, batch * H, "h0")
    _dev(h_out, torch.float32, T * batch * H, "h_out")
    _use_current_stream(lib)
    fn = lib.isam_gru_forward_reset_before if reset_before else lib.isam_gru_forward
    check(fn(T, batch, H, _ptr(x), _ptr(W), _ptr(U), _ptr(b), _ptr(h0), _ptr(h_out)))


def gru_forward_stack(layers, T, batch, hidden, x, W, U, b, h0, h_out, reset_before=False) -> None:
    """isam_gru_forward_stack: x [T,batch,H] bf16; W, U [layers,3H,H] bf16;
    b [layers,6H], h0 [layers,batch,H] (or None), h_out [layers,T,batch,H] fp32."""
    import torch
    lib = load()
    H, L = hidden, layers
    _dev(x, torch.bfloat16, T * batch * H, "x")
    _dev(W, torch.bfloat16, L * 3 * H * H, "W")
    _dev(U, torch.bfloat16, L * 3 * H * H, "U")
    _dev(b, torch.float32, L * 6 * H, "b")
    if h0 is not None:
        _dev(h0, torch.float32, L * batch * H, "h0")
    _dev(h_out, torch.float32, L * T * batch * H, "h_out")
    _use_current_stream(lib)
    check(lib.isam_gru_forward_stack(L, T, batch, H, int(bool(reset_before)), _ptr(x), _ptr(W),
                                     _ptr(U), _ptr(b), _ptr(h0), _ptr(h_out)))


def dwsep_conv(N, H, W, Cin, Cout, x, dw_w, pw_w, out) -> None:
    """isam_dwsep_conv: NHWC 3x3 depthwise (pad 1) then 1x1 pointwise."""
    import torch
    lib = load()
    _dev(x, torch.bfloat16, N * H * W * Cin, "x")
    _dev(dw_w, torch.bfloat16, 9 * Cin, "dw_w")
    _dev(pw_w, torch.bfloat16, Cin * Cout, "pw_w")
    _dev(out, torch.float32, N * H * W * Cout, "out")
    _use_current_stream(lib)
    check(lib.isam_dwsep_conv(N, H, W, Cin, Cout, _ptr(x), _ptr(dw_w), _ptr(pw_w), _ptr(out)))


def depthwise_conv3x3(N, H, W, C, x, dw_w, y) -> None:
    """isam_depthwise_conv3x3: NHWC 3x3 depthwise (pad 1), bf16 in and out."""
    import torch
    lib = load()
    _dev(x, torch.bfloat16, N * H * W * C, "x")
    _dev(dw_w, torch.bfloat16, 9 * C, "dw_w")
    _dev(y, torch.bfloat16, N * H * W * C, "y")
    _use_current_stream(lib)
    check(lib.isam_depthwise_conv3x3(N, H, W, C, _ptr(x), _ptr(dw_w), _ptr(y)))


_DWSEP_PLAN_KEYS = ("kernel", "rows_per_tile", "blocks", "block_cout")
_GRU_PLAN_KEYS = ("splits", "atoms", "batch_pad", "ctas", "smem", "path", "chunks")


def dwsep_plan(W, Cin, Cout, smem_optin=None) -> dict:
    """isam_dwsep_plan_info: the kernel, tile rows and output-channel blocks
    isam_dwsep_conv takes for this width and channel counts (nothing is
    launched); with smem_optin, isam_dwsep_plan_for on those limits (no GPU)."""
    lib = load()
    out = (ctypes.c_int * 4)()
    if smem_optin is None:
        check(lib.isam_dwsep_plan_info(W, Cin, Cout, out))
    else:
        check(lib.isam_dwsep_plan_for(W, Cin, Cout, smem_optin, out))
    return dict(zip(_DWSEP_PLAN_KEYS, list(out)))


def gru_plan(layers, batch, hidden, reset_before=False, num_sms=None, smem_optin=None) -> dict:
    """isam_gru_plan_info: K splits, padded batch, CTAs, shared memory and the
    layer schedule of a GRU call (nothing is launched); with num_sms and
    smem_optin, isam_gru_plan_for on those limits (no GPU)."""
    lib = load()
    out = (ctypes.c_int * 7)()
    if num_sms is None:
        check(lib.isam_gru_plan_info(layers, batch, hidden, int(bool(reset_before)), out))
    else:
        check(lib.isam_gru_plan_for(layers, batch, hidden, int(bool(reset_before)), num_sms, smem_optin, out))
    return dict(zip(_GRU_PLAN_KEYS, list(out)))
