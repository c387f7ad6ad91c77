"""Thin ctypes binding of libunisvq (argument marshalling only).

Every step of the layer runs in the library's CUDA kernels; PyTorch supplies
device memory (tensors) and the current CUDA stream. If the shared library has
not been built, `load()` raises instead of falling back to anything else.
"""
from __future__ import annotations

import ctypes
import os

import numpy as np

LIB_PATH = os.path.join(os.path.dirname(os.path.abspath(__file__)), "_lib", "libunisvq.so")

OK, ERR_INVALID_ARG, ERR_UNSUPPORTED, ERR_CUDA, ERR_OOM, ERR_TIMEOUT = range(6)
(KERNEL_AUTO, KERNEL_DECODE, KERNEL_PREFILL, KERNEL_GEMV, KERNEL_SKINNY, KERNEL_GEMV_ROWS, KERNEL_GROUPED,
 KERNEL_STREAM) = range(8)

# Every function include/unisvq.h declares.
EXPORTS = [
    "unisvq_pack", "unisvq_linear", "unisvq_linear_force", "unisvq_dequant_debug",
    "unisvq_query", "unisvq_sync_status", "unisvq_destroy", "unisvq_clone",
    "unisvq_status_string", "unisvq_packed_code_bytes", "unisvq_pack_host", "unisvq_version",
    "unisvq_linear_group", "unisvq_linear_group_force", "unisvq_linear_noalloc", "unisvq_query_group",
    "unisvq_pack_grouped", "unisvq_set_rht", "unisvq_hadamard", "unisvq_pack_bits",
    "unisvq_prefill_table_host", "unisvq_debug_wait_timeout",
]
MAX_GROUP = 4


class UnisvqError(RuntimeError):
    def __init__(self, status: int, what: str):
        self.status = status
        super().__init__(f"{what}: {status_string(status)} (status {status})")


class Info(ctypes.Structure):
    _fields_ = [("N", ctypes.c_int), ("K", ctypes.c_int), ("d", ctypes.c_int),
                ("Np", ctypes.c_int), ("Kp", ctypes.c_int), ("kernel", ctypes.c_int),
                ("split_k", ctypes.c_int), ("grid_ctas", ctypes.c_int),
                ("code_bytes", ctypes.c_longlong), ("meta_bytes", ctypes.c_longlong),
                ("algo_bytes", ctypes.c_longlong), ("flops", ctypes.c_double), ("launches", ctypes.c_int)]


_lib = None


def load():
    """Load libunisvq.so (built in-tree by `__graft_entry__.build()`)."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(LIB_PATH):
        raise ImportError(f"libunisvq is not built ({LIB_PATH} missing); run __graft_entry__.build()")
    lib = ctypes.CDLL(LIB_PATH)
    vp, i, sz = ctypes.c_void_p, ctypes.c_int, ctypes.c_size_t
    lib.unisvq_pack.argtypes = [vp, vp, vp, i, i, i, vp, ctypes.POINTER(vp)]
    lib.unisvq_pack_grouped.argtypes = [vp, vp, vp, i, i, i, i, vp, ctypes.POINTER(vp)]
    lib.unisvq_pack_bits.argtypes = [vp, vp, vp, i, i, i, i, vp, ctypes.POINTER(vp)]
    lib.unisvq_set_rht.argtypes = [vp, vp, vp, i, vp]
    lib.unisvq_hadamard.argtypes = [vp, vp, i, i, vp, i, vp]
    lib.unisvq_linear.argtypes = [vp, vp, vp, i, vp]
    lib.unisvq_linear_force.argtypes = [vp, i, vp, vp, i, vp]
    lib.unisvq_linear_group.argtypes = [vp, i, vp, vp, i, vp]
    lib.unisvq_linear_group_force.argtypes = [vp, i, i, vp, vp, i, vp]
    lib.unisvq_linear_noalloc.argtypes = [vp, vp, vp, i, vp]
    lib.unisvq_dequant_debug.argtypes = [vp, vp, vp]
    lib.unisvq_debug_wait_timeout.argtypes = [vp, vp, vp]
    lib.unisvq_query.argtypes = [vp, i, ctypes.POINTER(Info)]
    lib.unisvq_query_group.argtypes = [vp, i, i, ctypes.POINTER(Info)]
    lib.unisvq_sync_status.argtypes = [vp]
    lib.unisvq_destroy.argtypes = [vp]
    lib.unisvq_clone.argtypes = [vp, vp, ctypes.POINTER(vp)]
    lib.unisvq_status_string.argtypes = [i]
    lib.unisvq_status_string.restype = ctypes.c_char_p
    lib.unisvq_packed_code_bytes.argtypes = [i, i]
    lib.unisvq_packed_code_bytes.restype = sz
    lib.unisvq_pack_host.argtypes = [vp, i, i, vp, sz]
    lib.unisvq_prefill_table_host.argtypes = [vp, vp, i, i, vp, sz, ctypes.POINTER(sz)]
    lib.unisvq_version.argtypes = []
    _lib = lib
    return lib


def status_string(status: int) -> str:
    return load().unisvq_status_string(int(status)).decode()


def _check(status: int, what: str):
    if status != OK:
        raise UnisvqError(status, what)


def _stream_ptr(stream=None):
    import torch
    s = stream if stream is not None else torch.cuda.current_stream()
    return ctypes.c_void_p(s.cuda_stream)


def packed_code_bytes(N: int, K: int) -> int:
    return int(load().unisvq_packed_code_bytes(N, K))


def prefill_table_host(A, B, d: int, bits: int = 2) -> np.ndarray:
    """The prefill GEMM's table for this A (d x d), B (d), as unisvq_pack
    builds it (unisvq_prefill_table_host; uint32 words)."""
    a16 = np.ascontiguousarray(np.asarray(A, dtype=np.float16).reshape(-1)).view(np.uint16)
    b16 = np.ascontiguousarray(np.asarray(B, dtype=np.float16).reshape(-1)).view(np.uint16)
    words = ctypes.c_size_t(0)
    _check(load().unisvq_prefill_table_host(a16.ctypes.data, b16.ctypes.data, int(d), int(bits), None, 0,
                                            ctypes.byref(words)), "prefill_table_host")
    out = np.zeros(words.value, dtype=np.uint32)
    _check(load().unisvq_prefill_table_host(a16.ctypes.data, b16.ctypes.data, int(d), int(bits), out.ctypes.data,
                                            out.size, ctypes.byref(words)), "prefill_table_host")
    return out


def pack_host(codes: np.ndarray) -> np.ndarray:
    """Packed device layout of `codes` ([N][K] uint8), computed on the host."""
    codes = np.ascontiguousarray(codes, dtype=np.uint8)
    N, K = codes.shape
    out = np.zeros(packed_code_bytes(N, K), dtype=np.uint8)
    _check(load().unisvq_pack_host(codes.ctypes.data, N, K, out.ctypes.data, out.nbytes), "pack_host")
    return out


def _f16_bits(a) -> np.ndarray:
    a = np.asarray(a)
    if a.dtype == np.uint16:
        return np.ascontiguousarray(a)
    return np.ascontiguousarray(a.astype(np.float16)).view(np.uint16)


def _sign_bytes(s) -> np.ndarray:
    """+-1 values (or 0/1 bytes) -> uint8 with 1 = -1."""
    a = np.asarray(s)
    if a.dtype == np.uint8:
        return np.ascontiguousarray(a)
    return np.ascontiguousarray((a < 0).astype(np.uint8))


def hadamard_ptr(x_ptr: int, y_ptr: int, M: int, n: int, signs_ptr: int, signs_first: int, stream_ptr: int) -> int:
    """Raw-pointer unisvq_hadamard; returns the status."""
    return load().unisvq_hadamard(ctypes.c_void_p(x_ptr), ctypes.c_void_p(y_ptr), int(M), int(n),
                                  ctypes.c_void_p(signs_ptr or None), int(signs_first), ctypes.c_void_p(stream_ptr))


def sync_status(stream=None) -> int:
    return int(load().unisvq_sync_status(_stream_ptr(stream)))


def wait_timeout_probe_ptr(src16_ptr: int, out3_ptr: int, stream=None) -> int:
    """unisvq_debug_wait_timeout: a bounded device wait that runs out (test hook)."""
    return int(load().unisvq_debug_wait_timeout(ctypes.c_void_p(src16_ptr), ctypes.c_void_p(out3_ptr),
                                                 _stream_ptr(stream)))


class UniSVQLinear:
    """One packed UniSVQ linear layer resident on the current CUDA device."""

    def __init__(self, codes: np.ndarray, A, B, stream=None, _handle=None, group_cols: int | None = None,
                 bits: int = 2):
        """One (A [d][d], B [d]) for the matrix (unisvq_pack; `bits` = 3 for
        codes 0..7, unisvq_pack_bits), or, with `group_cols`, one per (row,
        group of columns): A [N][G][d][d], B [N][G][d] (unisvq_pack_grouped)."""
        lib = load()
        if _handle is not None:
            self._h = _handle
        else:
            codes = np.ascontiguousarray(codes, dtype=np.uint8)
            A16 = _f16_bits(A)
            B16 = _f16_bits(B)
            d = A16.shape[-1]
            N, K = codes.shape
            h = ctypes.c_void_p()
            if group_cols is None:
                _check(lib.unisvq_pack_bits(codes.ctypes.data, A16.ctypes.data, B16.ctypes.data, N, K, d, int(bits),
                                            _stream_ptr(stream), ctypes.byref(h)), "unisvq_pack_bits")
            else:
                G = -(-K // group_cols)
                if A16.shape != (N, G, d, d) or B16.shape != (N, G, d):
                    raise ValueError("per-group A must be [N][G][d][d] and B [N][G][d]")
                _check(lib.unisvq_pack_grouped(codes.ctypes.data, A16.ctypes.data, B16.ctypes.data, N, K, d,
                                               group_cols, _stream_ptr(stream), ctypes.byref(h)),
                       "unisvq_pack_grouped")
            self._h = h
        info = self.query(1)
        self.N, self.K, self.d = info["N"], info["K"], info["d"]

    def clone(self, stream=None) -> "UniSVQLinear":
        h = ctypes.c_void_p()
        _check(load().unisvq_clone(self._h, _stream_ptr(stream), ctypes.byref(h)), "unisvq_clone")
        return UniSVQLinear(None, None, None, _handle=h)

    def forward(self, x, out=None, kernel: int = KERNEL_AUTO, stream=None):
        """y = x W_hat^T for a bf16 CUDA tensor x [M][K]; returns y [M][N] bf16."""
        import torch
        if x.dtype != torch.bfloat16 or not x.is_cuda or x.dim() != 2 or x.shape[1] != self.K:
            raise ValueError("x must be a CUDA bf16 tensor of shape [M, K]")
        x = x.contiguous()
        M = x.shape[0]
        if out is None:
            out = torch.empty((M, self.N), dtype=torch.bfloat16, device=x.device)
        elif out.dtype != torch.bfloat16 or not out.is_contiguous() or tuple(out.shape) != (M, self.N):
            raise ValueError("out must be a contiguous bf16 tensor of shape [M, N]")
        st = load().unisvq_linear_force(self._h, int(kernel), ctypes.c_void_p(x.data_ptr()),
                                        ctypes.c_void_p(out.data_ptr()), M, _stream_ptr(stream))
        _check(st, "unisvq_linear")
        return out

    __call__ = forward

    def forward_ptr(self, x_ptr: int, y_ptr: int, M: int, stream_ptr: int, kernel: int = KERNEL_AUTO) -> int:
        """Raw-pointer call (no checks in Python); returns the status."""
        return load().unisvq_linear_force(self._h, kernel, ctypes.c_void_p(x_ptr), ctypes.c_void_p(y_ptr),
                                          M, ctypes.c_void_p(stream_ptr))

    def forward_noalloc_ptr(self, x_ptr: int, y_ptr: int, M: int, stream_ptr: int) -> int:
        """Raw-pointer unisvq_linear_noalloc (fold workspace in the library's
        static device array); returns the status."""
        return load().unisvq_linear_noalloc(self._h, ctypes.c_void_p(x_ptr), ctypes.c_void_p(y_ptr), M,
                                            ctypes.c_void_p(stream_ptr))

    def dequant_debug(self, stream=None):
        import torch
        W = torch.empty((self.N, self.K), dtype=torch.float32, device="cuda")
        _check(load().unisvq_dequant_debug(self._h, ctypes.c_void_p(W.data_ptr()), _stream_ptr(stream)),
               "unisvq_dequant_debug")
        return W

    def set_rht(self, s_in, s_out, max_tokens: int = 64, stream=None):
        """Rotate inputs by (S_V, V) and outputs by (U, S_U) around the layer
        (unisvq_set_rht). s_in [K], s_out [N]: +-1 values or 0/1 bytes (1 = -1);
        both None removes the transform."""
        if s_in is None and s_out is None:
            _check(load().unisvq_set_rht(self._h, None, None, 0, _stream_ptr(stream)), "unisvq_set_rht")
            return
        si = _sign_bytes(s_in)
        so = _sign_bytes(s_out)
        _check(load().unisvq_set_rht(self._h, si.ctypes.data, so.ctypes.data, int(max_tokens), _stream_ptr(stream)),
               "unisvq_set_rht")

    def query(self, M: int) -> dict:
        info = Info()
        _check(load().unisvq_query(self._h, int(M), ctypes.byref(info)), "unisvq_query")
        return {f: getattr(info, f) for f, _ in Info._fields_}

    def close(self):
        if getattr(self, "_h", None) is not None and self._h.value:
            load().unisvq_destroy(self._h)
            self._h = ctypes.c_void_p()

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


def linear_group_ptr(layers, x_ptr: int, y_ptrs, M: int, stream_ptr: int, kernel=None) -> int:
    """Raw-pointer unisvq_linear_group (or unisvq_linear_group_force when
    `kernel` is given) over `layers` (same K); returns the status."""
    n = len(layers)
    hs = (ctypes.c_void_p * n)(*[l._h.value if isinstance(l._h, ctypes.c_void_p) else l._h for l in layers])
    ys = (ctypes.c_void_p * n)(*[int(p) for p in y_ptrs])
    if kernel is None:
        return load().unisvq_linear_group(hs, n, ctypes.c_void_p(x_ptr), ys, M, ctypes.c_void_p(stream_ptr))
    return load().unisvq_linear_group_force(hs, n, int(kernel), ctypes.c_void_p(x_ptr), ys, M,
                                            ctypes.c_void_p(stream_ptr))


def query_group(layers, M: int) -> dict:
    """unisvq_query_group: the launches unisvq_linear_group makes for `layers`."""
    n = len(layers)
    hs = (ctypes.c_void_p * n)(*[l._h.value if isinstance(l._h, ctypes.c_void_p) else l._h for l in layers])
    info = Info()
    _check(load().unisvq_query_group(hs, n, int(M), ctypes.byref(info)), "unisvq_query_group")
    return {f: getattr(info, f) for f, _ in Info._fields_}


def linear_group(layers, x, outs=None, stream=None, kernel=None):
    """y_i = x W_hat_i^T for layers that share x ([M][K] bf16 CUDA tensor);
    `kernel` (a KERNEL_* value) forces the kernel, else the library picks."""
    import torch
    if x.dtype != torch.bfloat16 or not x.is_cuda or x.dim() != 2:
        raise ValueError("x must be a CUDA bf16 tensor of shape [M, K]")
    x = x.contiguous()
    M = x.shape[0]
    if outs is None:
        outs = [torch.empty((M, l.N), dtype=torch.bfloat16, device=x.device) for l in layers]
    _check(linear_group_ptr(layers, x.data_ptr(), [o.data_ptr() for o in outs], M,
                            _stream_ptr(stream).value or 0, kernel), "unisvq_linear_group")
    return outs
