"""ctypes binding of liblpvit.so: one Python function per C entry point, same names, argument
marshalling only (every step of the layer runs in the library's CUDA kernels).

The library must have been built (``paper_2407_02068_gb300.build.build()``); if it is missing,
loading raises instead of falling back to anything else.
"""
from __future__ import annotations

import ctypes
import os
import threading

from .build import LIB

LPVIT_OK = 0
LPVIT_ERR_INVALID_ARG = 1
LPVIT_ERR_UNSUPPORTED = 2
LPVIT_ERR_CUDA = 3
LPVIT_ERR_TIMEOUT = 4
LPVIT_ERR_WORKSPACE = 5
LPVIT_BF16 = 0
LPVIT_F32 = 1

EXPORTS = ("lpvit_sched_bytes", "lpvit_pack_bsr", "lpvit_taylor_pack_bsr", "lpvit_workspace_bytes", "lpvit_bsr_linear",
           "lpvit_bsr_linear_gelu", "lpvit_bsr_linear_noalloc", "lpvit_check", "lpvit_status_string",
           "lpvit_selftest_wait", "lpvit_pack_bsr_many", "lpvit_taylor_block_mask",
           "lpvit_delta_curve_workspace_bytes", "lpvit_delta_curve", "lpvit_lambda_search", "lpvit_mean_gradient",
           "lpvit_add_layernorm", "lpvit_attention", "lpvit_bsr_linear_residual", "lpvit_chain_workspace_bytes",
           "lpvit_bsr_linear_chain")
LPVIT_NOALLOC_SCRATCH_BYTES = 8 * 1024 * 1024


class lpvit_bsr(ctypes.Structure):
    _fields_ = [
        ("n", ctypes.c_int32), ("k", ctypes.c_int32), ("bn", ctypes.c_int32), ("bk", ctypes.c_int32),
        ("nnzb_capacity", ctypes.c_int32),
        ("row_ptr", ctypes.c_void_p), ("col_idx", ctypes.c_void_p), ("blocks", ctypes.c_void_p),
        ("sched", ctypes.c_void_p), ("sched_bytes", ctypes.c_size_t),
    ]


class lpvit_chain_link(ctypes.Structure):
    _fields_ = [
        ("bsr", ctypes.POINTER(lpvit_bsr)), ("X", ctypes.c_void_p), ("ldx", ctypes.c_int64),
        ("bias", ctypes.c_void_p), ("Y", ctypes.c_void_p), ("ldy", ctypes.c_int64), ("gelu", ctypes.c_int32),
    ]


class LpvitError(RuntimeError):
    def __init__(self, status: int, what: str):
        self.status = status
        super().__init__(f"{what}: status {status} ({status_string(status)})")


_lock = threading.Lock()
_lib = None


def load(path: str | None = None):
    """Load liblpvit.so (once). Raises if the library has not been built."""
    global _lib
    with _lock:
        if _lib is not None:
            return _lib
        p = path or LIB
        if not os.path.exists(p):
            raise RuntimeError(f"{p} is missing: build the CUDA library first "
                               "(python -c 'import __graft_entry__ as g; g.build()')")
        lib = ctypes.CDLL(p)
        V, I32, I64, SZ = ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64, ctypes.c_size_t
        BP = ctypes.POINTER(lpvit_bsr)
        lib.lpvit_sched_bytes.restype = SZ
        lib.lpvit_sched_bytes.argtypes = [I32, I32, I32, I32]
        lib.lpvit_pack_bsr.restype = ctypes.c_int
        lib.lpvit_pack_bsr.argtypes = [V, V, BP, ctypes.POINTER(I32), V]
        lib.lpvit_taylor_pack_bsr.restype = ctypes.c_int
        lib.lpvit_taylor_pack_bsr.argtypes = [V, V, ctypes.c_double, V, V, BP, ctypes.POINTER(I32), V]
        lib.lpvit_taylor_block_mask.restype = ctypes.c_int
        lib.lpvit_taylor_block_mask.argtypes = [V, V, I32, I32, I32, I32, ctypes.c_double, V, V, V]
        lib.lpvit_delta_curve_workspace_bytes.restype = SZ
        lib.lpvit_delta_curve_workspace_bytes.argtypes = [I32, I32, I32, I32, I32, I32]
        lib.lpvit_delta_curve.restype = ctypes.c_int
        lib.lpvit_delta_curve.argtypes = [V, V, I32, I32, I32, I32, I32, ctypes.c_double, I32, V, V, SZ, V]
        lib.lpvit_add_layernorm.restype = ctypes.c_int
        lib.lpvit_add_layernorm.argtypes = [V, V, V, V, I64, I32, ctypes.c_double, V, V, V]
        lib.lpvit_attention.restype = ctypes.c_int
        lib.lpvit_attention.argtypes = [V, I64, I32, I32, I32, V, V]
        lib.lpvit_mean_gradient.restype = ctypes.c_int
        lib.lpvit_mean_gradient.argtypes = [V, I32, I64, V, V]
        lib.lpvit_lambda_search.restype = ctypes.c_int
        lib.lpvit_lambda_search.argtypes = [I32, I32, V, V, V, ctypes.c_double, ctypes.c_double, V, V, V]
        lib.lpvit_pack_bsr_many.restype = ctypes.c_int
        lib.lpvit_pack_bsr_many.argtypes = [I32, ctypes.POINTER(V), ctypes.POINTER(V), BP, V]
        lib.lpvit_workspace_bytes.restype = SZ
        lib.lpvit_workspace_bytes.argtypes = [BP, I64]
        for name in ("lpvit_bsr_linear", "lpvit_bsr_linear_gelu"):
            f = getattr(lib, name)
            f.restype = ctypes.c_int
            f.argtypes = [BP, V, I64, I64, V, V, I64, ctypes.c_int, V, SZ, V]
        lib.lpvit_bsr_linear_residual.restype = ctypes.c_int
        lib.lpvit_bsr_linear_residual.argtypes = [BP, V, I64, I64, V, ctypes.c_int32, V, I64, V, I64, V, SZ, V]
        CL = ctypes.POINTER(lpvit_chain_link)
        lib.lpvit_chain_workspace_bytes.restype = SZ
        lib.lpvit_chain_workspace_bytes.argtypes = [CL, I32, I64]
        lib.lpvit_bsr_linear_chain.restype = ctypes.c_int
        lib.lpvit_bsr_linear_chain.argtypes = [CL, I32, I64, V, SZ, V]
        lib.lpvit_bsr_linear_noalloc.restype = ctypes.c_int
        lib.lpvit_bsr_linear_noalloc.argtypes = [BP, V, I64, I64, V, V, I64, ctypes.c_int, ctypes.c_int, V]
        lib.lpvit_check.restype = ctypes.c_int
        lib.lpvit_check.argtypes = [V, V]
        lib.lpvit_selftest_wait.restype = ctypes.c_int
        lib.lpvit_selftest_wait.argtypes = [V, ctypes.c_uint64, ctypes.c_uint64, V]
        lib.lpvit_status_string.restype = ctypes.c_char_p
        lib.lpvit_status_string.argtypes = [ctypes.c_int]
        _lib = lib
        return lib


def status_string(status: int) -> str:
    return load().lpvit_status_string(int(status)).decode()


def lpvit_sched_bytes(n: int, k: int, bn: int, bk: int) -> int:
    return int(load().lpvit_sched_bytes(n, k, bn, bk))


def lpvit_pack_bsr(W_ptr: int, mask_ptr: int, bsr: lpvit_bsr, want_count: bool, stream: int):
    """Returns (status, nnzb or None)."""
    cnt = ctypes.c_int32(0)
    st = load().lpvit_pack_bsr(W_ptr, mask_ptr, ctypes.byref(bsr), ctypes.byref(cnt) if want_count else None,
                               stream)
    return st, (cnt.value if want_count else None)


def lpvit_taylor_pack_bsr(W_ptr: int, G_ptr: int, prune_ratio: float, scores_ptr: int, mask_ptr: int,
                          bsr: lpvit_bsr, want_count: bool, stream: int):
    """Returns (status, nnzb or None)."""
    cnt = ctypes.c_int32(0)
    st = load().lpvit_taylor_pack_bsr(W_ptr, G_ptr, prune_ratio, scores_ptr, mask_ptr, ctypes.byref(bsr),
                                      ctypes.byref(cnt) if want_count else None, stream)
    return st, (cnt.value if want_count else None)


def lpvit_pack_bsr_many(W_ptrs, mask_ptrs, bsrs, stream: int) -> int:
    """Pack len(bsrs) weights in two launches. ``bsrs``: a ctypes array of lpvit_bsr (or a list)."""
    n = len(bsrs)
    if not isinstance(bsrs, ctypes.Array):
        arr = (lpvit_bsr * n)()
        for i, b in enumerate(bsrs):
            arr[i] = b
        bsrs = arr
    Wa = (ctypes.c_void_p * n)(*W_ptrs)
    Ma = (ctypes.c_void_p * n)(*mask_ptrs)
    return load().lpvit_pack_bsr_many(n, Wa, Ma, bsrs, stream)


def lpvit_taylor_block_mask(W_ptr, G_ptr, n, k, bn, bk, prune_ratio, scores_ptr, mask_ptr, stream) -> int:
    return load().lpvit_taylor_block_mask(W_ptr, G_ptr, n, k, bn, bk, float(prune_ratio), scores_ptr, mask_ptr,
                                          stream)


def lpvit_delta_curve_workspace_bytes(nsamples: int, n: int, k: int, bn: int, bk: int, steps: int) -> int:
    return int(load().lpvit_delta_curve_workspace_bytes(nsamples, n, k, bn, bk, steps))


def lpvit_delta_curve(W_ptr, G_ptr, nsamples, n, k, bn, bk, kappa, steps, delta_ptr, ws_ptr, ws_bytes,
                      stream) -> int:
    return load().lpvit_delta_curve(W_ptr, G_ptr, nsamples, n, k, bn, bk, float(kappa), steps, delta_ptr, ws_ptr,
                                    ws_bytes, stream)


def lpvit_add_layernorm(x_ptr, r_ptr, gamma_ptr, beta_ptr, rows, D, eps, sum_ptr, norm_ptr, stream) -> int:
    return load().lpvit_add_layernorm(x_ptr, r_ptr, gamma_ptr, beta_ptr, rows, D, float(eps), sum_ptr, norm_ptr, stream)


def lpvit_attention(qkv_ptr, images, tokens, heads, head_dim, out_ptr, stream) -> int:
    return load().lpvit_attention(qkv_ptr, images, tokens, heads, head_dim, out_ptr, stream)


def lpvit_mean_gradient(G_ptr, nsamples, count, g_ptr, stream) -> int:
    return load().lpvit_mean_gradient(G_ptr, nsamples, count, g_ptr, stream)


def lpvit_lambda_search(delta_rows, steps: int, flops, power_coef, beta: float, flops_ratio: float):
    """Host call. delta_rows: sequence of per-layer sequences of steps + 1 floats. Returns
    (status, [k_i], lambda, ratio)."""
    L = len(delta_rows)
    D = (ctypes.c_double * (L * (steps + 1)))(*[float(v) for row in delta_rows for v in row])
    F = (ctypes.c_double * L)(*[float(v) for v in flops])
    C = (ctypes.c_double * L)(*[float(v) for v in power_coef])
    K = (ctypes.c_int32 * L)()
    lam, ratio = ctypes.c_double(0.0), ctypes.c_double(0.0)
    st = load().lpvit_lambda_search(L, steps, D, F, C, float(beta), float(flops_ratio), K, ctypes.byref(lam),
                                    ctypes.byref(ratio))
    return st, list(K), lam.value, ratio.value


def lpvit_workspace_bytes(bsr: lpvit_bsr, m: int) -> int:
    return int(load().lpvit_workspace_bytes(ctypes.byref(bsr), m))


def lpvit_bsr_linear(bsr, X_ptr, m, ldx, bias_ptr, Y_ptr, ldy, y_dtype, ws_ptr, ws_bytes, stream) -> int:
    return load().lpvit_bsr_linear(ctypes.byref(bsr), X_ptr, m, ldx, bias_ptr, Y_ptr, ldy, y_dtype, ws_ptr,
                                   ws_bytes, stream)


def lpvit_bsr_linear_gelu(bsr, X_ptr, m, ldx, bias_ptr, Y_ptr, ldy, y_dtype, ws_ptr, ws_bytes, stream) -> int:
    return load().lpvit_bsr_linear_gelu(ctypes.byref(bsr), X_ptr, m, ldx, bias_ptr, Y_ptr, ldy, y_dtype, ws_ptr,
                                        ws_bytes, stream)


def lpvit_bsr_linear_residual(bsr, X_ptr, m, ldx, bias_ptr, gelu, R_ptr, ldr, Y_ptr, ldy, ws_ptr, ws_bytes,
                              stream) -> int:
    return load().lpvit_bsr_linear_residual(ctypes.byref(bsr), X_ptr, m, ldx, bias_ptr, int(gelu), R_ptr,
                                            ldr, Y_ptr, ldy, ws_ptr, ws_bytes, stream)


def chain_links(rows) -> ctypes.Array:
    """A ctypes array of lpvit_chain_link from (bsr, X_ptr, ldx, bias_ptr, Y_ptr, ldy, gelu) tuples; the
    lpvit_bsr structs must outlive the array."""
    arr = (lpvit_chain_link * len(rows))()
    for i, (bsr, X_ptr, ldx, bias_ptr, Y_ptr, ldy, gelu) in enumerate(rows):
        arr[i] = lpvit_chain_link(ctypes.pointer(bsr) if bsr is not None else None, X_ptr, ldx, bias_ptr, Y_ptr,
                                  ldy, int(gelu))
    return arr


def lpvit_chain_workspace_bytes(links, count: int, m: int) -> int:
    return int(load().lpvit_chain_workspace_bytes(links, count, m))


def lpvit_bsr_linear_chain(links, count: int, m: int, ws_ptr, ws_bytes, stream) -> int:
    return load().lpvit_bsr_linear_chain(links, count, m, ws_ptr, ws_bytes, stream)


def lpvit_bsr_linear_noalloc(bsr, X_ptr, m, ldx, bias_ptr, Y_ptr, ldy, y_dtype, gelu, stream) -> int:
    """The linear with the library's own scratch array as workspace (no allocation by anyone)."""
    return load().lpvit_bsr_linear_noalloc(ctypes.byref(bsr), X_ptr, m, ldx, bias_ptr, Y_ptr, ldy, y_dtype,
                                           1 if gelu else 0, stream)


def lpvit_check(ws_ptr: int, stream: int) -> int:
    return load().lpvit_check(ws_ptr, stream)


def lpvit_selftest_wait(ws_ptr: int, limit_ns: int, abort_after_ns: int, stream: int) -> int:
    """Force the bounded device wait to run out (diagnostic of the failure path)."""
    return load().lpvit_selftest_wait(ws_ptr, limit_ns, abort_after_ns, stream)


def lpvit_status_string(status: int) -> str:
    return status_string(status)
