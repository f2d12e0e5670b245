"""CPU oracle for the LPViT block-sparse linear layer (arXiv 2407.02068).

TEST INFRASTRUCTURE ONLY: this package is imported by ``tests/``, by
``__graft_entry__.smoke()`` (to check one small GPU result) and by ``bench.py``'s CPU-baseline
and reference arm. The product library never imports, links or calls it, and it imports
nothing from the product package.

The arithmetic lives in ``lpvit_oracle.c`` (plain C, IEEE double, no fused multiply-add
contraction); this module compiles it with gcc on first use and wraps it with ctypes:

* ``linear``   -- y = [gelu](X (W (.) M)^T + bias) in float64 (Sec. 3.1 mask, Sec. 3.3 matmul)
* ``pack``     -- BSR packing of the surviving blocks (Sec. 1, Sec. 3.3)
* ``round_bf16`` / ``bf16_to_f64`` / ``gelu``
* ``block_scores`` / ``prune_count`` / ``taylor_mask`` -- the block mask from first-order Taylor
  scores (Sec. 3.1): |W . grad W| average-pooled per block, bottom alpha of the blocks eliminated
* ``deit_stack_rows`` -- the 48-GEMM DeiT linear stack on a subset of token rows
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "lpvit_oracle.c")
_BUILD = os.path.join(_HERE, "_build")
_LIB_PATH = os.path.join(_BUILD, "liblpvit_oracle.so")
_lock = threading.Lock()
_lib = None


def build(force: bool = False) -> str:
    """Compile the C oracle into ``oracle/_build/liblpvit_oracle.so`` (host gcc, -O2, no
    FMA contraction so x86 and Arm builds give identical bits)."""
    os.makedirs(_BUILD, exist_ok=True)
    if force or not os.path.exists(_LIB_PATH) or os.path.getmtime(_LIB_PATH) < os.path.getmtime(_SRC):
        tmp = _LIB_PATH + f".{os.getpid()}.tmp"
        subprocess.check_call(
            ["gcc", "-O2", "-std=c11", "-ffp-contract=off", "-fno-fast-math", "-fPIC", "-shared",
             "-o", tmp, _SRC, "-lm", "-lpthread"])
        os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def _load():
    global _lib
    with _lock:
        if _lib is None:
            lib = ctypes.CDLL(build())
            P = ctypes.c_void_p
            lib.lpvit_oracle_bf16_to_f64.restype = ctypes.c_double
            lib.lpvit_oracle_bf16_to_f64.argtypes = [ctypes.c_uint16]
            lib.lpvit_oracle_round_bf16.restype = ctypes.c_uint16
            lib.lpvit_oracle_round_bf16.argtypes = [ctypes.c_double]
            lib.lpvit_oracle_gelu.restype = ctypes.c_double
            lib.lpvit_oracle_gelu.argtypes = [ctypes.c_double]
            lib.lpvit_oracle_pack.restype = ctypes.c_int64
            lib.lpvit_oracle_pack.argtypes = [P, P, ctypes.c_int32, ctypes.c_int32, ctypes.c_int32, ctypes.c_int32,
                                              P, P, P]
            lib.lpvit_oracle_linear.restype = ctypes.c_int
            lib.lpvit_oracle_linear.argtypes = [P, ctypes.c_int64, ctypes.c_int64, P, P, ctypes.c_int32,
                                                ctypes.c_int32, ctypes.c_int32, ctypes.c_int32, P, ctypes.c_int, P,
                                                ctypes.c_int64, ctypes.c_int]
            lib.lpvit_oracle_block_scores.restype = ctypes.c_int
            lib.lpvit_oracle_block_scores.argtypes = [P, P, ctypes.c_int32, ctypes.c_int32, ctypes.c_int32,
                                                      ctypes.c_int32, P]
            lib.lpvit_oracle_prune_count.restype = ctypes.c_int64
            lib.lpvit_oracle_prune_count.argtypes = [ctypes.c_double, ctypes.c_int64]
            lib.lpvit_oracle_taylor_mask.restype = ctypes.c_int
            lib.lpvit_oracle_taylor_mask.argtypes = [P, ctypes.c_int64, ctypes.c_int64, P]
            lib.lpvit_oracle_round_bf16_array.restype = None
            lib.lpvit_oracle_round_bf16_array.argtypes = [P, P, ctypes.c_int64]
            _lib = lib
    return _lib


def _ptr(a: np.ndarray | None):
    return None if a is None else a.ctypes.data_as(ctypes.c_void_p)


def block_shape(b) -> tuple[int, int]:
    """A block given as b (square, b x b) or (bn, bk): bn output rows by bk input columns."""
    if isinstance(b, (tuple, list)):
        bn, bk = int(b[0]), int(b[1])
    else:
        bn = bk = int(b)
    if bn <= 0 or bk <= 0:
        raise ValueError("block sides must be positive")
    return bn, bk


def bf16_to_f64(bits) -> np.ndarray:
    """Exact widening of bf16 bit patterns (uint16) to float64."""
    bits = np.ascontiguousarray(bits, dtype=np.uint16)
    return (bits.astype(np.uint32) << 16).view(np.float32).astype(np.float64)


def round_bf16(y) -> np.ndarray:
    """float64 -> bf16 bit patterns, round to nearest, ties to even (C oracle)."""
    y = np.ascontiguousarray(y, dtype=np.float64)
    out = np.empty(y.shape, dtype=np.uint16)
    _load().lpvit_oracle_round_bf16_array(_ptr(y), _ptr(out), y.size)
    return out


def round_bf16_scalar(y: float) -> int:
    return int(_load().lpvit_oracle_round_bf16(float(y)))


def gelu(y) -> np.ndarray:
    """Exact GELU 0.5*y*(1+erf(y/sqrt(2))) through the C oracle, element by element."""
    lib = _load()
    y = np.asarray(y, dtype=np.float64)
    return np.vectorize(lib.lpvit_oracle_gelu, otypes=[np.float64])(y)


def pack(W_bits: np.ndarray, mask: np.ndarray, b):
    """BSR pack of W (uint16 bf16 bits [n, k]) under the block mask ([n/bn, k/bk], nonzero = kept);
    b is the block: an int (square) or (bn, bk).

    Returns (row_ptr int32[n/bn+1], col_idx int32[nnzb], blocks uint16[nnzb, bn, bk])."""
    bn, bk = block_shape(b)
    W_bits = np.ascontiguousarray(W_bits, dtype=np.uint16)
    mask = np.ascontiguousarray(mask, dtype=np.uint8)
    n, k = W_bits.shape
    if n % bn or k % bk or mask.shape != (n // bn, k // bk):
        raise ValueError("shape mismatch")
    cap = (n // bn) * (k // bk)
    row_ptr = np.zeros(n // bn + 1, dtype=np.int32)
    col_idx = np.zeros(max(cap, 1), dtype=np.int32)
    blocks = np.zeros((max(cap, 1), bn, bk), dtype=np.uint16)
    nnzb = _load().lpvit_oracle_pack(_ptr(W_bits), _ptr(mask), n, k, bn, bk, _ptr(row_ptr), _ptr(col_idx),
                                     _ptr(blocks))
    if nnzb < 0:
        raise ValueError("oracle pack rejected the arguments")
    return row_ptr, col_idx[:nnzb].copy(), blocks[:nnzb].copy()


def block_scores(W_bits: np.ndarray, G: np.ndarray, b) -> np.ndarray:
    """Sec. 3.1 block scores: the average of |W . G| over each bn x bk block (b = int or (bn, bk)),
    float64 [n/bn, k/bk]. W_bits: uint16 bf16 bits [n, k]; G: float32 gradient [n, k]."""
    bn, bk = block_shape(b)
    W_bits = np.ascontiguousarray(W_bits, dtype=np.uint16)
    G = np.ascontiguousarray(G, dtype=np.float32)
    n, k = W_bits.shape
    if G.shape != (n, k) or n % bn or k % bk:
        raise ValueError("shape mismatch")
    out = np.empty((n // bn, k // bk), dtype=np.float64)
    if _load().lpvit_oracle_block_scores(_ptr(W_bits), _ptr(G), n, k, bn, bk, _ptr(out)) != 0:
        raise ValueError("oracle block_scores rejected the arguments")
    return out


def prune_count(alpha: float, count: int) -> int:
    """Blocks eliminated at pruning ratio alpha: round(alpha * count), half away from zero."""
    return int(_load().lpvit_oracle_prune_count(float(alpha), int(count)))


def taylor_mask(scores: np.ndarray, alpha: float) -> np.ndarray:
    """Sec. 3.1 block mask: rank the blocks by score (ties: lower linear index first) and eliminate
    the bottom prune_count(alpha, blocks). Returns uint8 of the scores' shape, 1 = kept."""
    scores = np.ascontiguousarray(scores, dtype=np.float64)
    mask = np.empty(scores.shape, dtype=np.uint8)
    if _load().lpvit_oracle_taylor_mask(_ptr(scores), scores.size, prune_count(alpha, scores.size),
                                        _ptr(mask)) != 0:
        raise ValueError("oracle taylor_mask rejected the arguments")
    return mask


def linear(X_bits: np.ndarray, W_bits: np.ndarray, mask: np.ndarray, b, bias: np.ndarray | None,
           gelu: bool = False, nthreads: int | None = None) -> np.ndarray:
    """y = [gelu](X (W (.) M)^T + bias) in float64.

    X_bits: uint16 [m, k] (a row-strided view is fine); W_bits: uint16 [n, k]; b: the block, int
    (square) or (bn, bk); mask: uint8 [n/bn, k/bk]; bias: float32 [n] or None. Returns float64
    [m, n]."""
    bn, bk = block_shape(b)
    X_bits = np.asarray(X_bits, dtype=np.uint16)
    if X_bits.ndim != 2 or X_bits.strides[1] != 2:
        X_bits = np.ascontiguousarray(X_bits)
    ldx = X_bits.strides[0] // 2
    W_bits = np.ascontiguousarray(W_bits, dtype=np.uint16)
    mask = np.ascontiguousarray(mask, dtype=np.uint8)
    m, k = X_bits.shape
    n = W_bits.shape[0]
    if W_bits.shape[1] != k or n % bn or k % bk or mask.shape != (n // bn, k // bk):
        raise ValueError("shape mismatch")
    if bias is not None:
        bias = np.ascontiguousarray(bias, dtype=np.float32)
    Y = np.empty((m, n), dtype=np.float64)
    if nthreads is None:
        nthreads = os.cpu_count() or 1
    rc = _load().lpvit_oracle_linear(_ptr(X_bits), m, ldx, _ptr(W_bits), _ptr(mask), n, k, bn, bk, _ptr(bias),
                                     1 if gelu else 0, _ptr(Y), n, int(nthreads))
    if rc != 0:
        raise ValueError("oracle linear rejected the arguments")
    return Y


def deit_stack_rows(h0_bits: np.ndarray, layers, nthreads: int | None = None) -> np.ndarray:
    """The DeiT linear stack on a set of token rows, as bf16 bits in and out.

    ``layers`` is a sequence of dicts with keys qkv/proj/fc1/fc2, each a tuple
    (W_bits, mask, bias, b). Per layer (attention and LayerNorm are not part of this path):
      qkv  = bf16(h @ W~qkv^T + b)                  [rows, 3D]
      proj = bf16(qkv[:, 2D:3D] @ W~proj^T + b)     the V third stands in for the attention output
      fc1  = bf16(gelu(proj @ W~fc1^T + b))
      h    = bf16(fc1 @ W~fc2^T + b)
    Every product is the float64 oracle ``linear``; every hand-off rounds to bf16 (RNE)."""
    h = np.ascontiguousarray(h0_bits, dtype=np.uint16)
    for L in layers:
        W, M, bias, b = L["qkv"]
        qkv = round_bf16(linear(h, W, M, b, bias, False, nthreads))
        d = qkv.shape[1] // 3
        W, M, bias, b = L["proj"]
        proj = round_bf16(linear(qkv[:, 2 * d:3 * d], W, M, b, bias, False, nthreads))
        W, M, bias, b = L["fc1"]
        fc1 = round_bf16(linear(proj, W, M, b, bias, True, nthreads))
        W, M, bias, b = L["fc2"]
        h = round_bf16(linear(fc1, W, M, b, bias, False, nthreads))
    return h
