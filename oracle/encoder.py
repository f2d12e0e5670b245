"""CPU oracle for the end-to-end DeiT encoder forward with block-sparse linears (arXiv 2407.02068:
the pruned ViTs of Sec. 4, whose linears are the Sec. 3.1 / 3.3 block-sparse layers).

TEST INFRASTRUCTURE ONLY, like the rest of ``oracle/``: used by ``tests/`` and ``bench.py``'s
CPU-baseline leg; the product library never imports it. numpy in float64.

The encoder is the standard pre-norm ViT block stack (DeiT): per layer
    h = LN1(x);  qkv = h W~qkv^T + b;  a = MHSA(qkv);  x = x + (a W~proj^T + b)
    h = LN2(x);  f = gelu(h W~fc1^T + b);  x = x + (f W~fc2^T + b)
and a final LayerNorm. LN(x) = (x - mean) / sqrt(var + eps) * gamma + beta over the feature axis
(biased variance). MHSA splits qkv's 3D columns as (3, heads, head_dim), softmax((q k^T) /
sqrt(head_dim)) v per image and head, heads concatenated. Every hand-off the GPU stores in bf16 is
rounded to bf16 here too (round to nearest even): LayerNorm outputs, linear outputs, the
attention output and the residual stream after each addition.
"""
from __future__ import annotations

import numpy as np

from . import bf16_to_f64, linear, round_bf16


def layernorm(x: np.ndarray, gamma: np.ndarray, beta: np.ndarray, eps: float) -> np.ndarray:
    """Row-wise LayerNorm in float64 (biased variance)."""
    x = np.asarray(x, dtype=np.float64)
    mu = x.mean(axis=-1, keepdims=True)
    var = ((x - mu) ** 2).mean(axis=-1, keepdims=True)
    return (x - mu) / np.sqrt(var + eps) * np.asarray(gamma, np.float64) + np.asarray(beta, np.float64)


def attention(qkv: np.ndarray, tokens: int, heads: int, head_dim: int) -> np.ndarray:
    """Multi-head self-attention in float64. qkv: [images * tokens, 3 * heads * head_dim];
    returns [images * tokens, heads * head_dim]."""
    qkv = np.asarray(qkv, dtype=np.float64)
    images = qkv.shape[0] // tokens
    D = heads * head_dim
    out = np.empty((images * tokens, D), dtype=np.float64)
    for b in range(images):
        rows = slice(b * tokens, (b + 1) * tokens)
        for h in range(heads):
            q = qkv[rows, h * head_dim:(h + 1) * head_dim]
            k = qkv[rows, D + h * head_dim:D + (h + 1) * head_dim]
            v = qkv[rows, 2 * D + h * head_dim:2 * D + (h + 1) * head_dim]
            s = q @ k.T / np.sqrt(head_dim)
            s = s - s.max(axis=1, keepdims=True)
            p = np.exp(s)
            p /= p.sum(axis=1, keepdims=True)
            out[rows, h * head_dim:(h + 1) * head_dim] = p @ v
    return out


def _bits_to_f64(bits):
    return bf16_to_f64(np.asarray(bits, dtype=np.uint16))


def layer_forward(x_bits: np.ndarray, L, tokens: int, heads: int, eps: float = 1e-6,
                  nthreads: int | None = None) -> np.ndarray:
    """One encoder layer on the bf16 residual stream x_bits [images * tokens, D] (uint16 bits):
    x + Attn(LN1(x)), then that + MLP(LN2(.)), every hand-off rounded to bf16; returns the new
    stream as bf16 bits. ``L`` as for ``encoder_forward``."""
    x = np.asarray(x_bits, dtype=np.uint16)
    head_dim = x.shape[1] // heads
    h = round_bf16(layernorm(_bits_to_f64(x), *L["ln1"], eps))
    W, M, bias, b = L["qkv"]
    qkv = round_bf16(linear(h, W, M, b, bias, False, nthreads))
    a = round_bf16(attention(_bits_to_f64(qkv), tokens, heads, head_dim))
    W, M, bias, b = L["proj"]
    p = round_bf16(linear(a, W, M, b, bias, False, nthreads))
    x = round_bf16(_bits_to_f64(x) + _bits_to_f64(p))
    h = round_bf16(layernorm(_bits_to_f64(x), *L["ln2"], eps))
    W, M, bias, b = L["fc1"]
    f = round_bf16(linear(h, W, M, b, bias, True, nthreads))
    W, M, bias, b = L["fc2"]
    o = round_bf16(linear(f, W, M, b, bias, False, nthreads))
    return round_bf16(_bits_to_f64(x) + _bits_to_f64(o))


def encoder_forward(x_bits: np.ndarray, layers, final, tokens: int, heads: int, eps: float = 1e-6,
                    nthreads: int | None = None) -> np.ndarray:
    """The encoder on bf16 token activations x_bits [images * tokens, D] (uint16 bits); returns the
    final LayerNorm output as bf16 bits.

    ``layers``: per layer a dict with ln1 / ln2 = (gamma, beta) float32 arrays and qkv / proj / fc1 /
    fc2 = (W_bits, mask, bias, b) as for ``oracle.linear``; ``final`` = (gamma, beta)."""
    x = np.asarray(x_bits, dtype=np.uint16)
    for L in layers:
        x = layer_forward(x, L, tokens, heads, eps, nthreads)
    return round_bf16(layernorm(_bits_to_f64(x), *final, eps))
