"""CPU oracle for LPViT's layer-wise pruning-ratio allocation (arXiv 2407.02068, Sec. 3.2-3.5).

TEST INFRASTRUCTURE ONLY, like the rest of ``oracle/``: used by ``tests/`` and ``bench.py``'s
CPU-baseline leg; the product library never imports it. Plain numpy in float64, written from the
definitions, slow on purpose.

What it computes:

* ``mean_gradient(G)`` -- the first-order gradient grad_W f as the average of N per-sample
  gradients, in float32 like the gradients themselves: summed over the samples in order with
  float32 additions, then divided by N (IEEE float32; the gradient the Taylor block scores of
  Sec. 3.1 take).
* ``delta_curve`` -- the per-layer curve of Sec. 3.4 / 3.5: for alpha_k = k / steps, k = 0..steps,
      delta(alpha_k) = g . dW_k + 1/2 dW_k^T H dW_k,
  where dW_k = -W on the blocks pruned at alpha_k (the bottom prune_count(alpha_k, blocks) blocks
  by Taylor score, ties kept by lower linear index, Sec. 3.1) and 0 elsewhere, g = mean_gradient,
  and H is the empirical Fisher of Sec. 3.5, kappa I + (1/N) sum_n g_n g_n^T. The quadratic form is
  evaluated as kappa |dW|^2 + (1/N) sum_n (g_n . dW)^2 (the same number, never forming D x D).
  Each alpha_k is evaluated directly, not through the incremental update of Eq. update.
* ``distortion(delta)`` -- the per-layer output-distortion term of Eq. obj_f, delta^2.
* ``lambda_search`` -- Sec. 3.4, Eq. langrangian2: for a multiplier lambda, layer i takes the
  largest alpha_k such that every discrete slope of its distortion curve up to k,
  (D_i(alpha_j) - D_i(alpha_{j-1})) * steps, is at most lambda_i = lambda + beta * c_i
  (c_i = M_i N_i K_i / (B_n B_k), the layer's power coefficient); lambda is traversed over every
  value where some layer's choice changes, and the smallest lambda whose FLOPs-remained ratio
  sum_i (1 - alpha_i) F_i / sum_i F_i is at most R is returned (the least pruning that meets the
  target; if no lambda meets it, the most pruning).
"""
from __future__ import annotations

import math

import numpy as np

from . import bf16_to_f64, block_scores, block_shape, taylor_mask


def mean_gradient(G: np.ndarray) -> np.ndarray:
    """float32 [n, k]: the samples of G (float32 [N, n, k]) summed in order in float32, / N."""
    G = np.asarray(G, dtype=np.float32)
    acc = np.zeros(G.shape[1:], dtype=np.float32)
    for i in range(G.shape[0]):
        acc = acc + G[i]
    return acc / np.float32(G.shape[0])


def pruned_delta_w(W_bits: np.ndarray, g32: np.ndarray, b, alpha: float) -> np.ndarray:
    """dW at pruning ratio alpha: -W on the blocks the Taylor ranking eliminates, 0 elsewhere."""
    bn, bk = block_shape(b)
    W = bf16_to_f64(W_bits)
    mask = taylor_mask(block_scores(W_bits, g32, b), alpha)
    keep = np.kron(mask, np.ones((bn, bk), dtype=np.uint8)).astype(bool)
    return np.where(keep, 0.0, -W)


def _delta(dW: np.ndarray, g: np.ndarray, Gd: np.ndarray, kappa: float) -> float:
    """g . dW + 1/2 (kappa |dW|^2 + (1/N) sum_n (g_n . dW)^2) for flattened float64 operands."""
    first = float(g @ dW)
    quad = kappa * float(dW @ dW) + float(np.sum((Gd @ dW) ** 2)) / Gd.shape[0]
    return first + 0.5 * quad


def delta_curve(W_bits: np.ndarray, G: np.ndarray, b, steps: int, kappa: float) -> np.ndarray:
    """delta(alpha_k) for alpha_k = k / steps, k = 0..steps (float64 [steps + 1]).

    W_bits: bf16 bits [n, k]; G: float32 per-sample gradients [N, n, k]; b: block (int or (bn, bk))."""
    G = np.asarray(G, dtype=np.float32)
    N = G.shape[0]
    g32 = mean_gradient(G)
    g = g32.astype(np.float64).ravel()
    Gd = G.reshape(N, -1).astype(np.float64)
    out = np.empty(steps + 1, dtype=np.float64)
    for kk in range(steps + 1):
        out[kk] = _delta(pruned_delta_w(W_bits, g32, b, kk / steps).ravel(), g, Gd, kappa)
    return out


def delta_at_mask(W_bits: np.ndarray, G: np.ndarray, b, mask: np.ndarray, kappa: float) -> float:
    """delta for a given block mask (1 = kept): dW = -W on the removed blocks, as in delta_curve."""
    bn, bk = block_shape(b)
    G = np.asarray(G, dtype=np.float32)
    N = G.shape[0]
    g = mean_gradient(G).astype(np.float64).ravel()
    Gd = G.reshape(N, -1).astype(np.float64)
    keep = np.kron(np.asarray(mask, dtype=np.uint8), np.ones((bn, bk), dtype=np.uint8)).astype(bool)
    dW = np.where(keep, 0.0, -bf16_to_f64(W_bits)).ravel()
    return _delta(dW, g, Gd, kappa)


def distortion(delta: np.ndarray) -> np.ndarray:
    return np.asarray(delta, dtype=np.float64) ** 2


def shifted_slopes(D: np.ndarray, steps: int, beta: float, c: float) -> np.ndarray:
    """t_j = (D[j] - D[j-1]) * steps - beta * c for j = 1..steps: the layer may move to alpha_j
    while every t up to j is at most lambda."""
    D = np.asarray(D, dtype=np.float64)
    return np.array([(D[j] - D[j - 1]) * steps - beta * c for j in range(1, steps + 1)])


def layer_index(t: np.ndarray, lam: float) -> int:
    """The largest k with t_1..t_k all <= lam (0 when t_1 > lam)."""
    k = 0
    for v in t:
        if v <= lam:
            k += 1
        else:
            break
    return k


def flops_remained(ks, steps: int, F) -> float:
    num = sum((1.0 - k / steps) * f for k, f in zip(ks, F))
    return num / sum(F)


def lambda_search(D_list, steps: int, F, c, beta: float, R: float):
    """Returns (lambda, [k_i], flops ratio): alpha_i = k_i / steps for every layer."""
    T = [shifted_slopes(D, steps, beta, ci) for D, ci in zip(D_list, c)]
    candidates = sorted(set(float(v) for t in T for v in t))
    best = None
    for lam in [-math.inf] + candidates:
        ks = [layer_index(t, lam) for t in T]
        r = flops_remained(ks, steps, F)
        best = (lam, ks, r)
        if r <= R:
            return best
    return best
