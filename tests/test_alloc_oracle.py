"""Pins for the pruning-ratio allocation oracle (oracle/alloc.py, Sec. 3.2-3.5) against what the
paper and the mathematics fix: a hand-worked lambda search (tests/golden/lambda_search_tiny.txt),
closed forms, the empirical Fisher written out as a dense D x D matrix, and the paper's own
incremental update (Eq. update) run on that matrix."""
import math
import os

import numpy as np
import pytest
import torch

import oracle
from oracle import alloc
from paper_2407_02068_gb300 import inputs

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _golden_lambda():
    vals, cases = {}, []
    with open(os.path.join(GOLDEN, "lambda_search_tiny.txt")) as f:
        for line in f:
            line = line.split("#", 1)[0].split()
            if not line:
                continue
            if line[0] == "case":
                beta, R, lam, k1, k2 = line[1:]
                cases.append((float(beta), float(R), float(lam), [int(k1), int(k2)]))
            else:
                vals[line[0]] = [float(v) for v in line[1:]]
    return vals, cases


def test_lambda_search_matches_the_hand_worked_example():
    v, cases = _golden_lambda()
    steps = int(v["steps"][0])
    for beta, R, lam, ks in cases:
        got_lam, got_ks, r = alloc.lambda_search([v["D1"], v["D2"]], steps, v["F"], v["c"], beta, R)
        assert got_ks == ks and got_lam == lam, (beta, R, got_lam, got_ks)
        assert r <= R or R < 0


def _case(n, k, b, N, seed, scale=1e-2):
    rng = np.random.default_rng(seed)
    W = (rng.standard_normal((n, k)) * 0.05).astype(np.float32)
    Wb = inputs.bf16_bits(torch.from_numpy(W).to(torch.bfloat16))
    G = (rng.standard_normal((N, n, k)) * scale).astype(np.float32)
    return Wb, G


def test_mean_gradient_sums_in_float32_in_sample_order():
    G = np.array([[[1e8]], [[1.0]], [[-1e8]]], dtype=np.float32)
    assert alloc.mean_gradient(G)[0, 0] == 0.0                    # 1e8 + 1 rounds back to 1e8 in float32
    G2 = np.array([[[1.0]], [[1e8]], [[-1e8]]], dtype=np.float32)
    assert alloc.mean_gradient(G2)[0, 0] == 0.0
    G3 = np.array([[[1e8]], [[-1e8]], [[1.0]]], dtype=np.float32)
    assert alloc.mean_gradient(G3)[0, 0] == np.float32(1.0) / np.float32(3.0)  # order decides
    G = (np.arange(24, dtype=np.float32).reshape(3, 2, 4) / 8)
    assert np.array_equal(alloc.mean_gradient(G), (G[0] + G[1] + G[2]) / np.float32(3))


def test_no_pruning_gives_zero_and_zero_gradients_give_the_kappa_closed_form():
    n, k, b, steps, kappa = 64, 96, 32, 6, 0.7
    Wb, _ = _case(n, k, b, 1, 3)
    G = np.zeros((4, n, k), dtype=np.float32)
    d = alloc.delta_curve(Wb, G, b, steps, kappa)
    assert d[0] == 0.0
    # zero gradients: every block scores 0, ties keep the lower linear index, so alpha_k removes
    # the last prune_count(alpha_k) blocks in linear order, and delta = kappa / 2 |W there|^2
    W = oracle.bf16_to_f64(Wb)
    blocks = [(r, j) for r in range(n // b) for j in range(k // b)]
    for kk in range(steps + 1):
        p = oracle.prune_count(kk / steps, len(blocks))
        gone = blocks[len(blocks) - p:]
        want = 0.5 * kappa * sum(float(np.sum(W[r * b:(r + 1) * b, j * b:(j + 1) * b] ** 2)) for r, j in gone)
        assert d[kk] == pytest.approx(want, rel=1e-13, abs=0)


@pytest.mark.parametrize("b", [8, (8, 16)])
def test_delta_equals_the_dense_fisher_quadratic_form(b):
    """H = kappa I + (1/N) sum g_n g_n^T built as a dense matrix (Sec. 3.5)."""
    n, k, N, steps, kappa = 16, 32, 5, 4, 0.3
    Wb, G = _case(n, k, b, N, 11)
    d = alloc.delta_curve(Wb, G, b, steps, kappa)
    g32 = alloc.mean_gradient(G)
    g = g32.astype(np.float64).ravel()
    Gd = G.reshape(N, -1).astype(np.float64)
    H = kappa * np.eye(n * k) + Gd.T @ Gd / N
    for kk in range(steps + 1):
        dW = alloc.pruned_delta_w(Wb, g32, b, kk / steps).ravel()
        assert d[kk] == pytest.approx(g @ dW + 0.5 * dW @ H @ dW, rel=1e-11, abs=1e-18)


def test_the_papers_incremental_update_reproduces_the_curve():
    """Eq. update: delta_k - delta_{k-1} = g'^T d + (d/2 + dW_{k-1})^T H' d with d = dW_k - dW_{k-1},
    run on the dense Fisher; it must land on the directly evaluated curve at every step."""
    n, k, b, N, steps, kappa = 32, 32, 8, 7, 8, 0.05
    Wb, G = _case(n, k, b, N, 12)
    d_direct = alloc.delta_curve(Wb, G, b, steps, kappa)
    g32 = alloc.mean_gradient(G)
    g = g32.astype(np.float64).ravel()
    Gd = G.reshape(N, -1).astype(np.float64)
    H = kappa * np.eye(n * k) + Gd.T @ Gd / N
    prev = np.zeros(n * k)
    delta = 0.0
    for kk in range(1, steps + 1):
        cur = alloc.pruned_delta_w(Wb, g32, b, kk / steps).ravel()
        dd = cur - prev
        idx = np.nonzero(dd)[0]  # the sub-vector of newly pruned weights
        delta += g[idx] @ dd[idx] + (0.5 * dd[idx] + prev[idx]) @ H[idx][:, idx] @ dd[idx] \
            + prev[np.setdiff1d(np.arange(n * k), idx)] @ H[np.setdiff1d(np.arange(n * k), idx)][:, idx] @ dd[idx]
        assert delta == pytest.approx(d_direct[kk], rel=1e-10, abs=1e-16)
        prev = cur


def test_lambda_search_invariants_on_random_curves():
    rng = np.random.default_rng(5)
    L, steps = 12, 10
    D = [np.concatenate([[0.0], np.cumsum(np.sort(rng.random(steps)) * rng.uniform(0.5, 3))]) for _ in range(L)]
    F = rng.uniform(1, 5, L)
    c = rng.uniform(0.1, 2, L)
    prev_k = [0] * L
    for R in (1.0, 0.8, 0.6, 0.4, 0.2, 0.0):
        lam, ks, r = alloc.lambda_search(D, steps, F, c, 0.5, R)
        assert r <= R + 1e-15
        assert all(a >= b_ for a, b_ in zip(ks, prev_k))  # less FLOPs never un-prunes a layer
        assert r == pytest.approx(alloc.flops_remained(ks, steps, F))
        prev_k = ks
    # the least pruning that meets R: one lambda step lower misses it
    lam, ks, r = alloc.lambda_search(D, steps, F, c, 0.5, 0.5)
    T = [alloc.shifted_slopes(d, steps, 0.5, ci) for d, ci in zip(D, c)]
    lower = max([v for t in T for v in t if v < lam], default=-math.inf)
    assert alloc.flops_remained([alloc.layer_index(t, lower) for t in T], steps, F) > 0.5


def test_power_term_moves_quota_to_the_larger_matmul():
    """Same distortion curve, different power coefficients: with beta > 0 the layer with the larger
    M N K / (B_n B_k) is pruned at least as far, and strictly further for some beta."""
    steps = 8
    D = np.concatenate([[0.0], np.cumsum(np.linspace(0.1, 2.0, steps))])
    F = [1.0, 1.0]
    strict = False
    for beta in (0.0, 0.05, 0.2, 1.0):
        lam, ks, r = alloc.lambda_search([D, D], steps, F, [1.0, 4.0], beta, 0.5)
        assert ks[1] >= ks[0]
        if beta == 0.0:
            assert ks[0] == ks[1]
        strict |= ks[1] > ks[0]
    assert strict
