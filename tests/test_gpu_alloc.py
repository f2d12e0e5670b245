"""Pruning-ratio allocation on the GPU (lpvit_mean_gradient, lpvit_delta_curve) against the oracle
(oracle/alloc.py): the mean gradient bit for bit (both float32 in sample order), the distortion
curves within 1e-9 of their largest magnitude (the GPU takes exact products, float-pair lane sums of
at most 128 terms, double beyond, and updates incrementally by Eq. update; the oracle evaluates
every alpha directly in double), and the whole allocation -- curves, lambda search,
Taylor masks at the allocated ratios, pack and linear -- on a small stack.

The GPU ranks blocks by float32 Taylor scores, the oracle by their exact averages (Sec. 3.1). A
ratio step whose cut-off falls within the float32 bound of two blocks' scores may prune either of
them (taylor_bounds); at such steps the oracle's delta is taken for the pruned set the GPU chose,
after that set is checked against the band rule, so every step is compared."""
import numpy as np
import pytest
import torch

import oracle
from oracle import alloc
from paper_2407_02068_gb300 import inputs
from taylor_bounds import ambiguous_steps, assert_mask_matches_away_from_cutoff

pytestmark = pytest.mark.gpu

CURVE_TOL = 1e-9


@pytest.fixture(scope="module")
def lp():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2407_02068_gb300 import build
    build.build()
    import paper_2407_02068_gb300 as lp
    return lp


def _wg(n, k, N, seed, gscale=1e-2):
    W = inputs.weight(n, k, seed, "cuda")
    g = torch.Generator(device="cuda").manual_seed(seed + 1)
    G = (torch.randn(N, n, k, generator=g, device="cuda") * gscale).contiguous()
    return W, G


def _resolve_ambiguous_steps(lp, W, G, b, steps, kappa, want):
    """At the ratio steps whose cut-off lies in the float32 band, replace the oracle's value by the
    oracle's delta for the pruned set the GPU chose there (its mask checked against the band rule
    first: the oracle's side for every block outside the band, the exact kept count). Returns the
    ambiguous steps; at most half of the steps may be ambiguous."""
    bn, bk = inputs.block_sides(b)
    Wb, Gh = inputs.bf16_bits(W), G.cpu().numpy()
    exact = oracle.block_scores(Wb, alloc.mean_gradient(Gh), b)
    amb = ambiguous_steps(exact, steps, bn, bk)
    assert len(amb) <= max(2, steps // 2), amb
    g = lp.mean_gradient(G)
    for s in amb:
        mask, _ = lp.taylor_block_mask(W, g, b, s / steps)
        m = mask.cpu().numpy()
        assert_mask_matches_away_from_cutoff(m, exact, s / steps, bn, bk)
        want[s] = alloc.delta_at_mask(Wb, Gh, b, m, kappa)
    return amb


def test_mean_gradient_bit_exact(lp):
    W, G = _wg(384, 256, 13, 70)
    got = lp.mean_gradient(G).cpu().numpy()
    assert np.array_equal(got, alloc.mean_gradient(G.cpu().numpy()))


@pytest.mark.parametrize("n,k,b,N,steps,kappa", [(128, 256, 32, 8, 10, 0.1), (256, 192, (64, 32), 5, 7, 1e-3),
                                                  (96, 128, 16, 33, 16, 0.0), (768, 3072, 32, 8, 20, 0.01),
                                                  (384, 1536, (16, 32), 4, 12, 0.05), (64, 64, 64, 1, 3, 2.0)])
def test_delta_curve_matches_the_oracle(lp, n, k, b, N, steps, kappa):
    bn, bk = inputs.block_sides(b)
    W, G = _wg(n, k, N, 7000 + n + k + N)
    got = lp.delta_curve(W, G, b, steps, kappa).cpu().numpy()
    want = alloc.delta_curve(inputs.bf16_bits(W), G.cpu().numpy(), b, steps, kappa)
    assert got[0] == 0.0
    scale = np.max(np.abs(want))
    assert scale > 0
    _resolve_ambiguous_steps(lp, W, G, b, steps, kappa, want)
    assert np.max(np.abs(got - want)) <= CURVE_TOL * scale, np.max(np.abs(got - want)) / scale


def test_zero_gradients_give_the_kappa_closed_form(lp):
    n, k, b, steps, kappa = 128, 128, 32, 4, 0.5
    W, _ = _wg(n, k, 1, 71)
    G = torch.zeros(3, n, k, device="cuda")
    got = lp.delta_curve(W, G, b, steps, kappa).cpu().numpy()
    Wd = oracle.bf16_to_f64(inputs.bf16_bits(W))
    blocks = [(r, j) for r in range(n // b) for j in range(k // b)]
    for s in range(steps + 1):
        p = oracle.prune_count(s / steps, len(blocks))
        want = 0.5 * kappa * sum(float(np.sum(Wd[r * b:(r + 1) * b, j * b:(j + 1) * b] ** 2))
                                 for r, j in blocks[len(blocks) - p:])
        assert got[s] == pytest.approx(want, rel=1e-12, abs=0)


def test_allocation_feeds_the_masks_and_the_linear(lp):
    """Four DeiT-S-shaped layers: GPU curves -> lambda search -> Taylor masks at the allocated ratios
    (ranked by the mean gradient) -> pack -> linear, each step against the oracle."""
    layers = [("qkv", 384, 1152), ("proj", 384, 384), ("fc1", 384, 1536), ("fc2", 1536, 384)]
    b, N, steps, kappa, beta, R, m = 32, 6, 8, 1e-3, 2e-9, 0.5, 197
    curves, refs, Ws, Gs = [], [], [], []
    for i, (name, k, n) in enumerate(layers):
        W, G = _wg(n, k, N, 7100 + i)
        Ws.append(W)
        Gs.append(G)
        curves.append(lp.delta_curve(W, G, b, steps, kappa).cpu().numpy())
        refs.append(alloc.delta_curve(inputs.bf16_bits(W), G.cpu().numpy(), b, steps, kappa))
        _resolve_ambiguous_steps(lp, W, G, b, steps, kappa, refs[-1])
        assert np.max(np.abs(curves[-1] - refs[-1])) <= CURVE_TOL * np.max(np.abs(refs[-1]))
    F = [m * n * k for _, k, n in layers]
    c = [m * n * k / (b * b) for _, k, n in layers]
    ks, lam, ratio = lp.lambda_search(curves, steps, F, c, beta, R)
    # the search itself, on the GPU's curves, is the oracle's search; and on the oracle's curves
    want = alloc.lambda_search([alloc.distortion(d) for d in curves], steps, F, c, beta, R)
    assert ks == want[1]
    assert ks == alloc.lambda_search([alloc.distortion(d) for d in refs], steps, F, c, beta, R)[1]
    assert ratio <= R
    for i, (name, k, n) in enumerate(layers):
        g = lp.mean_gradient(Gs[i])
        mask, _ = lp.taylor_block_mask(Ws[i], g, b, ks[i] / steps)
        g_ref = alloc.mean_gradient(Gs[i].cpu().numpy())
        exact = oracle.block_scores(inputs.bf16_bits(Ws[i]), g_ref, b)
        got_m = mask.cpu().numpy()
        assert_mask_matches_away_from_cutoff(got_m, exact, ks[i] / steps, b, b)
        X = inputs.activations(m, k, 7200 + i, "cuda")
        w = lp.pack_bsr(Ws[i], mask, b)
        Y = lp.bsr_linear(w, X, None, out_dtype=torch.float32)
        ref = oracle.linear(inputs.bf16_bits(X), inputs.bf16_bits(Ws[i]), got_m, b, None)
        err = np.max(np.abs(Y.cpu().double().numpy() - ref)) / max(np.sqrt(np.mean(ref ** 2)), 1e-30)
        assert err <= 1e-4
