"""The block mask of Sec. 3.1 from first-order Taylor scores on the GPU (lpvit_taylor_block_mask)
against the oracle's exact block averages of |W . grad W|:

* scores within the float32 accumulation bound (bn + bk) 2^-24 of the exact average, element by
  element (the kernel sums in float32; see taylor_bounds);
* the mask: the oracle's kept count exactly, the oracle's mask on every block outside the band
  around the cut-off that the score bound leaves open, and exactly the ranking of the definition
  (higher score first, ties to the lower block index, round(alpha * blocks) eliminated) applied to
  the GPU's own scores;
* integer-valued inputs, whose float32 sums are exact, bit for bit;
* then the mask drives the pack and the linear."""
import numpy as np
import pytest
import torch

import oracle
from paper_2407_02068_gb300 import inputs
from taylor_bounds import assert_mask_matches_away_from_cutoff, assert_scores_within_bound

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def lp():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2407_02068_gb300 import build
    build.build()
    import paper_2407_02068_gb300 as lp
    return lp


def _wg(n, k, seed, grad_scale=1e-3):
    W = inputs.weight(n, k, seed, "cuda")
    g = torch.Generator(device="cuda").manual_seed(seed + 1)
    G = torch.randn(n, k, generator=g, device="cuda") * grad_scale
    return W, G.contiguous()


def _oracle(W, G, b, alpha):
    s = oracle.block_scores(inputs.bf16_bits(W), G.cpu().numpy(), b)
    return s, oracle.taylor_mask(s, alpha)


@pytest.mark.parametrize("n,k,b", [(384, 256, 32), (208, 1536, 16), (768, 3072, 64), (3072, 768, 32),
                                   (768, 3072, 32), (1152, 384, 16), (768, 3072, (64, 32)), (384, 1536, (16, 32)),
                                   (192, 320, (32, 16))])
@pytest.mark.parametrize("alpha", [0.0, 0.3, 0.5, 0.8, 1.0])
def test_scores_within_bound_and_mask_away_from_cutoff(lp, n, k, b, alpha):
    bn, bk = inputs.block_sides(b)
    W, G = _wg(n, k, 4000 + n + k + (bn if bn == bk else 100 * bn + bk))
    mask, scores = lp.taylor_block_mask(W, G, b, alpha)
    exact = oracle.block_scores(inputs.bf16_bits(W), G.cpu().numpy(), b)
    got_s, got_m = scores.cpu().numpy(), mask.cpu().numpy()
    assert got_s.shape == (n // bn, k // bk)
    assert_scores_within_bound(got_s, exact, bn, bk)
    assert_mask_matches_away_from_cutoff(got_m, exact, alpha, bn, bk)
    # the selection itself, on the GPU's scores, is the ranking of the definition bit for bit
    assert np.array_equal(got_m, oracle.taylor_mask(got_s, alpha))
    assert int(got_m.sum()) == (n // bn) * (k // bk) - oracle.prune_count(alpha, (n // bn) * (k // bk))


@pytest.mark.parametrize("b", [16, 32, 64])
def test_ties_keep_the_lowest_block_indices(lp, b):
    n, k = 4 * b, 6 * b
    W = torch.ones(n, k, dtype=torch.bfloat16, device="cuda")
    W[::2] = -1
    G = torch.full((n, k), 0.5, device="cuda")
    for alpha in (0.25, 0.5, 0.7):
        mask, scores = lp.taylor_block_mask(W, G, b, alpha)
        assert bool((scores == 0.5).all())
        keep = 24 - oracle.prune_count(alpha, 24)
        assert np.array_equal(mask.cpu().numpy().ravel(), (np.arange(24) < keep).astype(np.uint8))


def test_integer_scores_with_many_ties(lp):
    n, k, b = 512, 512, 16
    gen = torch.Generator(device="cuda").manual_seed(77)
    W = torch.randint(-2, 3, (n, k), generator=gen, device="cuda").to(torch.bfloat16)
    G = torch.randint(-2, 3, (n, k), generator=gen, device="cuda").float()
    for alpha in (0.1, 0.5, 0.9):
        mask, scores = lp.taylor_block_mask(W, G, b, alpha)
        s_ref, m_ref = _oracle(W, G, b, alpha)
        assert np.array_equal(scores.cpu().numpy(), s_ref)
        assert np.array_equal(mask.cpu().numpy(), m_ref)


def test_mask_drives_pack_and_linear(lp):
    m, n, k, b = 300, 768, 768, 32
    W, G = _wg(n, k, 4321)
    mask, _ = lp.taylor_block_mask(W, G, b, 0.5)
    w = lp.pack_bsr(W, mask, b, count=True)
    X = inputs.activations(m, k, 4322, "cuda")
    bias = inputs.bias(n, 4323, "cuda")
    Y = lp.bsr_linear(w, X, bias, out_dtype=torch.float32)
    exact = oracle.block_scores(inputs.bf16_bits(W), G.cpu().numpy(), b)
    got_m = mask.cpu().numpy()
    assert_mask_matches_away_from_cutoff(got_m, exact, 0.5, b, b)
    ref = oracle.linear(inputs.bf16_bits(X), inputs.bf16_bits(W), got_m, b, bias.cpu().numpy(), False)
    err = np.max(np.abs(Y.cpu().double().numpy() - ref)) / np.sqrt(np.mean(ref ** 2))
    assert err <= 1e-4 and w.nnzb == int(got_m.sum())
