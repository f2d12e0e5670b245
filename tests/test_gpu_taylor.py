"""The block mask of Sec. 3.1 from first-order Taylor scores on the GPU (lpvit_taylor_block_mask)
against the oracle: block scores bit for bit (both take the same float32 operations in the same
order: products, row sums, the sum of the row sums) and masks bit for bit (rank by score, ties to the lower block index, round(alpha * blocks)
eliminated); then the mask drives the pack and the linear."""
import numpy as np
import pytest
import torch

import oracle
from paper_2407_02068_gb300 import inputs

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
def test_scores_and_mask_bit_exact(lp, n, k, b, alpha):
    bn, bk = inputs.block_sides(b)
    W, G = _wg(n, k, 4000 + n + k + (bn if bn == bk else 100 * bn + bk))
    mask, scores = lp.taylor_block_mask(W, G, b, alpha)
    s_ref, m_ref = _oracle(W, G, b, alpha)
    assert scores.shape == (n // bn, k // bk)
    assert np.array_equal(scores.cpu().numpy(), s_ref)
    assert np.array_equal(mask.cpu().numpy(), m_ref)
    assert int(mask.sum()) == (n // bn) * (k // bk) - oracle.prune_count(alpha, (n // bn) * (k // bk))


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
    _, m_ref = _oracle(W, G, b, 0.5)
    ref = oracle.linear(inputs.bf16_bits(X), inputs.bf16_bits(W), m_ref, b, bias.cpu().numpy(), False)
    err = np.max(np.abs(Y.cpu().double().numpy() - ref)) / np.sqrt(np.mean(ref ** 2))
    assert err <= 1e-4 and w.nnzb == int(m_ref.sum())
