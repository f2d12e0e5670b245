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


@pytest.mark.parametrize("n,k,b,alpha", [(384, 256, 32, 0.5), (768, 3072, 32, 0.3), (1152, 384, 16, 0.6),
                                         (768, 3072, (64, 32), 0.615), (384, 1536, (16, 32), 0.287),
                                         (256, 512, 64, 1.0), (256, 512, 32, 0.0)])
def test_fused_taylor_pack_matches_mask_then_pack(lp, n, k, b, alpha):
    """lpvit_taylor_pack_bsr (mask and pack in one call, no host step) gives bit for bit the scores,
    mask, BSR arrays and work list of lpvit_taylor_block_mask followed by lpvit_pack_bsr; its mask
    agrees with the oracle's away from the cut-off and its pack with the oracle's pack of that mask;
    a linear on it matches the oracle."""
    bn, bk = inputs.block_sides(b)
    W, G = _wg(n, k, 6100 + n + k + (bn if bn == bk else 100 * bn + bk))
    wf, mf, sf = lp.taylor_pack_bsr(W, G, b, alpha, count=True)
    ms, ss = lp.taylor_block_mask(W, G, b, alpha)
    ws = lp.pack_bsr(W, ms, b, count=True)
    torch.cuda.synchronize()
    assert torch.equal(sf.view(torch.int64), ss.view(torch.int64)) and torch.equal(mf, ms)
    assert wf.nnzb == ws.nnzb and torch.equal(wf.row_ptr, ws.row_ptr)
    assert torch.equal(wf.col_idx[:wf.nnzb], ws.col_idx[:ws.nnzb])
    assert torch.equal(wf.blocks[:wf.nnzb].view(torch.int16), ws.blocks[:ws.nnzb].view(torch.int16))
    hdr = wf.sched[:64].view(torch.int32).cpu().numpy()
    ng, kc = int(hdr[1]), -(-k // 64)
    table_end = 4 * (16 + ng + 1 + 16 * ng)              # header, group pointers, group table
    ent0 = 4 * ((16 + ng + 1 + 16 * ng + 3) // 4 * 4)   # entries (after padding to 16 bytes)
    ent_end = ent0 + 4 * int(hdr[2])
    stream = (4 * ((16 + ng + 1 + 16 * ng + 3) // 4 * 4 + ng * kc) + 1023) // 1024 * 1024
    used = stream + int(hdr[2]) * 256 * 64 * 2
    assert torch.equal(wf.sched[:table_end], ws.sched[:table_end])
    assert torch.equal(wf.sched[ent0:ent_end], ws.sched[ent0:ent_end])
    assert torch.equal(wf.sched[stream:used], ws.sched[stream:used])
    exact = oracle.block_scores(inputs.bf16_bits(W), G.cpu().numpy(), b)
    got_m = mf.cpu().numpy()
    assert_mask_matches_away_from_cutoff(got_m, exact, alpha, bn, bk)
    rp, ci, bl = oracle.pack(inputs.bf16_bits(W), got_m, b)
    assert np.array_equal(wf.row_ptr.cpu().numpy(), rp) and np.array_equal(wf.col_idx[:wf.nnzb].cpu().numpy(), ci)
    assert np.array_equal(wf.blocks[:wf.nnzb].contiguous().view(torch.int16).cpu().numpy().view(np.uint16), bl)
    X = inputs.activations(197, k, 6200 + n, "cuda")
    bias = inputs.bias(n, 6300 + n, "cuda")
    Y = lp.bsr_linear(wf, X, bias, out_dtype=torch.float32)
    ref = oracle.linear(inputs.bf16_bits(X), inputs.bf16_bits(W), got_m, b, bias.cpu().numpy())
    err = np.max(np.abs(Y.cpu().double().numpy() - ref)) / max(np.sqrt(np.mean(ref ** 2)), 1e-30)
    assert err <= 1e-4
