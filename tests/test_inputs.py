"""Host checks of the seeded input recipe (mask counts, Zipf water-fill, stack sparsities)."""
import numpy as np
import pytest

from paper_2407_02068_gb300 import inputs


@pytest.mark.parametrize("n,k,b,s", [(1152, 384, 32, 0.5), (384, 1536, 16, 0.3), (3072, 768, 32, 0.8),
                                     (768, 3072, 32, 0.0), (64, 64, 16, 1.0)])
def test_uniform_mask_exact_count_and_seeded(n, k, b, s):
    m1 = inputs.uniform_mask(n, k, b, s, 123)
    m2 = inputs.uniform_mask(n, k, b, s, 123)
    total = (n // b) * (k // b)
    assert m1.shape == (n // b, k // b) and m1.dtype.is_floating_point is False
    assert int((m1 == 0).sum()) == inputs.round_half_away(s * total)
    assert bool((m1 == m2).all())


def test_round_half_away():
    assert inputs.round_half_away(2.5) == 3 and inputs.round_half_away(-2.5) == -3
    assert inputs.round_half_away(2.4999) == 2


@pytest.mark.parametrize("n,k,b", [(3072, 768, 16), (768, 3072, 64), (3072, 768, 64), (768, 3072, 16)])
def test_zipf_counts_waterfill(n, k, b):
    P, kb = n // b, k // b
    T = inputs.round_half_away(0.4 * P * kb)
    c = inputs.zipf_counts(P, kb, T, 1.2, 77)
    assert sum(c) == T and max(c) <= kb and min(c) >= 0
    mask = inputs.zipf_mask(n, k, b, 0.6, 77)
    assert mask.sum(dim=1).tolist() == c
    # heavier-ranked panels never get fewer blocks than lighter ones (up to the +1 remainder)
    import torch
    g = torch.Generator(); g.manual_seed(77)
    ranks = (torch.randperm(P, generator=g) + 1).tolist()
    order = sorted(range(P), key=lambda i: ranks[i])
    assert all(c[order[i]] + 1 >= c[order[i + 1]] for i in range(P - 1))


def test_zipf_cap_binds_for_fc2_b64():
    c = inputs.zipf_counts(12, 48, inputs.round_half_away(0.4 * 12 * 48), 1.2, 5)
    assert max(c) == 48


def test_stack_sparsities_antithetic_mean():
    sp = np.array(inputs.stack_sparsities(4))
    assert sp.shape == (12, 4)
    assert np.all((sp >= 0.3) & (sp <= 0.7))
    assert np.allclose(sp.mean(axis=0), 0.5, atol=1e-15)
    assert np.allclose(sp[0::2] + sp[1::2], 1.0, atol=1e-15)
