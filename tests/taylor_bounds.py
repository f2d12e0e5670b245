"""Comparison rules for block Taylor scores (Sec. 3.1) computed in float32 against the oracle's
exact block averages.

A float32 score takes bn * bk products of a bf16 weight and a float32 gradient (each rounded once)
and adds their magnitudes in float32, in two levels of at most bk and bn terms. For sums of
non-negative terms every rounding is relative to the partial sum, so the result is within
(1 + u)^(bn + bk - 1) - 1 < (bn + bk) u of the exact average, u = 2^-24 (the final division by
bn * bk in double adds less than 2^-53). Blocks whose exact score lies that close to the cut-off of
the ranking may fall on either side of it; every other block has one correct side.
"""
import numpy as np

import oracle


def score_rel_bound(bn: int, bk: int) -> float:
    return (bn + bk) * 2.0 ** -24


def assert_scores_within_bound(got: np.ndarray, exact: np.ndarray, bn: int, bk: int):
    rel = score_rel_bound(bn, bk)
    err = np.abs(np.asarray(got, dtype=np.float64) - exact)
    bad = err > rel * exact
    assert not bad.any(), (int(bad.sum()), float(np.max(err / np.maximum(exact, 1e-300))), rel)


def ambiguous_blocks(exact: np.ndarray, alpha: float, bn: int, bk: int) -> np.ndarray:
    """Boolean array of exact.shape: the blocks whose side of the cut-off at pruning ratio alpha a
    float32 score within the bound may change (ties at the cut included)."""
    flat = np.asarray(exact, dtype=np.float64).ravel()
    count = flat.size
    keep = count - oracle.prune_count(alpha, count)
    amb = np.zeros(count, dtype=bool)
    if keep == 0 or keep == count:
        return amb.reshape(np.shape(exact))
    order = np.lexsort((np.arange(count), -flat))  # the ranking: higher score first, then lower index
    cut_hi = flat[order[keep - 1]]  # lowest kept score
    cut_lo = flat[order[keep]]      # highest pruned score
    e = score_rel_bound(bn, bk)
    kept = np.zeros(count, dtype=bool)
    kept[order[:keep]] = True
    amb |= kept & (flat * (1 - e) <= cut_lo * (1 + e))
    amb |= ~kept & (flat * (1 + e) >= cut_hi * (1 - e))
    return amb.reshape(np.shape(exact))


def assert_mask_matches_away_from_cutoff(mask: np.ndarray, exact: np.ndarray, alpha: float, bn: int, bk: int,
                                         max_ambiguous: int | None = None):
    """The mask keeps exactly the oracle's count, agrees with the oracle's mask on every block
    outside the cut-off band, and the band holds at most max_ambiguous blocks (default: 1% of the
    blocks, at least 2)."""
    mask = np.asarray(mask)
    want = oracle.taylor_mask(exact, alpha)
    amb = ambiguous_blocks(exact, alpha, bn, bk)
    count = want.size
    if max_ambiguous is None:
        max_ambiguous = max(2, count // 100)
    assert int(amb.sum()) <= max_ambiguous, (int(amb.sum()), count)
    assert int(mask.sum()) == int(want.sum())
    assert np.array_equal(mask[~amb], want[~amb])


def ambiguous_steps(exact: np.ndarray, steps: int, bn: int, bk: int) -> list[int]:
    """Ratio steps k (alpha = k / steps) whose pruned set a float32 score may change."""
    return [s for s in range(steps + 1) if ambiguous_blocks(exact, s / steps, bn, bk).any()]
