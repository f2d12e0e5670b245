"""Pins for the CPU oracle: each test checks it against something other than itself
(hand-worked values, textbook tables, numpy/torch library products, closed forms and
invariants), so that a dropped term, a wrong index or sign, or a transposed operand in the
oracle fails at least one of them."""
import math
import os

import numpy as np
import pytest
import torch

import oracle
from paper_2407_02068_gb300 import inputs

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _read_golden(name):
    """Parse 'key dims...' headers followed by rows of numbers."""
    sections, key, dims, rows = {}, None, None, []
    with open(os.path.join(GOLDEN, name)) as f:
        for line in f:
            line = line.split("#", 1)[0].strip()
            if not line:
                continue
            tok = line.split()
            if tok[0].isalpha() or "_" in tok[0]:
                if key is not None:
                    sections[key] = np.array(rows, dtype=np.float64).reshape(dims) if dims else rows
                key, dims, rows = tok[0], tuple(int(t) for t in tok[1:]), []
                if key == "b":
                    sections["b"] = int(tok[1])
                    key = None
                continue
            rows.extend(float(t) for t in tok)
        if key is not None:
            sections[key] = np.array(rows, dtype=np.float64).reshape(dims)
    return sections


def _bits(a):
    """float array -> bf16 bits (all golden values are exactly representable)."""
    t = torch.tensor(np.asarray(a, dtype=np.float32)).to(torch.bfloat16)
    bits = inputs.bf16_bits(t)
    assert np.array_equal(oracle.bf16_to_f64(bits), np.asarray(a, dtype=np.float64))
    return bits


def _expand(mask, b):
    bn, bk = oracle.block_shape(b)
    return np.kron(mask.astype(np.float64), np.ones((bn, bk)))


def _rand_case(rng, m, n, k, b, density=0.5, int_valued=False):
    if int_valued:
        X = rng.integers(-4, 5, size=(m, k)).astype(np.float32)
        W = (rng.integers(-4, 5, size=(n, k)) / 16.0).astype(np.float32)
        bias = (rng.integers(-8, 9, size=n) / 8.0).astype(np.float32)
    else:
        X = rng.standard_normal((m, k)).astype(np.float32)
        W = (0.02 * rng.standard_normal((n, k))).astype(np.float32)
        bias = (0.02 * rng.standard_normal(n)).astype(np.float32)
    Xb = inputs.bf16_bits(torch.tensor(X).to(torch.bfloat16))
    Wb = inputs.bf16_bits(torch.tensor(W).to(torch.bfloat16))
    bn, bk = oracle.block_shape(b)
    mask = (rng.random((n // bn, k // bk)) < density).astype(np.uint8)
    return Xb, Wb, mask, bias


# --------------------------------------------------------------------------- golden example

def test_golden_tiny_linear_and_pack():
    g = _read_golden("tiny_block_linear.txt")
    b = g["b"]
    Wb, Xb = _bits(g["W"]), _bits(g["X"])
    mask = g["mask"].astype(np.uint8)
    bias = g["bias"].astype(np.float32)
    Y = oracle.linear(Xb, Wb, mask, b, bias)
    assert np.array_equal(Y, g["Y"])
    row_ptr, col_idx, blocks = oracle.pack(Wb, mask, b)
    assert row_ptr.tolist() == g["row_ptr"].astype(int).tolist()
    assert col_idx.tolist() == g["col_idx"].astype(int).tolist()
    assert np.array_equal(oracle.bf16_to_f64(blocks), g["blocks"])


def test_golden_gelu_against_normal_cdf_table():
    tab = np.loadtxt(os.path.join(GOLDEN, "normal_cdf.txt"))
    x, phi = tab[:, 0], tab[:, 1]
    got = oracle.gelu(x)
    # relative accuracy everywhere, the far negative tail included (Phi(-6) ~ 1e-9)
    assert np.allclose(got, x * phi, rtol=1e-12, atol=0)
    # the tanh approximation misses by ~1.5e-4 at y=1: a swapped form fails here
    tanh_form = 0.5 * x * (1 + np.tanh(math.sqrt(2 / math.pi) * (x + 0.044715 * x ** 3)))
    assert abs(tanh_form[1] - got[1]) > 1e-5
    assert oracle.gelu(0.0) == 0.0


def test_gelu_matches_scipy_ndtr():
    sp = pytest.importorskip("scipy.special")
    y = np.linspace(-8, 8, 1001)
    assert np.allclose(oracle.gelu(y), y * sp.ndtr(y), rtol=1e-12, atol=0)
    # far tail: Phi(-z) = phi(z) M(z), M from scipy's scaled erfc, down to |GELU| ~ 1e-300
    z = np.linspace(8, 37, 300)
    tail = -z * np.exp(-z * z / 2) / np.sqrt(2 * np.pi) * np.sqrt(np.pi / 2) * sp.erfcx(z / np.sqrt(2))
    assert np.allclose(oracle.gelu(-z), tail, rtol=1e-11, atol=0)
    assert np.all(np.diff(oracle.gelu(np.linspace(0, 8, 100))) > 0)  # monotone for y > 0


# --------------------------------------------------------------------------- brute force

@pytest.mark.parametrize("m,n,k,b", [(3, 8, 12, 4), (5, 32, 16, 8), (8, 64, 32, 16), (4, 32, 64, 32), (2, 6, 4, 2),
                                     (4, 128, 64, (64, 32)), (3, 32, 96, (16, 32)), (2, 12, 8, (3, 2)),
                                     (3, 64, 64, (32, 16))])
def test_linear_matches_numpy_dense_masked_product(m, n, k, b):
    rng = np.random.default_rng(1000 + m * 7 + n)
    Xb, Wb, mask, bias = _rand_case(rng, m, n, k, b)
    X, W = oracle.bf16_to_f64(Xb), oracle.bf16_to_f64(Wb)
    ref = X @ (W * _expand(mask, b)).T + bias.astype(np.float64)
    got = oracle.linear(Xb, Wb, mask, b, bias)
    assert np.allclose(got, ref, rtol=1e-12, atol=1e-12 * np.abs(ref).max())
    got_g = oracle.linear(Xb, Wb, mask, b, bias, gelu=True)
    sp = pytest.importorskip("scipy.special")
    assert np.allclose(got_g, ref * sp.ndtr(ref), rtol=1e-12, atol=1e-14)


def test_non_square_mask_orientation():
    """mask[n/b][k/b] indexes (output panel, input block); transposing it must change the result."""
    rng = np.random.default_rng(7)
    m, n, k, b = 4, 16, 48, 8
    Xb, Wb, mask, bias = _rand_case(rng, m, n, k, b, density=0.5)
    X, W = oracle.bf16_to_f64(Xb), oracle.bf16_to_f64(Wb)
    ref = X @ (W * _expand(mask, b)).T + bias
    assert np.allclose(oracle.linear(Xb, Wb, mask, b, bias), ref, rtol=1e-12, atol=1e-14)


def test_non_square_blocks_are_rows_by_columns():
    """A (bn, bk) block is bn output rows by bk input columns: one kept block at (r, j) lets exactly
    W[r*bn:(r+1)*bn, j*bk:(j+1)*bk] through, and swapping the sides gives a different layer."""
    rng = np.random.default_rng(11)
    m, n, k = 3, 64, 64
    Xb, Wb, _, bias = _rand_case(rng, m, n, k, 8)
    X, W = oracle.bf16_to_f64(Xb), oracle.bf16_to_f64(Wb)
    mask = np.zeros((n // 32, k // 16), np.uint8)
    mask[1, 2] = 1
    got = oracle.linear(Xb, Wb, mask, (32, 16), None)
    want = np.zeros((m, n))
    want[:, 32:64] = X[:, 32:48] @ W[32:64, 32:48].T
    assert np.allclose(got, want, rtol=1e-13, atol=1e-15)
    mask2 = np.zeros((n // 16, k // 32), np.uint8)  # the sides swapped: rows 32..47, columns 32..63
    mask2[2, 1] = 1
    swapped = oracle.linear(Xb, Wb, mask2, (16, 32), None)
    want2 = np.zeros((m, n))
    want2[:, 32:48] = X[:, 32:64] @ W[32:48, 32:64].T
    assert np.allclose(swapped, want2, rtol=1e-13, atol=1e-15)
    assert not np.allclose(got, swapped)
    with pytest.raises(ValueError):
        oracle.linear(Xb, Wb, mask, (16, 32), None)  # mask shape is for (32, 16) blocks


def test_zero_sparsity_equals_dense_torch_matmul_on_config_shapes():
    for (k, n) in [(384, 1152), (1536, 384), (768, 3072), (3072, 768)]:
        Xb = inputs.bf16_bits(inputs.activations(4, k, 11 + k))
        Wb = inputs.bf16_bits(inputs.weight(n, k, 12 + n))
        bias = inputs.bias(n, 13).numpy()
        mask = np.ones((n // 32, k // 32), dtype=np.uint8)
        got = oracle.linear(Xb, Wb, mask, 32, bias)
        X = torch.from_numpy(oracle.bf16_to_f64(Xb))
        W = torch.from_numpy(oracle.bf16_to_f64(Wb))
        ref = (X @ W.T + torch.from_numpy(bias.astype(np.float64))).numpy()
        assert np.allclose(got, ref, rtol=1e-12, atol=1e-12)


def test_all_zero_mask_gives_bias_exactly():
    rng = np.random.default_rng(3)
    Xb, Wb, _, bias = _rand_case(rng, 5, 64, 64, 16)
    mask = np.zeros((4, 4), dtype=np.uint8)
    got = oracle.linear(Xb, Wb, mask, 16, bias)
    assert np.array_equal(got, np.broadcast_to(bias.astype(np.float64), got.shape))
    got_g = oracle.linear(Xb, Wb, mask, 16, bias, gelu=True)
    assert np.array_equal(got_g, np.broadcast_to(oracle.gelu(bias.astype(np.float64)), got.shape))
    assert np.array_equal(oracle.linear(Xb, Wb, mask, 16, None), np.zeros((5, 64)))


def test_pruned_blocks_are_never_read():
    rng = np.random.default_rng(4)
    Xb, Wb, mask, bias = _rand_case(rng, 6, 64, 96, 16)
    poisoned = Wb.copy()
    keep = np.kron(mask, np.ones((16, 16), dtype=np.uint8)).astype(bool)
    poisoned[~keep] = np.uint16(0x7FC0)  # NaN
    poisoned[~keep & (np.arange(96)[None, :] % 3 == 0)] = np.uint16(0x7F80)  # +Inf
    zeros = Wb.copy()
    zeros[~keep] = 0
    a = oracle.linear(Xb, poisoned, mask, 16, bias)
    c = oracle.linear(Xb, zeros, mask, 16, bias)
    assert np.array_equal(a, c) and np.isfinite(a).all()


def test_single_block_closed_form():
    rng = np.random.default_rng(5)
    m, n, k, b = 7, 64, 128, 32
    Xb, Wb, _, bias = _rand_case(rng, m, n, k, b)
    mask = np.zeros((n // b, k // b), dtype=np.uint8)
    r, j = 1, 2
    mask[r, j] = 1
    got = oracle.linear(Xb, Wb, mask, b, bias)
    X, W = oracle.bf16_to_f64(Xb), oracle.bf16_to_f64(Wb)
    expect = np.broadcast_to(bias.astype(np.float64), (m, n)).copy()
    expect[:, r * b:(r + 1) * b] += X[:, j * b:(j + 1) * b] @ W[r * b:(r + 1) * b, j * b:(j + 1) * b].T
    assert np.allclose(got, expect, rtol=1e-13, atol=1e-15)


def test_integer_mode_is_exact_and_permutation_invariant():
    """Small dyadic inputs: every product and partial sum is exact, so the result is exact in
    any order; permuting k-block columns of X, W and the mask together leaves it unchanged."""
    rng = np.random.default_rng(6)
    m, n, k, b = 9, 64, 256, 16
    Xb, Wb, mask, bias = _rand_case(rng, m, n, k, b, int_valued=True)
    X, W = oracle.bf16_to_f64(Xb), oracle.bf16_to_f64(Wb)
    got = oracle.linear(Xb, Wb, mask, b, bias)
    exact = X @ (W * _expand(mask, b)).T + bias
    assert np.array_equal(got, exact)
    perm = rng.permutation(k // b)
    cols = np.concatenate([np.arange(p * b, (p + 1) * b) for p in perm])
    got_p = oracle.linear(np.ascontiguousarray(Xb[:, cols]), np.ascontiguousarray(Wb[:, cols]),
                          np.ascontiguousarray(mask[:, perm]), b, bias)
    assert np.array_equal(got, got_p)


def test_thread_count_does_not_change_bits():
    rng = np.random.default_rng(8)
    Xb, Wb, mask, bias = _rand_case(rng, 37, 64, 64, 16)
    a = oracle.linear(Xb, Wb, mask, 16, bias, nthreads=1)
    c = oracle.linear(Xb, Wb, mask, 16, bias, nthreads=5)
    assert np.array_equal(a, c)


def test_row_strided_input_view():
    rng = np.random.default_rng(9)
    Xb, Wb, mask, bias = _rand_case(rng, 6, 32, 32, 16)
    wide = np.zeros((6, 96), dtype=np.uint16)
    wide[:, 64:96] = Xb
    assert np.array_equal(oracle.linear(wide[:, 64:96], Wb, mask, 16, bias), oracle.linear(Xb, Wb, mask, 16, bias))


# --------------------------------------------------------------------------- pack

@pytest.mark.parametrize("n,k,b", [(128, 64, (64, 32)), (64, 96, (16, 32)), (48, 32, (8, 16)), (64, 32, 16), (96, 192, 32), (128, 64, 64), (32, 32, 16)])
def test_pack_invariants_and_round_trip(n, k, b):
    rng = np.random.default_rng(n + k + sum(oracle.block_shape(b)))
    _, Wb, mask, _ = _rand_case(rng, 1, n, k, b, density=0.45)
    mask[0, :] = 0  # an empty panel
    bn, bk = oracle.block_shape(b)
    row_ptr, col_idx, blocks = oracle.pack(Wb, mask, b)
    assert blocks.shape[1:] == (bn, bk)
    assert row_ptr[0] == 0 and np.all(np.diff(row_ptr) >= 0)
    assert row_ptr[-1] == int(mask.astype(bool).sum()) == len(col_idx)
    for r in range(n // bn):
        cs = col_idx[row_ptr[r]:row_ptr[r + 1]]
        assert np.all(np.diff(cs) > 0)
        assert cs.tolist() == np.nonzero(mask[r])[0].tolist()
    # unpack(pack(W, M)) == W (.) expand(M), bitwise
    un = np.zeros_like(Wb)
    for r in range(n // bn):
        for t in range(row_ptr[r], row_ptr[r + 1]):
            j = col_idx[t]
            un[r * bn:(r + 1) * bn, j * bk:(j + 1) * bk] = blocks[t]
    keep = np.kron(mask, np.ones((bn, bk), dtype=np.uint8)).astype(bool)
    assert np.array_equal(un, np.where(keep, Wb, 0))


def test_pack_empty_matrix():
    Wb = np.ones((32, 64), dtype=np.uint16)
    row_ptr, col_idx, blocks = oracle.pack(Wb, np.zeros((2, 4), np.uint8), 16)
    assert row_ptr.tolist() == [0, 0, 0] and len(col_idx) == 0 and len(blocks) == 0


# --------------------------------------------------------------------------- bf16 rounding

def test_round_bf16_ties_and_specials():
    r = oracle.round_bf16_scalar
    assert r(1.0) == 0x3F80
    assert r(1.0 + 2.0 ** -8) == 0x3F80                # tie -> even (1.0)
    assert r(1.0 + 3 * 2.0 ** -8) == 0x3F82            # tie -> even (1 + 2^-6)
    assert r(1.0 + 2.0 ** -8 + 2.0 ** -30) == 0x3F81   # above the tie -> up
    assert r(-2.5) == 0xC020
    assert r(0.0) == 0x0000 and r(-0.0) == 0x8000
    assert r(float("inf")) == 0x7F80 and r(float("-inf")) == 0xFF80
    assert r(3.4e38) == 0x7F80                         # above bf16 max + half ulp -> inf
    assert r(2.0 ** -133) == 0x0001                    # smallest subnormal
    assert r(2.0 ** -134) == 0x0000                    # tie -> even (zero)


def test_round_bf16_matches_torch_on_float32_values():
    g = torch.Generator().manual_seed(0)
    x = torch.cat([torch.randn(20000, generator=g) * 10.0 ** torch.randint(-30, 30, (20000,), generator=g),
                   torch.randn(1000, generator=g) * 1e-39])
    want = inputs.bf16_bits(x.to(torch.bfloat16))
    got = oracle.round_bf16(x.double().numpy())
    assert np.array_equal(got, want)


# --------------------------------------------------------------------------- stack

def test_deit_stack_rows_is_row_independent_chain():
    """Rows of the stack are independent: the stack on a subset equals the subset of the stack."""
    rng = np.random.default_rng(10)
    d, h, b = 32, 64, 16
    layers = []
    for _ in range(2):
        L = {}
        for name, k, n in [("qkv", d, 3 * d), ("proj", d, d), ("fc1", d, h), ("fc2", h, d)]:
            _, Wb, mask, bias = _rand_case(rng, 1, n, k, b)
            L[name] = (Wb, mask, bias, b)
        layers.append(L)
    h0 = inputs.bf16_bits(torch.randn(6, d).to(torch.bfloat16))
    full = oracle.deit_stack_rows(h0, layers)
    part = oracle.deit_stack_rows(h0[[1, 4]], layers)
    assert np.array_equal(full[[1, 4]], part)
    # first layer by hand from the library product
    W, M, bias, _ = layers[0]["qkv"]
    X = oracle.bf16_to_f64(h0)
    qkv = X @ (oracle.bf16_to_f64(W) * _expand(M, b)).T + bias
    assert np.array_equal(oracle.round_bf16(oracle.linear(h0, W, M, b, bias)),
                          oracle.round_bf16(qkv)) or np.allclose(qkv, oracle.linear(h0, W, M, b, bias))


# ------------------------------------------------------------- block mask from Taylor scores

def _golden_taylor():
    rows = [l.split() for l in open(os.path.join(GOLDEN, "taylor_mask_tiny.txt")) if l.strip() and not l.startswith("#")]
    W = np.array([float(v) for v in rows[0][1:]], dtype=np.float32).reshape(4, 4)
    G = np.array([float(v) for v in rows[1][1:]], dtype=np.float32).reshape(4, 4)
    scores = np.array([float(v) for v in rows[2][1:]]).reshape(2, 2)
    cases = [(float(r[1]), int(r[2]), np.array([int(v) for v in r[3:]], dtype=np.uint8).reshape(2, 2)) for r in rows[3:]]
    return W, G, scores, cases


def _bits(a):
    """bf16 bits of a float32 array (round to nearest even, as the inputs module rounds)."""
    return inputs.bf16_bits(torch.from_numpy(np.ascontiguousarray(a, dtype=np.float32)).to(torch.bfloat16))


def test_taylor_scores_and_masks_match_the_hand_worked_example():
    W, G, scores, cases = _golden_taylor()
    got = oracle.block_scores(_bits(W), G, 2)
    assert np.array_equal(got, scores)
    for alpha, pruned, mask in cases:
        assert oracle.prune_count(alpha, 4) == pruned
        assert np.array_equal(oracle.taylor_mask(got, alpha), mask), alpha


def test_taylor_mask_equal_scores_keep_the_lowest_indices():
    s = np.full((3, 5), 0.75)
    for alpha in (0.2, 0.4, 0.6, 0.8):
        keep = 15 - oracle.prune_count(alpha, 15)
        assert np.array_equal(oracle.taylor_mask(s, alpha).ravel(), (np.arange(15) < keep).astype(np.uint8))


def test_taylor_scores_are_local_and_scale_exactly():
    rng = np.random.default_rng(5)
    W = (rng.standard_normal((64, 96)) * 0.02).astype(np.float32)
    G = (rng.standard_normal((64, 96)) * 1e-3).astype(np.float32)
    Wb = _bits(W)
    s = oracle.block_scores(Wb, G, 32)
    # a power-of-two factor on the gradient scales every score exactly and keeps the mask
    s4 = oracle.block_scores(Wb, G * np.float32(4.0), 32)
    assert np.array_equal(s4, 4.0 * s)
    assert np.array_equal(oracle.taylor_mask(s4, 0.5), oracle.taylor_mask(s, 0.5))
    # changing one block changes only that block's score
    G2 = G.copy()
    G2[32:64, 0:32] *= 3
    s2 = oracle.block_scores(Wb, G2, 32)
    changed = s2 != s
    assert changed[1, 0] and changed.sum() == 1


def test_taylor_scores_are_the_exact_block_average():
    """One 2 x 32 block: one product of 1 and 63 products of 2^-25. The exact average is
    (1 + 63 * 2^-25) / 64, representable in double; a float32 accumulation (any order that adds the
    small products to 1 one at a time, or row by row) loses some or all of the 2^-25 terms."""
    W = np.full((2, 32), 2.0 ** -8, dtype=np.float32)
    W[0, 0] = 1.0
    G = np.full((2, 32), 2.0 ** -17, dtype=np.float32)
    G[0, 0] = 1.0
    s = oracle.block_scores(_bits(W), G, (2, 32))
    assert s[0, 0] == (1.0 + 63 * 2.0 ** -25) / 64
    assert s[0, 0] != (1.0 + 2.0 ** -20) / 64   # row sums in float32, then their sum
    assert s[0, 0] != 1.0 / 64                  # one float32 sum over the block


def test_taylor_scores_ignore_the_sign_of_each_product():
    """|W . G| element by element, not |sum|: a block whose products cancel still scores their
    magnitudes (the hand-worked block (1,1) of the golden file, here on a 16 x 16 block)."""
    W = np.ones((16, 16), dtype=np.float32)
    W[::2] = -1.0
    G = np.full((16, 16), 0.5, dtype=np.float32)
    s = oracle.block_scores(_bits(W), G, 16)
    assert s[0, 0] == 0.5


def test_taylor_scores_brute_force_and_mask_order():
    rng = np.random.default_rng(6)
    for b in (16, 32, (64, 32), (16, 32)):
        bn, bk = oracle.block_shape(b)
        W = (rng.standard_normal((4 * bn, 3 * bk)) * 0.02).astype(np.float32)
        G = rng.standard_normal((4 * bn, 3 * bk)).astype(np.float32)
        Wb = _bits(W)
        Wd = oracle.bf16_to_f64(Wb)
        want = np.abs(Wd * G.astype(np.float64)).reshape(4, bn, 3, bk).sum(axis=(1, 3)) / (bn * bk)
        s = oracle.block_scores(Wb, G, b)
        # the same average by numpy's pairwise double sum: only the summation order differs
        assert np.allclose(s, want, rtol=1e-13, atol=0)
        for alpha in (0.0, 0.25, 0.5, 0.75, 1.0):
            m = oracle.taylor_mask(s, alpha)
            kept, pruned = s[m == 1], s[m == 0]
            assert m.sum() == 12 - oracle.prune_count(alpha, 12)
            if kept.size and pruned.size:
                assert kept.min() >= pruned.max()
