"""Seeded synthetic inputs for the block-sparse DeiT linears.

This module draws random numbers and nothing else: it holds none of the layer's arithmetic,
and both the CUDA path and the CPU oracle consume what it produces (the oracle never imports
the CUDA path and vice versa).

The paper's workloads are ImageNet DeiT activations and pretrained weights; none are
available, so these draws stand in with the same shapes:

* tokens M = batch * 197 (224x224 image, 16x16 patches, plus the class token);
* X ~ N(0, 1), W ~ N(0, 0.02), bias ~ N(0, 0.02), drawn in float32; X and W rounded to bf16
  (round to nearest even, done by torch's float32 -> bfloat16 conversion);
* block masks (nonzero = kept):
  - ``uniform_mask``: exactly round(s * nblocks) blocks pruned (ties away from zero),
    chosen by a seeded permutation of all blocks -- not a Bernoulli draw;
  - ``zipf_mask``: kept blocks per row panel follow Zipf(1.2) over a seeded rank order,
    water-filled under the cap of K/b blocks per panel;
  - ``stack_sparsities``: per-GEMM sparsities for the 12-layer stack, drawn U[0.30, 0.70] and
    given as antithetic pairs (s, 1-s) to layers 2j and 2j+1 so that the mean is exactly 50%.

Seeds: ``seed(config, gemm, what)`` = 20240702 + 1000*config + 10*gemm + what, with
what in {X: 0, W: 1, bias: 2, mask: 3, sparsity: 4}.
"""
from __future__ import annotations

import math

import numpy as np
import torch

BASE_SEED = 20240702
WHAT = {"X": 0, "W": 1, "bias": 2, "mask": 3, "sparsity": 4}

DEIT_S = {"dim": 384, "hidden": 1536}
DEIT_B = {"dim": 768, "hidden": 3072}
TOKENS_PER_IMAGE = 197


def seed(config: int, gemm: int, what: str) -> int:
    return BASE_SEED + 1000 * config + 10 * gemm + WHAT[what]


def _gen(s: int, device="cpu") -> torch.Generator:
    g = torch.Generator(device=device)
    g.manual_seed(s)
    return g


def round_half_away(x: float) -> int:
    return int(math.floor(abs(x) + 0.5)) * (1 if x >= 0 else -1)


def activations(m: int, k: int, s: int, device="cpu") -> torch.Tensor:
    """X ~ N(0,1) [m, k] as bf16 (float32 draw rounded to nearest even)."""
    return torch.randn(m, k, generator=_gen(s, device), device=device, dtype=torch.float32).to(torch.bfloat16)


def weight(n: int, k: int, s: int, device="cpu") -> torch.Tensor:
    """W ~ N(0, 0.02) [n, k] (out x in) as bf16."""
    w = torch.randn(n, k, generator=_gen(s, device), device=device, dtype=torch.float32) * 0.02
    return w.to(torch.bfloat16)


def bias(n: int, s: int, device="cpu") -> torch.Tensor:
    """bias ~ N(0, 0.02) [n] as float32."""
    return torch.randn(n, generator=_gen(s, device), device=device, dtype=torch.float32) * 0.02


def block_sides(b) -> tuple[int, int]:
    """A block given as b (b x b) or (bn, bk): bn output rows by bk input columns."""
    return (int(b[0]), int(b[1])) if isinstance(b, (tuple, list)) else (int(b), int(b))


def uniform_mask(n: int, k: int, b, sparsity: float, s: int) -> torch.Tensor:
    """[n/bn, k/bk] uint8 mask with exactly round(sparsity * nblocks) zero (pruned) blocks
    (b = int or (bn, bk))."""
    bn, bk = block_sides(b)
    nb, kb = n // bn, k // bk
    total = nb * kb
    npruned = min(total, max(0, round_half_away(sparsity * total)))
    perm = torch.randperm(total, generator=_gen(s))
    m = torch.ones(total, dtype=torch.uint8)
    m[perm[:npruned]] = 0
    return m.view(nb, kb)


def zipf_counts(panels: int, kb: int, keep_total: int, exponent: float, s: int) -> list[int]:
    """Kept blocks per panel: weights rank^-exponent over a seeded rank permutation, water-filled
    to ``keep_total`` under the cap ``kb``; the integer remainder goes to the largest fractional
    parts first (ties to the lower panel index)."""
    g = _gen(s)
    ranks = (torch.randperm(panels, generator=g) + 1).tolist()
    w = [float(r) ** (-exponent) for r in ranks]
    keep_total = min(keep_total, panels * kb)
    capped = [False] * panels
    ideal = [0.0] * panels
    while True:
        rem = keep_total - kb * sum(capped)
        wsum = sum(w[i] for i in range(panels) if not capped[i])
        changed = False
        for i in range(panels):
            if capped[i]:
                ideal[i] = float(kb)
                continue
            ideal[i] = rem * w[i] / wsum if wsum > 0 else 0.0
            if ideal[i] >= kb:
                capped[i] = True
                changed = True
        if not changed:
            break
    counts = [kb if capped[i] else int(math.floor(ideal[i])) for i in range(panels)]
    left = keep_total - sum(counts)
    order = sorted((i for i in range(panels) if not capped[i]), key=lambda i: (-(ideal[i] - counts[i]), i))
    for i in order[:left]:
        counts[i] += 1
    return counts


def zipf_mask(n: int, k: int, b, sparsity: float, s: int, exponent: float = 1.2) -> torch.Tensor:
    """[n/bn, k/bk] uint8 mask whose per-panel kept-block counts follow ``zipf_counts``; each panel's
    kept columns are a seeded random subset."""
    bn, bk = block_sides(b)
    nb, kb = n // bn, k // bk
    keep_total = round_half_away((1.0 - sparsity) * nb * kb)
    counts = zipf_counts(nb, kb, keep_total, exponent, s)
    g = _gen(s + 7919)
    m = torch.zeros(nb, kb, dtype=torch.uint8)
    for r in range(nb):
        cols = torch.randperm(kb, generator=g)[: counts[r]]
        m[r, cols] = 1
    return m


def stack_sparsities(config: int, layers: int = 12, types: int = 4, lo: float = 0.30, hi: float = 0.70):
    """sp[layer][type]: U[lo, hi] draws, antithetic over layer pairs (2j, 2j+1)."""
    g = _gen(seed(config, 0, "sparsity"))
    draws = (lo + (hi - lo) * torch.rand(types, layers // 2, generator=g, dtype=torch.float64)).tolist()
    sp = [[0.0] * types for _ in range(layers)]
    for t in range(types):
        for j in range(layers // 2):
            sp[2 * j][t] = draws[t][j]
            sp[2 * j + 1][t] = 1.0 - draws[t][j]
    return sp


def bf16_bits(t: torch.Tensor) -> np.ndarray:
    """The raw uint16 bit patterns of a bf16 tensor (on the host)."""
    assert t.dtype == torch.bfloat16
    return t.detach().cpu().contiguous().view(torch.int16).numpy().view(np.uint16)


# ---------------------------------------------------------------------------------------------
# Named workloads (the shapes of the paper's DeiT-S / DeiT-B linears)
# ---------------------------------------------------------------------------------------------

def deit_gemms(model: dict):
    """(name, K_in, N_out, gelu) for one encoder layer's linears."""
    d, h = model["dim"], model["hidden"]
    return [("qkv", d, 3 * d, False), ("proj", d, d, False), ("fc1", d, h, True), ("fc2", h, d, False)]


def make_gemm(config: int, gemm: int, m: int, k: int, n: int, b, sparsity: float, mask_kind="uniform",
              device="cpu", with_x: bool = True):
    """One seeded block-sparse linear: dict with X (bf16 [m,k] or None), W (bf16 [n,k]),
    bias (fp32 [n]) and mask (uint8 [n/bn, k/bk]); b = int (square) or (bn, bk)."""
    out = {
        "W": weight(n, k, seed(config, gemm, "W"), device),
        "bias": bias(n, seed(config, gemm, "bias"), device),
        "b": b, "m": m, "k": k, "n": n, "sparsity": sparsity,
    }
    if mask_kind == "uniform":
        out["mask"] = uniform_mask(n, k, b, sparsity, seed(config, gemm, "mask"))
    elif mask_kind == "zipf":
        out["mask"] = zipf_mask(n, k, b, sparsity, seed(config, gemm, "mask"))
    else:
        raise ValueError(mask_kind)
    out["X"] = activations(m, k, seed(config, gemm, "X"), device) if with_x else None
    return out


def deit_b_stack(config: int = 4, b: int = 32, device="cpu"):
    """The 12-layer DeiT-B linear stack: per layer dict of qkv/proj/fc1/fc2 gemms (no X),
    sparsities from ``stack_sparsities``."""
    sp = stack_sparsities(config)
    layers = []
    for l in range(12):
        L = {}
        for t, (name, k, n, gelu) in enumerate(deit_gemms(DEIT_B)):
            gi = 4 * l + t
            g = make_gemm(config, gi, 0, k, n, b, sp[l][t], device=device, with_x=False)
            g["gelu"] = gelu
            L[name] = g
        layers.append(L)
    return layers


def deit_encoder_params(model: dict, b=32, config: int = 9, layers: int = 12, device="cpu"):
    """Seeded parameters of a pre-norm DeiT encoder with block-sparse linears: per layer a dict with
    'ln1', 'ln2' = (gamma ~ 1 + N(0, 0.1), beta ~ N(0, 0.1)) float32 [D] and 'qkv', 'proj', 'fc1',
    'fc2' = (W bf16 [n, k], uniform mask uint8 [n/bn, k/bk] at the stack's per-GEMM sparsities,
    bias float32 [n]); plus the final LayerNorm's (gamma, beta)."""
    D = model["dim"]
    sp = stack_sparsities(config, layers)
    gen = _gen(seed(config, 0, "bias"), device)
    out = []
    for l in range(layers):
        lay = {"ln1": ((1 + 0.1 * torch.randn(D, generator=gen, device=device)).contiguous(),
                       (0.1 * torch.randn(D, generator=gen, device=device)).contiguous()),
               "ln2": ((1 + 0.1 * torch.randn(D, generator=gen, device=device)).contiguous(),
                       (0.1 * torch.randn(D, generator=gen, device=device)).contiguous())}
        for t, (name, k, n, _) in enumerate(deit_gemms(model)):
            gi = 4 * l + t
            lay[name] = (weight(n, k, seed(config, gi, "W"), device),
                         uniform_mask(n, k, b, sp[l][t], seed(config, gi, "mask")).to(device),
                         bias(n, seed(config, gi, "bias"), device))
        out.append(lay)
    final = ((1 + 0.1 * torch.randn(D, generator=gen, device=device)).contiguous(),
             (0.1 * torch.randn(D, generator=gen, device=device)).contiguous())
    return out, final
