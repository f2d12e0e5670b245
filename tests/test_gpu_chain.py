"""GPU parity of the chain entry point (lpvit_bsr_linear_chain): consecutive linears in one
persistent launch give the same bits as separate lpvit_bsr_linear[_gelu] calls, and the chained
DeiT stack matches the fp64 oracle chain on sampled token rows.

The chain orders the linears by per-(linear, 256-token tile) counters instead of launch
boundaries, so the cases cover: several tiles with a ragged last one, groups of 256 features with a
partial last group (n = 1152), non-square blocks, a linear whose mask keeps nothing (its units load
no X and wait in the epilogue), more linears than one launch takes (48), and the host's fallbacks
(m <= 256, split units, overlaps that are not row for row), where links run on their own."""
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
    import paper_2407_02068_gb300 as lp
    from paper_2407_02068_gb300 import build
    build.build()
    return lp


def _layers(nl, d, b, seed, empty=()):
    """nl DeiT layers (qkv, proj, fc1 + GELU, fc2) at width d with seeded weights, biases and uniform
    masks of sparsity 0.3 .. 0.7; (layer, name) in ``empty`` gets a mask that keeps nothing."""
    g = torch.Generator().manual_seed(seed)
    shapes = {"qkv": (3 * d, d), "proj": (d, d), "fc1": (4 * d, d), "fc2": (d, 4 * d)}
    out = []
    for li in range(nl):
        L = {}
        for gi, (name, (n, k)) in enumerate(shapes.items()):
            W = (torch.randn(n, k, generator=g) * 0.05).to(torch.bfloat16)
            bias = torch.randn(n, generator=g) * 0.05
            sp = 0.3 + 0.4 * ((li * 4 + gi) % 5) / 4
            mask = inputs.uniform_mask(n, k, b, sp, seed + 17 * li + gi)
            if (li, name) in empty:
                mask = torch.zeros_like(mask)
            L[name] = {"W": W.cuda(), "bias": bias.cuda(), "mask": mask.cuda(), "gelu": name == "fc1"}
        out.append(L)
    return out


def _packed(lp, layers, b):
    for L in layers:
        for G in L.values():
            G["w"] = lp.pack_bsr(G["W"], G["mask"], b)
    return layers


def _buffers(m, d):
    bf = torch.bfloat16
    return {"qkv": torch.empty(m, 3 * d, dtype=bf, device="cuda"),
            "proj": torch.empty(m, d, dtype=bf, device="cuda"),
            "fc1": torch.empty(m, 4 * d, dtype=bf, device="cuda"),
            "h": [torch.empty(m, d, dtype=bf, device="cuda") for _ in range(2)]}


def _steps(layers, h0, B, d):
    """The stack's (w, X, bias, out, gelu) sequence: proj reads the last third of qkv's columns."""
    steps, src = [], h0
    for li, L in enumerate(layers):
        steps.append((L["qkv"]["w"], src, L["qkv"]["bias"], B["qkv"], False))
        steps.append((L["proj"]["w"], B["qkv"][:, 2 * d:], L["proj"]["bias"], B["proj"], False))
        steps.append((L["fc1"]["w"], B["proj"], L["fc1"]["bias"], B["fc1"], True))
        src = B["h"][li % 2]
        steps.append((L["fc2"]["w"], B["fc1"], L["fc2"]["bias"], src, False))
    return steps, src


def _separate(lp, steps):
    for w, X, bias, out, gelu in steps:
        lp.bsr_linear(w, X, bias, gelu=gelu, out=out)


def _run_both(lp, layers, m, d, seed):
    h0 = inputs.activations(m, d, seed, "cuda")
    A, B = _buffers(m, d), _buffers(m, d)
    sa, outa = _steps(layers, h0, A, d)
    sb, outb = _steps(layers, h0, B, d)
    _separate(lp, sa)
    ws = torch.zeros(64 << 20, dtype=torch.uint8, device="cuda")
    lp.bsr_linear_chain(sb, workspace=ws)
    lp.check(ws)
    torch.cuda.synchronize()
    return h0, A, B, outa, outb, ws


def _same(A, B):
    for key in ("qkv", "proj", "fc1"):
        assert torch.equal(A[key], B[key]), key
    for i in range(2):
        assert torch.equal(A["h"][i], B["h"][i]), ("h", i)


@pytest.mark.parametrize("d,b,m", [(384, 16, 5000), (384, (16, 32), 5000), (768, 32, 3500), (768, (64, 32), 3500)])
def test_chain_equals_separate_calls(lp, d, b, m):
    layers = _packed(lp, _layers(2, d, b, 41), b)
    _, A, B, _, _, _ = _run_both(lp, layers, m, d, 43)
    _same(A, B)


def _ulp_bf16(x):
    return 2.0 ** (np.floor(np.log2(np.maximum(np.abs(x), 2.0 ** -126))) - 7)


@pytest.mark.parametrize("d,b,m", [(384, 16, 5000), (768, 32, 3500)])
def test_chained_linears_match_oracle(lp, d, b, m):
    """Each linear of the chain's last layer against the fp64 oracle on its own bf16 input (the
    chain's buffers after the call), on sampled token rows in several tiles: one bf16 ulp of the exact
    value plus the float32 accumulation bound k 2^-24 sum|x w~| (+|bias|), x1.13 under GELU."""
    layers = _packed(lp, _layers(2, d, b, 51), b)
    _, _, B, _, _, _ = _run_both(lp, layers, m, d, 53)
    rows = np.unique(np.concatenate([np.random.default_rng(2).choice(m, 12, replace=False),
                                     [0, 255, 256, m - 1]]))
    ri = torch.from_numpy(rows).cuda()
    L = layers[1]
    for name, X, out in (("qkv", B["h"][0], B["qkv"]), ("proj", B["qkv"][:, 2 * d:], B["proj"]),
                         ("fc1", B["proj"], B["fc1"]), ("fc2", B["fc1"], B["h"][1])):
        G = L[name]
        Xs = X[ri]
        mask = G["mask"].cpu().numpy()
        ref = oracle.linear(inputs.bf16_bits(Xs), inputs.bf16_bits(G["W"]), mask, b, G["bias"].cpu().numpy(),
                            G["gelu"])
        got = oracle.bf16_to_f64(inputs.bf16_bits(out[ri]))
        bn, bk = inputs.block_sides(b)
        keep = G["mask"].repeat_interleave(bn, 0).repeat_interleave(bk, 1).bool()
        Wa = torch.where(keep, G["W"], torch.zeros_like(G["W"])).double().abs().cpu()
        acc = (G["W"].shape[1] * 2.0 ** -24 * (Xs.double().abs().cpu() @ Wa.T + G["bias"].double().abs().cpu())).numpy()
        tol = _ulp_bf16(ref) + (1.13 * acc + 4 * 2.0 ** -23 * np.abs(ref) if G["gelu"] else acc)
        assert np.all(np.abs(got - ref) <= tol), (name, float(np.max(np.abs(got - ref) - tol)))


def test_chain_with_a_linear_that_keeps_nothing(lp):
    """proj of layer 0 and fc2 of layer 1 keep no block: their units load nothing and wait for the
    previous linear in the epilogue; the last output is then the bf16 bias of layer 1's fc2."""
    d, b, m = 384, 16, 5000
    layers = _packed(lp, _layers(2, d, b, 61, empty={(0, "proj"), (1, "fc2")}), b)
    _, A, B, _, _, _ = _run_both(lp, layers, m, d, 63)
    _same(A, B)
    bias = layers[1]["fc2"]["bias"].to(torch.bfloat16)
    assert torch.equal(B["h"][1], bias.expand(m, d))


def test_chain_repeats_and_leaves_its_workspace_clear(lp):
    """Three calls on one workspace give the same bits; afterwards every counter (queue, tiles, the
    CTA count) is back at zero, so the whole workspace reads zero."""
    d, b, m = 768, 32, 3500
    layers = _packed(lp, _layers(1, d, b, 71), b)
    h0 = inputs.activations(m, d, 73, "cuda")
    B = _buffers(m, d)
    steps, out = _steps(layers, h0, B, d)
    ws = torch.zeros(1 << 20, dtype=torch.uint8, device="cuda")
    runs = []
    for _ in range(3):
        lp.bsr_linear_chain(steps, workspace=ws)
        lp.check(ws)
        runs.append(out.clone())
    assert torch.equal(runs[0], runs[1]) and torch.equal(runs[0], runs[2])
    torch.cuda.synchronize()
    assert int(torch.count_nonzero(ws)) == 0
    # a workspace smaller than lpvit_chain_workspace_bytes is refused before anything runs
    from paper_2407_02068_gb300 import _lib
    rows = [(w.struct(), X.data_ptr(), X.stride(0), bias.data_ptr(), o.data_ptr(), o.stride(0), int(g))
            for w, X, bias, o, g in steps]
    links = _lib.chain_links(rows)
    need = _lib.lpvit_chain_workspace_bytes(links, len(rows), m)
    assert need > 256
    assert _lib.lpvit_bsr_linear_chain(links, len(rows), m, ws.data_ptr(), need - 256, 0) == _lib.LPVIT_ERR_WORKSPACE


def test_chain_longer_than_one_launch(lp):
    """13 layers = 52 linears: a launch of 48, then one of 4."""
    d, b, m = 384, 16, 5000
    layers = _packed(lp, _layers(13, d, b, 81), b)
    _, A, B, _, _, _ = _run_both(lp, layers, m, d, 83)
    _same(A, B)


@pytest.mark.parametrize("m", [197, 1000])   # every link on its own: the small-m kernel; split units
def test_chain_fallback_sizes(lp, m):
    d, b = 384, 16
    layers = _packed(lp, _layers(2, d, b, 91), b)
    _, A, B, _, _, _ = _run_both(lp, layers, m, d, 93)
    _same(A, B)


def test_chain_overlap_not_row_for_row_runs_apart(lp):
    """Link 2 reads link 1's output through another row stride (row r of its X is half of output
    row r / 2): the host starts a new launch there, and the result equals separate calls."""
    d, b, m = 768, 32, 3500
    layers = _packed(lp, _layers(1, d, b, 101), b)
    G1, G2 = layers[0]["proj"], layers[0]["fc2"]
    w2 = lp.pack_bsr(G2["W"][:, :384].contiguous(), G2["mask"][:, :384 // 32].contiguous(), b)
    h0 = inputs.activations(m, d, 103, "cuda")
    res = []
    for chained in (False, True):
        buf = torch.empty(m * d, dtype=torch.bfloat16, device="cuda")
        y1 = buf.view(m, d)
        x2 = buf[: m * 384].view(m, 384)
        y2 = torch.empty(m, d, dtype=torch.bfloat16, device="cuda")
        steps = [(G1["w"], h0, G1["bias"], y1, False), (w2, x2, G2["bias"], y2, True)]
        if chained:
            lp.bsr_linear_chain(steps)
        else:
            _separate(lp, steps)
        torch.cuda.synchronize()
        res.append((y1.clone(), y2.clone()))
    assert torch.equal(res[0][0], res[1][0]) and torch.equal(res[0][1], res[1][1])
