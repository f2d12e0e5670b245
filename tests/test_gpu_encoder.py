"""The end-to-end encoder on the GPU against the oracle (oracle/encoder.py): the residual add +
LayerNorm kernel, the attention kernel, and a whole DeiT-S encoder forward with block-sparse
linears. Tolerances follow the arithmetic: LayerNorm outputs within one bf16 ulp plus the float32
statistics' error; attention within the bf16 rounding of the softmax weights (2^-9 relative, times
max |v|) plus one output ulp; the chained encoder (every hand-off rounded to bf16 on both sides, so
differences come from rounding flips that later layers carry) within two ulps of each output plus
2^-7 of rms, and 1% of rms on average."""
import numpy as np
import pytest
import torch

import oracle
from oracle import encoder as oenc
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


def _ulp(x):
    return 2.0 ** (np.floor(np.log2(np.maximum(np.abs(x), 2.0 ** -126))) - 7)


def _b(t):
    return inputs.bf16_bits(t)


@pytest.mark.parametrize("D,rows", [(384, 1000), (768, 777), (64, 5), (1024, 33)])
@pytest.mark.parametrize("with_r", [False, True])
def test_add_layernorm(lp, D, rows, with_r):
    g = torch.Generator(device="cuda").manual_seed(D + rows)
    x = (torch.randn(rows, D, generator=g, device="cuda") * 2 + 0.5).to(torch.bfloat16)
    r = (torch.randn(rows, D, generator=g, device="cuda")).to(torch.bfloat16) if with_r else None
    gamma = (1 + 0.1 * torch.randn(D, generator=g, device="cuda")).contiguous()
    beta = (0.1 * torch.randn(D, generator=g, device="cuda")).contiguous()
    res = lp.add_layernorm(x, r, gamma, beta, 1e-6)
    xd = oracle.bf16_to_f64(_b(x))
    if with_r:
        s, y = res
        exact = xd + oracle.bf16_to_f64(_b(r))
        sd = oracle.bf16_to_f64(_b(s))
        assert np.all(np.abs(sd - exact) <= _ulp(exact) * 0.5 + 1e-300)   # round to nearest of the sum
        src = sd
    else:
        y, src = res, xd
    ref = oenc.layernorm(src, gamma.cpu().double().numpy(), beta.cpu().double().numpy(), 1e-6)
    yd = oracle.bf16_to_f64(_b(y))
    bound = _ulp(ref) + 2.0 ** -16 * (np.abs(ref) + np.abs(beta.cpu().double().numpy()) + 1)
    assert np.all(np.abs(yd - ref) <= bound)


@pytest.mark.parametrize("tokens,heads,images", [(197, 6, 3), (197, 12, 1), (49, 3, 5), (1, 2, 2), (208, 1, 2),
                                                 (16, 4, 1), (33, 2, 2), (128, 3, 2), (129, 2, 3), (177, 1, 2)])
def test_attention(lp, tokens, heads, images):
    g = torch.Generator(device="cuda").manual_seed(tokens * 100 + heads)
    qkv = (torch.randn(images * tokens, 3 * heads * 64, generator=g, device="cuda")).to(torch.bfloat16)
    out = lp.attention(qkv, tokens, heads)
    q = oracle.bf16_to_f64(_b(qkv))
    ref = oenc.attention(q, tokens, heads, 64)
    got = oracle.bf16_to_f64(_b(out))
    D = heads * 64
    vmax = np.abs(q[:, 2 * D:]).max()
    assert np.all(np.abs(got - ref) <= 2.0 ** -8 * vmax + _ulp(ref))


def test_attention_rejects_what_it_does_not_cover(lp):
    qkv = torch.zeros(209 * 2, 3 * 64, dtype=torch.bfloat16, device="cuda")
    with pytest.raises(lp.LpvitError):
        lp.attention(qkv, 209, 1)
    with pytest.raises(lp.LpvitError):
        lp.attention(torch.zeros(10, 3 * 2 * 32, dtype=torch.bfloat16, device="cuda"), 10, 2)   # head_dim 32


def _encoder(D, hidden, heads, L, b, seed, sparsity=0.5):
    gen = torch.Generator(device="cuda").manual_seed(seed)
    bn, bk = inputs.block_sides(b)
    layers = []
    for l in range(L):
        lay = {"ln1": ((1 + 0.1 * torch.randn(D, generator=gen, device="cuda")).contiguous(),
                       (0.1 * torch.randn(D, generator=gen, device="cuda")).contiguous()),
               "ln2": ((1 + 0.1 * torch.randn(D, generator=gen, device="cuda")).contiguous(),
                       (0.1 * torch.randn(D, generator=gen, device="cuda")).contiguous())}
        for t, (name, k, n) in enumerate((("qkv", D, 3 * D), ("proj", D, D), ("fc1", D, hidden), ("fc2", hidden, D))):
            W = inputs.weight(n, k, seed + 10 * l + t, "cuda")
            M = inputs.uniform_mask(n, k, b, sparsity, seed + 100 + 10 * l + t).cuda()
            bias = (0.02 * torch.randn(n, generator=gen, device="cuda")).contiguous()
            lay[name] = (W, M, bias)
        layers.append(lay)
    final = ((1 + 0.1 * torch.randn(D, generator=gen, device="cuda")).contiguous(),
             (0.1 * torch.randn(D, generator=gen, device="cuda")).contiguous())
    return layers, final


def _oracle_layers(layers, final, b):
    ol = []
    for L in layers:
        d = {"ln1": tuple(v.cpu().double().numpy() for v in L["ln1"]),
             "ln2": tuple(v.cpu().double().numpy() for v in L["ln2"])}
        for name in ("qkv", "proj", "fc1", "fc2"):
            W, M, bias = L[name]
            d[name] = (_b(W), M.cpu().numpy(), bias.cpu().numpy(), b)
        ol.append(d)
    return ol, tuple(v.cpu().double().numpy() for v in final)


@pytest.mark.parametrize("b", [32, (16, 32)])
def test_deit_s_encoder_forward(lp, b):
    from paper_2407_02068_gb300.encoder import SparseEncoder
    D, hidden, heads, T, L, images = 384, 1536, 6, 197, 2, 2
    layers, final = _encoder(D, hidden, heads, L, b, 900)
    enc = SparseEncoder(layers, final, heads, T, b)
    x = inputs.activations(images * T, D, 901, "cuda")
    y = enc.forward(x)
    ol, of = _oracle_layers(layers, final, b)
    ref = oracle.bf16_to_f64(oenc.encoder_forward(_b(x), ol, of, T, heads))
    got = oracle.bf16_to_f64(_b(y))
    rms = np.sqrt(np.mean(ref ** 2))
    err = np.abs(got - ref)
    # a hand-off whose exact value lies within the accumulation error of a bf16 rounding boundary can
    # round differently on the two sides: one ulp there, carried (and normalised) by later layers
    assert np.all(err <= 2 * _ulp(ref) + 2.0 ** -7 * rms), np.max(err / (_ulp(ref) + 1e-30))
    assert err.mean() <= 0.01 * rms, err.mean() / rms
    # the dense torch comparator computes the same model
    yd = enc.dense_forward(x).float().cpu().double().numpy()
    assert np.abs(yd - ref).mean() <= 0.02 * rms


def test_deit_b_encoder_at_the_timed_configuration(lp):
    """The configuration `bench.py --encoder deit_b` times: DeiT-B, 12 layers, 256 images of 197
    tokens (M = 50432: its token tiles, slicing and attention grid), 32x32 blocks at the stack's
    per-GEMM sparsities. Images are independent, so the oracle runs each sampled image alone: the
    first, the last and four seeded others. Layer by layer, the oracle layer applied to the GPU's
    input stream of that layer must give the GPU's output stream under the DeiT-S gate; the final
    LayerNorm likewise. Over all 12 layers the hand-off roundings compound (a value within the
    accumulation error of a bf16 boundary rounds differently on the two sides, and later layers
    carry that ulp), so end to end only the mean error is gated."""
    from paper_2407_02068_gb300.encoder import SparseEncoder
    model, b, config, images, T = inputs.DEIT_B, 32, 9, 256, 197
    D, heads = model["dim"], model["dim"] // 64
    layers, final = inputs.deit_encoder_params(model, b, config, 12, "cuda")
    enc = SparseEncoder(layers, final, heads, T, b)
    x = inputs.activations(images * T, D, inputs.seed(config, 0, "X"), "cuda")
    streams = []
    y = enc.forward(x, streams)
    torch.cuda.synchronize()
    assert len(streams) == 12
    ol, of = _oracle_layers(layers, final, b)
    rng = np.random.default_rng(20240702)
    sample = sorted({0, images - 1, *rng.choice(np.arange(1, images - 1), size=4, replace=False).tolist()})
    sb = [_b(x)] + [_b(st) for st in streams]
    yb = _b(y)

    def gate(got_bits, ref_bits, what):
        ref, got = oracle.bf16_to_f64(ref_bits), oracle.bf16_to_f64(got_bits)
        rms = np.sqrt(np.mean(ref ** 2))
        err = np.abs(got - ref)
        assert np.all(err <= 2 * _ulp(ref) + 2.0 ** -7 * rms), (what, float(np.max(err / (_ulp(ref) + 1e-30))))
        assert err.mean() <= 0.01 * rms, (what, err.mean() / rms)

    for img in sample:
        rows = slice(img * T, (img + 1) * T)
        for li in range(12):
            gate(sb[li + 1][rows], oenc.layer_forward(sb[li][rows], ol[li], T, heads), (img, li))
        gate(yb[rows], oenc.encoder_forward(sb[12][rows], [], of, T, heads), (img, "final LayerNorm"))
        ref = oracle.bf16_to_f64(oenc.encoder_forward(sb[0][rows], ol, of, T, heads))
        got = oracle.bf16_to_f64(yb[rows])
        assert np.abs(got - ref).mean() <= 0.01 * np.sqrt(np.mean(ref ** 2)), img
