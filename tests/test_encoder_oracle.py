"""Pins for the encoder oracle (oracle/encoder.py): LayerNorm and multi-head attention against
torch's float64 library routines and closed forms, and the encoder's independence across images."""
import numpy as np
import pytest
import torch

import oracle
from oracle import encoder
from paper_2407_02068_gb300 import inputs


def test_layernorm_closed_forms_and_library():
    g, b = np.ones(2), np.zeros(2)
    assert np.allclose(encoder.layernorm(np.array([[1.0, 3.0]]), g, b, 0.0), [[-1.0, 1.0]], atol=0)
    assert np.array_equal(encoder.layernorm(np.full((1, 8), 5.0), np.ones(8), np.arange(8.0), 1e-6),
                          np.arange(8.0)[None])                       # constant row -> beta
    rng = np.random.default_rng(0)
    x = rng.standard_normal((7, 384)) * 3 + 1
    gamma, beta = rng.standard_normal(384), rng.standard_normal(384)
    ref = torch.nn.functional.layer_norm(torch.tensor(x), (384,), torch.tensor(gamma), torch.tensor(beta), 1e-6)
    assert np.allclose(encoder.layernorm(x, gamma, beta, 1e-6), ref.numpy(), rtol=1e-12, atol=1e-12)
    # shift and scale invariance of the normalised part
    assert np.allclose(encoder.layernorm(4 * x + 9, gamma, beta, 0.0), encoder.layernorm(x, gamma, beta, 0.0),
                       rtol=1e-10, atol=1e-10)


def test_attention_closed_forms_and_library():
    T, H, d = 5, 2, 4
    rng = np.random.default_rng(1)
    v = rng.standard_normal((T, H * d))
    qkv = np.concatenate([np.zeros((T, H * d)), np.ones((T, H * d)), v], axis=1)  # equal scores
    out = encoder.attention(qkv, T, H, d)
    assert np.allclose(out, np.tile(v.mean(axis=0), (T, 1)), atol=1e-14)     # uniform weights
    q = np.zeros((T, H * d)); q[:, 0] = 100.0
    k = np.zeros((T, H * d)); k[3, 0] = 1.0
    out = encoder.attention(np.concatenate([q, k, v], axis=1), T, H, d)
    assert np.allclose(out[:, :d], np.tile(v[3, :d], (T, 1)), atol=1e-12)    # head 0 picks key 3
    # against torch's scaled dot-product attention in float64, 3 images of 197 tokens, 6 heads
    T, H, d, B = 197, 6, 64, 3
    qkv = rng.standard_normal((B * T, 3 * H * d))
    got = encoder.attention(qkv, T, H, d)
    t = torch.tensor(qkv).view(B, T, 3, H, d).permute(2, 0, 3, 1, 4)
    ref = torch.nn.functional.scaled_dot_product_attention(t[0], t[1], t[2])
    ref = ref.permute(0, 2, 1, 3).reshape(B * T, H * d).numpy()
    assert np.allclose(got, ref, rtol=1e-11, atol=1e-12)


def _tiny_encoder(D, hidden, heads, L, b, seed):
    rng = np.random.default_rng(seed)
    layers = []
    for l in range(L):
        lay = {"ln1": (1 + 0.1 * rng.standard_normal(D), 0.1 * rng.standard_normal(D)),
               "ln2": (1 + 0.1 * rng.standard_normal(D), 0.1 * rng.standard_normal(D))}
        for name, k, n in (("qkv", D, 3 * D), ("proj", D, D), ("fc1", D, hidden), ("fc2", hidden, D)):
            W = (rng.standard_normal((n, k)) * 0.05).astype(np.float32)
            Wb = inputs.bf16_bits(torch.from_numpy(W).to(torch.bfloat16))
            mask = (rng.random((n // b, k // b)) < 0.6).astype(np.uint8)
            bias = (0.02 * rng.standard_normal(n)).astype(np.float32)
            lay[name] = (Wb, mask, bias, b)
        layers.append(lay)
    final = (np.ones(D), np.zeros(D))
    return layers, final


def test_encoder_images_are_independent():
    D, hidden, heads, T, L, b = 64, 128, 2, 9, 2, 16
    layers, final = _tiny_encoder(D, hidden, heads, L, b, 3)
    rng = np.random.default_rng(4)
    x = inputs.bf16_bits(torch.from_numpy(rng.standard_normal((3 * T, D)).astype(np.float32)).to(torch.bfloat16))
    both = encoder.encoder_forward(x, layers, final, T, heads)
    for i in range(3):
        one = encoder.encoder_forward(x[i * T:(i + 1) * T], layers, final, T, heads)
        assert np.array_equal(both[i * T:(i + 1) * T], one)
    # permuting the tokens of an image permutes its outputs (attention has no position terms here)
    perm = np.random.default_rng(5).permutation(T)
    out_p = encoder.encoder_forward(x[:T][perm], layers, final, T, heads)
    assert np.array_equal(out_p, both[:T][perm])


def test_encoder_with_no_layers_is_the_final_layernorm():
    D, T = 32, 4
    x = inputs.bf16_bits(torch.randn(T, D).to(torch.bfloat16))
    g, bta = np.linspace(0.5, 1.5, D), np.linspace(-1, 1, D)
    out = encoder.encoder_forward(x, [], (g, bta), T, 2)
    assert np.array_equal(out, oracle.round_bf16(encoder.layernorm(oracle.bf16_to_f64(x), g, bta, 1e-6)))
