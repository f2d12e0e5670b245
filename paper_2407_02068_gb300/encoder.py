"""An end-to-end pre-norm ViT (DeiT) encoder forward whose linears are block-sparse: the pruned
ViTs of Sec. 4, with the Sec. 3.1 / 3.3 block-sparse layers in place of the dense linears. Every
step runs in liblpvit.so: residual add + LayerNorm, the four block-sparse linears of a block (fc1
with the exact GELU) and multi-head attention. Per layer:

    h = LN1(x);  qkv = h W~qkv^T + b;  a = MHSA(qkv);  x = x + (a W~proj^T + b)
    h = LN2(x);  f = gelu(h W~fc1^T + b);  x = x + (f W~fc2^T + b)

then a final LayerNorm. A residual addition is fused into the LayerNorm that follows it.

``dense_forward`` runs the same model with torch's dense bf16 operations on W (.) M (the
comparator the speedup is measured against; not part of the product path)."""
from __future__ import annotations

import torch

from . import (add_layernorm, alloc_bsr, attention, block_sides, bsr_linear, pack_bsr_many_into,
               workspace_for)

NAMES = ("qkv", "proj", "fc1", "fc2")


class SparseEncoder:
    """layers: per layer a dict with 'ln1', 'ln2' = (gamma, beta) float32 [D] tensors and 'qkv',
    'proj', 'fc1', 'fc2' = (W bf16 [n, k], mask uint8 [n/bn, k/bk], bias float32 [n]); final =
    (gamma, beta). All on one CUDA device; the weights are packed at construction."""

    def __init__(self, layers, final, heads: int, tokens: int, b, eps: float = 1e-6):
        self.heads, self.tokens, self.eps = heads, tokens, eps
        self.bn, self.bk = block_sides(b)
        self.layers, self.final = layers, final
        self.dim = layers[0]["qkv"][0].shape[1] if layers else final[0].numel()
        dev = final[0].device
        self.w: list[dict] = []
        flat_w, flat_W, flat_m = [], [], []
        for L in layers:
            packed = {}
            for name in NAMES:
                W, M, _ = L[name]
                packed[name] = alloc_bsr(W.shape[0], W.shape[1], b, device=dev)
                flat_w.append(packed[name])
                flat_W.append(W.contiguous())
                flat_m.append(M.to(dev).contiguous())
            self.w.append(packed)
        if flat_w:
            pack_bsr_many_into(flat_w, flat_W, flat_m)
        self._bufs = {}

    def _buffers(self, M: int, dev):
        if M not in self._bufs:
            D = self.dim
            hid = self.layers[0]["fc1"][0].shape[0] if self.layers else D
            e = lambda c: torch.empty((M, c), dtype=torch.bfloat16, device=dev)
            ws = {}
            for name in NAMES:
                if self.layers:
                    ws[name] = workspace_for(self.w[0][name], M, dev)
            self._bufs[M] = dict(h=e(D), qkv=e(3 * D), a=e(D), f=e(hid), s0=e(D), s1=e(D),
                                 out=e(D), ws=ws)
        return self._bufs[M]

    def forward(self, x: torch.Tensor, streams: list | None = None) -> torch.Tensor:
        """x: bf16 [images * tokens, D] contiguous CUDA token activations. Returns bf16 [images * tokens, D]
        (a buffer reused by the next call with the same shape). ``streams``: optional list that
        receives a copy of the residual stream after each layer."""
        M = x.shape[0]
        B = self._buffers(M, x.device)
        # the residual stream ping-pongs between s0 and s1 (x itself is never written); proj and fc2
        # add it in their epilogues, so every LayerNorm reads the finished sum
        s_cur, s_next = x, B["s0"]
        for L, W in zip(self.layers, self.w):
            add_layernorm(s_cur, None, *L["ln1"], eps=self.eps, norm_out=B["h"])
            bsr_linear(W["qkv"], B["h"], L["qkv"][2], out=B["qkv"], workspace=B["ws"]["qkv"])
            attention(B["qkv"], self.tokens, self.heads, out=B["a"])
            bsr_linear(W["proj"], B["a"], L["proj"][2], out=s_next, workspace=B["ws"]["proj"], residual=s_cur)
            s_cur, s_next = s_next, (B["s1"] if s_next is B["s0"] else B["s0"])
            add_layernorm(s_cur, None, *L["ln2"], eps=self.eps, norm_out=B["h"])
            bsr_linear(W["fc1"], B["h"], L["fc1"][2], gelu=True, out=B["f"], workspace=B["ws"]["fc1"])
            bsr_linear(W["fc2"], B["f"], L["fc2"][2], out=s_next, workspace=B["ws"]["fc2"], residual=s_cur)
            s_cur, s_next = s_next, (B["s1"] if s_next is B["s0"] else B["s0"])
            if streams is not None:
                streams.append(s_cur.clone())
        add_layernorm(s_cur, None, *self.final, eps=self.eps, norm_out=B["out"])
        return B["out"]

    def launches(self) -> int:
        """Library kernel launches per forward: per layer 2 LayerNorms, 4 linears (proj and fc2 adding
        the residual), 1 attention; plus the final LayerNorm."""
        return 7 * len(self.layers) + 1

    def dense_forward(self, x: torch.Tensor) -> torch.Tensor:
        """The same model with torch's dense bf16 operations on W (.) M (the comparator)."""
        F = torch.nn.functional
        if not hasattr(self, "_dense"):
            self._dense = []
            for L in self.layers:
                d = {}
                for name in NAMES:
                    W, M, bias = L[name]
                    keep = M.to(W.device).repeat_interleave(self.bn, 0).repeat_interleave(self.bk, 1).bool()
                    d[name] = (torch.where(keep, W, torch.zeros_like(W)), bias.to(torch.bfloat16))
                self._dense.append(d)
        D, T, H = self.dim, self.tokens, self.heads
        s = x
        for L, d in zip(self.layers, self._dense):
            h = F.layer_norm(s, (D,), L["ln1"][0].to(torch.bfloat16), L["ln1"][1].to(torch.bfloat16), self.eps)
            qkv = F.linear(h, *d["qkv"]).view(-1, T, 3, H, D // H).permute(2, 0, 3, 1, 4)
            a = F.scaled_dot_product_attention(qkv[0], qkv[1], qkv[2]).permute(0, 2, 1, 3).reshape(-1, D)
            s = s + F.linear(a, *d["proj"])
            h = F.layer_norm(s, (D,), L["ln2"][0].to(torch.bfloat16), L["ln2"][1].to(torch.bfloat16), self.eps)
            s = s + F.linear(F.gelu(F.linear(h, *d["fc1"])), *d["fc2"])
        return F.layer_norm(s, (D,), self.final[0].to(torch.bfloat16), self.final[1].to(torch.bfloat16), self.eps)
