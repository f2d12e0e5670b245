"""The DeiT linear stack on the block-sparse library: L encoder layers x (qkv, proj, fc1+GELU, fc2),
each a pruned linear (Sec. 3.1) run as a block-sparse matmul (Sec. 3.3).

One ``step`` is one pass of the whole block-sparse path over one batch: every weight is packed
(mask -> BSR + work list, all weights in one batched call) and every linear runs, chained layer to
layer on one stream:

    qkv  = X~qkv(h)                     [M, 3D]
    proj = X~proj(qkv[:, 2D:3D])        the V third stands in for the attention output
    fc1  = gelu(X~fc1(proj))            [M, 4D]
    h    = X~fc2(fc1)                   [M, D]

Attention, LayerNorm and residuals are not part of this path. All buffers are allocated once;
a step allocates nothing, so it can be captured in a CUDA graph. The C entry points are called
through pre-marshalled ctypes argument lists to keep host overhead per call at a few microseconds.
The linears run either as one library call each or, with ``chain=True``, as one chain call
(lpvit_bsr_linear_chain: the 48 linears in one persistent launch, each token tile of a linear
starting once the previous linear has stored it); both give the same bits.
"""
from __future__ import annotations

import ctypes

import torch

from . import _lib
from . import alloc_bsr, inputs


class DeitLinearStack:
    def __init__(self, m: int, layers, device="cuda"):
        """``layers``: list of dicts name -> {W, bias, mask, b, gelu} (see inputs.deit_b_stack)."""
        self.m = m
        self.device = device
        self.layers = layers
        lib = _lib.load()
        self._pack_fn = lib.lpvit_pack_bsr
        self._pack_many_fn = lib.lpvit_pack_bsr_many
        self._lin = {False: lib.lpvit_bsr_linear, True: lib.lpvit_bsr_linear_gelu}
        self._chain_fn = lib.lpvit_bsr_linear_chain
        d = layers[0]["qkv"]["W"].shape[1]
        h = layers[0]["fc1"]["W"].shape[0]
        self.d, self.h = d, h
        bf = torch.bfloat16
        self.h_in = torch.empty(m, d, dtype=bf, device=device)
        self.qkv = torch.empty(m, 3 * d, dtype=bf, device=device)
        self.proj = torch.empty(m, d, dtype=bf, device=device)
        self.fc1 = torch.empty(m, h, dtype=bf, device=device)
        self.hbuf = [torch.empty(m, d, dtype=bf, device=device) for _ in range(2)]
        self.gemms = []  # (name, layer, W, mask, bias, gelu, BsrWeight)
        for li, L in enumerate(layers):
            for name in ("qkv", "proj", "fc1", "fc2"):
                g = L[name]
                W = g["W"].to(device).contiguous()
                mask = g["mask"].to(device=device, dtype=torch.uint8).contiguous()
                bias = g["bias"].to(device).contiguous()
                w = alloc_bsr(W.shape[0], W.shape[1], g["b"], device=device)
                self.gemms.append({"name": name, "layer": li, "W": W, "mask": mask, "bias": bias,
                                   "gelu": bool(g["gelu"]), "w": w, "struct": w.struct(),
                                   "nnzb": int((g["mask"] != 0).sum())})
        ws_bytes = max(_lib.lpvit_workspace_bytes(G["struct"], m) for G in self.gemms)
        sizing = _lib.chain_links([(G["struct"], 0, 0, 0, 0, 0, 0) for G in self.gemms])
        ws_bytes = max(ws_bytes, _lib.lpvit_chain_workspace_bytes(sizing, len(self.gemms), m))
        self.ws = torch.zeros(max(ws_bytes, 256), dtype=torch.uint8, device=device)
        self._calls = None

    # ------------------------------------------------------------------ accounting
    def effective_flops(self, rows: int | None = None) -> int:
        """2 * rows * sum over GEMMs of (kept blocks) * bn * bk (bias and GELU not counted)."""
        r = self.m if rows is None else rows
        return sum(2 * r * G["nnzb"] * G["w"].bn * G["w"].bk for G in self.gemms)

    def algorithmic_bytes(self) -> int:
        """Per step of the linears: X read once, Y written once (bf16), kept blocks + indices + bias."""
        tot = 0
        for G in self.gemms:
            n, k, bn, bk = G["w"].n, G["w"].k, G["w"].bn, G["w"].bk
            tot += 2 * self.m * k + 2 * self.m * n + 2 * G["nnzb"] * bn * bk + 4 * G["nnzb"] + 4 * (n // bn + 1) + 4 * n
        return tot

    def launches_per_step(self, chain: bool = False) -> int:
        """Kernel launches of one step: one per linear (or one per 48 linears of a chain call), two per
        batched pack of up to 96 weights."""
        n = len(self.gemms)
        return ((n + 47) // 48 if chain else n) + 2 * ((n + 95) // 96)

    # ------------------------------------------------------------------ launches
    def _build_calls(self, stream: int):
        V = ctypes.c_void_p
        calls = []
        n = len(self.gemms)
        self._pack_many_args = (ctypes.c_int32(n), (V * n)(*[G["W"].data_ptr() for G in self.gemms]),
                                (V * n)(*[G["mask"].data_ptr() for G in self.gemms]),
                                (_lib.lpvit_bsr * n)(*[G["struct"] for G in self.gemms]), V(stream))
        ws = V(self.ws.data_ptr())
        wsn = ctypes.c_size_t(self.ws.numel())
        st = V(stream)
        src = self.h_in
        links = []
        for gi, G in enumerate(self.gemms):
            pack_args = (V(G["W"].data_ptr()), V(G["mask"].data_ptr()), ctypes.byref(G["struct"]), None, st)
            name = G["name"]
            if name == "qkv":
                X, ldx, Y = src, src.stride(0), self.qkv
            elif name == "proj":
                X, ldx, Y = self.qkv[:, 2 * self.d:], self.qkv.stride(0), self.proj
            elif name == "fc1":
                X, ldx, Y = self.proj, self.proj.stride(0), self.fc1
            else:
                X, ldx, Y = self.fc1, self.fc1.stride(0), self.hbuf[G["layer"] % 2]
                src = Y
            lin_args = (ctypes.byref(G["struct"]), V(X.data_ptr()), ctypes.c_int64(self.m), ctypes.c_int64(ldx),
                        V(G["bias"].data_ptr()), V(Y.data_ptr()), ctypes.c_int64(Y.stride(0)),
                        ctypes.c_int(_lib.LPVIT_BF16), ws, wsn, st)
            calls.append((pack_args, self._lin[G["gelu"]], lin_args))
            links.append((G["struct"], X.data_ptr(), ldx, G["bias"].data_ptr(), Y.data_ptr(), Y.stride(0), G["gelu"]))
        self.out = src
        arr = _lib.chain_links(links)
        self._chain_args = (arr, ctypes.c_int32(len(links)), ctypes.c_int64(self.m), ws, wsn, st)
        return calls

    def _calls_for(self, stream: int):
        if self._calls is None or self._calls[0] != stream:
            self._calls = (stream, self._build_calls(stream))
        return self._calls[1]

    def pack_all(self, stream=None):
        """Pack every weight: one lpvit_pack_bsr_many call (two launches for the whole stack)."""
        s = int((stream or torch.cuda.current_stream()).cuda_stream)
        self._calls_for(s)
        rc = self._pack_many_fn(*self._pack_many_args)
        if rc != 0:
            raise _lib.LpvitError(rc, "lpvit_pack_bsr_many")

    def pack_each(self, stream=None):
        """Pack every weight with its own lpvit_pack_bsr call (the per-weight path)."""
        s = int((stream or torch.cuda.current_stream()).cuda_stream)
        for pack_args, _, _ in self._calls_for(s):
            rc = self._pack_fn(*pack_args)
            if rc != 0:
                raise _lib.LpvitError(rc, "lpvit_pack_bsr")

    def forward(self, stream=None, events=None, chain: bool = False):
        """Chain the 4L linears from ``h_in``; returns the output buffer. ``events``: optional list of
        (start, end) CUDA event pairs recorded around each library call: one per linear, or one for
        the whole chain call (``chain=True``)."""
        s = stream or torch.cuda.current_stream()
        calls = self._calls_for(int(s.cuda_stream))
        if chain:
            if events is not None:
                events[0][0].record(s)
            rc = self._chain_fn(*self._chain_args)
            if events is not None:
                events[0][1].record(s)
            if rc != 0:
                raise _lib.LpvitError(rc, "lpvit_bsr_linear_chain")
            return self.out
        for i, (_, fn, lin_args) in enumerate(calls):
            if events is not None:
                events[i][0].record(s)
            rc = fn(*lin_args)
            if events is not None:
                events[i][1].record(s)
            if rc != 0:
                raise _lib.LpvitError(rc, "lpvit_bsr_linear")
        return self.out

    def step(self, stream=None, events=None, chain: bool = False):
        """One pass of the whole path: pack every weight, then run every linear."""
        self.pack_all(stream)
        return self.forward(stream, events, chain)

    def check(self, stream=None):
        st = _lib.lpvit_check(self.ws.data_ptr(), int((stream or torch.cuda.current_stream()).cuda_stream))
        if st != 0:
            raise _lib.LpvitError(st, "lpvit_check")

    # ------------------------------------------------------------------ dense comparator
    def dense_forward(self, h0: torch.Tensor) -> torch.Tensor:
        """Same chain with torch's dense bf16 linear on W (.) M (a comparator, not the product)."""
        if not hasattr(self, "_dense"):
            self._dense = []
            for G in self.gemms:
                bn, bk = G["w"].bn, G["w"].bk
                keep = G["mask"].repeat_interleave(bn, 0).repeat_interleave(bk, 1).bool()
                self._dense.append(torch.where(keep, G["W"], torch.zeros_like(G["W"])))
        F = torch.nn.functional
        h = h0
        for G, Wd in zip(self.gemms, self._dense):
            if G["name"] == "qkv":
                qkv = F.linear(h, Wd, G["bias"].to(torch.bfloat16))
            elif G["name"] == "proj":
                p = F.linear(qkv[:, 2 * self.d:], Wd, G["bias"].to(torch.bfloat16))
            elif G["name"] == "fc1":
                f1 = F.gelu(F.linear(p, Wd, G["bias"].to(torch.bfloat16)))
            else:
                h = F.linear(f1, Wd, G["bias"].to(torch.bfloat16))
        return h


def deit_b_stack(m: int = 50432, b: int = 32, config: int = 4, device="cuda") -> DeitLinearStack:
    """The 12-layer DeiT-B linear stack at m tokens with seeded weights, biases and masks."""
    return DeitLinearStack(m, inputs.deit_b_stack(config, b, device), device)
