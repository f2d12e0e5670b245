"""Block-sparse linear layers for LPViT-pruned vision transformers on GB300 (sm_103a).

LPViT (arXiv 2407.02068) prunes each linear weight of a ViT in blocks (Sec. 3.1) so that the
layer becomes a block-sparse matmul whose work is proportional to the kept blocks (Sec. 3.3). A
block ``b`` is an int (b x b) or a pair (bn, bk): bn output rows by bk input columns, each 16, 32
or 64 (Table 2 uses 32x32, 64x32, 16x32 and 16x16). This package wraps the C library
``liblpvit.so`` (include/lpvit.h):

* ``taylor_block_mask(W, G, b, alpha)`` -- the block mask from first-order Taylor scores (Sec. 3.1)
* ``pack_bsr(W, mask, b)``  -- mask -> BSR pack + work list, on the GPU
* ``taylor_pack_bsr(W, G, b, alpha)`` -- the Taylor mask and the pack in one call (no host step)
* ``pack_bsr_many_into(ws, Ws, masks)`` -- the same for a list of weights in two launches
* ``bsr_linear(w, X, bias, gelu=..., residual=...)`` -- Y = act(X (W (.) M)^T + bias), optionally
  plus a bf16 residual in the same pass (the x + sublayer(x) of a pre-norm block)
* ``delta_curve(W, G, b, steps, kappa)`` / ``lambda_search(...)`` -- the layer-wise pruning-ratio
  allocation of Sec. 3.4-3.5 (empirical-Fisher distortion curves, Lagrangian slope matching)
* ``add_layernorm`` / ``attention`` -- the rest of a pre-norm ViT block; ``encoder.SparseEncoder``
  runs a whole DeiT encoder forward on them and the block-sparse linears

PyTorch provides device memory and streams only; every step runs in the library's kernels.
"""
from __future__ import annotations

from dataclasses import dataclass

import torch

from . import _lib

__all__ = ["BsrWeight", "alloc_bsr", "pack_bsr", "pack_bsr_into", "pack_bsr_many_into", "taylor_block_mask",
           "taylor_pack_bsr",
           "workspace_for", "bsr_linear", "bsr_linear_chain", "check", "LpvitError", "delta_curve", "lambda_search", "mean_gradient",
           "add_layernorm", "attention"]

LpvitError = _lib.LpvitError


def block_sides(b) -> tuple[int, int]:
    """(bn, bk) of a block given as b (square) or (bn, bk)."""
    if isinstance(b, (tuple, list)):
        if len(b) != 2:
            raise ValueError("a block is b or (bn, bk)")
        return int(b[0]), int(b[1])
    return int(b), int(b)


def _stream_handle(stream) -> int:
    s = stream if stream is not None else torch.cuda.current_stream()
    return int(s.cuda_stream)


@dataclass
class BsrWeight:
    """A packed block-sparse weight (blocks of bn rows by bk columns): device tensors owned by
    this object."""
    n: int
    k: int
    bn: int
    bk: int
    capacity: int
    row_ptr: torch.Tensor   # int32 [n/bn + 1]
    col_idx: torch.Tensor   # int32 [capacity]
    blocks: torch.Tensor | None  # bf16 [capacity, bn, bk]; None: index and work list only
    sched: torch.Tensor     # uint8 [sched_bytes]
    nnzb: int | None = None

    @property
    def b(self):
        """The block as given to alloc_bsr: an int when square, else (bn, bk)."""
        return self.bn if self.bn == self.bk else (self.bn, self.bk)

    def struct(self) -> _lib.lpvit_bsr:
        return _lib.lpvit_bsr(self.n, self.k, self.bn, self.bk, self.capacity, self.row_ptr.data_ptr(),
                              self.col_idx.data_ptr(), 0 if self.blocks is None else self.blocks.data_ptr(),
                              self.sched.data_ptr(),
                              self.sched.numel())


def alloc_bsr(n: int, k: int, b, capacity: int | None = None, device="cuda", blocks: bool = True) -> BsrWeight:
    """Device buffers for a packed n x k weight with blocks b (int or (bn, bk)); the capacity
    defaults to every block. ``blocks=False`` leaves out the BSR copy of the kept tiles: the
    linear reads only the work list's weight stream, so packing then writes the block index and
    the work list alone."""
    bn, bk = block_sides(b)
    if capacity is None:
        capacity = (n // bn) * (k // bk) if bn > 0 and bk > 0 and n % bn == 0 and k % bk == 0 else 0
    sb = _lib.lpvit_sched_bytes(n, k, bn, bk)
    return BsrWeight(n, k, bn, bk, capacity,
                     torch.empty(max(n // max(bn, 1), 0) + 1, dtype=torch.int32, device=device),
                     torch.empty(max(capacity, 1), dtype=torch.int32, device=device),
                     torch.empty((max(capacity, 1), max(bn, 1), max(bk, 1)), dtype=torch.bfloat16, device=device)
                     if blocks else None,
                     torch.empty(max(sb, 16), dtype=torch.uint8, device=device))


def pack_bsr_into(w: BsrWeight, W: torch.Tensor, mask: torch.Tensor, count: bool = False, stream=None) -> BsrWeight:
    """Pack W (bf16 [n, k], contiguous CUDA) under the block mask (uint8 [n/bn, k/bk], contiguous
    CUDA, nonzero = kept) into the buffers of ``w``; asynchronous unless ``count``."""
    if W.dtype != torch.bfloat16 or not W.is_cuda or W.dim() != 2 or not W.is_contiguous():
        raise ValueError("W must be a contiguous 2-D bf16 CUDA tensor")
    if mask.dtype != torch.uint8 or not mask.is_contiguous() or mask.device != W.device:
        raise ValueError("mask must be a contiguous uint8 tensor on W's device")
    st, nnzb = _lib.lpvit_pack_bsr(W.data_ptr(), mask.data_ptr(), w.struct(), count, _stream_handle(stream))
    if st != _lib.LPVIT_OK:
        raise LpvitError(st, "lpvit_pack_bsr")
    w.nnzb = nnzb
    return w


def taylor_block_mask(W: torch.Tensor, G: torch.Tensor, b, prune_ratio: float, stream=None):
    """Block mask of Sec. 3.1 from first-order Taylor scores: W bf16 [n, k], G (the gradient)
    float32 [n, k], both contiguous CUDA; b = int or (bn, bk). Returns (mask uint8 [n/bn, k/bk],
    1 = kept; scores float64 [n/bn, k/bk]); round(prune_ratio * blocks) of the lowest-scored
    blocks are eliminated."""
    if W.dtype != torch.bfloat16 or not W.is_cuda or W.dim() != 2 or not W.is_contiguous():
        raise ValueError("W must be a contiguous 2-D bf16 CUDA tensor")
    if G.dtype != torch.float32 or G.shape != W.shape or not G.is_contiguous() or G.device != W.device:
        raise ValueError("G must be a contiguous float32 tensor shaped like W on W's device")
    n, k = W.shape
    bn, bk = block_sides(b)
    if bn <= 0 or bk <= 0 or n % bn or k % bk:
        raise ValueError("n and k must be multiples of the block sides")
    scores = torch.empty((n // bn, k // bk), dtype=torch.float64, device=W.device)
    mask = torch.empty((n // bn, k // bk), dtype=torch.uint8, device=W.device)
    st = _lib.lpvit_taylor_block_mask(W.data_ptr(), G.data_ptr(), n, k, bn, bk, prune_ratio, scores.data_ptr(),
                                      mask.data_ptr(), _stream_handle(stream))
    if st != _lib.LPVIT_OK:
        raise LpvitError(st, "lpvit_taylor_block_mask")
    return mask, scores


def taylor_pack_bsr(W: torch.Tensor, G: torch.Tensor, b, prune_ratio: float, capacity: int | None = None,
                    count: bool = False, stream=None):
    """Sec. 3.1 end to end: the block mask from first-order Taylor scores at ``prune_ratio`` and the
    pack of W under it, in one library call (lpvit_taylor_pack_bsr). W bf16 [n, k], G float32 [n, k],
    both contiguous CUDA. Returns (BsrWeight, mask uint8 [n/bn, k/bk], scores float64 [n/bn, k/bk])."""
    if W.dtype != torch.bfloat16 or not W.is_cuda or W.dim() != 2 or not W.is_contiguous():
        raise ValueError("W must be a contiguous 2-D bf16 CUDA tensor")
    if G.dtype != torch.float32 or G.shape != W.shape or not G.is_contiguous() or G.device != W.device:
        raise ValueError("G must be a contiguous float32 tensor shaped like W on W's device")
    n, k = W.shape
    bn, bk = block_sides(b)
    if bn <= 0 or bk <= 0 or n % bn or k % bk:
        raise ValueError("n and k must be multiples of the block sides")
    w = alloc_bsr(n, k, b, capacity, W.device)
    scores = torch.empty((n // bn, k // bk), dtype=torch.float64, device=W.device)
    mask = torch.empty((n // bn, k // bk), dtype=torch.uint8, device=W.device)
    st, nnzb = _lib.lpvit_taylor_pack_bsr(W.data_ptr(), G.data_ptr(), prune_ratio, scores.data_ptr(),
                                          mask.data_ptr(), w.struct(), count, _stream_handle(stream))
    if st != _lib.LPVIT_OK:
        raise LpvitError(st, "lpvit_taylor_pack_bsr")
    w.nnzb = nnzb
    return w, mask, scores


def delta_curve(W: torch.Tensor, G: torch.Tensor, b, steps: int, kappa: float, workspace: torch.Tensor | None = None,
                stream=None) -> torch.Tensor:
    """Sec. 3.4-3.5 distortion curve of one layer: W bf16 [n, k], G float32 per-sample gradients
    [N, n, k], both contiguous CUDA. Returns float64 [steps + 1] on the device: delta at
    alpha = s / steps (see lpvit_delta_curve)."""
    if W.dtype != torch.bfloat16 or not W.is_cuda or W.dim() != 2 or not W.is_contiguous():
        raise ValueError("W must be a contiguous 2-D bf16 CUDA tensor")
    if G.dtype != torch.float32 or G.dim() != 3 or tuple(G.shape[1:]) != tuple(W.shape) or not G.is_contiguous() \
            or G.device != W.device:
        raise ValueError("G must be a contiguous float32 [N, n, k] tensor on W's device")
    n, k = W.shape
    bn, bk = block_sides(b)
    N = G.shape[0]
    need = _lib.lpvit_delta_curve_workspace_bytes(N, n, k, bn, bk, steps)
    if workspace is None:
        workspace = torch.empty(max(need, 256), dtype=torch.uint8, device=W.device)
    out = torch.empty(steps + 1, dtype=torch.float64, device=W.device)
    st = _lib.lpvit_delta_curve(W.data_ptr(), G.data_ptr(), N, n, k, bn, bk, kappa, steps, out.data_ptr(),
                                workspace.data_ptr(), workspace.numel(), _stream_handle(stream))
    if st != _lib.LPVIT_OK:
        raise LpvitError(st, "lpvit_delta_curve")
    return out


def add_layernorm(x: torch.Tensor, r: torch.Tensor | None, gamma: torch.Tensor, beta: torch.Tensor,
                  eps: float = 1e-6, norm_out: torch.Tensor | None = None, sum_out: torch.Tensor | None = None,
                  stream=None):
    """s = bf16(x + r) (r may be None: s = x) and y = LayerNorm(s) * gamma + beta over the last axis.
    x, r: contiguous bf16 CUDA [rows, D]; gamma, beta: float32 [D]. Returns y, or (s, y) when r is
    given."""
    if x.dtype != torch.bfloat16 or not x.is_cuda or x.dim() != 2 or not x.is_contiguous():
        raise ValueError("x must be a contiguous 2-D bf16 CUDA tensor")
    rows, D = x.shape
    if r is not None and (r.shape != x.shape or r.dtype != x.dtype or not r.is_contiguous()):
        raise ValueError("r must match x")
    if gamma.dtype != torch.float32 or beta.dtype != torch.float32 or gamma.numel() != D or beta.numel() != D:
        raise ValueError("gamma and beta must be float32 [D]")
    y = norm_out if norm_out is not None else torch.empty_like(x)
    sm = None
    if r is not None:
        sm = sum_out if sum_out is not None else torch.empty_like(x)
    st = _lib.lpvit_add_layernorm(x.data_ptr(), 0 if r is None else r.data_ptr(), gamma.data_ptr(), beta.data_ptr(),
                                  rows, D, eps, 0 if sm is None else sm.data_ptr(), y.data_ptr(),
                                  _stream_handle(stream))
    if st != _lib.LPVIT_OK:
        raise LpvitError(st, "lpvit_add_layernorm")
    return y if r is None else (sm, y)


def attention(qkv: torch.Tensor, tokens: int, heads: int, out: torch.Tensor | None = None, stream=None):
    """softmax(q k^T / sqrt(head_dim)) v per image and head: qkv bf16 [images * tokens, 3 * heads * 64],
    contiguous CUDA; returns bf16 [images * tokens, heads * 64]."""
    if qkv.dtype != torch.bfloat16 or not qkv.is_cuda or qkv.dim() != 2 or not qkv.is_contiguous():
        raise ValueError("qkv must be a contiguous 2-D bf16 CUDA tensor")
    M, C = qkv.shape
    if M % tokens or C % (3 * heads):
        raise ValueError("qkv shape does not match tokens and heads")
    head_dim = C // (3 * heads)
    o = out if out is not None else torch.empty((M, C // 3), dtype=torch.bfloat16, device=qkv.device)
    st = _lib.lpvit_attention(qkv.data_ptr(), M // tokens, tokens, heads, head_dim, o.data_ptr(),
                              _stream_handle(stream))
    if st != _lib.LPVIT_OK:
        raise LpvitError(st, "lpvit_attention")
    return o


def mean_gradient(G: torch.Tensor, stream=None) -> torch.Tensor:
    """float32 [n, k]: the mean over the first axis of G (float32 [N, n, k], contiguous CUDA), summed in
    float32 in sample order (the gradient lpvit_delta_curve and the Taylor mask rank blocks by)."""
    if G.dtype != torch.float32 or not G.is_cuda or G.dim() < 2 or not G.is_contiguous():
        raise ValueError("G must be a contiguous float32 CUDA tensor [N, ...]")
    g = torch.empty(G.shape[1:], dtype=torch.float32, device=G.device)
    st = _lib.lpvit_mean_gradient(G.data_ptr(), G.shape[0], g.numel(), g.data_ptr(), _stream_handle(stream))
    if st != _lib.LPVIT_OK:
        raise LpvitError(st, "lpvit_mean_gradient")
    return g


def lambda_search(deltas, steps: int, flops, power_coef, beta: float, flops_ratio: float):
    """Sec. 3.4 lambda search (host): deltas = per-layer curves of steps + 1 values. Returns
    (k list with alpha_i = k_i / steps, lambda, FLOPs-remained ratio)."""
    rows = [d.tolist() if hasattr(d, "tolist") else list(d) for d in deltas]
    st, ks, lam, ratio = _lib.lpvit_lambda_search(rows, steps, flops, power_coef, beta, flops_ratio)
    if st != _lib.LPVIT_OK:
        raise LpvitError(st, "lpvit_lambda_search")
    return ks, lam, ratio


def pack_bsr_many_into(ws: list, Ws: list, masks: list, stream=None) -> list:
    """Pack Ws[i] under masks[i] into ws[i] for all i in two launches (lpvit_pack_bsr_many);
    asynchronous. Tensors as for pack_bsr_into."""
    if not (len(ws) == len(Ws) == len(masks)):
        raise ValueError("ws, Ws and masks must have the same length")
    for W, mask in zip(Ws, masks):
        if W.dtype != torch.bfloat16 or not W.is_cuda or W.dim() != 2 or not W.is_contiguous():
            raise ValueError("every W must be a contiguous 2-D bf16 CUDA tensor")
        if mask.dtype != torch.uint8 or not mask.is_contiguous() or mask.device != W.device:
            raise ValueError("every mask must be a contiguous uint8 tensor on its W's device")
    st = _lib.lpvit_pack_bsr_many([W.data_ptr() for W in Ws], [m.data_ptr() for m in masks],
                                  [w.struct() for w in ws], _stream_handle(stream))
    if st != _lib.LPVIT_OK:
        raise LpvitError(st, "lpvit_pack_bsr_many")
    return ws


def pack_bsr(W: torch.Tensor, mask: torch.Tensor, b, capacity: int | None = None, count: bool = False,
             stream=None) -> BsrWeight:
    """Pack W (bf16 [n, k], CUDA) under the block mask (uint8 [n/bn, k/bk], nonzero = kept);
    b = int (square) or (bn, bk)."""
    if W.dtype != torch.bfloat16 or not W.is_cuda or W.dim() != 2:
        raise ValueError("W must be a 2-D bf16 CUDA tensor")
    W = W.contiguous()
    mask = mask.to(device=W.device, dtype=torch.uint8).contiguous()
    n, k = W.shape
    w = alloc_bsr(n, k, b, capacity, W.device)
    return pack_bsr_into(w, W, mask, count, stream)


def workspace_for(w: BsrWeight, m: int, device=None) -> torch.Tensor:
    """A zero-filled workspace of lpvit_workspace_bytes(w, m) bytes (256-byte aligned)."""
    nbytes = _lib.lpvit_workspace_bytes(w.struct(), m)
    return torch.zeros(max(nbytes, 256), dtype=torch.uint8, device=device or w.sched.device)


def bsr_linear(w: BsrWeight, X: torch.Tensor, bias: torch.Tensor | None = None, gelu: bool = False,
               out: torch.Tensor | None = None, out_dtype=torch.bfloat16, workspace: torch.Tensor | None = None,
               stream=None, residual: torch.Tensor | None = None) -> torch.Tensor:
    """Y = act(X W~^T + bias). X: bf16 [m, k] CUDA (a row-strided view with unit column stride is
    fine); bias: fp32 [n] or None. Returns Y [m, n] (or writes ``out``). With ``residual`` (bf16
    [m, n], 16-byte rows; may be ``out`` itself) Y = round(round(act(...)) + residual), bf16
    (lpvit_bsr_linear_residual). The library picks the kernel: m <= 256 runs one launch of the
    small-m kernel, larger m the persistent CTA-pair kernel."""
    if X.dtype != torch.bfloat16 or X.dim() != 2 or X.stride(1) != 1:
        raise ValueError("X must be a 2-D bf16 tensor with unit column stride")
    m = X.shape[0]
    if out is None:
        out = torch.empty((m, w.n), dtype=out_dtype, device=X.device)
    if out.dtype not in (torch.bfloat16, torch.float32) or out.stride(1) != 1:
        raise ValueError("out must be bf16 or fp32 with unit column stride")
    if bias is not None:
        if bias.dtype != torch.float32 or not bias.is_contiguous():
            raise ValueError("bias must be a contiguous fp32 tensor")
    if workspace is None:
        workspace = workspace_for(w, m, X.device)
    if residual is not None:
        if residual.dtype != torch.bfloat16 or residual.dim() != 2 or residual.stride(1) != 1 \
                or tuple(residual.shape) != (m, w.n) or out.dtype != torch.bfloat16:
            raise ValueError("residual must be a bf16 [m, n] tensor with unit column stride, out bf16")
        st = _lib.lpvit_bsr_linear_residual(w.struct(), X.data_ptr(), m, X.stride(0),
                                            bias.data_ptr() if bias is not None else None, gelu,
                                            residual.data_ptr(), residual.stride(0), out.data_ptr(), out.stride(0),
                                            workspace.data_ptr(), workspace.numel(), _stream_handle(stream))
        if st != _lib.LPVIT_OK:
            raise LpvitError(st, "lpvit_bsr_linear_residual")
        return out
    fn = _lib.lpvit_bsr_linear_gelu if gelu else _lib.lpvit_bsr_linear
    st = fn(w.struct(), X.data_ptr(), m, X.stride(0), bias.data_ptr() if bias is not None else None,
            out.data_ptr(), out.stride(0), _lib.LPVIT_F32 if out.dtype == torch.float32 else _lib.LPVIT_BF16,
            workspace.data_ptr(), workspace.numel(), _stream_handle(stream))
    if st != _lib.LPVIT_OK:
        raise LpvitError(st, "lpvit_bsr_linear_gelu" if gelu else "lpvit_bsr_linear")
    return out


def bsr_linear_chain(steps, workspace: torch.Tensor | None = None, stream=None) -> None:
    """Consecutive linears over the same m tokens in one library call (lpvit_bsr_linear_chain).
    ``steps``: a sequence of (w, X, bias, out, gelu): X and out bf16 [m, k] / [m, n] CUDA tensors with
    unit column stride (row-strided views are fine; a later X may be an earlier out, or a column range
    of it), bias fp32 [n] or None. Each out = act(X W~^T + bias), in order, bit-identical to separate
    bsr_linear calls. The workspace defaults to a zero-filled one of lpvit_chain_workspace_bytes."""
    steps = list(steps)
    if not steps:
        return
    m = steps[0][1].shape[0]
    rows = []
    for w, X, bias, out, gelu in steps:
        for t in (X, out):
            if t.dtype != torch.bfloat16 or t.dim() != 2 or t.stride(1) != 1 or t.shape[0] != m:
                raise ValueError("X and out must be 2-D bf16 tensors of m rows with unit column stride")
        if bias is not None and (bias.dtype != torch.float32 or not bias.is_contiguous()):
            raise ValueError("bias must be a contiguous fp32 tensor")
        rows.append((w.struct(), X.data_ptr(), X.stride(0), bias.data_ptr() if bias is not None else None,
                     out.data_ptr(), out.stride(0), 1 if gelu else 0))
    links = _lib.chain_links(rows)
    if workspace is None:
        nbytes = _lib.lpvit_chain_workspace_bytes(links, len(rows), m)
        workspace = torch.zeros(max(nbytes, 256), dtype=torch.uint8, device=steps[0][1].device)
    st = _lib.lpvit_bsr_linear_chain(links, len(rows), m, workspace.data_ptr(), workspace.numel(),
                                     _stream_handle(stream))
    if st != _lib.LPVIT_OK:
        raise LpvitError(st, "lpvit_bsr_linear_chain")


def check(workspace: torch.Tensor, stream=None) -> None:
    """Synchronise and raise if a kernel that used ``workspace`` reported a device-side error."""
    st = _lib.lpvit_check(workspace.data_ptr(), _stream_handle(stream))
    if st != _lib.LPVIT_OK:
        raise LpvitError(st, "lpvit_check")
