"""GPU parity: the CUDA path through the C ABI against the fp64 CPU oracle.

Gates (from the method's stated bar): BSR pack bit-exact; GEMM with fp32 output within
max|y - y_ref| / rms(y_ref) <= 1e-2 (and, as a tighter diagnostic, <= 1e-4, since fp32
accumulation of bf16 products is accurate to ~1e-6); bf16 output within one bf16 ulp of the
exact value element-wise; integer-exact inputs bit-exact."""
import numpy as np
import pytest
import torch

import oracle
from paper_2407_02068_gb300 import inputs

pytestmark = pytest.mark.gpu

NORM_TOL = 1e-2      # max|y - y_ref| / rms(y_ref), fp32 output
TIGHT_TOL = 1e-4

# blocks: b (square) or (bn rows, bk columns); Table 2 uses 32x32, 64x32, 16x32 and 16x16
BLOCKS = [16, 32, 64, (64, 32), (16, 32)]
BLOCKS_ALL = BLOCKS + [(32, 16), (32, 64), (16, 64), (64, 16)]


def _sides(b):
    return inputs.block_sides(b)


def _sid(b):
    """A seed offset per block (square blocks keep their historic b)."""
    bn, bk = _sides(b)
    return bn if bn == bk else 100 * bn + bk


@pytest.fixture(scope="module")
def lp():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2407_02068_gb300 as lp
    from paper_2407_02068_gb300 import build
    build.build()
    return lp


def _bits(t):
    return inputs.bf16_bits(t)


def _oracle(X, W, mask, b, bias, gelu=False, rows=None):
    Xb = _bits(X if rows is None else X[rows])
    return oracle.linear(Xb, _bits(W), mask.cpu().numpy(), b, None if bias is None else bias.cpu().numpy(), gelu)


def _norm_err(y, ref):
    rms = np.sqrt(np.mean(ref ** 2))
    return np.max(np.abs(y - ref)) / max(rms, 1e-30)


def _ulp_bf16(x):
    a = np.abs(x)
    e = np.floor(np.log2(np.maximum(a, 2.0 ** -126)))
    return 2.0 ** (e - 7)


def _acc_bound(X, W, mask, b, bias):
    """Bound on the fp32 accumulation error of any summation order: k * 2^-24 * sum_k |x w~|."""
    bn, bk = _sides(b)
    keep = mask.repeat_interleave(bn, 0).repeat_interleave(bk, 1).bool()
    Wa = torch.where(keep, W, torch.zeros_like(W)).double().abs().cpu()
    S = X.double().abs().cpu() @ Wa.T + bias.double().abs().cpu()
    return (W.shape[1] * 2.0 ** -24 * S).numpy()


def _bf16_tol(ref, X, W, mask, b, bias, gelu=False):
    """One bf16 ulp of the exact value, plus the fp32 accumulation bound (scaled by max|gelu'| = 1.13),
    plus 4 fp32 ulps for erff."""
    acc = _acc_bound(X, W, mask, b, bias)
    return _ulp_bf16(ref) + (1.13 * acc + 4 * 2.0 ** -23 * np.abs(ref) if gelu else acc)


def _case(m, n, k, b, sp, seed, device="cuda", int_valued=False, mask_kind="uniform"):
    g = torch.Generator().manual_seed(seed)
    if int_valued:
        X = torch.randint(-4, 5, (m, k), generator=g).float().to(torch.bfloat16)
        W = (torch.randint(-4, 5, (n, k), generator=g).float() / 16).to(torch.bfloat16)
        bias = torch.randint(-8, 9, (n,), generator=g).float() / 8
    else:
        X = torch.randn(m, k, generator=g).to(torch.bfloat16)
        W = (torch.randn(n, k, generator=g) * 0.02).to(torch.bfloat16)
        bias = torch.randn(n, generator=g) * 0.02
    if mask_kind == "uniform":
        mask = inputs.uniform_mask(n, k, b, sp, seed + 1)
    else:
        mask = inputs.zipf_mask(n, k, b, sp, seed + 1)
    return X.to(device), W.to(device), bias.to(device), mask.to(device)


# ------------------------------------------------------------------------------------- pack

@pytest.mark.parametrize("n,k,b,sp", [(1152, 384, 32, 0.5), (384, 1536, 16, 0.5), (768, 3072, 64, 0.3),
                                      (3072, 768, 32, 0.0), (256, 256, 16, 1.0), (64, 48, 16, 0.4),
                                      (768, 3072, (64, 32), 0.6), (384, 1536, (16, 32), 0.3),
                                      (192, 128, (32, 64), 0.5), (64, 96, (64, 16), 0.4)])
def test_pack_bit_exact(lp, n, k, b, sp):
    X, W, bias, mask = _case(4, n, k, b, sp, 11)
    mask[0] = 0  # an empty panel
    w = lp.pack_bsr(W, mask, b, count=True)
    rp, ci, bl = oracle.pack(_bits(W), mask.cpu().numpy(), b)
    assert w.nnzb == len(ci)
    assert np.array_equal(w.row_ptr.cpu().numpy(), rp)
    assert np.array_equal(w.col_idx[:w.nnzb].cpu().numpy(), ci)
    got = w.blocks[:w.nnzb].contiguous().view(torch.int16).cpu().numpy().view(np.uint16)
    assert np.array_equal(got, bl)


GROUP = 256    # output features of a work unit
CHUNK = 64     # input columns of a work-list entry
SLOTS = 16     # group table width


def _decode_sched(w):
    """Header, group entry pointers, entries (chunk index each) and the group table (row panel of
    every slot, or -1)."""
    raw = w.sched.cpu().numpy().view(np.int32)
    ng = int(raw[1])
    gent = raw[16:16 + ng + 1]
    gpan = raw[16 + ng + 1:16 + ng + 1 + SLOTS * ng].reshape(ng, SLOTS)
    off = _entries_offset(ng)
    ent = raw[off:off + int(gent[-1])]
    return raw[:16], gent, ent, gpan


def _entries_offset(ng):
    return (16 + ng + 1 + SLOTS * ng + 3) // 4 * 4


def _chunk_bits(M, bk):
    """[panels, chunks]: does the panel keep a block in each 64-column chunk?"""
    npan, kb = M.shape
    bpc = CHUNK // bk
    kc = -(-kb * bk // CHUNK)
    C = np.zeros((npan, kc), dtype=bool)
    for c in range(kc):
        C[:, c] = M[:, c * bpc:(c + 1) * bpc].any(axis=1)
    return C


def _grouping(M, bn, bk):
    """The plan's grouping rule restated: a group starts with the unassigned panel keeping the most
    blocks, then takes the unassigned panel adding the fewest chunks to the group's union (ties to
    the lower index); kept only if it has fewer entries than consecutive panels, and only for up to
    1024 panels and 8192 bitmap words."""
    npan, kb = M.shape
    C = _chunk_bits(M, bk)
    kc = C.shape[1]
    gb = GROUP // bn
    ng = -(-npan // gb)
    ident = [[g * gb + p if p < gb and g * gb + p < npan else -1 for p in range(SLOTS)] for g in range(ng)]
    if not (gb >= 2 and npan <= 1024 and npan * ((kc + 31) // 32) <= 8192):
        return ident
    rows = [set(np.nonzero(C[r])[0].tolist()) for r in range(npan)]
    kept = [int(M[r].sum()) for r in range(npan)]
    asg, table = [False] * npan, []
    for g in range(ng):
        t, U = [], set()
        for sl in range(gb):
            cand = [p for p in range(npan) if not asg[p]]
            if not cand:
                t.append(-1)
                continue
            pick = min(cand, key=(lambda p: (-kept[p], p)) if sl == 0 else (lambda p: (len(rows[p] - U), p)))
            asg[pick] = True
            t.append(pick)
            U |= rows[pick]
        table.append(t + [-1] * (SLOTS - gb))

    def entries(tab):
        return sum(len(set().union(*[rows[r] for r in t if r >= 0])) for t in tab)
    return table if entries(table) < entries(ident) else ident


@pytest.mark.parametrize("n,k,b", [(1152, 384, 32), (384, 1536, 16), (768, 3072, 64), (200 * 16, 64, 16),
                                   (768, 768, (64, 32)), (208, 384, (16, 32)), (320, 128, (64, 16)),
                                   (1024 * 16, 64, 16),      # 1024 panels: the grouping's limit
                                   (1025 * 16, 64, 16),      # 1025 panels: consecutive groups
                                   (8192, 8704, 16),         # 512 panels x 17 bitmap words > 8192
                                   (100 * 32, 4096, 32),     # register grouping: 100 panels, 4 words
                                   (128 * 32, 4096, 32),     # register grouping at its limits: 128 panels, 4 words
                                   (129 * 32, 4096, 32),     # 129 panels: shared-memory grouping
                                   (128 * 32, 5120, 32)])    # 5 bitmap words: shared-memory grouping
def test_work_list_covers_every_kept_block_once(lp, n, k, b):
    X, W, bias, mask = _case(4, n, k, b, 0.55, 12)
    w = lp.pack_bsr(W, mask, b, count=True)
    hdr, gent, ent, gpan = _decode_sched(w)
    bn, bk = _sides(b)
    assert (int(hdr[4]), int(hdr[5]), int(hdr[6]), int(hdr[7]), int(hdr[8])) == (n, k, bn, bk, 2)
    gb = GROUP // bn
    M = mask.cpu().numpy()
    C = _chunk_bits(M, bk)
    # the group table: every row panel in exactly one slot, as the grouping rule picks them
    used = sorted(int(r) for r in gpan.ravel() if r >= 0)
    assert used == list(range(n // bn)) and np.all(gpan[:, gb:] == -1)
    assert gpan.tolist() == _grouping(M, bn, bk)
    # entries: per group the chunks where one of its panels keeps a block, ascending; so every
    # kept block lies in exactly one entry (its panel's group, its column's chunk)
    covered = np.zeros_like(M, dtype=np.int32)
    for g in range(int(hdr[1])):
        cs = [int(c) for c in ent[gent[g]:gent[g + 1]]]
        panels = [int(r) for r in gpan[g, :gb] if r >= 0]
        want = sorted(np.nonzero(C[panels].any(axis=0))[0].tolist()) if panels else []
        assert cs == want
        for c in cs:
            for r in panels:
                j0 = c * CHUNK // bk
                covered[r, j0:j0 + CHUNK // bk] += 1
    assert np.all(covered[M != 0] == 1)


@pytest.mark.parametrize("b", [32, 16, (64, 32)])
def test_grouping_pairs_panels_with_the_same_columns(lp, b):
    """Row panels of two kinds keep blocks in two disjoint sets of chunks (even panels in A, odd
    panels in B). Consecutive groups would mix the kinds and need |A u B| entries each; the plan's
    grouping puts panels of one kind together, so each group needs |A| or |B| entries. The linear on
    that work list still matches the oracle."""
    bn, bk = _sides(b)
    n, k = 1024, 512
    npan, kb, kc = n // bn, k // bk, k // CHUNK
    rng = np.random.default_rng(77)
    chunks = rng.permutation(kc)
    CA, CB = np.sort(chunks[:kc // 3]), np.sort(chunks[kc // 3:kc // 3 + kc // 4])
    bpc = CHUNK // bk
    A = np.concatenate([np.arange(c * bpc, (c + 1) * bpc) for c in CA])
    B = np.concatenate([np.arange(c * bpc, (c + 1) * bpc) for c in CB])
    M = np.zeros((npan, kb), np.uint8)
    M[0::2, A] = 1
    M[1::2, B] = 1
    X, W, bias, _ = _case(300, n, k, b, 0.5, 1234)
    mask = torch.from_numpy(M).cuda()
    w = lp.pack_bsr(W, mask, b, count=True)
    hdr, gent, ent, gpan = _decode_sched(w)
    gb = GROUP // bn
    assert gpan.tolist() == _grouping(M, bn, bk)
    for g in range(int(hdr[1])):
        kinds = {int(r) % 2 for r in gpan[g, :gb] if r >= 0}
        assert len(kinds) == 1                       # one kind of panel per group
    ng = npan // gb
    assert int(gent[-1]) == (ng // 2) * (len(CA) + len(CB))
    Y = lp.bsr_linear(w, X, bias, out_dtype=torch.float32)
    ref = _oracle(X, W, mask, b, bias)
    assert _norm_err(Y.cpu().double().numpy(), ref) <= TIGHT_TOL


def _check_weight_stream(w, W, mask):
    """The work list's weight stream: entry by entry, the 256-row tile of the entry's group over its
    64-column chunk, row-major: row r holds W[feature of group row r] over the chunk where that
    block is kept, zero where it is removed, where the slot has no panel and beyond column k."""
    n, k, bn, bk = w.n, w.k, w.bn, w.bk
    hdr, gent, ent, gpan = _decode_sched(w)
    ng, kc = int(hdr[1]), -(-k // CHUNK)
    raw = w.sched.cpu().numpy().view(np.uint8)
    ent_end = 4 * (_entries_offset(ng) + ng * kc)
    stream = raw[(ent_end + 1023) // 1024 * 1024:]
    Wb = _bits(W).reshape(n, k)
    M = mask.cpu().numpy()
    # the expected tile of group g at chunk c, built from the definition
    feat = np.full(GROUP, -1)
    for g in range(ng):
        for r in range(GROUP):
            panel = int(gpan[g, r // bn])
            feat[r] = panel * bn + r % bn if panel >= 0 else -1
        ri = np.nonzero(feat >= 0)[0]
        fr = feat[ri]
        for e in range(int(gent[g]), int(gent[g + 1])):
            c = int(ent[e])
            want = np.zeros((GROUP, CHUNK), np.uint16)
            cols = np.arange(c * CHUNK, min(k, (c + 1) * CHUNK))
            keep = M[fr // bn][:, cols // bk] != 0
            want[np.ix_(ri, cols - c * CHUNK)] = np.where(keep, Wb[fr][:, cols], 0)
            tile = stream[e * GROUP * CHUNK * 2:(e + 1) * GROUP * CHUNK * 2].view(np.uint16).reshape(GROUP, CHUNK)
            assert np.array_equal(tile, want), (g, c)


@pytest.mark.parametrize("n,k,b", [(384, 256, 32), (208, 128, 16), (384, 192, 64), (96, 64, 32), (384, 128, (64, 32)),
                                   (208, 128, (16, 32)), (192, 192, (32, 64))])
def test_weight_stream_holds_every_entry_tile(lp, n, k, b):
    X, W, bias, mask = _case(4, n, k, b, 0.5, 31)
    w = lp.pack_bsr(W, mask, b, count=True)
    _check_weight_stream(w, W, mask)


@pytest.mark.parametrize("count", [1, 5, 100])
def test_pack_many_matches_single_packs(lp, count):
    """The batched pack (all plans in one launch, all copies in another; 100 jobs span two launches
    of 96) gives, weight by weight, the bits of single packs and of the oracle."""
    shapes = [(384, 256, 32), (208, 128, 16), (384, 768, 64), (768, 3072, 32), (96, 64, 32)]
    Ws, masks, wm, ws = [], [], [], []
    for i in range(count):
        n, k, b = shapes[i % len(shapes)]
        X, W, bias, mask = _case(4, n, k, b, 0.3 + 0.1 * (i % 5), 2000 + i)
        Ws.append(W.contiguous())
        masks.append(mask.contiguous())
        wm.append(lp.alloc_bsr(n, k, b))
        ws.append(lp.pack_bsr(W, mask, b, count=True))
    lp.pack_bsr_many_into(wm, Ws, masks)
    torch.cuda.synchronize()
    for i in range(count):
        a, s1 = wm[i], ws[i]
        n, k, b = a.n, a.k, a.b
        nnzb = s1.nnzb
        assert torch.equal(a.row_ptr, s1.row_ptr)
        assert torch.equal(a.col_idx[:nnzb], s1.col_idx[:nnzb])
        assert torch.equal(a.blocks[:nnzb].view(torch.int16), s1.blocks[:nnzb].view(torch.int16))
        # header, group pointers and entries (the words padding the entries to 16 bytes are not defined)
        ha, hs, ea, es = _decode_sched(a)[0], _decode_sched(s1)[0], _decode_sched(a), _decode_sched(s1)
        assert np.array_equal(ha, hs) and np.array_equal(ea[1], es[1]) and np.array_equal(ea[2], es[2])
        assert np.array_equal(ea[3], es[3])
        assert np.array_equal(_stream_bytes(a), _stream_bytes(s1))
        if i < 5:
            _check_weight_stream(a, Ws[i], masks[i])
        rp, ci, bl = oracle.pack(_bits(Ws[i]), masks[i].cpu().numpy(), b)
        assert np.array_equal(a.row_ptr.cpu().numpy(), rp) and np.array_equal(a.col_idx[:nnzb].cpu().numpy(), ci)


def _stream_bytes(w):
    """The weight-stream tiles of w's work list (entries x 256 x 64 bf16) as raw bytes."""
    hdr, gent, ent, gpan = _decode_sched(w)
    ng, kc = int(hdr[1]), -(-w.k // CHUNK)
    raw = w.sched.cpu().numpy().view(np.uint8)
    start = (4 * (_entries_offset(ng) + ng * kc) + 1023) // 1024 * 1024
    return raw[start:start + int(hdr[2]) * GROUP * CHUNK * 2]


@pytest.mark.parametrize("many", [False, True])
def test_pack_without_blocks(lp, many):
    """A weight allocated without the BSR block copy packs to the same index, work list and weight
    stream, and its linear gives the same bits."""
    shapes = [(1152, 384, 32, 0.5), (384, 1536, 16, 0.4), (768, 3072, (64, 32), 0.6)]
    for i, (n, k, b, sp) in enumerate(shapes):
        X, W, bias, mask = _case(197, n, k, b, sp, 4100 + i)
        full = lp.pack_bsr(W, mask, b, count=True)
        bare = lp.alloc_bsr(n, k, b, blocks=False)
        assert bare.blocks is None
        if many:
            lp.pack_bsr_many_into([bare], [W.contiguous()], [mask.contiguous()])
        else:
            lp.pack_bsr_into(bare, W.contiguous(), mask.contiguous())
        torch.cuda.synchronize()
        nnzb = full.nnzb
        assert torch.equal(bare.row_ptr, full.row_ptr) and torch.equal(bare.col_idx[:nnzb], full.col_idx[:nnzb])
        hb, hf = _decode_sched(bare), _decode_sched(full)
        assert all(np.array_equal(u, v) for u, v in zip(hb, hf))
        assert np.array_equal(_stream_bytes(bare), _stream_bytes(full))
        yb = lp.bsr_linear(bare, X, bias)
        yf = lp.bsr_linear(full, X, bias)
        assert torch.equal(yb.view(torch.int16), yf.view(torch.int16))


# ------------------------------------------------------------------------------------- GEMM

@pytest.mark.parametrize("b", BLOCKS_ALL)
@pytest.mark.parametrize("m", [1, 197, 300, 777])
def test_linear_fp32_out(lp, b, m):
    n, k = 384, 256
    X, W, bias, mask = _case(m, n, k, b, 0.5, 100 + _sid(b) + m)
    w = lp.pack_bsr(W, mask, b)
    Y = lp.bsr_linear(w, X, bias, out_dtype=torch.float32)
    ws = lp.workspace_for(w, m)
    lp.check(ws)
    ref = _oracle(X, W, mask, b, bias)
    err = _norm_err(Y.cpu().double().numpy(), ref)
    assert err <= NORM_TOL
    assert err <= TIGHT_TOL


@pytest.mark.parametrize("m", [520, 200])   # the pair kernel; the small-m kernel
@pytest.mark.parametrize("b", BLOCKS)
def test_linear_integer_inputs_bit_exact(lp, b, m):
    n, k = 256, 512
    X, W, bias, mask = _case(m, n, k, b, 0.5, 200 + _sid(b), int_valued=True)
    w = lp.pack_bsr(W, mask, b)
    Y = lp.bsr_linear(w, X, bias, out_dtype=torch.float32)
    ref = _oracle(X, W, mask, b, bias)
    assert np.array_equal(Y.cpu().double().numpy(), ref)


@pytest.mark.parametrize("b", BLOCKS)
def test_linear_bf16_out_within_one_ulp(lp, b):
    m, n, k = 600, 512, 384
    X, W, bias, mask = _case(m, n, k, b, 0.5, 300 + _sid(b))
    w = lp.pack_bsr(W, mask, b)
    Y = lp.bsr_linear(w, X, bias)
    ref = _oracle(X, W, mask, b, bias)
    y = Y.float().cpu().double().numpy()
    assert np.all(np.abs(y - ref) <= _bf16_tol(ref, X, W, mask, b, bias))


@pytest.mark.parametrize("b", BLOCKS)
def test_linear_gelu(lp, b):
    m, n, k = 333, 256, 256
    X, W, bias, mask = _case(m, n, k, b, 0.4, 400 + _sid(b))
    w = lp.pack_bsr(W, mask, b)
    Y = lp.bsr_linear(w, X, bias, gelu=True, out_dtype=torch.float32)
    ref = _oracle(X, W, mask, b, bias, gelu=True)
    assert _norm_err(Y.cpu().double().numpy(), ref) <= TIGHT_TOL
    Yb = lp.bsr_linear(w, X, bias, gelu=True)
    assert np.all(np.abs(Yb.float().cpu().double().numpy() - ref) <= _bf16_tol(ref, X, W, mask, b, bias, gelu=True))


def test_gelu_epilogue_over_the_float32_range(lp):
    """All-zero mask: the output is GELU(bias). Biases sweep [-14, 14], tiny, huge and signed-zero
    values, against the oracle's exact GELU: float32 output within 5e-4 relative plus 2^-21 |t|
    (the epilogue's GELU: a polynomial for log2 of the normal tail and one single-precision MUFU
    exponential), relative alone where t > -3; bf16 output within one bf16 ulp plus that."""
    f32 = np.float32
    special = [0.0, -0.0, 1e-30, -1e-30, 1e-6, -1e-6, 20.0, -20.0, 1e4, -1e4, 3.0, -3.0]
    sweep = np.linspace(-14.0, 14.0, 4096 - len(special))
    t = np.concatenate([np.array(special, np.float64), sweep]).astype(np.float32)
    n, k, m = t.size, 32, 40
    bias = torch.from_numpy(t).cuda()
    W = torch.zeros(n, k, dtype=torch.bfloat16, device="cuda")
    X = torch.zeros(m, k, dtype=torch.bfloat16, device="cuda")
    mask = torch.zeros(n // 32, k // 32, dtype=torch.uint8, device="cuda")
    w = lp.pack_bsr(W, mask, 32)
    ref = oracle.gelu(t.astype(np.float64))
    Y = lp.bsr_linear(w, X, bias, gelu=True, out_dtype=torch.float32).cpu().double().numpy()
    assert np.all(Y == Y[0])
    y = Y[0]
    tol = 5e-4 * np.abs(ref) + 2.0 ** -21 * np.abs(t)
    assert np.all(np.abs(y - ref) <= tol)
    core = (t > -3) & (np.abs(ref) > 1e-36)
    assert np.all(np.abs(y[core] - ref[core]) <= 5e-4 * np.abs(ref[core]))   # relative where no cancellation
    assert y[0] == 0.0 and y[special.index(20.0)] == 20.0 and y[special.index(1e4)] == f32(1e4)
    Yb = lp.bsr_linear(w, X, bias, gelu=True).float().cpu().double().numpy()[0]
    assert np.all(np.abs(Yb - ref) <= _ulp_bf16(ref) + tol)


@pytest.mark.parametrize("b", BLOCKS)
def test_all_zero_mask_is_bias(lp, b):
    m, n, k = 260, 256, 128
    X, W, bias, _ = _case(m, n, k, b, 0.5, 500 + _sid(b))
    bn, bk = _sides(b)
    mask = torch.zeros(n // bn, k // bk, dtype=torch.uint8, device="cuda")
    w = lp.pack_bsr(W, mask, b)
    Y = lp.bsr_linear(w, X, bias, out_dtype=torch.float32)
    assert torch.equal(Y, bias.expand(m, n))
    Yg = lp.bsr_linear(w, X, bias, gelu=True, out_dtype=torch.float32)
    ref = oracle.gelu(bias.cpu().double().numpy())
    assert np.allclose(Yg[0].cpu().double().numpy(), ref, rtol=1e-6, atol=1e-9)
    Yn = lp.bsr_linear(w, X, None, out_dtype=torch.float32)
    assert torch.count_nonzero(Yn) == 0


@pytest.mark.parametrize("m", [300, 120])
@pytest.mark.parametrize("b", BLOCKS)
def test_pruned_blocks_never_read(lp, b, m):
    n, k = 256, 256
    X, W, bias, mask = _case(m, n, k, b, 0.5, 600 + _sid(b))
    bn, bk = _sides(b)
    keep = mask.repeat_interleave(bn, 0).repeat_interleave(bk, 1).bool()
    Wp = W.clone()
    Wp[~keep] = float("nan")
    Wz = W.clone()
    Wz[~keep] = 0
    Yp = lp.bsr_linear(lp.pack_bsr(Wp, mask, b), X, bias, out_dtype=torch.float32)
    Yz = lp.bsr_linear(lp.pack_bsr(Wz, mask, b), X, bias, out_dtype=torch.float32)
    assert torch.equal(Yp, Yz) and torch.isfinite(Yp).all()


@pytest.mark.parametrize("m", [290, 100])
def test_single_block_closed_form(lp, m):
    n, k, b = 256, 256, 32
    X, W, bias, _ = _case(m, n, k, b, 0.5, 700, int_valued=True)
    mask = torch.zeros(n // b, k // b, dtype=torch.uint8, device="cuda")
    mask[3, 5] = 1
    Y = lp.bsr_linear(lp.pack_bsr(W, mask, b), X, bias, out_dtype=torch.float32)
    Xd, Wd = X.double().cpu(), W.double().cpu()
    expect = bias.double().cpu().expand(m, n).clone()
    expect[:, 96:128] += Xd[:, 160:192] @ Wd[96:128, 160:192].T
    assert torch.equal(Y.double().cpu(), expect)


@pytest.mark.parametrize("m", [400, 150])
def test_strided_input_output_and_guard_band(lp, m):
    n, k, b = 256, 128, 32
    X, W, bias, mask = _case(m, n, k, b, 0.5, 800)
    Xw = torch.zeros(m, k + 64, dtype=torch.bfloat16, device="cuda")
    Xw[:, 64:] = X
    canary = -12345.0
    Yw = torch.full((m + 7, n + 32), canary, dtype=torch.float32, device="cuda")
    w = lp.pack_bsr(W, mask, b)
    lp.bsr_linear(w, Xw[:, 64:], bias, out=Yw[:m, 16:16 + n])
    ref = _oracle(X, W, mask, b, bias)
    assert _norm_err(Yw[:m, 16:16 + n].cpu().double().numpy(), ref) <= TIGHT_TOL
    assert torch.all(Yw[m:] == canary) and torch.all(Yw[:, :16] == canary) and torch.all(Yw[:, 16 + n:] == canary)


@pytest.mark.parametrize("m", [301, 101])
@pytest.mark.parametrize("col0,extra", [(1, 33), (2, 34)])
def test_bf16_output_offsets_and_row_strides(lp, col0, extra, m):
    """bf16 output inside a larger buffer, with bases and row strides that rule out 16-byte stores
    (element stores instead); the canary around the output region survives and the values are
    those of a contiguous output."""
    n, k, b = 256, 128, 32
    X, W, bias, mask = _case(m, n, k, b, 0.5, 850 + col0)
    canary = torch.tensor(-777.0, dtype=torch.bfloat16)
    Yw = torch.full((m + 3, n + extra), canary.item(), dtype=torch.bfloat16, device="cuda")
    w = lp.pack_bsr(W, mask, b)
    for gelu in (False, True):
        lp.bsr_linear(w, X, bias, gelu=gelu, out=Yw[:m, col0:col0 + n])
        Yc = lp.bsr_linear(w, X, bias, gelu=gelu)
        assert torch.equal(Yw[:m, col0:col0 + n], Yc)
        assert torch.all(Yw[m:] == canary) and torch.all(Yw[:, :col0] == canary)
        assert torch.all(Yw[:, col0 + n:] == canary)
    ref = _oracle(X, W, mask, b, bias, gelu=True)
    assert np.all(np.abs(Yc.float().cpu().double().numpy() - ref) <= _bf16_tol(ref, X, W, mask, b, bias, gelu=True))


@pytest.mark.parametrize("b,m,n,k,gelu", [(32, 333, 256, 256, False), (16, 197, 768, 3072, False),
                                          ((64, 32), 300, 384, 512, True), (16, 300, 768, 3072, False)])
def test_residual_linear_is_the_bf16_sum(lp, b, m, n, k, gelu):
    """lpvit_bsr_linear_residual: Y equals, bit for bit, the plain linear's bf16 output plus R
    rounded to bf16 (the sum formed in float32), into a new tensor and in place (R = Y); the
    197-row case runs the small-m kernel with K cut over a cluster, the 300-row K = 3072 case the
    pair kernel's split units (the fix-up path)."""
    X, W, bias, mask = _case(m, n, k, b, 0.5, 1300 + _sid(b))
    w = lp.pack_bsr(W, mask, b)
    R = torch.randn(m, n, generator=torch.Generator().manual_seed(9)).to(torch.bfloat16).cuda()
    Y0 = lp.bsr_linear(w, X, bias, gelu=gelu)
    want = (Y0.float() + R.float()).to(torch.bfloat16)
    Y = lp.bsr_linear(w, X, bias, gelu=gelu, residual=R)
    assert torch.equal(Y, want)
    Z = R.clone()
    lp.bsr_linear(w, X, bias, gelu=gelu, out=Z, residual=Z)
    assert torch.equal(Z, want)


@pytest.mark.parametrize("m", [197, 300])   # small-m kernel (K over a cluster); pair kernel split units
@pytest.mark.parametrize("b", [32, (64, 32), (16, 32)])
def test_deterministic_repeats(lp, b, m):
    n, k = 768, 3072
    X, W, bias, mask = _case(m, n, k, b, 0.5, 900 + (0 if b == 32 else _sid(b)))
    w = lp.pack_bsr(W, mask, b)
    ws = lp.workspace_for(w, m)
    Y1 = lp.bsr_linear(w, X, bias, out_dtype=torch.float32, workspace=ws)
    Y2 = lp.bsr_linear(w, X, bias, out_dtype=torch.float32, workspace=ws)
    lp.check(ws)
    assert torch.equal(Y1, Y2)
    ref = _oracle(X, W, mask, b, bias)
    assert _norm_err(Y1.cpu().double().numpy(), ref) <= TIGHT_TOL


# ------------------------------------------------------------------------------ small m

# (m, n, k, b, gelu, f32): one token, a 256-feature weight and K = 3072 (eight K parts in one
# cluster); 17 tokens (eight parts); k = 400, not a multiple of the 64-column chunk (the last
# chunk reads zeros past k); n = 1152, 4.5 groups (row slices with no panel); 197 tokens over
# 64 x 32 blocks with GELU; m = 256, the largest the small-m kernel takes (four parts).
SMALL_M_CASES = [(1, 256, 3072, 32, False, True), (17, 768, 3072, 16, True, True),
                 (64, 384, 400, 16, False, True), (65, 1152, 384, 32, True, False),
                 (197, 3072, 768, (64, 32), True, False), (256, 512, 1536, (16, 32), False, True)]


@pytest.mark.parametrize("m,n,k,b,gelu,f32", SMALL_M_CASES)
def test_small_m_kernel_against_oracle(lp, m, n, k, b, gelu, f32):
    """Token counts up to 256 run the small-m kernel: fp32 output within the tight gate of the
    oracle, bf16 output within one bf16 ulp plus the fp32 accumulation bound, and the workspace
    error word clear."""
    X, W, bias, mask = _case(m, n, k, b, 0.5, 1500 + m + _sid(b))
    w = lp.pack_bsr(W, mask, b)
    ws = lp.workspace_for(w, m)
    Y = lp.bsr_linear(w, X, bias, gelu=gelu, out_dtype=torch.float32 if f32 else torch.bfloat16, workspace=ws)
    lp.check(ws)
    ref = _oracle(X, W, mask, b, bias, gelu=gelu)
    y = Y.float().cpu().double().numpy()
    if f32:
        assert _norm_err(y, ref) <= TIGHT_TOL
    else:
        assert np.all(np.abs(y - ref) <= _bf16_tol(ref, X, W, mask, b, bias, gelu=gelu))


def test_small_and_pair_kernels_agree_at_the_boundary(lp):
    """m = 256 (small-m kernel) and m = 257 (pair kernel) on the same weight: the first 256 rows
    agree within the fp32 accumulation bound of two summation orders, and both meet the oracle."""
    n, k, b = 768, 1536, 32
    X, W, bias, mask = _case(257, n, k, b, 0.5, 1600)
    w = lp.pack_bsr(W, mask, b)
    Ys = lp.bsr_linear(w, X[:256], bias, out_dtype=torch.float32)
    Yp = lp.bsr_linear(w, X, bias, out_dtype=torch.float32)
    bound = 2 * _acc_bound(X[:256], W, mask, b, bias)
    assert np.all(np.abs(Ys.cpu().double().numpy() - Yp[:256].cpu().double().numpy()) <= bound)
    ref = _oracle(X, W, mask, b, bias)
    assert _norm_err(Yp.cpu().double().numpy(), ref) <= TIGHT_TOL
    assert _norm_err(Ys.cpu().double().numpy(), ref[:256]) <= TIGHT_TOL


@pytest.mark.parametrize("b", [16, 64, (16, 32)])
def test_zipf_imbalanced_masks(lp, b):
    m, n, k = 513, 768, 3072
    X, W, bias, mask = _case(m, n, k, b, 0.6, 1000 + _sid(b), mask_kind="zipf")
    w = lp.pack_bsr(W, mask, b)
    Y = lp.bsr_linear(w, X, bias, gelu=True, out_dtype=torch.float32)
    ref = _oracle(X, W, mask, b, bias, gelu=True)
    assert _norm_err(Y.cpu().double().numpy(), ref) <= TIGHT_TOL


def test_empty_input_rows(lp):
    X, W, bias, mask = _case(4, 128, 128, 32, 0.5, 1100)
    w = lp.pack_bsr(W, mask, 32)
    Y = lp.bsr_linear(w, X[:0], bias)
    assert Y.shape == (0, 128)


def test_full_size_deit_b_fc1_sampled_rows(lp):
    """DeiT-B fc1 at batch 256 (M = 50432), 32x32 blocks, 50% sparsity, launched as in the bench;
    the oracle checks a seeded sample of rows plus the first and last token tile."""
    m, k, n, b = 50432, 768, 3072, 32
    X = inputs.activations(m, k, inputs.seed(3, 0, "X"), "cuda")
    W = inputs.weight(n, k, inputs.seed(3, 0, "W"), "cuda")
    bias = inputs.bias(n, inputs.seed(3, 0, "bias"), "cuda")
    mask = inputs.uniform_mask(n, k, b, 0.5, inputs.seed(3, 0, "mask"))
    w = lp.pack_bsr(W, mask.cuda(), b)
    Y = lp.bsr_linear(w, X, bias, gelu=True, out_dtype=torch.float32)
    rows = np.unique(np.concatenate([np.random.default_rng(0).choice(m, 96, replace=False),
                                     np.arange(0, 8), np.arange(m - 8, m)]))
    ref = _oracle(X, W, mask, b, bias, gelu=True, rows=torch.from_numpy(rows).cuda())
    assert _norm_err(Y[torch.from_numpy(rows).cuda()].cpu().double().numpy(), ref) <= TIGHT_TOL
