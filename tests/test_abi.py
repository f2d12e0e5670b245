"""CPU checks of the C ABI: the library builds, loads, exports every function include/lpvit.h
declares, and rejects bad arguments before touching a GPU."""
import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def lib():
    from paper_2407_02068_gb300 import _lib, build
    build.build()
    return _lib


def _declared_functions():
    src = open(os.path.join(ROOT, "include", "lpvit.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(lpvit_[a-z_]+)\s*\(", src)))


def test_every_declared_symbol_is_exported(lib):
    names = _declared_functions()
    assert {"lpvit_pack_bsr", "lpvit_bsr_linear", "lpvit_bsr_linear_gelu"} <= set(names)
    raw = ctypes.CDLL(lib.LIB)
    for name in names:
        assert hasattr(raw, name), name
    assert set(names) == set(lib.EXPORTS)


def test_sched_bytes_and_status_strings(lib):
    assert lib.lpvit_sched_bytes(1152, 384, 32, 32) > 0
    assert lib.lpvit_sched_bytes(1152, 384, 64, 32) > 0   # 64 rows x 32 columns
    assert lib.lpvit_sched_bytes(1152, 384, 16, 32) == lib.lpvit_sched_bytes(1152, 384, 64, 32)  # bn: list only
    assert lib.lpvit_sched_bytes(1152, 384, 24, 32) == 0  # unsupported block height
    assert lib.lpvit_sched_bytes(1152, 384, 32, 24) == 0  # unsupported block width
    assert lib.lpvit_sched_bytes(1000, 384, 32, 32) == 0  # n not a multiple of bn
    assert lib.lpvit_sched_bytes(1152, 400, 64, 32) == 0  # k not a multiple of bk
    for st in range(6):
        assert lib.status_string(st)


def test_bad_arguments_are_rejected_without_a_gpu(lib):
    bsr = lib.lpvit_bsr(1152, 384, 32, 32, 432, None, None, None, None, 0)
    st, _ = lib.lpvit_pack_bsr(None, None, bsr, False, None)
    assert st == lib.LPVIT_ERR_INVALID_ARG
    bad_b = lib.lpvit_bsr(1152, 384, 24, 24, 432, None, None, None, None, 0)
    st, _ = lib.lpvit_pack_bsr(None, None, bad_b, False, None)
    assert st == lib.LPVIT_ERR_UNSUPPORTED
    for bn, bk in ((64, 24), (8, 32), (128, 32)):
        st, _ = lib.lpvit_pack_bsr(None, None, lib.lpvit_bsr(1152, 384, bn, bk, 432, None, None, None, None, 0),
                                   False, None)
        assert st == lib.LPVIT_ERR_UNSUPPORTED, (bn, bk)
    assert lib.lpvit_bsr_linear(bsr, None, 197, 384, None, None, 1152, 0, None, 0, None) == lib.LPVIT_ERR_INVALID_ARG
    assert lib.lpvit_bsr_linear(bsr, None, -1, 384, None, None, 1152, 0, None, 0, None) == lib.LPVIT_ERR_INVALID_ARG
    assert lib.lpvit_bsr_linear(bsr, None, 0, 384, None, None, 1152, 0, None, 0, None) == lib.LPVIT_OK  # empty
    assert lib.lpvit_bsr_linear_gelu(bad_b, None, 4, 384, None, None, 1152, 0, None, 0, None) == \
        lib.LPVIT_ERR_UNSUPPORTED
    # misaligned X (not 16-byte aligned) / ldx not a multiple of 8
    fake = ctypes.c_void_p(0x1000)
    assert lib.lpvit_bsr_linear(bsr, 0x1002, 4, 384, None, 0x200000, 1152, 0, 0x100000, 1 << 20, None) == \
        lib.LPVIT_ERR_INVALID_ARG
    assert lib.lpvit_bsr_linear(bsr, fake.value, 4, 388, None, 0x200000, 1152, 0, 0x100000, 1 << 20, None) == \
        lib.LPVIT_ERR_INVALID_ARG
    assert lib.lpvit_check(None, None) == lib.LPVIT_ERR_INVALID_ARG
    # residual linear: R present, gelu 0/1, R 16-byte aligned with ldr >= n and ldr % 8 == 0, R either
    # Y itself (then the call proceeds to the work-list size check) or clear of Y
    rb = lib.lpvit_bsr(1152, 384, 32, 32, 432, None, None, None, 0x400000, 0)
    X, Y, ws = 0x1000, 0x200000, 0x100000

    def res(R, ldr, gelu=0, ldy=1152):
        return lib.lpvit_bsr_linear_residual(rb, X, 4, 384, None, gelu, R, ldr, Y, ldy, ws, 1 << 20, None)
    assert res(None, 1152) == lib.LPVIT_ERR_INVALID_ARG
    assert res(0x300000, 1152, gelu=2) == lib.LPVIT_ERR_INVALID_ARG
    assert res(0x300002, 1152) == lib.LPVIT_ERR_INVALID_ARG           # misaligned
    assert res(0x300000, 1148) == lib.LPVIT_ERR_INVALID_ARG           # ldr < n
    assert res(0x300000, 1156) == lib.LPVIT_ERR_INVALID_ARG           # ldr % 8
    assert res(Y + 16, 1152) == lib.LPVIT_ERR_INVALID_ARG             # overlaps Y without being Y
    assert res(Y, 1160, ldy=1152) == lib.LPVIT_ERR_INVALID_ARG        # Y's rows, another stride
    assert res(Y, 1152) == lib.LPVIT_ERR_WORKSPACE                    # in place: accepted, no work list
    assert res(0x300000, 1152) == lib.LPVIT_ERR_WORKSPACE             # clear of Y: accepted
    # the batched pack checks every job before launching anything
    assert lib.load().lpvit_pack_bsr_many(0, None, None, None, None) == lib.LPVIT_OK
    assert lib.load().lpvit_pack_bsr_many(-1, None, None, None, None) == lib.LPVIT_ERR_INVALID_ARG
    assert lib.load().lpvit_pack_bsr_many(1, None, None, None, None) == lib.LPVIT_ERR_INVALID_ARG
    assert lib.lpvit_pack_bsr_many([0x1000], [0x2000], [bad_b], None) == lib.LPVIT_ERR_UNSUPPORTED
    assert lib.lpvit_pack_bsr_many([0x1000, 0], [0x2000, 0x2000], [bsr, bsr], None) == lib.LPVIT_ERR_INVALID_ARG
    # the Taylor block mask validates before launching anything
    tm = lib.lpvit_taylor_block_mask
    assert tm(0x1000, 0x2000, 64, 64, 24, 24, 0.5, 0x3000, 0x4000, None) == lib.LPVIT_ERR_UNSUPPORTED
    assert tm(0x1000, 0x2000, 64, 64, 32, 24, 0.5, 0x3000, 0x4000, None) == lib.LPVIT_ERR_UNSUPPORTED
    assert tm(0x1000, 0x2000, 64, 48, 32, 32, 0.5, 0x3000, 0x4000, None) == lib.LPVIT_ERR_INVALID_ARG   # k % bk
    assert tm(0x1000, 0x2000, 96, 64, 64, 32, 0.5, 0x3000, 0x4000, None) == lib.LPVIT_ERR_INVALID_ARG   # n % bn
    for bad_alpha in (-0.1, 1.5, float("nan")):
        assert tm(0x1000, 0x2000, 64, 64, 32, 32, bad_alpha, 0x3000, 0x4000, None) == lib.LPVIT_ERR_INVALID_ARG
    assert tm(0, 0x2000, 64, 64, 32, 32, 0.5, 0x3000, 0x4000, None) == lib.LPVIT_ERR_INVALID_ARG
    assert tm(0x1008, 0x2000, 64, 64, 32, 32, 0.5, 0x3000, 0x4000, None) == lib.LPVIT_ERR_INVALID_ARG  # W alignment
    assert tm(0x1000, 0x2000, 65536, 65536, 16, 16, 0.5, 0x3000, 0x4000, None) == \
        lib.LPVIT_ERR_UNSUPPORTED  # > 2^20 blocks
    # the wait self-test validates before launching anything
    assert lib.lpvit_selftest_wait(0, 10 ** 6, 0, None) == lib.LPVIT_ERR_INVALID_ARG          # no workspace
    assert lib.lpvit_selftest_wait(0x100010, 10 ** 6, 0, None) == lib.LPVIT_ERR_INVALID_ARG   # misaligned
    assert lib.lpvit_selftest_wait(0x100000, 0, 0, None) == lib.LPVIT_ERR_INVALID_ARG         # no limit
    assert lib.lpvit_selftest_wait(0x100000, 11 * 10 ** 9, 0, None) == lib.LPVIT_ERR_INVALID_ARG  # > 10 s
    assert lib.lpvit_selftest_wait(0x100000, 10 ** 6, 10 ** 6, None) == lib.LPVIT_ERR_INVALID_ARG  # abort >= limit


def test_lambda_search_host_matches_the_oracle(lib):
    """lpvit_lambda_search is host code: it runs here, without a GPU, against the oracle."""
    import math
    import numpy as np
    from oracle import alloc
    # the hand-worked example, given as delta curves (D = delta^2)
    d1 = [math.sqrt(v) for v in (0, 1, 3, 7)]
    d2 = [math.sqrt(v) for v in (0, 2, 4, 6)]
    for beta, R in ((0, 0.5), (0, 0.95), (2, 0.5), (2, 0.1), (0, 1.0)):
        st, ks, lam, ratio = lib.lpvit_lambda_search([d1, d2], 3, [1, 3], [1, 2], beta, R)
        want = alloc.lambda_search([alloc.distortion(d1), alloc.distortion(d2)], 3, [1, 3], [1, 2], beta, R)
        assert st == lib.LPVIT_OK and (lam, ks, ratio) == (want[0], want[1], want[2]), (beta, R)
    rng = np.random.default_rng(9)
    for trial in range(20):
        L, steps = int(rng.integers(1, 30)), int(rng.integers(1, 25))
        deltas = [np.concatenate([[0.0], np.cumsum(rng.standard_normal(steps))]) for _ in range(L)]
        F = rng.uniform(0.5, 4.0, L)
        c = rng.uniform(0.0, 3.0, L)
        beta, R = float(rng.uniform(0, 2)), float(rng.uniform(-0.1, 1.1))
        st, ks, lam, ratio = lib.lpvit_lambda_search(deltas, steps, F, c, beta, R)
        want = alloc.lambda_search([alloc.distortion(d) for d in deltas], steps, F, c, beta, R)
        assert st == lib.LPVIT_OK and ks == want[1] and lam == want[0] and ratio == want[2], trial


def test_allocation_arguments_are_checked_without_a_gpu(lib):
    L = lib.load()
    assert lib.lpvit_delta_curve_workspace_bytes(8, 768, 3072, 32, 32, 20) > 8 * 768 * 3072 // 1024 * 8
    assert lib.lpvit_delta_curve_workspace_bytes(0, 768, 3072, 32, 32, 20) == 0
    assert lib.lpvit_delta_curve_workspace_bytes(8, 768, 3000, 32, 32, 20) == 0
    assert lib.lpvit_delta_curve_workspace_bytes(8, 768, 3072, 32, 32, 0) == 0
    dc = lib.lpvit_delta_curve
    ok = dict(W_ptr=0x1000, G_ptr=0x2000, nsamples=8, n=256, k=256, bn=32, bk=32, kappa=0.1, steps=10,
              delta_ptr=0x3000, ws_ptr=0x100000, ws_bytes=1 << 30, stream=None)
    def call(**kw):
        a = dict(ok, **kw)
        return dc(a["W_ptr"], a["G_ptr"], a["nsamples"], a["n"], a["k"], a["bn"], a["bk"], a["kappa"], a["steps"],
                  a["delta_ptr"], a["ws_ptr"], a["ws_bytes"], a["stream"])
    assert call(bn=24) == lib.LPVIT_ERR_UNSUPPORTED
    assert call(n=65536, k=65536, bn=16, bk=16) == lib.LPVIT_ERR_UNSUPPORTED  # > 2^20 blocks
    for bad in (dict(nsamples=0), dict(nsamples=1025), dict(steps=0), dict(steps=5000), dict(kappa=-1.0),
                dict(kappa=float("inf")), dict(kappa=float("nan")), dict(W_ptr=0), dict(G_ptr=0x2004),
                dict(delta_ptr=0x3004), dict(ws_ptr=0x100010), dict(k=250)):
        assert call(**bad) == lib.LPVIT_ERR_INVALID_ARG, bad
    assert call(ws_bytes=16) == lib.LPVIT_ERR_WORKSPACE
    st, *_ = lib.lpvit_lambda_search([[0.0, 1.0]], 1, [0.0], [1.0], 0.0, 0.5)   # flops must be > 0
    assert st == lib.LPVIT_ERR_INVALID_ARG
    st, *_ = lib.lpvit_lambda_search([[0.0, float("nan")]], 1, [1.0], [1.0], 0.0, 0.5)
    assert st == lib.LPVIT_ERR_INVALID_ARG
    assert L.lpvit_lambda_search(0, 1, None, None, None, 0.0, 0.5, None, None, None) == lib.LPVIT_ERR_INVALID_ARG


def test_encoder_kernel_arguments_are_checked_without_a_gpu(lib):
    ln = lib.lpvit_add_layernorm
    assert ln(0x1000, None, 0x2000, 0x3000, 0, 384, 1e-6, None, 0x4000, None) == lib.LPVIT_OK   # no rows
    for bad in ((0x1000, None, 0x2000, 0x3000, 4, 1028, 1e-6, None, 0x4000),     # D > 1024
                (0x1000, None, 0x2000, 0x3000, 4, 100, 1e-6, None, 0x4000),      # D % 8
                (0x1000, None, 0x2000, 0x3000, 4, 384, 0.0, None, 0x4000),       # eps
                (0x1000, 0x5000, 0x2000, 0x3000, 4, 384, 1e-6, None, 0x4000),    # r without sum_out
                (0x1008, None, 0x2000, 0x3000, 4, 384, 1e-6, None, 0x4000),      # alignment
                (0, None, 0x2000, 0x3000, 4, 384, 1e-6, None, 0x4000)):
        assert ln(*bad, None) == lib.LPVIT_ERR_INVALID_ARG, bad
    at = lib.lpvit_attention
    assert at(0x1000, 2, 197, 6, 32, 0x2000, None) == lib.LPVIT_ERR_UNSUPPORTED    # head_dim
    assert at(0x1000, 2, 209, 6, 64, 0x2000, None) == lib.LPVIT_ERR_UNSUPPORTED    # tokens
    assert at(0x1000, 0, 197, 6, 64, 0x2000, None) == lib.LPVIT_OK                 # no images
    assert at(0x1008, 2, 197, 6, 64, 0x2000, None) == lib.LPVIT_ERR_INVALID_ARG
    assert at(0x1000, 2, 197, 0, 64, 0x2000, None) == lib.LPVIT_ERR_INVALID_ARG


def test_chain_arguments_are_checked_without_a_gpu(lib):
    """lpvit_bsr_linear_chain checks every link (as lpvit_bsr_linear would) before launching, and
    sizes its workspace as the control block, the largest split partials and a counter per
    (linear, token tile) of one launch."""
    L = lib.load()
    sched = 0x400000
    b_qkv = lib.lpvit_bsr(2304, 768, 32, 32, 1728, None, None, None, sched, 1 << 24)
    b_proj = lib.lpvit_bsr(768, 768, 32, 32, 576, None, None, None, sched, 1 << 24)
    X, Y, ws = 0x1000000, 0x8000000, 0x100000
    m = 50432
    rows = [(b_qkv, X, 768, None, Y, 2304, 0), (b_proj, Y + 2 * 1536, 2304, None, 0x20000000, 768, 0)]
    links = lib.chain_links(rows)
    # a counter per (linear, 256-token tile) after the 256-byte control block (no split at this m)
    tiles = (m + 255) // 256
    assert lib.lpvit_chain_workspace_bytes(links, 2, m) == 256 + (2 * tiles * 4 + 255) // 256 * 256
    assert lib.lpvit_chain_workspace_bytes(None, 2, m) == 0
    assert lib.lpvit_chain_workspace_bytes(links, 0, m) == 0
    bad = lib.chain_links([(lib.lpvit_bsr(2304, 770, 32, 32, 1, None, None, None, sched, 1 << 24),
                            X, 776, None, Y, 2304, 0)])
    assert lib.lpvit_chain_workspace_bytes(bad, 1, m) == 0
    chain = L.lpvit_bsr_linear_chain
    assert chain(links, 0, m, ws, 1 << 20, None) == lib.LPVIT_OK          # nothing to do
    assert chain(links, 2, 0, ws, 1 << 20, None) == lib.LPVIT_OK          # no tokens
    assert chain(links, -1, m, ws, 1 << 20, None) == lib.LPVIT_ERR_INVALID_ARG
    assert chain(None, 2, m, ws, 1 << 20, None) == lib.LPVIT_ERR_INVALID_ARG
    assert chain(links, 2, m, None, 1 << 20, None) == lib.LPVIT_ERR_INVALID_ARG
    assert chain(links, 2, m, ws + 16, 1 << 20, None) == lib.LPVIT_ERR_INVALID_ARG   # workspace alignment
    assert chain(links, 2, -5, ws, 1 << 20, None) == lib.LPVIT_ERR_INVALID_ARG

    def one(**kw):
        r = dict(bsr=b_qkv, X=X, ldx=768, bias=None, Y=Y, ldy=2304, gelu=0)
        r.update(kw)
        return chain(lib.chain_links([tuple(r.values())]), 1, m, ws, 1 << 20, None)
    assert one(gelu=2) == lib.LPVIT_ERR_INVALID_ARG
    assert one(bsr=None) == lib.LPVIT_ERR_INVALID_ARG
    assert one(X=X + 2) == lib.LPVIT_ERR_INVALID_ARG        # X not 16-byte aligned
    assert one(ldx=772) == lib.LPVIT_ERR_INVALID_ARG        # ldx % 8
    assert one(ldy=2300) == lib.LPVIT_ERR_INVALID_ARG       # ldy < n
    assert one(Y=X) == lib.LPVIT_ERR_INVALID_ARG            # Y overlaps X
    assert one(bsr=bad[0].bsr.contents) == lib.LPVIT_ERR_INVALID_ARG   # k not a multiple of bk
    # a bad second link stops the call before the first one runs
    rows_bad = [rows[0], (b_proj, Y + 2 * 1536, 2304, None, 0x20000000, 768, 5)]
    assert chain(lib.chain_links(rows_bad), 2, m, ws, 1 << 20, None) == lib.LPVIT_ERR_INVALID_ARG
