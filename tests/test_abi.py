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
