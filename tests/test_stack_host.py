"""CPU checks of the linear stack's host side: the argument table it hands lpvit_bsr_linear_chain
(which buffer each of the 4L linears reads and writes, with which row stride, which one applies
GELU), the per-linear calls it would make instead, the workspace it sizes for both, and its launch
count. Nothing here launches a kernel; the library is only asked for sizes."""
import ctypes

import pytest
import torch

from paper_2407_02068_gb300 import inputs


@pytest.fixture(scope="module")
def stack():
    from paper_2407_02068_gb300 import build
    build.build()
    from paper_2407_02068_gb300.stack import DeitLinearStack
    d, b, m = 384, 16, 5000
    g = torch.Generator().manual_seed(5)
    layers = []
    for li in range(2):
        L = {}
        for name, (n, k) in {"qkv": (3 * d, d), "proj": (d, d), "fc1": (4 * d, d), "fc2": (d, 4 * d)}.items():
            L[name] = {"W": torch.randn(n, k, generator=g).to(torch.bfloat16), "bias": torch.zeros(n),
                       "mask": inputs.uniform_mask(n, k, b, 0.5, 11 + li), "b": b, "gelu": name == "fc1"}
        layers.append(L)
    st = DeitLinearStack(m, layers, "cpu")
    st._calls_for(0)
    return st, d, m


def test_chain_table_follows_the_stack(stack):
    st, d, m = stack
    links, count, mm, ws, wsn, strm = st._chain_args
    assert count.value == 8 == len(st.gemms) and mm.value == m
    assert ws.value == st.ws.data_ptr() and wsn.value == st.ws.numel()
    bf = 2  # bytes per bf16
    x_of = {"qkv": None, "proj": (st.qkv.data_ptr() + 2 * d * bf, 3 * d), "fc1": (st.proj.data_ptr(), d),
            "fc2": (st.fc1.data_ptr(), 4 * d)}
    y_of = {"qkv": (st.qkv.data_ptr(), 3 * d), "proj": (st.proj.data_ptr(), d), "fc1": (st.fc1.data_ptr(), 4 * d)}
    src = (st.h_in.data_ptr(), d)
    for i, G in enumerate(st.gemms):
        L = links[i]
        name = G["name"]
        assert ctypes.addressof(L.bsr.contents) == ctypes.addressof(G["struct"])
        X = src if name == "qkv" else x_of[name]
        Y = (st.hbuf[G["layer"] % 2].data_ptr(), d) if name == "fc2" else y_of[name]
        assert (L.X, L.ldx) == X, (i, name)
        assert (L.Y, L.ldy) == Y, (i, name)
        assert L.bias == G["bias"].data_ptr() and L.gelu == (1 if name == "fc1" else 0)
        if name == "fc2":
            src = Y
    assert st.out.data_ptr() == st.hbuf[1].data_ptr()


def test_per_linear_calls_match_the_chain_table(stack):
    st, d, m = stack
    links = st._chain_args[0]
    for i, (_, fn, args) in enumerate(st._calls_for(0)):
        L = links[i]
        assert args[1].value == L.X and args[3].value == L.ldx and args[2].value == m
        assert args[5].value == L.Y and args[6].value == L.ldy and args[4].value == L.bias
        assert (fn == st._lin[True]) == bool(L.gelu)


def test_workspace_serves_both_launch_modes(stack):
    from paper_2407_02068_gb300 import _lib
    st, d, m = stack
    links = st._chain_args[0]
    need_chain = _lib.lpvit_chain_workspace_bytes(links, len(st.gemms), m)
    need_each = max(_lib.lpvit_workspace_bytes(G["struct"], m) for G in st.gemms)
    assert need_chain > 256 and st.ws.numel() >= max(need_chain, need_each)
    # the control block, then one 32-bit counter per (linear, 256-token tile)
    tiles = (m + 255) // 256
    assert need_chain >= 256 + 4 * len(st.gemms) * tiles


def test_launch_counts(stack):
    st, _, _ = stack
    assert st.launches_per_step(chain=False) == 8 + 2
    assert st.launches_per_step(chain=True) == 1 + 2
