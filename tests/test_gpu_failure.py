"""Failure detection on the GPU without a fault: every device wait is bounded, and a wait that runs
out is reported on the host (lpvit_check) while the context stays usable. lpvit_selftest_wait makes
the GEMM's bounded wait run out on an mbarrier that nothing arrives on (and, in the second case,
makes another role of the CTA give up first via the abort flag); then an ordinary linear on the same
stream must still match the oracle."""
import time

import numpy as np
import pytest
import torch

import oracle

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def lp():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2407_02068_gb300 import build
    build.build()
    import paper_2407_02068_gb300 as lp
    return lp


def _waited_us(ws):
    return int(ws[12:16].cpu().numpy().view(np.uint32)[0])


def _stream():
    return torch.cuda.current_stream().cuda_stream


def test_wait_runs_out_and_is_reported(lp):
    from paper_2407_02068_gb300 import _lib
    ws = torch.zeros(4096, dtype=torch.uint8, device="cuda")
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    assert _lib.lpvit_selftest_wait(ws.data_ptr(), 50_000_000, 0, _stream()) == _lib.LPVIT_OK
    assert _lib.lpvit_check(ws.data_ptr(), _stream()) == _lib.LPVIT_ERR_TIMEOUT
    wall = time.perf_counter() - t0
    assert 0.05 <= wall < 5.0
    assert 50_000 <= _waited_us(ws) < 1_000_000
    assert _lib.lpvit_check(ws.data_ptr(), _stream()) == _lib.LPVIT_OK   # the error word was cleared


def test_abort_flag_ends_the_wait_early(lp):
    from paper_2407_02068_gb300 import _lib
    ws = torch.zeros(4096, dtype=torch.uint8, device="cuda")
    assert _lib.lpvit_selftest_wait(ws.data_ptr(), 2_000_000_000, 20_000_000, _stream()) == _lib.LPVIT_OK
    assert _lib.lpvit_check(ws.data_ptr(), _stream()) == _lib.LPVIT_ERR_TIMEOUT
    assert 20_000 <= _waited_us(ws) < 1_000_000     # well before the 2 s limit


def test_context_still_computes_after_a_timeout(lp):
    from paper_2407_02068_gb300 import _lib, inputs
    ws = torch.zeros(4096, dtype=torch.uint8, device="cuda")
    assert _lib.lpvit_selftest_wait(ws.data_ptr(), 10_000_000, 0, _stream()) == _lib.LPVIT_OK
    assert _lib.lpvit_check(ws.data_ptr(), _stream()) == _lib.LPVIT_ERR_TIMEOUT
    m, n, k, b = 300, 256, 256, 32
    g = torch.Generator().manual_seed(99)
    X = torch.randn(m, k, generator=g).to(torch.bfloat16).cuda()
    W = (torch.randn(n, k, generator=g) * 0.02).to(torch.bfloat16).cuda()
    bias = (torch.randn(n, generator=g) * 0.02).cuda()
    mask = inputs.uniform_mask(n, k, b, 0.5, 5).cuda()
    w = lp.pack_bsr(W, mask, b)
    ws2 = lp.workspace_for(w, m)
    Y = lp.bsr_linear(w, X, bias, out_dtype=torch.float32, workspace=ws2)
    lp.check(ws2)   # raises if a wait of the GEMM ran out
    ref = oracle.linear(inputs.bf16_bits(X.cpu()), inputs.bf16_bits(W.cpu()), mask.cpu().numpy(), b,
                        bias.cpu().numpy(), False)
    y = Y.cpu().double().numpy()
    assert np.max(np.abs(y - ref)) / np.sqrt(np.mean(ref ** 2)) <= 1e-4
