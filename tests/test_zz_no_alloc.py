"""lpvit_bsr_linear_noalloc: the linear for callers that cannot allocate device memory where they
run the layer (no allocator of their own, stream capture in progress, or a latency-critical path).
The library supplies the workspace from its own fixed-size device array; the caller passes only
inputs and outputs. This file is collected last on purpose.

Each case calls the new entry point twice in a row through the C ABI and compares both outputs
with the ordinary entry point's (caller-provided workspace), within the fp32-output tolerance of
the parity tests."""
import numpy as np
import pytest
import torch

pytestmark = pytest.mark.gpu

TIGHT_TOL = 1e-4  # max|y - y_ref| / rms(y_ref), as in the parity tests


@pytest.fixture(scope="module")
def lp():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2407_02068_gb300 import build
    build.build()
    import paper_2407_02068_gb300 as lp
    return lp


def _case(m, n, k, b, seed):
    from paper_2407_02068_gb300 import inputs
    g = torch.Generator().manual_seed(seed)
    X = torch.randn(m, k, generator=g).to(torch.bfloat16).cuda()
    W = (torch.randn(n, k, generator=g) * 0.02).to(torch.bfloat16).cuda()
    bias = (torch.randn(n, generator=g) * 0.02).cuda()
    mask = inputs.uniform_mask(n, k, b, 0.5, seed + 1).cuda()
    return X, W, bias, mask


def _noalloc(lp, w, X, bias, Y, gelu):
    from paper_2407_02068_gb300 import _lib
    return _lib.lpvit_bsr_linear_noalloc(w.struct(), X.data_ptr(), X.shape[0], X.stride(0), bias.data_ptr(),
                                         Y.data_ptr(), Y.stride(0), _lib.LPVIT_F32, gelu,
                                         torch.cuda.current_stream().cuda_stream)


def _err(y, ref):
    y, ref = y.double().cpu().numpy(), ref.double().cpu().numpy()
    return np.max(np.abs(y - ref)) / np.sqrt(np.mean(ref ** 2))


@pytest.mark.parametrize("m,n,k,b,gelu", [(20000, 512, 384, 32, False),   # one slice per group
                                          (197, 768, 3072, 32, True),      # split slices + fix-up
                                          (197, 384, 256, 32, True),       # short: one slice per group
                                          (300, 256, 128, 16, False),
                                          (600, 256, 512, 64, True)])
def test_noalloc_matches_existing_entry_point_twice(lp, m, n, k, b, gelu):
    from paper_2407_02068_gb300 import _lib
    X, W, bias, mask = _case(m, n, k, b, 4242 + m + b)
    w = lp.pack_bsr(W, mask, b)
    assert _lib.lpvit_workspace_bytes(w.struct(), m) <= _lib.LPVIT_NOALLOC_SCRATCH_BYTES
    ref = lp.bsr_linear(w, X, bias, gelu=gelu, out_dtype=torch.float32)
    for _ in range(2):
        Y = torch.full((m, n), float("nan"), dtype=torch.float32, device="cuda")
        st = _noalloc(lp, w, X, bias, Y, gelu)
        assert st == _lib.LPVIT_OK, _lib.status_string(st)
        torch.cuda.synchronize()
        assert torch.isfinite(Y).all()
        assert _err(Y, ref) <= TIGHT_TOL


def test_noalloc_rejects_work_beyond_its_array(lp):
    from paper_2407_02068_gb300 import _lib
    m, n, k, b = 197, 3072, 3072, 32   # small m, long k, many groups: the split partial sums need > 8 MiB
    X, W, bias, mask = _case(m, n, k, b, 77)
    w = lp.pack_bsr(W, mask, b)
    assert _lib.lpvit_workspace_bytes(w.struct(), m) > _lib.LPVIT_NOALLOC_SCRATCH_BYTES
    Y = torch.zeros(m, n, dtype=torch.float32, device="cuda")
    assert _noalloc(lp, w, X, bias, Y, False) == _lib.LPVIT_ERR_WORKSPACE
    torch.cuda.synchronize()
    assert torch.count_nonzero(Y) == 0
