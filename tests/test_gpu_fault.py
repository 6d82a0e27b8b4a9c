"""Failure detection on the GPU without a GPU fault.

A host-side hook makes the GEMM's TMA producer skip its copies; every
consumer wait is time-bounded, so the kernel gives up after the set limit,
reports the timeout in the status word, releases its tensor memory and exits.
The context must stay usable: the same GEMM then runs correctly, and a slice
whose GEMMs timed out reports SKY_ERR_TIMEOUT from sky_slice_sync.
"""
import ctypes as C

import numpy as np
import pytest

from paper_2202_11836_gb300 import _lib as L
from paper_2202_11836_gb300 import synth
from parity_util import l2rel, to_device

pytestmark = pytest.mark.gpu
torch = pytest.importorskip("torch")


def P(t):
    return C.c_void_p(0 if t is None else int(t.data_ptr()))


def stream():
    return C.c_void_p(int(torch.cuda.current_stream().cuda_stream))


def test_gemm_wait_timeout_is_reported_and_context_survives():
    M, N, K = 256, 512, 256
    g = np.random.default_rng(1)
    A = synth.round_bf16(g.normal(0, 1, (M, K)).astype(np.float32))
    W = synth.round_bf16(g.normal(0, 0.05, (N, K)).astype(np.float32))
    a, w = to_device(A, "bf16"), to_device(W, "bf16")
    c = torch.zeros((M, N), dtype=torch.bfloat16, device="cuda")
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    L.lib().sky_debug_gemm_fault(50_000_000, 1)  # 50 ms per wait, no TMA copies
    try:
        L.call("sky_gemm", L.SKY_GEMM_XWT, M, N, K, 0, P(a), P(w), P(c), 0, 0, None, None, None,
               None, 0, P(status), stream())
        torch.cuda.synchronize()
    finally:
        L.lib().sky_debug_gemm_fault(0, 0)
    assert int(status.item()) & 2, "timeout bit not set"
    # the context is intact: the same GEMM now runs and is correct
    status.zero_()
    L.call("sky_gemm", L.SKY_GEMM_XWT, M, N, K, 0, P(a), P(w), P(c), 0, 0, None, None, None,
           None, 0, P(status), stream())
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    ref = A.astype(np.float64) @ W.astype(np.float64).T
    assert l2rel(c.float().cpu().numpy(), ref) <= 4e-3


def test_slice_reports_timeout_then_recovers():
    from paper_2202_11836_gb300.slice import EncoderSlice
    w = synth.custom("fault", layers=1, hidden=128, heads=2, ffn=256, seq=64, batch=2)
    X, lens = synth.activations(w), synth.lengths(w)
    with EncoderSlice(128, 2, 256, 0, 1, 2, 64) as s:
        s.set_params(0, synth.layer_params(0, 128, 256, "bf16", affine="random"))
        x = to_device(X, "bf16")
        ln = torch.from_numpy(lens).cuda()
        L.lib().sky_debug_gemm_fault(20_000_000, 1)
        try:
            s.forward(x, ln)
            with pytest.raises(L.SkyError) as e:
                s.sync()
            assert e.value.status == L.SKY_ERR_TIMEOUT
        finally:
            L.lib().sky_debug_gemm_fault(0, 0)
        y = s.forward(x, ln)
        s.sync()  # OK again
        assert torch.isfinite(y.float()).all()
