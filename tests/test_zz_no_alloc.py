"""sky_column_sum_noalloc: the bias-gradient column sum without any device
allocation (its scratch is a fixed device array inside the library), for
callers that draw all device memory from a pool they do not own, or must not
allocate inside their step loop.

Checked against sky_column_sum (caller workspace) on the same inputs, on two
calls in a row with different data (the shared scratch keeps the previous
call's contents), and for the clean rejection of a size beyond its scratch.
This file is collected last so that a failure here cannot hide another test.
"""
import ctypes as C

import numpy as np
import pytest

from paper_2202_11836_gb300 import _lib as L

pytestmark = pytest.mark.gpu
torch = pytest.importorskip("torch")


def P(t):
    return C.c_void_p(0 if t is None else int(t.data_ptr()))


def stream():
    return C.c_void_p(int(torch.cuda.current_stream().cuda_stream))


@pytest.mark.parametrize("dt,T,N", [("bf16", 8192, 4096), ("bf16", 333, 1000), ("fp32", 64, 384)])
def test_noalloc_matches_workspace_version(dt, T, N):
    td = torch.bfloat16 if dt == "bf16" else torch.float32
    code = L.SKY_DTYPE_BF16 if dt == "bf16" else L.SKY_DTYPE_FP32
    g = torch.Generator(device="cuda").manual_seed(T + N)
    for call in range(2):  # second call: new data over the previous call's scratch
        x = torch.randn((T, N), device="cuda", generator=g).to(td) * (1 + call)
        ref = torch.empty(N, dtype=torch.float32, device="cuda")
        wsb = L.lib().sky_column_sum_workspace_bytes(T, N)
        ws = torch.empty(wsb, dtype=torch.uint8, device="cuda")
        L.call("sky_column_sum", P(x), T, N, code, P(ref), P(ws), wsb, stream())
        got = torch.full((N,), float("nan"), dtype=torch.float32, device="cuda")
        L.call("sky_column_sum_noalloc", P(x), T, N, code, P(got), stream())
        torch.cuda.synchronize()
        r, o = ref.cpu().numpy(), got.cpu().numpy()
        assert np.isfinite(o).all()
        assert np.linalg.norm(o - r) <= 1e-6 * np.linalg.norm(r), call
        exact = x.double().sum(0).cpu().numpy()
        assert np.linalg.norm(o - exact) <= 1e-5 * np.linalg.norm(exact)


def test_noalloc_rejects_oversized_request():
    N = 1 << 19  # partials of 2 MiB: beyond the fixed scratch
    x = torch.zeros((1, N), dtype=torch.float32, device="cuda")
    out = torch.zeros(N, dtype=torch.float32, device="cuda")
    st = L.lib().sky_column_sum_noalloc(P(x), 1, N, L.SKY_DTYPE_FP32, P(out), stream())
    assert st == L.SKY_ERR_INVALID_ARG
    assert "scratch" in L.last_error()
