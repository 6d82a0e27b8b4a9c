"""Out-of-bounds write checks (GPU), in place of a memory sanitizer.

Every output and scratch buffer an op receives is the middle of a larger
allocation whose leading and trailing 4 KiB hold a byte pattern.  Each op
runs on ragged sizes (rows, columns and sequence lengths off the tile
grid), and afterwards both bands must still hold the pattern: no kernel
wrote outside the ranges its arguments describe.
"""
import ctypes as C
import math

import numpy as np
import pytest

from paper_2202_11836_gb300 import _lib as L
from paper_2202_11836_gb300 import synth

pytestmark = pytest.mark.gpu
torch = pytest.importorskip("torch")

GUARD = 4096      # bytes on each side (keeps the payload 256-byte aligned)
PATTERN = 0xA5


class Guarded:
    """A tensor of `shape` and `dtype` inside a patterned allocation."""

    def __init__(self, shape, dtype):
        shape = tuple(shape)
        esz = torch.empty((), dtype=dtype).element_size()
        n = max(1, math.prod(shape)) * esz
        self.raw = torch.full((GUARD + n + GUARD,), PATTERN, dtype=torch.uint8, device="cuda")
        self.t = self.raw[GUARD:GUARD + n].view(dtype)[:math.prod(shape)].view(shape)

    def intact(self):
        return bool((self.raw[:GUARD] == PATTERN).all()) and \
            bool((self.raw[-GUARD:] == PATTERN).all())


def P(t):
    if isinstance(t, Guarded):
        t = t.t
    return C.c_void_p(0 if t is None else int(t.data_ptr()))


def stream():
    return C.c_void_p(int(torch.cuda.current_stream().cuda_stream))


def code(dt):
    return L.SKY_DTYPE_BF16 if dt == "bf16" else L.SKY_DTYPE_FP32


def tdt(dt):
    return torch.bfloat16 if dt == "bf16" else torch.float32


def rand(shape, dt, std=1.0, seed=0):
    g = torch.Generator(device="cuda").manual_seed(seed)
    return (std * torch.randn(shape, device="cuda", generator=g)).to(tdt(dt))


def check(*bufs):
    torch.cuda.synchronize()
    for i, b in enumerate(bufs):
        assert b.intact(), f"buffer {i} written out of bounds"


@pytest.mark.parametrize("dt", ["bf16", "fp32"])
@pytest.mark.parametrize("form", [L.SKY_GEMM_XWT, L.SKY_GEMM_XW, L.SKY_GEMM_XTW])
# (512, 264, 8192): the fp32 outputs split K, with the partials in the workspace
@pytest.mark.parametrize("shape", [(200, 264, 72), (1000, 520, 136), (8, 8, 8), (512, 264, 8192)],
                         ids=lambda s: "x".join(map(str, s)))
def test_gemm_writes_in_bounds(dt, form, shape):
    M, N, K = shape
    a_shape = (K, M) if form == L.SKY_GEMM_XTW else (M, K)
    b_shape = (N, K) if form == L.SKY_GEMM_XWT else (K, N)
    A, B = rand(a_shape, dt, seed=1), rand(b_shape, dt, 0.05, seed=2)
    for out in (["bf16", "fp32"] if dt == "bf16" else ["fp32"]):
        wsb = L.lib().sky_gemm_workspace_bytes(form, M, N, K, code(dt), code(out))
        c = Guarded((M, N), tdt(out))
        ws = Guarded((max(wsb, 16),), torch.uint8)
        L.call("sky_gemm", form, M, N, K, code(dt), P(A), P(B), P(c), code(out), L.SKY_EPI_STORE,
               None, None, None, P(ws), wsb, None, stream())
        check(c, ws)
        assert torch.isfinite(c.t.float()).all()
    if form == L.SKY_GEMM_XWT:
        bias = rand((N,), dt, 0.5, seed=3)
        c = Guarded((M, N), tdt(dt))
        gp = Guarded((M, N), torch.float16 if dt == "bf16" else torch.float32)
        L.call("sky_gemm", form, M, N, K, code(dt), P(A), P(B), P(c), code(dt),
               L.SKY_EPI_BIAS_GELU, P(bias), None, P(gp), None, 0, None, stream())
        check(c, gp)
        d = Guarded((M, N), tdt(dt))
        L.call("sky_gemm", form, M, N, K, code(dt), P(A), P(B), P(d), code(dt),
               L.SKY_EPI_GELU_BWD, None, P(gp), None, None, 0, None, stream())
        check(d, gp)


@pytest.mark.parametrize("dt", ["bf16", "fp32"])
@pytest.mark.parametrize("case", [(3, 130, 1, [64, 65, 129]), (2, 100, 2, [100, 1]),
                                  (4, 1, 1, [1, 1, 1, 1])], ids=lambda c: f"B{c[0]}S{c[1]}A{c[2]}")
def test_attention_writes_in_bounds(dt, case):
    B, S, A, lens = case
    H = 64 * A
    qkv = rand((B * S, 3 * H), dt, seed=4)
    ln = torch.tensor(lens, dtype=torch.int32, device="cuda")
    ctx = Guarded((B * S, H), tdt(dt))
    lse = Guarded((B, A, S), torch.float32)
    st = Guarded((1,), torch.int32)
    st.t.zero_()
    L.call("sky_attention_fwd", P(qkv), P(ln), B, S, H, A, code(dt), P(ctx), P(lse), P(st),
           stream())
    check(ctx, lse, st)
    do = rand((B * S, H), dt, seed=5)
    dq = Guarded((B * S, 3 * H), tdt(dt))
    wsb = L.lib().sky_attention_bwd_workspace_bytes(B, S, H, A)
    ws = Guarded((max(wsb, 16),), torch.uint8)
    L.call("sky_attention_bwd", P(qkv), P(ctx), P(do), P(lse), P(ln), B, S, H, A, code(dt),
           P(dq), P(ws), wsb, P(st), stream())
    check(dq, ws, st)
    assert int(st.t.item()) == 0


@pytest.mark.parametrize("dt", ["bf16", "fp32"])
@pytest.mark.parametrize("TH", [(257, 1024), (300, 768), (33, 512)], ids=lambda t: f"T{t[0]}H{t[1]}")
def test_layernorm_writes_in_bounds(dt, TH):
    T, H = TH
    a = rand((T, H), "fp32", seed=6)
    r = rand((T, H), "fp32", seed=7)
    gam = (1.0 + rand((H,), "fp32", 0.1, seed=8)).to(tdt(dt))
    bet = rand((H,), dt, 0.1, seed=9)
    u = Guarded((T, H), torch.float32)
    y32 = Guarded((T, H), torch.float32)
    y = Guarded((T, H), tdt(dt))
    mean = Guarded((T,), torch.float32)
    rstd = Guarded((T,), torch.float32)
    L.call("sky_layernorm_fwd", P(a), P(r), P(gam), P(bet), T, H, C.c_float(1e-5), code(dt),
           P(u), P(y32), P(y), P(mean), P(rstd), stream())
    check(u, y32, y, mean, rstd)
    if dt == "bf16":  # u alone into a bf16 y (the slice's form)
        y2, m2, r2 = Guarded((T, H), torch.bfloat16), Guarded((T,), torch.float32), Guarded((T,), torch.float32)
        L.call("sky_layernorm_fwd", P(a), None, P(gam), P(bet), T, H, C.c_float(1e-5), code(dt),
               None, None, P(y2), P(m2), P(r2), stream())
        check(y2, m2, r2)
    dy = rand((T, H), dt, 1e-2, seed=10)
    dy2 = rand((T, H), "fp32", 1e-2, seed=11)
    wsb = L.lib().sky_layernorm_bwd_workspace_bytes(T, H)
    ws = Guarded((max(wsb, 16),), torch.uint8)
    du32 = Guarded((T, H), torch.float32)
    du = Guarded((T, H), tdt(dt))
    dg, db, dbias = (Guarded((H,), torch.float32) for _ in range(3))
    L.call("sky_layernorm_bwd", P(dy), code(dt), P(dy2), P(u), P(gam), P(mean), P(rstd), T, H,
           code(dt), P(du32), P(du), P(dg), P(db), P(dbias), P(ws), wsb, stream())
    check(du32, du, dg, db, dbias, ws)


@pytest.mark.parametrize("dt", ["bf16", "fp32"])
def test_row_kernels_write_in_bounds(dt):
    T, N = 333, 1000
    z, bias, dg = rand((T, N), dt, 2.0, seed=12), rand((N,), dt, 0.5, seed=13), \
        rand((T, N), dt, seed=14)
    hpre = Guarded((T, N), tdt(dt))
    gg = Guarded((T, N), tdt(dt))
    dh = Guarded((T, N), tdt(dt))
    L.call("sky_bias_gelu_fwd", P(z), P(bias), T, N, code(dt), P(hpre), P(gg), stream())
    L.call("sky_gelu_bwd", P(dg), P(hpre), T, N, code(dt), P(dh), stream())
    check(hpre, gg, dh)
    wsb = L.lib().sky_column_sum_workspace_bytes(T, N)
    ws = Guarded((max(wsb, 16),), torch.uint8)
    out = Guarded((N,), torch.float32)
    L.call("sky_column_sum", P(dg), T, N, code(dt), P(out), P(ws), wsb, stream())
    check(out, ws)
    out2 = Guarded((N,), torch.float32)
    L.call("sky_column_sum_noalloc", P(dg), T, N, code(dt), P(out2), stream())
    check(out2)
    r, o = out.t.double(), out2.t.double()
    assert float((o - r).norm()) <= 1e-6 * float(r.norm())


@pytest.mark.parametrize("io_fp32", [False, True])
def test_slice_writes_in_bounds(io_fp32):
    """Forward and backward of a ragged bf16 slice, direct and as a replayed
    step graph, into guarded y and dx."""
    from paper_2202_11836_gb300.slice import EncoderSlice
    w = synth.custom("bounds", layers=2, hidden=256, heads=4, ffn=1024, seq=80, batch=3,
                     len_lo=1, len_hi=80, dy_std=1e-2)
    io = torch.float32 if io_fp32 else torch.bfloat16
    x = torch.from_numpy(synth.activations(w)).cuda().to(io)
    dy = torch.from_numpy(synth.upstream_grad(w)).cuda().to(io)
    ln = torch.from_numpy(synth.lengths(w)).cuda()
    with EncoderSlice(w.hidden, w.heads, w.ffn, 0, w.layers, w.batch, w.seq, "bf16",
                      io_fp32=io_fp32) as s:
        for i, p in enumerate(synth.slice_params(w, affine="random")):
            s.set_params(i, p)
        y = Guarded(x.shape, io)
        dx = Guarded(x.shape, io)
        s.forward(x, ln, y.t)
        s.backward(dy, dx.t)
        s.sync()
        check(y, dx)
        y_ref, dx_ref = y.t.clone(), dx.t.clone()
        y2 = Guarded(x.shape, io)
        dx2 = Guarded(x.shape, io)
        s.step_graph(x, ln, y2.t, dy, dx2.t)
        s.launch_step_graph()
        s.sync()
        check(y2, dx2)
        assert torch.equal(y2.t, y_ref) and torch.equal(dx2.t, dx_ref)
        assert np.isfinite(y_ref.float().cpu().numpy()).all()
