"""Kernel-level parity through the C ABI of sky_ops.h (GPU).

Each kernel runs on seeded inputs whose sizes span several tiles and end in a
ragged tail; the reference is the plain definition in float64 (the oracle's
own functions for attention, LayerNorm and GELU).
"""
import ctypes as C

import numpy as np
import pytest

from oracle import encoder_f64 as ORC
from paper_2202_11836_gb300 import _lib as L
from paper_2202_11836_gb300.synth import round_bf16
from parity_util import assert_close, l2rel, maxrel, to_device, to_host

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")


def P(t):
    return C.c_void_p(0 if t is None else int(t.data_ptr()))


def stream():
    return C.c_void_p(int(torch.cuda.current_stream().cuda_stream))


def dt_code(dt):
    return L.SKY_DTYPE_BF16 if dt == "bf16" else L.SKY_DTYPE_FP32


def rnd(g, shape, std, dt):
    a = g.normal(0, std, shape).astype(np.float32)
    return round_bf16(a) if dt == "bf16" else a


GEMM_SHAPES = [(128, 256, 64), (200, 264, 72), (384, 768, 1024), (1000, 520, 136), (8, 8, 8)]


@pytest.mark.parametrize("dt", ["bf16", "fp32"])
@pytest.mark.parametrize("form", [L.SKY_GEMM_XWT, L.SKY_GEMM_XW, L.SKY_GEMM_XTW])
@pytest.mark.parametrize("shape", GEMM_SHAPES, ids=lambda s: "x".join(map(str, s)))
def test_gemm_store(dt, form, shape):
    M, N, K = shape
    g = np.random.default_rng(M * 7 + N * 3 + K + form)
    if form == L.SKY_GEMM_XWT:
        A, B = rnd(g, (M, K), 1.0, dt), rnd(g, (N, K), 0.05, dt)
        ref = A.astype(np.float64) @ B.astype(np.float64).T
    elif form == L.SKY_GEMM_XW:
        A, B = rnd(g, (M, K), 1.0, dt), rnd(g, (K, N), 0.05, dt)
        ref = A.astype(np.float64) @ B.astype(np.float64)
    else:
        A, B = rnd(g, (K, M), 1.0, dt), rnd(g, (K, N), 0.05, dt)
        ref = A.astype(np.float64).T @ B.astype(np.float64)
    for out_dt in (["bf16", "fp32"] if dt == "bf16" else ["fp32"]):
        a, b = to_device(A, dt), to_device(B, dt)
        c = torch.zeros((M, N), dtype=torch.bfloat16 if out_dt == "bf16" else torch.float32,
                        device="cuda")
        wsb = L.lib().sky_gemm_workspace_bytes(form, M, N, K, dt_code(dt), dt_code(out_dt))
        ws = torch.empty(max(wsb, 16), dtype=torch.uint8, device="cuda")
        L.call("sky_gemm", form, M, N, K, dt_code(dt), P(a), P(b), P(c), dt_code(out_dt),
               L.SKY_EPI_STORE, None, None, None, P(ws), wsb, None, stream())
        torch.cuda.synchronize()
        got = to_host(c)
        if out_dt == "fp32":
            tol = 1e-5 if dt == "bf16" else 1e-5
            assert l2rel(got, ref) <= tol and maxrel(got, ref) <= 10 * tol, (out_dt, l2rel(got, ref))
        else:
            assert l2rel(got, ref) <= 4e-3 and maxrel(got, ref) <= 8e-3, (l2rel(got, ref), maxrel(got, ref))


@pytest.mark.parametrize("dt", ["bf16", "fp32"])
# (256, 384, 128) and (512, 768, 192) run the 192-wide pair tiles in their
# plain-store (bias) products
@pytest.mark.parametrize("shape", [(256, 512, 128), (200, 264, 72), (256, 384, 128), (512, 768, 192)],
                         ids=lambda s: "x".join(map(str, s)))
def test_gemm_epilogues(dt, shape):
    M, N, K = shape
    g = np.random.default_rng(11)
    A, W = rnd(g, (M, K), 1.0, dt), rnd(g, (N, K), 0.1, dt)
    bias = rnd(g, (N,), 0.5, dt)
    acc = A.astype(np.float64) @ W.astype(np.float64).T
    a, w, b = to_device(A, dt), to_device(W, dt), to_device(bias, dt)
    td = torch.bfloat16 if dt == "bf16" else torch.float32
    tol_l2 = 4e-3 if dt == "bf16" else 1e-5
    # bias + GELU: C = GELU(acc + b), aux_out = GELU'(acc + b) (fp16 for bf16 inputs)
    c = torch.empty((M, N), dtype=td, device="cuda")
    gp = torch.empty((M, N), dtype=torch.float16 if dt == "bf16" else torch.float32, device="cuda")
    L.call("sky_gemm", L.SKY_GEMM_XWT, M, N, K, dt_code(dt), P(a), P(w), P(c), dt_code(dt),
           L.SKY_EPI_BIAS_GELU, P(b), None, P(gp), None, 0, None, stream())
    torch.cuda.synchronize()
    pre = acc + bias
    assert l2rel(to_host(c), ORC.gelu(pre)) <= tol_l2
    assert l2rel(to_host(gp), ORC.gelu_grad(pre)) <= (1e-3 if dt == "bf16" else 1e-5)
    # GELU backward: C = acc * aux, aux the stored derivative
    d = g.normal(0.5, 0.3, (M, N)).astype(np.float32)
    aux = torch.from_numpy(d).cuda().to(gp.dtype)
    dv = aux.float().cpu().numpy().astype(np.float64)
    L.call("sky_gemm", L.SKY_GEMM_XWT, M, N, K, dt_code(dt), P(a), P(w), P(c), dt_code(dt),
           L.SKY_EPI_GELU_BWD, None, P(aux), None, None, 0, None, stream())
    torch.cuda.synchronize()
    assert l2rel(to_host(c), acc * dv) <= tol_l2
    # bias into an fp32 output (the residual-branch linear layers)
    c32 = torch.empty((M, N), dtype=torch.float32, device="cuda")
    L.call("sky_gemm", L.SKY_GEMM_XWT, M, N, K, dt_code(dt), P(a), P(w), P(c32), 1,
           L.SKY_EPI_STORE, P(b), None, None, None, 0, None, stream())
    torch.cuda.synchronize()
    assert l2rel(to_host(c32), acc + bias) <= 1e-5
    # bias into an output of the input type (the QKV projection's form), with
    # the bias 16-byte aligned and 8 bytes off: the results agree bit for bit
    outs = []
    for off in (0, 4 if dt == "bf16" else 2):
        braw = torch.zeros(N + 8, dtype=td, device="cuda")
        braw[off:off + N] = b
        cb = torch.empty((M, N), dtype=td, device="cuda")
        L.call("sky_gemm", L.SKY_GEMM_XWT, M, N, K, dt_code(dt), P(a), P(w), P(cb), dt_code(dt),
               L.SKY_EPI_STORE, P(braw[off:off + N]), None, None, None, 0, None, stream())
        torch.cuda.synchronize()
        outs.append(to_host(cb))
        assert l2rel(outs[-1], acc + bias) <= tol_l2
    assert np.array_equal(outs[0], outs[1])


def test_gemm_wgrad_split_deterministic():
    """Split-K weight gradient over a long token dimension: bitwise repeatable."""
    M, N, K = 768, 768, 8192
    g = np.random.default_rng(5)
    A, B = rnd(g, (K, M), 1.0, "bf16"), rnd(g, (K, N), 1e-3, "bf16")
    a, b = to_device(A, "bf16"), to_device(B, "bf16")
    wsb = L.lib().sky_gemm_workspace_bytes(L.SKY_GEMM_XTW, M, N, K, 0, 1)
    assert wsb > 0  # this shape splits the token dimension
    ws = torch.empty(wsb, dtype=torch.uint8, device="cuda")
    outs = []
    for _ in range(2):
        c = torch.empty((M, N), dtype=torch.float32, device="cuda")
        L.call("sky_gemm", L.SKY_GEMM_XTW, M, N, K, 0, P(a), P(b), P(c), 1, 0, None, None, None,
               P(ws), wsb, None, stream())
        torch.cuda.synchronize()
        outs.append(c.cpu().numpy())
    assert np.array_equal(outs[0], outs[1])
    ref = A.astype(np.float64).T @ B.astype(np.float64)
    assert l2rel(outs[0], ref) <= 1e-5


def attn_case(dt, B, S, A, lens, seed=3):
    D = 64
    H = A * D
    g = np.random.default_rng(seed)
    qkv = rnd(g, (B * S, 3 * H), 1.0, dt)
    dctx = rnd(g, (B * S, H), 1.0, dt)
    return H, qkv, dctx, np.array(lens, dtype=np.int32)


@pytest.mark.parametrize("dt", ["bf16", "fp32"])
@pytest.mark.parametrize("case", [
    (2, 100, 2, [100, 1]), (3, 130, 1, [64, 65, 129]), (1, 64, 2, [63]), (2, 256, 4, [256, 200]),
    (4, 1, 1, [1, 1, 1, 1]),
], ids=lambda c: f"B{c[0]}S{c[1]}A{c[2]}")
def test_attention(dt, case):
    B, S, A, lens = case
    H, qkv, dctx, lens = attn_case(dt, B, S, A, lens)
    D = 64
    q = to_device(qkv, dt)
    ln = torch.from_numpy(lens).cuda()
    td = torch.bfloat16 if dt == "bf16" else torch.float32
    ctx = torch.empty((B * S, H), dtype=td, device="cuda")
    lse = torch.empty((B, A, S), dtype=torch.float32, device="cuda")
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    L.call("sky_attention_fwd", P(q), P(ln), B, S, H, A, dt_code(dt), P(ctx), P(lse), P(st), stream())
    do = to_device(dctx, dt)
    dq = torch.empty((B * S, 3 * H), dtype=td, device="cuda")
    wsb = L.lib().sky_attention_bwd_workspace_bytes(B, S, H, A)
    ws = torch.empty(wsb, dtype=torch.uint8, device="cuda")
    L.call("sky_attention_bwd", P(q), P(ctx), P(do), P(lse), P(ln), B, S, H, A, dt_code(dt),
           P(dq), P(ws), wsb, P(st), stream())
    torch.cuda.synchronize()
    assert int(st.item()) == 0
    Q = qkv[:, :H].reshape(B, S, A, D).astype(np.float64)
    K = qkv[:, H:2 * H].reshape(B, S, A, D).astype(np.float64)
    V = qkv[:, 2 * H:].reshape(B, S, A, D).astype(np.float64)
    ctx_o, Pm = ORC.attention_forward(Q, K, V, lens)
    assert_close("ctx", to_host(ctx), ctx_o.reshape(B * S, H), dt)
    # the kernel's backward consumes its own (rounded) ctx, as the slice does
    dQ, dK, dV = ORC.attention_backward(dctx.reshape(B, S, A, D).astype(np.float64), Q, K, V, Pm, lens)
    got = to_host(dq)
    assert_close("dQ", got[:, :H], dQ.reshape(B * S, H), dt)
    assert_close("dK", got[:, H:2 * H], dK.reshape(B * S, H), dt)
    assert_close("dV", got[:, 2 * H:], dV.reshape(B * S, H), dt)
    # padded keys get exactly zero dK and dV
    for b, n in enumerate(lens):
        assert np.all(got[b * S + n:(b + 1) * S, H:] == 0.0)
    # log-sum-exp of each row (the kernels keep it in base-2 units)
    for b, n in enumerate(lens):
        for a in range(A):
            s = Q[b, :, a] @ K[b, :n, a].T / 8.0
            m = s.max(1)
            ref = m + np.log(np.exp(s - m[:, None]).sum(1))
            got_ln = lse.cpu().numpy()[b, a].astype(np.float64) * np.log(2.0)
            assert np.max(np.abs(got_ln - ref)) <= (2e-2 if dt == "bf16" else 1e-4)


def test_attention_bad_length_sets_status():
    B, S, A = 2, 64, 1
    H, qkv, _, _ = attn_case("bf16", B, S, A, [1, 1])
    q = to_device(qkv, "bf16")
    ln = torch.tensor([0, 65], dtype=torch.int32, device="cuda")
    ctx = torch.empty((B * S, H), dtype=torch.bfloat16, device="cuda")
    lse = torch.empty((B, A, S), dtype=torch.float32, device="cuda")
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    L.call("sky_attention_fwd", P(q), P(ln), B, S, H, A, 0, P(ctx), P(lse), P(st), stream())
    torch.cuda.synchronize()
    assert int(st.item()) & 1
    assert torch.isfinite(ctx.float()).all()


def test_attention_bwd_rejects_misaligned_workspace():
    # checked on the host before any kernel is launched: nothing runs
    B, S, A = 1, 64, 1
    H, qkv, dctx, lens = attn_case("bf16", B, S, A, [64])
    q = to_device(qkv, "bf16")
    do = to_device(dctx, "bf16")
    ln = torch.from_numpy(lens).cuda()
    ctx = torch.zeros((B * S, H), dtype=torch.bfloat16, device="cuda")
    lse = torch.zeros((B, A, S), dtype=torch.float32, device="cuda")
    dq = torch.zeros((B * S, 3 * H), dtype=torch.bfloat16, device="cuda")
    wsb = L.lib().sky_attention_bwd_workspace_bytes(B, S, H, A)
    ws = torch.empty(wsb + 16, dtype=torch.uint8, device="cuda")
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    with pytest.raises(L.SkyError) as e:
        L.call("sky_attention_bwd", P(q), P(ctx), P(do), P(lse), P(ln), B, S, H, A, 0,
               P(dq), C.c_void_p(int(ws.data_ptr()) + 4), wsb, P(st), stream())
    assert e.value.status == L.SKY_ERR_INVALID_ARG
    torch.cuda.synchronize()
    assert int(st.item()) == 0 and not dq.any()


@pytest.mark.parametrize("dt", ["bf16", "fp32"])
@pytest.mark.parametrize("TH", [(300, 768), (257, 1024), (64, 128), (33, 2048)],
                         ids=lambda t: f"T{t[0]}H{t[1]}")
def test_layernorm(dt, TH):
    """Residual + LayerNorm of fp32 inputs; backward from a dtype or an fp32 dy
    plus an fp32 second gradient term."""
    T, H = TH
    if dt == "fp32" and H > 1024:
        pytest.skip("fp32 LayerNorm supports H <= 1024")
    g = np.random.default_rng(T + H)
    av = g.normal(0.5, 1.0, (T, H)).astype(np.float32)
    rv = g.normal(0.0, 1.0, (T, H)).astype(np.float32)
    dy = rnd(g, (T, H), 1e-2, dt)
    dy2 = g.normal(0, 1e-2, (T, H)).astype(np.float32)
    gam, bet = (1 + rnd(g, (H,), 0.1, dt)), rnd(g, (H,), 0.1, dt)
    gam = round_bf16(gam) if dt == "bf16" else gam
    td = torch.bfloat16 if dt == "bf16" else torch.float32
    A_ = torch.from_numpy(av).cuda()
    R_ = torch.from_numpy(rv).cuda()
    D2 = torch.from_numpy(dy2).cuda()
    G_, B_, DY = (to_device(v, dt) for v in (gam, bet, dy))
    y = torch.empty((T, H), dtype=td, device="cuda")
    y32 = torch.empty((T, H), dtype=torch.float32, device="cuda")
    mean = torch.empty(T, dtype=torch.float32, device="cuda")
    rstd = torch.empty(T, dtype=torch.float32, device="cuda")
    eps = 1e-5
    # u written in place over a
    L.call("sky_layernorm_fwd", P(A_), P(R_), P(G_), P(B_), T, H, C.c_float(eps), dt_code(dt),
           P(A_), P(y32), P(y), P(mean), P(rstd), stream())
    torch.cuda.synchronize()
    u = av.astype(np.float64) + rv
    assert l2rel(to_host(A_), u) <= 1e-7
    Yo, xhat, rs = ORC.layer_norm(u, gam.astype(np.float64), bet.astype(np.float64), eps)
    assert_close("y", to_host(y), Yo, dt)
    assert l2rel(to_host(y32), Yo) <= 1e-5
    wsb = L.lib().sky_layernorm_bwd_workspace_bytes(T, H)
    ws = torch.empty(wsb, dtype=torch.uint8, device="cuda")
    for dy_dt, second in ((dt, False), ("fp32", True)):
        dyt = DY if dy_dt == dt else DY.float()
        du = torch.empty((T, H), dtype=td, device="cuda")
        du32 = torch.empty((T, H), dtype=torch.float32, device="cuda")
        dg, db, dbias = (torch.empty(H, dtype=torch.float32, device="cuda") for _ in range(3))
        L.call("sky_layernorm_bwd", P(dyt), dt_code(dy_dt), P(D2) if second else None, P(A_),
               P(G_), P(mean), P(rstd), T, H, dt_code(dt), P(du32), P(du), P(dg), P(db),
               P(dbias), P(ws), wsb, stream())
        torch.cuda.synchronize()
        dyo = dy.astype(np.float64) + (dy2 if second else 0.0)
        dUo, dgo, dbo = ORC.layer_norm_backward(dyo, xhat, rs, gam.astype(np.float64))
        assert_close("du", to_host(du), dUo, dt)
        assert l2rel(to_host(du32), dUo) <= 1e-5
        assert l2rel(dg.cpu().numpy(), dgo) <= 1e-5
        assert l2rel(db.cpu().numpy(), dbo) <= 1e-5
        assert l2rel(dbias.cpu().numpy(), dUo.sum(0)) <= 1e-4
    # the two-term sum into the dtype
    s_out = torch.empty((T, H), dtype=td, device="cuda")
    L.call("sky_add_f32", P(R_), P(D2), T * H, dt_code(dt), P(s_out), stream())
    torch.cuda.synchronize()
    assert_close("add", to_host(s_out), rv.astype(np.float64) + dy2, dt)


@pytest.mark.parametrize("TH", [(1000, 1024), (300, 768), (200, 2048), (100, 512)],
                         ids=lambda t: f"T{t[0]}H{t[1]}")
def test_layernorm_fwd_of_u_only(TH):
    """bf16 LayerNorm of u alone (no residual operand, no u output), the form
    the slice uses: against the oracle, and bit for bit against the same rows
    with a zero residual added (which changes no sum).  Also with an fp32
    output only, whose bf16 rounding is the bf16 output."""
    T, H = TH
    g = np.random.default_rng(T * H)
    av = g.normal(0.5, 1.0, (T, H)).astype(np.float32)
    gam, bet = round_bf16(1 + g.normal(0, 0.1, H)), round_bf16(g.normal(0, 0.1, H))
    A_ = torch.from_numpy(av).cuda()
    Z_ = torch.zeros_like(A_)
    G_, B_ = to_device(gam, "bf16"), to_device(bet, "bf16")
    eps = 1e-12
    outs = []
    for r in (None, Z_):
        y = torch.empty((T, H), dtype=torch.bfloat16, device="cuda")
        mean = torch.empty(T, dtype=torch.float32, device="cuda")
        rstd = torch.empty(T, dtype=torch.float32, device="cuda")
        L.call("sky_layernorm_fwd", P(A_), P(r) if r is not None else None, P(G_), P(B_), T, H,
               C.c_float(eps), dt_code("bf16"), None, None, P(y), P(mean), P(rstd), stream())
        outs.append((y, mean, rstd))
    y32 = torch.empty((T, H), dtype=torch.float32, device="cuda")
    m2, r2 = (torch.empty(T, dtype=torch.float32, device="cuda") for _ in range(2))
    L.call("sky_layernorm_fwd", P(A_), None, P(G_), P(B_), T, H, C.c_float(eps), dt_code("bf16"),
           None, P(y32), None, P(m2), P(r2), stream())
    torch.cuda.synchronize()
    (ys, ms, rs), (yw, mw, rw) = outs
    assert torch.equal(ys, yw) and torch.equal(ms, mw) and torch.equal(rs, rw)
    assert torch.equal(m2, ms) and torch.equal(r2, rs)
    assert torch.equal(y32.bfloat16(), ys)
    Yo, _, rso = ORC.layer_norm(av.astype(np.float64), gam.astype(np.float64),
                                bet.astype(np.float64), eps)
    assert l2rel(to_host(y32), Yo) <= 1e-5
    assert_close("y", to_host(ys), Yo, "bf16")
    assert l2rel(rs.cpu().numpy().astype(np.float64), rso.reshape(-1)) <= 1e-5


def test_layernorm_rejects_misaligned_tensors():
    """The row kernels move 16-byte vectors: a tensor off a 16-byte boundary
    is refused on the host (UNSUPPORTED), before any launch."""
    T, H = 200, 256
    buf = torch.zeros(T * H + 1, dtype=torch.float32, device="cuda")
    a = buf[1:]
    G_ = torch.ones(H, dtype=torch.bfloat16, device="cuda")
    B_ = torch.zeros(H, dtype=torch.bfloat16, device="cuda")
    y = torch.empty((T, H), dtype=torch.bfloat16, device="cuda")
    mean, rstd = (torch.empty(T, dtype=torch.float32, device="cuda") for _ in range(2))
    with pytest.raises(L.SkyError) as e:
        L.call("sky_layernorm_fwd", P(a), None, P(G_), P(B_), T, H, C.c_float(1e-12),
               dt_code("bf16"), None, None, P(y), P(mean), P(rstd), stream())
    assert e.value.status == L.SKY_ERR_UNSUPPORTED


@pytest.mark.parametrize("dt", ["bf16", "fp32"])
def test_gelu_and_column_sum(dt):
    T, N = 333, 1000
    g = np.random.default_rng(2)
    z, bias, dgv = rnd(g, (T, N), 2.0, dt), rnd(g, (N,), 0.5, dt), rnd(g, (T, N), 1.0, dt)
    td = torch.bfloat16 if dt == "bf16" else torch.float32
    Z, Bv, DG = to_device(z, dt), to_device(bias, dt), to_device(dgv, dt)
    hpre = torch.empty((T, N), dtype=td, device="cuda")
    gg = torch.empty((T, N), dtype=td, device="cuda")
    dh = torch.empty((T, N), dtype=td, device="cuda")
    L.call("sky_bias_gelu_fwd", P(Z), P(Bv), T, N, dt_code(dt), P(hpre), P(gg), stream())
    L.call("sky_gelu_bwd", P(DG), P(hpre), T, N, dt_code(dt), P(dh), stream())
    out = torch.empty(N, dtype=torch.float32, device="cuda")
    wsb = L.lib().sky_column_sum_workspace_bytes(T, N)
    ws = torch.empty(wsb, dtype=torch.uint8, device="cuda")
    L.call("sky_column_sum", P(DG), T, N, dt_code(dt), P(out), P(ws), wsb, stream())
    torch.cuda.synchronize()
    pre = z.astype(np.float64) + bias
    assert_close("hpre", to_host(hpre), pre, dt)
    assert_close("gelu", to_host(gg), ORC.gelu(pre), dt)
    h_used = to_host(hpre)
    assert_close("gelu_bwd", to_host(dh), dgv * ORC.gelu_grad(h_used), dt)
    assert l2rel(out.cpu().numpy(), dgv.astype(np.float64).sum(0)) <= 1e-6
