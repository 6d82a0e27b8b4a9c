"""The local parameter update (sky_slice_optimizer_*, Sec. III) against the
float64 update oracle.  Each step runs a real forward and backward pass on
the GPU; the gradients it leaves are fed to the oracle too, so the update
rule itself is compared: fp32 master weights and state within 2e-6 relative
(fp32 arithmetic on values of order one), and the slice's bf16 parameters
equal to the master weights rounded to bf16."""
import numpy as np
import pytest

from oracle import optimizer as O
from paper_2202_11836_gb300 import synth
from parity_util import to_device

pytestmark = pytest.mark.gpu
torch = pytest.importorskip("torch")


def run(w, kind, steps=3):
    from paper_2202_11836_gb300.slice import EncoderSlice
    params = synth.slice_params(w, affine="random")
    X, lens, dY = synth.activations(w), synth.lengths(w), synth.upstream_grad(w)
    hp = dict(lr=1e-2, beta1=0.9, beta2=0.98, eps=1e-6, weight_decay=0.05, momentum=0.9)
    layers = range(w.layer_begin, w.layer_begin + w.layers)
    with EncoderSlice(w.hidden, w.heads, w.ffn, w.layer_begin, w.layer_begin + w.layers,
                      X.shape[0], w.seq, w.dtype) as s:
        for i, l in enumerate(layers):
            s.set_params(l, params[i])
        s.optimizer_init(kind, **hp)
        ref = {l: {n: [s.get_params(l)[n].astype(np.float64), 0.0, 0.0] for n in synth.PARAM_NAMES}
               for l in layers}
        x = to_device(X, w.dtype)
        dy = to_device(dY, w.dtype)
        ln = torch.from_numpy(np.asarray(lens, np.int32)).cuda()
        for t in range(1, steps + 1):
            s.forward(x, ln)
            s.backward(dy)
            s.sync()
            grads = {l: s.get_grads(l) for l in layers}
            s.optimizer_step(hp["lr"])
            s.sync()
            for l in layers:
                for n in synth.PARAM_NAMES:
                    st = ref[l][n]
                    decay = n in O.DECAYED
                    g = grads[l][n].astype(np.float64)
                    if kind == "adamw":
                        st[0], st[1], st[2] = O.adamw_step(st[0], g, st[1], st[2], t, hp["lr"],
                                                           hp["beta1"], hp["beta2"], hp["eps"],
                                                           hp["weight_decay"], decay)
                    else:
                        st[0], st[1] = O.sgd_step(st[0], g, st[1], t, hp["lr"], hp["momentum"],
                                                  hp["weight_decay"], decay)
        for l in layers:
            master = s.optimizer_state(l, 0)
            s1 = s.optimizer_state(l, 1)
            s2 = s.optimizer_state(l, 2) if kind == "adamw" else None
            p = s.get_params(l)
            for n in synth.PARAM_NAMES:
                w_ref, m_ref, v_ref = ref[l][n]
                scale = np.abs(w_ref).max() + 1e-30
                assert np.abs(master[n] - w_ref).max() <= 2e-6 * scale, (l, n)
                assert np.abs(s1[n] - m_ref).max() <= 2e-6 * (np.abs(m_ref).max() + 1e-30), (l, n)
                if s2 is not None:
                    assert np.abs(s2[n] - v_ref).max() <= 2e-6 * (np.abs(v_ref).max() + 1e-30), (l, n)
                if w.dtype == "bf16":
                    assert np.array_equal(p[n], synth.round_bf16(master[n])), (l, n)
                else:
                    assert np.array_equal(p[n], master[n]), (l, n)


@pytest.mark.parametrize("kind", ["adamw", "sgd"])
def test_update_bf16_slice(kind):
    w = synth.custom("opt", layers=2, hidden=256, heads=4, ffn=512, seq=64, batch=4,
                     len_lo=16, len_hi=64)
    run(w, kind)


@pytest.mark.parametrize("kind", ["adamw", "sgd"])
def test_update_fp32_slice(kind):
    run(synth.WORKLOADS["tiny-fp32"], kind)


def test_update_requires_init():
    from paper_2202_11836_gb300 import _lib as L
    from paper_2202_11836_gb300.slice import EncoderSlice
    with EncoderSlice(256, 4, 512, 0, 1, 2, 64) as s:
        with pytest.raises(L.SkyError) as e:
            s.optimizer_step(1e-3)
        assert e.value.status == L.SKY_ERR_STATE
        with pytest.raises(L.SkyError) as e:
            s.optimizer_init("adamw", beta1=1.0)
        assert e.value.status == L.SKY_ERR_INVALID_ARG
