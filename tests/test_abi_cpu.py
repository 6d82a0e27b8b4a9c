"""Host-side checks of the C ABI that need no GPU: the library builds and
loads, exports every function include/*.h declares, and rejects bad
arguments (and an over-cap allocation) before touching a device."""
import ctypes as C
import os
import re

import numpy as np
import pytest

from paper_2202_11836_gb300 import _lib as L
from paper_2202_11836_gb300 import synth

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def lib():
    if not os.path.exists(L.LIB_PATH):
        from paper_2202_11836_gb300 import build
        build.build()
    return L.lib()


def declared_functions():
    names = set()
    for h in sorted(os.listdir(os.path.join(ROOT, "include"))):
        if not h.endswith(".h"):
            continue
        src = open(os.path.join(ROOT, "include", h)).read()
        src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
        names |= set(re.findall(r"\b(sky_\w+)\s*\(", src))
    return sorted(names)


def test_exports_every_declared_symbol(lib):
    names = declared_functions()
    assert len(names) >= 25
    for n in names:
        assert hasattr(lib, n), f"{n} declared in include/ but not exported"
    assert set(names) == set(L._SIGNATURES), "binding and headers disagree"


def test_status_strings(lib):
    for code, name in L.STATUS_NAMES.items():
        assert lib.sky_status_string(code).decode() == name


def cfg(**kw):
    base = dict(width=768, heads=12, ffn=3072, layer_begin=0, layer_end=4, max_batch=32,
                max_seq=128, dtype=L.SKY_DTYPE_BF16, ln_eps=1e-12)
    base.update(kw)
    return L.SkySliceConfig(**base)


@pytest.mark.parametrize("bad,status", [
    (dict(heads=5), L.SKY_ERR_INVALID_ARG),          # width % heads
    (dict(layer_begin=3, layer_end=3), L.SKY_ERR_INVALID_ARG),
    (dict(max_batch=0), L.SKY_ERR_INVALID_ARG),
    (dict(width=768, heads=6), L.SKY_ERR_UNSUPPORTED),  # bf16 head dim 128
    (dict(ln_eps=-1.0), L.SKY_ERR_INVALID_ARG),
])
def test_create_rejects_bad_config(lib, bad, status):
    h = C.c_void_p()
    assert lib.sky_slice_create(C.byref(cfg(**bad)), C.byref(h)) == status
    assert not h.value
    assert L.last_error()


def test_create_over_allocation_cap_is_oom(lib):
    lib.sky_debug_set_alloc_cap(1 << 20)
    try:
        h = C.c_void_p()
        assert lib.sky_slice_create(C.byref(cfg()), C.byref(h)) == L.SKY_ERR_OOM
        assert "cap" in L.last_error()
    finally:
        lib.sky_debug_set_alloc_cap(0)


def test_null_arguments(lib):
    assert lib.sky_slice_destroy(None) == L.SKY_OK
    assert lib.sky_slice_forward(None, None, None, 1, 1, None, None) == L.SKY_ERR_INVALID_ARG
    assert lib.sky_slice_backward(None, None, None, None) == L.SKY_ERR_INVALID_ARG
    assert lib.sky_slice_step_graph_create(None, None, None, 1, 1, None, None, None,
                                           None) == L.SKY_ERR_INVALID_ARG
    assert lib.sky_slice_step_graph_launch(None, None) == L.SKY_ERR_INVALID_ARG
    assert lib.sky_gemm(0, 8, 8, 8, 0, None, None, None, 0, 0, None, None, None, None, 0, None,
                        None) == L.SKY_ERR_INVALID_ARG
    assert lib.sky_column_sum_workspace_bytes(0, 5) == 0


def test_split_choice_is_a_host_decision(lib):
    # weight-gradient shapes split the token dimension; activations shapes never do
    assert lib.sky_gemm_workspace_bytes(L.SKY_GEMM_XTW, 1024, 1024, 8192, 0, 1) > 0
    assert lib.sky_gemm_workspace_bytes(L.SKY_GEMM_XWT, 8192, 1024, 1024, 0, 0) == 0


def test_synth_generator_is_seeded_and_bf16_exact():
    w = synth.WORKLOADS["base-s128"]
    a, b = synth.activations(w), synth.activations(w)
    assert np.array_equal(a, b)
    assert np.array_equal(synth.round_bf16(a), a)
    lens = synth.lengths(w)
    assert lens.min() >= 64 and lens.max() <= 128
    w5 = synth.WORKLOADS["large-s2048"]
    l5 = synth.lengths(w5)
    assert l5[0] == 2048 and l5[1] == 2048 and 512 <= l5[2] <= 2048
    # per-layer parameters depend only on (seed, layer)
    p3 = synth.layer_params(3, 64, 128, "bf16")
    assert np.array_equal(p3["W1"], synth.layer_params(3, 64, 128, "bf16")["W1"])
    assert not np.array_equal(p3["W1"], synth.layer_params(4, 64, 128, "bf16")["W1"])


def test_bf16_rounding_matches_torch():
    torch = pytest.importorskip("torch")
    g = np.random.default_rng(0)
    x = np.concatenate([g.normal(0, 1, 10000), g.normal(0, 1e-30, 100), [0.0, -0.0, 1.0 + 2 ** -8]])
    x = x.astype(np.float32)
    ref = torch.from_numpy(x).to(torch.bfloat16).float().numpy()
    assert np.array_equal(synth.round_bf16(x), ref)


def _kind_c(t, enums):
    """Storage class of a C type as written in include/*.h."""
    t = " ".join(t.replace("const", " ").split())
    if "*" in t:
        return ("ptr",)
    table = {"int32_t": ("i", 4), "int": ("i", 4), "int64_t": ("i", 8), "uint64_t": ("u", 8),
             "size_t": ("u", 8), "float": ("f", 4), "double": ("f", 8), "sky_status": ("i", 4),
             "void": None}
    if t in enums:
        return ("i", 4)
    assert t in table, f"unmapped C type {t!r}"
    return table[t]


def _kind_ctypes(ct):
    if ct is None:
        return None
    if ct in (C.c_void_p, C.c_char_p) or issubclass(ct, C._Pointer):
        return ("ptr",)
    if ct in (C.c_float, C.c_double):
        return ("f", C.sizeof(ct))
    signed = ct(-1).value < 0
    return ("i" if signed else "u", C.sizeof(ct))


def test_binding_signatures_match_headers():
    """Every declared function has the same parameter count, parameter
    storage classes and return class in the ctypes table as in its header."""
    decls, enums = {}, set()
    for h in sorted(os.listdir(os.path.join(ROOT, "include"))):
        if not h.endswith(".h"):
            continue
        src = open(os.path.join(ROOT, "include", h)).read()
        src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
        src = re.sub(r"//[^\n]*", "", src)
        enums |= set(re.findall(r"typedef\s+enum\s*\{[^}]*\}\s*(\w+)\s*;", src))
        for ret, name, params in re.findall(r"([\w\s\*]+?)\b(sky_\w+)\s*\(([^)]*)\)\s*;", src):
            ret = ret.split("\n")[-1].strip()
            ps = [p.strip() for p in params.split(",") if p.strip() and p.strip() != "void"]
            # drop the parameter name: the last identifier of each declarator
            types = [re.sub(r"\b\w+\s*$", "", p) if re.search(r"[\s\*]\w+\s*$", p) else p
                     for p in ps]
            decls[name] = (ret, types)
    assert set(decls) == set(L._SIGNATURES)
    for name, (ret, types) in decls.items():
        restype, argtypes = L._SIGNATURES[name]
        assert len(argtypes) == len(types), (name, types)
        assert _kind_ctypes(restype) == _kind_c(ret, enums), (name, ret, restype)
        for i, (ct, t) in enumerate(zip(argtypes, types)):
            assert _kind_ctypes(ct) == _kind_c(t, enums), (name, i, t, ct)
