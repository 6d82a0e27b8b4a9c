"""Seeded synthetic inputs for the encoder-slice workloads.

This module only draws random numbers and formats them (bf16 rounding); it
holds none of the encoder layer's arithmetic.  Both the CUDA path (through the
tests and the bench) and the float64 oracle consume what it produces, so the
two sides always see the same values.

The paper trains BERT on MNLI with 16 heads and batch 32 (Sec. VI-A); its
hidden size and sequence length are not stated and the dataset is not used
here.  Throughput depends only on shapes and on the padding mask, so seeded
Gaussian activations, weights and upstream gradients, with per-sequence valid
lengths drawn uniformly, stand in for it.

Parameters of global layer index ``l`` are drawn from ``(seed, l)`` alone, so
any contiguous slice ``[l0, l1)`` of a deep model (the unit of work the
allocator hands a device, Sec. IV-D) is well defined and slices compose.
"""
from __future__ import annotations

import dataclasses

import numpy as np

SEED = 20220223

# Order of the 12 per-layer parameter tensors everywhere in this library.
PARAM_NAMES = (
    "Wqkv", "bqkv", "Wo", "bo", "gamma1", "beta1",
    "W1", "b1", "W2", "b2", "gamma2", "beta2",
)


@dataclasses.dataclass(frozen=True)
class Workload:
    """Shape and value distribution of one synthetic encoder-slice workload."""
    name: str
    layers: int          # slice length l1 - l0
    hidden: int          # H
    heads: int           # A  (head dim D = H / A)
    ffn: int             # F
    seq: int             # S (padded)
    batch: int           # B
    dtype: str           # "fp32" or "bf16"
    len_lo: int          # valid lengths uniform in [len_lo, len_hi]
    len_hi: int
    dy_std: float        # upstream gradient ~ N(0, dy_std)
    full_len: int = 0    # this many leading sequences get len = S
    layer_begin: int = 0

    @property
    def tokens(self) -> int:
        return self.batch * self.seq


WORKLOADS = {
    # tiny fp32 slice of 2 layers (parity at 1e-4)
    "tiny-fp32": Workload("tiny-fp32", 2, 128, 2, 512, 32, 4, "fp32", 16, 32, 1e-2),
    # BERT-base width, 4 layers, S=128, B=32
    "base-s128": Workload("base-s128", 4, 768, 12, 3072, 128, 32, "bf16", 64, 128, 1e-3),
    # BERT-large width, 8 layers, S=512, B=16
    "large-s512": Workload("large-s512", 8, 1024, 16, 4096, 512, 16, "bf16", 256, 512, 1e-3),
    # BERT-base width, S=128, B=16: uneven slices {1,3,7,17} of a 160-layer model
    "base-s128-b16": Workload("base-s128-b16", 1, 768, 12, 3072, 128, 16, "bf16", 64, 128, 1e-3),
    # BERT-large width, long sequence S=2048, B=4, two full-length sequences
    "large-s2048": Workload("large-s2048", 4, 1024, 16, 4096, 2048, 4, "bf16", 512, 2048, 1e-3,
                            full_len=2),
}

# Uneven load-balanced slices of the 160-layer base-width model.
UNEVEN_SLICES = ((0, 1), (1, 4), (4, 11), (11, 28))


def round_bf16(x: np.ndarray) -> np.ndarray:
    """Round float32 values to the nearest bfloat16 (ties to even); returns float32."""
    u = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32).astype(np.uint64)
    u = (u + 0x7FFF + ((u >> 16) & 1)) & 0xFFFF0000
    return u.astype(np.uint32).view(np.float32)


def to_bf16_bits(x: np.ndarray) -> np.ndarray:
    """bfloat16 bit patterns (uint16) of float32 values that are already bf16-exact."""
    u = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32)
    return (u >> 16).astype(np.uint16)


def from_bf16_bits(b: np.ndarray) -> np.ndarray:
    return (np.ascontiguousarray(b, dtype=np.uint16).astype(np.uint32) << 16).view(np.float32)


def _rng(seed: int, *stream: int) -> np.random.Generator:
    return np.random.Generator(np.random.PCG64(np.random.SeedSequence([seed, *stream])))


def _finish(a: np.ndarray, dtype: str) -> np.ndarray:
    a = a.astype(np.float32)
    return round_bf16(a) if dtype == "bf16" else a


def layer_params(layer: int, hidden: int, ffn: int, dtype: str, seed: int = SEED,
                 affine: str = "bert") -> dict:
    """Parameters of global layer ``layer``; layouts are ``[out, in]`` row-major.

    ``affine="bert"`` gives the workload's initialisation (weights N(0, 0.02),
    biases 0, gamma 1, beta 0).  ``affine="random"`` also draws biases
    N(0, 0.02), gamma 1 + N(0, 0.1) and beta N(0, 0.02) so that tests exercise
    every parameter path.
    """
    H, F = hidden, ffn
    g = _rng(seed, 1, layer)
    shapes = {"Wqkv": (3 * H, H), "bqkv": (3 * H,), "Wo": (H, H), "bo": (H,),
              "gamma1": (H,), "beta1": (H,), "W1": (F, H), "b1": (F,),
              "W2": (H, F), "b2": (H,), "gamma2": (H,), "beta2": (H,)}
    out = {}
    for name in PARAM_NAMES:
        shp = shapes[name]
        if name.startswith("W"):
            v = g.normal(0.0, 0.02, shp)
        elif affine == "random":
            if name.startswith("gamma"):
                v = 1.0 + g.normal(0.0, 0.1, shp)
            else:
                v = g.normal(0.0, 0.02, shp)
        else:
            v = np.ones(shp) if name.startswith("gamma") else np.zeros(shp)
        out[name] = _finish(v, dtype)
    return out


def lengths(w: Workload, seed: int = SEED, batch: int | None = None) -> np.ndarray:
    B = w.batch if batch is None else batch
    g = _rng(seed, 3)
    lens = g.integers(w.len_lo, w.len_hi, size=B, endpoint=True)
    lens[: min(w.full_len, B)] = w.seq
    return lens.astype(np.int32)


def activations(w: Workload, seed: int = SEED, batch: int | None = None) -> np.ndarray:
    """Slice input X ~ N(0, 1), shape [B, S, H]."""
    B = w.batch if batch is None else batch
    return _finish(_rng(seed, 2).normal(0.0, 1.0, (B, w.seq, w.hidden)), w.dtype)


def upstream_grad(w: Workload, seed: int = SEED, batch: int | None = None) -> np.ndarray:
    """Upstream gradient dY ~ N(0, dy_std), shape [B, S, H], padded rows included."""
    B = w.batch if batch is None else batch
    return _finish(_rng(seed, 4).normal(0.0, w.dy_std, (B, w.seq, w.hidden)), w.dtype)


def slice_params(w: Workload, seed: int = SEED, affine: str = "bert") -> list:
    return [layer_params(l, w.hidden, w.ffn, w.dtype, seed, affine)
            for l in range(w.layer_begin, w.layer_begin + w.layers)]


def custom(name: str = "custom", **kw) -> Workload:
    """A workload with explicit sizes (used for small parity cases)."""
    base = dict(layers=1, hidden=128, heads=2, ffn=512, seq=64, batch=2, dtype="bf16",
                len_lo=1, len_hi=64, dy_std=1e-2)
    base.update(kw)
    return Workload(name, **base)
