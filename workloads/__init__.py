"""Seeded synthetic inputs for the MoE-ViE MoE FFN layer.

This module is the one piece shared by the CPU oracle and the CUDA library's
tests and benchmark.  It draws random numbers and lays them out; it holds none
of the method's arithmetic (no routing, no sigmoid, no top-k, no GELU).

Recipe (seed 0, ``numpy.random.default_rng``, draw order fixed as below):

* ``x   [T, d]``       N(0, 1) rounded to bf16 (tokens as after a LayerNorm)
* ``W_r [d, E]``       N(0, 0.02^2) fp32 (0.02 read as the standard deviation)
* ``b   [E]``          U(-0.1, 0.1) fp32
* ``W1  [E, d, h]``    N(0, 1/d) rounded to bf16 (1/fan_in read as the variance)
* ``W2  [E, h, d]``    N(0, 1/h) rounded to bf16
* ``Ws1 [d, h_s]``, ``Ws2 [h_s, d]``  the same rule, only when ``h_s > 0``

Skewed expert loads (the video and stress layers) are made by one constant
feature: ``x[:, d-1] = 1`` and ``W_r[d-1, e] = o_e``, so every logit of expert e
is shifted by ``o_e``.  The offsets ``o_e`` are stored in ``skew_offsets.json``;
they were fitted once, offline, by ``oracle/calibrate_skew.py`` against a target
per-expert load (Zipf with a few empty experts), and are plain input data here.

bf16 values travel as ``uint16`` bit patterns (the upper half of an fp32).
"""
from __future__ import annotations

import json
import os
from dataclasses import dataclass, field

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
SKEW_FILE = os.path.join(_HERE, "skew_offsets.json")


@dataclass(frozen=True)
class LayerConfig:
    """Shape and input recipe of one MoE FFN layer workload."""
    name: str
    T: int
    d: int
    E: int
    k: int
    h: int
    h_s: int = 0            # shared expert width, 0 = none
    lam: float = 1.0        # weight of the shared expert
    seed: int = 0
    skew: str | None = None  # key into skew_offsets.json, or None for no skew
    note: str = ""
    act: str = "gelu"       # expert FFN: "gelu", or "swiglu" (W1 gate, W3 up; App. B)

    @property
    def slots(self) -> int:
        return self.T * self.k


# The five layer workloads: token counts are whole images / clips of ViT patches
# (256 patches per 224^2 image at patch 14-16, 1024 for 448^2 at patch 14).
CONFIGS = {
    "c0": LayerConfig("c0", T=512, d=768, E=16, k=2, h=768,
                      note="2 images x 256 patches, no shared expert"),
    "c1": LayerConfig("c1", T=8192, d=1024, E=64, k=8, h=512, h_s=1024, lam=1.0,
                      note="32 images x 256 patches, one shared expert h_s=1024"),
    "c2": LayerConfig("c2", T=1024, d=1536, E=64, k=8, h=768,
                      note="batch-1 448x448 image at patch 14 (weight-bandwidth bound)"),
    "c3": LayerConfig("c3", T=32768, d=1536, E=128, k=8, h=384, skew="c3",
                      note="4 clips x 32 frames x 256 patches, Zipf(1.0) loads, 4 empty experts"),
    "c4": LayerConfig("c4", T=65536, d=1664, E=256, k=8, h=416, skew="c4",
                      note="stress layer: one saturated expert, Zipf(1.1) over the rest, 3 empty"),
    # SwiGLU experts (the paper's own FFN, App. B) at the image-batch layer's routed shape
    "s1": LayerConfig("s1", T=8192, d=1024, E=64, k=8, h=512, act="swiglu",
                      note="32 images x 256 patches, SwiGLU experts (W1 gate, W3 up), no shared expert"),
    # The paper's own MoE-ViE-B / L / H layers (App. D, model table): 32 experts of width
    # 512 / 684 / 854 per layer, one of them shared, 4 / 4 / 8 activated counting the
    # shared one: E = 31 routed, k = 3 / 3 / 7, h_s = h, SwiGLU.  8192 tokens: 32 images
    # x 256 patches (B, L), 8 images x 1024 patches at 448^2, patch 14 (H).
    "pB": LayerConfig("pB", T=8192, d=768, E=31, k=3, h=512, h_s=512, act="swiglu",
                      note="MoE-ViE-B layer: 31 routed + 1 shared SwiGLU experts of width 512"),
    "pL": LayerConfig("pL", T=8192, d=1024, E=31, k=3, h=684, h_s=684, act="swiglu",
                      note="MoE-ViE-L layer: 31 routed + 1 shared SwiGLU experts of width 684"),
    "pH": LayerConfig("pH", T=8192, d=1280, E=31, k=7, h=854, h_s=854, act="swiglu",
                      note="MoE-ViE-H layer: 31 routed + 1 shared SwiGLU experts of width 854"),
}


def f32_to_bf16_bits(a: np.ndarray) -> np.ndarray:
    """Round fp32 values to the nearest bf16 (ties to even); return the bit patterns.

    The rounding is torch's fp32 -> bf16 conversion on the CPU (round to nearest,
    ties to even: add 0x7FFF plus the lowest kept bit, drop the low 16 bits), used
    here only because it is multithreaded."""
    import torch
    t = torch.from_numpy(np.ascontiguousarray(a, dtype=np.float32))
    return t.to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16).copy()


def bf16_bits_to_f32(b: np.ndarray) -> np.ndarray:
    """Widen bf16 bit patterns to fp32 (exact)."""
    b = np.ascontiguousarray(b, dtype=np.uint16)
    return (b.astype(np.uint32) << 16).view(np.float32)


@dataclass
class LayerInputs:
    cfg: LayerConfig
    x: np.ndarray            # uint16 [T, d] (bf16 bits)
    Wr: np.ndarray           # float32 [d, E]
    b: np.ndarray            # float32 [E]
    W1: np.ndarray           # uint16 [E, d, h]
    W2: np.ndarray           # uint16 [E, h, d]
    Ws1: np.ndarray | None = None   # uint16 [d, h_s]
    Ws2: np.ndarray | None = None   # uint16 [h_s, d]
    extra: dict = field(default_factory=dict)
    W3: np.ndarray | None = None    # uint16 [E, d, h], SwiGLU layers only
    Ws3: np.ndarray | None = None   # uint16 [d, h_s], SwiGLU layers with a shared expert


def _normal_bf16(rng: np.random.Generator, shape, std: float) -> np.ndarray:
    v = rng.standard_normal(size=shape, dtype=np.float32)
    if std != 1.0:
        np.multiply(v, np.float32(std), out=v)
    return f32_to_bf16_bits(v)


def load_skew_offsets(key: str) -> np.ndarray | None:
    if not os.path.exists(SKEW_FILE):
        return None
    with open(SKEW_FILE) as f:
        table = json.load(f)
    if key not in table:
        return None
    return np.asarray(table[key]["offsets"], dtype=np.float32)


def make_layer(cfg: LayerConfig, skew_offsets: np.ndarray | None = None,
               require_skew: bool = True) -> LayerInputs:
    """Draw the layer inputs of ``cfg``.

    For a skewed config the stored offsets are applied (pass ``skew_offsets`` to
    override, e.g. zeros while fitting them).  ``require_skew`` makes a missing
    table an error instead of silently producing an unskewed layer.
    """
    rng = np.random.default_rng(cfg.seed)
    T, d, E, h = cfg.T, cfg.d, cfg.E, cfg.h
    x = _normal_bf16(rng, (T, d), 1.0)
    Wr = (rng.standard_normal(size=(d, E), dtype=np.float32) * np.float32(0.02)).astype(np.float32)
    b = rng.uniform(-0.1, 0.1, size=E).astype(np.float32)
    W1 = _normal_bf16(rng, (E, d, h), 1.0 / np.sqrt(d))
    W2 = _normal_bf16(rng, (E, h, d), 1.0 / np.sqrt(h))
    Ws1 = Ws2 = None
    if cfg.h_s > 0:
        Ws1 = _normal_bf16(rng, (d, cfg.h_s), 1.0 / np.sqrt(d))
        Ws2 = _normal_bf16(rng, (cfg.h_s, d), 1.0 / np.sqrt(cfg.h_s))
    W3 = Ws3 = None
    if cfg.act == "swiglu":   # drawn last: the GELU layers' draws are unchanged
        W3 = _normal_bf16(rng, (E, d, h), 1.0 / np.sqrt(d))
        if cfg.h_s > 0:
            Ws3 = _normal_bf16(rng, (d, cfg.h_s), 1.0 / np.sqrt(d))
    extra = {}
    if cfg.skew is not None:
        offs = skew_offsets if skew_offsets is not None else load_skew_offsets(cfg.skew)
        if offs is None:
            if require_skew:
                raise FileNotFoundError(f"no skew offsets for {cfg.skew!r} in {SKEW_FILE}")
        else:
            offs = np.asarray(offs, dtype=np.float32)
            assert offs.shape == (E,)
            x[:, d - 1] = f32_to_bf16_bits(np.ones(1, np.float32))[0]
            Wr[d - 1, :] = offs
            extra["skew_offsets"] = offs
    return LayerInputs(cfg, x, Wr, b, W1, W2, Ws1, Ws2, extra, W3, Ws3)


def small_config(T, d, E, k, h, h_s=0, lam=1.0, seed=0, name="small", act="gelu") -> LayerConfig:
    """An unskewed layer of arbitrary shape (tests)."""
    return LayerConfig(name, T=T, d=d, E=E, k=k, h=h, h_s=h_s, lam=lam, seed=seed, act=act)


# ---------------------------------------------------------------- skew targets

def skew_layout(cfg: LayerConfig) -> dict:
    """Target per-expert load of a skewed layer (number of routed slots per expert).

    c3: Zipf(s=1.0) over the 124 non-empty experts, 4 experts empty.
    c4: one expert takes every token (T slots, the most one expert can hold, as
    each token picks k distinct experts), Zipf(s=1.1) over 252 others, 3 empty.
    Loads above T are capped at T and the excess is water-filled onto the rest in
    proportion.  Which expert ids are hot, empty or where in the Zipf order they
    sit comes from a permutation drawn with seed ``cfg.seed + 1``.
    """
    E, T, total = cfg.E, cfg.T, cfg.T * cfg.k
    perm = np.random.default_rng(cfg.seed + 1).permutation(E)
    if cfg.skew == "c3":
        n_empty, n_hot, s = 4, 0, 1.0
    elif cfg.skew == "c4":
        n_empty, n_hot, s = 3, 1, 1.1
    else:
        raise ValueError(cfg.skew)
    empty = np.sort(perm[:n_empty])
    hot = perm[n_empty:n_empty + n_hot]
    rest = perm[n_empty + n_hot:]
    target = np.zeros(E, np.float64)
    target[hot] = T
    remaining = total - n_hot * T
    w = 1.0 / np.arange(1, rest.size + 1, dtype=np.float64) ** s
    alloc = np.zeros(rest.size)
    free = np.ones(rest.size, bool)
    for _ in range(rest.size):
        share = remaining * w * free / (w * free).sum()
        alloc = np.where(free, share, alloc)
        over = free & (alloc > T)
        if not over.any():
            break
        alloc[over] = T
        remaining -= T * over.sum()
        free &= ~over
    target[rest] = alloc
    return {"target": target, "empty": empty, "hot": hot}
