"""Seeded synthetic inputs for the QSVD latent-attention path.

This module is shared by the CPU oracle, the GPU tests and the benchmark.  It
draws random numbers and stores them in the formats the path consumes (bf16
bit patterns, fp32 values); it contains none of the method's arithmetic (no
SVD, no quantization, no projection, no attention).

Recipe (every draw from ``numpy.random.default_rng(seed)``, PCG64, fp64):

* Joint QKV weight of the tiny layer: ``W_qkv`` [d, 3d] ~ N(0, 1/d), the
  column blocks being W_q | W_k | W_v as in Eq. 2.
* Down-projection weight of the LLaVA-shaped layers (fp32 values):
  ``W_d[k, j] ~ N(0, 1/d) * (j+1)**-0.5`` -- column j scaled by sigma_j =
  j^-1/2 (1-based), the spread of singular values that Eq. 13 says the
  Sigma^beta factor puts on the latent's columns.
* Up-projections ``U_q, U_k, U_v`` [r, d] ~ N(0, 1/H_r) with H_r the r-th
  harmonic number, so that ``W_d @ U`` has the per-entry variance 1/d of a
  standard-initialised projection; rounded to bf16.
* Activations: rows ~ N(0, 1); image-like rows at unit scale, text-like rows
  at scale 0.5; a seeded set of outlier channels (1% of d, at least one)
  multiplied by 20 in every row -- the channel-wise outliers of Sec. 3.3.
  Rounded to bf16.

Draw order within a layer is fixed: weights (W, U_q, U_k, U_v), outlier
channels, prefill activations, then the decode activations step by step.
"""
from __future__ import annotations

import dataclasses
import math
from typing import List, Optional

import numpy as np

__all__ = [
    "bf16_bits", "bf16_from_bits", "LayerShape", "Workload", "WORKLOADS",
    "LayerInputs", "gen_layer", "gen_joint_qkv", "harmonic",
]


# --------------------------------------------------------------------------
# bf16 storage format (data representation only)
# --------------------------------------------------------------------------
def bf16_bits(x) -> np.ndarray:
    """fp64 -> fp32 (round to nearest even) -> bf16 bit pattern (round to
    nearest even on the 16 dropped bits).  Returns uint16."""
    f = np.ascontiguousarray(np.asarray(x, dtype=np.float64).astype(np.float32))
    u = f.view(np.uint32).astype(np.uint64)
    bias = np.uint64(0x7FFF) + ((u >> np.uint64(16)) & np.uint64(1))
    return ((u + bias) >> np.uint64(16)).astype(np.uint16)


def bf16_from_bits(b) -> np.ndarray:
    """bf16 bit pattern (uint16) -> exact fp64 value."""
    b = np.ascontiguousarray(np.asarray(b, dtype=np.uint16))
    return (b.astype(np.uint32) << np.uint32(16)).view(np.float32).astype(np.float64)


def harmonic(n: int) -> float:
    return float(np.sum(1.0 / np.arange(1, n + 1, dtype=np.float64)))


# --------------------------------------------------------------------------
# Shapes and workloads
# --------------------------------------------------------------------------
@dataclasses.dataclass(frozen=True)
class LayerShape:
    d: int      # hidden size E
    H: int      # heads
    dh: int     # head dim (H * dh == d)
    r: int      # joint rank

    def __post_init__(self):
        assert self.H * self.dh == self.d


@dataclasses.dataclass(frozen=True)
class Workload:
    name: str
    shape: LayerShape
    B: int                 # sequences
    n_image: int           # image-like prefill tokens per sequence
    n_text: int            # text-like prefill tokens per sequence
    decode_steps: int
    lat_bits: int          # 8 or 4 (latent cache precision)
    tiny_svd: bool = False  # weights from the joint SVD of a Gaussian W_qkv

    @property
    def prefill(self) -> int:
        return self.n_image + self.n_text

    @property
    def tmax(self) -> int:
        return self.prefill + self.decode_steps


_S7B = LayerShape(d=4096, H=32, dh=128, r=1536)
WORKLOADS = {
    # tiny single layer: d=256, H=4, dh=64, r=96, prefill 64, 16 decode steps
    "tiny": Workload("tiny", LayerShape(256, 4, 64, 96), B=1, n_image=0, n_text=64,
                     decode_steps=16, lat_bits=8, tiny_svd=True),
    # LLaVA-7B-shaped layer: 576 image + 64 text tokens, 128 decode steps, int8 cache
    "llava7b": Workload("llava7b", _S7B, B=1, n_image=576, n_text=64,
                        decode_steps=128, lat_bits=8),
    # decode-heavy 7B: batch 16, 4096 cached tokens each, int4 cache, 256 steps
    "decode7b_int4": Workload("decode7b_int4", _S7B, B=16, n_image=4096, n_text=0,
                              decode_steps=256, lat_bits=4),
    # LLaVA-13B-shaped layer: batch 8 of 5x576 image + 128 text, 512 steps
    "llava13b": Workload("llava13b", LayerShape(5120, 40, 128, 2048), B=8,
                         n_image=2880, n_text=128, decode_steps=512, lat_bits=8),
}


def sweep_point(r: int, L: int, B: int, lat_bits: int, steps: int = 1) -> Workload:
    """One point of the 32-layer 7B-shaped sweep (cache length L per sequence)."""
    return Workload(f"sweep_r{r}_L{L}_B{B}_i{lat_bits}", LayerShape(4096, 32, 128, r),
                    B=B, n_image=L, n_text=0, decode_steps=steps, lat_bits=lat_bits)


# --------------------------------------------------------------------------
# Draws
# --------------------------------------------------------------------------
def gen_joint_qkv(d: int, rng: np.random.Generator) -> np.ndarray:
    """W_concat = [W_q, W_k, W_v] in R^{d x 3d}, entries N(0, 1/d) (fp64)."""
    return rng.standard_normal((d, 3 * d)) / math.sqrt(d)


def _down_weight(d: int, r: int, rng) -> np.ndarray:
    w = rng.standard_normal((d, r)) / math.sqrt(d)
    w = w * (np.arange(1, r + 1, dtype=np.float64) ** -0.5)[None, :]
    return w.astype(np.float32).astype(np.float64)      # fp32 values


def _up_weight(r: int, d: int, rng) -> np.ndarray:
    return bf16_bits(rng.standard_normal((r, d)) / math.sqrt(harmonic(r)))


def _outlier_channels(d: int, rng) -> np.ndarray:
    n = max(1, int(round(0.01 * d)))
    return np.sort(rng.choice(d, size=n, replace=False))


def _activations(n_rows: int, d: int, row_scale: float, outliers, rng) -> np.ndarray:
    x = rng.standard_normal((n_rows, d)) * row_scale
    x[:, outliers] *= 20.0
    return bf16_bits(x)


@dataclasses.dataclass
class LayerInputs:
    """Everything one layer of a workload consumes, as stored bit patterns.

    ``W_qkv`` is set for the tiny workload (its W_d / U come from the joint
    SVD the caller performs); otherwise ``W_d`` (fp32 values, [d, r]) and the
    bf16 bit patterns of ``U_q, U_k, U_v`` ([r, d]) are set.
    ``X_prefill``: bf16 bits [B, prefill, d]; ``X_decode``: bf16 bits
    [steps, B, d] (``None`` when ``decode_steps == 0``).
    """
    workload: Workload
    seed: int
    W_qkv: Optional[np.ndarray]
    W_d: Optional[np.ndarray]
    U_q: Optional[np.ndarray]
    U_k: Optional[np.ndarray]
    U_v: Optional[np.ndarray]
    outliers: np.ndarray
    X_prefill: np.ndarray
    X_decode: Optional[np.ndarray]


def gen_layer(wl: Workload, seed: int = 0, layer: int = 0,
              prefill_rows: Optional[int] = None,
              decode_steps: Optional[int] = None) -> LayerInputs:
    """Draw one layer's inputs.  ``prefill_rows``/``decode_steps`` truncate
    the draws (the draw order is unchanged, so a truncated draw is a prefix
    of the full one for the weights and the prefill rows of sequence 0)."""
    s = wl.shape
    rng = np.random.default_rng(seed + layer)
    W_qkv = W_d = U_q = U_k = U_v = None
    if wl.tiny_svd:
        W_qkv = gen_joint_qkv(s.d, rng)
    else:
        W_d = _down_weight(s.d, s.r, rng)
        U_q = _up_weight(s.r, s.d, rng)
        U_k = _up_weight(s.r, s.d, rng)
        U_v = _up_weight(s.r, s.d, rng)
    outl = _outlier_channels(s.d, rng)
    if wl.tiny_svd:     # tiny layer: 4 outlier channels
        outl = np.sort(rng.choice(s.d, size=4, replace=False))
    n_pre = wl.prefill if prefill_rows is None else prefill_rows
    rows: List[np.ndarray] = []
    for _b in range(wl.B):
        n_img = min(wl.n_image, n_pre)
        n_txt = min(wl.n_text, max(0, n_pre - n_img))
        parts = []
        if n_img:
            parts.append(_activations(n_img, s.d, 1.0, outl, rng))
        if n_txt:
            parts.append(_activations(n_txt, s.d, 1.0 if wl.tiny_svd else 0.5, outl, rng))
        rows.append(np.concatenate(parts, axis=0) if parts else
                    np.zeros((0, s.d), np.uint16))
    X_prefill = np.stack(rows, axis=0)
    steps = wl.decode_steps if decode_steps is None else decode_steps
    X_decode = None
    if steps:
        X_decode = np.stack([_activations(wl.B, s.d, 1.0 if wl.tiny_svd else 0.5, outl, rng)
                             for _ in range(steps)], axis=0)
    return LayerInputs(wl, seed, W_qkv, W_d, U_q, U_k, U_v, outl, X_prefill, X_decode)


def latent_rows(n_rows: int, r: int, rng) -> np.ndarray:
    """Latent rows shaped like x W_d of the synthetic layers: channel j has
    standard deviation (j+1)^-0.5 (the spectrum decay of the down-projection)
    times a per-token magnitude drawn log-uniformly from [0.5, 2]; fp32
    values as fp64 [n_rows, r]."""
    decay = np.arange(1, r + 1, dtype=np.float64) ** -0.5
    mag = np.exp(rng.uniform(math.log(0.5), math.log(2.0), size=(n_rows, 1)))
    x = rng.standard_normal((n_rows, r)) * decay[None, :] * mag
    return x.astype(np.float32).astype(np.float64)
