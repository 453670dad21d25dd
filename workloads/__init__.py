"""Seeded synthetic inputs for the block-CAT W4A4 linear layer.

This module only draws random inputs: activations (calibration and evaluation
splits), weights, outlier-channel choices and the random signs of a randomized
Hadamard transform.  It contains none of the layer's arithmetic (no transform,
no quantizer, no GEMM), so the CPU oracle and the CUDA path can both take their
inputs from here without sharing any method code.

The paper calibrates and evaluates on real LLM layers (Sec. 6: Llama/Qwen
linear layers, 128 x 2048 DCLM-edu calibration tokens).  Those weights and
datasets are not available, so the generators below stand in for them with
layer shapes taken from Llama-3-8B / Llama-3-70B and activation statistics that
reproduce what the paper's analysis is about (Sec. 2 "Concentration" and
"Alignment"): correlated bulk channels, a few massive outlier channels, heavy
tails, and weight rows with unequal energy.

Every array is drawn in float64 (weights of the large layers in float32 to keep
host memory bounded) with ``numpy.random.default_rng`` and cast once to the
layer dtype.  bf16 layers keep both the bf16 bit patterns (``uint16``) and the
same values widened to float32, so both sides read identical numbers.
"""
from __future__ import annotations

import dataclasses
from typing import Dict, Optional, Tuple

import numpy as np


@dataclasses.dataclass(frozen=True)
class LayerConfig:
    """One synthetic linear layer y = W x with its calibration split."""

    name: str
    d_in: int
    d_out: int
    n_eval: int
    n_calib: int
    k: int                      # CAT block size
    dtype: str                  # "f32" or "bf16"
    seed: int
    act: str                    # activation recipe: "lowrank_outlier", "wishart_outlier", "swiglu"
    outlier_frac: float = 0.0
    outlier_count: int = 0      # used instead of outlier_frac when > 0
    outlier_scale: float = 1.0
    lowrank: int = 64
    iso_var: float = 0.1
    w_dist: str = "normal"      # "normal" or "student_t"
    w_std: float = 0.02
    w_row_lognormal_sigma: float = 0.0   # > 0: rows scaled by LogNormal(0, sigma^2)
    k_sweep: Tuple[int, ...] = ()
    description: str = ""

    @property
    def n_outliers(self) -> int:
        if self.outlier_count > 0:
            return self.outlier_count
        return int(round(self.outlier_frac * self.d_in))


CONFIGS: Dict[str, LayerConfig] = {
    "c1_256x256_k32_f32": LayerConfig(
        name="c1_256x256_k32_f32", d_in=256, d_out=256, n_eval=512, n_calib=128, k=32,
        dtype="f32", seed=0, act="wishart_outlier", outlier_count=4, outlier_scale=50.0,
        w_dist="student_t", w_std=0.02,
        description="single linear layer 256->256, 512 tokens, k=32, fp32; x ~ N(0, A A^T/256) with 4 "
                    "outlier channels x50; W ~ Student-t(5) x 0.02"),
    "c2_qkv_4096x6144_k128_bf16": LayerConfig(
        name="c2_qkv_4096x6144_k128_bf16", d_in=4096, d_out=6144, n_eval=2048, n_calib=512, k=128,
        dtype="bf16", seed=2, act="lowrank_outlier", outlier_frac=0.01, outlier_scale=100.0,
        w_std=0.02, w_row_lognormal_sigma=0.5,
        description="Llama-3-8B fused QKV projection 4096->6144, 2048 tokens, k=128, bf16; low-rank(64) "
                    "correlated bulk + isotropic 0.1, 1% outlier channels x100; W ~ N(0, 0.02^2) with "
                    "LogNormal(0, 0.5^2) row scales"),
    "c3_down_14336x4096_k128_bf16": LayerConfig(
        name="c3_down_14336x4096_k128_bf16", d_in=14336, d_out=4096, n_eval=4096, n_calib=512, k=128,
        dtype="bf16", seed=3, act="swiglu", w_std=0.015,
        description="Llama-3-8B MLP down projection 14336->4096, 4096 tokens, k=128, bf16; x = SiLU(g)*u; "
                    "W ~ N(0, 0.015^2)"),
    "c4_decode_up_4096x14336_k128_bf16": LayerConfig(
        name="c4_decode_up_4096x14336_k128_bf16", d_in=4096, d_out=14336, n_eval=16, n_calib=512, k=128,
        dtype="bf16", seed=4, act="lowrank_outlier", outlier_frac=0.01, outlier_scale=100.0,
        w_std=0.02, w_row_lognormal_sigma=0.5,
        description="decode-shaped up projection 4096->14336, 16 tokens, k=128, bf16; generators of the "
                    "QKV layer"),
    "c5_gateup_8192x28672_bf16": LayerConfig(
        name="c5_gateup_8192x28672_bf16", d_in=8192, d_out=28672, n_eval=8192, n_calib=512, k=128,
        dtype="bf16", seed=5, act="lowrank_outlier", outlier_frac=0.005, outlier_scale=200.0,
        w_std=0.01, k_sweep=(32, 64, 128, 256),
        description="Llama-3-70B gate/up projection 8192->28672, 8192 tokens, bf16, k in {32,64,128,256}; "
                    "low-rank bulk, 0.5% outlier channels x200; W ~ N(0, 0.01^2)"),
}

# Order in which the configurations are usually listed.
CONFIG_ORDER = ("c1_256x256_k32_f32", "c2_qkv_4096x6144_k128_bf16", "c3_down_14336x4096_k128_bf16",
                "c4_decode_up_4096x14336_k128_bf16", "c5_gateup_8192x28672_bf16")


def small_config(name: str, d_in: int, d_out: int, n_eval: int, n_calib: int, k: int, dtype: str = "bf16",
                 seed: int = 11, act: str = "lowrank_outlier", **kw) -> LayerConfig:
    """A reduced layer with the generators of the large ones (tests use these for
    tile-spanning, ragged shapes that the oracle finishes in seconds)."""
    base = dict(outlier_frac=0.01, outlier_scale=100.0, w_std=0.02, w_row_lognormal_sigma=0.5, lowrank=16)
    if act == "wishart_outlier":
        base = dict(outlier_count=2, outlier_scale=50.0, w_dist="student_t", w_std=0.02)
    if act == "swiglu":
        base = dict(w_std=0.015)
    base.update(kw)
    return LayerConfig(name=name, d_in=d_in, d_out=d_out, n_eval=n_eval, n_calib=n_calib, k=k, dtype=dtype,
                       seed=seed, act=act, **base)


# ----------------------------------------------------------------------------------------------
# dtype handling
# ----------------------------------------------------------------------------------------------

def to_bf16_bits(a: np.ndarray) -> np.ndarray:
    """Round float values to bfloat16 (round to nearest, ties to even); return the uint16 bit patterns."""
    f = np.ascontiguousarray(a, dtype=np.float32)
    u = f.view(np.uint32)  # finite values: u + 0x8000 cannot overflow 32 bits
    rounded = (u + np.uint32(0x7FFF) + ((u >> np.uint32(16)) & np.uint32(1))) >> np.uint32(16)
    return rounded.astype(np.uint16)


def bf16_bits_to_f32(b: np.ndarray) -> np.ndarray:
    """Widen bfloat16 bit patterns to float32 (exact)."""
    return (b.astype(np.uint32) << 16).view(np.float32)


@dataclasses.dataclass
class Tensor:
    """A host array in the layer dtype.

    ``values`` holds the numbers as float32 (exact for both dtypes); ``raw`` holds what a
    device buffer of the layer dtype contains (float32 values, or uint16 bf16 bit patterns)."""

    values: np.ndarray
    raw: np.ndarray
    dtype: str

    @property
    def shape(self):
        return self.values.shape


def cast(a: np.ndarray, dtype: str) -> Tensor:
    if dtype == "f32":
        v = np.ascontiguousarray(a, dtype=np.float32)
        return Tensor(values=v, raw=v, dtype="f32")
    if dtype == "bf16":
        bits = to_bf16_bits(a)
        return Tensor(values=bf16_bits_to_f32(bits), raw=bits, dtype="bf16")
    raise ValueError(f"unknown dtype {dtype}")


# ----------------------------------------------------------------------------------------------
# generators
# ----------------------------------------------------------------------------------------------

def _streams(seed: int):
    """Independent streams: distribution parameters, calibration draw, evaluation draw, weights, signs."""
    ss = np.random.SeedSequence(seed)
    dist, calib, ev, wt, signs = ss.spawn(5)
    return (np.random.default_rng(dist), np.random.default_rng(calib), np.random.default_rng(ev),
            np.random.default_rng(wt), np.random.default_rng(signs))


class _ActDist:
    """Activation distribution of one layer; draws token batches [n, d_in] in float64."""

    def __init__(self, cfg: LayerConfig, rng_dist: np.random.Generator):
        self.cfg = cfg
        d = cfg.d_in
        if cfg.act == "wishart_outlier":
            self.A = rng_dist.standard_normal((d, d))
        elif cfg.act == "lowrank_outlier":
            self.F = rng_dist.standard_normal((d, cfg.lowrank)) / np.sqrt(cfg.lowrank)
        elif cfg.act != "swiglu":
            raise ValueError(cfg.act)
        n_out = cfg.n_outliers
        self.outliers = np.sort(rng_dist.choice(d, size=n_out, replace=False)) if n_out > 0 else np.zeros(0, int)

    def draw(self, rng: np.random.Generator, n: int) -> np.ndarray:
        cfg, d = self.cfg, self.cfg.d_in
        if cfg.act == "wishart_outlier":
            z = rng.standard_normal((n, d))
            x = z @ self.A.T / np.sqrt(d)          # x_t = A z_t / sqrt(d): covariance A A^T / d
        elif cfg.act == "lowrank_outlier":
            z = rng.standard_normal((n, cfg.lowrank))
            eps = rng.standard_normal((n, d))
            x = z @ self.F.T + np.sqrt(cfg.iso_var) * eps
        else:  # swiglu: SiLU(g) * u
            g = rng.standard_normal((n, d))
            u = rng.standard_normal((n, d))
            x = g / (1.0 + np.exp(-g)) * u
        if self.outliers.size:
            x[:, self.outliers] *= cfg.outlier_scale
        return x


def _weights(cfg: LayerConfig, rng: np.random.Generator) -> np.ndarray:
    shape = (cfg.d_out, cfg.d_in)
    big = cfg.d_out * cfg.d_in > (1 << 24)
    if cfg.w_dist == "student_t":
        w = rng.standard_t(5.0, size=shape) * cfg.w_std
    else:
        w = rng.standard_normal(shape, dtype=np.float32 if big else np.float64)
        w *= cfg.w_std
    if cfg.w_row_lognormal_sigma > 0:
        rho = np.exp(cfg.w_row_lognormal_sigma * rng.standard_normal(cfg.d_out))
        w *= rho[:, None].astype(w.dtype)
    return w


@dataclasses.dataclass
class Layer:
    cfg: LayerConfig
    x_calib: Tensor            # [n_calib, d_in]
    x_eval: Tensor             # [n_eval, d_in]
    W: Tensor                  # [d_out, d_in]
    rht_signs: np.ndarray      # [d_in] float64 in {-1, +1}
    outlier_channels: np.ndarray


def make_layer(cfg: LayerConfig, n_eval: Optional[int] = None, with_weights: bool = True) -> Layer:
    """Draw one layer.  ``n_eval`` overrides the number of evaluation tokens."""
    rng_dist, rng_calib, rng_eval, rng_w, rng_sign = _streams(cfg.seed)
    dist = _ActDist(cfg, rng_dist)
    xc = cast(dist.draw(rng_calib, cfg.n_calib), cfg.dtype)
    xe = cast(dist.draw(rng_eval, cfg.n_eval if n_eval is None else n_eval), cfg.dtype)
    if with_weights:
        W = cast(_weights(cfg, rng_w), cfg.dtype)
    else:
        W = cast(np.zeros((0, cfg.d_in)), cfg.dtype)
    signs = rng_sign.choice(np.array([-1.0, 1.0]), size=cfg.d_in)
    return Layer(cfg=cfg, x_calib=xc, x_eval=xe, W=W, rht_signs=signs, outlier_channels=dist.outliers)


def random_codes(rng: np.random.Generator, shape, qmax: int = 7) -> np.ndarray:
    """Uniform integer codes in [-qmax, qmax] (int8), for GEMM tests fed with given codes."""
    return rng.integers(-qmax, qmax + 1, size=shape, dtype=np.int64).astype(np.int8)
