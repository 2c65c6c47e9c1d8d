"""Seeded synthetic inputs for the block-calibration step.

This module only draws random numbers and shapes them; it holds none of the
method's arithmetic (no quantizer, no transformation, no block forward).  Both
the CUDA path and the fp64 oracle are fed from here, so the two sides see the
same tensors.

The calibration data of the paper (128 segments of 2048 tokens, Sec. 4.1
"Training") and the LLaMA weights are not available, so seeded tensors of the
same shapes and of the distributions below stand in for them:

* block input x [T, d]: N(0, 1), with a fixed random set of outlier channels
  scaled by a constant factor (1% x50 for the 7B/13B shapes, 0.5% x100 for the
  70B shape).  The outlier channels are chosen once from the weight seed, so
  every sample of a block shares them, as activation outliers do (Sec. 3.3).
* weights [Cout, Cin]: N(0, std) rounded to bf16 (the frozen weights are bf16
  in HBM).  The single-linear case draws Student-t(3) samples scaled to unit
  variance and then to std 0.02.
* LWC logits: gamma_hat = beta_hat = 4.0 (sigmoid ~ 0.982); test cases can
  perturb them so that clipping is active.
* LET parameters, drawn rather than computed: per-channel scales exp(N(0, 0.1))
  times sqrt(outlier factor) on the generator's own outlier channels (the
  magnitude pattern a smoothing initialisation gives them), shifts N(0, 0.05);
  the [v, o] pair and the Q/K scale start near identity with a small seeded
  perturbation.  The method's own initialisation (SmoothQuant-style scales and
  channel means of the block's statistics) is computed by the library's LET
  initialisation and by the oracle, not here.
"""
from __future__ import annotations

import dataclasses
import math
from typing import Dict, Optional

import numpy as np

__all__ = ["BlockShape", "LinearShape", "SHAPES", "block_shape", "make_linear_case",
           "make_block_weights", "make_block_input", "make_block_theta", "bf16_representable"]


@dataclasses.dataclass(frozen=True)
class LinearShape:
    """Single quantized linear layer (the W4A16 g128 unit case)."""
    name: str
    T: int
    Cin: int
    Cout: int
    wbits: int = 4
    abits: int = 16
    group: int = 128
    w_std: float = 0.02
    gamma0: float = 4.0
    beta0: float = 4.0


@dataclasses.dataclass(frozen=True)
class BlockShape:
    """LLaMA-style decoder block: RMSNorm, RoPE attention, SwiGLU FFN."""
    name: str
    T: int
    d: int
    n_heads: int
    n_kv: int
    ffn: int
    wbits: int
    abits: int
    group: int          # 0 = one group per output channel
    let: int            # learnable equivalent transformation on/off
    head_dim: int = 128
    w_std: float = 0.02
    outlier_frac: float = 0.01
    outlier_scale: float = 50.0
    rms_eps: float = 1e-6
    rope_theta: float = 10000.0
    gamma0: float = 4.0
    beta0: float = 4.0

    @property
    def dq(self) -> int:
        return self.n_heads * self.head_dim

    @property
    def dkv(self) -> int:
        return self.n_kv * self.head_dim

    def with_(self, **kw) -> "BlockShape":
        return dataclasses.replace(self, **kw)


SHAPES: Dict[str, object] = {
    "linear_w4a16_g128": LinearShape("linear_w4a16_g128", T=256, Cin=512, Cout=512),
    "llama7b_w3a16_g128": BlockShape("llama7b_w3a16_g128", T=2048, d=4096, n_heads=32, n_kv=32,
                                     ffn=11008, wbits=3, abits=16, group=128, let=0),
    "llama7b_w4a4": BlockShape("llama7b_w4a4", T=2048, d=4096, n_heads=32, n_kv=32,
                               ffn=11008, wbits=4, abits=4, group=0, let=1),
    "llama13b_w2a16_g64": BlockShape("llama13b_w2a16_g64", T=2048, d=5120, n_heads=40, n_kv=40,
                                     ffn=13824, wbits=2, abits=16, group=64, let=0),
    "llama2_70b_w4a4_gqa": BlockShape("llama2_70b_w4a4_gqa", T=2048, d=8192, n_heads=64, n_kv=8,
                                      ffn=28672, wbits=4, abits=4, group=0, let=1,
                                      w_std=0.015, outlier_frac=0.005, outlier_scale=100.0,
                                      rms_eps=1e-5),
}


def block_shape(name: str, **override) -> BlockShape:
    s = SHAPES[name]
    assert isinstance(s, BlockShape)
    return s.with_(**override) if override else s


def bf16_representable(a: np.ndarray) -> np.ndarray:
    """Return float32 values that are exactly representable in bf16.

    Uses round-to-nearest-even on the float32 bit pattern; this is the storage
    format of the frozen weights, not part of the method."""
    a = np.ascontiguousarray(a, dtype=np.float32)
    u = a.view(np.uint32)
    lsb = (u >> np.uint32(16)) & np.uint32(1)
    u = (u + np.uint32(0x7FFF) + lsb) & np.uint32(0xFFFF0000)
    return u.view(np.float32)


def _rng(seed: int) -> np.random.Generator:
    return np.random.Generator(np.random.PCG64(seed))


# ----------------------------------------------------------------------------------------------
# single linear case
# ----------------------------------------------------------------------------------------------

def make_linear_case(shape: LinearShape, seed: int = 0, perturb_theta: bool = False):
    """X [T, Cin] fp32 N(0,1); W [Cout, Cin] Student-t(3) scaled to std w_std, bf16 values;
    B = 0; LWC logits [Cout, Cin/group] at gamma0/beta0 (optionally perturbed)."""
    rng = _rng(seed)
    X = rng.standard_normal((shape.T, shape.Cin)).astype(np.float32)
    t = rng.standard_t(3, size=(shape.Cout, shape.Cin)) / math.sqrt(3.0)   # unit variance
    W = bf16_representable((shape.w_std * t).astype(np.float32))
    ng = shape.Cin // (shape.group if shape.group > 0 else shape.Cin)
    gl = np.full((shape.Cout, ng), shape.gamma0, np.float32)
    bl = np.full((shape.Cout, ng), shape.beta0, np.float32)
    if perturb_theta:
        gl = gl + rng.normal(-2.5, 1.0, gl.shape).astype(np.float32)
        bl = bl + rng.normal(-2.5, 1.0, bl.shape).astype(np.float32)
    B = np.zeros((shape.Cout,), np.float32)
    return dict(X=X, W=W, B=B, gamma_logit=gl, beta_logit=bl)


# ----------------------------------------------------------------------------------------------
# decoder block
# ----------------------------------------------------------------------------------------------

def _outlier_channels(shape: BlockShape, seed: int) -> np.ndarray:
    rng = _rng(seed + 7919)
    n = int(round(shape.outlier_frac * shape.d))
    return np.sort(rng.choice(shape.d, size=n, replace=False))


def make_block_weights(shape: BlockShape, seed: int = 1) -> Dict[str, np.ndarray]:
    """Frozen weights of one block, [Cout, Cin] row-major, values exactly representable in bf16."""
    rng = _rng(seed)
    d, dq, dkv, f = shape.d, shape.dq, shape.dkv, shape.ffn

    def w(cout, cin):
        v = rng.standard_normal((cout, cin), dtype=np.float32)
        v *= np.float32(shape.w_std)
        return bf16_representable(v)

    return dict(wq=w(dq, d), wk=w(dkv, d), wv=w(dkv, d), wo=w(d, dq),
                wg=w(f, d), wu=w(f, d), wd=w(d, f))


def make_block_input(shape: BlockShape, sample: int = 0, weight_seed: int = 1) -> np.ndarray:
    """Block input x [T, d] fp32 for calibration sample `sample`."""
    rng = _rng(1000 + sample)
    x = rng.standard_normal((shape.T, shape.d), dtype=np.float32)
    ch = _outlier_channels(shape, weight_seed)
    x[:, ch] *= np.float32(shape.outlier_scale)
    return x


def make_block_theta(shape: BlockShape, weights: Dict[str, np.ndarray], x: Optional[np.ndarray] = None,
                     seed: int = 2, perturb: bool = False, weight_seed: int = 1) -> Dict[str, np.ndarray]:
    """Learnable parameters Theta1 (LWC logits per linear) and Theta2 (LET s, delta, s_a), drawn.

    `perturb` spreads the LWC logits so that clipping is active in many groups (test cases).
    `x` is not used (kept for call compatibility); `weight_seed` selects the outlier channels that
    make_block_input scaled."""
    rng = _rng(seed)
    th: Dict[str, np.ndarray] = {}
    for name in ("wq", "wk", "wv", "wo", "wg", "wu", "wd"):
        cout, cin = weights[name].shape
        ng = cin // (shape.group if shape.group > 0 else cin)
        g = np.full((cout, ng), shape.gamma0, np.float32)
        b = np.full((cout, ng), shape.beta0, np.float32)
        if perturb:
            g = g + rng.normal(-2.0, 1.5, g.shape).astype(np.float32)
            b = b + rng.normal(-2.0, 1.5, b.shape).astype(np.float32)
        th["gamma_" + name[1:]] = g
        th["beta_" + name[1:]] = b
    if shape.let:
        ch = _outlier_channels(shape, weight_seed)
        boost = np.ones(shape.d, np.float32)
        boost[ch] = np.float32(math.sqrt(shape.outlier_scale))
        th["s1"] = (np.exp(rng.normal(0.0, 0.1, shape.d)) * boost).astype(np.float32)
        th["d1"] = rng.normal(0.0, 0.05, shape.d).astype(np.float32)
        th["s2"] = (np.exp(rng.normal(0.0, 0.1, shape.d)) * boost).astype(np.float32)
        th["d2"] = rng.normal(0.0, 0.05, shape.d).astype(np.float32)
        th["so"] = np.exp(rng.normal(0.0, 0.1, shape.dkv)).astype(np.float32)
        th["do"] = rng.normal(0.0, 0.01, shape.dkv).astype(np.float32)
        th["sa"] = np.exp(rng.normal(0.0, 0.1, shape.dkv)).astype(np.float32)
        if perturb:
            th["s1"] *= np.exp(rng.normal(0.0, 0.1, shape.d)).astype(np.float32)
            th["d1"] += rng.normal(0.0, 0.05, shape.d).astype(np.float32)
            th["s2"] *= np.exp(rng.normal(0.0, 0.1, shape.d)).astype(np.float32)
            th["d2"] += rng.normal(0.0, 0.05, shape.d).astype(np.float32)
    return th
