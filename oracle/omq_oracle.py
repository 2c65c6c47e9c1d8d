"""fp64 CPU oracle of one OmniQuant block-calibration step (Algorithm 1, inner loop).

TEST INFRASTRUCTURE ONLY: imported by `tests/`, `__graft_entry__.smoke()` and the
CPU legs of `bench.py`, never by the product path.  Plain PyTorch CPU ops in
float64; a matrix product is the only library primitive used as a step.

What it computes, in the paper's notation:

* Eq. 2 (LWC):  W_q = clamp(round(W/h) + z, 0, 2^N - 1),
  h = (gamma*max(W) - beta*min(W)) / (2^N - 1),  z = -round(beta*min(W)/h),
  gamma = sigmoid(gamma_hat), beta = sigmoid(beta_hat)  (Sec. 3.2).
  The fake-quantized value fed to the matmul is (W_q - z) * h.
* Q_a, the per-token MinMax activation quantizer (Sec. 3.3 after Eq. 4; per-token
  granularity in Sec. 4.1) = the same map with gamma = beta = 1, one group per
  token row.
* Eq. 3 / Eq. 4 (LET on a linear): X~ = (X - delta) / s,  W~ = s (.) W,
  B~ = B + delta W,  Y = Q_a(X~) Q_w(W~) + B~.
* Eq. 5 (LET on Q K^T):  Q~ = Q / s_a,  K~ = K (.) s_a, both quantized per token.
* Eq. 1 / Algorithm 1: loss = mean((x_fp - x_q')^2) of one transformer block, then
  the gradient of the loss w.r.t. Theta1 = {gamma_hat, beta_hat} and
  Theta2 = {s, delta, s_a}.

Readings where the paper is silent (each is listed with its reason in the design
notes of the repository):

 R1  dequantisation: W_hat = (W_q - z) * h.
 R2  round = half to even.
 R3  h is floored at eps (1e-5); a floored h has zero gradient.
 R4  min/max are taken literally (not forced to straddle 0); z is not clamped.
 R5  gamma, beta are sigmoids of fp32 logits (default 4.0).
 R6  groups are contiguous runs of `group` input channels of one output channel;
     group 0 means one group per output channel.
 R7  backward = straight-through estimator: every round() has derivative 1;
     clamp passes the gradient for 0 <= c <= 2^N-1 (inclusive); max and min pass
     their gradient to the first index that attains them; h is not detached.
 R8  Q, K, V are quantized per token over the full projected width.
 R9  s_a is applied after RoPE; with grouped KV heads it is broadcast to the
     query heads of each group, and so are s_o, delta_o of the [v, out] pair.
 R10 the attention scores are scaled by 1/sqrt(head_dim).
 R11 the block loss is the mean over all T*d elements of the squared error.
 R12 at W-A settings the inputs of all seven linears and Q~, K~, V' are
     quantized; the softmax output stays unquantized (Sec. 4.1).
 R13 precision policy ("emulate" mode): each operand of every matrix product,
     forward and backward, is rounded to bf16 (nearest, ties to even) right
     before the product; accumulation is exact (fp64 here).  "exact" mode skips
     the rounding.  Nothing else is rounded: every quantizer decision (max/min and
     their first index, the floor of h, the zero point, every code) is taken in
     float64 on float64 values, as Eq. 2 states it, and the softmax enters P V
     normalised (Eq. 5).
 R14 LLaMA blocks have no linear biases (B = 0); the [v, out] LET pair moves
     its transform into v_proj: W_v' = diag(1/s_o) W_v diag(s1),
     b_v' = (W_v delta1 - delta_o) / s_o, and the out_proj input is P V'
     (Sec. 3.3, last paragraph).
 R16 LET initialisation (Sec. 4.1 "Training": scaling as in SmoothQuant, shifting as in
     Outlier Suppression+), statistics of the full-precision block over the calibration
     tokens: s = max(max|X|^alpha / max|W|^(1-alpha), 1e-5) per input channel (alpha 0.5,
     max|W| over every output row of the weights sharing the input), delta = the channel mean
     of X; [ln1, (q,k,v)] on the ln1 output, [ln2, (gate,up)] on the ln2 output; the [v, out]
     pair the same recipe on the attention output O and W_o, per value channel (maxima and
     mean taken over the query heads of its group); [Q, K]: s_a = sqrt(max|Q| / max|K|) per
     channel after RoPE (max over the group's query heads), no shift.
 R17 fold & pack (Algorithm 1, after training: transform with the learned parameters, then
     quantize): the scales and shifts of the [ln, linears] pairs are absorbed into the
     RMSNorm as a gain 1/s and a bias -delta/s (the block's RMSNorm has unit gain and no bias
     of its own), the linear biases B~ of Eq. 3 and the [v, out] pair's row scale stay in the
     quantized weights and biases (R14), s_a stays a per-channel scale of the Q / K cache
     (it sits after RoPE, R9, so it cannot be folded into the projection weights).  Weight
     codes are packed per output row as a little-endian bit stream: code i occupies bits
     [N i, N i + N) of the row.
 R18 optimizer (Sec. 4.1 "Training": AdamW, zero weight decay, lr 5e-3 for the LWC logits and
     1e-2 for the LET vectors): betas 0.9 / 0.999, eps 1e-8, bias-corrected moments, decoupled
     weight decay; one update after every calibration sample (batch size 1).  Algorithm 1's
     LET statistics (R16) are taken on the fp inputs of each block before they are advanced.
 R21 the zero point rounds u = beta*min/h with h unfloored written as
     Q*beta*min / (gamma*max - beta*min), and as Q*min / (max - min) when gamma = beta (the
     clipping strengths cancel): the same value without the intermediate rounding of h, so a
     quotient that is exactly a half (gamma = beta and max = -min give u = -Q/2) stays exact
     and rounds to even (R2).
 R20 softmax-output quantization (the ablation of Table A7, off by default): the causal softmax
     output is quantized per query row with the MinMax Q_a (gamma = beta = 1, the floor of h
     included) over the visible keys j <= t only; the masked entries stay 0.  Its backward is the
     STE of R7.
"""
from __future__ import annotations

import dataclasses
import math
from typing import Dict, Optional, Tuple

import torch

F64 = torch.float64

__all__ = [
    "rne", "to_bf16", "sigmoid", "quant_fwd", "quant_bwd", "quant_ste", "codes_from_scale",
    "lwc_fakequant_fwd", "lwc_fakequant_bwd", "act_quant_per_token", "act_quant_per_token_bwd",
    "let_apply", "block_loss", "qlinear_step", "BlockCfg", "block_forward", "block_step",
    "rmsnorm", "rope", "silu", "FrozenTape", "use_tape", "block_fp_forward",
    "THETA_NAMES_LWC", "THETA_NAMES_LET", "let_init", "pack_codes", "unpack_codes", "block_fold_pack",
    "folded_forward", "adamw_step", "calibrate_blocks", "softmax_quant",
    "stage_attn_in", "stage_attention", "stage_attn_out", "stage_ffn_in", "stage_ffn_out",
]


# ----------------------------------------------------------------------------------------------
# elementary maps
# ----------------------------------------------------------------------------------------------

def rne(v: torch.Tensor) -> torch.Tensor:
    """round(.) of Eq. 2, read as round half to even (R2)."""
    return torch.round(v)


def to_bf16(v: torch.Tensor) -> torch.Tensor:
    """Nearest bf16 value (ties to even), returned in float64 (R13).

    The value is first rounded to float32, the precision in which the CUDA path
    holds every intermediate before it rounds a matmul operand."""
    return v.to(torch.float32).to(torch.bfloat16).to(F64)


def sigmoid(t: torch.Tensor) -> torch.Tensor:
    """gamma = sigmoid(gamma_hat), footnote to Sec. 3.2."""
    return 1.0 / (1.0 + torch.exp(-t))


def _first_argmax(w: torch.Tensor) -> torch.Tensor:
    """Index of the first maximum along the last axis (R7)."""
    M = w.max(dim=-1, keepdim=True).values
    hit = (w == M).to(torch.int64)
    return hit.argmax(dim=-1)          # argmax of a 0/1 vector = first 1


def _first_argmin(w: torch.Tensor) -> torch.Tensor:
    m = w.min(dim=-1, keepdim=True).values
    hit = (w == m).to(torch.int64)
    return hit.argmax(dim=-1)


# ----------------------------------------------------------------------------------------------
# Eq. 2, explicit forward and STE backward of one quantizer over groups on the last axis
# ----------------------------------------------------------------------------------------------

def _zero_point_round(a, b, M, m, Q: float, floored, eps: float) -> torch.Tensor:
    """round(u) for the zero point z = -round(u), u = beta*min/h (Eq. 2), read as R21: with h
    unfloored, u = Q*beta*min / (gamma*max - beta*min), or Q*min / (max - min) when gamma = beta;
    with h floored, u = beta*min/eps."""
    with torch.no_grad():
        M, m = M.detach(), m.detach()
        a = torch.as_tensor(a, dtype=F64).detach().expand_as(M)
        b = torch.as_tensor(b, dtype=F64).detach().expand_as(M)
        den = a * M - b * m
        rng_ = M - m
        u_same = Q * m / torch.where(rng_ == 0, torch.ones_like(rng_), rng_)
        u_gen = Q * b * m / torch.where(den == 0, torch.ones_like(den), den)
        u = torch.where(torch.as_tensor(floored), b * m / eps, torch.where(a == b, u_same, u_gen))
        return rne(u)


def quant_fwd(w: torch.Tensor, a, b, nbits: int, eps: float = 1e-5) -> Dict[str, torch.Tensor]:
    """Eq. 2 over groups laid out on the last axis of `w` (shape [..., g]).

    a, b are the clipping strengths gamma, beta (tensors of shape [...] or floats; 1.0 gives
    MinMax, the special case stated after Eq. 2).  Every decision is taken in float64.
    Returns every intermediate."""
    w = w.to(F64)
    Q = float(2 ** nbits - 1)
    a = torch.as_tensor(a, dtype=F64)
    b = torch.as_tensor(b, dtype=F64)
    imax = _first_argmax(w)
    imin = _first_argmin(w)
    M = torch.gather(w, -1, imax[..., None])[..., 0]
    m = torch.gather(w, -1, imin[..., None])[..., 0]
    h_raw = (a * M - b * m) / Q
    floored = h_raw < eps                                  # R3
    h = torch.where(floored, torch.full_like(h_raw, eps), h_raw)
    u = b * m / h
    x = w / h[..., None]
    z = -_zero_point_round(a, b, M, m, Q, floored, eps)
    c = rne(x) + z[..., None]
    q = torch.clamp(c, 0.0, Q)
    what = (q - z[..., None]) * h[..., None]               # R1
    return dict(a=a, b=b, M=M, m=m, imax=imax, imin=imin, h=h, floored=floored, u=u, z=z,
                x=x, c=c, q=q, what=what, Q=torch.tensor(Q, dtype=F64))


def quant_bwd(st: Dict[str, torch.Tensor], g: torch.Tensor) -> Dict[str, torch.Tensor]:
    """Straight-through backward of `quant_fwd` (R7), given g = dL/d what.

    Per group: an element whose code c lies in [0, Q] passes g to w directly and
    contributes (round(x) - x) * g to dL/dh; a clipped element contributes
    (round(u) - u) * g (below) or (Q + round(u) - u) * g (above) to dL/dh and g to
    dL/d(beta*min).  With h = (a*M - b*m)/Q the totals reach a*M and b*m, then
    gamma_hat, beta_hat through the sigmoid, and M, m through their first index.
    Returns dw (same shape as w), dgamma_logit and dbeta_logit (= dL/da * a(1-a)),
    and dL/da, dL/db."""
    g = g.to(F64)
    Q = st["Q"]
    c, x, u = st["c"], st["x"], st["u"]
    a, b, M, m = st["a"], st["b"], st["M"], st["m"]
    inr = (c >= 0) & (c <= Q)
    below = c < 0
    ru = -st["z"] - u                                      # round(u) is -z
    dh_elem = torch.where(inr, rne(x) - x,
                          torch.where(below, ru[..., None], (Q + ru)[..., None]))
    G_h = (g * dh_elem).sum(-1)
    G_h = torch.where(st["floored"], torch.zeros_like(G_h), G_h)
    G_bm = (g * (~inr).to(F64)).sum(-1)
    G_aM = G_h / Q
    G_bm_tot = G_bm - G_h / Q
    dw = g * inr.to(F64)
    dw = dw.scatter_add(-1, st["imax"][..., None], (G_aM * a)[..., None])
    dw = dw.scatter_add(-1, st["imin"][..., None], (G_bm_tot * b)[..., None])
    da = G_aM * M
    db = G_bm_tot * m
    return dict(dw=dw, da=da, db=db, dgamma_logit=da * a * (1 - a), dbeta_logit=db * b * (1 - b),
                G_h=G_h, G_bm=G_bm)


def _ste_round(v: torch.Tensor) -> torch.Tensor:
    """round(v) in the forward, identity in the backward (R7)."""
    return v + (rne(v) - v).detach()


class FrozenTape:
    """Records, then replays, the non-smooth decisions of every `quant_ste` call.

    In "record" mode each call stores its argmax/argmin, its floor flag, the rounding
    offsets round(v) - v and its clamp branches.  In "replay" mode the same calls evaluate
    the frozen-offset surrogate: round(v) becomes v + (offset recorded at theta_0), clamp
    and max/min keep the recorded branches.  The surrogate is smooth near theta_0 and its
    derivative there is, by R7, the STE gradient; finite differences of it therefore test
    the backward."""

    def __init__(self):
        self.mode = "record"
        self.rec = []
        self.i = 0

    def replay(self):
        self.mode = "replay"
        self.i = 0
        return self


_TAPE: Optional[FrozenTape] = None


class use_tape:
    """Context manager that routes every `quant_ste` call through `tape`."""

    def __init__(self, tape: FrozenTape):
        self.tape = tape

    def __enter__(self):
        global _TAPE
        self.prev, _TAPE = _TAPE, self.tape
        return self.tape

    def __exit__(self, *exc):
        global _TAPE
        _TAPE = self.prev


def quant_ste(w: torch.Tensor, a, b, nbits: int, eps: float = 1e-5) -> torch.Tensor:
    """Eq. 2 fake quantization as an autograd graph whose gradient is the STE of R7.

    Groups on the last axis; a, b broadcast against w[..., 0] (tensors that may require
    grad, or floats for Q_a)."""
    Q = float(2 ** nbits - 1)
    tape = _TAPE
    if tape is not None and tape.mode == "replay":
        r = tape.rec[tape.i]
        tape.i += 1
        M = torch.gather(w, -1, r["imax"][..., None])[..., 0]
        m = torch.gather(w, -1, r["imin"][..., None])[..., 0]
        h_raw = (a * M - b * m) / Q
        h = torch.where(r["floored"], torch.full_like(h_raw, eps), h_raw)
        u = b * m / h
        z = -(u + r["ru"])
        c = w / h[..., None] + r["rx"] + z[..., None]
        q = torch.where(r["inr"], c, torch.where(r["below"], torch.zeros_like(c), torch.full_like(c, Q)))
        return (q - z[..., None]) * h[..., None]
    imax = _first_argmax(w.detach())
    imin = _first_argmin(w.detach())
    M = torch.gather(w, -1, imax[..., None])[..., 0]
    m = torch.gather(w, -1, imin[..., None])[..., 0]
    h_raw = (a * M - b * m) / Q
    h = torch.clamp(h_raw, min=eps)                        # R3: gradient 0 when floored
    u = b * m / h
    ru = _zero_point_round(a, b, M, m, Q, (h_raw < eps).detach(), eps) - u.detach()
    z = -(u + ru)                                          # round(u) forward (R21), identity backward
    c = _ste_round(w / h[..., None]) + z[..., None]
    q = torch.clamp(c, 0.0, Q)
    if tape is not None:
        with torch.no_grad():
            h_raw = (a * M - b * m) / Q
            u = b * m / h
            x = w / h[..., None]
            tape.rec.append(dict(imax=imax, imin=imin, floored=torch.as_tensor(h_raw < eps),
                                 ru=ru.detach(), rx=(rne(x) - x).detach(),
                                 inr=((c >= 0) & (c <= Q)).detach(), below=(c < 0).detach()))
    return (q - z[..., None]) * h[..., None]


def codes_from_scale(w: torch.Tensor, h: torch.Tensor, z: torch.Tensor, nbits: int,
                     tie_window: float = 1e-6) -> Tuple[torch.Tensor, torch.Tensor]:
    """Codes clamp(round(w/h) + z, 0, Q) for given per-group h, z (groups on the last
    axis), and a mask of the elements whose w/h lies within `tie_window` of a .5
    boundary (those are exempt from bit-exact comparison)."""
    w = w.to(F64)
    x = w / h.to(F64)[..., None]
    Q = 2 ** nbits - 1
    c = torch.clamp(rne(x) + z.to(F64)[..., None], 0, Q)
    frac = x - torch.floor(x)
    near = (frac - 0.5).abs() < tie_window
    return c.to(torch.int64), near


# ----------------------------------------------------------------------------------------------
# kernel-level operations (one per C-ABI entry point)
# ----------------------------------------------------------------------------------------------

def _groups(W: torch.Tensor, group: int) -> torch.Tensor:
    cout, cin = W.shape
    g = cin if group == 0 else group
    assert cin % g == 0
    return W.reshape(cout, cin // g, g)                    # R6


def lwc_fakequant_fwd(W, gamma_logit, beta_logit, nbits: int, group: int,
                      s: Optional[torch.Tensor] = None, eps: float = 1e-5,
                      row_scale: Optional[torch.Tensor] = None) -> Dict[str, torch.Tensor]:
    """LWC of Eq. 2 on W~ = s (.) W (Eq. 3) for W [Cout, Cin].

    row_scale (optional, [Cout]) multiplies each output row before quantization; it is how
    the [v, out] LET pair divides v_proj's rows by s_o (R14).  Returns h, z [Cout, ngroups],
    the first argmax/argmin inside each group (as column indices into Cin), integer codes,
    W_hat [Cout, Cin] and the quantizer input Wt."""
    W = W.to(F64)
    Wt = W if s is None else W * s.to(F64)[None, :]
    if row_scale is not None:
        Wt = Wt * row_scale.to(F64)[:, None]
    G = _groups(Wt, group)
    a = sigmoid(gamma_logit.to(F64))
    b = sigmoid(beta_logit.to(F64))
    st = quant_fwd(G, a, b, nbits, eps)
    gsz = G.shape[-1]
    base = torch.arange(G.shape[1], dtype=torch.int64)[None, :] * gsz
    return dict(st=st, Wt=Wt, h=st["h"], z=st["z"], argmax=st["imax"] + base, argmin=st["imin"] + base,
                codes=st["q"].reshape(Wt.shape).to(torch.int64), what=st["what"].reshape(Wt.shape))


def lwc_fakequant_bwd(fwd: Dict[str, torch.Tensor], W, dWhat, s: Optional[torch.Tensor] = None,
                      row_scale: Optional[torch.Tensor] = None) -> Dict[str, torch.Tensor]:
    """STE backward of `lwc_fakequant_fwd`: dgamma_logit, dbeta_logit [Cout, ngroups], dWt
    [Cout, Cin] (gradient w.r.t. the quantizer input), ds [Cin] = sum_o dWt_oi * W_oi * r_o
    (Eq. 3 with W~ = s (.) W) and d(row_scale) [Cout] when a row scale is present."""
    W = W.to(F64)
    st = fwd["st"]
    cout, cin = W.shape
    gb = quant_bwd(st, dWhat.to(F64).reshape(st["x"].shape))
    dWt = gb["dw"].reshape(cout, cin)
    out = dict(dgamma_logit=gb["dgamma_logit"], dbeta_logit=gb["dbeta_logit"], dWt=dWt)
    r = torch.ones(cout, dtype=F64) if row_scale is None else row_scale.to(F64)
    if s is not None:
        out["ds"] = (dWt * W * r[:, None]).sum(0)
    if row_scale is not None:
        sv = torch.ones(cin, dtype=F64) if s is None else s.to(F64)
        out["drow_scale"] = (dWt * W * sv[None, :]).sum(1)
    return out


def act_quant_per_token(X, nbits: int, s: Optional[torch.Tensor] = None,
                        delta: Optional[torch.Tensor] = None, eps: float = 1e-5) -> Dict[str, torch.Tensor]:
    """LET on activations (Eq. 3: X~ = (X - delta)/s) followed by Q_a, the per-token MinMax
    quantizer (gamma = beta = 1 in Eq. 2; one group per token row)."""
    Xt = X.to(F64)
    if delta is not None:
        Xt = Xt - delta.to(F64)[None, :]
    if s is not None:
        Xt = Xt / s.to(F64)[None, :]
    st = quant_fwd(Xt, 1.0, 1.0, nbits, eps)
    return dict(st=st, Xt=Xt, Xq=st["what"], codes=st["q"].to(torch.int64), h=st["h"], z=st["z"],
                argmax=st["imax"], argmin=st["imin"])


def act_quant_per_token_bwd(fwd: Dict[str, torch.Tensor], dXq, s: Optional[torch.Tensor] = None,
                            delta: Optional[torch.Tensor] = None) -> Dict[str, torch.Tensor]:
    """STE backward of `act_quant_per_token`: dX, and the LET column reductions
    ds_i = -sum_t dX~_ti X~_ti / s_i, ddelta_i = -sum_t dX~_ti / s_i (Eq. 3)."""
    gb = quant_bwd(fwd["st"], dXq)
    dXt = gb["dw"]
    out = dict(dXt=dXt)
    sv = torch.ones(dXt.shape[1], dtype=F64) if s is None else s.to(F64)
    out["dX"] = dXt / sv[None, :]
    if s is not None:
        out["ds"] = -(dXt * fwd["Xt"]).sum(0) / sv
    if delta is not None:
        out["ddelta"] = -dXt.sum(0) / sv
    return out


def let_apply(X, W, B, s, delta) -> Dict[str, torch.Tensor]:
    """Eq. 3 with W stored [Cout, Cin]: X~ = (X - delta)/s, W~ = W diag(s), B~ = B + W delta."""
    X, W = X.to(F64), W.to(F64)
    s, delta = s.to(F64), delta.to(F64)
    Bv = torch.zeros(W.shape[0], dtype=F64) if B is None else B.to(F64)
    return dict(Xt=(X - delta[None, :]) / s[None, :], Wt=W * s[None, :], Bt=Bv + W @ delta)


def block_loss(Yq, Yfp) -> Tuple[torch.Tensor, torch.Tensor]:
    """Eq. 1 / Algorithm 1 loss, read as the mean squared error (R11); returns (loss, dY)."""
    Yq, Yfp = Yq.to(F64), Yfp.to(F64)
    n = Yq.numel()
    diff = Yq - Yfp
    return (diff * diff).sum() / n, 2.0 * diff / n


# ----------------------------------------------------------------------------------------------
# matrix products with the precision policy of R13
# ----------------------------------------------------------------------------------------------

class _MatmulBF16(torch.autograd.Function):
    """C = bf16(A) @ bf16(B)^T with exact accumulation; the backward rounds the incoming
    gradient to bf16 and multiplies it with the rounded operands (R13).  The rounding is a
    forward perturbation only: the gradient reaches A and B unchanged by it."""

    @staticmethod
    def forward(ctx, A, B):
        Ab, Bb = to_bf16(A), to_bf16(B)
        ctx.save_for_backward(Ab, Bb)
        return Ab @ Bb.transpose(-1, -2)

    @staticmethod
    def backward(ctx, gC):
        Ab, Bb = ctx.saved_tensors
        gb = to_bf16(gC)
        return gb @ Bb, gb.transpose(-1, -2) @ Ab


def _mm(A, B, mode: str):
    """A @ B^T (batched over leading axes)."""
    if mode == "emulate":
        return _MatmulBF16.apply(A, B)
    return A @ B.transpose(-1, -2)


# ----------------------------------------------------------------------------------------------
# single quantized linear step (LWC only, optional LET): the single-linear workload
# ----------------------------------------------------------------------------------------------

def qlinear_step(X, W, B, gamma_logit, beta_logit, Yfp, wbits: int, group: int, abits: int = 16,
                 s=None, delta=None, mode: str = "emulate", eps: float = 1e-5) -> Dict[str, torch.Tensor]:
    """Forward Y = Q_a(X~) Q_w(W~)^T + B~ (Eq. 4), loss against Yfp (Eq. 1), and the STE
    gradients of the loss w.r.t. gamma_hat, beta_hat (and s, delta when LET is on)."""
    gl = gamma_logit.to(F64).clone().requires_grad_(True)
    bl = beta_logit.to(F64).clone().requires_grad_(True)
    leaves = [gl, bl]
    sv = dv = None
    if s is not None:
        sv = s.to(F64).clone().requires_grad_(True)
        dv = delta.to(F64).clone().requires_grad_(True)
        leaves += [sv, dv]
    X = X.to(F64)
    W = W.to(F64)
    Xt = X if sv is None else (X - dv) / sv
    Wt = W if sv is None else W * sv[None, :]
    Bt = (torch.zeros(W.shape[0], dtype=F64) if B is None else B.to(F64))
    if sv is not None:
        Bt = Bt + W @ dv
    Xh = Xt if abits >= 16 else quant_ste(Xt, 1.0, 1.0, abits, eps)
    cout, cin = W.shape
    gsz = cin if group == 0 else group
    Wh = quant_ste(Wt.reshape(cout, cin // gsz, gsz), sigmoid(gl), sigmoid(bl), wbits, eps).reshape(cout, cin)
    Y = _mm(Xh, Wh, mode) + Bt
    loss, _ = block_loss(Y, Yfp)
    grads = torch.autograd.grad(loss, leaves)
    out = dict(Y=Y.detach(), loss=loss.detach(), dgamma_logit=grads[0], dbeta_logit=grads[1])
    if sv is not None:
        out["ds"], out["ddelta"] = grads[2], grads[3]
    return out


# ----------------------------------------------------------------------------------------------
# decoder block (LLaMA layout: RMSNorm, RoPE causal attention, SwiGLU FFN)
# ----------------------------------------------------------------------------------------------

@dataclasses.dataclass
class BlockCfg:
    d: int
    n_heads: int
    n_kv: int
    ffn: int
    wbits: int            # 16 = weights not quantized
    abits: int            # 16 = activations not quantized
    group: int            # 0 = per output channel
    let: bool
    head_dim: int = 128
    rms_eps: float = 1e-6
    rope_theta: float = 10000.0
    h_eps: float = 1e-5
    mode: str = "emulate"
    pbits: int = 16       # softmax-output bits (R20); 16 = kept at full precision (the default)

    @staticmethod
    def from_shape(shape, **kw) -> "BlockCfg":
        base = dict(d=shape.d, n_heads=shape.n_heads, n_kv=shape.n_kv, ffn=shape.ffn,
                    wbits=shape.wbits, abits=shape.abits, group=shape.group, let=bool(shape.let),
                    head_dim=shape.head_dim, rms_eps=shape.rms_eps, rope_theta=shape.rope_theta)
        base.update(kw)
        return BlockCfg(**base)


def rmsnorm(x, eps):
    """RMSNorm with unit gain: x / sqrt(mean(x^2) + eps) per token."""
    return x / torch.sqrt((x * x).mean(-1, keepdim=True) + eps)


def silu(v):
    return v * sigmoid(v)


def rope(v, n_heads: int, head_dim: int, theta: float):
    """Rotary position embedding, rotate-half pairing (i, i + head_dim/2) in each head,
    position = token index, frequency theta^(-2j/head_dim)."""
    T = v.shape[0]
    half = head_dim // 2
    j = torch.arange(half, dtype=F64)
    inv_freq = 1.0 / (theta ** (2.0 * j / head_dim))
    ang = torch.arange(T, dtype=F64)[:, None] * inv_freq[None, :]
    cos, sin = torch.cos(ang)[:, None, :], torch.sin(ang)[:, None, :]
    vh = v.reshape(T, n_heads, head_dim)
    v1, v2 = vh[..., :half], vh[..., half:]
    return torch.cat([v1 * cos - v2 * sin, v2 * cos + v1 * sin], dim=-1).reshape(T, n_heads * head_dim)


def _expand_kv(vec, cfg: BlockCfg):
    """Broadcast a per-KV-channel vector [n_kv*hd] to the query heads [n_heads*hd] (R9)."""
    rep = cfg.n_heads // cfg.n_kv
    return vec.reshape(cfg.n_kv, 1, cfg.head_dim).expand(cfg.n_kv, rep, cfg.head_dim).reshape(-1)


def _qw(Wt, gl, bl, cfg: BlockCfg):
    """LWC fake quantization (Eq. 2) of a (LET-scaled) weight [Cout, Cin]."""
    if cfg.wbits >= 16:
        return Wt
    cout, cin = Wt.shape
    gsz = cin if cfg.group == 0 else cfg.group
    return quant_ste(Wt.reshape(cout, cin // gsz, gsz), sigmoid(gl), sigmoid(bl),
                     cfg.wbits, cfg.h_eps).reshape(cout, cin)


def _qa(X, cfg: BlockCfg):
    """Q_a, the per-token MinMax quantizer (R8, R12)."""
    if cfg.abits >= 16:
        return X
    return quant_ste(X, 1.0, 1.0, cfg.abits, cfg.h_eps)


def softmax_quant(P, nbits: int, eps: float = 1e-5):
    """Q_p (R20): the causal softmax output P [..., T, T] quantized per query row with the
    MinMax quantizer of Eq. 2 (gamma = beta = 1) over the row's visible keys j <= t, as an
    autograd graph with the STE of R7 (h not detached; max / min pass their gradient to the first
    index).  The masked entries stay exactly 0 and take no part in the row's range.  nbits >= 16
    returns P."""
    if nbits >= 16:
        return P
    T = P.shape[-1]
    causal = torch.ones(T, T, dtype=torch.bool).tril()
    # the masked entries are filled with the row's diagonal probability: a value inside the row's
    # range at an index after every visible key, so max, min and their first indices are unchanged
    diag = torch.diagonal(P, dim1=-2, dim2=-1)[..., :, None]
    Pf = torch.where(causal, P, diag.detach().expand_as(P))
    return quant_ste(Pf, 1.0, 1.0, nbits, eps).masked_fill(~causal, 0.0)


def _attn_pv(S, Vh, cfg: BlockCfg):
    """The attention output from the masked scores: softmax(S) (Eq. 5; quantized per query row
    when the ablation of R20 is on) times V, both operands rounded to bf16 in emulate mode (R13)."""
    P = torch.softmax(S, dim=-1)
    if cfg.pbits < 16:
        P = softmax_quant(P, cfg.pbits, cfg.h_eps)
    return _mm(P, Vh.transpose(-1, -2), cfg.mode)


# The block forward in five stages; each stage takes its inputs as tensors, so a test can start
# any stage from another implementation's values of its input (stage-wise comparison).

def stage_attn_in(x, Wd: Dict[str, torch.Tensor], th: Dict[str, torch.Tensor], cfg: BlockCfg):
    """RMSNorm, the [ln1, (q, k, v)] LET pair (Eq. 3) with the [v, out] pair moved into v_proj
    (R14), Q_a and the three quantized projections (Eq. 4): q, k, v before RoPE, LET biases
    included."""
    mode = cfg.mode
    wq, wk, wv = Wd["wq"], Wd["wk"], Wd["wv"]
    a = rmsnorm(x, cfg.rms_eps)
    if cfg.let:
        s1, d1, so, do_ = th["s1"], th["d1"], th["so"], th["do"]
        at = (a - d1) / s1
        wq_t, wk_t = wq * s1, wk * s1
        wv_t = (wv * s1) / so[:, None]
        bq, bk = wq @ d1, wk @ d1
        bv = (wv @ d1 - do_) / so
    else:
        at, wq_t, wk_t, wv_t = a, wq, wk, wv
    ah = _qa(at, cfg)
    q = _mm(ah, _qw(wq_t, th.get("gamma_q"), th.get("beta_q"), cfg), mode)
    k = _mm(ah, _qw(wk_t, th.get("gamma_k"), th.get("beta_k"), cfg), mode)
    v = _mm(ah, _qw(wv_t, th.get("gamma_v"), th.get("beta_v"), cfg), mode)
    if cfg.let:
        q, k, v = q + bq, k + bk, v + bv
    return q, k, v, a


def stage_attention(q, k, v, th: Dict[str, torch.Tensor], cfg: BlockCfg):
    """RoPE, the [Q, K] LET pair after RoPE (Eq. 5, R9), Q_a of Q~, K~, V' (R8, R12) and causal
    attention with scores scaled by 1/sqrt(head_dim) (R10).  Returns O [T, H * hd] and the
    post-RoPE q, k."""
    H, Hkv, hd = cfg.n_heads, cfg.n_kv, cfg.head_dim
    T = q.shape[0]
    q = rope(q, H, hd, cfg.rope_theta)
    k = rope(k, Hkv, hd, cfg.rope_theta)
    if cfg.let:
        sa = th["sa"]
        q = q / _expand_kv(sa, cfg)
        k = k * sa
    qh, kh, vh = _qa(q, cfg), _qa(k, cfg), _qa(v, cfg)
    rep = H // Hkv
    Qh = qh.reshape(T, H, hd).transpose(0, 1)                            # [H, T, hd]
    Kh = kh.reshape(T, Hkv, hd).transpose(0, 1).repeat_interleave(rep, 0)
    Vh = vh.reshape(T, Hkv, hd).transpose(0, 1).repeat_interleave(rep, 0)
    S = _mm(Qh, Kh, cfg.mode) / math.sqrt(hd)
    causal = torch.ones(T, T, dtype=torch.bool).tril()
    S = S.masked_fill(~causal, float("-inf"))
    O = _attn_pv(S, Vh, cfg).transpose(0, 1).reshape(T, H * hd)
    return O, q, k


def stage_attn_out(O, x, Wd: Dict[str, torch.Tensor], th: Dict[str, torch.Tensor], cfg: BlockCfg):
    """Q_a of the attention output and the quantized o_proj with the [v, out] pair's column scale
    and bias (Eq. 3, Eq. 4, R14), plus the residual: h1 = x + o."""
    wo = Wd["wo"]
    oh = _qa(O, cfg)
    if cfg.let:
        wo_t = wo * _expand_kv(th["so"], cfg)[None, :]
        bo = wo @ _expand_kv(th["do"], cfg)
    else:
        wo_t, bo = wo, None
    o = _mm(oh, _qw(wo_t, th.get("gamma_o"), th.get("beta_o"), cfg), cfg.mode)
    if bo is not None:
        o = o + bo
    return x + o


def stage_ffn_in(h1, Wd: Dict[str, torch.Tensor], th: Dict[str, torch.Tensor], cfg: BlockCfg):
    """RMSNorm, the [ln2, (gate, up)] LET pair, Q_a and the quantized gate and up projections."""
    mode = cfg.mode
    wg, wu = Wd["wg"], Wd["wu"]
    b_ = rmsnorm(h1, cfg.rms_eps)
    if cfg.let:
        s2, d2 = th["s2"], th["d2"]
        bt = (b_ - d2) / s2
        wg_t, wu_t = wg * s2, wu * s2
        bg, bu = wg @ d2, wu @ d2
    else:
        bt, wg_t, wu_t, bg, bu = b_, wg, wu, None, None
    bh = _qa(bt, cfg)
    gt = _mm(bh, _qw(wg_t, th.get("gamma_g"), th.get("beta_g"), cfg), mode)
    up = _mm(bh, _qw(wu_t, th.get("gamma_u"), th.get("beta_u"), cfg), mode)
    if cfg.let:
        gt, up = gt + bg, up + bu
    return gt, up


def stage_ffn_out(gt, up, h1, Wd: Dict[str, torch.Tensor], th: Dict[str, torch.Tensor], cfg: BlockCfg):
    """SwiGLU, Q_a, the quantized down_proj (no LET on its input, Sec. 3.3) and the residual."""
    m = silu(gt) * up
    mh = _qa(m, cfg)
    return h1 + _mm(mh, _qw(Wd["wd"], th.get("gamma_d"), th.get("beta_d"), cfg), cfg.mode), m


def block_forward(x, Wd: Dict[str, torch.Tensor], th: Dict[str, torch.Tensor], cfg: BlockCfg,
                  keep: Optional[Dict[str, torch.Tensor]] = None):
    """Forward of the LET'd, LWC-quantized block (Algorithm 1, LET then
    Quantization_with_LWC then the block on x_q), the five stages in order.  `th` holds the
    learnable parameters (gamma_*/beta_* logits per linear; s1, d1, so, do, sa, s2, d2 when LET
    is on).  With wbits = abits = 16 and LET off this is the full-precision block F(W, X)."""
    q0, k0, v, a = stage_attn_in(x, Wd, th, cfg)
    O, q, k = stage_attention(q0, k0, v, th, cfg)
    h1 = stage_attn_out(O, x, Wd, th, cfg)
    gt, up = stage_ffn_in(h1, Wd, th, cfg)
    y, m = stage_ffn_out(gt, up, h1, Wd, th, cfg)
    if keep is not None:
        keep.update(dict(a=a, q=q, k=k, v=v, O=O, h1=h1, gate=gt, up=up, m=m))
    return y


THETA_NAMES_LWC = ["gamma_q", "beta_q", "gamma_k", "beta_k", "gamma_v", "beta_v", "gamma_o", "beta_o",
                   "gamma_g", "beta_g", "gamma_u", "beta_u", "gamma_d", "beta_d"]
THETA_NAMES_LET = ["s1", "d1", "so", "do", "sa", "s2", "d2"]


def block_step(x, y_fp, weights: Dict[str, object], theta: Dict[str, object], cfg: BlockCfg,
               keep: Optional[Dict[str, torch.Tensor]] = None) -> Dict[str, torch.Tensor]:
    """One step of Algorithm 1's inner loop without the parameter update: forward of the
    quantized block on x, loss against y_fp, and the STE gradient of the loss w.r.t. every
    learnable parameter.  Returns y, loss and d<name> for each parameter."""
    t = lambda v: torch.as_tensor(v).to(F64)
    Wd = {k: t(v) for k, v in weights.items()}
    names = (THETA_NAMES_LWC if cfg.wbits < 16 else []) + (THETA_NAMES_LET if cfg.let else [])
    th = {k: t(theta[k]).clone().requires_grad_(True) for k in names}
    y = block_forward(t(x), Wd, th, cfg, keep)
    loss, _ = block_loss(y, t(y_fp))
    out = dict(y=y.detach(), loss=loss.detach())
    if names:
        grads = torch.autograd.grad(loss, [th[k] for k in names])
        for k, gk in zip(names, grads):
            out["d" + k] = gk
    return out


def block_fp_forward(x, weights: Dict[str, object], cfg: BlockCfg) -> torch.Tensor:
    """Full-precision block F(W, X) in fp64 (Eq. 1 target; Algorithm 1 updates X_fp with it)."""
    fp = dataclasses.replace(cfg, wbits=16, abits=16, let=False, mode="exact")
    t = lambda v: torch.as_tensor(v).to(F64)
    with torch.no_grad():
        return block_forward(t(x), {k: t(v) for k, v in weights.items()}, {}, fp)


# ----------------------------------------------------------------------------------------------
# LET initialisation (R16)
# ----------------------------------------------------------------------------------------------

def let_init(xs, weights: Dict[str, object], cfg: BlockCfg, alpha: float = 0.5, floor: float = 1e-5):
    """Initial LET parameters s1, d1, so, do, sa, s2, d2 from the calibration inputs `xs` (a list
    of [T, d] block inputs) through the full-precision block (reading R16)."""
    fp = dataclasses.replace(cfg, wbits=16, abits=16, let=False, mode="exact")
    t = lambda v: torch.as_tensor(v).to(F64)
    Wd = {k: t(v) for k, v in weights.items()}
    H, Hkv, hd = cfg.n_heads, cfg.n_kv, cfg.head_dim
    rep = H // Hkv
    amax = {}
    sums = {}
    n = 0
    with torch.no_grad():
        for x in xs:
            keep: Dict[str, torch.Tensor] = {}
            block_forward(t(x), Wd, {}, fp, keep)
            stats = dict(a=keep["a"], q=keep["q"], k=keep["k"], O=keep["O"], b=rmsnorm(keep["h1"], cfg.rms_eps))
            for key, v in stats.items():
                m = v.abs().max(0).values
                amax[key] = m if key not in amax else torch.maximum(amax[key], m)
                sm = v.sum(0)
                sums[key] = sm if key not in sums else sums[key] + sm
            n += x.shape[0]

    def smooth(xmax, wmax):
        return torch.clamp(xmax ** alpha / wmax ** (1.0 - alpha), min=floor)

    def per_kv(v, op):                    # [H*hd] -> [Hkv*hd] over the query heads of each group
        g = v.reshape(Hkv, rep, hd)
        return (g.max(1).values if op == "max" else g.mean(1)).reshape(Hkv * hd)

    wmax_qkv = torch.cat([Wd["wq"], Wd["wk"], Wd["wv"]]).abs().max(0).values
    wmax_gu = torch.cat([Wd["wg"], Wd["wu"]]).abs().max(0).values
    wmax_o = per_kv(Wd["wo"].abs().max(0).values, "max")
    out = dict(
        s1=smooth(amax["a"], wmax_qkv), d1=sums["a"] / n,
        s2=smooth(amax["b"], wmax_gu), d2=sums["b"] / n,
        so=smooth(per_kv(amax["O"], "max"), wmax_o), do=per_kv(sums["O"] / n, "mean"),
        sa=torch.clamp(torch.sqrt(per_kv(amax["q"], "max") / amax["k"]), min=floor),
    )
    return out


# ----------------------------------------------------------------------------------------------
# fold & pack (R17)
# ----------------------------------------------------------------------------------------------

def pack_codes(codes: torch.Tensor, nbits: int) -> torch.Tensor:
    """Integer codes [Cout, Cin] (0 <= c < 2^nbits) -> uint8 [Cout, Cin * nbits / 8]: code i of a
    row at bits [nbits i, nbits i + nbits) of the row's little-endian bit stream."""
    cout, cin = codes.shape
    assert (cin * nbits) % 8 == 0
    bits = ((codes.to(torch.int64)[..., None] >> torch.arange(nbits)) & 1).reshape(cout, cin * nbits)
    bytes_ = bits.reshape(cout, -1, 8)
    return (bytes_ << torch.arange(8)).sum(-1).to(torch.uint8)


def unpack_codes(packed: torch.Tensor, nbits: int, cin: int) -> torch.Tensor:
    cout = packed.shape[0]
    bits = ((packed.to(torch.int64)[..., None] >> torch.arange(8)) & 1).reshape(cout, -1)[:, :cin * nbits]
    return (bits.reshape(cout, cin, nbits) << torch.arange(nbits)).sum(-1)


def block_fold_pack(weights: Dict[str, object], theta: Dict[str, object], cfg: BlockCfg) -> Dict[str, torch.Tensor]:
    """The block after calibration, with its learned parameters folded in and its weights
    quantized (Algorithm 1, last steps; reading R17): per linear (q|k|v stacked, o, gate|up,
    down) packed codes, h and z per group; biases of q|k|v, o, gate|up; the two RMSNorm gains
    and biases; s_a."""
    t = lambda v: torch.as_tensor(v).to(F64)
    Wd = {k: t(v) for k, v in weights.items()}
    th = {k: t(v) for k, v in theta.items()}
    H, Hkv, hd = cfg.n_heads, cfg.n_kv, cfg.head_dim
    out: Dict[str, torch.Tensor] = {}
    let = cfg.let
    with torch.no_grad():
        if let:
            s1, d1, so, do_, s2, d2 = th["s1"], th["d1"], th["so"], th["do"], th["s2"], th["d2"]
            r_o = 1.0 / so
            rows = torch.cat([torch.ones(H * hd + Hkv * hd, dtype=F64), r_o])
            so_e, do_e = _expand_kv(so, cfg), _expand_kv(do_, cfg)
        lin = dict(
            qkv=(torch.cat([Wd["wq"], Wd["wk"], Wd["wv"]]), ("q", "k", "v"), s1 if let else None, rows if let else None),
            o=(Wd["wo"], ("o",), so_e if let else None, None),
            gu=(torch.cat([Wd["wg"], Wd["wu"]]), ("g", "u"), s2 if let else None, None),
            d=(Wd["wd"], ("d",), None, None))
        for name, (Wl, parts, s, r) in lin.items():
            gl = torch.cat([th["gamma_" + p_] for p_ in parts])
            bl = torch.cat([th["beta_" + p_] for p_ in parts])
            f = lwc_fakequant_fwd(Wl, gl, bl, cfg.wbits, cfg.group, s=s, eps=cfg.h_eps, row_scale=r)
            out["codes_" + name] = pack_codes(f["codes"], cfg.wbits)
            out["h_" + name] = f["h"]
            out["z_" + name] = f["z"]
        if let:
            wv_b = (Wd["wv"] @ d1 - do_) / so
            out["b_qkv"] = torch.cat([Wd["wq"] @ d1, Wd["wk"] @ d1, wv_b])
            out["b_o"] = Wd["wo"] @ do_e
            out["b_gu"] = torch.cat([Wd["wg"], Wd["wu"]]) @ d2
            out["ln1_gain"], out["ln1_bias"] = 1.0 / s1, -d1 / s1
            out["ln2_gain"], out["ln2_bias"] = 1.0 / s2, -d2 / s2
            out["sa"] = th["sa"]
    return out


def folded_forward(folded: Dict[str, torch.Tensor], x, cfg: BlockCfg) -> torch.Tensor:
    """The deployed block built only from block_fold_pack's output: dequantized weights
    (code - z) h, folded RMSNorm gains and biases, biases, s_a on Q / K; activations quantized
    per token as in the calibrated block."""
    H, Hkv, hd = cfg.n_heads, cfg.n_kv, cfg.head_dim
    mode = cfg.mode
    T = x.shape[0]
    let = cfg.let

    def deq(name, cout, cin):
        c = unpack_codes(folded["codes_" + name], cfg.wbits, cin).to(F64)
        g = cin if cfg.group == 0 else cfg.group
        h = folded["h_" + name].to(F64).repeat_interleave(g, 1)
        z = folded["z_" + name].to(F64).repeat_interleave(g, 1)
        return (c - z) * h

    d, f = cfg.d, cfg.ffn
    dq, dkv = H * hd, Hkv * hd
    x = torch.as_tensor(x).to(F64)
    with torch.no_grad():
        a = rmsnorm(x, cfg.rms_eps)
        if let:
            a = a * folded["ln1_gain"] + folded["ln1_bias"]
        y = _mm(_qa(a, cfg), deq("qkv", dq + 2 * dkv, d), mode)
        if let:
            y = y + folded["b_qkv"]
        q, k, v = y[:, :dq], y[:, dq:dq + dkv], y[:, dq + dkv:]
        q = rope(q, H, hd, cfg.rope_theta)
        k = rope(k, Hkv, hd, cfg.rope_theta)
        if let:
            q = q / _expand_kv(folded["sa"], cfg)
            k = k * folded["sa"]
        qh, kh, vh = _qa(q, cfg), _qa(k, cfg), _qa(v, cfg)
        rep = H // Hkv
        Qh = qh.reshape(T, H, hd).transpose(0, 1)
        Kh = kh.reshape(T, Hkv, hd).transpose(0, 1).repeat_interleave(rep, 0)
        Vh = vh.reshape(T, Hkv, hd).transpose(0, 1).repeat_interleave(rep, 0)
        S = _mm(Qh, Kh, mode) / math.sqrt(hd)
        S = S.masked_fill(~torch.ones(T, T, dtype=torch.bool).tril(), float("-inf"))
        O = _attn_pv(S, Vh, cfg).transpose(0, 1).reshape(T, dq)
        o = _mm(_qa(O, cfg), deq("o", d, dq), mode)
        if let:
            o = o + folded["b_o"]
        h1 = x + o
        b = rmsnorm(h1, cfg.rms_eps)
        if let:
            b = b * folded["ln2_gain"] + folded["ln2_bias"]
        gu = _mm(_qa(b, cfg), deq("gu", 2 * f, d), mode)
        if let:
            gu = gu + folded["b_gu"]
        m = silu(gu[:, :f]) * gu[:, f:]
        return h1 + _mm(_qa(m, cfg), deq("d", d, f), mode)


# ----------------------------------------------------------------------------------------------
# Algorithm 1: block-wise calibration (R18)
# ----------------------------------------------------------------------------------------------

def adamw_step(p, g, m, v, lr: float, t: int, b1: float = 0.9, b2: float = 0.999, eps: float = 1e-8,
               wd: float = 0.0):
    """One AdamW update (in place) of parameter p with gradient g and moments m, v; t >= 1."""
    m.mul_(b1).add_((1 - b1) * g)
    v.mul_(b2).add_((1 - b2) * g * g)
    mh = m / (1 - b1 ** t)
    vh = v / (1 - b2 ** t)
    p.sub_(lr * mh / (torch.sqrt(vh) + eps) + lr * wd * p)


def calibrate_blocks(blocks, xs, cfg: BlockCfg, theta0, epochs: int = 1, lr_lwc: float = 5e-3,
                     lr_let: float = 1e-2, let_init_alpha: Optional[float] = 0.5):
    """Algorithm 1 over a stack of blocks: X_fp = X_q = X; per block: X_fp <- B(X_fp), initialise
    Theta1 (theta0's LWC logits) and Theta2 (let_init on the block's fp inputs, R16), train on the
    (x_q, x_fp) pairs for `epochs` epochs with AdamW (R18), then X_q <- the quantized block(X_q).
    Returns the per-block parameters and the final X_fp, X_q."""
    t = lambda v: torch.as_tensor(v).to(F64)
    x_fp = [t(x) for x in xs]
    x_q = [t(x) for x in xs]
    names = (THETA_NAMES_LWC if cfg.wbits < 16 else []) + (THETA_NAMES_LET if cfg.let else [])
    out = []
    for W in blocks:
        th = {k: t(theta0[k]).clone() for k in names}
        if cfg.let and let_init_alpha is not None:
            th.update(let_init(x_fp, W, cfg, alpha=let_init_alpha))
        y_fp = [block_fp_forward(x, W, cfg) for x in x_fp]
        mom = {k: (torch.zeros_like(v), torch.zeros_like(v)) for k, v in th.items()}
        step = 0
        for _ in range(epochs):
            for xq, yf in zip(x_q, y_fp):
                r = block_step(xq, yf, W, th, cfg)
                step += 1
                for k in names:
                    lr = lr_let if k in THETA_NAMES_LET else lr_lwc
                    adamw_step(th[k], r["d" + k], mom[k][0], mom[k][1], lr, step)
        with torch.no_grad():
            Wd = {k: t(v) for k, v in W.items()}
            x_q = [block_forward(xq, Wd, th, cfg) for xq in x_q]
        x_fp = y_fp
        out.append({k: v.clone() for k, v in th.items()})
    return out, x_fp, x_q
