"""Pins of the fp64 oracle against facts fixed by the paper and by mathematics.

Each test ties one oracle function to something other than itself: hand-evaluated
values of Eq. 2, the MinMax special case stated after Eq. 2, brute-force code
enumeration, the exact equivalence of Eq. 3 / Eq. 5 with quantization off,
finite differences of the frozen-offset surrogate (the STE gradient of R7), and a
naive loop implementation of causal attention.
"""
import json
import math
import os

import numpy as np
import pytest
import torch

import oracle as O
from paper_2308_13137_gb300 import inputs as I

F64 = torch.float64
GOLD = os.path.join(os.path.dirname(__file__), "golden")


def _rel(a, b):
    a, b = torch.as_tensor(a, dtype=F64), torch.as_tensor(b, dtype=F64)
    return float((a - b).norm() / max(float(b.norm()), 1e-300))


# ------------------------------------------------------------------------------------------------
# elementary maps
# ------------------------------------------------------------------------------------------------

def test_rne_ties_to_even():
    v = torch.tensor([0.5, 1.5, 2.5, -0.5, -1.5, -2.5, 0.49999999, 2.5000001], dtype=F64)
    assert O.rne(v).tolist() == [0.0, 2.0, 2.0, -0.0, -2.0, -2.0, 0.0, 3.0]


def test_to_bf16_is_nearest_even_bf16():
    rng = np.random.default_rng(5)
    vals = np.concatenate([rng.standard_normal(2000) * 10.0 ** rng.integers(-6, 6, 2000),
                           [1.0 + 2 ** -8, 1.0 + 3 * 2 ** -8, -(1.0 + 2 ** -8)]])
    out = O.to_bf16(torch.tensor(vals, dtype=F64)).numpy()
    for v, o in zip(vals, out):
        f = np.float32(v)
        e = math.frexp(float(f))[1]                # f = mant * 2^e, mant in [0.5, 1)
        ulp = 2.0 ** (e - 8)                       # bf16 keeps 8 significant bits
        lo = math.floor(float(f) / ulp) * ulp
        cands = [lo, lo + ulp]
        d = [abs(c - float(f)) for c in cands]
        if d[0] == d[1]:                           # tie: even significand
            best = cands[0] if int(round(cands[0] / ulp)) % 2 == 0 else cands[1]
        else:
            best = cands[int(np.argmin(d))]
        assert o == best, (v, o, best)


# ------------------------------------------------------------------------------------------------
# Eq. 2
# ------------------------------------------------------------------------------------------------

def test_lwc_hand_examples():
    with open(os.path.join(GOLD, "lwc_hand_examples.json")) as fh:
        cases = json.load(fh)["cases"]
    for cs in cases:
        w = torch.tensor(cs["w"], dtype=F64)[None, :]
        st = O.quant_fwd(w, cs["a"], cs["b"], cs["nbits"])
        assert abs(float(st["h"][0]) - cs["h"]) < 1e-12, cs["comment"]
        assert int(st["z"][0]) == cs["z"], cs["comment"]
        assert st["q"][0].tolist() == cs["codes"], cs["comment"]
        assert torch.allclose(st["what"][0] / st["h"][0], torch.tensor(cs["what_over_h"], dtype=F64))


def _textbook_minmax(w, nbits):
    """Asymmetric min-max round-to-nearest, written independently: scale = range / (2^N-1),
    zero point = round(-min/scale), value = (clamp(round(w/scale)+zp) - zp) * scale."""
    qmax = 2 ** nbits - 1
    lo, hi = w.min(-1, keepdim=True).values, w.max(-1, keepdim=True).values
    scale = (hi - lo) / qmax
    zp = torch.round(-lo / scale)
    code = torch.clamp(torch.round(w / scale) + zp, 0, qmax)
    return code, (code - zp) * scale


@pytest.mark.parametrize("nbits", [2, 3, 4, 8])
def test_lwc_reduces_to_minmax(nbits):
    g = torch.Generator().manual_seed(nbits)
    w = torch.randn(64, 128, generator=g, dtype=F64) * 0.02
    big = torch.full((64, 1), 40.0, dtype=F64)     # sigmoid(40) == 1.0 in float64
    f = O.lwc_fakequant_fwd(w, big, big, nbits, group=0)
    code, val = _textbook_minmax(w, nbits)
    assert torch.equal(f["codes"], code.to(torch.int64))
    assert torch.allclose(f["what"], val, rtol=0, atol=1e-15)


@pytest.mark.parametrize("nbits", [2, 3, 4])
def test_codes_are_nearest_level_bruteforce(nbits):
    g = torch.Generator().manual_seed(10 + nbits)
    w = torch.randn(16, 64, generator=g, dtype=F64) * 0.05
    gl = torch.randn(16, 4, generator=g, dtype=F64) + 1.0
    bl = torch.randn(16, 4, generator=g, dtype=F64) + 1.0
    f = O.lwc_fakequant_fwd(w, gl, bl, nbits, group=16)
    h = f["h"].reshape(16, 4, 1)
    z = f["z"].reshape(16, 4, 1)
    wg = w.reshape(16, 4, 16)
    levels = torch.arange(2 ** nbits, dtype=F64)
    dist = (wg[..., None] - (levels - z[..., None]) * h[..., None]).abs()      # [16,4,16,L]
    best = dist.argmin(-1)
    srt = dist.sort(-1).values
    ambiguous = (srt[..., 1] - srt[..., 0]) < 1e-12 * h[..., 0:1].expand_as(srt[..., 0])
    codes = f["codes"].reshape(16, 4, 16)
    assert torch.equal(codes[~ambiguous], best[~ambiguous])


def test_group_layout_matches_loop():
    g = torch.Generator().manual_seed(3)
    w = torch.randn(6, 48, generator=g, dtype=F64)
    gl = torch.randn(6, 3, generator=g, dtype=F64)
    bl = torch.randn(6, 3, generator=g, dtype=F64)
    f = O.lwc_fakequant_fwd(w, gl, bl, 3, group=16)
    for o in range(6):
        for j in range(3):
            seg = w[o, 16 * j:16 * (j + 1)][None]
            st = O.quant_fwd(seg, O.sigmoid(gl[o, j]), O.sigmoid(bl[o, j]), 3)
            assert torch.equal(f["what"][o, 16 * j:16 * (j + 1)], st["what"][0])
            assert int(f["argmax"][o, j]) == 16 * j + int(st["imax"][0])


def test_fakequant_idempotent_with_fixed_scale():
    g = torch.Generator().manual_seed(4)
    w = torch.randn(32, 64, generator=g, dtype=F64) * 0.02
    gl = torch.randn(32, 1, generator=g, dtype=F64) + 2
    bl = torch.randn(32, 1, generator=g, dtype=F64) + 2
    f = O.lwc_fakequant_fwd(w, gl, bl, 4, group=0)
    c2, _ = O.codes_from_scale(f["what"].reshape(32, 1, 64), f["h"], f["z"], 4)
    assert torch.equal(c2.reshape(32, 64), f["codes"])
    w2 = (c2.to(F64) - f["z"][..., None]) * f["h"][..., None]
    assert torch.allclose(w2.reshape(32, 64), f["what"], rtol=0, atol=1e-15)


def test_first_index_on_ties():
    w = torch.tensor([[0.3, -0.2, 0.3, -0.2, 0.1]], dtype=F64)
    st = O.quant_fwd(w, 1.0, 1.0, 4)
    assert int(st["imax"][0]) == 0 and int(st["imin"][0]) == 1


def test_h_floor():
    w = torch.full((1, 8), 0.25, dtype=F64)        # constant group: range 0
    st = O.quant_fwd(w, 1.0, 1.0, 4, eps=1e-5)
    assert bool(st["floored"][0]) and float(st["h"][0]) == 1e-5


# ------------------------------------------------------------------------------------------------
# STE backward: explicit formulas == autograd of the STE graph == finite differences of the
# frozen-offset surrogate
# ------------------------------------------------------------------------------------------------

def _surrogate_fd(fn, params, direction, eps=1e-6):
    with torch.no_grad():
        plus = fn([p + eps * d for p, d in zip(params, direction)])
        minus = fn([p - eps * d for p, d in zip(params, direction)])
    return float((plus - minus) / (2 * eps))


@pytest.mark.parametrize("nbits,floor", [(2, False), (3, False), (4, False), (4, True)])
def test_quant_bwd_explicit_vs_autograd_vs_fd(nbits, floor):
    g = torch.Generator().manual_seed(20 + nbits)
    w = torch.randn(6, 5, 8, generator=g, dtype=F64) * 0.05
    if floor:
        w[0, 0] = 0.125                            # constant group -> floored h
    gl = torch.randn(6, 5, generator=g, dtype=F64)
    bl = torch.randn(6, 5, generator=g, dtype=F64)
    gup = torch.randn(6, 5, 8, generator=g, dtype=F64)

    st = O.quant_fwd(w, O.sigmoid(gl), O.sigmoid(bl), nbits)
    ex = O.quant_bwd(st, gup)

    wv, gv, bv = (t.clone().requires_grad_(True) for t in (w, gl, bl))
    out = O.quant_ste(wv, O.sigmoid(gv), O.sigmoid(bv), nbits)
    assert torch.allclose(out, st["what"], rtol=0, atol=1e-15)
    dw, dg, db = torch.autograd.grad((out * gup).sum(), [wv, gv, bv])
    assert _rel(dw, ex["dw"]) < 1e-12
    assert _rel(dg, ex["dgamma_logit"]) < 1e-12
    assert _rel(db, ex["dbeta_logit"]) < 1e-12

    tape = O.FrozenTape()
    with O.use_tape(tape):
        O.quant_ste(w, O.sigmoid(gl), O.sigmoid(bl), nbits)

    def loss(ps):
        tape.replay()
        with O.use_tape(tape):
            return (O.quant_ste(ps[0], O.sigmoid(ps[1]), O.sigmoid(ps[2]), nbits) * gup).sum()

    for k in range(3):
        dirs = [torch.randn(t.shape, generator=g, dtype=F64) for t in (w, gl, bl)]
        fd = _surrogate_fd(loss, [w, gl, bl], dirs)
        an = float(sum((d * gr).sum() for d, gr in zip(dirs, (ex["dw"], ex["dgamma_logit"], ex["dbeta_logit"]))))
        assert abs(fd - an) <= 1e-6 * max(abs(an), 1e-8), (fd, an)


def test_clamp_boundary_is_inclusive():
    # c == Q exactly must pass the gradient: MinMax puts the max at code Q.
    w = torch.tensor([[-0.3, 0.0, 0.7]], dtype=F64)
    st = O.quant_fwd(w, 1.0, 1.0, 2)
    assert float(st["c"][0, 2]) == 3.0 and float(st["c"][0, 0]) == 0.0
    gb = O.quant_bwd(st, torch.tensor([[1.0, 1.0, 1.0]], dtype=F64))
    assert float(gb["G_bm"][0]) == 0.0             # nothing clipped


# ------------------------------------------------------------------------------------------------
# Eq. 3 / Eq. 4 on one linear
# ------------------------------------------------------------------------------------------------

def test_let_linear_equivalence():
    g = torch.Generator().manual_seed(7)
    X = torch.randn(33, 24, generator=g, dtype=F64)
    W = torch.randn(40, 24, generator=g, dtype=F64)
    B = torch.randn(40, generator=g, dtype=F64)
    s = torch.exp(torch.randn(24, generator=g, dtype=F64))
    d = torch.randn(24, generator=g, dtype=F64)
    r = O.let_apply(X, W, B, s, d)
    assert _rel(r["Xt"] @ r["Wt"].T + r["Bt"], X @ W.T + B) < 1e-13


def test_act_quant_bwd_let_terms_vs_fd():
    g = torch.Generator().manual_seed(8)
    X = torch.randn(10, 16, generator=g, dtype=F64)
    s = torch.exp(0.3 * torch.randn(16, generator=g, dtype=F64))
    d = 0.2 * torch.randn(16, generator=g, dtype=F64)
    gup = torch.randn(10, 16, generator=g, dtype=F64)
    f = O.act_quant_per_token(X, 4, s, d)
    b = O.act_quant_per_token_bwd(f, gup, s, d)
    tape = O.FrozenTape()
    with O.use_tape(tape):
        O.quant_ste((X - d) / s, 1.0, 1.0, 4)

    def loss(ps):
        tape.replay()
        with O.use_tape(tape):
            return (O.quant_ste((ps[0] - ps[2]) / ps[1], 1.0, 1.0, 4) * gup).sum()

    for k in range(3):
        dirs = [torch.randn(t.shape, generator=g, dtype=F64) for t in (X, s, d)]
        fd = _surrogate_fd(loss, [X, s, d], dirs)
        an = float((dirs[0] * b["dX"]).sum() + (dirs[1] * b["ds"]).sum() + (dirs[2] * b["ddelta"]).sum())
        assert abs(fd - an) <= 1e-6 * max(abs(an), 1e-8), (fd, an)


def test_lwc_bwd_let_scale_vs_fd():
    g = torch.Generator().manual_seed(9)
    W = torch.randn(12, 32, generator=g, dtype=F64) * 0.05
    s = torch.exp(0.3 * torch.randn(32, generator=g, dtype=F64))
    r = torch.exp(0.3 * torch.randn(12, generator=g, dtype=F64))
    gl = torch.randn(12, 4, generator=g, dtype=F64) + 1
    bl = torch.randn(12, 4, generator=g, dtype=F64) + 1
    gup = torch.randn(12, 32, generator=g, dtype=F64)
    f = O.lwc_fakequant_fwd(W, gl, bl, 3, 8, s=s, row_scale=r)
    b = O.lwc_fakequant_bwd(f, W, gup, s=s, row_scale=r)
    tape = O.FrozenTape()
    with O.use_tape(tape):
        O.quant_ste((W * s * r[:, None]).reshape(12, 4, 8), O.sigmoid(gl), O.sigmoid(bl), 3)

    def loss(ps):
        tape.replay()
        with O.use_tape(tape):
            wt = (W * ps[0] * ps[1][:, None]).reshape(12, 4, 8)
            return (O.quant_ste(wt, O.sigmoid(ps[2]), O.sigmoid(ps[3]), 3).reshape(12, 32) * gup).sum()

    for k in range(3):
        dirs = [torch.randn(t.shape, generator=g, dtype=F64) for t in (s, r, gl, bl)]
        fd = _surrogate_fd(loss, [s, r, gl, bl], dirs)
        an = float((dirs[0] * b["ds"]).sum() + (dirs[1] * b["drow_scale"]).sum()
                   + (dirs[2] * b["dgamma_logit"]).sum() + (dirs[3] * b["dbeta_logit"]).sum())
        assert abs(fd - an) <= 1e-6 * max(abs(an), 1e-8), (fd, an)


def test_qlinear_step_matches_explicit_chain():
    """Autograd through Eq. 4 == the explicit chain the kernels follow: loss -> dY ->
    dW_hat = dY^T X_hat -> LWC backward; dX_hat = dY W_hat -> Q_a/LET backward."""
    g = torch.Generator().manual_seed(11)
    T, Cin, Cout = 24, 32, 16
    X = torch.randn(T, Cin, generator=g, dtype=F64)
    W = torch.randn(Cout, Cin, generator=g, dtype=F64) * 0.05
    gl = torch.randn(Cout, 4, generator=g, dtype=F64) + 2
    bl = torch.randn(Cout, 4, generator=g, dtype=F64) + 2
    s = torch.exp(0.2 * torch.randn(Cin, generator=g, dtype=F64))
    d = 0.1 * torch.randn(Cin, generator=g, dtype=F64)
    Yfp = X @ W.T
    r = O.qlinear_step(X, W, None, gl, bl, Yfp, wbits=3, group=8, abits=4, s=s, delta=d, mode="exact")
    fa = O.act_quant_per_token(X, 4, s, d)
    fw = O.lwc_fakequant_fwd(W, gl, bl, 3, 8, s=s)
    Y = fa["Xq"] @ fw["what"].T + W @ d
    loss, dY = O.block_loss(Y, Yfp)
    assert abs(float(loss) - float(r["loss"])) < 1e-14 * max(1.0, float(loss))
    bw = O.lwc_fakequant_bwd(fw, W, dY.T @ fa["Xq"], s=s)
    ba = O.act_quant_per_token_bwd(fa, dY @ fw["what"], s, d)
    dB = dY.sum(0)
    assert _rel(bw["dgamma_logit"], r["dgamma_logit"]) < 1e-11
    assert _rel(bw["dbeta_logit"], r["dbeta_logit"]) < 1e-11
    assert _rel(bw["ds"] + ba["ds"], r["ds"]) < 1e-11
    assert _rel(ba["ddelta"] + W.T @ dB, r["ddelta"]) < 1e-11


def test_block_loss_grad_fd():
    g = torch.Generator().manual_seed(12)
    Y = torch.randn(7, 9, generator=g, dtype=F64)
    Yf = torch.randn(7, 9, generator=g, dtype=F64)
    loss, dY = O.block_loss(Y, Yf)
    assert abs(float(loss) - float(((Y - Yf) ** 2).mean())) < 1e-15
    D = torch.randn(7, 9, generator=g, dtype=F64)
    fd = (O.block_loss(Y + 1e-6 * D, Yf)[0] - O.block_loss(Y - 1e-6 * D, Yf)[0]) / 2e-6
    assert abs(float(fd) - float((D * dY).sum())) < 1e-8


# ------------------------------------------------------------------------------------------------
# block
# ------------------------------------------------------------------------------------------------

def _tiny_block(let=True, abits=4, wbits=4, group=0, n_kv=2, seed=0, T=12):
    shape = I.BlockShape("tiny", T=T, d=32, n_heads=4, n_kv=n_kv, ffn=48, wbits=wbits, abits=abits,
                         group=group, let=int(let), head_dim=8, outlier_frac=0.1, outlier_scale=20.0)
    W = I.make_block_weights(shape, seed=seed + 1)
    W = {k: v * 4.0 for k, v in W.items()}         # std 0.08: outputs of order one at d = 32
    x = I.make_block_input(shape, sample=seed, weight_seed=seed + 1)
    th = I.make_block_theta(shape, W, x, seed=seed + 2, perturb=True)
    cfg = O.BlockCfg.from_shape(shape)
    return shape, W, x, th, cfg


def _t(d):
    return {k: torch.as_tensor(v, dtype=F64) for k, v in d.items()}


@pytest.mark.parametrize("n_kv", [4, 2])
def test_block_let_equivalence_without_quant(n_kv):
    """Eq. 3 and Eq. 5 are exact transformations: with both quantizers off, the LET'd block
    equals the full-precision block for any s, delta, s_a, and the loss against the fp output
    is zero with zero gradient for every LET parameter."""
    shape, W, x, th, cfg = _tiny_block(n_kv=n_kv)
    yfp = O.block_fp_forward(x, W, cfg)
    c = O.BlockCfg.from_shape(shape, wbits=16, abits=16, let=True, mode="exact")
    r = O.block_step(x, yfp, W, th, c)
    assert _rel(r["y"], yfp) < 1e-13
    assert float(r["loss"]) < 1e-26
    for k in O.THETA_NAMES_LET:
        assert float(r["d" + k].abs().max()) < 1e-13, k


@pytest.mark.parametrize("let,abits,wbits,group,n_kv", [(True, 4, 4, 0, 2), (True, 4, 4, 0, 4),
                                                         (False, 16, 3, 8, 4), (False, 16, 2, 16, 4)])
def test_block_gradient_vs_surrogate_fd(let, abits, wbits, group, n_kv):
    """Directional finite differences of the frozen-offset surrogate of the whole block match
    the STE gradients the oracle returns (exact mode, so no bf16 rounding)."""
    shape, W, x, th, cfg = _tiny_block(let=let, abits=abits, wbits=wbits, group=group, n_kv=n_kv)
    cfg = O.BlockCfg.from_shape(shape, mode="exact")
    g = torch.Generator().manual_seed(99)
    yfp = O.block_fp_forward(x, W, cfg) + 0.01 * torch.randn(shape.T, shape.d, generator=g, dtype=F64)
    names = O.THETA_NAMES_LWC + (O.THETA_NAMES_LET if let else [])
    tape = O.FrozenTape()
    with O.use_tape(tape):
        r = O.block_step(x, yfp, W, th, cfg)
    Wt, xt = _t(W), torch.as_tensor(x, dtype=F64)
    base = [torch.as_tensor(th[k], dtype=F64) for k in names]

    def loss(ps):
        tape.replay()
        with O.use_tape(tape):
            y = O.block_forward(xt, Wt, dict(zip(names, ps)), cfg)
        return O.block_loss(y, yfp)[0]

    for k in range(3):
        dirs = [torch.randn(p.shape, generator=g, dtype=F64) for p in base]
        fd = _surrogate_fd(loss, base, dirs, eps=1e-6)
        an = float(sum((d * r["d" + n]).sum() for d, n in zip(dirs, names)))
        assert abs(fd - an) <= 1e-6 * max(abs(an), 1e-12), (fd, an)


def test_attention_matches_naive_loops():
    """Causal RoPE attention of the fp block against a per-(head, query, key) loop."""
    shape, W, x, th, cfg = _tiny_block(n_kv=2, T=6)
    c = O.BlockCfg.from_shape(shape, wbits=16, abits=16, let=False, mode="exact")
    keep = {}
    with torch.no_grad():
        O.block_forward(torch.as_tensor(x, dtype=F64), _t(W), {}, c, keep)
    q, k, v, Ok = keep["q"], keep["k"], keep["v"], keep["O"]
    T, H, Hkv, hd = shape.T, shape.n_heads, shape.n_kv, shape.head_dim
    out = torch.zeros(T, H * hd, dtype=F64)
    for h in range(H):
        kvh = h // (H // Hkv)
        for t in range(T):
            sc = []
            for j in range(t + 1):
                sc.append(sum(float(q[t, h * hd + e]) * float(k[j, kvh * hd + e]) for e in range(hd)) / math.sqrt(hd))
            mx = max(sc)
            ex = [math.exp(s_ - mx) for s_ in sc]
            tot = sum(ex)
            for e in range(hd):
                out[t, h * hd + e] = sum(ex[j] / tot * float(v[j, kvh * hd + e]) for j in range(t + 1))
    assert _rel(Ok, out) < 1e-13


def _causal_probs(H, T, seed, spread=2.0):
    g = torch.Generator().manual_seed(seed)
    S = torch.randn(H, T, T, generator=g, dtype=F64) * spread
    S = S.masked_fill(~torch.ones(T, T, dtype=torch.bool).tril(), float("-inf"))
    return torch.softmax(S, -1)


def test_softmax_quant_hand_example():
    """R20 on a 3-key causal matrix, 2 bits (Q = 3).  Row 2, P = (0.6, 0.3, 0.1): h = 0.5/3 = 1/6,
    z = -round(0.1 * 6) = -1, codes 3, 1, 0, values (code - z) h = 4/6, 2/6, 1/6.  Row 0 has one
    key: range 0, h floored at eps, z = -round(1/eps), value (0 - z) eps = 1.  Row 1,
    P = (0.7, 0.3): h = 0.4/3 = 2/15, z = -round(2.25) = -2, codes round(5.25) - 2 = 3 and
    round(2.25) - 2 = 0, values 5 h = 2/3 and 2 h = 4/15."""
    P = torch.tensor([[[1.0, 0.0, 0.0], [0.7, 0.3, 0.0], [0.6, 0.3, 0.1]]], dtype=F64)
    got = O.softmax_quant(P, 2)
    want = torch.tensor([[[1.0, 0.0, 0.0], [2 / 3, 4 / 15, 0.0], [4 / 6, 2 / 6, 1 / 6]]], dtype=F64)
    assert torch.allclose(got, want, rtol=0, atol=1e-12)
    assert float(got[0, 0, 1]) == 0.0 and float(got[0, 1, 2]) == 0.0


@pytest.mark.parametrize("nbits", [8, 6, 4, 3])
def test_softmax_quant_is_rowwise_minmax_over_visible_keys(nbits):
    """Each query row equals Eq. 2's MinMax quantizer applied to the row's visible slice
    P[t, :t+1] alone (a per-row loop, no filling of the masked part); masked entries are 0."""
    H, T = 2, 9
    P = _causal_probs(H, T, 30 + nbits)
    got = O.softmax_quant(P, nbits)
    for hh in range(H):
        for t in range(T):
            st = O.quant_fwd(P[hh, t, :t + 1][None], 1.0, 1.0, nbits)
            assert torch.allclose(got[hh, t, :t + 1], st["what"][0], rtol=0, atol=1e-15)
            assert bool((got[hh, t, t + 1:] == 0).all())


@pytest.mark.parametrize("nbits", [8, 4])
def test_softmax_quant_ste_gradient_is_per_row_quant_bwd(nbits):
    """Autograd through Q_p equals the explicit STE backward of Eq. 2 (pinned above against finite
    differences) applied to each row's visible slice; masked entries get no gradient."""
    H, T = 2, 8
    P = _causal_probs(H, T, 40 + nbits, spread=1.0).requires_grad_(True)
    g = torch.Generator().manual_seed(41)
    gq = torch.randn(H, T, T, generator=g, dtype=F64)
    (dP,) = torch.autograd.grad(O.softmax_quant(P, nbits), [P], gq)
    Pd = P.detach()
    for hh in range(H):
        for t in range(T):
            st = O.quant_fwd(Pd[hh, t, :t + 1][None], 1.0, 1.0, nbits)
            ex = O.quant_bwd(st, gq[hh, t, :t + 1][None])
            assert torch.allclose(dP[hh, t, :t + 1], ex["dw"][0], rtol=1e-12, atol=1e-14)
            assert bool((dP[hh, t, t + 1:] == 0).all())


def test_zero_point_exact_halves_round_to_even():
    """R21 with R2: when gamma = beta the zero point's quotient is u = Q min / (max - min), so a
    group with max = -min gives u = -Q/2 exactly and one with max = 5 |min| gives u = -Q/6; hand
    values.  N = 4, group (-1, 0.25, 1): u = 15 (-1) / 2 = -7.5, half to even -8, z = 8; N = 2:
    u = -1.5 -> -2, z = 2; N = 4, group (-1, 0, 5): u = 15 (-1) / 6 = -2.5 -> -2, z = 2.  The same
    holds for Q_a (gamma = beta = 1).  With gamma != beta there is no exact half: z = -round(beta
    min / h) of the plain formula."""
    t = lambda v: torch.tensor(v, dtype=F64)
    g4 = t([[-1.0, 0.25, 1.0]])
    a = O.sigmoid(t([4.0]))
    assert float(O.quant_fwd(g4, a, a, 4)["z"][0]) == 8.0
    assert float(O.quant_fwd(g4, a, a, 2)["z"][0]) == 2.0
    assert float(O.quant_fwd(t([[-1.0, 0.0, 5.0]]), a, a, 4)["z"][0]) == 2.0
    assert float(O.quant_fwd(g4, 1.0, 1.0, 4)["z"][0]) == 8.0
    st = O.quant_fwd(t([[-1.0, 0.3, 2.0]]), O.sigmoid(t([3.0])), O.sigmoid(t([1.0])), 4)
    assert float(st["z"][0]) == -round(float(st["b"][0] * -1.0 / st["h"][0]))
    # the STE surrogate and the explicit backward see the same zero point
    w = g4.clone().requires_grad_(True)
    y = O.quant_ste(w, a, a, 4)
    assert torch.allclose(y.detach(), O.quant_fwd(g4, a, a, 4)["what"], rtol=0, atol=1e-15)


def test_sigmoid_silu_hand_values():
    """sigmoid(t) = 1 / (1 + e^-t) (the footnote to Sec. 3.2): sigmoid(0) = 1/2 and
    sigmoid(ln 3) = 1 / (1 + 1/3) = 3/4.  SwiGLU's silu(v) = v sigmoid(v): silu(0) = 0,
    silu(ln 3) = (3/4) ln 3, silu(-ln 3) = -(1/4) ln 3, and silu(v) - silu(-v) = v."""
    l3 = math.log(3.0)
    s = O.sigmoid(torch.tensor([0.0, l3, -l3], dtype=F64)).tolist()
    assert abs(s[0] - 0.5) < 1e-16 and abs(s[1] - 0.75) < 1e-15 and abs(s[2] - 0.25) < 1e-15
    v = O.silu(torch.tensor([0.0, l3, -l3, 2.5], dtype=F64)).tolist()
    assert v[0] == 0.0
    assert abs(v[1] - 0.75 * l3) < 1e-15 and abs(v[2] + 0.25 * l3) < 1e-15
    w = torch.linspace(-6, 6, 25, dtype=F64)
    assert torch.allclose(O.silu(w) - O.silu(-w), w, rtol=0, atol=1e-14)


def test_rmsnorm_hand_values():
    """RMSNorm with unit gain: x / sqrt(mean(x^2) + eps) per token.  Row (3, 4) has mean square
    12.5; with eps = 3.5 the root is sqrt(16) = 4, so the row maps to (0.75, 1.0) (a sum instead
    of the mean, a variance instead of the mean square, or eps outside the root all give other
    values).  Row (2, 2, 2, 2) with eps = 0 maps to ones, and every row is scale invariant up to
    eps."""
    got = O.rmsnorm(torch.tensor([[3.0, 4.0]], dtype=F64), 3.5)
    assert torch.allclose(got, torch.tensor([[0.75, 1.0]], dtype=F64), rtol=0, atol=1e-15)
    assert torch.equal(O.rmsnorm(torch.full((1, 4), 2.0, dtype=F64), 0.0), torch.ones(1, 4, dtype=F64))
    g = torch.Generator().manual_seed(15)
    x = torch.randn(3, 16, generator=g, dtype=F64)
    assert torch.allclose(O.rmsnorm(7.0 * x, 0.0), O.rmsnorm(x, 0.0), rtol=1e-14, atol=0)
    r = O.rmsnorm(x, 0.0)
    assert torch.allclose((r * r).mean(-1), torch.ones(3, dtype=F64), rtol=1e-14, atol=0)


def test_attention_stage_emulate_rounds_normalised_probabilities():
    """In emulate mode (R13) the attention's second product takes the normalised softmax output
    (Eq. 5) rounded to bf16 against bf16(V): equal scores give the causal prefix mean of bf16(V)
    divided exactly, since 1/n rounds to bf16 exactly only for powers of two; the value is the
    plain product bf16(softmax(S)) bf16(V)."""
    g = torch.Generator().manual_seed(19)
    H, T, hd = 2, 7, 4
    cfg = O.BlockCfg(d=H * hd, n_heads=H, n_kv=H, ffn=8, wbits=16, abits=16, group=0, let=False, head_dim=hd)
    V = torch.randn(H, T, hd, generator=g, dtype=F64)
    causal = torch.ones(T, T, dtype=torch.bool).tril()
    S = (torch.randn(H, T, T, generator=g, dtype=F64) * 3).masked_fill(~causal, float("-inf"))
    from oracle.omq_oracle import _attn_pv
    got = _attn_pv(S, V, cfg)
    want = O.to_bf16(torch.softmax(S, -1)) @ O.to_bf16(V)
    assert torch.equal(got, want)
    S0 = torch.zeros(H, T, T, dtype=F64).masked_fill(~causal, float("-inf"))
    n = torch.arange(1, T + 1, dtype=F64)
    want0 = (O.to_bf16(1.0 / n)[None, :, None] * torch.cumsum(O.to_bf16(V), 1))
    assert torch.allclose(_attn_pv(S0, V, cfg), want0, rtol=0, atol=1e-14)


def test_rope_properties():
    g = torch.Generator().manual_seed(13)
    T, H, hd = 9, 2, 8
    q = torch.randn(T, H * hd, generator=g, dtype=F64)
    k = torch.randn(T, H * hd, generator=g, dtype=F64)
    rq = O.rope(q, H, hd, 10000.0)
    assert torch.allclose(rq[0], q[0], atol=0)                     # position 0: identity
    half = hd // 2
    n0 = (q.reshape(T, H, 2, half) ** 2).sum(2)
    n1 = (rq.reshape(T, H, 2, half) ** 2).sum(2)
    assert torch.allclose(n0, n1, atol=1e-12)                      # pair norms kept
    # relative position: <rope(a, t1), rope(b, t2)> depends on t1 - t2 only
    a = torch.randn(1, hd, generator=g, dtype=F64).expand(T, hd).contiguous()
    b = torch.randn(1, hd, generator=g, dtype=F64).expand(T, hd).contiguous()
    ra, rb = O.rope(a, 1, hd, 10000.0), O.rope(b, 1, hd, 10000.0)
    assert abs(float(ra[5] @ rb[3]) - float(ra[4] @ rb[2])) < 1e-12
    assert abs(float(ra[7] @ rb[3]) - float(ra[4] @ rb[0])) < 1e-12


def test_emulate_mode_rounds_matmul_operands():
    g = torch.Generator().manual_seed(14)
    A = torch.randn(5, 7, generator=g, dtype=F64)
    B = torch.randn(3, 7, generator=g, dtype=F64)
    from oracle.omq_oracle import _mm
    C = _mm(A, B, "emulate")
    assert torch.equal(C, O.to_bf16(A) @ O.to_bf16(B).T)


def test_rope_rotation_direction():
    """RoFormer's rotation R(t*w) = [[cos, -sin], [sin, cos]] applied to (x_j, x_{j+hd/2}):
    with head_dim 2 the single frequency is 1, so position 1 maps (1, 0) to (cos 1, sin 1)."""
    v = torch.tensor([[1.0, 0.0], [1.0, 0.0]], dtype=F64)
    r = O.rope(v, 1, 2, 10000.0)
    assert torch.allclose(r[1], torch.tensor([math.cos(1.0), math.sin(1.0)], dtype=F64), atol=1e-15)


@pytest.mark.parametrize("n_kv", [4, 2])
def test_let_init_balances_ranges_and_centres(n_kv):
    """LET initialisation (Sec. 4.1: scaling as SmoothQuant, shifting as OS+; reading R16),
    checked through the properties that define it rather than its formula: with alpha = 0.5
    every unclamped channel of X / s and of W * s has the same maximum magnitude (the difficulty
    is split evenly between activation and weight), the shift makes the channel mean of X - delta
    zero over the calibration tokens, and s_a equalises max|Q / s_a| and max|K * s_a| per channel
    (maxima over the query heads of a kv group).  Statistics are recomputed here in numpy from
    the full-precision block's intermediates."""
    shape, W, _, _, cfg = _tiny_block(n_kv=n_kv)
    xs = [I.make_block_input(shape, sample=i, weight_seed=1) for i in range(3)]
    th = O.let_init(xs, W, cfg)
    H, Hkv, hd = shape.n_heads, shape.n_kv, shape.head_dim
    rep = H // Hkv
    keeps = []
    for x in xs:
        k = {}
        O.block_forward(torch.as_tensor(x, dtype=F64), _t(W), {},
                        O.BlockCfg.from_shape(shape, wbits=16, abits=16, let=False, mode="exact"), k)
        keeps.append({n: v.numpy() for n, v in k.items()})
    rms = lambda v: v / np.sqrt((v * v).mean(1, keepdims=True) + shape.rms_eps)
    A = np.concatenate([rms(np.asarray(x, np.float64)) for x in xs])
    B = np.concatenate([rms(k["h1"]) for k in keeps])
    Q = np.concatenate([k["q"] for k in keeps]).reshape(-1, Hkv, rep, hd)
    K = np.concatenate([k["k"] for k in keeps]).reshape(-1, Hkv, hd)
    Ob = np.concatenate([k["O"] for k in keeps]).reshape(-1, Hkv, rep, hd)
    g = {n: v.numpy() for n, v in th.items()}

    def balanced(Xa, Wa, s):
        lhs = np.abs(Xa / s).max(0)
        rhs = np.abs(Wa * s).max(0)
        free = s > 1e-5 * (1 + 1e-9)
        assert free.any()
        assert np.allclose(lhs[free], rhs[free], rtol=1e-12, atol=0)

    balanced(A, np.concatenate([W["wq"], W["wk"], W["wv"]]).astype(np.float64), g["s1"])
    balanced(B, np.concatenate([W["wg"], W["wu"]]).astype(np.float64), g["s2"])
    assert np.abs((A - g["d1"]).mean(0)).max() < 1e-12
    assert np.abs((B - g["d2"]).mean(0)).max() < 1e-12
    # [v, out]: per value channel, maxima over the group's heads of O / s_o and W_o * s_o columns
    Wo = np.asarray(W["wo"], np.float64).reshape(-1, Hkv, rep, hd)
    lhs = np.abs(Ob / g["so"].reshape(1, Hkv, 1, hd)).max(axis=(0, 2))
    rhs = np.abs(Wo * g["so"].reshape(1, Hkv, 1, hd)).max(axis=(0, 2))
    assert np.allclose(lhs, rhs, rtol=1e-12, atol=0)
    assert np.abs((Ob - g["do"].reshape(1, Hkv, 1, hd)).mean(axis=(0, 2))).max() < 1e-12
    # [Q, K]
    qs = np.abs(Q / g["sa"].reshape(1, Hkv, 1, hd)).max(axis=(0, 2))
    ks = np.abs(K * g["sa"].reshape(1, Hkv, hd)).max(0)
    assert np.allclose(qs, ks, rtol=1e-12, atol=0)


def test_pack_codes_bit_layout_by_hand():
    """Packed codes (reading R17): code i of a row occupies bits [N i, N i + N) of the row's
    little-endian bit stream.  Hand-packed bytes for N = 4, 2 and 3."""
    c4 = torch.tensor([[1, 2, 3, 4, 15, 0, 7, 8]])
    assert O.pack_codes(c4, 4).tolist() == [[0x21, 0x43, 0x0F, 0x87]]
    c2 = torch.tensor([[1, 2, 3, 0, 3, 3, 0, 1]])
    assert O.pack_codes(c2, 2).tolist() == [[0b00111001, 0b01001111]]
    # N = 3: stream 001 010 011 100 101 110 111 000 (LSB first) -> bytes 0xD1, 0x58, 0x1F
    c3 = torch.tensor([[1, 2, 3, 4, 5, 6, 7, 0]])
    bits = [(v >> b) & 1 for v in [1, 2, 3, 4, 5, 6, 7, 0] for b in range(3)]
    hand = [sum(bits[8 * k + j] << j for j in range(8)) for k in range(3)]
    assert hand == [0xD1, 0x58, 0x1F]
    assert O.pack_codes(c3, 3).tolist() == [hand]
    g = torch.Generator().manual_seed(5)
    for n in (2, 3, 4, 8):
        c = torch.randint(0, 2 ** n, (6, 64), generator=g)
        assert torch.equal(O.unpack_codes(O.pack_codes(c, n), n, 64), c)


@pytest.mark.parametrize("let,abits,wbits,group,n_kv", [(True, 4, 4, 0, 4), (True, 4, 4, 0, 2),
                                                         (False, 16, 3, 8, 4)])
def test_folded_block_equals_calibrated_block(let, abits, wbits, group, n_kv):
    """Fold & pack (Algorithm 1's transform-then-quantize; reading R17): the deployed block built
    only from the packed codes, h, z, biases, folded RMSNorm gains / biases and s_a computes the
    same output as the calibrated block with its LET and LWC parameters (fp64, decisions in fp64)."""
    shape, W, x, th, cfg = _tiny_block(let=let, abits=abits, wbits=wbits, group=group, n_kv=n_kv)
    c = O.BlockCfg.from_shape(shape, mode="exact")
    folded = O.block_fold_pack(W, th, c)
    y_fold = O.folded_forward(folded, x, c)
    y_ref = O.block_forward(torch.as_tensor(x, dtype=F64), _t(W), _t(th), c)
    assert _rel(y_fold, y_ref) < 1e-12
    assert folded["codes_qkv"].dtype == torch.uint8
    assert folded["codes_qkv"].shape[1] * 8 == shape.d * wbits


def test_adamw_step_matches_library_adamw():
    """The oracle's AdamW update (Sec. 4.1 "Training"; reading R18) equals torch.optim.AdamW over
    several steps, with and without decoupled weight decay."""
    g = torch.Generator().manual_seed(3)
    for wd in (0.0, 0.1):
        p0 = torch.randn(7, generator=g, dtype=F64)
        p_ref = p0.clone().requires_grad_(True)
        opt = torch.optim.AdamW([p_ref], lr=1e-2, betas=(0.9, 0.999), eps=1e-8, weight_decay=wd)
        p, m, v = p0.clone(), torch.zeros(7, dtype=F64), torch.zeros(7, dtype=F64)
        for step in range(1, 6):
            grad = torch.randn(7, generator=g, dtype=F64)
            p_ref.grad = grad.clone()
            opt.step()
            O.adamw_step(p, grad, m, v, 1e-2, step, wd=wd)
        assert torch.allclose(p, p_ref.detach(), rtol=1e-12, atol=1e-14)


def test_calibration_driver_data_flow():
    """Algorithm 1's data flow: with zero epochs, after each block X_fp is the full-precision block
    of the previous X_fp and X_q the quantized block (initial parameters) of the previous X_q, and
    the LET parameters of each block are let_init of that block's fp inputs."""
    shape, W0, x, th, cfg = _tiny_block(let=True, abits=4, wbits=4, n_kv=2)
    W1 = {k: v[::-1].copy() for k, v in W0.items()}
    xs = [x, I.make_block_input(shape, sample=1, weight_seed=1)]
    params, x_fp, x_q = O.calibrate_blocks([W0, W1], xs, cfg, th, epochs=0)
    f0 = [O.block_fp_forward(xx, W0, cfg) for xx in xs]
    f1 = [O.block_fp_forward(xx, W1, cfg) for xx in f0]
    for a, b in zip(x_fp, f1):
        assert torch.equal(a, b)
    p0 = dict(_t(th), **O.let_init(xs, W0, cfg))
    q0 = [O.block_forward(torch.as_tensor(xx, dtype=F64), _t(W0), p0, cfg) for xx in xs]
    p1 = dict(_t(th), **O.let_init(f0, W1, cfg))
    q1 = [O.block_forward(xx, _t(W1), p1, cfg) for xx in q0]
    for a, b in zip(x_q, q1):
        assert torch.equal(a, b)
    for k in O.THETA_NAMES_LET:
        assert torch.equal(params[1][k], p1[k])
