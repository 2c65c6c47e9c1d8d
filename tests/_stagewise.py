"""Stage-wise comparison of one GPU calibration step with the fp64 oracle.

The block is cut where the GPU keeps a stage value (omq_block_saved_layout): q|k|v before RoPE,
the attention output O, h1, gate|up and the output y.  Each oracle stage starts from the GPU's
own value of its input, and each stage's backward from the GPU's own gradient of its output, so a
4-bit code that flips in one stage (a quotient within rounding of a half) cannot carry into the
next.  Every learnable parameter's gradient is the sum of its stages' contributions (s_o and
delta_o appear in the q|k|v stage through v_proj and in the o_proj stage); the sums are compared
with the GPU's gradients.  Stage outputs and the loss are held to 1e-2, gradients to 3e-2
(relative Frobenius error).  The code decisions of every quantizer the step saves are checked
with the shared-scale protocol of `_parity`.
"""
from __future__ import annotations

from typing import Dict

import numpy as np
import torch

import oracle as O
from oracle.omq_oracle import _expand_kv
from _parity import (GRAD_TOL, OUT_TOL, add_counts, check_codes, check_h, check_zero_points, code_counts, fp32_band,
                     grad_errors, record, record_codes, rel)

F64 = torch.float64


def _t(v):
    return torch.as_tensor(np.asarray(v) if not torch.is_tensor(v) else v).to(F64)


def _host(v):
    return v.detach().float().cpu().to(F64) if v.dtype != torch.int32 else v.detach().cpu()


def _param_names(shape):
    return (O.THETA_NAMES_LWC if shape.wbits < 16 else []) + (O.THETA_NAMES_LET if shape.let else [])


def _grads(outs, leaves, gouts):
    g = torch.autograd.grad(outs, leaves, gouts, allow_unused=True)
    return [torch.zeros_like(l) if gi is None else gi for gi, l in zip(g, leaves)]


def compare_step(shape, W: Dict[str, np.ndarray], x: np.ndarray, th: Dict[str, np.ndarray], yfp, y_gpu,
                 loss_gpu: float, grads_gpu: Dict[str, np.ndarray], sv: Dict[str, object], tag: str,
                 codes: bool = True, pbits: int = 16):
    """Asserts the stage-wise bounds; returns {check: relative error}."""
    cfg = O.BlockCfg.from_shape(shape, pbits=pbits)
    T, f = shape.T, shape.ffn
    dq, dkv = shape.dq, shape.dkv
    Wd = {k: _t(v) for k, v in W.items()}
    names = _param_names(shape)
    leaf = {k: _t(th[k]).clone().requires_grad_(True) for k in names}
    P = [leaf[k] for k in names]
    G = {k: _host(v) for k, v in sv.items() if not isinstance(v, list)}
    xx = _t(x)
    yq = _t(y_gpu)
    err, total = {}, [torch.zeros_like(p) for p in P]

    def add(gs):
        for i, gi in enumerate(gs):
            total[i] = total[i] + gi

    # stage A: x -> q|k|v (RMSNorm, LET [ln1,(q,k,v)] and [v,out] on v_proj, Q_a, three products)
    q0, k0, v0, _ = O.stage_attn_in(xx, Wd, leaf, cfg)
    qkv = torch.cat([q0, k0, v0], 1)
    err["fwd q|k|v"] = rel(G["y_qkv"], qkv.detach())
    add(_grads(qkv, P, G["dy_qkv"]) if P else [])
    del q0, k0, v0, qkv

    # stage B: GPU q|k|v -> O (RoPE, [Q,K] LET, Q_a, causal attention)
    qkv_in = G["y_qkv"].clone().requires_grad_(True)
    Oref, _, _ = O.stage_attention(qkv_in[:, :dq], qkv_in[:, dq:dq + dkv], qkv_in[:, dq + dkv:], leaf, cfg)
    err["fwd O"] = rel(G["o"], Oref.detach())
    gB = _grads(Oref, P + [qkv_in], G["do_bf16"])
    add(gB[:-1])
    err["bwd d(q|k|v)"] = rel(G["dy_qkv"], gB[-1])
    del Oref, gB, qkv_in

    # stage C: GPU O -> h1 (Q_a, o_proj with the [v,out] column scale and bias, residual)
    O_in = G["o"].clone().requires_grad_(True)
    h1 = O.stage_attn_out(O_in, xx, Wd, leaf, cfg)
    err["fwd h1"] = rel(G["h1"], h1.detach())
    gC = _grads(h1, P + [O_in], G["dh1"])
    add(gC[:-1])
    err["bwd dO"] = rel(G["do_bf16"], gC[-1])
    del h1, gC, O_in

    # stage D: GPU h1 -> gate|up (RMSNorm, LET [ln2,(gate,up)], Q_a, two products)
    h1_in = G["h1"].clone().requires_grad_(True)
    gt, up = O.stage_ffn_in(h1_in, Wd, leaf, cfg)
    err["fwd gate|up"] = rel(G["y_gu"], torch.cat([gt, up], 1).detach())
    gD = _grads([gt, up], P + [h1_in], [G["dy_gu"][:, :f], G["dy_gu"][:, f:]])
    add(gD[:-1])
    dh1_norm = gD[-1]
    del gt, up, gD, h1_in

    # stage E: GPU gate|up -> y (SwiGLU, Q_a, down_proj, residual)
    gu_in = G["y_gu"].clone().requires_grad_(True)
    yref, _ = O.stage_ffn_out(gu_in[:, :f], gu_in[:, f:], G["h1"], Wd, leaf, cfg)
    err["fwd y"] = rel(yq, yref.detach())
    gE = _grads(yref, P + [gu_in], G["dy"])
    add(gE[:-1])
    err["bwd d(gate|up)"] = rel(G["dy_gu"], gE[-1])
    err["bwd dh1"] = rel(G["dh1"], dh1_norm + G["dy"])
    del yref, gE, gu_in

    # loss (Eq. 1, mean squared error) on the GPU's output
    lref, dyref = O.block_loss(yq, _t(yfp))
    err["loss"] = abs(loss_gpu - float(lref)) / float(lref)
    err["bwd dy"] = rel(G["dy"], dyref)

    err.update(grad_errors(grads_gpu, {"d" + n: gsum for n, gsum in zip(names, total)}, names))
    record("stage-wise", tag, **{k: float(v) for k, v in err.items()})
    bad = {k: v for k, v in err.items() if not v < (OUT_TOL if not (k.startswith("d") or k.startswith("bwd")) else GRAD_TOL)}
    if codes:
        check_step_codes(shape, W, x, th, sv, tag)
    assert not bad, bad
    return err


def _expand(vec, shape):
    rep = shape.n_heads // shape.n_kv
    v = torch.as_tensor(np.asarray(vec), dtype=torch.float32)
    return v.reshape(shape.n_kv, 1, shape.head_dim).expand(shape.n_kv, rep, shape.head_dim).reshape(-1)


def weight_inputs_fp32(shape, W, th, dtype=torch.float32):
    """The quantizer inputs of the block's four weight operands (q|k|v, o, gate|up, down):
    W~ = W s r (Eq. 3; the v rows of q|k|v carry the [v, out] pair's row scale 1 / s_o, o_proj's
    columns s_o, R14).  In float32 each product is one correctly rounded operation and the row
    scale is fl32(1 / s_o), the GPU's fp32 input; with dtype float64 the exact values."""
    lins = [(("wq", "wk", "wv"), "s1", True), (("wo",), "so", False), (("wg", "wu"), "s2", False),
            (("wd",), None, False)]
    out = []
    for parts, skey, rows in lins:
        Wl = torch.cat([torch.from_numpy(np.asarray(W[p], np.float32)) for p in parts]).to(dtype)
        if shape.let and skey is not None:
            sv_ = _expand(th["so"], shape) if skey == "so" else torch.as_tensor(np.asarray(th[skey]), dtype=torch.float32)
            Wl = Wl * sv_.to(dtype)[None, :]
            if rows:
                so = torch.as_tensor(np.asarray(th["so"]), dtype=torch.float32).to(dtype)
                Wl = Wl * torch.cat([torch.ones(shape.dq + shape.dkv, dtype=dtype), 1.0 / so])[:, None]
        out.append(Wl)
    return out


def check_step_codes(shape, W, x, th, sv, tag):
    """Codes of the four weight quantizers (shared scale, fp32 input W~ = fl32(fl32(W s) r)) and of
    the per-token quantizers of the linear inputs (the oracle's float64 input against the GPU's h,
    z, exempting the fp32 rounding band of the GPU's producer)."""
    # codes are recovered from the bf16 operand (code - z) h, which holds them exactly only while
    # |code - z| * 2^-8 < 1/2 (bf16 keeps 8 significant bits): up to 6 bits
    parts = [("q", "k", "v"), ("o",), ("g", "u"), ("d",)]
    if shape.wbits < 16:                    # h and z of every weight group against the oracle
        for i, Wx in enumerate(weight_inputs_fp32(shape, W, th, torch.float64)):
            cout, cin = Wx.shape
            gl = torch.cat([torch.as_tensor(np.asarray(th["gamma_" + p])) for p in parts[i]]).double()
            bl = torch.cat([torch.as_tensor(np.asarray(th["beta_" + p])) for p in parts[i]]).double()
            f = O.lwc_fakequant_fwd(Wx, gl, bl, shape.wbits, shape.group, eps=1e-5)
            st = f["st"]
            name = f"{tag} W{['qkv', 'o', 'gu', 'd'][i]}"
            check_h(name, sv["w_h"][i].cpu(), f["h"], st["a"] * st["M"], st["b"] * st["m"], 2 ** shape.wbits - 1)
            check_zero_points(name, st["u"], sv["w_z"][i].cpu(), f["z"])
            del f, st
    if shape.wbits <= 6:
        for i, Wl in enumerate(weight_inputs_fp32(shape, W, th)):
            cout, cin = Wl.shape
            g = cin if shape.group == 0 else shape.group
            h = sv["w_h"][i].cpu().double()
            z = sv["w_z"][i].cpu()
            wh = sv["w_hat"][i]
            n = None
            for r0 in range(0, cout, 4096):            # row blocks bound the host memory
                r1 = min(cout, r0 + 4096)
                hb = h[r0:r1]
                x_ = Wl[r0:r1].double().reshape(r1 - r0, cin // g, g) / hb[..., None]
                qz = torch.round(wh[r0:r1].cpu().double().reshape(r1 - r0, cin // g, g) / hb[..., None])
                c = code_counts(f"{tag} W{['qkv', 'o', 'gu', 'd'][i]}", x_, qz + z[r0:r1, :, None].double(),
                                z[r0:r1], shape.wbits)
                n = c if n is None else add_counts(n, c)
            record_codes(n)
    if shape.abits <= 6:
        cfg = O.BlockCfg.from_shape(shape)
        xx = _t(x)
        a = O.rmsnorm(xx, shape.rms_eps)
        s1, d1 = (_t(th["s1"]), _t(th["d1"])) if shape.let else (1.0, 0.0)
        at = (a - d1) / s1
        h, z = sv["a_h"].cpu().double(), sv["a_z"].cpu()
        qz = torch.round(sv["a_hat"].cpu().double() / h[:, None])
        band = fp32_band((a.abs() + abs(torch.as_tensor(d1))) / torch.as_tensor(s1), h[:, None], 32) + \
            fp32_band(at, h[:, None], 4)
        check_codes(f"{tag} A q|k|v input", at / h[:, None], qz + z[:, None].double(), z, shape.abits, band)
        # Q~, K~, V' from the GPU's own q|k|v: V' is the fp32 input itself; Q~ and K~ pass RoPE (an fp32
        # sin / cos table) and s_a, a few roundings of the rotated pair's magnitude
        dq, dkv, hd = shape.dq, shape.dkv, shape.head_dim
        Y = sv["y_qkv"].cpu().double()
        qh, zh = sv["qkv_h"].cpu().double(), sv["qkv_z"].cpu()
        sa = _t(th["sa"]) if shape.let else torch.ones(dkv, dtype=F64)
        for seg, (lo, hi, key) in enumerate([(0, dq, "q_hat"), (dq, dq + dkv, "k_hat"), (dq + dkv, dq + 2 * dkv, "v_hat")]):
            v = Y[:, lo:hi]
            band = None
            if seg < 2:
                nh = (hi - lo) // hd
                pair = v.reshape(-1, nh, 2, hd // 2).abs().sum(2, keepdim=True).expand(-1, nh, 2, hd // 2).reshape(v.shape)
                v = O.rope(v, nh, hd, shape.rope_theta)
                if seg == 0:
                    v = v / _expand_kv(sa, cfg)
                    pair = pair / _expand_kv(sa, cfg)
                else:
                    v = v * sa
                    pair = pair * sa
            h, z = qh[seg], zh[seg]
            if seg < 2:
                band = fp32_band(pair, h[:, None], 8)
            qz = torch.round(sv[key].cpu().double() / h[:, None])
            check_codes(f"{tag} A {key[0]} (attention input)", v / h[:, None], qz + z[:, None].double(), z,
                        shape.abits, band)
        # o_proj input: Q_a of the GPU's own O (plain producer: the fp32 input is exact)
        Og = sv["o"].cpu().double()
        h, z = sv["o_h"].cpu().double(), sv["o_z"].cpu()
        qz = torch.round(sv["o_hat"].cpu().double() / h[:, None])
        check_codes(f"{tag} A o_proj input", Og / h[:, None], qz + z[:, None].double(), z, shape.abits)
        # gate|up input from the GPU's own h1 (RMSNorm + LET as for the q|k|v input)
        b = O.rmsnorm(sv["h1"].cpu().double(), shape.rms_eps)
        s2, d2 = (_t(th["s2"]), _t(th["d2"])) if shape.let else (1.0, 0.0)
        bt = (b - d2) / s2
        h, z = sv["b_h"].cpu().double(), sv["b_z"].cpu()
        qz = torch.round(sv["b_hat"].cpu().double() / h[:, None])
        band = fp32_band((b.abs() + abs(torch.as_tensor(d2))) / torch.as_tensor(s2), h[:, None], 32) + \
            fp32_band(bt, h[:, None], 4)
        check_codes(f"{tag} A gate|up input", bt / h[:, None], qz + z[:, None].double(), z, shape.abits, band)
        # down_proj input silu(gate) up from the GPU's own gate|up (an fp32 exp and two roundings)
        f = shape.ffn
        gu = sv["y_gu"].cpu().double()
        m = O.silu(gu[:, :f]) * gu[:, f:]
        h, z = sv["m_h"].cpu().double(), sv["m_z"].cpu()
        qz = torch.round(sv["m_hat"].cpu().double() / h[:, None])
        check_codes(f"{tag} A down_proj input", m / h[:, None], qz + z[:, None].double(), z, shape.abits,
                    fp32_band(m, h[:, None], 8))
        del cfg
