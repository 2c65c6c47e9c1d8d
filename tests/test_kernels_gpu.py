"""Kernel-level parity of every C-ABI entry point against the fp64 oracle.

Code decisions follow the shared-scale protocol of `_parity`: the codes must equal
round(w / h) + z, clamped, for the exact quotient of the fp32 quantizer input w (W~ = fl32(s W),
times fl32 of the row scale; X~ = fl32(fl32(X - delta) / s)) and the kernel's own h and z, except
elements within 1e-6 of a .5 boundary, which are counted and reported.  h is compared with the
fp64 oracle (1e-6 relative), z with the oracle's float64 decision (exemptions counted), the
max/min indices with the first index of the fp32 input's extremes.  Real-valued outputs are
compared with the fp64 oracle (gradients to 3e-2 relative Frobenius error, the benchmark spec's bound)."""
import numpy as np
import pytest
import torch

import oracle as O
from _parity import GRAD_TOL, OUT_TOL, check_codes, check_h, check_zero_points, rel as _rel
from paper_2308_13137_gb300 import _lib, inputs as I

pytestmark = pytest.mark.gpu
F64 = torch.float64


def _dev(a, dtype=torch.float32):
    return torch.as_tensor(np.asarray(a)).to(dtype).cuda().contiguous()


def _first_extremes(G32):
    """First index of the max and of the min along the last axis (R7) of an fp32 tensor."""
    imax = (G32 == G32.max(-1, keepdim=True).values).int().argmax(-1)
    imin = (G32 == G32.min(-1, keepdim=True).values).int().argmax(-1)
    return imax, imin


LWC_CASES = [  # Cout, Cin, nbits, group, let, rowscale, perturb
    (512, 512, 4, 128, False, False, False),       # the single-linear workload
    (512, 512, 4, 128, False, False, True),
    (384, 1024, 4, 0, True, False, True),          # per-channel with LET scale
    (256, 768, 3, 128, False, False, True),
    (256, 512, 2, 64, False, False, True),
    (192, 512, 4, 0, True, True, True),            # v_proj rows divided by s_o
    (64, 11008, 4, 0, False, False, True),         # down_proj row length
    (128, 512, 8, 128, True, False, True),         # 8 bits: quotients up to 255
]


@pytest.mark.parametrize("Cout,Cin,nbits,group,let,rowscale,perturb", LWC_CASES)
def test_lwc_fwd_bwd(cuda_lib, Cout, Cin, nbits, group, let, rowscale, perturb):
    rng = np.random.default_rng(Cout + Cin + nbits)
    W = I.bf16_representable((0.02 * rng.standard_t(3, (Cout, Cin)) / np.sqrt(3)).astype(np.float32))
    ng = Cin // (group or Cin)
    gl = (4.0 + (rng.normal(-2.5, 1.5, (Cout, ng)) if perturb else np.zeros((Cout, ng)))).astype(np.float32)
    bl = (4.0 + (rng.normal(-2.5, 1.5, (Cout, ng)) if perturb else np.zeros((Cout, ng)))).astype(np.float32)
    s = np.exp(rng.normal(0, 0.5, Cin)).astype(np.float32) if let else None
    r = np.exp(rng.normal(0, 0.3, Cout)).astype(np.float32) if rowscale else None
    delta = rng.normal(0, 0.3, Cin).astype(np.float32) if let else None
    shift = rng.normal(0, 0.1, Cout).astype(np.float32) if rowscale else None
    cfg = _lib.make_cfg(wbits=nbits, group=group)
    Wd = _dev(W, torch.bfloat16)
    Wq = torch.empty(Cout, Cin, dtype=torch.bfloat16, device="cuda")
    codes = torch.empty(Cout, Cin, dtype=torch.uint8, device="cuda")
    h = torch.empty(Cout, ng, device="cuda")
    z = torch.empty(Cout, ng, dtype=torch.int32, device="cuda")
    imax = torch.empty_like(z)
    imin = torch.empty_like(z)
    Bt = torch.empty(Cout, device="cuda") if let else None
    sd = _dev(s) if let else None
    rd = _dev(r) if rowscale else None
    _lib.omq_lwc_fakequant_fwd(Cout, Cin, Wd, sd, rd, _dev(gl), _dev(bl), Wq, codes, h, z, imax, imin,
                               _dev(delta) if let else None, _dev(shift) if rowscale else None, Bt, cfg)
    torch.cuda.synchronize()
    tag = f"lwc {Cout}x{Cin} W{nbits} g{group}{' LET' if let else ''}{' rows' if rowscale else ''}"

    # -- the fp32 quantizer input W~ = fl32(fl32(W s) r) (one correctly rounded product each) --
    wt32 = torch.from_numpy(W)
    if let:
        wt32 = wt32 * torch.from_numpy(s)[None, :]
    if rowscale:
        wt32 = wt32 * torch.from_numpy(r)[:, None]
    gsz = group or Cin
    G32 = wt32.reshape(Cout, ng, gsz)
    hg, zg = h.cpu(), z.cpu()
    fmax, fmin = _first_extremes(G32)
    base = torch.arange(ng) * gsz
    assert torch.equal(imax.cpu().long(), fmax + base) and torch.equal(imin.cpu().long(), fmin + base)
    x = G32.double() / hg.double()[..., None]
    check_codes(tag, x, codes.cpu().reshape(Cout, ng, gsz), zg, nbits)
    qz = codes.cpu().reshape(Cout, ng, gsz).float() - zg.float()[..., None]
    assert torch.equal(Wq.cpu(), (qz * hg[..., None]).reshape(Cout, Cin).to(torch.bfloat16))

    # -- h and z against the fp64 oracle --
    f = O.lwc_fakequant_fwd(torch.from_numpy(W), torch.from_numpy(gl), torch.from_numpy(bl), nbits, group,
                            s=torch.from_numpy(s) if let else None,
                            row_scale=torch.from_numpy(r) if rowscale else None)
    st = f["st"]
    check_h(tag, hg, f["h"], st["a"] * st["M"], st["b"] * st["m"], 2 ** nbits - 1)
    check_zero_points(tag, st["u"], zg, f["z"])
    if let:
        ref_B = (torch.from_numpy(W).double() @ torch.from_numpy(delta).double()
                 - (torch.from_numpy(shift).double() if rowscale else 0)) * (torch.from_numpy(r).double() if rowscale else 1)
        assert _rel(Bt.cpu(), ref_B) < 1e-5

    # -- backward against the oracle's own (float64-decided) forward --
    g = np.random.default_rng(7).standard_normal((Cout, Cin)).astype(np.float32)
    dBt = rng.standard_normal(Cout).astype(np.float32) if let else None
    dgl = torch.empty(Cout, ng, device="cuda")
    dbl = torch.empty_like(dgl)
    dWt = torch.empty(Cout, Cin, device="cuda")
    ds = torch.empty(Cin, device="cuda") if let else None
    dr = torch.empty(Cout, device="cuda") if rowscale else None
    dd = torch.empty(Cin, device="cuda") if let else None
    ws = torch.empty(_lib.omq_lwc_bwd_workspace_size(Cout, Cin), dtype=torch.uint8, device="cuda")
    _lib.omq_lwc_fakequant_bwd(Cout, Cin, Wd, sd, rd, _dev(gl), _dev(bl), h, z, imax, imin, _dev(g), dgl, dbl, dWt,
                               ds, dr, _dev(dBt) if let else None, dd, ws, cfg)
    torch.cuda.synchronize()
    b = O.lwc_fakequant_bwd(f, torch.from_numpy(W), torch.from_numpy(g), s=torch.from_numpy(s) if let else None,
                            row_scale=torch.from_numpy(r) if rowscale else None)
    assert _rel(dgl.cpu(), b["dgamma_logit"]) < GRAD_TOL
    assert _rel(dbl.cpu(), b["dbeta_logit"]) < GRAD_TOL
    assert _rel(dWt.cpu(), b["dWt"]) < GRAD_TOL
    if let:
        assert _rel(ds.cpu(), b["ds"]) < GRAD_TOL
        rv = torch.from_numpy(r).double() if rowscale else 1.0
        ref_dd = torch.from_numpy(W).double().T @ (torch.from_numpy(dBt).double() * rv)
        assert _rel(dd.cpu(), ref_dd) < 1e-5
    if rowscale:
        assert _rel(dr.cpu(), b["drow_scale"]) < GRAD_TOL


ACT_CASES = [  # T, C, nbits, let
    (256, 512, 4, False),
    (300, 4096, 4, True),
    (64, 11008, 8, False),
    (128, 1024, 2, True),
    (96, 512, 16, True),
    (80, 2048, 8, True),
]


@pytest.mark.parametrize("T,C,nbits,let", ACT_CASES)
def test_act_quant_fwd_bwd(cuda_lib, T, C, nbits, let):
    rng = np.random.default_rng(T + C)
    X = rng.standard_normal((T, C)).astype(np.float32)
    X[:, rng.choice(C, max(1, C // 100), replace=False)] *= 50
    s = np.exp(rng.normal(0, 0.5, C)).astype(np.float32) if let else None
    d = rng.normal(0, 0.5, C).astype(np.float32) if let else None
    cfg = _lib.make_cfg(abits=nbits)
    Xq = torch.empty(T, C, dtype=torch.bfloat16, device="cuda")
    codes = torch.empty(T, C, dtype=torch.uint8, device="cuda") if nbits < 16 else None
    h = torch.empty(T, device="cuda")
    z = torch.empty(T, dtype=torch.int32, device="cuda")
    imax, imin = torch.empty_like(z), torch.empty_like(z)
    Xd = _dev(X)
    sd, dd = (_dev(s), _dev(d)) if let else (None, None)
    _lib.omq_act_quant_per_token(T, C, Xd, sd, dd, Xq, codes, h, z, imax, imin, cfg)
    torch.cuda.synchronize()
    # the fp32 quantizer input X~ = fl32(fl32(X - delta) / s), each operation correctly rounded
    Xt32 = torch.from_numpy(X)
    if let:
        Xt32 = (Xt32 - torch.from_numpy(d)) / torch.from_numpy(s)
    tag = f"act {T}x{C} A{nbits}{' LET' if let else ''}"
    if nbits >= 16:
        assert torch.equal(Xq.cpu(), Xt32.to(torch.bfloat16))
        fa = None
    else:
        hg, zg = h.cpu(), z.cpu()
        fmax, fmin = _first_extremes(Xt32)
        assert torch.equal(imax.cpu().long(), fmax) and torch.equal(imin.cpu().long(), fmin)
        check_codes(tag, Xt32.double() / hg.double()[:, None], codes.cpu(), zg, nbits)
        qz = codes.cpu().float() - zg.float()[:, None]
        assert torch.equal(Xq.cpu(), (qz * hg[:, None]).to(torch.bfloat16))
        fa = O.act_quant_per_token(torch.from_numpy(X), nbits, torch.from_numpy(s) if let else None,
                                   torch.from_numpy(d) if let else None)
        st = fa["st"]
        check_h(tag, hg, fa["h"], st["M"], st["m"], 2 ** nbits - 1)
        check_zero_points(tag, st["u"], zg, fa["z"])
    # backward
    g = np.random.default_rng(9).standard_normal((T, C)).astype(np.float32)
    dX = torch.empty(T, C, device="cuda")
    ds = torch.empty(C, device="cuda") if let else None
    ddl = torch.empty(C, device="cuda") if let else None
    ws = torch.empty(_lib.omq_act_bwd_workspace_size(T, C), dtype=torch.uint8, device="cuda")
    _lib.omq_act_quant_per_token_bwd(T, C, Xd, sd, dd, h, z, imax, imin, _dev(g), dX, ds, ddl, ws, cfg)
    torch.cuda.synchronize()
    if nbits >= 16:
        ref = torch.from_numpy(g).double() / (torch.from_numpy(s).double() if let else 1.0)
        assert _rel(dX.cpu(), ref) < 1e-6
        return
    ba = O.act_quant_per_token_bwd(fa, torch.from_numpy(g), torch.from_numpy(s) if let else None,
                                   torch.from_numpy(d) if let else None)
    assert _rel(dX.cpu(), ba["dX"]) < GRAD_TOL
    if let:
        assert _rel(ds.cpu(), ba["ds"]) < GRAD_TOL
        assert _rel(ddl.cpu(), ba["ddelta"]) < GRAD_TOL


def test_block_loss(cuda_lib):
    g = torch.Generator().manual_seed(3)
    n = 2048 * 520
    Yq, Yf = torch.randn(n, generator=g), torch.randn(n, generator=g)
    loss = torch.zeros(1, device="cuda")
    dY = torch.empty(n, device="cuda")
    dYb = torch.empty(n, dtype=torch.bfloat16, device="cuda")
    ws = torch.empty(_lib.omq_loss_workspace_size(n), dtype=torch.uint8, device="cuda")
    _lib.omq_block_loss(n, Yq.cuda(), Yf.cuda(), loss, dY, dYb, ws)
    torch.cuda.synchronize()
    rl, rd = O.block_loss(Yq, Yf)
    assert abs(float(loss) - float(rl)) / float(rl) < 1e-5
    assert _rel(dY.cpu(), rd) < 1e-6
    assert torch.equal(dYb.cpu(), dY.cpu().to(torch.bfloat16))


def test_let_apply(cuda_lib):
    rng = np.random.default_rng(4)
    T, Cin, Cout = 64, 256, 128
    X = rng.standard_normal((T, Cin)).astype(np.float32)
    W = I.bf16_representable(rng.standard_normal((Cout, Cin)).astype(np.float32) * 0.02)
    B = rng.standard_normal(Cout).astype(np.float32)
    s = np.exp(rng.normal(0, 0.5, Cin)).astype(np.float32)
    d = rng.normal(0, 0.5, Cin).astype(np.float32)
    Xt, Wt, Bt = torch.empty(T, Cin, device="cuda"), torch.empty(Cout, Cin, device="cuda"), torch.empty(Cout, device="cuda")
    _lib.omq_let_apply(T, Cin, Cout, _dev(X), _dev(W, torch.bfloat16), _dev(B), _dev(s), _dev(d), Xt, Wt, Bt,
                       _lib.make_cfg())
    torch.cuda.synchronize()
    r = O.let_apply(torch.from_numpy(X), torch.from_numpy(W), torch.from_numpy(B), torch.from_numpy(s), torch.from_numpy(d))
    assert _rel(Xt.cpu(), r["Xt"]) < 1e-6 and _rel(Wt.cpu(), r["Wt"]) < 1e-6 and _rel(Bt.cpu(), r["Bt"]) < 1e-5
    assert _rel((Xt.double() @ Wt.double().T + Bt.double()).cpu(), torch.from_numpy(X).double() @ torch.from_numpy(W).double().T + torch.from_numpy(B).double()) < 1e-5


def _qlinear_gpu(case, nbits, group, abits, let, s=None, d=None, Yfp=None):
    T, Cin, Cout = case["X"].shape[0], case["X"].shape[1], case["W"].shape[0]
    ng = Cin // (group or Cin)
    cfg = _lib.make_cfg(wbits=nbits, abits=abits, group=group, let=let)
    sv = dict(w_hat=torch.empty(Cout, Cin, dtype=torch.bfloat16, device="cuda"),
              h_w=torch.empty(Cout, ng, device="cuda"), z_w=torch.empty(Cout, ng, dtype=torch.int32, device="cuda"),
              imax_w=torch.empty(Cout, ng, dtype=torch.int32, device="cuda"),
              imin_w=torch.empty(Cout, ng, dtype=torch.int32, device="cuda"),
              x_hat=torch.empty(T, Cin, dtype=torch.bfloat16, device="cuda"), h_a=torch.empty(T, device="cuda"),
              z_a=torch.empty(T, dtype=torch.int32, device="cuda"), imax_a=torch.empty(T, dtype=torch.int32, device="cuda"),
              imin_a=torch.empty(T, dtype=torch.int32, device="cuda"), b_tilde=torch.empty(Cout, device="cuda"))
    saved = _lib.omq_qlinear_saved(*[sv[k].data_ptr() for k in ("w_hat", "h_w", "z_w", "imax_w", "imin_w", "x_hat",
                                                                "h_a", "z_a", "imax_a", "imin_a", "b_tilde")])
    X, W = _dev(case["X"]), _dev(case["W"], torch.bfloat16)
    gl, bl = _dev(case["gamma_logit"]), _dev(case["beta_logit"])
    sd, dd = (_dev(s), _dev(d)) if let else (None, None)
    Y = torch.empty(T, Cout, device="cuda")
    _lib.omq_qlinear_fwd(T, Cin, Cout, X, W, _dev(case["B"]), sd, dd, gl, bl, Y, saved, cfg)
    loss = torch.zeros(1, device="cuda")
    dY = torch.empty(T, Cout, device="cuda")
    lws = torch.empty(_lib.omq_loss_workspace_size(T * Cout), dtype=torch.uint8, device="cuda")
    _lib.omq_block_loss(T * Cout, Y, _dev(Yfp), loss, dY, None, lws)
    dgl, dbl = torch.empty(Cout, ng, device="cuda"), torch.empty(Cout, ng, device="cuda")
    ds = torch.empty(Cin, device="cuda") if let else None
    ddl = torch.empty(Cin, device="cuda") if let else None
    ws = torch.empty(_lib.omq_qlinear_workspace_size(T, Cin, Cout, cfg), dtype=torch.uint8, device="cuda")
    _lib.omq_qlinear_bwd(T, Cin, Cout, X, W, sd, dd, gl, bl, saved, dY, None, dgl, dbl, ds, ddl, ws, cfg)
    torch.cuda.synchronize()
    return dict(Y=Y.cpu(), loss=float(loss), dgamma_logit=dgl.cpu(), dbeta_logit=dbl.cpu(),
                ds=None if ds is None else ds.cpu(), ddelta=None if ddl is None else ddl.cpu())


@pytest.mark.parametrize("perturb", [False, True])
def test_qlinear_step_single_linear_workload(cuda_lib, perturb):
    """The single-linear W4A16 g128 workload: X 256x512, W 512x512 Student-t, gamma=beta=4."""
    sh = I.SHAPES["linear_w4a16_g128"]
    case = I.make_linear_case(sh, seed=0, perturb_theta=perturb)
    Yfp = (torch.from_numpy(case["X"]).double() @ torch.from_numpy(case["W"]).double().T).float().numpy()
    got = _qlinear_gpu(case, 4, 128, 16, 0, Yfp=Yfp)
    t = {k: torch.from_numpy(v) for k, v in case.items()}
    ref = O.qlinear_step(t["X"], t["W"], t["B"], t["gamma_logit"], t["beta_logit"], torch.from_numpy(Yfp), 4, 128, 16)
    assert _rel(got["Y"], ref["Y"]) < OUT_TOL
    assert abs(got["loss"] - float(ref["loss"])) / float(ref["loss"]) < OUT_TOL
    assert _rel(got["dgamma_logit"], ref["dgamma_logit"]) < GRAD_TOL
    assert _rel(got["dbeta_logit"], ref["dbeta_logit"]) < GRAD_TOL


def test_qlinear_step_w4a4_let(cuda_lib):
    sh = I.LinearShape("w4a4", T=384, Cin=1024, Cout=512)
    case = I.make_linear_case(sh, seed=3, perturb_theta=True)
    case["gamma_logit"] = case["gamma_logit"][:, :1].copy()
    case["beta_logit"] = case["beta_logit"][:, :1].copy()
    rng = np.random.default_rng(11)
    case["X"][:, rng.choice(1024, 10, replace=False)] *= 50
    s = np.exp(rng.normal(0, 0.5, 1024)).astype(np.float32)
    d = rng.normal(0, 0.2, 1024).astype(np.float32)
    Yfp = (torch.from_numpy(case["X"]).double() @ torch.from_numpy(case["W"]).double().T).float().numpy()
    got = _qlinear_gpu(case, 4, 0, 4, 1, s=s, d=d, Yfp=Yfp)
    t = {k: torch.from_numpy(v) for k, v in case.items()}
    ref = O.qlinear_step(t["X"], t["W"], t["B"], t["gamma_logit"], t["beta_logit"], torch.from_numpy(Yfp), 4, 0, 4,
                         s=torch.from_numpy(s), delta=torch.from_numpy(d))
    assert _rel(got["Y"], ref["Y"]) < OUT_TOL
    assert abs(got["loss"] - float(ref["loss"])) / float(ref["loss"]) < OUT_TOL
    for k in ("dgamma_logit", "dbeta_logit", "ds", "ddelta"):
        assert _rel(got[k], ref[k]) < GRAD_TOL, k


def test_adamw(cuda_lib):
    g = torch.Generator().manual_seed(2)
    n = 1000
    p, gr = torch.randn(n, generator=g), torch.randn(n, generator=g)
    m, v = torch.randn(n, generator=g) * 0.1, torch.rand(n, generator=g) * 0.1
    pd, md, vd = p.cuda(), m.cuda(), v.cuda()
    _lib.omq_adamw_update(n, pd, gr.cuda(), md, vd, 5e-3, 0.9, 0.999, 1e-8, 0.0, 3)
    torch.cuda.synchronize()
    m2 = 0.9 * m.double() + 0.1 * gr.double()
    v2 = 0.999 * v.double() + 0.001 * gr.double() ** 2
    p2 = p.double() - 5e-3 * (m2 / (1 - 0.9 ** 3)) / ((v2 / (1 - 0.999 ** 3)).sqrt() + 1e-8)
    assert _rel(pd.cpu(), p2) < 1e-6 and _rel(md.cpu(), m2) < 1e-6 and _rel(vd.cpu(), v2) < 1e-6


def test_adamw_device_step(cuda_lib):
    """The device-counter form: three advances then one update equals the update at step 3."""
    g = torch.Generator().manual_seed(3)
    n = 1000
    p, gr = torch.randn(n, generator=g), torch.randn(n, generator=g)
    m, v = torch.randn(n, generator=g) * 0.1, torch.rand(n, generator=g) * 0.1
    pd, md, vd = p.cuda(), m.cuda(), v.cuda()
    t = torch.zeros(1, dtype=torch.int32, device="cuda")
    for _ in range(3):
        _lib.omq_step_advance(t)
    _lib.omq_adamw_update_dev(n, pd, gr.cuda(), md, vd, 5e-3, 0.9, 0.999, 1e-8, 0.0, t)
    torch.cuda.synchronize()
    assert int(t.item()) == 3
    m2 = 0.9 * m.double() + 0.1 * gr.double()
    v2 = 0.999 * v.double() + 0.001 * gr.double() ** 2
    p2 = p.double() - 5e-3 * (m2 / (1 - 0.9 ** 3)) / ((v2 / (1 - 0.999 ** 3)).sqrt() + 1e-8)
    assert _rel(pd.cpu(), p2) < 1e-6 and _rel(md.cpu(), m2) < 1e-6 and _rel(vd.cpu(), v2) < 1e-6
