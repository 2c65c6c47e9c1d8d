"""Parity at the full workload sizes (2048 tokens, LLaMA-7B/13B/70B block shapes), through the
same BlockState calls and kernel launch configurations that bench.py times.

* LLaMA-7B W4A4 LWC+LET (the timed workload): the whole calibration step against the fp64 oracle
  (emulate mode): block output, loss and every parameter gradient.  At 2048 tokens the W4A4 step
  is discontinuous in its input: every rounding decision of Eq. 2 on the per-token 4-bit q, k,
  v, o and FFN activations is a step function, and a flipped code in k or v reaches every later
  query through attention.  Moving the input by 2 ulps moves the oracle's own output by about
  1.3 % and its gradients by up to 3 % (most rows unchanged, a few late tokens by 5-10 %).  So the
  test measures that spread in the oracle (the same step on the input scaled by 1 + 2^-22) and
  asks of the GPU step: at least 90 % of the output rows within 1e-3 of the oracle (the tokens
  whose decisions agree), the loss within 1e-2, and the output and every gradient within the
  small-shape tolerances or twice the oracle's own spread, whichever is larger.  The GPU
  full-precision forward that produces the Eq. 1 target is checked as well.
* LLaMA-7B W3A16 g128, LLaMA-13B W2A16 g64 and LLaMA-2-70B W4A4 GQA: block output and loss of
  the step against the oracle's quantized forward (the gradient paths of these configurations
  are covered element by element at small sizes).
* Every weight operand of the 7B W4A4 block: the LWC fake-quant of the full weight on the GPU,
  with the codes of a seeded sample of rows bit-exact against the oracle (rows are independent).

Inputs follow the bench recipe: weights seed 1, calibration sample 0, parameters seed 2.
"""
import numpy as np
import pytest
import torch

import oracle as O
from paper_2308_13137_gb300 import _lib
from paper_2308_13137_gb300 import inputs as I
from paper_2308_13137_gb300.block import BlockState

pytestmark = [pytest.mark.gpu, pytest.mark.full]
OUT_TOL, GRAD_TOL = 1e-2, 3e-2
F64 = torch.float64


def _rel(a, b):
    a, b = torch.as_tensor(a).double().cpu(), torch.as_tensor(b).double().cpu()
    return float((a - b).norm() / b.norm().clamp_min(1e-300))


def _inputs(shape):
    W = I.make_block_weights(shape, seed=1)
    x = I.make_block_input(shape, sample=0, weight_seed=1)
    th = I.make_block_theta(shape, W, x, seed=2)
    return W, x, th


def _gpu_step(shape, W, x, th, yfp):
    st = BlockState(shape, W, th)
    xd = torch.from_numpy(x).cuda()
    y_fp_gpu = torch.empty_like(xd)
    st.fp_forward(xd, y_fp_gpu)
    y = torch.empty_like(xd)
    st.step(xd, yfp.cuda(), y)
    torch.cuda.synchronize()
    assert int(st.status.item()) == 0
    out = dict(y=y.cpu(), loss=float(st.loss.item()), y_fp=y_fp_gpu.cpu(), **st.split_grads())
    del st
    torch.cuda.empty_cache()
    return out


@pytest.fixture(scope="module")
def c2_full(cuda_lib):
    shape = I.block_shape("llama7b_w4a4")
    W, x, th = _inputs(shape)
    cfg = O.BlockCfg.from_shape(shape)
    yfp = O.block_fp_forward(x, W, cfg).float()
    got = _gpu_step(shape, W, x, th, yfp)
    ref = O.block_step(x, yfp, W, th, cfg)
    x2 = (x.astype(np.float64) * (1.0 + 2.0 ** -22)).astype(np.float32)     # the input moved by 2 ulps
    ref2 = O.block_step(x2, yfp, W, th, cfg)
    spread = {"y": _rel(ref2["y"], ref["y"])}
    for n in O.THETA_NAMES_LWC + O.THETA_NAMES_LET:
        spread["d" + n] = _rel(ref2["d" + n], ref["d" + n])
    return shape, got, ref, yfp, spread


def test_full_c2_fp_target(c2_full):
    _, got, _, yfp, _ = c2_full
    assert _rel(got["y_fp"], yfp) < OUT_TOL


def test_full_c2_step(c2_full):
    shape, got, ref, _, spread = c2_full
    y, yr = torch.as_tensor(got["y"]).double(), torch.as_tensor(ref["y"]).double()
    row_err = (y - yr).norm(dim=1) / yr.norm(dim=1)
    agree = float((row_err <= 1e-3).double().mean())
    print(f"rows within 1e-3: {agree:.4f}; y error {_rel(y, yr):.3e} (oracle 2-ulp spread {spread['y']:.3e})")
    assert agree >= 0.9, (agree, spread["y"])
    assert _rel(y, yr) < max(OUT_TOL, 2 * spread["y"]), (_rel(y, yr), spread["y"])
    assert abs(got["loss"] - float(ref["loss"])) / float(ref["loss"]) < OUT_TOL
    bad = {}
    for n in O.THETA_NAMES_LWC + O.THETA_NAMES_LET:
        e = _rel(got["d" + n], ref["d" + n])
        if not e < max(GRAD_TOL, 2 * spread["d" + n]):
            bad[n] = (e, spread["d" + n])
    assert not bad, bad


FWD_ONLY = ["llama7b_w3a16_g128", "llama13b_w2a16_g64", "llama2_70b_w4a4_gqa"]


@pytest.mark.parametrize("name", FWD_ONLY)
def test_full_forward_and_loss(cuda_lib, name):
    shape = I.block_shape(name)
    W, x, th = _inputs(shape)
    cfg = O.BlockCfg.from_shape(shape)
    yfp = O.block_fp_forward(x, W, cfg).float()
    got = _gpu_step(shape, W, x, th, yfp)
    with torch.no_grad():
        t = lambda v: torch.as_tensor(v).to(F64)
        y = O.block_forward(t(x), {k: t(v) for k, v in W.items()}, {k: t(v) for k, v in th.items()}, cfg)
        loss, _ = O.block_loss(y, yfp.to(F64))
    assert _rel(got["y"], y) < OUT_TOL
    assert abs(got["loss"] - float(loss)) / float(loss) < OUT_TOL


def _stacked_linears(shape, W, th):
    """The four weight operands of the block exactly as its LWC launches see them: stacked q|k|v
    (LET scale s1, rows of v divided by s_o) and gate|up (LET scale s2), o (scale s_o, Eq. 5's
    [v, out] pair) and down (no LET)."""
    f32 = np.float32
    dq, dkv = shape.dq, shape.dkv
    rep = shape.n_heads // shape.n_kv
    so_exp = np.repeat(th["so"].reshape(shape.n_kv, 1, shape.head_dim), rep, axis=1).reshape(-1)
    do_exp = np.repeat(th["do"].reshape(shape.n_kv, 1, shape.head_dim), rep, axis=1).reshape(-1)
    r_qkv = np.concatenate([np.ones(dq + dkv, f32), f32(1.0) / th["so"]]).astype(f32)
    sh_qkv = np.concatenate([np.zeros(dq + dkv, f32), th["do"]]).astype(f32)
    cat = lambda *k: np.concatenate([th[n] for n in k], axis=0)
    return [
        ("qkv", np.concatenate([W["wq"], W["wk"], W["wv"]]), th["s1"], r_qkv, th["d1"], sh_qkv,
         cat("gamma_q", "gamma_k", "gamma_v"), cat("beta_q", "beta_k", "beta_v")),
        ("o", W["wo"], so_exp.astype(f32), None, do_exp.astype(f32), None, th["gamma_o"], th["beta_o"]),
        ("gu", np.concatenate([W["wg"], W["wu"]]), th["s2"], None, th["d2"], None,
         cat("gamma_g", "gamma_u"), cat("beta_g", "beta_u")),
        ("d", W["wd"], None, None, None, None, th["gamma_d"], th["beta_d"]),
    ]


@pytest.fixture(scope="module")
def c2_linears():
    shape = I.block_shape("llama7b_w4a4")
    W, _, th = _inputs(shape)
    return _stacked_linears(shape, W, th)


@pytest.mark.parametrize("which", range(4), ids=["qkv", "o", "gu", "d"])
def test_full_lwc_rows_sampled(cuda_lib, c2_linears, which):
    """Full-size LWC fake-quant (per-channel W4) of each weight operand of the 7B W4A4 block
    through omq_lwc_fakequant_fwd: on a seeded sample of 64 rows the integer codes, z, the first
    argmax/argmin and h equal the oracle with its decisions in fp32, W_hat is (code - z) h
    rounded to bf16, and the LET bias B~ = r (W delta - shift) agrees to fp32 accuracy."""
    tag, Wn, s, r, delta, shift, gl, bl = c2_linears[which]
    Cout, Cin = Wn.shape
    dev = lambda a, dt=torch.float32: None if a is None else torch.from_numpy(np.ascontiguousarray(a)).to(dt).cuda()
    Wd = dev(Wn, torch.bfloat16)
    Wq = torch.empty(Cout, Cin, dtype=torch.bfloat16, device="cuda")
    codes = torch.empty(Cout, Cin, dtype=torch.uint8, device="cuda")
    h = torch.empty(Cout, 1, device="cuda")
    z = torch.empty(Cout, 1, dtype=torch.int32, device="cuda")
    imax, imin = torch.empty_like(z), torch.empty_like(z)
    Bt = torch.empty(Cout, device="cuda") if s is not None else None
    cfg = _lib.make_cfg(wbits=4, group=0)
    _lib.omq_lwc_fakequant_fwd(Cout, Cin, Wd, dev(s), dev(r), dev(gl), dev(bl), Wq, codes, h, z, imax, imin,
                               dev(delta), dev(shift), Bt, cfg)
    torch.cuda.synchronize()
    rows = np.sort(np.random.default_rng(11).choice(Cout, size=64, replace=False))
    ri = torch.from_numpy(rows).cuda()
    t64 = lambda a: None if a is None else torch.from_numpy(np.ascontiguousarray(a))
    ref = O.lwc_fakequant_fwd(t64(Wn[rows]), t64(gl[rows]), t64(bl[rows]), 4, 0, s=t64(s),
                              row_scale=None if r is None else t64(r[rows]), decide="fp32")
    hg, zg = h[ri].cpu(), z[ri].cpu()
    assert torch.equal(codes[ri].cpu().long(), ref["codes"])
    assert torch.equal(zg.double(), ref["z"]) and torch.equal(hg.double(), ref["h"])
    assert torch.equal(imax[ri].cpu().long(), ref["argmax"]) and torch.equal(imin[ri].cpu().long(), ref["argmin"])
    what = ((ref["codes"].float() - zg.float()) * hg.float()).to(torch.bfloat16)
    assert torch.equal(Wq[ri].cpu(), what)
    if s is not None:
        Bref = torch.from_numpy(Wn[rows]).double() @ torch.from_numpy(delta).double()
        if shift is not None:
            Bref = Bref - torch.from_numpy(shift[rows]).double()
        if r is not None:
            Bref = Bref * torch.from_numpy(r[rows]).double()
        assert _rel(Bt[ri].cpu(), Bref) < 1e-5
