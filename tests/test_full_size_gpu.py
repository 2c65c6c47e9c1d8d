"""Parity at the full workload sizes (2048 tokens, LLaMA-7B/13B/70B block shapes), through the
same BlockState calls and kernel launch configurations that bench.py times.

* Stage-wise (`_stagewise`): for LLaMA-7B W4A4 LWC+LET (the timed workload), LLaMA-7B W3A16
  g128, LLaMA-13B W2A16 g64 and LLaMA-2-70B W4A4 GQA, every stage of the GPU step (q|k|v, the
  attention, o_proj, gate|up, down_proj, the loss) against the fp64 oracle started from the GPU's
  own stage input and output gradient: stage outputs and the loss within 1e-2, every stage input
  gradient and every parameter gradient (each the sum of its stages) within 3e-2; the codes of
  all four weight quantizers and of the per-token quantizers the step keeps, under the
  shared-scale protocol (exempt elements counted in the parity report).
* End to end (7B W4A4): the oracle's whole step from the block input, recorded in the parity
  report.  At 2048 tokens the W4A4 step is discontinuous in its input (every per-token 4-bit
  decision is a step function and a flipped code in k or v reaches every later query), so the
  end-to-end distance measures that sensitivity as much as the kernels; the loss is held to 1e-2.
* The GPU full-precision forward that produces the Eq. 1 target, against the oracle's.
* omq_lwc_fakequant_fwd on each full 7B weight operand: codes of a seeded sample of rows under
  the shared-scale protocol, z, h and the first max/min indices.

Inputs follow the bench recipe: weights seed 1, calibration sample 0, parameters seed 2.
"""
import numpy as np
import pytest
import torch

import oracle as O
from _parity import OUT_TOL, check_codes, check_h, check_zero_points, record, rel as _rel
from _stagewise import compare_step
from paper_2308_13137_gb300 import _lib
from paper_2308_13137_gb300 import inputs as I
from paper_2308_13137_gb300.block import BlockState

pytestmark = [pytest.mark.gpu, pytest.mark.full]
F64 = torch.float64


def _inputs(shape):
    W = I.make_block_weights(shape, seed=1)
    x = I.make_block_input(shape, sample=0, weight_seed=1)
    th = I.make_block_theta(shape, W, x, seed=2)
    return W, x, th


def _gpu_step(shape, W, x, th, yfp, fp_target=False):
    """One GPU step; returns the output, loss, gradients and the saved stage values on the host."""
    st = BlockState(shape, W, th)
    xd = torch.from_numpy(x).cuda()
    out = {}
    if fp_target:
        y_fp_gpu = torch.empty_like(xd)
        st.fp_forward(xd, y_fp_gpu)
        out["y_fp"] = y_fp_gpu.cpu()
    y = torch.empty_like(xd)
    st.step(xd, yfp.cuda(), y)
    torch.cuda.synchronize()
    assert int(st.status.item()) == 0
    sv = st.saved()
    host = {k: ([t.cpu() for t in v] if isinstance(v, list) else v.cpu()) for k, v in sv.items()}
    out.update(y=y.cpu(), loss=float(st.loss.item()), grads=st.split_grads(), saved=host)
    del st, sv
    torch.cuda.empty_cache()
    return out


@pytest.fixture(scope="module")
def c2_full(cuda_lib):
    shape = I.block_shape("llama7b_w4a4")
    W, x, th = _inputs(shape)
    cfg = O.BlockCfg.from_shape(shape)
    yfp = O.block_fp_forward(x, W, cfg).float()
    got = _gpu_step(shape, W, x, th, yfp, fp_target=True)
    return shape, W, x, th, yfp, got


def test_full_c2_fp_target(c2_full):
    _, _, _, _, yfp, got = c2_full
    assert _rel(got["y_fp"], yfp) < OUT_TOL


def test_full_c2_stagewise(c2_full):
    shape, W, x, th, yfp, got = c2_full
    compare_step(shape, W, x, th, yfp, got["y"], got["loss"], got["grads"], got["saved"], "llama7b_w4a4 full")


def test_full_c2_end_to_end(c2_full):
    shape, W, x, th, yfp, got = c2_full
    ref = O.block_step(x, yfp, W, th, O.BlockCfg.from_shape(shape))
    y, yr = torch.as_tensor(got["y"]).double(), ref["y"]
    row_err = (y - yr).norm(dim=1) / yr.norm(dim=1)
    errs = dict(y=_rel(y, yr), loss=abs(got["loss"] - float(ref["loss"])) / float(ref["loss"]),
                rows_within_1e3=float((row_err <= 1e-3).double().mean()))
    for n in O.THETA_NAMES_LWC + O.THETA_NAMES_LET:
        errs["d" + n] = _rel(got["grads"]["d" + n], ref["d" + n])
    record("end to end", "llama7b_w4a4 full", **errs)
    assert errs["loss"] < OUT_TOL, errs


STAGEWISE = ["llama7b_w3a16_g128", "llama13b_w2a16_g64", "llama2_70b_w4a4_gqa"]


@pytest.mark.parametrize("name", STAGEWISE)
def test_full_stagewise(cuda_lib, name):
    shape = I.block_shape(name)
    W, x, th = _inputs(shape)
    yfp = O.block_fp_forward(x, W, O.BlockCfg.from_shape(shape)).float()
    got = _gpu_step(shape, W, x, th, yfp)
    compare_step(shape, W, x, th, yfp, got["y"], got["loss"], got["grads"], got["saved"], f"{name} full")


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
    through omq_lwc_fakequant_fwd: on a seeded sample of 64 rows the codes under the shared-scale
    protocol, z against the oracle's float64 decision, h within 1e-6 of the oracle, the first
    argmax/argmin of the fp32 input, W_hat = bf16((code - z) h), and the LET bias
    B~ = r (W delta - shift) to fp32 accuracy."""
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
    # the fp32 quantizer input W~ = fl32(fl32(W s) r)
    w32 = torch.from_numpy(np.ascontiguousarray(Wn[rows]))
    if s is not None:
        w32 = w32 * torch.from_numpy(s)[None, :]
    if r is not None:
        w32 = w32 * torch.from_numpy(r[rows])[:, None]
    hg, zg = h[ri].cpu(), z[ri].cpu()
    name = f"lwc full 7B {tag} (64 rows)"
    x = (w32.double() / hg.double()).reshape(64, 1, Cin)
    check_codes(name, x, codes[ri].cpu().reshape(64, 1, Cin), zg, 4)
    assert torch.equal(imax[ri].cpu()[:, 0].long(), (w32 == w32.max(1, keepdim=True).values).int().argmax(1))
    assert torch.equal(imin[ri].cpu()[:, 0].long(), (w32 == w32.min(1, keepdim=True).values).int().argmax(1))
    what = ((codes[ri].cpu().float() - zg.float()) * hg).to(torch.bfloat16)
    assert torch.equal(Wq[ri].cpu(), what)
    ref = O.lwc_fakequant_fwd(t64(Wn[rows]), t64(gl[rows]), t64(bl[rows]), 4, 0, s=t64(s),
                              row_scale=None if r is None else t64(r[rows]))
    st = ref["st"]
    check_h(name, hg, ref["h"], st["a"] * st["M"], st["b"] * st["m"], 15)
    check_zero_points(name, st["u"], zg, ref["z"])
    if s is not None:
        Bref = torch.from_numpy(Wn[rows]).double() @ torch.from_numpy(delta).double()
        if shift is not None:
            Bref = Bref - torch.from_numpy(shift[rows]).double()
        if r is not None:
            Bref = Bref * torch.from_numpy(r[rows]).double()
        assert _rel(Bt[ri].cpu(), Bref) < 1e-5
