"""Edge cases of the quantizers and the block step on the GPU, element by element against the oracle.

* Eq. 2 degenerate groups (R3, R4, R7): a constant group and a constant token row (h floored at
  eps, no gradient through h), max and min repeated at several positions (first index takes the
  routed gradient), all-positive and all-negative groups (z outside [0, 2^N - 1]).
* Quotients exactly on a .5 boundary (R2, R21): a per-token row with max = -min = 7.5 has h = 1,
  so elements k + 1/2 are exact halves, and so is u = -7.5; with the clipping strengths at 1
  (logits 80) the same holds for a weight group.  Both sides round half to even; the halves are
  counted in the parity report.
* A group as wide as the row (group = Cin) equals the per-channel form.
* The block step at T = 1, 3 and 127 tokens (a single token, fewer tokens than a vector, a ragged
  last tile), stage-wise and end to end."""
import numpy as np
import pytest
import torch

import oracle as O
from _parity import GRAD_TOL, OUT_TOL, check_codes, check_h, check_zero_points, grad_errors, record, rel
from _stagewise import compare_step
from paper_2308_13137_gb300 import _lib, inputs as I
from paper_2308_13137_gb300.block import BlockState

pytestmark = pytest.mark.gpu
F64 = torch.float64


def _dev(a, dtype=torch.float32):
    return torch.as_tensor(np.asarray(a)).to(dtype).cuda().contiguous()


def _lwc(W, gl, bl, nbits, group, g):
    """GPU forward and backward of LWC on W [Cout, Cin] (no LET) with upstream gradient g."""
    Cout, Cin = W.shape
    ng = Cin // (group or Cin)
    cfg = _lib.make_cfg(wbits=nbits, group=group)
    Wd = _dev(W, torch.bfloat16)
    out = dict(Wq=torch.empty(Cout, Cin, dtype=torch.bfloat16, device="cuda"),
               codes=torch.empty(Cout, Cin, dtype=torch.uint8, device="cuda"),
               h=torch.empty(Cout, ng, device="cuda"), z=torch.empty(Cout, ng, dtype=torch.int32, device="cuda"),
               imax=torch.empty(Cout, ng, dtype=torch.int32, device="cuda"),
               imin=torch.empty(Cout, ng, dtype=torch.int32, device="cuda"))
    gld, bld = _dev(gl), _dev(bl)
    _lib.omq_lwc_fakequant_fwd(Cout, Cin, Wd, None, None, gld, bld, out["Wq"], out["codes"], out["h"], out["z"],
                               out["imax"], out["imin"], None, None, None, cfg)
    dgl, dbl = torch.empty(Cout, ng, device="cuda"), torch.empty(Cout, ng, device="cuda")
    dWt = torch.empty(Cout, Cin, device="cuda")
    ws = torch.empty(_lib.omq_lwc_bwd_workspace_size(Cout, Cin), dtype=torch.uint8, device="cuda")
    _lib.omq_lwc_fakequant_bwd(Cout, Cin, Wd, None, None, gld, bld, out["h"], out["z"], out["imax"], out["imin"],
                               _dev(g), dgl, dbl, dWt, None, None, None, None, ws, cfg)
    torch.cuda.synchronize()
    out.update(dgl=dgl, dbl=dbl, dWt=dWt)
    return {k: v.cpu() for k, v in out.items()}


def _check_lwc(tag, W, gl, bl, nbits, group, g, got):
    Cout, Cin = W.shape
    gsz = group or Cin
    ng = Cin // gsz
    G = torch.from_numpy(W).reshape(Cout, ng, gsz)
    hg, zg = got["h"], got["z"]
    check_codes(tag, G.double() / hg.double()[..., None], got["codes"].reshape(Cout, ng, gsz), zg, nbits)
    f = O.lwc_fakequant_fwd(torch.from_numpy(W), torch.from_numpy(gl), torch.from_numpy(bl), nbits, group)
    st = f["st"]
    check_h(tag, hg, f["h"], st["a"] * st["M"], st["b"] * st["m"], 2 ** nbits - 1)
    check_zero_points(tag, st["u"], zg, f["z"])
    assert torch.equal(got["imax"].long(), f["argmax"]) and torch.equal(got["imin"].long(), f["argmin"])
    b = O.lwc_fakequant_bwd(f, torch.from_numpy(W), torch.from_numpy(g))
    errs = dict(dgamma=rel(got["dgl"], b["dgamma_logit"]), dbeta=rel(got["dbl"], b["dbeta_logit"]),
                dW=rel(got["dWt"], b["dWt"]))
    record("edge case", tag, **errs)
    assert all(v < GRAD_TOL for v in errs.values()), errs
    return f, b


def _student(rng, shape, std=0.02):
    return I.bf16_representable((std * rng.standard_t(3, shape) / np.sqrt(3)).astype(np.float32))


def test_lwc_degenerate_groups(cuda_lib):
    """Row 0: constant group (h floored, no gradient through h); row 1: an all-zero group; row 2:
    max and min each repeated at three positions (the first takes the routing); row 3: all
    positive (z < 0); row 4: all negative (z > Q); the rest ordinary."""
    rng = np.random.default_rng(41)
    Cout, Cin, group, nbits = 16, 256, 128, 4
    W = _student(rng, (Cout, Cin))
    W[0, :128] = np.float32(0.0078125)
    W[1, 128:] = 0.0
    W[2, [5, 40, 100]] = np.float32(0.5)
    W[2, [7, 70, 127]] = np.float32(-0.5)
    W[3] = np.abs(W[3]) + np.float32(0.015625)
    W[4] = -np.abs(W[4]) - np.float32(0.015625)
    W = I.bf16_representable(W)
    ng = Cin // group
    gl = rng.normal(2.0, 1.0, (Cout, ng)).astype(np.float32)
    bl = rng.normal(2.0, 1.0, (Cout, ng)).astype(np.float32)
    bl[0, 0] = gl[0, 0]                 # gamma = beta on the constant group: h = 0, floored
    gl[3:5], bl[3:5] = 4.0, 4.0         # one-signed groups with a positive range
    g = np.random.default_rng(42).standard_normal((Cout, Cin)).astype(np.float32)
    got = _lwc(W, gl, bl, nbits, group, g)
    f, b = _check_lwc("lwc degenerate groups", W, gl, bl, nbits, group, g, got)
    assert float(got["h"][0, 0]) == float(np.float32(1e-5)) and float(got["h"][1, 1]) == float(np.float32(1e-5))
    assert bool(f["st"]["floored"][0, 0]) and bool(f["st"]["floored"][1, 1])
    assert float(got["dgl"][0, 0]) == 0.0 and float(got["dgl"][1, 1]) == 0.0     # no gradient through h
    assert int(got["imax"][2, 0]) == 5 and int(got["imin"][2, 0]) == 7
    assert int(got["z"][3].max()) < 0 and int(got["z"][4].min()) > 2 ** nbits - 1


def test_exact_halves_round_to_even(cuda_lib):
    """Per-token rows with max = -min = 7.5 (h = 1, u = -7.5 exactly) and elements k + 1/2; a weight
    group of the same values scaled by 2^-7 with clipping strengths exactly 1 (logits 80)."""
    half = np.arange(-7, 8, dtype=np.float32) + np.float32(0.5)           # -6.5 .. 7.5
    row = np.concatenate([[-7.5], half, np.linspace(-7, 7, 16, dtype=np.float32)]).astype(np.float32)
    T, C = 4, row.size
    X = np.stack([row, row[::-1], row * np.float32(0.5), row * np.float32(2.0)]).astype(np.float32)
    cfg = _lib.make_cfg(abits=4)
    Xq = torch.empty(T, C, dtype=torch.bfloat16, device="cuda")
    codes = torch.empty(T, C, dtype=torch.uint8, device="cuda")
    h = torch.empty(T, device="cuda")
    z = torch.empty(T, dtype=torch.int32, device="cuda")
    imax, imin = torch.empty_like(z), torch.empty_like(z)
    _lib.omq_act_quant_per_token(T, C, _dev(X), None, None, Xq, codes, h, z, imax, imin, cfg)
    torch.cuda.synchronize()
    fa = O.act_quant_per_token(torch.from_numpy(X), 4)
    n = check_codes("act exact halves", torch.from_numpy(X).double() / h.cpu().double()[:, None], codes.cpu(), z.cpu(), 4)
    assert n["near_ties"] >= 3 * 15 and n["mismatches"] == 0
    assert torch.equal(codes.cpu().long(), fa["codes"])            # half to even on both sides
    assert torch.equal(z.cpu().double(), fa["z"]) and int(z[0]) == 8
    # weights: clipping strengths exactly 1, step exactly 2^-7
    Wrow = (np.concatenate([[-7.5], half, np.zeros(16, np.float32)]) * np.float32(2.0 ** -7)).astype(np.float32)
    W = np.stack([Wrow, Wrow[::-1]] * 4).astype(np.float32)
    gl = np.full((W.shape[0], 1), 80.0, np.float32)
    g = np.random.default_rng(3).standard_normal(W.shape).astype(np.float32)
    got = _lwc(W, gl, gl, 4, 0, g)
    assert bool((got["h"] == np.float32(2.0 ** -7)).all())
    f, _ = _check_lwc("lwc exact halves", W, gl, gl, 4, 0, g, got)
    assert torch.equal(got["codes"].long(), f["codes"]) and torch.equal(got["z"].double(), f["z"])


def test_constant_token_row(cuda_lib):
    """A constant activation row: range 0, h floored at eps, every element on one code."""
    rng = np.random.default_rng(5)
    T, C = 6, 512
    X = rng.standard_normal((T, C)).astype(np.float32)
    X[1] = np.float32(0.75)
    X[4] = 0.0
    cfg = _lib.make_cfg(abits=4)
    Xq = torch.empty(T, C, dtype=torch.bfloat16, device="cuda")
    codes = torch.empty(T, C, dtype=torch.uint8, device="cuda")
    h = torch.empty(T, device="cuda")
    z = torch.empty(T, dtype=torch.int32, device="cuda")
    imax, imin = torch.empty_like(z), torch.empty_like(z)
    Xd = _dev(X)
    _lib.omq_act_quant_per_token(T, C, Xd, None, None, Xq, codes, h, z, imax, imin, cfg)
    torch.cuda.synchronize()
    fa = O.act_quant_per_token(torch.from_numpy(X), 4)
    check_codes("act constant rows", torch.from_numpy(X).double() / h.cpu().double()[:, None], codes.cpu(), z.cpu(), 4)
    assert float(h[1]) == float(np.float32(1e-5)) and float(h[4]) == float(np.float32(1e-5))
    check_zero_points("act constant rows", fa["st"]["u"], z.cpu(), fa["z"])
    assert int(imax[1]) == 0 and int(imin[1]) == 0
    g = np.random.default_rng(6).standard_normal((T, C)).astype(np.float32)
    dX = torch.empty(T, C, device="cuda")
    ws = torch.empty(_lib.omq_act_bwd_workspace_size(T, C), dtype=torch.uint8, device="cuda")
    _lib.omq_act_quant_per_token_bwd(T, C, Xd, None, None, h, z, imax, imin, _dev(g), dX, None, None, ws, cfg)
    torch.cuda.synchronize()
    ba = O.act_quant_per_token_bwd(fa, torch.from_numpy(g))
    assert rel(dX.cpu(), ba["dX"]) < GRAD_TOL
    assert rel(dX.cpu()[[1, 4]], ba["dX"][[1, 4]]) < GRAD_TOL


def test_group_equal_to_row(cuda_lib):
    """group = Cin gives exactly the per-channel form (group = 0), and both match the oracle."""
    rng = np.random.default_rng(8)
    Cout, Cin = 64, 128
    W = _student(rng, (Cout, Cin))
    gl = rng.normal(2.0, 1.5, (Cout, 1)).astype(np.float32)
    bl = rng.normal(2.0, 1.5, (Cout, 1)).astype(np.float32)
    g = np.random.default_rng(9).standard_normal((Cout, Cin)).astype(np.float32)
    a = _lwc(W, gl, bl, 4, 0, g)
    b = _lwc(W, gl, bl, 4, Cin, g)
    for k in a:
        assert torch.equal(a[k], b[k]), k
    _check_lwc("lwc group = Cin", W, gl, bl, 4, Cin, g, b)


TOKENS = [1, 3, 127]


@pytest.mark.parametrize("T", TOKENS)
def test_block_step_token_counts(cuda_lib, T):
    shape = I.BlockShape(f"w4a4_let_T{T}", T=T, d=256, n_heads=2, n_kv=1, ffn=512, wbits=4, abits=4, group=0, let=1)
    W = I.make_block_weights(shape, seed=1)
    x = I.make_block_input(shape, sample=0, weight_seed=1)
    th = I.make_block_theta(shape, W, x, seed=2, perturb=True)
    cfg = O.BlockCfg.from_shape(shape)
    yfp = O.block_fp_forward(x, W, cfg).float()
    st = BlockState(shape, W, th)
    xd = torch.from_numpy(x).cuda()
    y = torch.empty_like(xd)
    st.step(xd, yfp.cuda(), y)
    torch.cuda.synchronize()
    assert int(st.status.item()) == 0
    sv = {k: ([t.cpu() for t in v] if isinstance(v, list) else v.cpu()) for k, v in st.saved().items()}
    grads = st.split_grads()
    compare_step(shape, W, x, th, yfp, y.cpu(), float(st.loss.item()), grads, sv, shape.name)
    ref = O.block_step(x, yfp, W, th, cfg)
    errs = dict(y=rel(y.cpu(), ref["y"]), loss=abs(float(st.loss.item()) - float(ref["loss"])) / float(ref["loss"]))
    errs.update(grad_errors(grads, ref, O.THETA_NAMES_LWC + O.THETA_NAMES_LET))
    record("end to end", shape.name, **errs)
    assert errs["y"] < OUT_TOL and errs["loss"] < OUT_TOL
