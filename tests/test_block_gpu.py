"""Block-level parity: one calibration step through omq_block_step against the fp64 oracle
(every quantizer decision in float64, the normalised softmax, matmul operands rounded to bf16,
R13).  End to end from the block input: output and loss within 1e-2 relative, every gradient
within 3e-2 relative Frobenius error.  Stage-wise (`_stagewise`: each oracle stage started from
the GPU's stage input and output gradient) under the same bounds, with the code decisions of
every saved quantizer under the shared-scale protocol."""
import numpy as np
import pytest
import torch

import oracle as O
from _parity import grad_errors, record
from _stagewise import compare_step
from paper_2308_13137_gb300 import inputs as I
from paper_2308_13137_gb300.block import BlockState

pytestmark = pytest.mark.gpu
OUT_TOL, GRAD_TOL = 1e-2, 3e-2


def _rel(a, b):
    a, b = torch.as_tensor(a).double().cpu(), torch.as_tensor(b).double().cpu()
    return float((a - b).norm() / b.norm().clamp_min(1e-300))


def _run(shape, perturb=True, seed=0, pbits=16, run_cuda=True):
    W = I.make_block_weights(shape, seed=seed + 1)
    x = I.make_block_input(shape, sample=seed, weight_seed=seed + 1)
    th = I.make_block_theta(shape, W, x, seed=seed + 2, perturb=perturb)
    cfg = O.BlockCfg.from_shape(shape, pbits=pbits)
    yfp = O.block_fp_forward(x, W, O.BlockCfg.from_shape(shape)).float()
    ref = O.block_step(x, yfp, W, th, cfg)
    if not run_cuda:
        return ref, None
    st = BlockState(shape, W, th, pbits=pbits)
    xd, yfd = torch.from_numpy(x).cuda(), yfp.cuda()
    y = torch.empty_like(xd)
    st.step(xd, yfd, y)
    torch.cuda.synchronize()
    assert int(st.status.item()) == 0
    got = dict(y=y.cpu(), loss=float(st.loss.item()), **st.split_grads())
    sv = st.saved()
    got["saved"] = {k: ([t.cpu() for t in v] if isinstance(v, list) else v.cpu()) for k, v in sv.items()}
    got["inputs"] = (W, x, th, yfp)
    return ref, got


SMALL = [
    I.BlockShape("w4a4_let", T=256, d=256, n_heads=2, n_kv=2, ffn=512, wbits=4, abits=4, group=0, let=1),
    I.BlockShape("w4a4_let_gqa", T=256, d=512, n_heads=4, n_kv=2, ffn=768, wbits=4, abits=4, group=0, let=1),
    I.BlockShape("w3a16_g128", T=256, d=256, n_heads=2, n_kv=2, ffn=512, wbits=3, abits=16, group=128, let=0),
    I.BlockShape("w2a16_g64", T=384, d=384, n_heads=3, n_kv=3, ffn=640, wbits=2, abits=16, group=64, let=0),
    I.BlockShape("w4a8_let_ragged", T=200, d=256, n_heads=2, n_kv=1, ffn=520, wbits=4, abits=8, group=0, let=1),
    # the other weight-activation settings the paper reports: W6A6 (its main weight-activation results) and the asymmetric
    # W4A6, W8A4 of its asymmetric-bits table (W4A8 above)
    I.BlockShape("w4a6_let", T=256, d=256, n_heads=2, n_kv=2, ffn=512, wbits=4, abits=6, group=0, let=1),
    I.BlockShape("w6a6_let", T=256, d=256, n_heads=2, n_kv=2, ffn=512, wbits=6, abits=6, group=0, let=1),
    I.BlockShape("w8a4_let", T=256, d=256, n_heads=2, n_kv=2, ffn=512, wbits=8, abits=4, group=0, let=1),
    # mid-size blocks (T = d = 1024): every product spans tens of 256 x 256 tiles and at least 16 k-blocks,
    # including the weight-gradient products with the LWC backward fused in their epilogue (per channel with LET,
    # and grouped)
    I.BlockShape("w4a4_let_mid", T=1024, d=1024, n_heads=8, n_kv=8, ffn=2816, wbits=4, abits=4, group=0, let=1),
    I.BlockShape("w3a16_g128_mid", T=1024, d=1024, n_heads=8, n_kv=4, ffn=2816, wbits=3, abits=16, group=128, let=0),
]


@pytest.mark.parametrize("shape", SMALL, ids=[s.name for s in SMALL])
def test_block_step_small(cuda_lib, shape):
    ref, got = _run(shape)
    W, x, th, yfp = got["inputs"]
    grads = {k: v for k, v in got.items() if k.startswith("d")}
    compare_step(shape, W, x, th, yfp, got["y"], got["loss"], grads, got["saved"], shape.name)
    errs = dict(y=_rel(got["y"], ref["y"]), loss=abs(got["loss"] - float(ref["loss"])) / float(ref["loss"]))
    names = O.THETA_NAMES_LWC + (O.THETA_NAMES_LET if shape.let else [])
    errs.update(grad_errors(got, ref, names))
    record("end to end", shape.name, **errs)
    assert errs["y"] < OUT_TOL and errs["loss"] < OUT_TOL, errs
    if shape.abits >= 16:
        # weight-only: the step is continuous in its input between weight-code ties, so the
        # end-to-end gradients meet the bound as well; with quantized activations a per-token code
        # that flips near a half moves the later stages, and the gradients are held stage-wise
        bad = {n: errs["d" + n] for n in names if not errs["d" + n] < GRAD_TOL}
        assert not bad, bad


# softmax-output quantization (the ablation beside Table A7: W4A4 with the softmax output at 8, 6
# and 4 bits), per query row over the visible keys
PQ_CASES = [
    (I.BlockShape("w4a4_let_p8", T=256, d=256, n_heads=2, n_kv=2, ffn=512, wbits=4, abits=4, group=0, let=1), 8),
    (I.BlockShape("w4a4_let_gqa_p6", T=256, d=512, n_heads=4, n_kv=2, ffn=768, wbits=4, abits=4, group=0, let=1), 6),
    (I.BlockShape("w4a4_let_ragged_p4", T=200, d=256, n_heads=2, n_kv=1, ffn=520, wbits=4, abits=4, group=0, let=1), 4),
    (I.BlockShape("w4a4_let_p2", T=256, d=256, n_heads=2, n_kv=2, ffn=512, wbits=4, abits=4, group=0, let=1), 2),
]


@pytest.mark.parametrize("shape,pbits", PQ_CASES, ids=[s.name for s, _ in PQ_CASES])
def test_block_step_softmax_quant(cuda_lib, shape, pbits):
    ref, got = _run(shape, pbits=pbits)
    W, x, th, yfp = got["inputs"]
    grads = {k: v for k, v in got.items() if k.startswith("d")}
    compare_step(shape, W, x, th, yfp, got["y"], got["loss"], grads, got["saved"], f"{shape.name} softmax {pbits} bits",
                 pbits=pbits)
    names = O.THETA_NAMES_LWC + O.THETA_NAMES_LET
    errs = dict(y=_rel(got["y"], ref["y"]), loss=abs(got["loss"] - float(ref["loss"])) / float(ref["loss"]))
    errs.update(grad_errors(got, ref, names))
    record("end to end", f"{shape.name} softmax {pbits} bits", **errs)
    assert errs["y"] < OUT_TOL and errs["loss"] < OUT_TOL, errs
    if pbits == 2:
        # the quantizer is really in the path: at 2 bits the s_a gradient moves by ~15% between the
        # quantized and the unquantized softmax; the kernels must sit much closer to the former
        ref0, _ = _run(shape, pbits=16, run_cuda=False)
        assert _rel(got["dsa"], ref["dsa"]) < 0.25 * _rel(ref0["dsa"], ref["dsa"])
