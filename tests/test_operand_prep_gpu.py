"""LWC fake quantization as GEMM operand preparation (Eq. 2 applied to each weight tile in shared
memory, omq_qcfg.wprep = 1) against the materialised path (the LWC forward writes W_hat to HBM and
the products read it).

Both paths feed the tensor cores the same bf16 operand values in the same order, so the forward
q|k|v product, the dX product that takes W_hat (dL/da = dY_qkv W_hat) and everything downstream
must agree bit for bit: output, loss, every gradient and every saved stage value.  The shapes
cover CTA pairs and single CTAs, per-channel and grouped weights, LET (row and column scales in
the prepared operand) and without, a ragged token count and a hidden size whose last k-block and
last dX column tile are partial.  The full 7B W4A4 block is the workload the step is timed on.
"""
import numpy as np
import pytest
import torch

from paper_2308_13137_gb300 import inputs as I
from paper_2308_13137_gb300.block import BlockState

pytestmark = pytest.mark.gpu

SHAPES = [
    I.BlockShape("w4a4_let", T=256, d=256, n_heads=2, n_kv=2, ffn=512, wbits=4, abits=4, group=0, let=1),
    I.BlockShape("w4a4_let_gqa", T=256, d=512, n_heads=4, n_kv=2, ffn=768, wbits=4, abits=4, group=0, let=1),
    I.BlockShape("w3a16_g128", T=256, d=256, n_heads=2, n_kv=2, ffn=512, wbits=3, abits=16, group=128, let=0),
    I.BlockShape("w2a16_g64", T=384, d=384, n_heads=3, n_kv=3, ffn=640, wbits=2, abits=16, group=64, let=0),
    I.BlockShape("w4a8_let_ragged", T=200, d=264, n_heads=2, n_kv=1, ffn=520, wbits=4, abits=8, group=0, let=1),
    I.BlockShape("w3a16_g128_let", T=128, d=384, n_heads=2, n_kv=2, ffn=512, wbits=3, abits=16, group=128, let=1),
    I.BlockShape("w4a4_let_mid", T=1024, d=1024, n_heads=8, n_kv=8, ffn=2816, wbits=4, abits=4, group=0, let=1),
]


def _step(shape, W, x, th, yfp, wprep):
    st = BlockState(shape, W, th, wprep=wprep)
    xd, yd = torch.from_numpy(x).cuda(), yfp.cuda()
    y = torch.empty_like(xd)
    st.step(xd, yd, y)
    torch.cuda.synchronize()
    assert int(st.status.item()) == 0
    sv = st.saved()
    saved = {k: ([None if t is None else t.cpu() for t in v] if isinstance(v, list) else v.cpu())
             for k, v in sv.items()}
    out = dict(y=y.cpu(), loss=st.loss.cpu(), grads={k: v.cpu() for k, v in st.grads.items()}, saved=saved)
    del st, sv
    torch.cuda.empty_cache()
    return out


def _same(a, b, what):
    assert a.dtype == b.dtype and a.shape == b.shape, what
    if not torch.equal(a.view(torch.uint8) if a.dtype == torch.bfloat16 else a, b.view(torch.uint8)
                       if b.dtype == torch.bfloat16 else b):
        d = (a.double() - b.double()).abs()
        raise AssertionError(f"{what}: {int((d > 0).sum())} elements differ, max |diff| {float(d.max()):.3e}")


def _compare(shape, seed=0):
    W = I.make_block_weights(shape, seed=seed + 1)
    x = I.make_block_input(shape, sample=seed, weight_seed=seed + 1)
    th = I.make_block_theta(shape, W, x, seed=seed + 2, perturb=True)
    yfp = torch.from_numpy(np.asarray(x, dtype=np.float32)) * 0.5      # any fixed target: both paths see the same
    ref = _step(shape, W, x, th, yfp, 0)
    got = _step(shape, W, x, th, yfp, 1)
    _same(got["y"], ref["y"], "y")
    _same(got["loss"], ref["loss"], "loss")
    for k in ref["grads"]:
        _same(got["grads"][k], ref["grads"][k], "d" + k)
    assert got["saved"]["w_hat"][0] is None and ref["saved"]["w_hat"][0] is not None
    for k, v in ref["saved"].items():
        if isinstance(v, list):
            for i in range(4):
                if got["saved"][k][i] is not None:
                    _same(got["saved"][k][i], v[i], f"{k}[{i}]")
        elif shape.abits < 16 or not k.endswith(("_h", "_z")):   # per-token quantizer state exists only with Q_a on
            _same(got["saved"][k], v, k)


@pytest.mark.parametrize("shape", SHAPES, ids=[s.name for s in SHAPES])
def test_operand_prep_bit_identical(cuda_lib, shape):
    _compare(shape)


@pytest.mark.full
def test_operand_prep_bit_identical_7b_w4a4(cuda_lib):
    _compare(I.block_shape("llama7b_w4a4"))
