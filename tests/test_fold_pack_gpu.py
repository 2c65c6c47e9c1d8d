"""Fold & pack on the GPU (omq_block_fold_pack through BlockState.fold_pack) against the oracle's
block_fold_pack (Algorithm 1's transform-then-quantize; reading R17) on the same seeded block:
packed codes and zero points bit-exact (decisions in fp32 on both sides, R15), h equal, biases
and folded RMSNorm vectors to fp32 accuracy, s_a copied."""
import numpy as np
import pytest
import torch

import oracle as O
from paper_2308_13137_gb300 import inputs as I
from paper_2308_13137_gb300.block import BlockState

pytestmark = pytest.mark.gpu

SHAPES = [
    I.BlockShape("pack_w4a4_let", T=128, d=256, n_heads=2, n_kv=2, ffn=512, wbits=4, abits=4, group=0, let=1),
    I.BlockShape("pack_w4a4_gqa", T=128, d=512, n_heads=4, n_kv=2, ffn=768, wbits=4, abits=4, group=0, let=1),
    I.BlockShape("pack_w3a16_g128", T=128, d=256, n_heads=2, n_kv=2, ffn=512, wbits=3, abits=16, group=128, let=0),
    I.BlockShape("pack_w2a16_g64", T=128, d=384, n_heads=3, n_kv=3, ffn=640, wbits=2, abits=16, group=64, let=0),
]


def _rel(a, b):
    a, b = torch.as_tensor(a).double().cpu(), torch.as_tensor(b).double().cpu()
    return float((a - b).norm() / b.norm().clamp_min(1e-300))


@pytest.mark.parametrize("shape", SHAPES, ids=[s.name for s in SHAPES])
def test_fold_pack_matches_oracle(cuda_lib, shape):
    W = I.make_block_weights(shape, seed=1)
    x = I.make_block_input(shape, sample=0, weight_seed=1)
    th = I.make_block_theta(shape, W, x, seed=2, perturb=True)
    ref = O.block_fold_pack(W, th, O.BlockCfg.from_shape(shape))
    st = BlockState(shape, W, th)
    got = st.fold_pack()
    torch.cuda.synchronize()
    for k in ("qkv", "o", "gu", "d"):
        assert torch.equal(got["codes_" + k].cpu(), ref["codes_" + k]), k
        assert torch.equal(got["z_" + k].cpu().double(), ref["z_" + k]), k
        assert torch.equal(got["h_" + k].cpu().double(), ref["h_" + k]), k
    if shape.let:
        for k in ("b_qkv", "b_o", "b_gu"):
            assert _rel(got[k], ref[k]) < 1e-5, k
        for k in ("ln1_gain", "ln1_bias", "ln2_gain", "ln2_bias"):
            assert _rel(got[k], ref[k]) < 1e-6, k
        assert torch.equal(got["sa"].cpu(), torch.as_tensor(th["sa"]))
