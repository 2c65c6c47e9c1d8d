"""Fold & pack on the GPU (omq_block_fold_pack through BlockState.fold_pack) against the oracle's
block_fold_pack (Algorithm 1's transform-then-quantize; reading R17) on the same seeded block:
the packed codes unpacked by the oracle's own bit layout and compared under the shared-scale
protocol (round of the fp32 quantizer input over the GPU's h, plus its z; exempt elements
counted), z against the oracle's float64 decision, h within 1e-6 of the oracle, biases and folded
RMSNorm vectors to fp32 accuracy, s_a copied."""
import numpy as np
import pytest
import torch

import oracle as O
from _parity import check_codes, check_h, check_zero_points
from _stagewise import weight_inputs_fp32
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
    cfg = O.BlockCfg.from_shape(shape)
    Q = 2 ** shape.wbits - 1
    exact = weight_inputs_fp32(shape, W, th, torch.float64)
    for i, (k, Wl) in enumerate(zip(("qkv", "o", "gu", "d"), weight_inputs_fp32(shape, W, th))):
        cout, cin = Wl.shape
        g = cin if shape.group == 0 else shape.group
        hg, zg = got["h_" + k].cpu(), got["z_" + k].cpu()
        codes = O.unpack_codes(got["codes_" + k].cpu(), shape.wbits, cin).reshape(cout, cin // g, g)
        tag = f"fold&pack {shape.name} {k}"
        check_codes(tag, Wl.double().reshape(cout, cin // g, g) / hg.double()[..., None], codes, zg, shape.wbits)
        parts = dict(qkv=("q", "k", "v"), o=("o",), gu=("g", "u"), d=("d",))[k]
        gl = torch.cat([torch.as_tensor(th["gamma_" + p_]) for p_ in parts]).double()
        bl = torch.cat([torch.as_tensor(th["beta_" + p_]) for p_ in parts]).double()
        a, b = O.sigmoid(gl), O.sigmoid(bl)
        G = exact[i].reshape(cout, cin // g, g)
        check_h(tag, hg, ref["h_" + k], a * G.max(-1).values, b * G.min(-1).values, Q)
        check_zero_points(tag, b * G.min(-1).values / ref["h_" + k], zg, ref["z_" + k])
        assert torch.allclose(ref["h_" + k], torch.clamp((a * G.max(-1).values - b * G.min(-1).values) / Q, min=1e-5),
                              rtol=1e-14, atol=0)
    if shape.let:
        for k in ("b_qkv", "b_o", "b_gu"):
            assert _rel(got[k], ref[k]) < 1e-5, k
        for k in ("ln1_gain", "ln1_bias", "ln2_gain", "ln2_bias"):
            assert _rel(got[k], ref[k]) < 1e-6, k
        assert torch.equal(got["sa"].cpu(), torch.as_tensor(th["sa"]))
