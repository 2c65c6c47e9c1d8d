"""Algorithm 1 over a stack of blocks on the GPU (paper_2308_13137_gb300.calibrate) against the
oracle's calibrate_blocks (Sec. 4.1 "Training"; readings R16, R18), and block-granular resume:
an interrupted run continued from its checkpoints ends where the uninterrupted run ends."""
import numpy as np
import pytest
import torch

import oracle as O
from paper_2308_13137_gb300 import inputs as I
from paper_2308_13137_gb300.calibrate import calibrate_blocks

pytestmark = pytest.mark.gpu

SHAPE = I.BlockShape("calib_w4a4_gqa", T=128, d=256, n_heads=4, n_kv=2, ffn=512, wbits=4, abits=4, group=0, let=1)
SHAPE_LWC = I.BlockShape("calib_w3a16_g64", T=128, d=256, n_heads=2, n_kv=2, ffn=512, wbits=3, abits=16, group=64,
                         let=0)


def _rel(a, b):
    a, b = torch.as_tensor(a).double().cpu(), torch.as_tensor(b).double().cpu()
    return float((a - b).norm() / b.norm().clamp_min(1e-300))


def _stack(shape=SHAPE, n=3):
    blocks = [I.make_block_weights(shape, seed=1 + 10 * i) for i in range(n)]
    xs = [I.make_block_input(shape, sample=i, weight_seed=1) for i in range(2)]
    th0 = I.make_block_theta(shape, blocks[0], xs[0], seed=2)
    return blocks, xs, th0


def test_calibration_matches_oracle_lwc_only(cuda_lib):
    """Weight-only W3A16 g64: after two blocks of two epochs every parameter, X_fp and X_q agree."""
    blocks, xs, th0 = _stack(SHAPE_LWC, 2)
    params, packed, x_fp, x_q = calibrate_blocks(SHAPE_LWC, blocks, xs, th0, epochs=2)
    ref_params, ref_fp, ref_q = O.calibrate_blocks(blocks, xs, O.BlockCfg.from_shape(SHAPE_LWC), th0, epochs=2)
    for got, ref in zip(x_fp + x_q, ref_fp + ref_q):
        assert _rel(got, ref) < 1e-2
    for b in range(2):
        for k, v in ref_params[b].items():
            assert _rel(params[b][k], v) < 1e-2, (b, k)
    assert packed[1]["codes_qkv"].dtype == torch.uint8


def test_calibration_matches_oracle_let(cuda_lib):
    """W4A4 with LET: the block outputs X_fp, X_q and the LWC logits agree.  The LET vectors are
    bounded instead: Adam moves a component by about lr per step whatever the gradient's size, so
    components whose gradients are near zero (their sign set by 4-bit decision noise) may walk in
    opposite directions on the two sides; no component may differ by more than 2 lr per step."""
    blocks, xs, th0 = _stack(SHAPE, 2)
    epochs, lr_let = 2, 1e-2
    params, packed, x_fp, x_q = calibrate_blocks(SHAPE, blocks, xs, th0, epochs=epochs, lr_let=lr_let)
    ref_params, ref_fp, ref_q = O.calibrate_blocks(blocks, xs, O.BlockCfg.from_shape(SHAPE), th0, epochs=epochs,
                                                   lr_let=lr_let)
    for got, ref in zip(x_fp + x_q, ref_fp + ref_q):
        assert _rel(got, ref) < 1e-2
    steps = epochs * len(xs)
    for b in range(2):
        for k, v in ref_params[b].items():
            if k in O.THETA_NAMES_LET:
                assert float((params[b][k].double() - v).abs().max()) <= 2 * lr_let * steps, (b, k)
            else:
                assert _rel(params[b][k], v) < 1e-2, (b, k)


def test_calibration_resumes_from_checkpoints(cuda_lib, tmp_path):
    blocks, xs, th0 = _stack()
    full = calibrate_blocks(SHAPE, blocks, xs, th0, epochs=1)
    ck = str(tmp_path / "ck")
    part = calibrate_blocks(SHAPE, blocks, xs, th0, epochs=1, ckpt_dir=ck, stop_after=1)
    assert len(part[0]) == 1
    resumed = calibrate_blocks(SHAPE, blocks, xs, th0, epochs=1, ckpt_dir=ck)
    assert len(resumed[0]) == 3
    for a, b in zip(full[3], resumed[3]):
        assert _rel(a, b) < 1e-4
    for b in range(3):
        for k in full[0][b]:
            assert _rel(resumed[0][b][k], full[0][b][k]) < 1e-4, (b, k)
