"""The calibration step replayed from a CUDA graph (BlockState.step_adamw_graph) gives the results of
the same step launched directly (step + adamw) over several steps and two input samples, bit for
bit: the same launches run in the same order and every reduction of the step has a fixed order
(no floating-point atomics), so the step is deterministic."""
import pytest
import torch

from paper_2308_13137_gb300 import inputs as I
from paper_2308_13137_gb300.block import BlockState

pytestmark = pytest.mark.gpu


def test_graph_replay_equals_direct_steps(cuda_lib):
    shape = I.BlockShape("w4a4_let_graph", T=256, d=512, n_heads=4, n_kv=2, ffn=768, wbits=4, abits=4, group=0, let=1)
    W = I.make_block_weights(shape, seed=1)
    xs = [I.make_block_input(shape, sample=i, weight_seed=1) for i in range(2)]
    th = I.make_block_theta(shape, W, xs[0], seed=2, perturb=True)
    a, b = BlockState(shape, W, th), BlockState(shape, W, th)
    xd = [torch.from_numpy(x).cuda() for x in xs]
    yfp = [torch.empty_like(v) for v in xd]
    for v, y in zip(xd, yfp):
        a.fp_forward(v, y)
    losses_a, losses_b = [], []
    for i in range(5):
        a.step(xd[i % 2], yfp[i % 2])
        a.adamw()
        losses_a.append(float(a.loss.item()))
        b.step_adamw_graph(xd[i % 2], yfp[i % 2])
        losses_b.append(float(b.loss.item()))
    torch.cuda.synchronize()
    assert int(a.status.item()) == 0 and int(b.status.item()) == 0
    assert losses_a == losses_b
    assert int(a.adam_step_dev.item()) == int(b.adam_step_dev.item()) == 5
    for g in a.theta_flat:
        assert torch.equal(b.theta_flat[g], a.theta_flat[g])
        assert torch.equal(b.adam[g][0], a.adam[g][0]) and torch.equal(b.adam[g][1], a.adam[g][1])


def test_step_is_deterministic(cuda_lib):
    """Two blocks stepped on the same input give identical gradients (the LET column gradients include
    the max / min routing of every weight row)."""
    shape = I.BlockShape("w4a4_let_det", T=256, d=512, n_heads=4, n_kv=2, ffn=768, wbits=4, abits=4, group=0, let=1)
    W = I.make_block_weights(shape, seed=3)
    x = I.make_block_input(shape, sample=0, weight_seed=3)
    th = I.make_block_theta(shape, W, x, seed=4, perturb=True)
    a, b = BlockState(shape, W, th), BlockState(shape, W, th)
    xd = torch.from_numpy(x).cuda()
    yfp = torch.empty_like(xd)
    a.fp_forward(xd, yfp)
    a.step(xd, yfp)
    b.step(xd, yfp)
    torch.cuda.synchronize()
    for g in a.grads_flat:
        assert torch.equal(a.grads_flat[g], b.grads_flat[g])
