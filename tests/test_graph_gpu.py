"""The calibration step replayed from a CUDA graph (BlockState.step_adamw_graph) gives the results of
the same step launched directly (step + adamw) over several steps and two input samples: the same
launches run in the same order.  The only reduction without a fixed order is the routing of the
LET column gradient ds to each weight row's max/min column (float atomics, Eq. 2's max/min path),
so values agree to rounding, not bit for bit."""
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
    for la, lb in zip(losses_a, losses_b):
        assert abs(la - lb) <= 1e-6 * abs(la)
    assert int(a.adam_step_dev.item()) == int(b.adam_step_dev.item()) == 5
    rel = lambda u, w: float((u.double() - w.double()).norm() / w.double().norm().clamp_min(1e-30))
    for g in a.theta_flat:
        assert rel(b.theta_flat[g], a.theta_flat[g]) < 1e-5
        assert rel(b.adam[g][0], a.adam[g][0]) < 1e-3 and rel(b.adam[g][1], a.adam[g][1]) < 1e-3
