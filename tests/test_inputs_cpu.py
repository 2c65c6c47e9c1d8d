"""The seeded input module that feeds both the CUDA path and the oracle: deterministic in its
seeds and independent of any global random state, weights stored as bf16 values (checked against
PyTorch's own bf16 conversion), the block input's outlier channels shared by every sample of a
block, and the documented shapes."""
import numpy as np
import torch

from paper_2308_13137_gb300 import inputs as I

SMALL = I.BlockShape("tiny", T=64, d=256, n_heads=2, n_kv=1, ffn=384, wbits=4, abits=4, group=0, let=1)


def test_seeded_and_independent_of_global_state():
    np.random.seed(1)
    torch.manual_seed(1)
    a = I.make_block_weights(SMALL, seed=5)
    np.random.seed(2)
    torch.manual_seed(2)
    b = I.make_block_weights(SMALL, seed=5)
    c = I.make_block_weights(SMALL, seed=6)
    for k in a:
        assert np.array_equal(a[k], b[k])
        assert not np.array_equal(a[k], c[k])
    x0 = I.make_block_input(SMALL, sample=0, weight_seed=5)
    assert np.array_equal(x0, I.make_block_input(SMALL, sample=0, weight_seed=5))
    assert not np.array_equal(x0, I.make_block_input(SMALL, sample=1, weight_seed=5))
    t0 = I.make_block_theta(SMALL, a, x0, seed=2, perturb=True)
    t1 = I.make_block_theta(SMALL, a, x0, seed=2, perturb=True)
    assert t0.keys() == t1.keys() and all(np.array_equal(t0[k], t1[k]) for k in t0)


def test_bf16_storage_matches_torch_rounding():
    rng = np.random.default_rng(3)
    v = (rng.standard_normal(4096) * 10.0 ** rng.integers(-4, 4, 4096)).astype(np.float32)
    got = I.bf16_representable(v)
    want = torch.from_numpy(v).to(torch.bfloat16).float().numpy()
    assert np.array_equal(got, want)
    W = I.make_block_weights(SMALL, seed=1)
    for k, w in W.items():
        assert w.dtype == np.float32 and not (w.view(np.uint32) & np.uint32(0xFFFF)).any(), k


def test_block_shapes_and_outlier_channels():
    W = I.make_block_weights(SMALL, seed=1)
    d, dq, dkv, f = SMALL.d, SMALL.dq, SMALL.dkv, SMALL.ffn
    assert {k: v.shape for k, v in W.items()} == dict(wq=(dq, d), wk=(dkv, d), wv=(dkv, d), wo=(d, dq),
                                                      wg=(f, d), wu=(f, d), wd=(d, f))
    xs = [I.make_block_input(SMALL, sample=s, weight_seed=1) for s in range(3)]
    n_out = int(round(SMALL.outlier_frac * d))
    big = [set(np.argsort(-np.abs(x).mean(0))[:n_out]) for x in xs]
    assert n_out >= 1 and big[0] == big[1] == big[2]          # the same channels in every sample
    x = xs[0]
    ch = sorted(big[0])
    rest = np.setdiff1d(np.arange(d), ch)
    assert np.abs(x[:, ch]).mean() > 0.5 * SMALL.outlier_scale * np.abs(x[:, rest]).mean()
    full = I.block_shape("llama7b_w4a4")
    assert (full.T, full.d, full.n_heads, full.n_kv, full.head_dim, full.ffn) == (2048, 4096, 32, 32, 128, 11008)
    assert (full.wbits, full.abits, full.group, full.let) == (4, 4, 0, 1)
