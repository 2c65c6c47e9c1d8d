"""The N > 1 path of bench.py without a GPU: two gloo ranks on 127.0.0.1 read their rank from the
environment the way torchrun sets it, take the slowest rank's time with the same MAX reduction the
bench applies to its CUDA-event times, and get distinct block replicas; the reference arm leaves
every rank but 0 without work.  The path is replicas only: the ranks exchange nothing but the
timing."""
import os
import socket
import sys

import numpy as np
import pytest
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, ws, port, q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(ws),
                      LOCAL_RANK=str(rank))
    sys.path.insert(0, ROOT)
    import torch.distributed as dist
    import bench
    dist.init_process_group("gloo", rank=rank, world_size=ws)
    wsz, r, local = bench._dist()
    slowest = bench.max_over_ranks(10.0 + 5.0 * r, wsz, "cpu")      # rank r took 10 + 5 r ms
    ref = bench.run_reference(None, None) if r != 0 else None        # returns before touching its args
    dist.barrier()
    dist.destroy_process_group()
    q.put((r, wsz, local, slowest, bench.replica_seeds(r), ref))


def test_two_gloo_ranks():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    out = sorted(q.get(timeout=120) for _ in procs)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    assert [o[0] for o in out] == [0, 1] and all(o[1] == 2 for o in out) and [o[2] for o in out] == [0, 1]
    assert all(o[3] == 15.0 for o in out)                           # both ranks see the slowest time
    assert out[0][4] != out[1][4]                                   # distinct replicas
    assert out[1][5] == 0                                           # reference arm: rank 1 does no work


def test_job_throughput_and_replicas():
    sys.path.insert(0, ROOT)
    import bench
    from paper_2308_13137_gb300 import inputs as I
    # whole-job tokens/s: all ranks' tokens over the slowest rank's seconds
    assert bench.job_throughput(2, 2048, 10, 0.015) == pytest.approx(2 * 2048 * 10 / 0.015)
    assert bench.max_over_ranks(3.5, 1, "cpu") == 3.5
    shape = I.BlockShape("tiny", T=64, d=128, n_heads=1, n_kv=1, ffn=256, wbits=4, abits=4, group=0, let=1)
    w0 = I.make_block_weights(shape, seed=bench.replica_seeds(0)["weights"])
    w1 = I.make_block_weights(shape, seed=bench.replica_seeds(1)["weights"])
    assert w0.keys() == w1.keys()
    assert all(w0[k].shape == w1[k].shape and not np.array_equal(w0[k], w1[k]) for k in w0)


def test_oracle_baseline_pieces_are_one_block_step():
    """The CPU baseline times the oracle's step cut into eleven pieces (five forward stages, the loss,
    five stage backwards); one pass over them must be exactly the oracle's block_step: same loss,
    same gradient of every parameter."""
    import torch
    import bench
    import oracle as O
    from paper_2308_13137_gb300 import inputs as I
    shape = I.BlockShape("tiny", T=16, d=64, n_heads=2, n_kv=1, ffn=96, wbits=4, abits=4, group=0, let=1,
                         head_dim=32)
    W = I.make_block_weights(shape, seed=1)
    x = I.make_block_input(shape, sample=0, weight_seed=1)
    th = I.make_block_theta(shape, W, x, seed=2, perturb=True)
    yfp = bench._oracle_yfp(shape, W, x)
    out = {}
    it = bench._oracle_pieces(shape, W, th, x, yfp, out)
    names = [next(it)[0] for _ in bench.PIECES]
    assert names == bench.PIECES
    ref = O.block_step(x, yfp, W, th, O.BlockCfg.from_shape(shape))
    assert abs(float(out["loss"]) - float(ref["loss"])) <= 1e-12 * float(ref["loss"])
    for n in O.THETA_NAMES_LWC + O.THETA_NAMES_LET:
        assert torch.allclose(out["d" + n], ref["d" + n], rtol=1e-9, atol=1e-15), n
