#!/usr/bin/env python3
"""Throughput of one OmniQuant block-calibration step on GB300.

A step is one iteration of Algorithm 1's inner loop on one calibration sample: LET + LWC on the
block's weights, the quantized block forward on 2048 tokens, the MSE loss against the
full-precision block output, the straight-through backward to every learnable parameter, and
the AdamW update.  Metric: calibration tokens per second per block (whole job over N GPUs).

Default workload: the LLaMA-7B decoder block at W4A4 (per-channel weights, per-token activations)
with LWC + LET, 2048 tokens per step; synthetic seeded weights and activations.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--config NAME] [--impl ours|reference]

With N > 1 (launched by torch.distributed.run) every rank calibrates its own block replica; the
path has no data exchange ("replicas only"), so no collective runs inside the step.
"""
from __future__ import annotations

import argparse
import json
import math
import os
import statistics
import subprocess
import sys
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

METRIC = "calibration tokens/sec per block (fwd+bwd, fused LWC+LET) and % of step roofline"
UNIT = "tokens/s"
DEFAULT_CONFIG = "llama7b_w4a4"


def _peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as fh:
            d = json.load(fh)
        return dict(hbm=float(d["hbm_gbs"]), bf16=float(d["bf16_tflops"]),
                    bf16_sus=float(d.get("bf16_tflops_sustained", d["bf16_tflops"])), src="measured")
    except Exception:
        return dict(hbm=6800.0, bf16=1900.0, bf16_sus=1700.0, src="fallback")


def _dist():
    ws = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return ws, rank, local


def replica_seeds(rank: int):
    """Seeds of rank `rank`'s block replica: every rank calibrates its own block (distinct weights,
    same shapes), so the ranks share no data and exchange nothing but the timing."""
    return {"weights": 1 + rank, "theta": 2 + rank}


def max_over_ranks(value: float, ws: int, device) -> float:
    """The largest of every rank's `value` (the slowest rank's time); the value itself alone."""
    import torch
    t = torch.tensor([float(value)], dtype=torch.float64, device=device)
    if ws > 1:
        torch.distributed.all_reduce(t, op=torch.distributed.ReduceOp.MAX)
    return float(t.item())


def job_throughput(ws: int, tokens_per_step: int, steps: int, seconds: float) -> float:
    """Whole-job tokens per second: all ranks' tokens over the slowest rank's time (weak scaling)."""
    return ws * tokens_per_step * steps / seconds


# ------------------------------------------------------------------------------------------------
# clocks during the timed region
# ------------------------------------------------------------------------------------------------
class ClockSampler:
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.proc = None

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.gpu), f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                 "-lms", "100"], stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except Exception:
            self.proc = None

    def stop(self):
        if self.proc is None:
            return dict(sm_mhz=None, sm_max_mhz=None, reasons=["nvidia-smi unavailable"], samples=0)
        self.proc.terminate()
        try:
            out, _ = self.proc.communicate(timeout=5)
        except Exception:
            self.proc.kill()
            out, _ = self.proc.communicate()
        sm, smax, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in out.strip().splitlines():
            f = [x.strip() for x in line.split(",")]
            if len(f) < 9:
                continue
            try:
                sm.append(float(f[1]))
                smax.append(float(f[2]))
            except ValueError:
                continue
            for n, v in zip(names, f[5:9]):
                if v.lower() in ("active", "1", "0x1"):
                    reasons.add(n)
        return dict(sm_mhz=statistics.median(sm) if sm else None, sm_max_mhz=max(smax) if smax else None,
                    reasons=sorted(reasons), samples=len(sm))


# ------------------------------------------------------------------------------------------------
# the oracle on host cores: bounded samples of the same workload
# ------------------------------------------------------------------------------------------------
def _oracle_sampler(shape, W, th, x):
    """Yields (seconds, block-equivalent seconds) per sample.  A sample is one oracle calibration
    step (Eq. 4 quantized linear, LWC + LET where the block has them, MSE to the fp output, STE
    gradients) of a 128-output-channel slice of one of the block's seven projections, at the full
    token count, cycling q, k, v, o, gate, up, down; its time is scaled by Cout/128 to the whole
    projection.  Attention and the norms (about 4% of the step's flops) are not sampled."""
    import numpy as np
    import torch
    import oracle as O
    torch.manual_seed(0)
    T, d, f = shape.T, shape.d, shape.ffn
    x64 = torch.from_numpy(x).double()
    a = x64 / torch.sqrt((x64 * x64).mean(-1, keepdim=True) + shape.rms_eps)
    rng = np.random.default_rng(5)
    m_in = torch.from_numpy(rng.standard_normal((T, f)).astype(np.float32)).double()
    let = bool(shape.let)
    lin = [("q", "wq", a, "s1", "d1"), ("k", "wk", a, "s1", "d1"), ("v", "wv", a, "s1", "d1"),
           ("o", "wo", x64, None, None), ("g", "wg", a, "s2", "d2"), ("u", "wu", a, "s2", "d2"),
           ("d", "wd", m_in, None, None)]
    rows = 128
    i = 0
    while True:
        name, wn, X, sn, dn = lin[i % 7]
        Wfull = torch.from_numpy(W[wn])
        Wsl = Wfull[:rows]
        gl = torch.from_numpy(th["gamma_" + name][:rows])
        bl = torch.from_numpy(th["beta_" + name][:rows])
        s = torch.from_numpy(th[sn]) if (let and sn) else None
        dl = torch.from_numpy(th[dn]) if (let and dn) else None
        yfp = X @ Wsl.double().T
        t0 = time.perf_counter()
        O.qlinear_step(X, Wsl, None, gl, bl, yfp, shape.wbits, shape.group, shape.abits, s=s, delta=dl,
                       mode="emulate")
        dt = time.perf_counter() - t0
        yield dt, dt * Wfull.shape[0] / rows
        i += 1


def _oracle_value(shape, W, th, x, n_samples):
    import torch
    it = _oracle_sampler(shape, W, th, x)
    wall, eq = 0.0, 0.0
    for _ in range(n_samples):
        a, b = next(it)
        wall += a
        eq += b
    cycles = n_samples / 7.0
    return shape.T * cycles / eq, wall, torch.get_num_threads()


def run_reference(args, shape):
    ws, rank, _ = _dist()
    if rank != 0:
        return 0
    import numpy as np
    from paper_2308_13137_gb300 import inputs as I
    W = I.make_block_weights(shape, seed=1)
    x = I.make_block_input(shape, 0, 1)
    th = I.make_block_theta(shape, W, x, seed=2)
    it = _oracle_sampler(shape, W, th, x)
    for _ in range(args.warmup):
        next(it)
    t0 = time.perf_counter()
    eq = 0.0
    for _ in range(args.steps):
        eq += next(it)[1]
    wall = time.perf_counter() - t0
    import torch
    value = shape.T * (args.steps / 7.0) / eq
    sample = ("each step: one fp64 oracle calibration step of a 128-output-channel slice of one block "
              "projection (cycling q,k,v,o,gate,up,down) at %d tokens; value scales each slice's time by "
              "Cout/128 to whole projections (attention and norms not sampled)" % shape.T)
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": ws, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": 1e3 * wall / args.steps, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": {"workload": shape.name, "tokens_per_step": shape.T, "wbits": shape.wbits,
                       "abits": shape.abits, "group": shape.group, "let": shape.let},
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": torch.get_num_threads(), "kind": "oracle",
                             "sample": sample},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)
    return 0


# ------------------------------------------------------------------------------------------------
# the GPU path
# ------------------------------------------------------------------------------------------------
def algorithmic_bytes(shape) -> float:
    """HBM bytes a fully fused step must move: every bf16 weight read three times (forward operand
    preparation, input-gradient operand, weight-gradient epilogue), plus one more stats pass for
    per-channel groups; the saved activations written once and read once; activation gradients the
    same; fp32 block input, target, output and residual streams."""
    T, d, f, dq, dkv = shape.T, shape.d, shape.ffn, shape.dq, shape.dkv
    P = d * (dq + 2 * dkv) + d * dq + 3 * d * f
    w_reads = (4 if shape.group == 0 else 3) * 2 * P
    acts = T * (d + (dq + 2 * dkv) + dq + d + 2 * f + f) * 2          # bf16 GEMM operands saved
    grads = acts
    streams = T * d * 4 * 6
    return float(w_reads + 2 * acts + 2 * grads + streams)


def algorithmic_flops(shape) -> float:
    """Flops of one step counted from the method, not from the launches: each linear's forward and
    weight-gradient product (2 T P each), the input-gradient products (q|k|v only when LET needs
    them), and the causal attention, lower triangle only: Q K^T and P V forward (2 * 128 H T (T+1))
    and twice that backward."""
    T, d, f, dq, dkv, H = shape.T, shape.d, shape.ffn, shape.dq, shape.dkv, shape.n_heads
    P_qkv = d * (dq + 2 * dkv)
    P = P_qkv + d * dq + 3 * d * f
    lin = 2 * T * P * 2 + 2 * T * (P if shape.let else P - P_qkv)
    attn = 3 * 2 * shape.head_dim * H * T * (T + 1)
    return float(lin + attn)


def _gemm_traffic():
    """DRAM bytes per GEMM launch from the committed ncu capture, if it was taken of this exact
    kernel source (else None)."""
    import hashlib
    try:
        with open(os.path.join(ROOT, "profiles", "gemm_traffic.json")) as fh:
            d = json.load(fh)
        with open(os.path.join(ROOT, d["source"]), "rb") as fh:
            sha = hashlib.sha256(fh.read()).hexdigest()
        return float(d["dram_bytes_per_launch"]) if sha == d["source_sha256"] else None
    except Exception:
        return None


def run_ours(args, shape):
    import numpy as np
    import torch
    ws, rank, local = _dist()
    if ws > 1:
        import torch.distributed as dist
        torch.cuda.set_device(local)
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    else:
        torch.cuda.set_device(0)
    dev = torch.cuda.current_device()
    from paper_2308_13137_gb300 import _lib, inputs as I
    from paper_2308_13137_gb300.block import BlockState
    _lib.lib()

    # every rank calibrates its own block: distinct weight seeds, same shapes
    seeds = replica_seeds(rank)
    W = I.make_block_weights(shape, seed=seeds["weights"])
    n_samples = 4
    xs = [I.make_block_input(shape, sample=i, weight_seed=seeds["weights"]) for i in range(n_samples)]
    th = I.make_block_theta(shape, W, xs[0], seed=seeds["theta"])
    st = BlockState(shape, W, th, pbits=args.pbits)
    xd = [torch.from_numpy(x).cuda() for x in xs]
    yfp = [torch.empty_like(v) for v in xd]
    for v, y in zip(xd, yfp):          # Eq. 1 targets: the full-precision block (not timed)
        st.fp_forward(v, y)
    torch.cuda.synchronize()

    def step_eager(i):
        st.step(xd[i % n_samples], yfp[i % n_samples])
        st.adamw()

    def step(i):                        # the same launches, replayed from a CUDA graph per sample
        st.step_adamw_graph(xd[i % n_samples], yfp[i % n_samples])

    for i in range(args.warmup):
        step_eager(i)
    for i in range(n_samples):          # each sample's first call runs one step and captures its graph
        step(i)
    torch.cuda.synchronize()
    if int(st.status.item()) != 0:
        raise RuntimeError(f"device status {int(st.status.item())} after warm-up")

    def barrier():
        if ws > 1:
            torch.distributed.barrier()

    # ---- timed region: K steps on the current stream --------------------------------------------
    vis = os.environ.get("CUDA_VISIBLE_DEVICES", "").split(",")
    clocks = ClockSampler(int(vis[dev]) if len(vis) > dev and vis[dev].strip().isdigit() else dev)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    barrier()
    torch.cuda.synchronize()
    clocks.start()
    time.sleep(0.3)
    e0.record()
    for i in range(args.steps):
        step(i)
    e1.record()
    torch.cuda.synchronize()
    barrier()
    clk = clocks.stop()
    ms = e0.elapsed_time(e1)
    if int(st.status.item()) != 0:
        raise RuntimeError(f"device status {int(st.status.item())} in the timed region")
    # per-launch GEMM durations (CUDA events on the launching streams) and the launch count, from
    # ordinary (not replayed) steps of the same workload right after the timed region
    n_prof = max(1, min(args.steps, 5))
    torch.cuda.synchronize()
    launches0 = _lib.omq_launch_count()
    _lib.omq_profile_begin()
    for i in range(n_prof):
        step_eager(i)
    torch.cuda.synchronize()
    gemm_ms, gemm_flops, gemm_launches = _lib.omq_profile_end()
    launches_per_step = (_lib.omq_launch_count() - launches0) / n_prof
    launches = int(round(launches_per_step * args.steps))
    gemm_ms, gemm_flops, gemm_launches = (gemm_ms * args.steps / n_prof, gemm_flops * args.steps / n_prof,
                                          gemm_launches * args.steps / n_prof)
    ms_max = max_over_ranks(ms, ws, "cuda")
    ms_step = ms_max / args.steps
    value = job_throughput(ws, shape.T, args.steps, ms_max / 1e3)

    # ---- end to end through the public API: host buffers in, loss out ----------------------------
    # each step's inputs go host -> device on a copy stream into one of two device buffers while the
    # step before runs; the step waits for its copy, and its loss is read back before the next step
    pin_x = [torch.from_numpy(x).pin_memory() for x in xs]
    pin_y = [y.cpu().pin_memory() for y in yfp]
    xin = [torch.empty_like(xd[0]) for _ in range(2)]
    yin = [torch.empty_like(yfp[0]) for _ in range(2)]
    loss_h = torch.zeros(1).pin_memory()
    main_stream = torch.cuda.current_stream()
    copy_stream = torch.cuda.Stream()
    copied = [torch.cuda.Event() for _ in range(2)]
    consumed = [torch.cuda.Event() for _ in range(2)]

    def enqueue_copy(i):
        b = i % 2
        with torch.cuda.stream(copy_stream):
            copy_stream.wait_event(consumed[b])   # the step that last read buffer b is done with it
            xin[b].copy_(pin_x[i % n_samples], non_blocking=True)
            yin[b].copy_(pin_y[i % n_samples], non_blocking=True)
            copied[b].record(copy_stream)

    e2e_steps = max(3, min(args.steps, 50))
    for b in range(2):                  # captures the graphs for the two input buffers (not timed)
        enqueue_copy(b)
        main_stream.wait_event(copied[b])
        st.step_adamw_graph(xin[b], yin[b])
        consumed[b].record(main_stream)
    torch.cuda.synchronize()
    barrier()
    t0 = time.perf_counter()
    enqueue_copy(0)
    for i in range(e2e_steps):
        b = i % 2
        if i + 1 < e2e_steps:
            enqueue_copy(i + 1)
        main_stream.wait_event(copied[b])
        st.step_adamw_graph(xin[b], yin[b])
        consumed[b].record(main_stream)
        loss_h.copy_(st.loss, non_blocking=True)
        main_stream.synchronize()
        _ = float(loss_h[0])
    e2e_s = max_over_ranks(time.perf_counter() - t0, ws, "cuda")
    e2e_value = job_throughput(ws, shape.T, e2e_steps, e2e_s)

    peaks = _peaks()
    gemm_flops_step = gemm_flops / args.steps
    gemm_ms_step = gemm_ms / args.steps
    achieved = gemm_flops / (gemm_ms / 1e3) / 1e12
    B = algorithmic_bytes(shape)
    F = algorithmic_flops(shape)
    t_roof = max(F / (peaks["bf16"] * 1e12), B / (peaks["hbm"] * 1e9))
    line = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": ws, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": ms_step, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
        "config": {"workload": shape.name + ("" if args.pbits == 16 else "_softmax%d" % args.pbits),
                   "tokens_per_step": shape.T, "hidden": shape.d,
                   "heads": shape.n_heads, "kv_heads": shape.n_kv, "ffn": shape.ffn, "wbits": shape.wbits,
                   "abits": shape.abits, "group": shape.group, "let": shape.let, "softmax_bits": args.pbits,
                   "step": "LET+LWC fake-quant, block fwd, MSE loss, STE bwd, AdamW",
                   "launch": "each step replays a CUDA graph of its launches (one graph per input sample)",
                   "l2": "inputs larger than L2 (bf16 weights %.0f MB per block)" % (
                       sum(v.size for v in W.values()) * 2 / 1e6),
                   "parallelism": "replicas" if ws > 1 else "single"},
        "roofline": {"bound": "tensor", "kernel": "gemm_bf16_kernel (tcgen05)",
                     "achieved": achieved, "peak": peaks["bf16_sus"], "unit": "TFLOP/s",
                     "frac": achieved / peaks["bf16_sus"], "traffic": _gemm_traffic(),
                     "traffic_unit": "bytes per launch (ncu dram read+write, averaged over one step)",
                     "peak_kind": "%s bf16_tflops_sustained (timed inside the step)" % peaks["src"],
                     "gemm_share_of_step": gemm_ms_step / ms_step, "gemm_launches_per_step":
                         gemm_launches / args.steps, "gemm_flops_per_step": gemm_flops_step,
                     "timing_note": "per-launch CUDA events over %d ordinary (not graph-replayed) steps right "
                                    "after the timed region; launches on the auxiliary stream overlap other "
                                    "kernels, so durations include co-scheduled work (a lower bound on the "
                                    "rate)" % n_prof},
        "step_roofline": {"flops_per_step": F, "bytes_per_step": B, "t_roof_ms": t_roof * 1e3,
                          "frac": t_roof * 1e3 / ms_step, "peak_tflops": peaks["bf16"], "peak_gbs": peaks["hbm"],
                          "peak_kind": peaks["src"] + " burst"},
        "e2e": {"value": e2e_value, "unit": UNIT, "h2d_bytes_per_step": 2 * xin[0].numel() * 4,
                "d2h_bytes_per_step": 4, "steps": e2e_steps,
                "copies": "pinned host -> device on a copy stream into one of two buffers while the previous "
                          "step runs; the loss is read back to the host after every step"},
        "gpu_launches": launches,
        "clocks": {"sm_mhz": clk["sm_mhz"], "sm_max_mhz": clk["sm_max_mhz"], "reasons": clk["reasons"],
                   "samples": clk["samples"]},
    }
    if rank == 0 and ws == 1 and not args.no_cpu_baseline:
        v, wall, cores = _oracle_value(shape, W, th, xs[0], args.cpu_samples)
        line["cpu_baseline"] = {"value": v, "unit": UNIT, "cores": cores, "kind": "oracle",
                                "sample": "%d oracle calibration steps (%.1f s) of 128-output-channel slices of "
                                          "the block's projections, cycling q,k,v,o,gate,up,down at %d tokens; each "
                                          "scaled by Cout/128 (attention and norms not sampled)" % (
                                              args.cpu_samples, wall, shape.T)}
    if rank == 0:
        print(json.dumps(line), flush=True)
    if ws > 1:
        torch.distributed.destroy_process_group()
    return 0


def main():
    ap = argparse.ArgumentParser(description=__doc__.split("\n")[0])
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=200)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--config", default=DEFAULT_CONFIG)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--cpu-samples", type=int, default=14)
    ap.add_argument("--pbits", type=int, default=16,
                    help="softmax-output bits (2..8: the quantized-softmax ablation; 16: not quantized, the default)")
    args = ap.parse_args()
    from paper_2308_13137_gb300 import inputs as I
    shape = I.block_shape(args.config)
    if args.impl == "reference":
        return run_reference(args, shape)
    return run_ours(args, shape)


if __name__ == "__main__":
    sys.exit(main())
