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
# the oracle on host cores
# ------------------------------------------------------------------------------------------------
PIECES = ["fwd q|k|v", "fwd attention", "fwd o_proj", "fwd gate|up", "fwd down_proj", "loss",
          "bwd down_proj", "bwd gate|up", "bwd o_proj", "bwd attention", "bwd q|k|v"]


def _oracle_pieces(shape, W, th, x, yfp, out=None):
    """Yields (piece name, seconds) forever: the oracle's calibration step (forward of the quantized
    block, loss against y_fp, straight-through backward to every parameter) cut at the block's
    five stages, in the order one step runs them (five forward stages, the loss, the five stage
    backwards), and again for the next step.  One pass over the eleven pieces is exactly one oracle
    block_step; each piece is a bounded sample of it.  `out` (a dict), when given, receives the
    step's loss and parameter gradients after every pass."""
    import torch
    import oracle as O
    cfg = O.BlockCfg.from_shape(shape)
    t = lambda v: torch.as_tensor(v).to(torch.float64)
    Wd = {k: t(v) for k, v in W.items()}
    names = (O.THETA_NAMES_LWC if shape.wbits < 16 else []) + (O.THETA_NAMES_LET if shape.let else [])
    dq, dkv, f = shape.dq, shape.dkv, shape.ffn
    xx, yf = t(x), t(yfp)

    def grad(out, inp, gout):
        inps = [] if inp is None else (list(inp) if isinstance(inp, (list, tuple)) else [inp])
        return torch.autograd.grad(out, [leaf[k] for k in names] + inps, gout, allow_unused=True)

    while True:
        leaf = {k: t(th[k]).clone().requires_grad_(True) for k in names}
        c = time.perf_counter()
        q, k, v, _ = O.stage_attn_in(xx, Wd, leaf, cfg)
        qkv = torch.cat([q, k, v], 1)
        yield PIECES[0], time.perf_counter() - c
        c = time.perf_counter()
        qkv_in = qkv.detach().requires_grad_(True)
        Ob, _, _ = O.stage_attention(qkv_in[:, :dq], qkv_in[:, dq:dq + dkv], qkv_in[:, dq + dkv:], leaf, cfg)
        yield PIECES[1], time.perf_counter() - c
        c = time.perf_counter()
        O_in = Ob.detach().requires_grad_(True)
        h1 = O.stage_attn_out(O_in, xx, Wd, leaf, cfg)
        yield PIECES[2], time.perf_counter() - c
        c = time.perf_counter()
        h1_in = h1.detach().requires_grad_(True)
        gt, up = O.stage_ffn_in(h1_in, Wd, leaf, cfg)
        gu = torch.cat([gt, up], 1)
        yield PIECES[3], time.perf_counter() - c
        c = time.perf_counter()
        gu_in = gu.detach().requires_grad_(True)
        h1_res = h1_in.detach().requires_grad_(True)
        y, _ = O.stage_ffn_out(gu_in[:, :f], gu_in[:, f:], h1_res, Wd, leaf, cfg)
        yield PIECES[4], time.perf_counter() - c
        c = time.perf_counter()
        y_in = y.detach().requires_grad_(True)
        loss, _ = O.block_loss(y_in, yf)
        (dy,) = torch.autograd.grad(loss, [y_in])
        yield PIECES[5], time.perf_counter() - c
        c = time.perf_counter()
        gE = grad(y, [gu_in, h1_res], dy)
        yield PIECES[6], time.perf_counter() - c
        c = time.perf_counter()
        gD = grad(gu, h1_in, gE[-2])
        dh1 = gD[-1] + gE[-1]
        yield PIECES[7], time.perf_counter() - c
        c = time.perf_counter()
        gC = grad(h1, O_in, dh1)
        yield PIECES[8], time.perf_counter() - c
        c = time.perf_counter()
        gB = grad(Ob, qkv_in, gC[-1])
        yield PIECES[9], time.perf_counter() - c
        c = time.perf_counter()
        gA = grad(qkv, None, gB[-1]) if names else []
        dt = time.perf_counter() - c
        if out is not None:
            out["loss"] = loss.detach()
            for i, n in enumerate(names):
                out["d" + n] = sum(gg[i] for gg in (gA, gB, gC, gD, gE) if gg[i] is not None)
        yield PIECES[10], dt
        del q, k, v, qkv, Ob, h1, gt, up, gu, y, gE, gD, gC, gB, gA


def _oracle_yfp(shape, W, x):
    import oracle as O
    return O.block_fp_forward(x, W, O.BlockCfg.from_shape(shape)).float().numpy()


def cpu_baseline(shape, W, th, x):
    """The oracle on the host cores, timed: one full calibration step (forward, loss, STE backward)
    of the block at the workload's token count."""
    import torch
    yfp = _oracle_yfp(shape, W, x)
    it = _oracle_pieces(shape, W, th, x, yfp)
    secs = sum(next(it)[1] for _ in PIECES)
    return dict(value=shape.T / secs, unit=UNIT, cores=torch.get_num_threads(), kind="oracle",
                sample="one full fp64 oracle calibration step (forward, loss, STE backward; %.1f s) at %d tokens"
                       % (secs, shape.T), seconds=secs)


def run_reference(args, shape):
    ws, rank, _ = _dist()
    if rank != 0:
        return 0
    import torch
    from paper_2308_13137_gb300 import inputs as I
    W = I.make_block_weights(shape, seed=1)
    x = I.make_block_input(shape, 0, 1)
    th = I.make_block_theta(shape, W, x, seed=2)
    it = _oracle_pieces(shape, W, th, x, _oracle_yfp(shape, W, x))
    for _ in range(args.warmup):
        next(it)
    per = {p: [] for p in PIECES}
    t0 = time.perf_counter()
    k = 0
    # time K pieces, and at least one of each so that every part of the step is measured
    while k < args.steps or any(not v for v in per.values()):
        name, dt = next(it)
        per[name].append(dt)
        k += 1
    wall = time.perf_counter() - t0
    step_s = sum(statistics.mean(v) for v in per.values())
    value = shape.T / step_s
    sample = ("each step one piece of the fp64 oracle's calibration step (the five forward stages, the loss, the five "
              "stage backwards, in a step's order); value = %d tokens / the sum of the pieces' mean times (%d pieces "
              "timed)" % (shape.T, k))
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": ws, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": 1e3 * step_s, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": {"workload": shape.name, "tokens_per_step": shape.T, "wbits": shape.wbits,
                       "abits": shape.abits, "group": shape.group, "let": shape.let},
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": torch.get_num_threads(), "kind": "oracle",
                             "sample": sample},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
            "wall_s": wall}
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


def step_roofline(F: float, B: float, ms_step: float, peaks: dict, bound=None) -> dict:
    """The line's roofline with one calibration step (one graph replay) as the unit: the step's
    algorithmic flops F and bytes B against the burst bf16 peak and the HBM peak, whichever bounds
    it; achieved = the algorithmic work of one step / the step's CUDA-event time, so frac =
    t_roof / t_step.  `bound` overrides the label (the single-linear case is latency-bound)."""
    t_f = F / (peaks["bf16"] * 1e12)
    t_b = B / (peaks["hbm"] * 1e9) if B else 0.0
    tensor = t_f >= t_b
    s = ms_step / 1e3
    achieved = F / s / 1e12 if tensor else B / s / 1e9
    peak = peaks["bf16"] if tensor else peaks["hbm"]
    return {"bound": bound or ("tensor" if tensor else "hbm"), "unit": "TFLOP/s" if tensor else "GB/s",
            "achieved": achieved, "peak": peak, "frac": achieved / peak, "traffic": None,
            "scope": "one whole calibration step (every kernel of it), algorithmic work / step time",
            "flops_per_step": F, "bytes_per_step": B, "t_roof_ms": max(t_f, t_b) * 1e3,
            "peak_kind": "%s %s" % (peaks["src"], "bf16_tflops burst" if tensor else "hbm_gbs"),
            "traffic_note": "no per-step DRAM capture: ncu counters beyond time are taken one kernel at a "
                            "time (the GEMM's in roofline.gemm.traffic, the others in profiles/)"}


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
    th = I.make_block_theta(shape, W, xs[0], seed=seeds["theta"], weight_seed=seeds["weights"])
    st = BlockState(shape, W, th, pbits=args.pbits, wprep=args.wprep)
    xd = [torch.from_numpy(x).cuda() for x in xs]
    yfp = [torch.empty_like(v) for v in xd]
    for v, y in zip(xd, yfp):          # Eq. 1 targets: the full-precision block (not timed)
        st.fp_forward(v, y)
    if shape.let:                       # Algorithm 1's LET initialisation from the samples (not timed)
        st.let_init(xd)
    torch.cuda.synchronize()
    th_host = st.split_theta()          # the parameters the timed steps start from

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
                   "qkv_weight_operand": ("fake-quantized tile by tile in the GEMM's shared memory" if args.wprep
                                          else "W_hat written to HBM by the LWC forward"),
                   "step": "LET+LWC fake-quant, block fwd, MSE loss, STE bwd, AdamW",
                   "launch": "each step replays a CUDA graph of its launches (one graph per input sample)",
                   "l2": "inputs larger than L2 (bf16 weights %.0f MB per block)" % (
                       sum(v.size for v in W.values()) * 2 / 1e6),
                   "parallelism": "replicas" if ws > 1 else "single"},
        "roofline": dict(step_roofline(F, B, ms_step, peaks), gemm={
                     "bound": "tensor", "kernel": "gemm_bf16_kernel (tcgen05)",
                     "achieved": achieved, "peak": peaks["bf16_sus"], "unit": "TFLOP/s",
                     "frac": achieved / peaks["bf16_sus"], "traffic": _gemm_traffic(),
                     "traffic_unit": "bytes per launch (ncu dram read+write, averaged over one step)",
                     "peak_kind": "%s bf16_tflops_sustained (timed inside the step)" % peaks["src"],
                     "gemm_share_of_step": gemm_ms_step / ms_step, "gemm_launches_per_step":
                         gemm_launches / args.steps, "gemm_flops_per_step": gemm_flops_step,
                     "timing_note": "per-launch CUDA events over %d ordinary (not graph-replayed) steps right "
                                    "after the timed region; launches on the auxiliary stream overlap other "
                                    "kernels, so durations include co-scheduled work (a lower bound on the "
                                    "rate)" % n_prof}),
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
        cb = cpu_baseline(shape, W, th_host, xs[0])
        cb.pop("seconds")
        line["cpu_baseline"] = cb
    if rank == 0:
        print(json.dumps(line), flush=True)
    if ws > 1:
        torch.distributed.destroy_process_group()
    return 0


def run_reference_linear(args, lsh):
    """The fp64 oracle's step of the single quantized linear on the host cores, one per step."""
    ws, rank, _ = _dist()
    if rank != 0:
        return 0
    import torch
    import oracle as O
    from paper_2308_13137_gb300 import inputs as I
    tt = {k: torch.from_numpy(v) for k, v in I.make_linear_case(lsh, seed=0).items()}
    yfp = tt["X"].double() @ tt["W"].double().T

    def one():
        O.qlinear_step(tt["X"], tt["W"], tt["B"], tt["gamma_logit"], tt["beta_logit"], yfp, lsh.wbits, lsh.group, lsh.abits)

    for _ in range(args.warmup):
        one()
    t0 = time.perf_counter()
    for _ in range(args.steps):
        one()
    wall = time.perf_counter() - t0
    value = lsh.T * args.steps / wall
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": ws, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": 1e3 * wall / args.steps, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": {"workload": lsh.name, "tokens_per_step": lsh.T, "wbits": lsh.wbits, "abits": lsh.abits,
                       "group": lsh.group, "let": 0},
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": torch.get_num_threads(), "kind": "oracle",
                             "sample": "each step one fp64 oracle calibration step of the linear"},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)
    return 0


def run_ours_linear(args, lsh):
    """The single quantized linear (W4A16 g128, LWC only, Eq. 4 with Eq. 2): one step is the forward,
    the MSE loss against the full-precision output, the STE backward to gamma_hat, beta_hat and the
    AdamW update, replayed from a CUDA graph (the step is launch-bound at this size)."""
    import numpy as np
    import torch
    ws, rank, local = _dist()
    torch.cuda.set_device(local if ws > 1 else 0)
    from paper_2308_13137_gb300 import _lib, inputs as I
    _lib.lib()
    if ws > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    case = I.make_linear_case(lsh, seed=rank)
    T, Cin, Cout = lsh.T, lsh.Cin, lsh.Cout
    ng = Cin // lsh.group
    cfg = _lib.make_cfg(wbits=lsh.wbits, abits=lsh.abits, group=lsh.group)
    f32, bf = dict(device="cuda", dtype=torch.float32), dict(device="cuda", dtype=torch.bfloat16)
    X = torch.from_numpy(case["X"]).cuda()
    W = torch.from_numpy(case["W"]).cuda().to(torch.bfloat16)
    B = torch.from_numpy(case["B"]).cuda()
    Yfp = X @ W.float().T                       # Eq. 1 target: the full-precision output (not timed)
    theta = torch.cat([torch.from_numpy(case["gamma_logit"]).reshape(-1), torch.from_numpy(case["beta_logit"]).reshape(-1)]).cuda()
    grads = torch.zeros_like(theta)
    m, v = torch.zeros_like(theta), torch.zeros_like(theta)
    gl, bl = theta[:Cout * ng].view(Cout, ng), theta[Cout * ng:].view(Cout, ng)
    dgl, dbl = grads[:Cout * ng].view(Cout, ng), grads[Cout * ng:].view(Cout, ng)
    sv = dict(w_hat=torch.empty(Cout, Cin, **bf), h_w=torch.empty(Cout, ng, **f32),
              z_w=torch.empty(Cout, ng, device="cuda", dtype=torch.int32),
              imax_w=torch.empty(Cout, ng, device="cuda", dtype=torch.int32),
              imin_w=torch.empty(Cout, ng, device="cuda", dtype=torch.int32), x_hat=torch.empty(T, Cin, **bf),
              h_a=torch.empty(T, **f32), z_a=torch.empty(T, device="cuda", dtype=torch.int32),
              imax_a=torch.empty(T, device="cuda", dtype=torch.int32), imin_a=torch.empty(T, device="cuda", dtype=torch.int32),
              b_tilde=torch.empty(Cout, **f32))
    saved = _lib.omq_qlinear_saved(*[sv[k].data_ptr() for k in ("w_hat", "h_w", "z_w", "imax_w", "imin_w", "x_hat",
                                                                "h_a", "z_a", "imax_a", "imin_a", "b_tilde")])
    Y = torch.empty(T, Cout, **f32)
    dY = torch.empty(T, Cout, **f32)
    loss = torch.zeros(1, **f32)
    lws = torch.empty(_lib.omq_loss_workspace_size(T * Cout), device="cuda", dtype=torch.uint8)
    qws = torch.empty(_lib.omq_qlinear_workspace_size(T, Cin, Cout, cfg), device="cuda", dtype=torch.uint8)
    step_dev = torch.zeros(1, device="cuda", dtype=torch.int32)

    def step(x):
        _lib.omq_qlinear_fwd(T, Cin, Cout, x, W, B, None, None, gl, bl, Y, saved, cfg)
        _lib.omq_block_loss(T * Cout, Y, Yfp, loss, dY, None, lws)
        _lib.omq_qlinear_bwd(T, Cin, Cout, x, W, None, None, gl, bl, saved, dY, None, dgl, dbl, None, None, qws, cfg)
        _lib.omq_step_advance(step_dev)
        _lib.omq_adamw_update_dev(theta.numel(), theta, grads, m, v, 5e-3, 0.9, 0.999, 1e-8, 0.0, step_dev)

    for _ in range(max(3, args.warmup)):
        step(X)
    torch.cuda.synchronize()
    xin = torch.empty_like(X)
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        step(xin)
    xin.copy_(X)
    for _ in range(3):
        g.replay()
    torch.cuda.synchronize()
    reps = max(20, args.steps)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    clocks = ClockSampler(0)
    clocks.start()
    time.sleep(0.3)
    if ws > 1:
        torch.distributed.barrier()
    torch.cuda.synchronize()
    e0.record()
    for _ in range(reps):
        g.replay()
    e1.record()
    torch.cuda.synchronize()
    clk = clocks.stop()
    ms = max_over_ranks(e0.elapsed_time(e1), ws, "cuda")
    value = job_throughput(ws, T, reps, ms / 1e3)
    # GEMM rate from ordinary steps
    _lib.omq_profile_begin()
    l0 = _lib.omq_launch_count()
    for _ in range(5):
        step(X)
    torch.cuda.synchronize()
    gemm_ms, gemm_flops, gemm_n = _lib.omq_profile_end()
    launches = (_lib.omq_launch_count() - l0) / 5
    # end to end: X from pinned host memory each step, the loss read back
    xh = torch.from_numpy(case["X"]).pin_memory()
    lh = torch.zeros(1).pin_memory()
    t0 = time.perf_counter()
    for _ in range(reps):
        xin.copy_(xh, non_blocking=True)
        g.replay()
        lh.copy_(loss, non_blocking=True)
        torch.cuda.current_stream().synchronize()
    e2e_s = max_over_ranks(time.perf_counter() - t0, ws, "cuda")
    peaks = _peaks()
    F = 3 * 2.0 * T * Cin * Cout
    line = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": ws, "steps": reps, "warmup": args.warmup,
        "ms_per_step": ms / reps, "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
        "data": "synthetic",
        "config": {"workload": lsh.name, "tokens_per_step": T, "Cin": Cin, "Cout": Cout, "wbits": lsh.wbits,
                   "abits": lsh.abits, "group": lsh.group, "let": 0,
                   "step": "LWC fake-quant, quantized linear fwd, MSE loss, STE bwd, AdamW",
                   "launch": "each step replays a CUDA graph of its launches",
                   "l2": "inputs smaller than L2 (the single-linear case is launch-bound)",
                   "parallelism": "replicas" if ws > 1 else "single"},
        "roofline": dict(step_roofline(F, 0.0, ms / reps, peaks, bound="latency"), gemm={
                     "bound": "latency", "kernel": "gemm_bf16_kernel (tcgen05)", "achieved": gemm_flops / (gemm_ms / 1e3) / 1e12,
                     "peak": peaks["bf16"], "unit": "TFLOP/s", "frac": gemm_flops / (gemm_ms / 1e3) / 1e12 / peaks["bf16"],
                     "traffic": None, "peak_kind": "%s bf16_tflops burst" % peaks["src"]},
                     note="%.2e flop per step: far below what fills the GPU; the step is set by launch latency" % F),
        "step_roofline": {"flops_per_step": F, "t_roof_ms": F / (peaks["bf16"] * 1e12) * 1e3,
                          "frac": F / (peaks["bf16"] * 1e12) * 1e3 / (ms / reps)},
        "e2e": {"value": job_throughput(ws, T, reps, e2e_s), "unit": UNIT, "h2d_bytes_per_step": X.numel() * 4,
                "d2h_bytes_per_step": 4, "steps": reps},
        "gpu_launches": int(round(launches * reps)),
        "clocks": {"sm_mhz": clk["sm_mhz"], "sm_max_mhz": clk["sm_max_mhz"], "reasons": clk["reasons"],
                   "samples": clk["samples"]},
    }
    if rank == 0 and ws == 1 and not args.no_cpu_baseline:
        import oracle as O
        tt = {k: torch.from_numpy(v) for k, v in case.items()}
        yfp64 = tt["X"].double() @ tt["W"].double().T
        n_rep, c = 5, time.perf_counter()
        for _ in range(n_rep):
            O.qlinear_step(tt["X"], tt["W"], tt["B"], tt["gamma_logit"], tt["beta_logit"], yfp64, lsh.wbits, lsh.group,
                           lsh.abits)
        secs = (time.perf_counter() - c) / n_rep
        line["cpu_baseline"] = {"value": T / secs, "unit": UNIT, "cores": torch.get_num_threads(), "kind": "oracle",
                                "sample": "fp64 oracle calibration step of the linear, mean of %d (%.3f s each)" % (
                                    n_rep, secs)}
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
    ap.add_argument("--pbits", type=int, default=16,
                    help="softmax-output bits (2..8: the quantized-softmax ablation; 16: not quantized, the default)")
    ap.add_argument("--wprep", type=int, choices=[0, 1], default=0,
                    help="q|k|v weight operand: 0 = W_hat materialised in HBM, 1 = fake-quantized inside the GEMM")
    args = ap.parse_args()
    from paper_2308_13137_gb300 import inputs as I
    if isinstance(I.SHAPES.get(args.config), I.LinearShape):
        if args.impl == "reference":
            return run_reference_linear(args, I.SHAPES[args.config])
        return run_ours_linear(args, I.SHAPES[args.config])
    shape = I.block_shape(args.config)
    if args.impl == "reference":
        return run_reference(args, shape)
    return run_ours(args, shape)


if __name__ == "__main__":
    sys.exit(main())
