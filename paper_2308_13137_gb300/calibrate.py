"""Algorithm 1 (block-wise calibration) over a stack of decoder blocks on the GPU, with a
checkpoint after every block so that an interrupted run resumes at the next block.

Per block i (Algorithm 1): the full-precision inputs X_fp are advanced through the full-precision
block to give the Eq. 1 targets; the LWC logits start at gamma_hat = beta_hat = 4 and the LET
vectors from the block's statistics on X_fp (Sec. 4.1 "Training": SmoothQuant scaling, OS+
shifting); every calibration sample x_q is one step (forward, loss against its target, STE
backward, AdamW with zero weight decay at lr 5e-3 / 1e-2); after the epochs the quantized block's
outputs become the next block's X_q, and the block is folded and packed.  Every kernel runs through
libomq (BlockState); this module only sequences the calls and writes checkpoints.
"""
from __future__ import annotations

import os
from typing import Dict, List, Optional

import numpy as np

from .block import BlockState

__all__ = ["calibrate_blocks"]


def _ckpt_path(ckpt_dir: str, i: int) -> str:
    return os.path.join(ckpt_dir, f"block_{i:04d}.pt")


def calibrate_blocks(shape, blocks: List[Dict[str, np.ndarray]], xs, theta0: Dict[str, np.ndarray], epochs: int = 1,
                     lr_lwc: float = 5e-3, lr_let: float = 1e-2, let_init: bool = True,
                     ckpt_dir: Optional[str] = None, stop_after: Optional[int] = None, device: str = "cuda"):
    """Calibrate `blocks` (host weight dicts of one shape) on calibration inputs `xs` (host or
    device [T, d] fp32).  theta0 holds the initial LWC logits (and LET vectors, overwritten by the
    statistics when let_init).  With ckpt_dir, block i's parameters, packed form and the advanced
    X_fp, X_q are saved after it finishes, and blocks already saved are skipped on a later call.
    stop_after = n returns after n blocks of this call (an interruption, for resuming).
    Returns (per-block parameter dicts on the host, per-block packed dicts on the host, X_fp, X_q)."""
    import torch
    dev = lambda x: torch.as_tensor(np.asarray(x) if not torch.is_tensor(x) else x).to(device, torch.float32).contiguous()
    x_fp = [dev(x) for x in xs]
    x_q = [dev(x) for x in xs]
    params, packed = [], []
    done_now = 0
    for i, W in enumerate(blocks):
        if ckpt_dir is not None and os.path.exists(_ckpt_path(ckpt_dir, i)):
            ck = torch.load(_ckpt_path(ckpt_dir, i), map_location="cpu", weights_only=True)
            params.append(ck["theta"])
            packed.append(ck["packed"])
            x_fp = [v.to(device) for v in ck["x_fp"]]
            x_q = [v.to(device) for v in ck["x_q"]]
            continue
        if stop_after is not None and done_now >= stop_after:
            break
        st = BlockState(shape, W, theta0, device=device)
        if shape.let and let_init:
            st.let_init(x_fp)
        y_fp = []
        for x in x_fp:
            y = torch.empty_like(x)
            st.fp_forward(x, y)
            y_fp.append(y)
        for _ in range(epochs):
            for xq, yf in zip(x_q, y_fp):
                st.step(xq, yf)
                st.adamw(lr_lwc, lr_let)
        new_q = []
        for xq in x_q:
            y = torch.empty_like(xq)
            st.forward(xq, y)
            new_q.append(y)
        torch.cuda.synchronize()
        if int(st.status.item()) != 0:
            raise RuntimeError(f"device status {int(st.status.item())} while calibrating block {i}")
        x_fp, x_q = y_fp, new_q
        theta = {k: torch.from_numpy(v.copy()) for k, v in st.split_theta().items()}
        pk = {k: v.detach().cpu().clone() for k, v in st.fold_pack().items()}
        params.append(theta)
        packed.append(pk)
        if ckpt_dir is not None:
            os.makedirs(ckpt_dir, exist_ok=True)
            tmp = _ckpt_path(ckpt_dir, i) + ".tmp"
            torch.save(dict(theta=theta, packed=pk, x_fp=[v.cpu() for v in x_fp], x_q=[v.cpu() for v in x_q]), tmp)
            os.replace(tmp, _ckpt_path(ckpt_dir, i))       # a checkpoint is complete or absent
        done_now += 1
        del st
    return params, packed, x_fp, x_q
