"""Device-resident state of one decoder block for libomq's block entry points.

PyTorch only allocates: this module stacks the frozen weights and the learnable parameters in
the layout include/omq.h documents (q|k|v rows in one matrix, gate|up rows in another), holds
the gradient buffers and the workspace, and passes pointers to omq_block_step /
omq_block_forward.  All arithmetic of the step runs in libomq's kernels.
"""
from __future__ import annotations

from typing import Dict, Optional

import numpy as np

from . import _lib

LWC_PARTS = {"qkv": ("q", "k", "v"), "o": ("o",), "gu": ("g", "u"), "d": ("d",)}
LET_NAMES = {"s1": "s1", "d1": "d1", "so": "so", "do": "do_", "sa": "sa", "s2": "s2", "d2": "d2"}


class BlockState:
    """Weights, parameters, gradients and workspace of one block on the current CUDA device."""

    def __init__(self, shape, weights: Dict[str, np.ndarray], theta: Dict[str, np.ndarray], device: str = "cuda",
                 wbits: Optional[int] = None, abits: Optional[int] = None, group: Optional[int] = None,
                 let: Optional[int] = None, pbits: int = 16, wprep: int = 0):
        import torch
        self.torch = torch
        self.shape = shape
        self.device = device
        self.wbits = shape.wbits if wbits is None else wbits
        self.abits = shape.abits if abits is None else abits
        self.group = shape.group if group is None else group
        self.let = shape.let if let is None else let
        self.pbits = pbits                 # softmax-output bits; 16 = not quantized (the default)
        self.wprep = wprep                 # 1: the q|k|v products fake-quantize the raw weight tile by tile
        bf = torch.bfloat16

        def dev_bf16(a):
            return torch.from_numpy(np.ascontiguousarray(a, dtype=np.float32)).to(device=device).to(bf).contiguous()

        def dev_f32(a):
            return torch.from_numpy(np.ascontiguousarray(a, dtype=np.float32)).to(device=device).contiguous()

        self.W = dict(
            qkv=dev_bf16(np.concatenate([weights["wq"], weights["wk"], weights["wv"]], 0)),
            o=dev_bf16(weights["wo"]),
            gu=dev_bf16(np.concatenate([weights["wg"], weights["wu"]], 0)),
            d=dev_bf16(weights["wd"]))
        # learnable parameters live in two flat fp32 buffers (LWC logits | LET vectors) so that one
        # optimizer launch per learning-rate group updates them; the names below are views
        host = {}
        if self.wbits < 16:
            for key, parts in LWC_PARTS.items():
                for gb in ("gamma", "beta"):
                    host[f"{gb}_{key}"] = np.concatenate([theta[f"{gb}_{p}"] for p in parts], 0)
        n_lwc = sum(v.size for v in host.values())
        if self.let:
            for k in LET_NAMES:
                host[k] = np.asarray(theta[k])
        self.theta_flat, self.grads_flat = {}, {}
        self.theta, self.grads = {}, {}
        groups = dict(lwc=[k for k in host if k not in LET_NAMES], let=[k for k in host if k in LET_NAMES])
        for gname, keys in groups.items():
            if not keys:
                continue
            # pad each view to a multiple of 4 floats so every view stays 16-byte aligned
            sizes = [host[k].size for k in keys]
            offs = np.cumsum([0] + [(n + 3) // 4 * 4 for n in sizes])
            flat = torch.zeros(int(offs[-1]), dtype=torch.float32, device=device)
            gflat = torch.zeros_like(flat)
            for k, o, n in zip(keys, offs[:-1], sizes):
                flat[o:o + n] = dev_f32(host[k].reshape(-1))
                self.theta[k] = flat[o:o + n].view(host[k].shape)
                self.grads[k] = gflat[o:o + n].view(host[k].shape)
            self.theta_flat[gname], self.grads_flat[gname] = flat, gflat
        self.n_lwc = n_lwc
        self.adam = {g: (torch.zeros_like(f), torch.zeros_like(f)) for g, f in self.theta_flat.items()}
        self.adam_step = 0
        # the AdamW step count also lives on the device, so that captured graphs replay correctly
        self.adam_step_dev = torch.zeros(1, dtype=torch.int32, device=device)
        self._graphs = {}
        self.c_shape = _lib.omq_block_shape(shape.T, shape.d, shape.n_heads, shape.n_kv, shape.head_dim, shape.ffn,
                                            shape.rms_eps, shape.rope_theta)
        self.c_w = _lib.omq_block_weights(*[self.W[k].data_ptr() for k in ("qkv", "o", "gu", "d")])
        self.c_theta = self._params(self.theta)
        self.c_grads = self._params(self.grads)
        self.status = torch.zeros(1, dtype=torch.int32, device=device)
        self.cfg = _lib.make_cfg(self.wbits, self.abits, self.group, self.let, 1e-5, 0, self.status, self.pbits,
                                 self.wprep)
        ws = _lib.omq_block_workspace_size(self.c_shape, self.cfg)
        if ws == 0:
            raise ValueError("block shape or configuration rejected by libomq")
        self.workspace = torch.empty(ws, dtype=torch.uint8, device=device)
        self.loss = torch.zeros(1, dtype=torch.float32, device=device)

    @staticmethod
    def _params(d) -> "_lib.omq_block_params":
        p = _lib.omq_block_params()
        for k, v in d.items():
            setattr(p, LET_NAMES.get(k, k), v.data_ptr())
        return p

    def step(self, x, y_fp, y=None, stream=None):
        """One calibration step: forward, loss (device scalar self.loss) and gradients (self.grads)."""
        _lib.omq_block_step(self.c_shape, self.c_w, self.c_theta, x, y_fp, y, self.loss, self.c_grads,
                            self.workspace, self.cfg, stream)
        return self.loss

    def saved(self, backward: bool = True) -> Dict[str, "object"]:
        """The stage values the last forward / step left in the workspace (omq_block_saved_layout),
        as device tensor views named like the layout's fields; w_hat, w_h, w_z become lists over
        q|k|v, o, gate|up, down.  Views, not copies: the next call overwrites them."""
        torch = self.torch
        sh = self.shape
        lay = _lib.omq_block_saved_layout(self.c_shape, self.cfg)
        T, d, f = sh.T, sh.d, sh.ffn
        nqkv = sh.dq + 2 * sh.dkv
        bf, f32, i32 = torch.bfloat16, torch.float32, torch.int32
        spec = dict(a_hat=(bf, (T, d)), a_h=(f32, (T,)), a_z=(i32, (T,)), y_qkv=(f32, (T, nqkv)),
                    qkv_h=(f32, (3, T)), qkv_z=(i32, (3, T)), q_hat=(bf, (T, sh.dq)), k_hat=(bf, (T, sh.dkv)),
                    v_hat=(bf, (T, sh.dkv)), o=(f32, (T, sh.dq)), o_hat=(bf, (T, sh.dq)),
                    o_h=(f32, (T,)), o_z=(i32, (T,)), h1=(f32, (T, d)), b_hat=(bf, (T, d)), b_h=(f32, (T,)),
                    b_z=(i32, (T,)), y_gu=(f32, (T, 2 * f)), m_hat=(bf, (T, f)), m_h=(f32, (T,)), m_z=(i32, (T,)))
        if backward:
            spec.update(dy=(f32, (T, d)), dy_gu=(bf, (T, 2 * f)), dh1=(bf, (T, d)), do_bf16=(bf, (T, sh.dq)),
                        dy_qkv=(bf, (T, nqkv)))

        def view(off, dtype, shp):
            n = int(np.prod(shp)) * torch.empty(0, dtype=dtype).element_size()
            return self.workspace[off:off + n].view(dtype).view(shp)

        out = {k: view(getattr(lay, k), dt, shp) for k, (dt, shp) in spec.items()}
        ng = lambda cin: 1 if self.group == 0 else cin // self.group
        lins = [(nqkv, d), (d, sh.dq), (2 * f, d), (d, f)]
        out["w_hat"] = [None if lay.w_hat[i] < 0 else view(lay.w_hat[i], bf, (co, ci)) for i, (co, ci) in enumerate(lins)]
        out["w_h"] = [view(lay.w_h[i], f32, (co, ng(ci))) for i, (co, ci) in enumerate(lins)]
        out["w_z"] = [view(lay.w_z[i], i32, (co, ng(ci))) for i, (co, ci) in enumerate(lins)]
        return out

    def adamw(self, lr_lwc: float = 5e-3, lr_let: float = 1e-2, stream=None):
        """AdamW with zero weight decay on both parameter groups (Sec. 4.1 "Training"); the step
        count advances on the device."""
        self.adam_step += 1
        _lib.omq_step_advance(self.adam_step_dev, stream)
        for g, flat in self.theta_flat.items():
            m, v = self.adam[g]
            _lib.omq_adamw_update_dev(flat.numel(), flat, self.grads_flat[g], m, v, lr_lwc if g == "lwc" else lr_let,
                                      0.9, 0.999, 1e-8, 0.0, self.adam_step_dev, stream)

    def step_adamw_graph(self, x, y_fp, lr_lwc: float = 5e-3, lr_let: float = 1e-2):
        """One calibration step and its AdamW update, replayed from a CUDA graph of the same launches
        (one graph per input pair (x, y_fp) and learning rates, captured on first use after one
        ordinary step has set up the library's state).  The result equals step() + adamw().

        A graph holds the device addresses it was captured with and is looked up by the addresses of
        x and y_fp: a caller refills the same tensors in place between calls (new tensors, even of
        equal contents, capture a new graph), and must keep them alive while this state may replay
        it.  Weights, parameters, gradients and workspace are this object's own buffers."""
        torch = self.torch
        key = (x.data_ptr(), y_fp.data_ptr(), lr_lwc, lr_let)
        g = self._graphs.get(key)
        if g is not None:
            self.adam_step += 1
            g.replay()
            return self.loss
        self.step(x, y_fp)                  # one ordinary step: lazy set-up inside libomq happens here
        self.adamw(lr_lwc, lr_let)
        torch.cuda.synchronize()
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g):
            self.step(x, y_fp)
            _lib.omq_step_advance(self.adam_step_dev)
            for name, flat in self.theta_flat.items():
                m, v = self.adam[name]
                _lib.omq_adamw_update_dev(flat.numel(), flat, self.grads_flat[name], m, v,
                                          lr_lwc if name == "lwc" else lr_let, 0.9, 0.999, 1e-8, 0.0,
                                          self.adam_step_dev)
        self._graphs[key] = g
        return self.loss

    def forward(self, x, y, stream=None, cfg=None):
        _lib.omq_block_forward(self.c_shape, self.c_w, self.c_theta, x, y, self.workspace, cfg or self.cfg, stream)
        return y

    def fp_forward(self, x, y, stream=None):
        """Full-precision block (quantization and LET off): the target of Eq. 1."""
        cfg = _lib.make_cfg(16, 16, 0, 0, 1e-5, 0, self.status)
        return self.forward(x, y, stream, cfg)

    def let_init(self, xs, alpha: float = 0.5, stream=None):
        """Initial LET parameters (Sec. 4.1 "Training": SmoothQuant scaling, OS+ shifting) from
        the calibration inputs xs (device [T, d] fp32 tensors), written into the LET views of the
        parameter buffer; returns them as a dict of device tensors."""
        torch = self.torch
        if not self.let:
            raise ValueError("LET is off for this block")
        sh = self.shape
        f32 = dict(dtype=torch.float32, device=self.device)
        st = {n: torch.empty(sz, **f32) for n, sz in
              dict(a_absmax=sh.d, a_sum=sh.d, q_absmax=sh.dq, k_absmax=sh.dkv, o_absmax=sh.dq, o_sum=sh.dq,
                   b_absmax=sh.d, b_sum=sh.d).items()}
        c_st = _lib.omq_let_stats(*[st[n].data_ptr() for n in _lib.LET_STATS_FIELDS])
        for i, x in enumerate(xs):
            _lib.omq_let_stats_accumulate(self.c_shape, self.c_w, x, c_st, i == 0, self.workspace, self.status,
                                          stream)
        ws = torch.empty(_lib.omq_let_init_workspace_size(self.c_shape), dtype=torch.uint8, device=self.device)
        _lib.omq_let_init(self.c_shape, self.c_w, c_st, sum(int(x.shape[0]) for x in xs), alpha, self.c_theta, ws,
                          stream)
        return {k: self.theta[k] for k in LET_NAMES}

    def fold_pack(self, stream=None):
        """The calibrated block with its LET parameters folded in and its weights quantized and
        packed (Algorithm 1, after training): device tensors named as in omq_block_packed."""
        torch = self.torch
        sh = self.shape
        dev = self.device
        nq = sh.dq + 2 * sh.dkv
        ng = lambda cin: cin // (self.group if self.group else cin)
        lins = dict(qkv=(nq, sh.d), o=(sh.d, sh.dq), gu=(2 * sh.ffn, sh.d), d=(sh.d, sh.ffn))
        out = {}
        for k, (co, ci) in lins.items():
            out["codes_" + k] = torch.empty(co, ci * self.wbits // 8, dtype=torch.uint8, device=dev)
            out["h_" + k] = torch.empty(co, ng(ci), dtype=torch.float32, device=dev)
            out["z_" + k] = torch.empty(co, ng(ci), dtype=torch.int32, device=dev)
        if self.let:
            f32 = dict(dtype=torch.float32, device=dev)
            out.update(b_qkv=torch.empty(nq, **f32), b_o=torch.empty(sh.d, **f32), b_gu=torch.empty(2 * sh.ffn, **f32),
                       ln1_gain=torch.empty(sh.d, **f32), ln1_bias=torch.empty(sh.d, **f32),
                       ln2_gain=torch.empty(sh.d, **f32), ln2_bias=torch.empty(sh.d, **f32),
                       sa=torch.empty(sh.dkv, **f32))
        c_out = _lib.omq_block_packed(*[(out[n].data_ptr() if n in out else None) for n in _lib.PACKED_FIELDS])
        ws = torch.empty(_lib.omq_block_pack_workspace_size(self.c_shape, self.cfg), dtype=torch.uint8, device=dev)
        _lib.omq_block_fold_pack(self.c_shape, self.c_w, self.c_theta, self.cfg, c_out, ws, stream)
        return out

    def _split(self, src, prefix: str) -> Dict[str, np.ndarray]:
        out = {}
        sh = self.shape
        sizes = dict(qkv=[sh.dq, sh.dkv, sh.dkv], o=[sh.d], gu=[sh.ffn, sh.ffn], d=[sh.d])
        for key, parts in LWC_PARTS.items():
            for gb in ("gamma", "beta"):
                name = f"{gb}_{key}"
                if name not in src:
                    continue
                g = src[name].float().cpu().numpy()
                off = 0
                for p, n in zip(parts, sizes[key]):
                    out[f"{prefix}{gb}_{p}"] = g[off:off + n]
                    off += n
        for k in LET_NAMES:
            if k in src:
                out[prefix + k] = src[k].float().cpu().numpy()
        return out

    def split_grads(self) -> Dict[str, np.ndarray]:
        """Gradients on the host, named like the oracle's parameters (d<name>)."""
        return self._split(self.grads, "d")

    def split_theta(self) -> Dict[str, np.ndarray]:
        """Parameters on the host, named like the oracle's parameters."""
        return self._split(self.theta, "")
