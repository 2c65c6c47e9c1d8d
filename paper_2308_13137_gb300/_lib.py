"""ctypes binding of libomq (include/omq.h).

Every function here has the name of the C entry point it calls and only marshals arguments:
torch tensors become device pointers, the current CUDA stream becomes the stream argument, and
a non-zero status raises OmqError.  There is no fallback: when libomq.so is missing or no GPU
is visible the calls raise.
"""
from __future__ import annotations

import ctypes
import os
import re
from ctypes import POINTER, Structure, c_float, c_int32, c_int64, c_size_t, c_void_p, c_char_p
from typing import Optional

PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(PKG, "libomq.so")
HEADER = os.path.join(os.path.dirname(PKG), "include", "omq.h")

OMQ_OK = 0
STATUS_NAMES = {0: "OMQ_OK", 1: "OMQ_ERR_INVALID_ARG", 2: "OMQ_ERR_SHAPE", 3: "OMQ_ERR_ALIGN",
                4: "OMQ_ERR_UNSUPPORTED", 5: "OMQ_ERR_CUDA", 6: "OMQ_ERR_TIMEOUT", 7: "OMQ_ERR_WORKSPACE"}


class OmqError(RuntimeError):
    def __init__(self, fn: str, code: int):
        super().__init__(f"{fn} returned {STATUS_NAMES.get(code, code)}")
        self.code = code


class omq_qcfg(Structure):
    _fields_ = [("wbits", c_int32), ("abits", c_int32), ("group", c_int32), ("let", c_int32),
                ("h_eps", c_float), ("accumulate", c_int32), ("dev_status", c_void_p), ("pbits", c_int32),
                ("wprep", c_int32)]


class omq_qlinear_saved(Structure):
    _fields_ = [("w_hat", c_void_p), ("h_w", c_void_p), ("z_w", c_void_p), ("imax_w", c_void_p),
                ("imin_w", c_void_p), ("x_hat", c_void_p), ("h_a", c_void_p), ("z_a", c_void_p),
                ("imax_a", c_void_p), ("imin_a", c_void_p), ("b_tilde", c_void_p)]


class omq_block_shape(Structure):
    _fields_ = [("T", c_int32), ("d", c_int32), ("n_heads", c_int32), ("n_kv", c_int32),
                ("head_dim", c_int32), ("ffn", c_int32), ("rms_eps", c_float), ("rope_theta", c_float)]


class omq_block_weights(Structure):
    _fields_ = [("wqkv", c_void_p), ("wo", c_void_p), ("wgu", c_void_p), ("wd", c_void_p)]


PARAM_FIELDS = ["gamma_qkv", "beta_qkv", "gamma_o", "beta_o", "gamma_gu", "beta_gu", "gamma_d", "beta_d",
                "s1", "d1", "so", "do_", "sa", "s2", "d2"]


class omq_block_params(Structure):
    _fields_ = [(n, c_void_p) for n in PARAM_FIELDS]


PACKED_FIELDS = ["codes_qkv", "codes_o", "codes_gu", "codes_d", "h_qkv", "z_qkv", "h_o", "z_o", "h_gu", "z_gu",
                 "h_d", "z_d", "b_qkv", "b_o", "b_gu", "ln1_gain", "ln1_bias", "ln2_gain", "ln2_bias", "sa"]


class omq_block_packed(Structure):
    _fields_ = [(n, c_void_p) for n in PACKED_FIELDS]


SAVED_FIELDS = ["a_hat", "a_h", "a_z", "y_qkv", "qkv_h", "qkv_z", "q_hat", "k_hat", "v_hat", "o", "o_hat", "o_h", "o_z", "h1", "b_hat", "b_h",
                "b_z", "y_gu", "m_hat", "m_h", "m_z"]
SAVED_BWD_FIELDS = ["dy", "dy_gu", "dh1", "do_bf16", "dy_qkv"]


class omq_block_saved(Structure):
    _fields_ = ([(n, c_int64) for n in SAVED_FIELDS] + [("w_hat", c_int64 * 4), ("w_h", c_int64 * 4),
                                                          ("w_z", c_int64 * 4)] +
                [(n, c_int64) for n in SAVED_BWD_FIELDS])


LET_STATS_FIELDS = ["a_absmax", "a_sum", "q_absmax", "k_absmax", "o_absmax", "o_sum", "b_absmax", "b_sum"]


class omq_let_stats(Structure):
    _fields_ = [(n, c_void_p) for n in LET_STATS_FIELDS]


P, I64, I32, F32, SZ = c_void_p, c_int64, c_int32, c_float, c_size_t
_SIGS = {
    "omq_let_apply": (I32, [P, I64, I64, I64, P, P, P, P, P, P, P, P, P]),
    "omq_lwc_fakequant_fwd": (I32, [P, I64, I64, P, P, P, P, P, P, P, P, P, P, P, P, P, P, P]),
    "omq_lwc_fakequant_bwd": (I32, [P, I64, I64, P, P, P, P, P, P, P, P, P, P, P, P, P, P, P, P, P, P, SZ, P]),
    "omq_lwc_bwd_workspace_size": (SZ, [I64, I64]),
    "omq_act_quant_per_token": (I32, [P, I64, I64, P, P, P, P, P, P, P, P, P, P]),
    "omq_act_quant_per_token_bwd": (I32, [P, I64, I64, P, P, P, P, P, P, P, P, P, P, P, P, SZ, P]),
    "omq_act_bwd_workspace_size": (SZ, [I64, I64]),
    "omq_block_loss": (I32, [P, I64, P, P, P, P, P, P, SZ]),
    "omq_loss_workspace_size": (SZ, [I64]),
    "omq_block_loss_noalloc": (I32, [P, I64, P, P, P, P, P]),
    "omq_gemm_bf16": (I32, [P, I64, I64, I64, I64, P, I64, I64, I32, P, I64, I64, I32, P, P, I64, I64, F32,
                            P, P, I64, F32, I32, P]),
    "omq_selftest_bounded_wait": (I32, [P, I64, I64, I64, P, P, P, ctypes.c_uint64, I32, P]),
    "omq_qlinear_fwd": (I32, [P, I64, I64, I64, P, P, P, P, P, P, P, P, P, P]),
    "omq_qlinear_bwd": (I32, [P, I64, I64, I64, P, P, P, P, P, P, P, P, P, P, P, P, P, P, SZ, P]),
    "omq_qlinear_workspace_size": (SZ, [I64, I64, I64, P]),
    "omq_block_workspace_size": (SZ, [P, P]),
    "omq_block_forward": (I32, [P, P, P, P, P, P, P, SZ, P]),
    "omq_block_step": (I32, [P, P, P, P, P, P, P, P, P, P, SZ, P]),
    "omq_block_saved_layout": (I32, [P, P, P]),
    "omq_attention_fwd": (I32, [P, I32, I32, I32, P, I64, P, P, I64, P, I64, P, P]),
    "omq_attention_bwd": (I32, [P, I32, I32, I32, P, I64, P, P, I64, P, I64, P, P, I64, P, P, I64, P, P, I64,
                                P]),
    "omq_qlinear_saved_sizes": (I32, [I64, I64, I64, P, P]),
    "omq_attention_pq_fwd": (I32, [P, I32, I32, I32, P, I64, P, P, I64, P, I64, P, I32, F32, P, P]),
    "omq_attention_pq_bwd": (I32, [P, I32, I32, I32, P, I64, P, P, I64, P, P, I64, P, I64, P, P, I64, I32, P, P,
                                   P]),
    "omq_block_pack_workspace_size": (SZ, [P, P]),
    "omq_block_fold_pack": (I32, [P, P, P, P, P, P, P, SZ]),
    "omq_let_stats_accumulate": (I32, [P, P, P, P, P, I32, P, SZ, P]),
    "omq_let_init_workspace_size": (SZ, [P]),
    "omq_let_init": (I32, [P, P, P, P, I64, F32, P, P, SZ]),
    "omq_adamw_update": (I32, [P, I64, P, P, P, P, F32, F32, F32, F32, F32, I32]),
    "omq_adamw_update_dev": (I32, [P, I64, P, P, P, P, F32, F32, F32, F32, F32, P]),
    "omq_step_advance": (I32, [P, P]),
    "omq_stream_status": (I32, [P, P, POINTER(c_int32)]),
    "omq_status_string": (c_char_p, [I32]),
    "omq_version": (I32, []),
    "omq_launch_count": (I64, []),
    "omq_profile_begin": (None, []),
    "omq_profile_end": (I32, [POINTER(ctypes.c_double), POINTER(ctypes.c_double), POINTER(c_int64)]),
}

_LIB: Optional[ctypes.CDLL] = None


def header_functions():
    """Names of the functions include/omq.h declares."""
    with open(HEADER) as fh:
        text = fh.read()
    return sorted(set(re.findall(r"^\s*(?:omq_status|size_t|int32_t|int64_t|void|const char\*)\s+(omq_\w+)\s*\(",
                                 text, re.M)))


def lib() -> ctypes.CDLL:
    """Load libomq.so (raises when it has not been built)."""
    global _LIB
    if _LIB is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError(f"{LIB_PATH} is missing: build it with `python -m paper_2308_13137_gb300.build`")
        L = ctypes.CDLL(LIB_PATH)
        for name, (res, args) in _SIGS.items():
            fn = getattr(L, name)
            fn.restype = res
            fn.argtypes = args
        _LIB = L
    return _LIB


# ------------------------------------------------------------------------------------------------
# marshalling helpers
# ------------------------------------------------------------------------------------------------

def ptr(t) -> Optional[int]:
    """Device pointer of a CUDA tensor (None passes NULL)."""
    if t is None:
        return None
    if not t.is_cuda:
        raise ValueError("libomq takes device tensors only")
    if not t.is_contiguous():
        raise ValueError("libomq takes contiguous tensors only")
    return t.data_ptr()


def stream_handle(stream=None) -> Optional[int]:
    import torch
    s = stream if stream is not None else torch.cuda.current_stream()
    return s.cuda_stream


def check(name: str, code: int):
    if code != OMQ_OK:
        raise OmqError(name, code)


def make_cfg(wbits=4, abits=16, group=0, let=0, h_eps=1e-5, accumulate=0, dev_status=None, pbits=16,
             wprep=0) -> omq_qcfg:
    return omq_qcfg(wbits, abits, group, int(let), h_eps, accumulate, ptr(dev_status), pbits, int(wprep))


# ------------------------------------------------------------------------------------------------
# same-name wrappers
# ------------------------------------------------------------------------------------------------

def omq_let_apply(T, Cin, Cout, X, W, B, s, delta, Xt, Wt, Bt, cfg, stream=None):
    check("omq_let_apply", lib().omq_let_apply(stream_handle(stream), T, Cin, Cout, ptr(X), ptr(W), ptr(B), ptr(s),
                                               ptr(delta), ptr(Xt), ptr(Wt), ptr(Bt), ctypes.byref(cfg)))


def omq_lwc_fakequant_fwd(Cout, Cin, W, s, r, gamma_logit, beta_logit, Wq, codes, h, z, argmax, argmin,
                          bias_delta, bias_shift, Bt, cfg, stream=None):
    check("omq_lwc_fakequant_fwd", lib().omq_lwc_fakequant_fwd(
        stream_handle(stream), Cout, Cin, ptr(W), ptr(s), ptr(r), ptr(gamma_logit), ptr(beta_logit), ptr(Wq),
        ptr(codes), ptr(h), ptr(z), ptr(argmax), ptr(argmin), ptr(bias_delta), ptr(bias_shift), ptr(Bt),
        ctypes.byref(cfg)))


def omq_lwc_bwd_workspace_size(Cout, Cin) -> int:
    return lib().omq_lwc_bwd_workspace_size(Cout, Cin)


def omq_lwc_fakequant_bwd(Cout, Cin, W, s, r, gamma_logit, beta_logit, h, z, argmax, argmin, dWq, dgamma, dbeta,
                          dWt, ds, dr, dBt, ddelta, workspace, cfg, stream=None):
    ws_bytes = 0 if workspace is None else workspace.numel() * workspace.element_size()
    check("omq_lwc_fakequant_bwd", lib().omq_lwc_fakequant_bwd(
        stream_handle(stream), Cout, Cin, ptr(W), ptr(s), ptr(r), ptr(gamma_logit), ptr(beta_logit), ptr(h), ptr(z),
        ptr(argmax), ptr(argmin), ptr(dWq), ptr(dgamma), ptr(dbeta), ptr(dWt), ptr(ds), ptr(dr), ptr(dBt),
        ptr(ddelta), ptr(workspace), ws_bytes, ctypes.byref(cfg)))


def omq_act_quant_per_token(T, C, X, s, delta, Xq, codes, h, z, argmax, argmin, cfg, stream=None):
    check("omq_act_quant_per_token", lib().omq_act_quant_per_token(
        stream_handle(stream), T, C, ptr(X), ptr(s), ptr(delta), ptr(Xq), ptr(codes), ptr(h), ptr(z), ptr(argmax),
        ptr(argmin), ctypes.byref(cfg)))


def omq_act_bwd_workspace_size(T, C) -> int:
    return lib().omq_act_bwd_workspace_size(T, C)


def omq_act_quant_per_token_bwd(T, C, X, s, delta, h, z, argmax, argmin, dXq, dX, ds, ddelta, workspace, cfg,
                                stream=None):
    ws_bytes = 0 if workspace is None else workspace.numel() * workspace.element_size()
    check("omq_act_quant_per_token_bwd", lib().omq_act_quant_per_token_bwd(
        stream_handle(stream), T, C, ptr(X), ptr(s), ptr(delta), ptr(h), ptr(z), ptr(argmax), ptr(argmin), ptr(dXq),
        ptr(dX), ptr(ds), ptr(ddelta), ptr(workspace), ws_bytes, ctypes.byref(cfg)))


def omq_loss_workspace_size(n) -> int:
    return lib().omq_loss_workspace_size(n)


def omq_block_loss(n, Yq, Yfp, loss, dY, dY_bf16, workspace, stream=None):
    ws_bytes = workspace.numel() * workspace.element_size()
    check("omq_block_loss", lib().omq_block_loss(stream_handle(stream), n, ptr(Yq), ptr(Yfp), ptr(loss), ptr(dY),
                                                 ptr(dY_bf16), ptr(workspace), ws_bytes))


def omq_block_loss_noalloc(n, Yq, Yfp, loss, dY, dY_bf16, stream=None):
    """omq_block_loss without a workspace: the scratch is a 4 KB device array inside the library.
    For callers that cannot allocate device memory; calls that overlap on the GPU race."""
    check("omq_block_loss_noalloc", lib().omq_block_loss_noalloc(stream_handle(stream), n, ptr(Yq), ptr(Yfp),
                                                                 ptr(loss), ptr(dY), ptr(dY_bf16)))


def omq_gemm_bf16(M, N, K, batch, A, a_ld, a_bs, a_kmajor, B, b_ld, b_bs, b_kmajor, Cf, Cb, ldc, c_bs, alpha=1.0,
                  bias=None, R=None, ldr=0, beta_acc=0.0, causal=0, dev_status=None, stream=None):
    check("omq_gemm_bf16", lib().omq_gemm_bf16(
        stream_handle(stream), M, N, K, batch, ptr(A), a_ld, a_bs, a_kmajor, ptr(B), b_ld, b_bs, b_kmajor, ptr(Cf),
        ptr(Cb), ldc, c_bs, alpha, ptr(bias), ptr(R), ldr, beta_acc, causal, ptr(dev_status)))


def omq_attention_fwd(T, n_heads, n_kv, Q, ldq, K, V, ldkv, O, ldo, lse, dev_status=None, stream=None):
    check("omq_attention_fwd", lib().omq_attention_fwd(
        stream_handle(stream), T, n_heads, n_kv, ptr(Q), ldq, ptr(K), ptr(V), ldkv, ptr(O), ldo, ptr(lse),
        ptr(dev_status)))


def omq_attention_bwd(T, n_heads, n_kv, Q, ldq, K, V, ldkv, O, ldo, lse, dO, lddo, D, dQ, ldg, dK, dV, ldgkv,
                      dev_status=None, stream=None):
    check("omq_attention_bwd", lib().omq_attention_bwd(
        stream_handle(stream), T, n_heads, n_kv, ptr(Q), ldq, ptr(K), ptr(V), ldkv, ptr(O), ldo, ptr(lse), ptr(dO),
        lddo, ptr(D), ptr(dQ), ldg, ptr(dK), ptr(dV), ldgkv, ptr(dev_status)))


def omq_qlinear_saved_sizes(T, Cin, Cout, cfg):
    sizes = (c_int64 * 11)()
    check("omq_qlinear_saved_sizes", lib().omq_qlinear_saved_sizes(T, Cin, Cout, ctypes.byref(cfg), sizes))
    return list(sizes)


def omq_attention_pq_fwd(T, n_heads, n_kv, Q, ldq, K, V, ldkv, O, ldo, lse, pbits, h_eps, pq_rows,
                         dev_status=None, stream=None):
    check("omq_attention_pq_fwd", lib().omq_attention_pq_fwd(
        stream_handle(stream), T, n_heads, n_kv, ptr(Q), ldq, ptr(K), ptr(V), ldkv, ptr(O), ldo, ptr(lse), pbits,
        h_eps, ptr(pq_rows), ptr(dev_status)))


def omq_attention_pq_bwd(T, n_heads, n_kv, Q, ldq, K, V, ldkv, lse, dO, lddo, dQ, ldg, dK, dV, ldgkv, pbits,
                         pq_rows, pq_stats, dev_status=None, stream=None):
    check("omq_attention_pq_bwd", lib().omq_attention_pq_bwd(
        stream_handle(stream), T, n_heads, n_kv, ptr(Q), ldq, ptr(K), ptr(V), ldkv, ptr(lse), ptr(dO), lddo,
        ptr(dQ), ldg, ptr(dK), ptr(dV), ldgkv, pbits, ptr(pq_rows), ptr(pq_stats), ptr(dev_status)))


def omq_block_pack_workspace_size(shape, cfg) -> int:
    return lib().omq_block_pack_workspace_size(ctypes.byref(shape), ctypes.byref(cfg))


def omq_block_fold_pack(shape, weights, theta, cfg, out, workspace, stream=None):
    ws_bytes = workspace.numel() * workspace.element_size()
    check("omq_block_fold_pack", lib().omq_block_fold_pack(
        stream_handle(stream), ctypes.byref(shape), ctypes.byref(weights), ctypes.byref(theta), ctypes.byref(cfg),
        ctypes.byref(out), ptr(workspace), ws_bytes))


def omq_let_stats_accumulate(shape, weights, x, stats, first, workspace, dev_status=None, stream=None):
    ws_bytes = workspace.numel() * workspace.element_size()
    check("omq_let_stats_accumulate", lib().omq_let_stats_accumulate(
        stream_handle(stream), ctypes.byref(shape), ctypes.byref(weights), ptr(x), ctypes.byref(stats), int(first),
        ptr(workspace), ws_bytes, ptr(dev_status)))


def omq_let_init_workspace_size(shape) -> int:
    return lib().omq_let_init_workspace_size(ctypes.byref(shape))


def omq_let_init(shape, weights, stats, ntok, alpha, theta, workspace, stream=None):
    ws_bytes = workspace.numel() * workspace.element_size()
    check("omq_let_init", lib().omq_let_init(
        stream_handle(stream), ctypes.byref(shape), ctypes.byref(weights), ctypes.byref(stats), ntok, alpha,
        ctypes.byref(theta), ptr(workspace), ws_bytes))


def omq_qlinear_fwd(T, Cin, Cout, X, W, B, s, delta, gamma_logit, beta_logit, Y, saved, cfg, stream=None):
    check("omq_qlinear_fwd", lib().omq_qlinear_fwd(
        stream_handle(stream), T, Cin, Cout, ptr(X), ptr(W), ptr(B), ptr(s), ptr(delta), ptr(gamma_logit),
        ptr(beta_logit), ptr(Y), ctypes.byref(saved), ctypes.byref(cfg)))


def omq_qlinear_workspace_size(T, Cin, Cout, cfg) -> int:
    return lib().omq_qlinear_workspace_size(T, Cin, Cout, ctypes.byref(cfg))


def omq_qlinear_bwd(T, Cin, Cout, X, W, s, delta, gamma_logit, beta_logit, saved, dY, dX, dgamma, dbeta, ds, ddelta,
                    workspace, cfg, stream=None):
    ws_bytes = workspace.numel() * workspace.element_size()
    check("omq_qlinear_bwd", lib().omq_qlinear_bwd(
        stream_handle(stream), T, Cin, Cout, ptr(X), ptr(W), ptr(s), ptr(delta), ptr(gamma_logit), ptr(beta_logit),
        ctypes.byref(saved), ptr(dY), ptr(dX), ptr(dgamma), ptr(dbeta), ptr(ds), ptr(ddelta), ptr(workspace),
        ws_bytes, ctypes.byref(cfg)))


def omq_block_workspace_size(shape: omq_block_shape, cfg: omq_qcfg) -> int:
    return lib().omq_block_workspace_size(ctypes.byref(shape), ctypes.byref(cfg))


def omq_selftest_bounded_wait(M, N, K, A, B, C, wait_limit_ns, withhold, dev_status, stream=None):
    check("omq_selftest_bounded_wait", lib().omq_selftest_bounded_wait(
        stream_handle(stream), M, N, K, ptr(A), ptr(B), ptr(C), int(wait_limit_ns), int(withhold), ptr(dev_status)))


def omq_block_saved_layout(shape: omq_block_shape, cfg: omq_qcfg) -> omq_block_saved:
    out = omq_block_saved()
    check("omq_block_saved_layout", lib().omq_block_saved_layout(ctypes.byref(shape), ctypes.byref(cfg),
                                                                 ctypes.byref(out)))
    return out


def omq_block_forward(shape, weights, theta, x, y, workspace, cfg, stream=None):
    ws_bytes = workspace.numel() * workspace.element_size()
    check("omq_block_forward", lib().omq_block_forward(
        stream_handle(stream), ctypes.byref(shape), ctypes.byref(weights), ctypes.byref(theta), ptr(x), ptr(y),
        ptr(workspace), ws_bytes, ctypes.byref(cfg)))


def omq_block_step(shape, weights, theta, x, y_fp, y, loss, grads, workspace, cfg, stream=None):
    ws_bytes = workspace.numel() * workspace.element_size()
    check("omq_block_step", lib().omq_block_step(
        stream_handle(stream), ctypes.byref(shape), ctypes.byref(weights), ctypes.byref(theta), ptr(x), ptr(y_fp),
        ptr(y), ptr(loss), ctypes.byref(grads), ptr(workspace), ws_bytes, ctypes.byref(cfg)))


def omq_adamw_update(n, p, g, m, v, lr, beta1, beta2, eps, weight_decay, step, stream=None):
    check("omq_adamw_update", lib().omq_adamw_update(stream_handle(stream), n, ptr(p), ptr(g), ptr(m), ptr(v), lr,
                                                     beta1, beta2, eps, weight_decay, step))


def omq_adamw_update_dev(n, p, g, m, v, lr, beta1, beta2, eps, weight_decay, step_dev, stream=None):
    check("omq_adamw_update_dev", lib().omq_adamw_update_dev(stream_handle(stream), n, ptr(p), ptr(g), ptr(m), ptr(v),
                                                             lr, beta1, beta2, eps, weight_decay, ptr(step_dev)))


def omq_step_advance(step_dev, stream=None):
    check("omq_step_advance", lib().omq_step_advance(stream_handle(stream), ptr(step_dev)))


def omq_stream_status(dev_status, stream=None) -> int:
    out = c_int32(0)
    check("omq_stream_status", lib().omq_stream_status(stream_handle(stream), ptr(dev_status), ctypes.byref(out)))
    return out.value


def omq_status_string(code: int) -> str:
    return lib().omq_status_string(code).decode()


def omq_version() -> int:
    return lib().omq_version()


def omq_launch_count() -> int:
    return lib().omq_launch_count()


def omq_profile_begin():
    lib().omq_profile_begin()


def omq_profile_end():
    """Returns (GEMM device ms, algorithmic GEMM flops, GEMM launches) traced since begin."""
    ms, fl, n = ctypes.c_double(0), ctypes.c_double(0), c_int64(0)
    check("omq_profile_end", lib().omq_profile_end(ctypes.byref(ms), ctypes.byref(fl), ctypes.byref(n)))
    return ms.value, fl.value, n.value
