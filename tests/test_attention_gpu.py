"""Causal attention through omq_attention_fwd / omq_attention_bwd against the plain definition
(Sec. 3.3: softmax(Q K^T / sqrt(d)) V over keys j <= t, softmax output not quantized) in fp64 on
the same bf16 inputs, with gradients by autograd.  Several 128-row blocks, a ragged tail, GQA."""
import math

import numpy as np
import pytest
import torch

from paper_2308_13137_gb300 import _lib

pytestmark = pytest.mark.gpu

CASES = [  # T, heads, kv heads
    (256, 2, 2),
    (200, 2, 1),        # ragged last block, two query heads per kv head
    (384, 4, 2),
    (128, 1, 1),
]


def _rel(a, b):
    a, b = torch.as_tensor(a).double().cpu(), torch.as_tensor(b).double().cpu()
    return float((a - b).norm() / b.norm().clamp_min(1e-300))


def _ref(Q, K, V, dO, H, Hkv):
    T = Q.shape[0]
    rep = H // Hkv
    q = Q.double().reshape(T, H, 128).transpose(0, 1).requires_grad_(True)
    k = K.double().reshape(T, Hkv, 128).transpose(0, 1).requires_grad_(True)
    v = V.double().reshape(T, Hkv, 128).transpose(0, 1).requires_grad_(True)
    kk, vv = k.repeat_interleave(rep, 0), v.repeat_interleave(rep, 0)
    s = q @ kk.transpose(-1, -2) / math.sqrt(128)
    s = s.masked_fill(~torch.ones(T, T, dtype=torch.bool).tril(), float("-inf"))
    lse2 = torch.logsumexp(s, -1) / math.log(2.0)
    o = torch.softmax(s, -1) @ vv
    O = o.transpose(0, 1).reshape(T, H * 128)
    gq, gk, gv = torch.autograd.grad(O, [q, k, v], dO.double())
    f = lambda g, n: g.transpose(0, 1).reshape(T, n * 128)
    return O.detach(), lse2.detach(), f(gq, H), f(gk, Hkv), f(gv, Hkv)


@pytest.mark.parametrize("T,H,Hkv", CASES)
def test_attention_fwd_bwd(cuda_lib, T, H, Hkv):
    g = torch.Generator().manual_seed(T * 7 + H)
    Q = (torch.randn(T, H * 128, generator=g) * 1.5).to(torch.bfloat16)
    K = (torch.randn(T, Hkv * 128, generator=g) * 1.5).to(torch.bfloat16)
    V = torch.randn(T, Hkv * 128, generator=g).to(torch.bfloat16)
    dO = torch.randn(T, H * 128, generator=g).to(torch.bfloat16)
    rO, rL, rdQ, rdK, rdV = _ref(Q.float(), K.float(), V.float(), dO.float(), H, Hkv)
    d = lambda t: t.cuda().contiguous()
    Qd, Kd, Vd, dOd = d(Q), d(K), d(V), d(dO)
    O = torch.empty(T, H * 128, device="cuda")
    lse = torch.empty(H, T, device="cuda")
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    _lib.omq_attention_fwd(T, H, Hkv, Qd, H * 128, Kd, Vd, Hkv * 128, O, H * 128, lse, st)
    D = torch.empty(H, T, device="cuda")
    dQ = torch.empty(T, H * 128, device="cuda")
    dK = torch.empty(T, Hkv * 128, device="cuda")
    dV = torch.empty(T, Hkv * 128, device="cuda")
    _lib.omq_attention_bwd(T, H, Hkv, Qd, H * 128, Kd, Vd, Hkv * 128, O, H * 128, lse, dOd, H * 128, D,
                           dQ, H * 128, dK, dV, Hkv * 128, st)
    torch.cuda.synchronize()
    assert int(st.item()) == 0
    # P enters the P V product rounded to bf16 (relative error <= 2^-9 per element)
    assert _rel(O, rO) < 1e-2
    # fp32 max and sum of exp2 (ex2.approx, relative error ~2^-22) against fp64
    assert float((lse.cpu().double() - rL).abs().max()) < 1e-4
    for got, ref in ((dQ, rdQ), (dK, rdK), (dV, rdV)):
        assert _rel(got, ref) < 2e-2
