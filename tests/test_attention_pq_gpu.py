"""Softmax-output quantization variant of the attention (the ablation beside Table A7) through
omq_attention_pq_fwd / omq_attention_pq_bwd against the oracle's `softmax_quant` (per query row
MinMax over the visible keys, STE backward with the h path) composed with the plain causal
attention in fp64 on the same bf16 inputs; the quantized probabilities enter P V rounded to bf16
as in the kernel (R13).  Several 128-row blocks, a ragged tail, GQA, 2 to 8 bits."""
import math

import pytest
import torch

import oracle as O
from paper_2308_13137_gb300 import _lib

pytestmark = pytest.mark.gpu

CASES = [  # T, heads, kv heads, bits
    (256, 2, 2, 8),
    (200, 2, 1, 6),     # ragged last block, two query heads per kv head
    (384, 2, 2, 4),
    (256, 2, 1, 3),
    (128, 1, 1, 2),
]
EPS = 1e-5


def _rel(a, b):
    a, b = torch.as_tensor(a).double().cpu(), torch.as_tensor(b).double().cpu()
    return float((a - b).norm() / b.norm().clamp_min(1e-300))


def _ref(Q, K, V, dO, H, Hkv, bits, plain_ste=False):
    T = Q.shape[0]
    rep = H // Hkv
    q = Q.double().reshape(T, H, 128).transpose(0, 1).requires_grad_(True)
    k = K.double().reshape(T, Hkv, 128).transpose(0, 1).requires_grad_(True)
    v = V.double().reshape(T, Hkv, 128).transpose(0, 1).requires_grad_(True)
    kk, vv = k.repeat_interleave(rep, 0), v.repeat_interleave(rep, 0)
    s = q @ kk.transpose(-1, -2) / math.sqrt(128)
    s = s.masked_fill(~torch.ones(T, T, dtype=torch.bool).tril(), float("-inf"))
    P = torch.softmax(s, -1)
    Pq = O.softmax_quant(P, bits, EPS)
    if plain_ste:              # identity gradient: no clamp mask, no h path (a deliberately wrong backward)
        Pq = P + (Pq - P).detach()
    Pb = Pq + (O.to_bf16(Pq.detach()) - Pq.detach())          # bf16 operand, gradient unchanged
    o = Pb @ vv
    Ot = o.transpose(0, 1).reshape(T, H * 128)
    gq, gk, gv = torch.autograd.grad(Ot, [q, k, v], dO.double())
    f = lambda g, n: g.transpose(0, 1).reshape(T, n * 128)
    return Ot.detach(), f(gq, H), f(gk, Hkv), f(gv, Hkv), P.detach()


@pytest.mark.parametrize("T,H,Hkv,bits", CASES)
def test_attention_pq_fwd_bwd(cuda_lib, T, H, Hkv, bits):
    g = torch.Generator().manual_seed(T * 11 + bits)
    Q = (torch.randn(T, H * 128, generator=g) * 1.5).to(torch.bfloat16)
    K = (torch.randn(T, Hkv * 128, generator=g) * 1.5).to(torch.bfloat16)
    V = torch.randn(T, Hkv * 128, generator=g).to(torch.bfloat16)
    dO = torch.randn(T, H * 128, generator=g).to(torch.bfloat16)
    rO, rdQ, rdK, rdV, P = _ref(Q.float(), K.float(), V.float(), dO.float(), H, Hkv, bits)
    d = lambda t: t.cuda().contiguous()
    Qd, Kd, Vd, dOd = d(Q), d(K), d(V), d(dO)
    Od = torch.empty(T, H * 128, device="cuda")
    lse = torch.empty(H, T, device="cuda")
    pqr = torch.empty(H, T, 8, device="cuda")
    pqb = torch.empty(H, T, 4, device="cuda")
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    _lib.omq_attention_pq_fwd(T, H, Hkv, Qd, H * 128, Kd, Vd, Hkv * 128, Od, H * 128, lse, bits, EPS, pqr, st)
    dQ = torch.empty(T, H * 128, device="cuda")
    dK = torch.empty(T, Hkv * 128, device="cuda")
    dV = torch.empty(T, Hkv * 128, device="cuda")
    _lib.omq_attention_pq_bwd(T, H, Hkv, Qd, H * 128, Kd, Vd, Hkv * 128, lse, dOd, H * 128, dQ, H * 128, dK, dV,
                              Hkv * 128, bits, pqr, pqb, st)
    torch.cuda.synchronize()
    assert int(st.item()) == 0
    # the row quantizers: first indices of the extremes exact, h and z from the fp32 decision
    pr = pqr.cpu().double()
    causal = torch.ones(T, T, dtype=torch.bool).tril()
    Pv = P.masked_fill(~causal, float("nan"))
    want_imax = torch.nan_to_num(Pv, nan=-1.0).argmax(-1)
    want_imin = torch.nan_to_num(Pv, nan=2.0).argmin(-1)
    assert torch.equal(pr[..., 6].long(), want_imax)
    assert torch.equal(pr[..., 7].long(), want_imin)
    Mx = P.gather(-1, want_imax[..., None])[..., 0]
    mn = P.gather(-1, want_imin[..., None])[..., 0]
    h_ref = torch.clamp((Mx - mn) / (2 ** bits - 1), min=EPS)
    assert float(((pr[..., 0] - h_ref).abs() / h_ref).max()) < 1e-5
    z_ref = -torch.round(mn / h_ref)
    assert float((pr[..., 2] != z_ref).double().mean()) < 0.01
    errs = dict(O=_rel(Od, rO), dQ=_rel(dQ, rdQ), dK=_rel(dK, rdK), dV=_rel(dV, rdV))
    print(T, H, Hkv, bits, errs)
    assert errs["O"] < 1e-2
    for n in ("dQ", "dK", "dV"):
        assert errs[n] < 2e-2, (n, errs)
    if bits <= 3:
        # the h path matters at low bit widths: a backward without it would be far off
        _, wdQ, wdK, _, _ = _ref(Q.float(), K.float(), V.float(), dO.float(), H, Hkv, bits, plain_ste=True)
        assert errs["dQ"] < 0.2 * _rel(wdQ, rdQ) and errs["dK"] < 0.2 * _rel(wdK, rdK)


@pytest.mark.full
@pytest.mark.parametrize("bits", [8, 4])
def test_attention_pq_full_size(cuda_lib, bits):
    """The LLaMA-7B attention of the step (2048 tokens, 32 heads of 128) with the softmax output
    quantized: the kernels run the whole grid; heads 0 and 31 are checked against the oracle
    composition in full (every row, every key)."""
    T, H, Hkv = 2048, 32, 32
    g = torch.Generator().manual_seed(2048 + bits)
    Q = (torch.randn(T, H * 128, generator=g) * 1.5).to(torch.bfloat16)
    K = (torch.randn(T, Hkv * 128, generator=g) * 1.5).to(torch.bfloat16)
    V = torch.randn(T, Hkv * 128, generator=g).to(torch.bfloat16)
    dO = torch.randn(T, H * 128, generator=g).to(torch.bfloat16)
    d = lambda t: t.cuda().contiguous()
    Od = torch.empty(T, H * 128, device="cuda")
    lse = torch.empty(H, T, device="cuda")
    pqr = torch.empty(H, T, 8, device="cuda")
    pqb = torch.empty(H, T, 4, device="cuda")
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    dQ = torch.empty(T, H * 128, device="cuda")
    dK = torch.empty(T, Hkv * 128, device="cuda")
    dV = torch.empty(T, Hkv * 128, device="cuda")
    Qd, Kd, Vd, dOd = d(Q), d(K), d(V), d(dO)
    _lib.omq_attention_pq_fwd(T, H, Hkv, Qd, H * 128, Kd, Vd, Hkv * 128, Od, H * 128, lse, bits, EPS, pqr, st)
    _lib.omq_attention_pq_bwd(T, H, Hkv, Qd, H * 128, Kd, Vd, Hkv * 128, lse, dOd, H * 128, dQ, H * 128, dK, dV,
                              Hkv * 128, bits, pqr, pqb, st)
    torch.cuda.synchronize()
    assert int(st.item()) == 0
    for hh in (0, H - 1):
        cols = slice(hh * 128, (hh + 1) * 128)
        rO, rdQ, rdK, rdV, _ = _ref(Q[:, cols].float(), K[:, cols].float(), V[:, cols].float(),
                                    dO[:, cols].float(), 1, 1, bits)
        errs = dict(O=_rel(Od[:, cols], rO), dQ=_rel(dQ[:, cols], rdQ), dK=_rel(dK[:, cols], rdK),
                    dV=_rel(dV[:, cols], rdV))
        print(hh, bits, errs)
        assert errs["O"] < 1e-2
        for n in ("dQ", "dK", "dV"):
            assert errs[n] < 2e-2, (n, errs)
