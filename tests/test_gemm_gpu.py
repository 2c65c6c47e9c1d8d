"""tcgen05 GEMM through the C ABI against the exact (fp64) product of the same bf16 operands."""
import pytest
import torch

from paper_2308_13137_gb300 import _lib

pytestmark = pytest.mark.gpu
F64 = torch.float64


def _bf16(shape, gen, scale=1.0):
    return (torch.randn(*shape, generator=gen) * scale).to(torch.bfloat16)


def _rel(a, b):
    return float((a.double() - b.double()).norm() / b.double().norm().clamp_min(1e-300))


def _logical(t, kmajor, rows, k):
    """[rows, k] view of a stored operand (K-major: stored [rows, k]; MN-major: stored [k, rows])."""
    return t if kmajor else t.T


CASES = [  # M, N, K, a_kmajor, b_kmajor
    (256, 512, 320, 1, 1),
    (200, 384, 200, 1, 1),
    (256, 256, 192, 0, 1),
    (256, 512, 256, 1, 0),
    (384, 256, 128, 0, 0),
    (128, 128, 72, 0, 0),
    (136, 264, 136, 1, 0),
]


@pytest.mark.parametrize("M,N,K,ak,bk", CASES)
def test_gemm_layouts(cuda_lib, M, N, K, ak, bk):
    g = torch.Generator().manual_seed(M * 7 + N + K + 3 * ak + bk)
    A = _bf16((M, K) if ak else (K, M), g)
    B = _bf16((N, K) if bk else (K, N), g)
    ref = _logical(A, ak, M, K).double() @ _logical(B, bk, N, K).double().T
    Ad, Bd = A.cuda(), B.cuda()
    C = torch.full((M, N), float("nan"), device="cuda")
    Cb = torch.empty((M, N), dtype=torch.bfloat16, device="cuda")
    _lib.omq_gemm_bf16(M, N, K, 1, Ad, K if ak else M, 0, ak, Bd, K if bk else N, 0, bk, C, Cb, N, 0)
    torch.cuda.synchronize()
    assert _rel(C.cpu(), ref) < 2e-5
    assert torch.equal(Cb.cpu(), C.cpu().to(torch.bfloat16))


def test_gemm_epilogue(cuda_lib):
    g = torch.Generator().manual_seed(5)
    M, N, K = 256, 512, 256
    A, B = _bf16((M, K), g), _bf16((N, K), g)
    bias = torch.randn(N, generator=g)
    R = torch.randn(M, N, generator=g)
    C0 = torch.randn(M, N, generator=g)
    ref = 0.5 * (A.double() @ B.double().T) + bias.double() + R.double() + 2.0 * C0.double()
    C = C0.cuda()
    _lib.omq_gemm_bf16(M, N, K, 1, A.cuda(), K, 0, 1, B.cuda(), K, 0, 1, C, None, N, 0, alpha=0.5, bias=bias.cuda(),
                       R=R.cuda(), ldr=N, beta_acc=2.0)
    torch.cuda.synchronize()
    assert _rel(C.cpu(), ref) < 2e-5


def test_gemm_batched_strided_heads(cuda_lib):
    """Per-head products on a [T, H*128] layout (the attention scores), batch = head."""
    g = torch.Generator().manual_seed(6)
    T, H, hd = 256, 3, 128
    Q, K_ = _bf16((T, H * hd), g), _bf16((T, H * hd), g)
    S = torch.zeros(H, T, T, device="cuda")
    _lib.omq_gemm_bf16(T, T, hd, H, Q.cuda(), H * hd, hd, 1, K_.cuda(), H * hd, hd, 1, S, None, T, T * T, alpha=0.25)
    torch.cuda.synchronize()
    for h in range(H):
        ref = 0.25 * Q[:, h * hd:(h + 1) * hd].double() @ K_[:, h * hd:(h + 1) * hd].double().T
        assert _rel(S[h].cpu(), ref) < 2e-5


def test_gemm_causal_modes(cuda_lib):
    g = torch.Generator().manual_seed(7)
    T, hd = 384, 128
    Q, K_ = _bf16((T, hd), g), _bf16((T, hd), g)
    P = torch.tril(torch.rand(T, T, generator=g)).to(torch.bfloat16)        # zero above the diagonal
    V = _bf16((T, hd), g)
    # mode 1: tiles entirely above the diagonal are not written
    S = torch.full((T, T), 7.0, device="cuda")
    _lib.omq_gemm_bf16(T, T, hd, 1, Q.cuda(), hd, 0, 1, K_.cuda(), hd, 0, 1, S, None, T, 0, causal=1)
    # mode 2: O = P V with k < end of the query tile
    O = torch.zeros(T, hd, device="cuda")
    _lib.omq_gemm_bf16(T, hd, T, 1, P.cuda(), T, 0, 1, V.cuda(), hd, 0, 0, O, None, hd, 0, causal=2)
    # mode 3: dV = P^T dO with k >= start of the key tile
    dO = _bf16((T, hd), g)
    dV = torch.zeros(T, hd, device="cuda")
    _lib.omq_gemm_bf16(T, hd, T, 1, P.cuda(), T, 0, 0, dO.cuda(), hd, 0, 0, dV, None, hd, 0, causal=3)
    torch.cuda.synchronize()
    full = Q.double() @ K_.double().T
    Sc = S.cpu()
    lower = torch.tril(torch.ones(T, T, dtype=torch.bool))
    assert _rel(Sc[lower], full[lower]) < 2e-5
    assert float(Sc[0:128, 128:].sub(7.0).abs().max()) == 0.0               # skipped tiles untouched
    assert _rel(O.cpu(), P.double() @ V.double()) < 2e-5
    assert _rel(dV.cpu(), P.double().T @ dO.double()) < 2e-5


def test_gemm_large_weight_shape(cuda_lib):
    """One projection-sized product (2048 x 4096 x 4096), sampled rows checked exactly."""
    g = torch.Generator().manual_seed(8)
    M, N, K = 2048, 4096, 4096
    A, B = _bf16((M, K), g), _bf16((N, K), g, 0.02)
    C = torch.empty(M, N, device="cuda")
    _lib.omq_gemm_bf16(M, N, K, 1, A.cuda(), K, 0, 1, B.cuda(), K, 0, 1, C, None, N, 0)
    torch.cuda.synchronize()
    rows = torch.randint(0, M, (64,), generator=g)
    ref = A[rows].double() @ B.double().T
    assert _rel(C.cpu()[rows], ref) < 2e-5


# Shapes whose tiles do not fill whole waves of the 76 CTA pairs (or 152 CTAs): fewer tiles than
# CTAs, a partial last wave, ragged rows, short K; with bias and residual in the epilogue.
SPLIT_CASES = [  # M, N, K, a_kmajor, b_kmajor
    (1024, 2816, 4096, 1, 1),   # 44 pair tiles: fewer tiles than workers, each tile cut over 2-3 pairs
    (2048, 5376, 1024, 1, 0),   # 168 pair tiles: one wave of whole tiles, then a cut tail
    (1000, 1152, 2048, 0, 1),   # one CTA per 128 x 128 tile (N not a multiple of 256), ragged M, 72 tiles
    (4096, 2304, 512, 0, 0),    # 144 pair tiles of 8 k-blocks
    # projection-shaped products (N = 4096, 12288) with K-major and MN-major B
    (2048, 4096, 512, 1, 1),
    (2048, 4096, 512, 1, 0),
    (2048, 4096, 320, 0, 0),
    (2048, 12288, 256, 1, 1),
    (2048, 12288, 256, 1, 0),
]


@pytest.mark.parametrize("M,N,K,ak,bk", SPLIT_CASES)
def test_gemm_split_tail(cuda_lib, M, N, K, ak, bk):
    g = torch.Generator().manual_seed(M + N + K + 3 * ak + bk)
    A = _bf16((M, K) if ak else (K, M), g)
    B = _bf16((N, K) if bk else (K, N), g, 0.05)
    bias = torch.randn(N, generator=g)
    R = torch.randn(M, N, generator=g)
    ref = 0.5 * (_logical(A, ak, M, K).double() @ _logical(B, bk, N, K).double().T) + bias.double() + R.double()
    Ad, Bd, bd, Rd = A.cuda(), B.cuda(), bias.cuda(), R.cuda()
    outs = []
    for _ in range(3):   # repeated launches give identical results
        C = torch.full((M, N), float("nan"), device="cuda")
        Cb = torch.empty((M, N), dtype=torch.bfloat16, device="cuda")
        _lib.omq_gemm_bf16(M, N, K, 1, Ad, K if ak else M, 0, ak, Bd, K if bk else N, 0, bk, C, Cb, N, 0, alpha=0.5,
                           bias=bd, R=Rd, ldr=N)
        outs.append((C.cpu(), Cb.cpu()))
    torch.cuda.synchronize()
    for C, Cb in outs:
        assert _rel(C, ref) < 2e-5
        assert torch.equal(Cb, C.to(torch.bfloat16))
        assert torch.equal(C, outs[0][0])
