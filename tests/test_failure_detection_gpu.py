"""Failure detection on the GPU without a fault: a bounded device wait that runs out.

omq_selftest_bounded_wait runs the library's tensor-core product on one CTA with a short wait
limit and, on request, without its first operand load (nothing ever completes that wait).  The
kernel must end on its own, report OMQ_ERR_TIMEOUT through the status word, and leave the
context usable: the same product and an ordinary omq_gemm_bf16 right afterwards are exact."""
import pytest
import torch

from paper_2308_13137_gb300 import _lib

pytestmark = pytest.mark.gpu


def _operands(M, N, K, seed):
    g = torch.Generator().manual_seed(seed)
    A = torch.randn(M, K, generator=g).to(torch.bfloat16)
    B = torch.randn(N, K, generator=g).to(torch.bfloat16)
    return A, B, A.double() @ B.double().T


def _rel(a, b):
    a, b = a.double().cpu(), b.double().cpu()
    return float((a - b).norm() / b.norm())


@pytest.mark.parametrize("K", [64, 256, 1024])
def test_expired_wait_reports_timeout_and_context_stays_usable(cuda_lib, K):
    M, N = 128, 128
    A, B, ref = _operands(M, N, K, K)
    Ad, Bd = A.cuda(), B.cuda()
    C = torch.empty(M, N, device="cuda")
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    # an ordinary product under a 100 ms limit
    _lib.omq_selftest_bounded_wait(M, N, K, Ad, Bd, C, 100_000_000, 0, st)
    assert _lib.omq_stream_status(st) == 0
    assert _rel(C, ref) < 1e-5
    # the first load withheld: every wait is limited to 50 us and the one for that load expires
    _lib.omq_selftest_bounded_wait(M, N, K, Ad, Bd, C, 50_000, 1, st)
    assert _lib.omq_stream_status(st) == 6                 # OMQ_ERR_TIMEOUT
    # the context is intact: the status word is cleared and both entry points compute exactly
    st.zero_()
    C.zero_()
    _lib.omq_selftest_bounded_wait(M, N, K, Ad, Bd, C, 100_000_000, 0, st)
    assert _lib.omq_stream_status(st) == 0
    assert _rel(C, ref) < 1e-5
    C2 = torch.empty(M, N, device="cuda")
    assert _lib.lib().omq_gemm_bf16(_lib.stream_handle(), M, N, K, 1, Ad.data_ptr(), K, 0, 1, Bd.data_ptr(), K, 0, 1,
                                    C2.data_ptr(), None, N, 0, 1.0, None, None, 0, 0.0, 0, st.data_ptr()) == 0
    assert _lib.omq_stream_status(st) == 0
    assert _rel(C2, ref) < 1e-5


def test_selftest_argument_checks(cuda_lib):
    A = torch.zeros(128, 64, dtype=torch.bfloat16, device="cuda")
    C = torch.empty(128, 128, device="cuda")
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    L = _lib.lib()
    h = _lib.stream_handle()
    # more rows than one CTA takes, a limit above one second, a bad withhold flag: refused on the host
    assert L.omq_selftest_bounded_wait(h, 256, 128, 64, A.data_ptr(), A.data_ptr(), C.data_ptr(), 50_000, 1,
                                       st.data_ptr()) == 2
    assert L.omq_selftest_bounded_wait(h, 128, 128, 64, A.data_ptr(), A.data_ptr(), C.data_ptr(), 2_000_000_000, 1,
                                       st.data_ptr()) == 1
    assert L.omq_selftest_bounded_wait(h, 128, 128, 64, A.data_ptr(), A.data_ptr(), C.data_ptr(), 50_000, 2,
                                       st.data_ptr()) == 1
    assert _lib.omq_stream_status(st) == 0
