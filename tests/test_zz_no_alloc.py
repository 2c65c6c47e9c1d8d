"""The allocation-free block loss (omq_block_loss_noalloc) against omq_block_loss.

Callers that cannot allocate device memory (a fixed arena owned by another framework, an interface
that passes only inputs and outputs, or code that must not call cudaMalloc/cudaFree while work is in
flight) use the variant whose scratch is a static array inside the library.  Two calls in a row,
with different sizes and data, must give what the workspace entry point gives, and sizes outside
the stated limit must be refused before anything runs."""
import pytest
import torch

from paper_2308_13137_gb300 import _lib

pytestmark = pytest.mark.gpu


def _workspace_loss(n, Yq, Yf):
    loss = torch.zeros(1, device="cuda")
    dY = torch.empty(n, device="cuda")
    dYb = torch.empty(n, dtype=torch.bfloat16, device="cuda")
    ws = torch.empty(_lib.omq_loss_workspace_size(n), dtype=torch.uint8, device="cuda")
    _lib.omq_block_loss(n, Yq, Yf, loss, dY, dYb, ws)
    return loss, dY, dYb


def test_noalloc_loss_matches_workspace_loss(cuda_lib):
    for n, seed in ((2048 * 4096 + 8, 1), (3000, 2)):          # two calls in a row
        g = torch.Generator().manual_seed(seed)
        Yq = torch.randn(n, generator=g).cuda()
        Yf = torch.randn(n, generator=g).cuda()
        loss = torch.full((1,), float("nan"), device="cuda")
        dY = torch.empty(n, device="cuda")
        dYb = torch.empty(n, dtype=torch.bfloat16, device="cuda")
        _lib.omq_block_loss_noalloc(n, Yq, Yf, loss, dY, dYb)
        ref_loss, ref_dY, ref_dYb = _workspace_loss(n, Yq, Yf)
        torch.cuda.synchronize()
        assert abs(float(loss) - float(ref_loss)) <= 1e-5 * abs(float(ref_loss))
        assert float((dY - ref_dY).norm() / ref_dY.norm()) <= 1e-6
        assert torch.equal(dYb, ref_dYb)


def test_noalloc_loss_rejects_sizes_outside_the_limit(cuda_lib):
    t = torch.zeros(8, device="cuda")
    for n in (0, -5, 2 ** 31):
        with pytest.raises(_lib.OmqError) as e:
            _lib.omq_block_loss_noalloc(n, t, t, t[:1], None, None)
        assert e.value.code == 2                                 # OMQ_ERR_SHAPE
