"""Host-side checks of the C ABI that need no GPU: the library loads, exports every function
include/omq.h declares, sizes its workspaces, and rejects bad arguments before any launch."""
import ctypes
import os

import pytest

from paper_2308_13137_gb300 import _lib, inputs as I

pytestmark = pytest.mark.skipif(not os.path.exists(_lib.LIB_PATH), reason="libomq.so not built")


def test_exports_every_declared_function():
    L = _lib.lib()
    names = _lib.header_functions()
    assert len(names) >= 15
    for n in names:
        assert hasattr(L, n), n
        assert n in _lib._SIGS, f"binding lacks {n}"
    assert _lib.omq_version() == 1
    assert _lib.omq_status_string(3).startswith("misaligned")


def test_every_exported_function_is_declared():
    """The reverse direction: no omq_ symbol leaves the library undocumented by the header."""
    import shutil
    import subprocess
    if not shutil.which("nm"):
        pytest.skip("nm not available")
    out = subprocess.run(["nm", "-D", "--defined-only", _lib.LIB_PATH], capture_output=True, text=True,
                         check=True).stdout
    exported = {f[2] for f in (line.split() for line in out.splitlines())
                if len(f) == 3 and f[1] == "T" and f[2].startswith("omq_")}
    assert exported and exported <= set(_lib.header_functions()), sorted(exported - set(_lib.header_functions()))


def _cfg(**kw):
    base = dict(wbits=4, abits=16, group=128, let=0, h_eps=1e-5, accumulate=0, dev_status=None, pbits=0, wprep=0)
    base.update(kw)
    return _lib.omq_qcfg(base["wbits"], base["abits"], base["group"], base["let"], base["h_eps"],
                         base["accumulate"], base["dev_status"], base["pbits"], base["wprep"])


FAKE = 0x10000     # 16-byte aligned dummy address: every call below returns before touching it


def _lwc_fwd(Cout, Cin, cfg, W=FAKE, Wq=FAKE):
    L = _lib.lib()
    return L.omq_lwc_fakequant_fwd(None, Cout, Cin, W, None, None, FAKE, FAKE, Wq, None, FAKE, FAKE, FAKE, FAKE,
                                   None, None, None, ctypes.byref(cfg) if cfg is not None else None)


def test_argument_errors_before_launch():
    assert _lwc_fwd(0, 512, _cfg()) == 2                       # OMQ_ERR_SHAPE
    assert _lwc_fwd(64, 500, _cfg(group=0)) == 3               # inner dimension not a multiple of 8
    assert _lwc_fwd(64, 512, _cfg(group=96)) == 2              # group does not divide Cin
    assert _lwc_fwd(64, 512, _cfg(wbits=1)) == 4               # OMQ_ERR_UNSUPPORTED
    assert _lwc_fwd(64, 512, _cfg(wbits=12)) == 4
    assert _lwc_fwd(64, 512, None) == 1                        # OMQ_ERR_INVALID_ARG
    assert _lwc_fwd(64, 512, _cfg(wprep=2)) == 1               # operand preparation mode outside {0, 1}
    assert _lwc_fwd(64, 512, _cfg(), W=FAKE + 4) == 3          # misaligned pointer
    L = _lib.lib()
    # workspace too small
    assert L.omq_block_loss(None, 1024, FAKE, FAKE, FAKE, None, None, FAKE, 4) == 7
    # GEMM: misaligned leading dimension
    assert L.omq_gemm_bf16(None, 128, 128, 64, 1, FAKE, 60, 0, 1, FAKE, 64, 0, 1, FAKE, None, 128, 0, 1.0,
                           None, None, 0, 0.0, 0, None) == 3
    # GEMM: bad causal mode
    assert L.omq_gemm_bf16(None, 128, 128, 64, 1, FAKE, 64, 0, 1, FAKE, 64, 0, 1, FAKE, None, 128, 0, 1.0,
                           None, None, 0, 0.0, 7, None) == 1


def test_softmax_quant_argument_errors():
    """The softmax-output quantizer's bit width and step floor are checked before any launch."""
    L = _lib.lib()
    assert _lwc_fwd(64, 512, _cfg(pbits=9)) == 4               # pbits outside 2..8 (0 / 16 = off)
    assert _lwc_fwd(64, 512, _cfg(pbits=1)) == 4
    for bits in (1, 9, 16, 0):
        assert L.omq_attention_pq_fwd(None, 256, 2, 2, FAKE, 256, FAKE, FAKE, 256, FAKE, 256, FAKE, bits, 1e-5,
                                      FAKE, None) == 4
        assert L.omq_attention_pq_bwd(None, 256, 2, 2, FAKE, 256, FAKE, FAKE, 256, FAKE, FAKE, 256, FAKE, 256, FAKE,
                                      FAKE, 256, bits, FAKE, FAKE, None) == 4
    assert L.omq_attention_pq_fwd(None, 256, 2, 2, FAKE, 256, FAKE, FAKE, 256, FAKE, 256, FAKE, 8, 0.0,
                                  FAKE, None) == 1             # h_eps must be positive
    assert L.omq_attention_pq_fwd(None, 256, 2, 2, FAKE, 256, FAKE, FAKE, 256, FAKE, 256, FAKE, 8, 1e-5,
                                  None, None) == 1             # the row records are required


def test_qlinear_saved_sizes():
    """Element counts of the single linear's saved arrays, in the struct's field order."""
    n = _lib.omq_qlinear_saved_sizes(256, 512, 384, _cfg(group=128))
    ng = 384 * 4
    assert n == [384 * 512, ng, ng, ng, ng, 256 * 512, 256, 256, 256, 256, 384]
    assert _lib.omq_qlinear_saved_sizes(256, 512, 384, _cfg(group=0))[1] == 384
    with pytest.raises(_lib.OmqError):
        _lib.omq_qlinear_saved_sizes(256, 512, 384, _cfg(group=96))       # 96 does not divide 512


def test_block_workspace_sizes():
    sh = I.SHAPES["llama7b_w4a4"]
    s = _lib.omq_block_shape(sh.T, sh.d, sh.n_heads, sh.n_kv, sh.head_dim, sh.ffn, sh.rms_eps, sh.rope_theta)
    ws = _lib.omq_block_workspace_size(s, _cfg(wbits=4, abits=4, group=0, let=1))
    assert 2e9 < ws < 8e9                                      # a few GB for the 7B block step
    bad = _lib.omq_block_shape(sh.T, sh.d, 32, 5, 128, sh.ffn, 1e-6, 1e4)    # heads not divisible
    assert _lib.omq_block_workspace_size(bad, _cfg()) == 0
    hd64 = _lib.omq_block_shape(sh.T, sh.d, 64, 64, 64, sh.ffn, 1e-6, 1e4)   # head_dim must be 128
    assert _lib.omq_block_workspace_size(hd64, _cfg()) == 0
    assert _lib.omq_qlinear_workspace_size(256, 512, 512, _cfg()) > 512 * 512 * 4
    # the softmax-quantized step carries two small per-row arrays more
    ws8 = _lib.omq_block_workspace_size(s, _cfg(wbits=4, abits=4, group=0, let=1, pbits=8))
    assert ws < ws8 < ws + 16 * sh.n_heads * sh.T * 4
    assert _lib.omq_block_workspace_size(s, _cfg(wbits=4, abits=4, group=0, let=1, pbits=12)) == 0
