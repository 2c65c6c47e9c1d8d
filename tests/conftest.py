import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)
TESTS = os.path.dirname(os.path.abspath(__file__))
if TESTS not in sys.path:
    sys.path.insert(0, TESTS)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (sm_103a) and the built libomq")
    config.addinivalue_line("markers", "full: runs the full workload sizes (minutes of oracle time on the host)")


def pytest_terminal_summary(terminalreporter, exitstatus, config):
    """Code-decision and stage parity counts of the GPU tests (exempt elements are reported, not
    hidden): one line per check; also written as JSON lines to $OMQ_PARITY_REPORT when set."""
    import _parity
    if not _parity.REPORT:
        return
    _parity.dump_report()
    tr = terminalreporter
    tr.section("parity report")
    for r in _parity.REPORT:
        if r["kind"] in ("codes", "zero points"):
            tr.write_line(f"{r['kind']:>11} {r['name']}: {r['elements']} elements, {r['mismatches']} differ "
                          f"({r['in_tie_window']} within 1e-6 of a tie, {r['in_input_band']} within the input's "
                          f"rounding band, {r['outside']} outside); {r['near_ties']} within 1e-6 of a tie")
        else:
            vals = ", ".join(f"{k}={v:.3e}" if isinstance(v, float) else f"{k}={v}"
                             for k, v in r.items() if k not in ("kind", "name"))
            tr.write_line(f"{r['kind']:>11} {r['name']}: {vals}")


@pytest.fixture(scope="session")
def cuda_lib():
    """The C-ABI library on cuda:0; fails loudly when the GPU or the build is missing."""
    import torch
    if not torch.cuda.is_available():
        pytest.fail("gpu test selected but no CUDA device is visible")
    from paper_2308_13137_gb300 import _lib
    return _lib.lib()
