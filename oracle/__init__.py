"""fp64 CPU oracle of the OmniQuant block-calibration step.

TEST INFRASTRUCTURE ONLY.  Only `tests/`, `__graft_entry__.smoke()` and the
`cpu_baseline` / `--impl reference` legs of `bench.py` may import or run this
package.  It shares no code with the CUDA path (`paper_2308_13137_gb300`) and
imports nothing from it; the two are fed the same seeded tensors from
`paper_2308_13137_gb300.inputs`, a module that holds no arithmetic of the
method.
"""
from .omq_oracle import *  # noqa: F401,F403
