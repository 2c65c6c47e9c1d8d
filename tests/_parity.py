"""Shared parity helpers of the GPU tests: relative errors and the code-decision protocol.

Code decisions (Eq. 2, Sec. 3.2): the GPU's codes are compared with round(w / h) + z clamped to
[0, 2^N - 1], where w is the quantizer's input and h, z are the GPU's own step and zero point
(the shared-scale protocol: computing h separately in fp32 and fp64 moves w / h by a few 1e-7,
which alone would flip codes near a half).  The quotient is taken in float64.  Every element must
agree bit for bit except

* those whose exact quotient lies within TIE_WINDOW = 1e-6 of a .5 boundary (exempt, counted);
* where the GPU's fp32 quantizer input is itself a rounded value of the exact one (the LET
  division, RMSNorm, RoPE ...), those whose quotient lies within the input's rounding band of a
  .5 boundary (exempt, counted separately; the band is stated by each caller in quotient units).

Where the quantizer input is an exactly defined fp32 value (a weight W~ = fl32(s W), an
activation without a producer), the band is zero and only the tie window exempts.  Each check
appends a line to REPORT, which the session prints at its end.
"""
from __future__ import annotations

import json
import os

import torch

F64 = torch.float64
TIE_WINDOW = 1e-6
OUT_TOL, GRAD_TOL = 1e-2, 3e-2
REPORT = []


def rel(a, b) -> float:
    a, b = torch.as_tensor(a).double().cpu(), torch.as_tensor(b).double().cpu()
    return float((a - b).norm() / b.norm().clamp_min(1e-300))


def grad_errors(got, ref, names):
    """{d<name>: relative error} over parameter gradients; a gradient that is zero by structure in
    the reference (one token: the softmax of a single key has no gradient, so d s_a = 0 exactly) is
    measured by its size against the largest reference gradient instead."""
    scale = max([float(torch.as_tensor(ref["d" + n]).double().norm()) for n in names] + [1e-300])
    out = {}
    for n in names:
        r = torch.as_tensor(ref["d" + n]).double()
        if float(r.norm()) > 1e-9 * scale:
            out["d" + n] = rel(got["d" + n], r)
        else:
            out["d" + n] = float(torch.as_tensor(got["d" + n]).double().norm()) / scale
    return out


def fp32_band(mag, h, ulps: float):
    """Rounding band in quotient units of an fp32 value of magnitude `mag` formed with `ulps`
    single-precision roundings (each at most 2^-24 relative), divided by the step h."""
    return ulps * 2.0 ** -24 * torch.as_tensor(mag, dtype=F64).abs() / torch.as_tensor(h, dtype=F64)


def code_counts(name: str, x, codes_gpu, z, nbits: int, band=None):
    """Counts of the code comparison (see check_codes) without asserting or recording."""
    x = torch.as_tensor(x, dtype=F64)
    Q = 2 ** nbits - 1
    ref = torch.clamp(torch.round(x) + torch.as_tensor(z, dtype=F64)[..., None], 0, Q).to(torch.int64)
    got = torch.as_tensor(codes_gpu).to(torch.int64)
    dist = ((x - torch.floor(x)) - 0.5).abs()
    tie = dist < TIE_WINDOW
    inband = tie.clone() if band is None else dist < TIE_WINDOW + torch.as_tensor(band, dtype=F64)
    mism = got != ref
    return dict(name=name, elements=int(x.numel()), mismatches=int(mism.sum()),
                in_tie_window=int((mism & tie).sum()), in_input_band=int((mism & inband & ~tie).sum()),
                outside=int((mism & ~inband).sum()), near_ties=int(tie.sum()))


def add_counts(a, b):
    return {k: (a[k] + b[k] if k != "name" else a[k]) for k in a}


def record_codes(n):
    REPORT.append(dict(kind="codes", **n))
    assert n["outside"] == 0, n
    return n


def check_codes(name: str, x, codes_gpu, z, nbits: int, band=None):
    """x: float64 quotients w / h (groups on the last axis); codes_gpu: the GPU's codes, same shape;
    z: the GPU's zero points [...]; band: None or a tensor broadcastable to x (quotient units).
    Asserts that every mismatch is exempt; returns the counts."""
    return record_codes(code_counts(name, x, codes_gpu, z, nbits, band))


def check_zero_points(name: str, u_ref, z_gpu, z_ref=None, band_rel: float = 1e-6):
    """Zero points z = -round(beta min / h): GPU against the oracle's (z_ref; default -round(u_ref)),
    u_ref the oracle's float64 quotient.  The GPU forms u from its own fp32 clipping strengths and
    extremes, each within a few 1e-7 relative of the oracle's, so a mismatch is exempt where u lies
    within 1e-6 + band_rel |u| of a .5 boundary."""
    u = torch.as_tensor(u_ref, dtype=F64)
    ref = -torch.round(u) if z_ref is None else torch.as_tensor(z_ref, dtype=F64)
    got = torch.as_tensor(z_gpu, dtype=F64)
    dist = ((u - torch.floor(u)) - 0.5).abs()
    tie = dist < TIE_WINDOW
    inband = dist < TIE_WINDOW + band_rel * u.abs()
    mism = got != ref
    n = dict(name=name, elements=int(u.numel()), mismatches=int(mism.sum()),
             in_tie_window=int((mism & tie).sum()), in_input_band=int((mism & inband & ~tie).sum()),
             outside=int((mism & ~inband).sum()), near_ties=int(tie.sum()))
    REPORT.append(dict(kind="zero points", **n))
    assert n["outside"] == 0, n
    return n


def check_h(name: str, h_gpu, h_ref, aM=None, bm=None, Q: float = 1.0):
    """Step h: within 1e-6 relative of the oracle's float64 h, or, where a M and b m cancel (a group
    whose range is small against its magnitude), within the fp32 rounding of the difference."""
    hg, hr = torch.as_tensor(h_gpu, dtype=F64), torch.as_tensor(h_ref, dtype=F64)
    tol = 1e-6 * hr.abs()
    if aM is not None:
        tol = tol + 2.0 ** -22 * (torch.as_tensor(aM, dtype=F64).abs() + torch.as_tensor(bm, dtype=F64).abs()) / Q
    err = (hg - hr).abs()
    worst = float((err / hr.abs()).max())
    REPORT.append(dict(kind="step h", name=name, elements=int(hr.numel()), max_rel=worst))
    assert bool((err <= tol).all()), (name, worst)
    return worst


def record(kind: str, name: str, **vals):
    REPORT.append(dict(kind=kind, name=name, **vals))


def dump_report(path: str = None):
    path = path or os.environ.get("OMQ_PARITY_REPORT")
    if path and REPORT:
        os.makedirs(os.path.dirname(os.path.abspath(path)), exist_ok=True)
        with open(path, "w") as fh:
            for r in REPORT:
                fh.write(json.dumps(r) + "\n")
