"""The bench line's roofline: one calibration step as the unit, its algorithmic flops and bytes
against the measured peaks (no GPU needed: the arithmetic of the fraction only)."""
import os
import sys

import pytest

sys.path.insert(0, os.path.dirname(os.path.dirname(os.path.abspath(__file__))))
import bench  # noqa: E402

PEAKS = dict(hbm=6780.0, bf16=1908.6, bf16_sus=1705.1, src="measured")


def test_tensor_bound_step():
    # the LLaMA-7B W4A4 step: 2.59 TFLOP and 2.76 GB of algorithmic work in 2.657 ms
    F, B, ms = 2589915611136.0, 2764046336.0, 2.6569534
    r = bench.step_roofline(F, B, ms, PEAKS)
    assert r["bound"] == "tensor" and r["unit"] == "TFLOP/s" and r["peak"] == 1908.6
    assert r["achieved"] == pytest.approx(F / (ms * 1e-3) / 1e12)
    assert r["frac"] == pytest.approx(r["achieved"] / r["peak"])
    assert r["frac"] == pytest.approx(r["t_roof_ms"] / ms)           # the same as t_roof / t_step
    assert r["frac"] == pytest.approx(0.5107, abs=1e-4)
    assert r["traffic"] is None


def test_hbm_bound_step():
    F, B, ms = 1e9, 6.78e9, 2.0                                      # 0.5 us of flops, 1 ms of bytes
    r = bench.step_roofline(F, B, ms, PEAKS)
    assert r["bound"] == "hbm" and r["unit"] == "GB/s" and r["peak"] == 6780.0
    assert r["achieved"] == pytest.approx(B / (ms * 1e-3) / 1e9)
    assert r["frac"] == pytest.approx(0.5)
    assert r["t_roof_ms"] == pytest.approx(1.0)


def test_latency_label_keeps_the_arithmetic():
    r = bench.step_roofline(4.0e8, 0.0, 0.055, PEAKS, bound="latency")
    assert r["bound"] == "latency" and r["unit"] == "TFLOP/s"
    assert r["frac"] == pytest.approx(4.0e8 / 0.055e-3 / 1e12 / 1908.6)
