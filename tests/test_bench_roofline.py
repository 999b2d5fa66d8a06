"""bench.py's roofline entries, checked on CPU: the attention kernel is put on
the HBM or the tensor roofline by its arithmetic intensity against the ridge
of the two peaks, and the T > 0 draw on the integer-multiply roofline of
Philox4x32-10 (10 multiply results per logit)."""
import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

import bench  # noqa: E402


def test_low_intensity_goes_on_the_hbm_roofline():
    counts = {"attn_bytes": 70e6, "flops": 4.3e9}          # 61 flop/byte, below a 288 ridge
    e = bench.roofline_entry(counts, attn_gbs=4000.0, attn_tflops=246.0, hbm_peak=6691.1,
                             tf_peak=1926.3, peak_src="measured", traffic=None)
    assert e["bound"] == "hbm" and e["unit"] == "GB/s"
    assert e["frac"] == pytest.approx(4000.0 / 6691.1, abs=1e-4)


def test_high_intensity_goes_on_the_tensor_roofline():
    counts = {"attn_bytes": 1e6, "flops": 1e9}             # 1000 flop/byte, above the ridge
    e = bench.roofline_entry(counts, attn_gbs=1000.0, attn_tflops=1400.0, hbm_peak=6691.1,
                             tf_peak=1926.3, peak_src="measured", traffic=123)
    assert e["bound"] == "tensor" and e["unit"] == "TFLOP/s"
    assert e["frac"] == pytest.approx(1400.0 / 1926.3, abs=1e-4)
    assert e["traffic"] == 123


def test_alu_roofline_counts_philox_multiplies():
    n_logits, ms = 1_000_000, 0.5
    e = bench.alu_roofline_entry(n_logits, ms, sms=152, mhz=2070.0, kernel="k")
    assert e["bound"] == "alu"
    assert e["peak"] == pytest.approx(64 * 152 * 2070e6 / 1e9, abs=0.1)
    achieved = n_logits * 10 / (ms * 1e-3) / 1e9                # 10 results per logit
    assert e["achieved"] == pytest.approx(achieved, abs=0.1)
    assert e["frac"] == pytest.approx(achieved / e["peak"], abs=1e-4)
    assert e["algorithmic_muls"] == 10 * n_logits
