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


def _uniform_workload(mode):
    from paper_2609_19868_gb300 import workloads as wl

    return wl.make("decode_small", small=True).with_mode(mode)


@pytest.mark.parametrize("mode", [0, 1])
def test_per_sequence_roofline_of_a_uniform_batch_is_the_single_intensity_one(mode):
    """Every sequence of decode_small has the same shape, so the per-sequence
    ideal time is the batch's bytes / HBM (or flops / bf16), whichever is
    larger, and the entry's peak is the measured one."""
    w = _uniform_workload(mode)
    c = bench.algorithmic_counts(w)
    ideal, hbm, tc, wide = bench.per_sequence_roofline(w, 6691.1, 1926.3)
    assert ideal == pytest.approx(max(c["attn_bytes"] / 6691.1e9, c["flops"] / 1926.3e12))
    assert ideal == pytest.approx(wide)
    e = bench.roofline_per_sequence(w, c, attn_ms=ideal * 1e3 * 2, hbm_peak=6691.1,
                                    tf_peak=1926.3, peak_src="measured", traffic=None)
    assert e["peak"] in (6691.1, 1926.3)
    assert e["frac"] == pytest.approx(0.5, abs=1e-4)


def test_per_sequence_roofline_of_a_mixed_batch():
    """Hand-built two-sequence batch: one sequence is HBM-bound (a long prefix
    read by 4 rows), the other tensor-bound (a short prefix read by 512 rows).
    The ideal time is the sum of their own bounds, which is at least the
    batch-wide max(bytes / HBM, flops / bf16), and frac = ideal / measured."""
    from dataclasses import replace

    import numpy as np

    w = _uniform_workload(1)
    w = replace(w, B=2, cache_lens=np.array([16384, 1024], np.int32),
                n_slots=np.array([1, 16], np.int32), slot_len=np.array([4, 32], np.int32),
                mask_mode=np.array([1, 0], np.int32), Hq=32, Hkv=8, D=128,
                q_row_offsets=np.array([0, 4, 516], np.int32))
    hbm_gbs, tf = 6691.1, 1926.3
    P = np.array([16384, 1024]); R = np.array([4, 512])
    byts = 8 * (P + R) * 128 * 2 * 2 + 2 * R * 32 * 128 * 2
    pairs = np.array([32 * (4 * 16384 + 4 * 5 // 2), 32 * 512 * (1024 + 512)])
    flops = 4 * 128 * pairs
    t_h, t_t = byts / (hbm_gbs * 1e9), flops / (tf * 1e12)
    assert t_h[0] > t_t[0] and t_t[1] > t_h[1]
    ideal, hbm, tc, wide = bench.per_sequence_roofline(w, hbm_gbs, tf)
    assert ideal == pytest.approx(t_h[0] + t_t[1])
    assert hbm == pytest.approx(t_h[0]) and tc == pytest.approx(t_t[1])
    assert wide == pytest.approx(max(byts.sum() / (hbm_gbs * 1e9), flops.sum() / (tf * 1e12)))
    assert wide <= ideal
    c = {"attn_bytes": int(byts.sum()), "flops": int(flops.sum())}
    e = bench.roofline_per_sequence(w, c, attn_ms=ideal * 1e3 / 0.8, hbm_peak=hbm_gbs,
                                    tf_peak=tf, peak_src="measured", traffic=None)
    assert e["frac"] == pytest.approx(0.8, abs=1e-4)
    assert e["achieved"] / e["peak"] == pytest.approx(e["frac"], abs=1e-3)
    assert e["peak_measured"] == (tf if e["bound"] == "tensor" else hbm_gbs)


def test_sustained_tensor_peak_and_the_burst_fraction_beside_it():
    """Launches timed in long loops are held against the sustained bf16 rate;
    the entry also gives the fraction against the burst rate, which is lower
    for a tensor-bound batch (its ideal time is shorter)."""
    w = wl_make_long()
    c = bench.algorithmic_counts(w)
    ideal_s = bench.per_sequence_roofline(w, 6691.1, 1749.2)[0]
    ideal_b = bench.per_sequence_roofline(w, 6691.1, 1926.3)[0]
    e = bench.roofline_per_sequence(w, c, attn_ms=ideal_s * 1e3 / 0.7, hbm_peak=6691.1,
                                    tf_peak=1749.2, peak_src="measured", traffic=None,
                                    tf_kind="sustained", tf_burst=1926.3)
    assert e["bound"] == "tensor" and e["peak"] == 1749.2
    assert e["frac"] == pytest.approx(0.7, abs=1e-4)
    assert e["frac_of_burst_bf16"] == pytest.approx(0.7 * ideal_b / ideal_s, abs=1e-4)
    assert e["frac_of_burst_bf16"] < e["frac"]
    assert "sustained" in e["peak_source"]


def wl_make_long():
    from paper_2609_19868_gb300 import workloads as wl

    return wl.make("long_ctx", small=True).with_mode(0)


def test_paged_subset_keeps_each_sequences_attention(oracle_mod):
    """bench's oracle samples of a paged batch keep only the sampled
    sequences' pages, renumbered: their attention must be unchanged."""
    import numpy as np

    from _helpers import oracle_full, oracle_staged
    from paper_2609_19868_gb300 import workloads as wl

    w = wl.make("serving_mix", small=True, B=4)
    full = oracle_full(oracle_mod, w, *oracle_staged(oracle_mod, w))
    sub = bench.workload_subset(w, [0, 2])
    assert sub.n_pages < w.n_pages
    got = oracle_full(oracle_mod, sub, *oracle_staged(oracle_mod, sub))
    offs = w.q_row_offsets
    want = np.concatenate([full[offs[0]:offs[1]], full[offs[2]:offs[3]]])
    assert np.array_equal(got, want)
