"""Slot-decode step benchmark (one layer of Zarya Mode B, Sec. 5.2).

One step = the whole hot path over one batch:
  stage + attend  zarya_slot_attn_staged  the block's K/V -> cache positions
                  P_b.., then block rows over prefix + block (mask per sequence)
  commit          zarya_kv_commit_staged  P_b += accepted (the accepted rows,
                  first in the block, are already in place)
The commit writes the advanced lengths into a second array (a decoding
loop's ping-pong), so every step sees the same prefix lengths.

Default workload: serving_mix (B64, 32/8 heads, D128, bf16, paged cache of
16-token pages, prefixes log-uniform in [1024, 16384], 8 slots of 4 to 32
tokens, mask mode per sequence), the largest configuration. Inputs are
seeded and synthetic. Several independent copies of the KV cache rotate so
that the data touched between two uses of one copy exceeds the L2 cache.

Every measurement is a series of timed regions of K steps (at least --reps
of them, lasting at least --min-seconds), reported as the median region
(the minimum beside it). The line's `per_config` object repeats the
measurement for every configuration (tiny_fp32, decode_small, ragged_mid,
long_ctx in both mask modes, serving_mix), each with its roofline, the
oracle's time on the host cores and the end-to-end rate with host buffers.

Prints one JSON line. `--impl reference` times the fp64 CPU oracle instead
(rank 0 only), each step a bounded sample of the same workload.

`--path select` measures slot selection and token acceptance (Sec. 5.2
steps 3-6) instead: zarya_draft_select over a block's logits, then
zarya_verify_accept over the verification block it laid out.
"""
from __future__ import annotations

import argparse
import json
import math
import os
import subprocess
import sys
import tempfile
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

FALLBACK_HBM_GBS = 6800.0
FALLBACK_BF16_TFLOPS = 1900.0
FALLBACK_BF16_TFLOPS_SUSTAINED = 1700.0

WORKLOAD_LABELS = {
    "tiny_fp32": "tiny_fp32: B1, Hq4/Hkv2, D64, fp32, prefix 128, contiguous cache, "
                 "2 slots x 4 tokens, slot-causal, accept 3",
    "decode_small": "decode_small: B8, Hq16/Hkv8, D128, bf16, prefix 2048, contiguous cache, "
                    "4 slots x 8 tokens, slot-causal, accept ~U[0,R]",
    "ragged_mid": "ragged_mid: B32, Hq32/Hkv8, D128, bf16, prefix ~U[512,8192], contiguous, "
                  "8 slots x 16 tokens, block-bidirectional",
    "long_ctx_bidir": "long_ctx: B4, Hq32/Hkv8, D128, bf16, prefix 32768, contiguous, "
                      "16 slots x 32 tokens, block-bidirectional, accept ~U[0,512]",
    "long_ctx_causal": "long_ctx: B4, Hq32/Hkv8, D128, bf16, prefix 32768, contiguous, "
                       "16 slots x 32 tokens, slot-causal, accept ~U[0,512]",
    "serving_mix": "serving_mix: B64, Hq32/Hkv8, D128, bf16, paged 16-token pages, prefix "
                   "log-U[1024,16384], slot_len in {4,8,16,32} x 8 slots, mixed modes",
}
# older name of the slot-causal long_ctx entry
WORKLOAD_ALIASES = {"long_ctx": "long_ctx_causal"}


def algorithmic_counts(w):
    """Bytes / flops the method needs for one step, by the counting rules:
    K and V of every key a block row can see read once per KV head, Q read
    once, O written once; 4*D flops per visible (row, head, key) pair;
    staging and committing move R_b (resp. accepted) rows of K and V, read
    and written."""
    eb = 2 if w.dtype == "bf16" else 4
    P = w.cache_lens.astype(np.int64)
    R = w.R
    kv = int((w.Hkv * (P + R) * w.D * eb * 2).sum())
    qo = int(2 * w.rows * w.Hq * w.D * eb)
    pairs = 0
    for b in range(w.B):
        if w.mask_mode[b] == 0:
            pairs += w.Hq * int(R[b]) * int(P[b] + R[b])
        else:
            pairs += w.Hq * (int(R[b]) * int(P[b]) + int(R[b]) * (int(R[b]) + 1) // 2)
    row = w.Hkv * w.D * eb
    return dict(attn_bytes=kv + qo, kv_bytes=kv, flops=4 * w.D * pairs,
                stage_bytes=int(2 * 2 * R.sum() * row),
                commit_bytes=int(2 * 2 * w.accept_len.astype(np.int64).sum() * row))


def recorded_traffic(workload: str, kernel: str = "slot_attn_tc_kernel"):
    """DRAM bytes (read + write) of one attention launch from the committed ncu
    summary (profiles/<kernel>_<workload>.json), if it was taken on the current
    kernel sources; else None."""
    import hashlib

    path = os.path.join(ROOT, "profiles", f"{kernel}_{workload}.json")
    try:
        with open(path) as f:
            rec = json.load(f)
        h = hashlib.sha256()
        for src in rec["kernel_sources"]:
            with open(os.path.join(ROOT, src), "rb") as f:
                h.update(f.read())
        if h.hexdigest() != rec["kernel_sources_sha256"]:
            return None
        return int(rec["dram_bytes_read"]) + int(rec["dram_bytes_write"])
    except Exception:
        return None


def read_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            d = json.load(f)
        return float(d["hbm_gbs"]), float(d["bf16_tflops"]), "measured"
    except Exception:
        return FALLBACK_HBM_GBS, FALLBACK_BF16_TFLOPS, "fallback"


def read_sustained_bf16():
    """The bf16 GEMM rate held for seconds under the power cap: the tensor
    peak for kernels timed in long back-to-back loops, as the attention
    launches are here (the burst figure is for a kernel timed alone)."""
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            return float(json.load(f)["bf16_tflops_sustained"]), "measured"
    except Exception:
        return FALLBACK_BF16_TFLOPS_SUSTAINED, "fallback"


# ALU roofline of the draw at T > 0, bound by Philox4x32-10: 10 rounds per 4
# words (one word per logit), each round two 32 x 32 -> 64-bit products, i.e.
# four 32-bit multiply results: 10 integer multiply results per logit. Peak:
# 64 such results per clock per SM (the CUDA programming guide's throughput
# for compute capabilities 7.0 to 9.0, taken as unchanged) x SMs x max clock.
PHILOX_MULS_PER_LOGIT = 10
INT_MUL_PER_CLK_PER_SM = 64


def alu_roofline_entry(n_logits, ms, sms, mhz, kernel):
    """The T > 0 draw against the integer-multiply peak of `sms` SMs at `mhz`."""
    peak = INT_MUL_PER_CLK_PER_SM * sms * mhz * 1e6 / 1e9
    achieved = n_logits * PHILOX_MULS_PER_LOGIT / (ms * 1e-3) / 1e9
    return {"bound": "alu", "achieved": round(achieved, 1), "peak": round(peak, 1),
            "unit": "G int32 mul/s", "frac": round(achieved / peak, 4), "traffic": None,
            "kernel": kernel, "algorithmic_muls": n_logits * PHILOX_MULS_PER_LOGIT,
            "peak_source": (f"{INT_MUL_PER_CLK_PER_SM} 32-bit integer multiply results per clock "
                            f"per SM x {sms} SMs x {mhz:.0f} MHz "
                            "(Philox4x32-10: 10 multiply results per logit)")}


def alu_roofline(n_logits, ms, dev, kernel):
    import torch

    props = torch.cuda.get_device_properties(dev)
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            mhz = float(json.load(f)["sm_max_mhz"])
    except Exception:
        mhz = 2070.0
    return alu_roofline_entry(n_logits, ms, props.multi_processor_count, mhz, kernel)


def roofline_entry(counts, attn_gbs, attn_tflops, hbm_peak, tf_peak, peak_src, traffic):
    """The attention kernel against the roofline that bounds it: HBM when its
    arithmetic intensity (algorithmic flops per algorithmic byte) is below the
    ridge of the measured peaks, the bf16 tensor pipe above it."""
    ridge = tf_peak * 1e12 / (hbm_peak * 1e9)
    intensity = counts["flops"] / counts["attn_bytes"]
    if intensity <= ridge:
        entry = {"bound": "hbm", "achieved": round(attn_gbs, 1), "peak": hbm_peak, "unit": "GB/s",
                 "frac": round(attn_gbs / hbm_peak, 4), "traffic": traffic,
                 "peak_source": f"{peak_src} HBM copy bandwidth"}
    else:
        entry = {"bound": "tensor", "achieved": round(attn_tflops, 1), "peak": tf_peak,
                 "unit": "TFLOP/s", "frac": round(attn_tflops / tf_peak, 4), "traffic": traffic,
                 "peak_source": f"{peak_src} cuBLAS bf16 GEMM (burst)"}
    entry["intensity_flop_per_byte"] = round(intensity, 1)
    entry["ridge_flop_per_byte"] = round(ridge, 1)
    entry["kernel"] = "slot_attn_tc_kernel"
    return entry


class ClockSampler:
    """nvidia-smi sampling of SM clocks and throttle reasons."""
    FIELDS = ("index,timestamp,clocks.sm,clocks.max.sm,power.draw,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index: int):
        self.index = index
        self.proc = None
        out_dir = os.environ.get("ZARYA_CLOCKS_DIR") or tempfile.gettempdir()
        self.path = os.path.join(out_dir, f"zarya_clocks_rank{index}.csv")

    def start(self):
        try:
            os.makedirs(os.path.dirname(self.path), exist_ok=True)
            self.fh = open(self.path, "w")
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.index), f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "100"],
                stdout=self.fh, stderr=subprocess.DEVNULL)
        except Exception:
            self.proc = None
        return self

    def stop(self, t0: float, t1: float, keep: bool = False):
        """Ends the sampling and returns the clocks seen in [t0, t1]; with
        `keep`, the samples stay available to window()."""
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        self.fh.close()
        rows = []
        with open(self.path) as f:
            for line in f:
                parts = [p.strip() for p in line.split(",")]
                if len(parts) < 9:
                    continue
                try:
                    ts = time.mktime(time.strptime(parts[1].split(".")[0], "%Y/%m/%d %H:%M:%S"))
                    frac = float("0." + parts[1].split(".")[1]) if "." in parts[1] else 0.0
                    rows.append((ts + frac, float(parts[2]), float(parts[3]), parts[5:9]))
                except Exception:
                    continue
        self.rows = rows
        return self.window(t0, t1)

    def window(self, t0: float, t1: float):
        """Median SM clock, maximum clock and throttle reasons of the samples
        taken in [t0, t1] (the nearest sample when none falls inside)."""
        rows = getattr(self, "rows", None)
        if self.proc is None or rows is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        inside = [r for r in rows if t0 - 0.05 <= r[0] <= t1 + 0.05]
        used = inside
        note = None
        if not inside and rows:
            mid = 0.5 * (t0 + t1)
            used = [min(rows, key=lambda r: abs(r[0] - mid))]
            note = "timed region shorter than the sampling period: nearest sample"
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for r in used for i, v in enumerate(r[3]) if v == "Active"})
        out = {"sm_mhz": float(np.median([r[1] for r in used])) if used else None,
               "sm_max_mhz": max(r[2] for r in used) if used else None,
               "reasons": reasons, "samples": len(inside),
               "window_s": round(t1 - t0, 3)}
        if note:
            out["note"] = note
        return out


def dist_setup():
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return world, rank, local


def max_over_ranks(x: float, device, world: int) -> float:
    """The maximum of a per-rank time over all ranks: the slowest replica
    sets the job's time (a no-op on one rank)."""
    if world <= 1:
        return x
    import torch
    import torch.distributed as dist

    t = torch.tensor([x], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def replica_throughput(steps: int, world: int, total_ms: float) -> float:
    """Whole-job steps/s of `world` replicas that each ran `steps` steps, the
    slowest taking total_ms (weak scaling: every rank has its own batch)."""
    return steps * world / (total_ms * 1e-3)


def per_sequence_roofline(w, hbm_peak, tf_peak):
    """Ideal time of the attention launch under a roofline taken sequence by
    sequence: every sequence b needs at least max(bytes_b / HBM, flops_b /
    bf16) (its K/V, Q and O bytes; 4 D flops per visible pair), and the batch
    needs their sum. For a batch whose sequences all have the same shape this
    is the usual single-intensity roofline. Returns (ideal_s, hbm_part_s,
    tensor_part_s, batch_wide_s), the last being max(sum bytes / HBM,
    sum flops / bf16), a lower bound on the same time."""
    eb = 2 if w.dtype == "bf16" else 4
    P = w.cache_lens.astype(np.int64)
    R = w.R
    kv = w.Hkv * (P + R) * w.D * eb * 2
    qo = 2 * R * w.Hq * w.D * eb
    pairs = np.where(w.mask_mode == 0, w.Hq * R * (P + R), w.Hq * (R * P + R * (R + 1) // 2))
    byts = (kv + qo).astype(np.float64)
    flops = (4 * w.D * pairs).astype(np.float64)
    t_hbm = byts / (hbm_peak * 1e9)
    t_tc = flops / (tf_peak * 1e12)
    ideal = float(np.maximum(t_hbm, t_tc).sum())
    hbm_part = float(np.where(t_hbm >= t_tc, t_hbm, 0.0).sum())
    batch_wide = max(float(byts.sum()) / (hbm_peak * 1e9), float(flops.sum()) / (tf_peak * 1e12))
    return ideal, hbm_part, ideal - hbm_part, batch_wide


def roofline_per_sequence(w, counts, attn_ms, hbm_peak, tf_peak, peak_src, traffic,
                          kernel=None, tf_kind="burst", tf_burst=None):
    """The attention launch against the per-sequence roofline of its batch.

    `bound` names the resource that bounds most of the ideal time. When every
    sequence is bound by the same resource, `peak` is that resource's measured
    peak and `achieved` the algorithmic bytes (HBM) or flops (tensor) per
    second. When the batch mixes HBM-bound and tensor-bound sequences, the
    bound is the dominant one and `peak` is the rate the roofline allows for
    this batch (its algorithmic amount / the ideal time), so that
    frac = achieved / peak = ideal time / measured time."""
    ideal, hbm_part, tc_part, batch_wide = per_sequence_roofline(w, hbm_peak, tf_peak)
    t = attn_ms * 1e-3
    frac = ideal / t
    if tc_part >= hbm_part:
        bound, unit, amount, peak_meas = "tensor", "TFLOP/s", counts["flops"] / 1e12, tf_peak
        src = f"{peak_src} cuBLAS bf16 GEMM ({tf_kind})"
    else:
        bound, unit, amount, peak_meas = "hbm", "GB/s", counts["attn_bytes"] / 1e9, hbm_peak
        src = f"{peak_src} HBM copy bandwidth"
    achieved = amount / t
    mixed = hbm_part > 0 and tc_part > 0
    peak = amount / ideal if mixed else peak_meas
    entry = {"bound": bound, "achieved": round(achieved, 1), "peak": round(peak, 1), "unit": unit,
             "frac": round(achieved / peak, 4), "traffic": traffic,
             "peak_source": (f"per-sequence roofline of this batch (sum over sequences of "
                             f"max(bytes_b / {hbm_peak:.0f} GB/s, flops_b / {tf_peak:.0f} TFLOP/s), "
                             f"{peak_src} peaks, bf16 {tf_kind}): the attainable rate"
                             if mixed else src),
             "ideal_us": round(ideal * 1e6, 2),
             "ideal_us_hbm_bound_sequences": round(hbm_part * 1e6, 2),
             "ideal_us_tensor_bound_sequences": round(tc_part * 1e6, 2),
             "frac_of_batch_wide_bound": round(batch_wide / t, 4),
             "intensity_flop_per_byte": round(counts["flops"] / counts["attn_bytes"], 1),
             "ridge_flop_per_byte": round(tf_peak * 1e12 / (hbm_peak * 1e9), 1),
             "kernel": kernel or ("slot_attn_tc_kernel" if w.dtype == "bf16"
                                  else "slot_attn_f32_kernel")}
    if mixed:
        entry["peak_measured"] = peak_meas
    if tf_burst is not None and tf_burst != tf_peak:
        # the same launch against the burst bf16 rate (the stricter ideal)
        entry["frac_of_burst_bf16"] = round(per_sequence_roofline(w, hbm_peak, tf_burst)[0] / t, 4)
    if w.dtype != "bf16":
        entry["note"] = ("fp32 correctness configuration on the CUDA cores: a few microseconds "
                         "of launch latency, far from any throughput roof")
    return entry


def timed_reps(enqueue, stream, min_reps, min_seconds, max_reps=20000):
    """Times `enqueue()` (which enqueues one K-step region on `stream`) over
    repeated regions: one calibration region, then n >= min_reps regions back
    to back with a CUDA event between consecutive ones, n chosen so that the
    whole run lasts at least min_seconds. Returns (per-region ms list,
    wall-clock start, wall-clock end)."""
    import torch

    c0, c1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    c0.record(stream)
    enqueue()
    c1.record(stream)
    torch.cuda.synchronize()
    one = max(c0.elapsed_time(c1), 1e-3)
    n = int(min(max_reps, max(min_reps, math.ceil(min_seconds * 1e3 / one))))
    evs = [torch.cuda.Event(enable_timing=True) for _ in range(n + 1)]
    torch.cuda.synchronize()
    t0 = time.time()
    evs[0].record(stream)
    for i in range(n):
        enqueue()
        evs[i + 1].record(stream)
    torch.cuda.synchronize()
    t1 = time.time()
    return [evs[i].elapsed_time(evs[i + 1]) for i in range(n)], t0, t1


def rep_stats(ms, K, dev, world):
    """Median and minimum of the per-region times (max over ranks), per step."""
    med = max_over_ranks(float(np.median(ms)), dev, world)
    mn = max_over_ranks(float(np.min(ms)), dev, world)
    return med / K, mn / K, len(ms)


# The configurations reported in `per_config`: (entry, workload, mask mode
# override). long_ctx runs in both of its modes; tiny_fp32 (both modes in its
# parity tests) is timed in slot-causal mode.
PER_CONFIG = [("tiny_fp32", "tiny_fp32", 1), ("decode_small", "decode_small", None),
              ("ragged_mid", "ragged_mid", None), ("long_ctx_bidir", "long_ctx", 0),
              ("long_ctx_causal", "long_ctx", 1), ("serving_mix", "serving_mix", None)]


def entry_workload(entry):
    for e, name, mode in PER_CONFIG:
        if e == entry:
            return name, mode
    raise KeyError(entry)


def measure_workload(entry, args, dev, stream, world, rank, K, W, min_reps, min_seconds,
                     cpu_budget, full, sampler_windows):
    """Measures one configuration: the slot-decode step (staged attention +
    length commit) over K steps, the attention launches alone, and the step
    end to end through the public API with host buffers; each as repeated
    K-step regions (median and minimum). With `full`, also the step with the
    copying commit. Returns a dict (see run_ours)."""
    import torch

    from paper_2609_19868_gb300 import _binding as zb
    from paper_2609_19868_gb300 import session
    from paper_2609_19868_gb300 import workloads as wl

    name, mode = entry_workload(entry)
    # weak scaling: every rank runs its own batch (distinct seed)
    seed = wl.SPECS[name]["seed"] + 1000 * rank
    w = wl.make(name, seed=seed)
    if mode is not None:
        w = w.with_mode(mode)
    counts = algorithmic_counts(w)
    l2 = torch.cuda.get_device_properties(dev).L2_cache_size
    cache_bytes = (w.k_cache.numel() + w.v_cache.numel()) * w.k_cache.element_size()
    n_rot = max(2, math.ceil(3 * l2 / max(cache_bytes, 1)))
    rots = []
    with torch.cuda.stream(stream):
        base = session.upload(w, dev)
        rots.append(base)
        for _ in range(n_rot - 1):
            kc, vc = base.k_cache.clone(), base.v_cache.clone()
            rots.append(session.upload(w, dev, caches=(kc, vc)))
    kernel = zb.slot_attn_kernel(base.desc)   # the kernel the plan launches
    # kernels per step: the attention call's (a dispatch-order kernel first
    # when the plan sorts its tiles; the fp32 path stages with an append), and
    # the length commit
    launches_per_step = zb.slot_attn_launches(base.desc) + (w.dtype != "bf16") + 1
    # The commit writes the advanced lengths into a second array (the
    # ping-pong a decoding loop would use), so every step starts from the same
    # prefix lengths: a stationary workload with no copy between steps.
    lens_next = {id(db): torch.empty_like(db.cache_lens) for db in rots}
    torch.cuda.synchronize()

    def step(db):
        # stage the block's own K/V and attend in one launch; the accepted
        # rows are then already in place, so the commit advances the lengths
        db.stage_and_attend(stream)
        db.commit_staged(stream, new_lens=lens_next[id(db)])

    def attend(db):
        db.attend(stream)

    def step_copy(db):
        # the same step with the commit copying the accepted rows again
        db.stage_and_attend(stream)
        db.commit(stream, new_lens=lens_next[id(db)])

    with torch.cuda.stream(stream):
        for i in range(max(W, n_rot)):
            step(rots[i % n_rot])
    torch.cuda.synchronize()
    assert zb.check_device_error(stream) == 0

    # CUDA graphs hold n_rot consecutive steps, one per cache rotation (as a
    # serving loop captures a whole forward pass): the kernels of successive
    # steps chain through programmatic dependent launch instead of paying a
    # graph launch each. A tail graph with the first K % n_rot steps makes each
    # timed region exactly K steps.
    def capture(fn, count):
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=stream):
            for r in range(count):
                fn(rots[r])
        return g

    def capture_fn(fn):
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=stream):
            fn()
        return g

    full_n, tail = divmod(K, n_rot)

    def region(graph, tail_graph):
        def enqueue():
            for _ in range(full_n):
                graph.replay()
            if tail_graph is not None:
                tail_graph.replay()
        return enqueue

    graphs = {"step": (capture(step, n_rot), capture(step, tail) if tail else None),
              "attn": (capture(attend, n_rot), capture(attend, tail) if tail else None)}
    if full:
        graphs["copy"] = (capture(step_copy, n_rot), capture(step_copy, tail) if tail else None)
    with torch.cuda.stream(stream):
        for g, gt in graphs.values():
            for _ in range(max(1, -(-W // n_rot))):
                g.replay()
    torch.cuda.synchronize()
    assert zb.check_device_error(stream) == 0

    res = {}
    with torch.cuda.stream(stream):
        for key, (g, gt) in graphs.items():
            if world > 1:
                import torch.distributed as dist

                dist.barrier()
            ms, t0, t1 = timed_reps(region(g, gt), stream, min_reps, min_seconds)
            res[key] = rep_stats(ms, K, dev, world)
            sampler_windows.append((entry, key, t0, t1))
    torch.cuda.synchronize()
    assert zb.check_device_error(stream) == 0

    # End to end through the public API, every step: the step's inputs (q,
    # k_new, v_new, accept_len, packed in one pinned host buffer) copied to the
    # device, the step, and its output copied back to pinned host memory.
    # The transfers are zarya_copy kernels (a few CTAs moving the bytes through
    # the pinned buffers' device mapping) or copy-engine memcpys, on their own
    # streams, pipelined with the computation as a serving loop overlaps
    # transfers with compute: step i's copy-in runs during step i - 1, its
    # copy-out during step i + 1. Step i uses rotation i % n_rot; events keep
    # each rotation's buffers in order (its copy-in waits for the step before
    # on that rotation to have read them, its step for that step's copy-out to
    # have read the output). The K steps of a timed region, copies included,
    # are one CUDA graph.
    def align(x):
        return (x + 255) // 256 * 256

    parts = [("q", w.q), ("k_new", w.k_new), ("v_new", w.v_new),
             ("accept_len", torch.as_tensor(w.accept_len))]
    offs, total = [], 0
    for _, t in parts:
        offs.append(total)
        total = align(total + t.numel() * t.element_size())
    host_in = torch.zeros(total, dtype=torch.uint8).pin_memory()
    for (_, t), o in zip(parts, offs):
        nbytes = t.numel() * t.element_size()
        host_in[o:o + nbytes].copy_(t.contiguous().view(-1).view(torch.uint8))
    out_h = torch.empty_like(w.q).pin_memory()
    h2d = sum(t.numel() * t.element_size() for _, t in parts)
    d2h = out_h.numel() * out_h.element_size()
    dev_in = []
    for db in rots:
        buf = torch.empty(total, dtype=torch.uint8, device=dev)
        dev_in.append(buf)
        for (nm, t), o in zip(parts, offs):
            nbytes = t.numel() * t.element_size()
            setattr(db, nm, buf[o:o + nbytes].view(t.dtype).view(t.shape))
    s_in, s_out = torch.cuda.Stream(dev), torch.cuda.Stream(dev)
    ev_in = [torch.cuda.Event() for _ in rots]
    ev_done = [torch.cuda.Event() for _ in rots]
    ev_out = [torch.cuda.Event() for _ in rots]

    def e2e_steps(count, engine):
        # stream forks off `stream` and joins back (valid inside a capture);
        # engine: the transfers are copy-engine memcpys instead of zarya_copy
        s_in.wait_stream(stream)
        s_out.wait_stream(stream)
        for i in range(count):
            r = i % n_rot
            db = rots[r]
            with torch.cuda.stream(s_in):
                if i >= n_rot:
                    s_in.wait_event(ev_done[r])    # step i - n_rot has read dev_in[r]
                if engine:
                    dev_in[r].copy_(host_in, non_blocking=True)
                else:
                    zb.copy(dev_in[r], host_in, s_in)
                ev_in[r].record(s_in)
            with torch.cuda.stream(stream):
                stream.wait_event(ev_in[r])
                if i >= n_rot:
                    stream.wait_event(ev_out[r])   # its output has been copied out
                step(db)
                ev_done[r].record(stream)
            with torch.cuda.stream(s_out):
                s_out.wait_event(ev_done[r])
                if engine:
                    out_h.copy_(db.out, non_blocking=True)
                else:
                    zb.copy(out_h, db.out, s_out)
                ev_out[r].record(s_out)
        stream.wait_stream(s_in)
        stream.wait_stream(s_out)

    # Both transfer forms are timed and the faster one is reported: copy
    # kernels avoid the hand-over cost of memcpy nodes between kernels (short
    # steps), copy engines run beside an attention grid that fills every SM
    # (long steps).
    e2e = {}
    for engine in (False, True):
        with torch.cuda.stream(stream):
            e2e_steps(n_rot, engine)   # eager warm-up through the public API
        torch.cuda.synchronize()
        e2e_graph = capture_fn(lambda: e2e_steps(K, engine))
        with torch.cuda.stream(stream):
            for _ in range(max(1, -(-W // K))):
                e2e_graph.replay()
        torch.cuda.synchronize()
        if world > 1:
            import torch.distributed as dist

            dist.barrier()
        with torch.cuda.stream(stream):
            ms, t0, t1 = timed_reps(e2e_graph.replay, stream, min_reps, min_seconds)
        sampler_windows.append((entry, "e2e", t0, t1))
        e2e["copy engines" if engine else "zarya_copy kernels"] = rep_stats(ms, K, dev, world)
        del e2e_graph
        assert zb.check_device_error(stream) == 0
        # every step computes the same output (a stationary workload): what
        # the last copy-out left in pinned memory is the device's result
        assert torch.equal(out_h.view(torch.uint8), rots[(K - 1) % n_rot].out.cpu().view(torch.uint8)), \
            "end-to-end output differs from the device result"
    e2e_how = min(e2e, key=lambda k: e2e[k][0])
    res["e2e"] = e2e[e2e_how]

    hbm_peak, tf_burst, peak_src = read_peaks()
    tf_peak, _ = read_sustained_bf16()
    attn_ms = res["attn"][0]
    step_ms = res["step"][0]
    out = {
        "workload": WORKLOAD_LABELS[entry],
        "w": w,
        "counts": counts,
        "n_rot": n_rot,
        "cache_bytes": cache_bytes,
        "l2": l2,
        "step_ms": res["step"],
        "attn_ms": res["attn"],
        "copy_ms": res.get("copy"),
        "e2e_ms": res["e2e"],
        "e2e_how": e2e_how,
        "e2e_all": {k: round(replica_throughput(K, world, v[0] * K), 2) for k, v in e2e.items()},
        "h2d": int(h2d),
        "d2h": int(d2h),
        "roofline": roofline_per_sequence(w, counts, attn_ms, hbm_peak, tf_peak, peak_src,
                                          recorded_traffic(entry, kernel), kernel,
                                          tf_kind="sustained: the launches are timed back to "
                                                  "back for a second or more",
                                          tf_burst=tf_burst),
        "hbm_gbs": counts["attn_bytes"] / (attn_ms * 1e-3) / 1e9,
        "tflops": counts["flops"] / (attn_ms * 1e-3) / 1e12,
        "steps_per_s": replica_throughput(K, world, step_ms * K),
        "launches_per_step": launches_per_step,
    }
    del rots, graphs, dev_in, base
    torch.cuda.synchronize()
    torch.cuda.empty_cache()
    if rank == 0 and world == 1 and cpu_budget > 0:
        out["cpu_baseline"] = cpu_baseline(w, budget_s=cpu_budget)
    return out


def config_entry(m, K, world):
    """The per_config record of one measured configuration."""
    (s_med, s_min, s_n), (a_med, a_min, a_n) = m["step_ms"], m["attn_ms"]
    e_med, e_min, e_n = m["e2e_ms"]
    c = m["counts"]
    rec = {
        "workload": m["workload"],
        "ms_per_step": round(s_med, 5),
        "ms_per_step_min": round(s_min, 5),
        "steps_per_s": round(replica_throughput(K, world, s_med * K), 2),
        "attn_ms_per_launch": round(a_med, 5),
        "attn_ms_per_launch_min": round(a_min, 5),
        "hbm_gbs": round(m["hbm_gbs"], 1),
        "tflops": round(m["tflops"], 2),
        "algorithmic_bytes": c["attn_bytes"],
        "algorithmic_flops": c["flops"],
        "roofline": m["roofline"],
        "e2e": {"value": round(replica_throughput(K, world, e_med * K), 2), "unit": "steps/s",
                "h2d_bytes_per_step": m["h2d"], "d2h_bytes_per_step": m["d2h"],
                "transfers": m["e2e_how"], "steps_per_s_by_transfer": m["e2e_all"]},
        "timing": f"{s_n} regions of {K} steps (median; min also given)",
    }
    if "cpu_baseline" in m:
        rec["cpu_baseline"] = m["cpu_baseline"]
    return rec


def run_ours(args):
    import torch
    import torch.distributed as dist

    world, rank, local = dist_setup()
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    if world > 1:
        dist.init_process_group("nccl", device_id=dev)
    from paper_2609_19868_gb300 import build as zbuild

    if rank == 0:
        zbuild.build()
    if world > 1:
        dist.barrier()
    from paper_2609_19868_gb300 import _binding as zb

    zb.load()
    zb.check_device_error()
    K, W = args.steps, args.warmup
    stream = torch.cuda.Stream(dev)
    sampler = ClockSampler(local).start() if args.clocks else None
    if sampler:
        time.sleep(0.3)
    windows = []
    head = measure_workload(args.workload, args, dev, stream, world, rank, K, W, args.reps,
                            args.min_seconds, 0.0 if args.no_cpu_baseline else args.cpu_budget,
                            True, windows)
    per_config = {}
    if args.per_config:
        for entry, _, _ in PER_CONFIG:
            if entry == args.workload:
                m = head
            else:
                m = measure_workload(entry, args, dev, stream, world, rank, K, W,
                                     args.reps, args.config_seconds,
                                     0.0 if args.no_cpu_baseline else args.cpu_budget / 4,
                                     False, windows)
            per_config[entry] = config_entry(m, K, world)
            if m is not head:
                del m
    clocks_all = None
    if sampler:
        step_win = [(t0, t1) for e, key, t0, t1 in windows if e == args.workload and key == "step"]
        clocks = sampler.stop(*step_win[0], keep=True)
        for entry in per_config:
            wins = [(t0, t1) for e, key, t0, t1 in windows if e == entry]
            per_config[entry]["clocks"] = sampler.window(wins[0][0], wins[-1][1])
        clocks_all = sampler.window(windows[0][2], windows[-1][3])
    else:
        clocks = None

    w = head["w"]
    (s_med, s_min, s_n), (a_med, a_min, a_n) = head["step_ms"], head["attn_ms"]
    e_med = head["e2e_ms"][0]
    c_med = head["copy_ms"][0]
    value = replica_throughput(K, world, s_med * K)
    line = {
        "metric": "slot-decode steps/s (one layer: stage + slot attention + commit)",
        "value": round(value, 2),
        "unit": "steps/s",
        "n_gpus": world,
        "steps": K,
        "warmup": W,
        "ms_per_step": round(s_med, 5),
        "higher_is_better": True,
        "scaling": "weak",
        "vs_baseline": None,
        "dtype": "bf16" if w.dtype == "bf16" else "f32",
        "data": "synthetic (seeded N(0,1), random-init; no weights or datasets)",
        "config": {
            "workload": head["workload"],
            "global_batch": w.B * world,
            "block_rows_per_seq_max": int(w.max_rows),
            "kv_len_max": int((w.cache_lens + w.R).max()),
            "l2": f"{head['n_rot']} rotating KV caches of {head['cache_bytes'] / 1e6:.1f} MB "
                  f"(> L2 {head['l2'] / 1e6:.0f} MB between reuses)",
            "parallelism": f"replicas x{world}" if world > 1 else "single GPU",
            "launch": f"CUDA graphs of {head['n_rot']} steps (programmatic dependent launch "
                      "between kernels)",
        },
        "timing": {"regions": s_n, "steps_per_region": K, "statistic": "median region",
                   "ms_per_step_min": round(s_min, 5),
                   "method": "CUDA events between back-to-back K-step regions on the "
                             "launching stream; max over ranks"},
        "attn": {
            "ms_per_launch": round(a_med, 5),
            "ms_per_launch_min": round(a_min, 5),
            "timing": f"{a_n} regions of {K} attention launches back to back ({head['n_rot']} per "
                      "CUDA graph, one per cache rotation), CUDA events on the launching stream; "
                      "median region",
            "hbm_gbs": round(head["hbm_gbs"], 1),
            "tflops": round(head["tflops"], 2),
            "algorithmic_bytes": head["counts"]["attn_bytes"],
            "algorithmic_flops": head["counts"]["flops"],
        },
        "roofline": head["roofline"],
        "e2e": {
            "value": round(replica_throughput(K, world, e_med * K), 2),
            "unit": "steps/s",
            "h2d_bytes_per_step": head["h2d"],
            "d2h_bytes_per_step": head["d2h"],
            "transfers": f"{head['e2e_how']} on side streams pipelined with the steps (step "
                         "i's copy-in during step i - 1, its copy-out during step i + 1; the K "
                         "steps and their copies one CUDA graph); the faster of zarya_copy "
                         "kernels and copy-engine memcpys",
            "steps_per_s_by_transfer": head["e2e_all"],
        },
        "step_forms": {
            "commit_staged": {"ms_per_step": round(s_med, 5),
                              "note": "zarya_slot_attn_staged + zarya_kv_commit_staged (the "
                                      "accepted rows are already in place: lengths advance)"},
            "commit_copy": {"ms_per_step": round(c_med, 5),
                            "steps_per_s": round(replica_throughput(K, world, c_med * K), 2),
                            "note": "zarya_slot_attn_staged + zarya_kv_append_commit_to (the "
                                    "accepted rows copied again)"},
        },
        "model_projection": {
            "note": "context only: one step per layer, attention path alone",
            "layers_28_steps_per_s": round(value / 28, 2),
            "layers_36_steps_per_s": round(value / 36, 2),
        },
        # the attention call's kernels + the length commit, every timed region
        "gpu_launches": head["launches_per_step"] * K * s_n,
        "gpu_launches_note": f"{head['launches_per_step']} kernels per step x {K} steps x "
                             f"{s_n} timed regions",
        "clocks": clocks,
    }
    if per_config:
        line["per_config"] = per_config
        if clocks_all is not None:
            line["clocks_whole_run"] = clocks_all
    if "cpu_baseline" in head:
        line["cpu_baseline"] = head["cpu_baseline"]
    if rank == 0:
        print(json.dumps(line), flush=True)
    if world > 1:
        dist.destroy_process_group()


SELECT_LABELS = {
    "select_decode_small": "select_decode_small: B8, 4 slots x 8 tokens, V 151936 (Qwen3 vocabulary), "
                           "bf16 logits, thresholds 0.9 / 0.4",
    "select_serving_mix": "select_serving_mix: B64, 8 slots, slot_len in {4,8,16,32}, V 151936, "
                          "bf16 logits, thresholds 0.9 / 0.4",
    "select_long_ctx": "select_long_ctx: B4, 16 slots x 32 tokens, V 151936, bf16 logits, "
                       "thresholds 0.9 / 0.4",
}


def run_select(args):
    """Slot selection and token acceptance (Sec. 5.2 steps 3-6): one step =
    zarya_draft_select over the draft block's logits, then zarya_verify_accept
    over the verification block the draft laid out (its tokens and layout
    taken from the draft's outputs on the device)."""
    import torch
    import torch.distributed as dist

    world, rank, local = dist_setup()
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    if world > 1:
        dist.init_process_group("nccl", device_id=dev)
    from paper_2609_19868_gb300 import build as zbuild

    if rank == 0:
        zbuild.build()
    if world > 1:
        dist.barrier()
    from paper_2609_19868_gb300 import _binding as zb
    from paper_2609_19868_gb300 import session
    from paper_2609_19868_gb300 import workloads as wl

    zb.load()
    zb.check_device_error()
    name = args.workload if args.workload in SELECT_LABELS else "select_decode_small"
    seed = wl.SAMPLE_SPECS[name]["seed"] + 1000 * rank
    w = wl.make_sampling(name, device=dev, seed=seed)
    T = args.temperature
    l2 = torch.cuda.get_device_properties(dev).L2_cache_size
    eb = 2 if w.dtype == "bf16" else 4
    logit_bytes = (w.draft_logits.numel() + w.verify_logits.numel()) * eb
    n_rot = max(1, math.ceil(3 * l2 / max(logit_bytes, 1))) if logit_bytes < 3 * l2 else 1
    stream = torch.cuda.Stream(dev)
    with torch.cuda.stream(stream):
        rots = [session.upload_sampling(w, dev, temperature=T, seed=seed, offset=r, chain=True)
                for r in range(n_rot)]
    torch.cuda.synchronize()

    def step(sb):
        sb.draft(stream)
        sb.verify(stream)

    K, W = args.steps, args.warmup
    with torch.cuda.stream(stream):
        for i in range(max(W, n_rot)):
            step(rots[i % n_rot])
    torch.cuda.synchronize()
    assert zb.check_device_error(stream) == 0
    vrows = int(rots[0].verify_row_offsets[-1].item())
    draft_bytes = w.rows * w.V * eb
    verify_bytes = vrows * w.V * eb

    def capture(fn, count):
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=stream):
            for r in range(count):
                fn(rots[r])
        return g

    full, tail = divmod(K, n_rot)
    step_graph = capture(step, n_rot)
    step_tail = capture(step, tail) if tail else None
    draft_graph = capture(lambda sb: sb.draft(stream), n_rot)
    draft_tail = capture(lambda sb: sb.draft(stream), tail) if tail else None

    def run(graph, tail_graph):
        for _ in range(full):
            graph.replay()
        if tail_graph is not None:
            tail_graph.replay()

    for _ in range(max(1, -(-W // n_rot))):
        step_graph.replay()
    torch.cuda.synchronize()
    sampler = ClockSampler(local).start() if args.clocks else None
    if sampler:
        time.sleep(0.3)
    if world > 1:
        dist.barrier()
    start, end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    torch.cuda.synchronize()
    t0 = time.time()
    with torch.cuda.stream(stream):
        start.record(stream)
        run(step_graph, step_tail)
        end.record(stream)
    torch.cuda.synchronize()
    t1 = time.time()
    total_ms = max_over_ranks(start.elapsed_time(end), dev, world)
    d0, d1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with torch.cuda.stream(stream):
        d0.record(stream)
        run(draft_graph, draft_tail)
        d1.record(stream)
    torch.cuda.synchronize()
    clocks = sampler.stop(t0, time.time()) if sampler else None
    assert zb.check_device_error(stream) == 0
    draft_ms = max_over_ranks(d0.elapsed_time(d1) / K, dev, world)

    # End to end through the public API: every step copies its draft logits
    # from pinned host memory, runs both calls, and reads accept_len and the
    # drafted tokens back (the verification logits stay resident: they are the
    # output of a forward pass that runs between the two calls on the device).
    host = w.draft_logits.cpu().pin_memory()
    out_tok = torch.empty(w.rows, dtype=torch.int32).pin_memory()
    out_acc = torch.empty(w.B, dtype=torch.int32).pin_memory()
    s_in, s_out = torch.cuda.Stream(dev), torch.cuda.Stream(dev)
    ev_in = [torch.cuda.Event() for _ in rots]
    ev_done = [torch.cuda.Event() for _ in rots]

    def e2e_steps(count):
        s_in.wait_stream(stream)
        s_out.wait_stream(stream)
        for r in range(count):
            sb = rots[r]
            with torch.cuda.stream(s_in):
                sb.draft_logits.copy_(host, non_blocking=True)
                ev_in[r].record(s_in)
            with torch.cuda.stream(stream):
                stream.wait_event(ev_in[r])
                step(sb)
                ev_done[r].record(stream)
            with torch.cuda.stream(s_out):
                s_out.wait_event(ev_done[r])
                out_tok.copy_(sb.draft_tokens, non_blocking=True)
                out_acc.copy_(sb.accept_len, non_blocking=True)
        stream.wait_stream(s_in)
        stream.wait_stream(s_out)

    with torch.cuda.stream(stream):
        e2e_steps(n_rot)
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=stream):
        e2e_steps(n_rot)
    gt = None
    if tail:
        gt = torch.cuda.CUDAGraph()
        with torch.cuda.graph(gt, stream=stream):
            e2e_steps(tail)
    g.replay()
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with torch.cuda.stream(stream):
        e0.record(stream)
        run(g, gt)
        e1.record(stream)
    torch.cuda.synchronize()
    e2e_ms = max_over_ranks(e0.elapsed_time(e1), dev, world)
    assert zb.check_device_error(stream) == 0

    hbm_peak, _, peak_src = read_peaks()
    draft_gbs = draft_bytes / (draft_ms * 1e-3) / 1e9
    line = {
        "metric": "slot select + token accept steps/s (draft select over the block's logits, "
                  "then acceptance over the verification block)",
        "value": round(replica_throughput(K, world, total_ms), 2),
        "unit": "steps/s",
        "n_gpus": world,
        "steps": K,
        "warmup": W,
        "ms_per_step": round(total_ms / K, 5),
        "higher_is_better": True,
        "scaling": "weak",
        "vs_baseline": None,
        "dtype": "f32 (bf16 logits)",
        "data": "synthetic (seeded N(0,2^2) logits with peaked tokens; no weights or datasets)",
        "config": {
            "workload": SELECT_LABELS[name],
            "temperature": T,
            "global_batch": w.B * world,
            "draft_rows": w.rows,
            "verify_rows": vrows,
            "l2": (f"{n_rot} rotating logits copies of {logit_bytes / 1e6:.1f} MB (> L2 between "
                   f"reuses)" if n_rot > 1 else
                   f"logits {logit_bytes / 1e6:.0f} MB per step (> L2 {l2 / 1e6:.0f} MB)"),
            "launch": f"CUDA graphs of {n_rot} steps (programmatic dependent launch)",
        },
        "roofline": {
            "bound": "hbm",
            "achieved": round(draft_gbs, 1),
            "peak": hbm_peak,
            "unit": "GB/s",
            "frac": round(draft_gbs / hbm_peak, 4),
            "traffic": None,
            "kernel": "zarya_draft_select (row pass + selection), per call",
            "algorithmic_bytes": draft_bytes,
            "peak_source": f"{peak_src} HBM copy bandwidth",
        } if T == 0 else alu_roofline(w.rows * w.V, draft_ms, dev,
                                      "zarya_draft_select (row pass + selection), per call"),
        "e2e": {
            "value": round(replica_throughput(K, world, e2e_ms), 2),
            "unit": "steps/s",
            "h2d_bytes_per_step": int(draft_bytes),
            "d2h_bytes_per_step": int(4 * (w.rows + w.B)),
        },
        "gpu_launches": 4 * K,
        "clocks": clocks,
    }
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        line["cpu_baseline"] = select_cpu_baseline(w, T, rots[0], budget_s=args.cpu_budget)
    if rank == 0:
        print(json.dumps(line), flush=True)
    if world > 1:
        dist.destroy_process_group()


REORDER_LABELS = {
    "reorder_serving": "reorder_serving: B64 token rows of up to 2048 (context length, Table 1), "
                       "lengths ~U[512,2048], per-sequence mask fraction ~U(0.1,0.9)",
}


def run_reorder(args):
    """Reordering + restoration (Sec. 5.1 steps 2/4, Sec. 5.2 steps 1/8): one
    step = zarya_reorder of a batch of token rows, then zarya_restore of the
    reordered rows. Stable form (Mode B) in `value`; the keyed form (Mode A's
    token shuffling) alongside."""
    import torch

    world, rank, local = dist_setup()
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    from paper_2609_19868_gb300 import build as zbuild

    zbuild.build()
    from paper_2609_19868_gb300 import _binding as zb
    from paper_2609_19868_gb300 import workloads as wl

    zb.load()
    zb.check_device_error()
    name = "reorder_serving"
    w = wl.make_reorder(name, seed=wl.REORDER_SPECS[name]["seed"] + 1000 * rank)
    stream = torch.cuda.Stream(dev)
    B, L = w.B, w.max_len
    t = torch.as_tensor(w.tokens).to(dev)
    m = torch.as_tensor(w.is_masked).to(dev)
    k = torch.as_tensor(w.order_key.view(np.int32)).to(dev)
    ln = torch.as_tensor(w.lens).to(dev)
    perm, out, back = (torch.empty_like(t) for _ in range(3))
    nv = torch.empty(B, dtype=torch.int32, device=dev)

    def step(keyed):
        zb.reorder(t, m, ln, perm, out, nv, order_key=k if keyed else None, stream=stream)
        zb.restore(out, perm, ln, back, stream=stream)

    K, W = args.steps, args.warmup
    res = {}
    for keyed in (False, True):
        with torch.cuda.stream(stream):
            for _ in range(W):
                step(keyed)
        torch.cuda.synchronize()
        assert zb.check_device_error(stream) == 0
        g = torch.cuda.CUDAGraph()
        per = 20
        with torch.cuda.graph(g, stream=stream):
            for _ in range(per):
                step(keyed)
        g.replay()
        torch.cuda.synchronize()
        reps = max(1, K // per)
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        with torch.cuda.stream(stream):
            e0.record(stream)
            for _ in range(reps):
                g.replay()
            e1.record(stream)
        torch.cuda.synchronize()
        res[keyed] = e0.elapsed_time(e1) / (reps * per)
    assert np.array_equal(back.cpu().numpy(), w.tokens)
    ms = res[False]
    # algorithmic bytes: reorder reads tokens + mask, writes perm + tokens;
    # restore reads tokens + perm, writes tokens (4-byte ints, 1-byte mask)
    n_pos = int(w.lens.sum())
    nbytes = n_pos * (4 + 1 + 4 + 4 + 4 + 4 + 4)
    hbm_peak, _, peak_src = read_peaks()
    gbs = nbytes / (ms * 1e-3) / 1e9
    # e2e: tokens and mask copied in from pinned host memory, restored tokens
    # copied back, every step; the copies are zarya_copy kernels on the step's
    # stream, and 20 steps (copies included) form one CUDA graph.
    ht, hm, hb = t.cpu().pin_memory(), m.cpu().pin_memory(), torch.empty_like(t, device="cpu").pin_memory()

    def e2e_step():
        zb.copy(t, ht, stream)
        zb.copy(m, hm, stream)
        step(False)
        zb.copy(hb, back, stream)

    with torch.cuda.stream(stream):
        for _ in range(W):
            e2e_step()
    torch.cuda.synchronize()
    ge = torch.cuda.CUDAGraph()
    with torch.cuda.graph(ge, stream=stream):
        for _ in range(per):
            e2e_step()
    ge.replay()
    hb.zero_()
    torch.cuda.synchronize()
    reps_e2e = max(1, K // per)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with torch.cuda.stream(stream):
        e0.record(stream)
        for _ in range(reps_e2e):
            ge.replay()
        e1.record(stream)
    torch.cuda.synchronize()
    assert zb.check_device_error(stream) == 0
    assert np.array_equal(hb.numpy(), w.tokens)
    e2e_ms = e0.elapsed_time(e1) / (reps_e2e * per)
    line = {
        "metric": "reorder + restore steps/s (a batch of token rows reordered visible-first, "
                  "then restored)",
        "value": round(1e3 / ms, 2), "unit": "steps/s", "n_gpus": 1, "steps": K, "warmup": W,
        "ms_per_step": round(ms, 5), "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "int32", "data": "synthetic (seeded token ids and masks)",
        "config": {"workload": REORDER_LABELS[name], "global_batch": B,
                   "keyed_ms_per_step": round(res[True], 5),
                   "launch": "CUDA graphs of 20 steps (programmatic dependent launch)",
                   "l2": "inputs resident (1.6 MB); latency-bound"},
        "roofline": {"bound": "hbm", "achieved": round(gbs, 1), "peak": hbm_peak, "unit": "GB/s",
                     "frac": round(gbs / hbm_peak, 4), "traffic": None,
                     "kernel": "reorder_kernel + restore_kernel (launch-latency bound)",
                     "algorithmic_bytes": nbytes, "peak_source": f"{peak_src} HBM copy bandwidth"},
        "e2e": {"value": round(1e3 / e2e_ms, 2), "unit": "steps/s",
                "h2d_bytes_per_step": int(t.numel() * 4 + m.numel()),
                "d2h_bytes_per_step": int(back.numel() * 4),
                "transfers": "zarya_copy kernels on the step's stream (CUDA graphs of 20 steps)"},
        "gpu_launches": 2 * K,
    }
    if not args.no_cpu_baseline:
        from oracle import reorder as ro

        nb = 8
        t0 = time.perf_counter()
        p_, o_, _ = ro.reorder(w.tokens[:nb], w.is_masked[:nb], w.lens[:nb])
        ro.restore(o_, p_, w.lens[:nb])
        dt = (time.perf_counter() - t0) * B / nb
        line["cpu_baseline"] = {"value": round(1.0 / dt, 4), "unit": "steps/s", "cores": 1,
                                "kind": "oracle",
                                "sample": f"{nb} of {B} sequences (python oracle), scaled"}
    print(json.dumps(line), flush=True)


def run_mode_a(args):
    """Mode A (Sec. 5.1): the mask-budget plan of a batch (once per
    generation), then per step the draw of every revealed position's token
    (zarya_sample_rows over those rows' logits). Batch of 64 sequences with 256
    masked tokens each, T = 64 diffusion steps, alpha_0 = 0.25 (the paper's
    default): a plan of about 64 + 192 steps revealing one token per sequence
    at most steps, so a step samples 64 rows of the Qwen3 vocabulary."""
    import torch

    world, rank, local = dist_setup()
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    from paper_2609_19868_gb300 import build as zbuild

    zbuild.build()
    from paper_2609_19868_gb300 import _binding as zb
    from paper_2609_19868_gb300 import session
    from paper_2609_19868_gb300 import workloads as wl

    zb.load()
    zb.check_device_error()
    B, n_mask, T_steps, a0 = 64, 256, 64, 0.25
    temp = args.temperature
    stream = torch.cuda.Stream(dev)
    nm = torch.full((B,), n_mask, dtype=torch.int32, device=dev)
    counts = torch.zeros((B, T_steps + n_mask), dtype=torch.int32, device=dev)
    steps = torch.zeros(B, dtype=torch.int32, device=dev)
    # logits of one revealed row per sequence (64 rows), rotated copies > L2
    w = wl.make_sampling("select_decode_small", device=dev)
    rows = B
    eb = 2
    l2 = torch.cuda.get_device_properties(dev).L2_cache_size
    n_rot = max(2, math.ceil(3 * l2 / (rows * w.V * eb)))
    src = w.draft_logits[:rows]
    rots = []
    for r in range(n_rot):
        sw = wl.SamplingWorkload(name="mode_a", B=rows, V=w.V, dtype="bf16",
                                 n_slots=np.ones(rows, dtype=np.int32),
                                 slot_len=np.ones(rows, dtype=np.int32),
                                 row_offsets=np.arange(rows + 1, dtype=np.int32),
                                 draft_logits=src.roll(r, 0), n_verify=np.ones(rows, dtype=np.int32),
                                 verify_offsets=np.arange(rows + 1, dtype=np.int32),
                                 verify_tokens=np.zeros(rows, dtype=np.int32),
                                 verify_logits=src[:1])
        rots.append(session.upload_sampling(sw, dev, temperature=temp, seed=9, offset=r))
    K, W = args.steps, args.warmup

    def plan():
        zb.mode_a_budget(nm, T_steps, a0, 9, 0, counts, steps, stream=stream)

    def sample(sb):
        zb.sample_rows(sb.draft_logits, sb.draft_tokens, sb.draft_prob, sb.draft_desc,
                       stream=stream)

    def timed(fn_graph, reps):
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        with torch.cuda.stream(stream):
            e0.record(stream)
            for _ in range(reps):
                fn_graph.replay()
            e1.record(stream)
        torch.cuda.synchronize()
        return e0.elapsed_time(e1) / reps

    with torch.cuda.stream(stream):
        for i in range(max(W, n_rot)):
            plan()
            sample(rots[i % n_rot])
    torch.cuda.synchronize()
    assert zb.check_device_error(stream) == 0
    gp = torch.cuda.CUDAGraph()
    with torch.cuda.graph(gp, stream=stream):
        for _ in range(10):
            plan()
    gs = torch.cuda.CUDAGraph()
    with torch.cuda.graph(gs, stream=stream):
        for sb in rots:
            sample(sb)
    gp.replay()
    gs.replay()
    torch.cuda.synchronize()
    plan_ms = timed(gp, max(1, K // 10)) / 10
    step_ms = timed(gs, max(1, K // n_rot)) / n_rot
    assert zb.check_device_error(stream) == 0
    n_steps = steps.cpu().numpy()
    nbytes = rows * w.V * eb
    hbm_peak, _, peak_src = read_peaks()
    gbs = nbytes / (step_ms * 1e-3) / 1e9
    line = {
        "metric": "Mode A sampling steps/s (the revealed rows' tokens drawn from their logits)",
        "value": round(1e3 / step_ms, 2), "unit": "steps/s", "n_gpus": 1, "steps": K,
        "warmup": W, "ms_per_step": round(step_ms, 5), "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f32 (bf16 logits)",
        "data": "synthetic (seeded N(0,2^2) logits with peaked tokens)",
        "config": {"workload": f"mode_a: B{B}, {n_mask} masked tokens, T={T_steps}, alpha_0={a0}, "
                               f"{rows} revealed rows per step, V {w.V}",
                   "temperature": temp,
                   "plan_ms": round(plan_ms, 5),
                   "plan_steps_mean": float(n_steps.mean()),
                   "l2": f"{n_rot} rotating logits copies (> L2 between reuses)"},
        "roofline": {"bound": "hbm", "achieved": round(gbs, 1),
                     "peak": hbm_peak, "unit": "GB/s", "frac": round(gbs / hbm_peak, 4),
                     "traffic": None, "kernel": "row_pass_kernel (zarya_sample_rows)",
                     "algorithmic_bytes": nbytes, "peak_source": f"{peak_src} HBM copy bandwidth"}
        if temp == 0 else alu_roofline(rows * w.V, step_ms, dev,
                                       "row_pass_kernel (zarya_sample_rows)"),
        "e2e": None,
        "gpu_launches": K,
    }
    print(json.dumps(line), flush=True)


def run_top_p(args):
    """top_p truncation of the draft block's logits (Sec. 5.1 step 3, Table 2):
    zarya_top_p in place over the decode block's 256 rows of the Qwen3
    vocabulary (bf16). The call changes its input, so every call gets a fresh
    copy of the logits, written just before it (as the LM head would leave
    them, in L2); CUDA events bracket the top_p call alone. A draft pass over
    the same logits is timed beside it for scale."""
    import torch

    world, rank, local = dist_setup()
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    from paper_2609_19868_gb300 import build as zbuild

    zbuild.build()
    from paper_2609_19868_gb300 import _binding as zb
    from paper_2609_19868_gb300 import session
    from paper_2609_19868_gb300 import workloads as wl

    zb.load()
    zb.check_device_error()
    name = args.workload if args.workload in SELECT_LABELS else "select_decode_small"
    w = wl.make_sampling(name, device=dev)
    T, top_p = args.temperature, args.top_p
    sb = session.upload_sampling(w, dev, temperature=T)
    src = sb.draft_logits.clone()
    stream = torch.cuda.Stream(dev)
    K, W = args.steps, args.warmup
    evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
           for _ in range(K)]
    with torch.cuda.stream(stream):
        for i in range(W + K):
            sb.draft_logits.copy_(src)
            if i >= W:
                evs[i - W][0].record(stream)
            zb.top_p(sb.draft_logits, top_p, sb.draft_desc, stream=stream)
            if i >= W:
                evs[i - W][1].record(stream)
    torch.cuda.synchronize()
    assert zb.check_device_error(stream) == 0
    ms = sorted(a.elapsed_time(b) for a, b in evs)
    med = float(np.median(ms))
    kept = int(torch.isfinite(sb.draft_logits.float()).sum().item())
    with torch.cuda.stream(stream):
        sb.draft_logits.copy_(src)
        d0, d1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        sb.draft(stream)
        d0.record(stream)
        for _ in range(K):
            sb.draft(stream)
        d1.record(stream)
    torch.cuda.synchronize()
    draft_ms = d0.elapsed_time(d1) / K
    nbytes = w.rows * w.V * 2
    line = {
        "metric": "top_p calls/s (nucleus truncation of every row of a block's logits)",
        "value": round(1e3 / med, 2), "unit": "calls/s", "n_gpus": 1, "steps": K, "warmup": W,
        "ms_per_step": round(med, 5), "ms_per_step_min": round(ms[0], 5),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
        "dtype": "f32 masses in 2^-40 fixed point (bf16 logits)",
        "data": "synthetic (seeded N(0,2^2) logits with peaked tokens)",
        "config": {"workload": SELECT_LABELS[name], "temperature": T, "top_p": top_p,
                   "rows": w.rows, "kept_tokens": kept,
                   "l2": "logits rewritten before every call (L2-warm, as after the LM head)"},
        "draft_pass_ms": round(draft_ms, 5),
        "ratio_to_draft_pass": round(med / draft_ms, 2),
        "row_bytes_read_per_call": nbytes,
        "gpu_launches": K,
    }
    print(json.dumps(line), flush=True)


def _oracle_select_rows(w, T, n_draft, n_verify, vtokens):
    """The sampling oracle over the first n_draft draft rows and n_verify
    verification rows (the per-row work dominates; the per-sequence rules are
    negligible)."""
    from oracle import sampling as smp

    xd = w.draft_logits[:n_draft].float().cpu().numpy()
    xv = w.verify_logits[:n_verify].float().cpu().numpy()
    t0 = time.perf_counter()
    smp.draft_select(xd, [n_draft], [1], temperature=T, slot_threshold=0.9, seed=1, fast=True,
                     rows=range(n_draft))
    smp.verify_accept(xv, vtokens[:n_verify], [n_verify], [1], temperature=T, token_threshold=0.4,
                      rows=range(n_verify))
    return time.perf_counter() - t0


def select_cpu_baseline(w, T, sb, budget_s=20.0):
    vrows = int(sb.verify_row_offsets[-1].item())
    vt = sb.verify_tokens.cpu().numpy()
    t1 = _oracle_select_rows(w, T, 1, 1, vt)
    per_row = t1 / 2
    n = int(max(1, min(w.rows, budget_s / 2 / max(per_row, 1e-6))))
    nd, nv = n, min(n, max(vrows, 1))
    t = _oracle_select_rows(w, T, nd, nv, vt)
    frac_d, frac_v = nd / w.rows, nv / max(vrows, 1)
    step_s = t / (nd + nv) * (w.rows + vrows)
    return {"value": round(1.0 / step_s, 4), "unit": "steps/s", "cores": 1, "kind": "oracle",
            "sample": f"{nd} of {w.rows} draft rows and {nv} of {vrows} verification rows "
                      f"(numpy fp64 oracle), scaled to the whole step by rows"}


def workload_subset(w, seqs):
    """The workload restricted to sequences ``seqs`` (their rows, lengths and
    caches; a paged cache keeps only their pages, renumbered)."""
    from dataclasses import replace

    sub = w
    if len(seqs) < w.B:
        idx = np.asarray(seqs)
        offs = w.q_row_offsets
        rows = np.concatenate([np.arange(offs[b], offs[b + 1]) for b in idx])
        new_offs = np.concatenate([[0], np.cumsum(w.R[idx])]).astype(np.int32)
        import torch

        ridx = torch.as_tensor(rows)
        if w.page_size:
            # the subset's own pages, renumbered into a compact pool
            table = w.page_table[idx]
            used = np.unique(table[table >= 0])
            remap = np.full(w.n_pages, -1, dtype=np.int64)
            remap[used] = np.arange(len(used))
            new_table = np.where(table >= 0, remap[np.maximum(table, 0)], -1).astype(np.int32)
            pidx = torch.as_tensor(used)
            caches = dict(k_cache=w.k_cache[pidx], v_cache=w.v_cache[pidx],
                          page_table=new_table, n_pages=len(used))
        else:
            caches = dict(k_cache=w.k_cache[torch.as_tensor(idx)],
                          v_cache=w.v_cache[torch.as_tensor(idx)])
        sub = replace(w, B=len(idx), cache_lens=w.cache_lens[idx], n_slots=w.n_slots[idx],
                      slot_len=w.slot_len[idx], mask_mode=w.mask_mode[idx],
                      accept_len=w.accept_len[idx], q_row_offsets=new_offs,
                      q=w.q[ridx], k_new=w.k_new[ridx], v_new=w.v_new[ridx], **caches)
    return sub


def _oracle_step(oracle, w, seqs, threads=0):
    """The oracle's version of one step restricted to sequences ``seqs``."""
    sub = workload_subset(w, seqs)
    t0 = time.perf_counter()
    kc, vc, lens = oracle.kv_append(sub.k_new, sub.v_new, sub.R, sub.k_cache, sub.v_cache,
                                    sub.cache_lens, sub.page_table, sub.q_row_offsets,
                                    page_size=sub.page_size, commit=False)
    oracle.slot_attn(sub.q, kc, vc, sub.cache_lens, sub.page_table, sub.n_slots, sub.slot_len,
                     sub.mask_mode, sub.q_row_offsets, scale=sub.scale,
                     page_size=sub.page_size, capacity=sub.capacity,
                     n_pages=sub.n_pages if sub.page_size else -1, threads=threads)
    oracle.kv_append(sub.k_new, sub.v_new, sub.accept_len, kc, vc, lens, sub.page_table,
                     sub.q_row_offsets, page_size=sub.page_size, commit=True)
    return time.perf_counter() - t0


def _visible_pairs(w):
    """Visible (row, head, key) pairs of every sequence: the oracle's work."""
    P = w.cache_lens.astype(np.int64)
    R = w.R
    return np.where(w.mask_mode == 0, w.Hq * R * (P + R), w.Hq * (R * P + R * (R + 1) // 2))


def cpu_baseline(w, budget_s=20.0):
    """The oracle, as it stands, on the host cores: whole steps over the
    first sequences of the batch, scaled to the full batch by the visible
    (row, head, key) pairs (the oracle's work is proportional to them)."""
    import oracle

    oracle.build()
    cores = oracle.max_threads()
    pairs = _visible_pairs(w)
    t1 = _oracle_step(oracle, w, [0])
    per_pair = t1 / max(int(pairs[0]), 1)
    n_seq = int(np.searchsorted(np.cumsum(pairs), budget_s / max(per_pair, 1e-15), side="right"))
    n_seq = max(1, min(w.B, n_seq))
    t = _oracle_step(oracle, w, list(range(n_seq)))
    step_s = t * float(pairs.sum()) / float(pairs[:n_seq].sum())
    return {"value": round(1.0 / step_s, 4), "unit": "steps/s", "cores": cores,
            "kind": "oracle",
            "sample": f"{n_seq} of {w.B} sequences of one step (stage + attention + commit, "
                      f"fp64 C oracle with OpenMP, {t:.1f} s), scaled to the full batch by "
                      f"visible (row, head, key) pairs"}


def run_reference(args):
    """The fp64 CPU oracle as the reference arm (rank 0 only)."""
    world, rank, local = dist_setup()
    if rank != 0:
        return
    import oracle
    from paper_2609_19868_gb300 import workloads as wl

    oracle.build()
    name, mode = entry_workload(args.workload)
    w = wl.make(name)
    if mode is not None:
        w = w.with_mode(mode)
    cores = oracle.max_threads()
    # size each step's sample so the whole run stays within ~2 minutes
    pairs = _visible_pairs(w)
    per_pair = _oracle_step(oracle, w, [0]) / max(int(pairs[0]), 1)
    budget = 120.0 / max(1, args.steps + args.warmup)
    n_seq = int(np.searchsorted(np.cumsum(pairs), budget / max(per_pair, 1e-15), side="right"))
    n_seq = max(1, min(w.B, n_seq))
    for _ in range(args.warmup):
        _oracle_step(oracle, w, list(range(n_seq)))
    total = 0.0
    for _ in range(args.steps):
        total += _oracle_step(oracle, w, list(range(n_seq)))
    step_s = total / args.steps * float(pairs.sum()) / float(pairs[:n_seq].sum())
    value = 1.0 / step_s
    sample = (f"{n_seq} of {w.B} sequences per step (stage + attention + commit), "
              f"scaled to the full batch by visible (row, head, key) pairs")
    line = {
        "impl": "reference",
        "metric": "slot-decode steps/s (one layer: stage + slot attention + commit)",
        "value": round(value, 4),
        "unit": "steps/s",
        "n_gpus": world,
        "steps": args.steps,
        "warmup": args.warmup,
        "ms_per_step": round(step_s * 1e3, 3),
        "higher_is_better": True,
        "scaling": "weak",
        "vs_baseline": None,
        "dtype": "f64",
        "data": "synthetic (seeded N(0,1), random-init; no weights or datasets)",
        "config": {"workload": WORKLOAD_LABELS.get(args.workload, args.workload),
                   "global_batch": w.B},
        "cpu_baseline": {"value": round(value, 4), "unit": "steps/s", "cores": cores,
                         "kind": "oracle", "sample": sample},
        "e2e": {"value": round(value, 4), "unit": "steps/s", "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


def run_select_reference(args):
    """The sampling oracle as the reference arm of --path select (rank 0)."""
    world, rank, local = dist_setup()
    if rank != 0:
        return
    from oracle import sampling as smp
    from paper_2609_19868_gb300 import workloads as wl

    name = args.workload if args.workload in SELECT_LABELS else "select_decode_small"
    w = wl.make_sampling(name)
    T = args.temperature
    xv = w.verify_logits.float().numpy()
    xd = w.draft_logits.float().numpy()
    t0 = time.perf_counter()
    smp.draft_select(xd[:1], [1], [1], temperature=T, slot_threshold=0.9, fast=True)
    per_row = time.perf_counter() - t0
    budget = 120.0 / max(1, args.steps + args.warmup)
    n = int(max(1, min(w.rows, budget / 2 / max(per_row, 1e-6))))
    nv = min(n, w.verify_rows)

    def one():
        t = time.perf_counter()
        smp.draft_select(xd[:n], [n], [1], temperature=T, slot_threshold=0.9, fast=True,
                         rows=range(n))
        smp.verify_accept(xv[:nv], w.verify_tokens[:nv], [nv], [1], temperature=T,
                          token_threshold=0.4, rows=range(nv))
        return time.perf_counter() - t

    for _ in range(args.warmup):
        one()
    total = sum(one() for _ in range(args.steps))
    step_s = total / args.steps / (n + nv) * (w.rows + w.verify_rows)
    value = 1.0 / step_s
    sample = (f"{n} of {w.rows} draft rows and {nv} of {w.verify_rows} verification rows per "
              f"step (numpy fp64 oracle), scaled to the whole step by rows")
    line = {
        "impl": "reference",
        "metric": "slot select + token accept steps/s (draft select over the block's logits, "
                  "then acceptance over the verification block)",
        "value": round(value, 4), "unit": "steps/s", "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": round(step_s * 1e3, 3), "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic (seeded N(0,2^2) logits with peaked tokens; no weights or datasets)",
        "config": {"workload": SELECT_LABELS[name], "temperature": T, "global_batch": w.B},
        "cpu_baseline": {"value": round(value, 4), "unit": "steps/s", "cores": 1,
                         "kind": "oracle", "sample": sample},
        "e2e": {"value": round(value, 4), "unit": "steps/s", "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=100)
    ap.add_argument("--warmup", type=int, default=10)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--workload", default=None,
                    choices=list(WORKLOAD_LABELS) + list(WORKLOAD_ALIASES) + list(SELECT_LABELS))
    ap.add_argument("--reps", type=int, default=30,
                    help="at least this many timed K-step regions (median and min reported)")
    ap.add_argument("--min-seconds", type=float, default=1.0,
                    help="the headline's repeated regions last at least this long")
    ap.add_argument("--config-seconds", type=float, default=0.3,
                    help="each per_config entry's repeated regions last at least this long")
    ap.add_argument("--no-per-config", dest="per_config", action="store_false",
                    help="measure the chosen workload only")
    ap.add_argument("--path", choices=["attention", "select", "reorder", "mode_a", "top_p"],
                    default="attention",
                    help="attention: the slot-decode layer step (stage + attention + commit); "
                         "select: slot selection + token acceptance over logits")
    ap.add_argument("--temperature", type=float, default=0.0)
    ap.add_argument("--top-p", type=float, default=0.9)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--cpu-budget", type=float, default=20.0)
    ap.add_argument("--no-clocks", dest="clocks", action="store_false")
    args = ap.parse_args()
    if args.warmup < 3:
        args.warmup = 3
    if args.workload is None:
        args.workload = ("select_decode_small" if args.path in ("select", "top_p")
                         else "serving_mix")
    args.workload = WORKLOAD_ALIASES.get(args.workload, args.workload)
    if args.path in ("attention",) and args.workload not in WORKLOAD_LABELS:
        ap.error(f"--workload {args.workload} is not an attention workload")
    if args.path == "top_p":
        if args.impl == "reference":
            print(json.dumps({"impl": "reference", "unavailable":
                              "the top_p path is measured against a draft pass only"}), flush=True)
        else:
            run_top_p(args)
    elif args.path == "mode_a":
        if args.impl == "reference":
            print(json.dumps({"impl": "reference", "unavailable":
                              "the Mode A path is measured against its roofline only"}), flush=True)
        else:
            run_mode_a(args)
    elif args.path == "reorder":
        if args.impl == "reference":
            print(json.dumps({"impl": "reference", "unavailable":
                              "the reorder path's reference arm is its oracle, timed as "
                              "cpu_baseline in the --path reorder line"}), flush=True)
        else:
            run_reorder(args)
    elif args.path == "select":
        if args.impl == "reference":
            run_select_reference(args)
        else:
            run_select(args)
    elif args.impl == "reference":
        run_reference(args)
    else:
        run_ours(args)


if __name__ == "__main__":
    main()
