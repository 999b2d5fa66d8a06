"""GPU parity of zarya_slot_attn against the fp64 CPU oracle.

Every test calls the CUDA library through the C ABI (the ctypes binding) on
seeded synthetic inputs of the five workloads; the oracle sees the same
bytes. Reduced workloads are compared element by element on every output;
full-size workloads, in the launch configuration the benchmark uses, on
sampled rows the oracle computes one by one.
"""
from dataclasses import replace

import numpy as np
import pytest
import torch

from paper_2609_19868_gb300 import workloads as wl
from _helpers import (gather_rows, oracle_full, oracle_rows, oracle_staged, sample_rows,
                      tolerance_ok)

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def zs():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2609_19868_gb300 import build, session
    from paper_2609_19868_gb300 import _binding as zb

    build.build()
    zb.load()
    zb.check_device_error()
    return session, zb


def _cases():
    out = []
    for name in wl.ORDER:
        spec = wl.SPECS[name]
        if spec["mode"][0] == "both":
            out += [(name, 0), (name, 1)]
        else:
            out.append((name, None))
    return out


def _run(zs, w, mode=None, kv_splits=0):
    session, zb = zs
    db = session.upload(w, "cuda", kv_splits=kv_splits, mask_mode=mode)
    db.stage()
    db.attend()
    torch.cuda.synchronize()
    assert zb.check_device_error() == 0
    return db


@pytest.mark.parametrize("name,mode", _cases())
def test_reduced_workload_matches_oracle_everywhere(zs, oracle_mod, name, mode):
    w = wl.make(name, small=True)
    db = _run(zs, w, mode)
    kc, vc = oracle_staged(oracle_mod, w)
    ref = oracle_full(oracle_mod, w, kc, vc, mode)
    got = db.out
    assert not torch.isnan(got).any()
    ok, err, scale = tolerance_ok(got, ref, w.dtype)
    assert ok, f"{name} mode={mode}: max|err|={err:.3e} max|ref|={scale:.3f}"


@pytest.mark.parametrize("name,mode", [("decode_small", None), ("long_ctx", 0), ("long_ctx", 1),
                                       ("ragged_mid", None)])
@pytest.mark.parametrize("splits", [1, 2, 3, 7])
def test_split_kv_merge_matches_oracle(zs, oracle_mod, name, mode, splits):
    """Forcing the key range to be split n ways (up to 3 splits form a
    thread-block cluster and merge through distributed shared memory, more
    merge through the workspace) still matches the oracle."""
    w = wl.make(name, small=True)
    db = _run(zs, w, mode, kv_splits=splits)
    kc, vc = oracle_staged(oracle_mod, w)
    ref = oracle_full(oracle_mod, w, kc, vc, mode)
    ok, err, scale = tolerance_ok(db.out, ref, w.dtype)
    assert ok, f"{name} splits={splits}: max|err|={err:.3e}"


@pytest.mark.parametrize("name,small,override,splits", [("long_ctx", True, {}, 9),
                                                        ("long_ctx", True, {}, 13),
                                                        ("decode_small", False, {"B": 2}, 17)])
def test_workspace_merge_beyond_a_cluster_matches_oracle(zs, oracle_mod, name, small, override,
                                                         splits):
    """More than 8 key splits merge through the workspace (last CTA to arrive,
    in split order) instead of a cluster; still matches the oracle."""
    session, zb = zs
    w = wl.make(name, small=small, **override)
    for mode in (0, 1):
        db = session.upload(w, "cuda", kv_splits=splits, mask_mode=mode)
        assert zb.workspace_size(db.desc) > 0
        db.stage()
        db.attend()
        torch.cuda.synchronize()
        assert zb.check_device_error() == 0
        kc, vc = oracle_staged(oracle_mod, w)
        sel = sample_rows(w, 96, seed=3)
        ref = oracle_rows(oracle_mod, w, kc, vc, sel, mode)
        ok, err, _ = tolerance_ok(gather_rows(db.out, w, sel), ref, w.dtype)
        assert ok, f"{name} splits={splits} mode={mode}: max|err|={err:.3e}"


@pytest.mark.parametrize("splits", [2, 3, 17])
def test_split_merge_is_bitwise_deterministic(zs, splits):
    """The merged result does not depend on which split finishes first."""
    session, zb = zs
    w = wl.make("decode_small", B=2)
    outs = []
    for _ in range(3):
        db = session.upload(w, "cuda", kv_splits=splits)
        db.stage()
        db.attend()
        torch.cuda.synchronize()
        outs.append(db.out.clone())
    assert torch.equal(outs[0], outs[1]) and torch.equal(outs[0], outs[2])


def test_workspace_counters_return_to_zero(zs):
    """The workspace merge leaves its arrival counters at zero, so a workspace
    can be reused: two calls in a row give identical results."""
    w = wl.make("decode_small", B=2)
    session, zb = zs
    db = session.upload(w, "cuda", kv_splits=12)
    db.stage()
    db.attend()
    first = db.out.clone()
    db.out.zero_()
    db.attend()
    torch.cuda.synchronize()
    assert zb.check_device_error() == 0
    assert torch.equal(first, db.out)
    # the counters are the last units*4 bytes (rounded) of the workspace
    assert db.workspace is not None


def test_repeat_runs_are_bitwise_deterministic(zs):
    w = wl.make("serving_mix", small=True)
    a = _run(zs, w).out.clone()
    b = _run(zs, w).out.clone()
    assert torch.equal(a, b)


def test_paged_cache_equals_contiguous_bitwise(zs):
    """The same logical keys behind a random page table give bit-identical
    outputs (same key tiles, same order)."""
    session, zb = zs
    wc = wl.make("ragged_mid", small=True)
    rng = np.random.default_rng(5)
    ps = 16
    P = wc.cache_lens.astype(np.int64)
    R = wc.R
    npg = (P + R + ps - 1) // ps
    n_pages = int(npg.sum()) + 3
    perm = rng.permutation(n_pages)
    pt = np.full((wc.B, int(npg.max())), -1, dtype=np.int32)
    kp = torch.full((n_pages, ps, wc.Hkv, wc.D), float("nan"), dtype=torch.bfloat16)
    vp = torch.full_like(kp, float("nan"))
    start = 0
    for b in range(wc.B):
        pt[b, :npg[b]] = perm[start:start + npg[b]]
        start += int(npg[b])
        for lp in range(int(npg[b])):
            lo = lp * ps
            hi = min(lo + ps, int(P[b]))
            if hi > lo:
                kp[pt[b, lp], :hi - lo] = wc.k_cache[b, lo:hi]
                vp[pt[b, lp], :hi - lo] = wc.v_cache[b, lo:hi]
    from dataclasses import replace
    wp = replace(wc, page_size=ps, capacity=int(npg.max()) * ps, n_pages=n_pages, page_table=pt,
                 k_cache=kp, v_cache=vp)
    oc = _run(zs, wc, kv_splits=1).out
    op = _run(zs, wp, kv_splits=1).out
    assert torch.equal(oc, op)


@pytest.mark.parametrize("name,mode", _cases())
def test_full_size_sampled_rows_match_oracle(zs, oracle_mod, name, mode):
    """Full-size workloads in the benchmark's launch configuration (automatic
    split plan): sampled (sequence, head, row) outputs against the oracle."""
    w = wl.make(name)
    db = _run(zs, w, mode)
    out = db.out
    assert not torch.isnan(out).any()
    del db
    kc, vc = oracle_staged(oracle_mod, w)
    sel = sample_rows(w, 192, seed=7)
    ref = oracle_rows(oracle_mod, w, kc, vc, sel, mode)
    got = gather_rows(out, w, sel)
    ok, err, scale = tolerance_ok(got, ref, w.dtype)
    assert ok, f"{name} mode={mode}: max|err|={err:.3e} max|ref|={scale:.3f}"


def test_cuda_graph_capture_of_a_step_matches_eager(zs):
    """A whole step (stage, attention, commit) captured into a CUDA graph and
    replayed gives the same output bits and lengths as eager calls."""
    session, zb = zs
    w = wl.make("decode_small", small=True)
    s = torch.cuda.Stream()
    with torch.cuda.stream(s):
        eager = session.upload(w, "cuda", kv_splits=2)
        eager.stage(s)
        eager.attend(s)
        eager.commit(s)
        db = session.upload(w, "cuda", kv_splits=2)
        db.stage(s)      # warm-up outside the capture
        db.attend(s)
    torch.cuda.synchronize()
    db.cache_lens.copy_(torch.as_tensor(w.cache_lens))
    db.out.zero_()
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=s):
        db.stage(s)
        db.attend(s)
        db.commit(s)
    g.replay()
    torch.cuda.synchronize()
    assert zb.check_device_error() == 0
    assert torch.equal(db.out, eager.out)
    assert torch.equal(db.cache_lens, eager.cache_lens)


# Ragged batches whose grids take several waves of CTAs (one CTA per SM),
# compared on every output.
@pytest.mark.parametrize("name,override", [
    ("ragged_mid", dict(B=48, prefix=("uniform", 37, 400))),        # distinct lengths
    ("ragged_mid", dict(B=128, prefix=("uniform", 100, 103))),      # many equal lengths
    ("ragged_mid", dict(B=129, prefix=("uniform", 37, 150))),
    ("serving_mix", dict(B=40, prefix=("loguniform", 20, 900))),    # paged, mixed L and masks
])
def test_multi_wave_ragged_batch_matches_oracle_everywhere(zs, oracle_mod, name, override):
    w = wl.make(name, seed=11, **override)
    db = _run(zs, w)
    kc, vc = oracle_staged(oracle_mod, w)
    ref = oracle_full(oracle_mod, w, kc, vc)
    got = db.out
    assert not torch.isnan(got).any()
    ok, err, scale = tolerance_ok(got, ref, w.dtype)
    assert ok, f"{name} {override}: max|err|={err:.3e} max|ref|={scale:.3f}"


def _one_sequence(w, b):
    """Sequence b of a contiguous-cache workload as a batch of one."""
    lo, hi = int(w.q_row_offsets[b]), int(w.q_row_offsets[b + 1])
    sl = slice(b, b + 1)
    return replace(w, B=1, cache_lens=w.cache_lens[sl].copy(), n_slots=w.n_slots[sl].copy(),
                   slot_len=w.slot_len[sl].copy(), mask_mode=w.mask_mode[sl].copy(),
                   accept_len=w.accept_len[sl].copy(),
                   q_row_offsets=np.array([0, hi - lo], dtype=w.q_row_offsets.dtype),
                   q=w.q[lo:hi].clone(), k_cache=w.k_cache[sl].clone(),
                   v_cache=w.v_cache[sl].clone(), k_new=w.k_new[lo:hi].clone(),
                   v_new=w.v_new[lo:hi].clone())


def test_batching_leaves_each_sequence_bitwise_unchanged(zs):
    """With one split per tile a sequence's outputs are the same bits whether
    its CTAs run inside a multi-wave batch or alone."""
    w = wl.make("ragged_mid", seed=13, B=48, prefix=("uniform", 37, 400))
    full = _run(zs, w, kv_splits=1).out
    order = np.argsort(-(w.cache_lens.astype(np.int64) + w.R), kind="stable")
    for b in sorted({int(order[0]), int(order[-1]), 0, 17, 47}):
        lo, hi = int(w.q_row_offsets[b]), int(w.q_row_offsets[b + 1])
        alone = _run(zs, _one_sequence(w, b), kv_splits=1).out
        assert torch.equal(full[lo:hi], alone), f"sequence {b}"


def test_dispatch_order_is_longest_first_and_changes_no_byte(zs, oracle_mod):
    """A paired launch of several waves first sorts its work items: the
    workspace then holds a permutation of (sequence, pair) items in
    non-increasing cost (M-tiles x key tiles, the tile loop's work; empty
    items last), ties in item order, and the output matches the oracle. The
    same batch in grid order (a forced split: the single-tile kernel, no
    order) matches it too."""
    session, zb = zs
    w = wl.make("serving_mix", seed=11, B=40, prefix=("loguniform", 20, 900))
    db = _run(zs, w)
    assert zb.slot_attn_kernel(db.desc) == "slot_attn_pair_kernel"
    assert zb.slot_attn_launches(db.desc) == 2
    T = int(db.desc.max_rows * (w.Hq // w.Hkv) + 127) // 128
    T = (T + 1) // 2
    perm = db.workspace[: 4 * w.B * T].view(torch.int32).cpu().numpy()
    assert sorted(perm.tolist()) == list(range(w.B * T))
    rpt = 128 // (w.Hq // w.Hkv)
    cost = []
    for item in perm:
        b, t = divmod(int(item), T)
        R, P = int(w.R[b]), int(w.cache_lens[b])
        r0 = 2 * t * rpt
        if r0 >= R:
            cost.append(0)
            continue
        m = min(2, -(-(R - r0) // rpt))
        r_hi = min(r0 + 2 * rpt, R) - 1
        kv = P + R if w.mask_mode[b] == 0 else P + r_hi + 1
        cost.append(m * (-(-kv // 128)) + 1)
    keys = [(-c, int(i)) for c, i in zip(cost, perm)]
    assert keys == sorted(keys)
    kc, vc = oracle_staged(oracle_mod, w)
    ok, err, _ = tolerance_ok(db.out, oracle_full(oracle_mod, w, kc, vc), w.dtype)
    assert ok, f"max|err|={err:.3e}"
    grid_order = _run(zs, w, kv_splits=1)
    assert zb.slot_attn_kernel(grid_order.desc) == "slot_attn_tc_kernel"
    assert zb.slot_attn_launches(grid_order.desc) == 1
    ok, err, _ = tolerance_ok(grid_order.out, oracle_full(oracle_mod, w, kc, vc), w.dtype)
    assert ok, f"grid order: max|err|={err:.3e}"


@pytest.mark.parametrize("D,page_size,mode", [(32, 0, 1), (64, 16, 0), (96, 16, 1), (128, 0, 2),
                                              (128, 16, 2), (256, 0, 0)])
def test_fp32_tier_shapes_and_masks_match_oracle(zs, oracle_mod, D, page_size, mode):
    """The fp32 kernel over head sizes 32..256, contiguous and paged caches,
    all three masks, prefixes from 0 (chunks of 32 keys with ragged tails)."""
    w = wl.make("tiny_fp32", seed=13, B=5, Hq=8, Hkv=2, D=D, page_size=page_size,
                prefix=("uniform", 0, 300), slot_len=("choice", [2, 3, 8]),
                mode=("fixed", mode), accept=("upto_R",))
    w = replace(w, cache_lens=w.cache_lens.copy())
    w.cache_lens[0] = 0
    db = _run(zs, w)
    kc, vc = oracle_staged(oracle_mod, w)
    ok, err, scale = tolerance_ok(db.out, oracle_full(oracle_mod, w, kc, vc), w.dtype)
    assert ok, f"D={D} page={page_size} mode={mode}: max|err|={err:.3e} max|ref|={scale:.3f}"
