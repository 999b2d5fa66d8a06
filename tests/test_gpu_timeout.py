"""Failure detection of the attention kernel: every pipeline wait is bounded.

A wait that runs out records ZARYA_DEVERR_TIMEOUT in the device error word,
and the CTA unwinds: it lets its own tensor copies and MMAs finish, frees its
tensor memory and writes no output, so the context stays usable. These tests
make a wait run out on purpose, with no fault: the descriptor's debug stall
has the MMA warp wait on a barrier that nothing completes, under a 1 ms limit
instead of the default 2 s. They check the error word, that the output was
left alone, that the call ended promptly, and that the next call at the
default limit matches the fp64 oracle.
"""
import ctypes
import time

import numpy as np
import pytest
import torch

from paper_2609_19868_gb300 import workloads as wl
from _helpers import oracle_full, oracle_staged, tolerance_ok

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


def _with_limit(zb, desc, wait_limit_us, debug_flags):
    d = zb.AttnDesc.from_buffer_copy(desc)
    d._keep = desc._keep
    d.wait_limit_us, d.debug_flags = wait_limit_us, debug_flags
    return d


def _attend(zb, db, desc, out, staged):
    if staged:
        zb.slot_attn_staged(db.q, db.k_new, db.v_new, db.k_cache, db.v_cache, db.cache_lens,
                            db.page_table, db.n_slots, db.slot_len, db.mask_mode, out, desc,
                            db.workspace)
    else:
        zb.slot_attn(db.q, db.k_cache, db.v_cache, db.cache_lens, db.page_table, db.n_slots,
                     db.slot_len, db.mask_mode, out, desc, db.workspace)


# kv_splits 1: one CTA per tile; 5: five CTAs per tile merging through the
# workspace. Paged and contiguous caches, plain and staged attention.
@pytest.mark.parametrize("name,splits,staged", [("decode_small", 1, False),
                                                ("decode_small", 5, False),
                                                ("decode_small", 1, True),
                                                ("serving_mix", 1, True)])
def test_a_wait_that_runs_out_unwinds_and_reports_it(zs, oracle_mod, name, splits, staged):
    session, zb = zs
    w = wl.make(name, small=True)
    db = session.upload(w, "cuda", kv_splits=splits)
    if not staged:
        db.stage()
    torch.cuda.synchronize()
    assert zb.check_device_error() == 0
    stall = _with_limit(zb, db.desc, 1000, zb.DEBUG_STALL)
    out = torch.full_like(db.out, float("nan"))
    t0 = time.perf_counter()
    _attend(zb, db, stall, out, staged)
    code = zb.check_device_error()
    elapsed = time.perf_counter() - t0
    assert code == zb.DEVERR_TIMEOUT
    assert elapsed < 1.0, f"the unwound launch took {elapsed:.3f} s"
    assert torch.isnan(out).all(), "a CTA that gave up wrote output"
    # After a call that set the error word the workspace is zeroed again
    # (zarya_slot_attn_workspace_size's contract), then the default limit.
    if db.workspace is not None:
        db.workspace.zero_()
    for call in range(2):
        out.fill_(float("nan"))
        _attend(zb, db, db.desc, out, staged)
        torch.cuda.synchronize()
        assert zb.check_device_error() == 0
        kc, vc = oracle_staged(oracle_mod, w)
        ok, err, _ = tolerance_ok(out, oracle_full(oracle_mod, w, kc, vc), w.dtype)
        assert ok, f"call {call} after the timeout: max|err| = {err:.3e}"


def test_a_short_limit_that_is_not_reached_changes_nothing(zs):
    """A 100 ms limit bounds waits that last microseconds: the result is the
    default limit's, bit for bit."""
    session, zb = zs
    w = wl.make("ragged_mid", small=True)
    db = session.upload(w, "cuda")
    db.stage()
    db.attend()
    ref = db.out.clone()
    out = torch.zeros_like(ref)
    _attend(zb, db, _with_limit(zb, db.desc, 100_000, 0), out, False)
    torch.cuda.synchronize()
    assert zb.check_device_error() == 0
    assert torch.equal(out, ref)
