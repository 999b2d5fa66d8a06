"""GPU parity of the slot-independent verification mask (mask mode 2: block
row r = s*L + j sees the prefix and rows s*L .. r of its own slot), on every
workload's shapes, against the fp64 oracle."""
import numpy as np
import pytest
import torch

from paper_2609_19868_gb300 import workloads as wl
from _helpers import gather_rows, oracle_full, oracle_rows, oracle_staged, sample_rows, tolerance_ok

pytestmark = pytest.mark.gpu
MODE = 2


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


def _run(zs, w, kv_splits=0, staged=False):
    session, zb = zs
    db = session.upload(w, "cuda", kv_splits=kv_splits, mask_mode=MODE)
    if staged:
        db.stage_and_attend()
    else:
        db.stage()
        db.attend()
    torch.cuda.synchronize()
    assert zb.check_device_error() == 0
    return db


@pytest.mark.parametrize("name", wl.ORDER)
def test_reduced_workload_matches_oracle_everywhere(zs, oracle_mod, name):
    w = wl.make(name, small=True)
    db = _run(zs, w)
    kc, vc = oracle_staged(oracle_mod, w)
    ref = oracle_full(oracle_mod, w, kc, vc, MODE)
    assert not torch.isnan(db.out.float()).any()
    ok, err, scale = tolerance_ok(db.out, ref, w.dtype)
    assert ok, f"{name}: max|err|={err:.3e} max|ref|={scale:.3f}"


@pytest.mark.parametrize("name", ["decode_small", "ragged_mid", "serving_mix", "long_ctx"])
def test_full_size_sampled_rows_match_oracle(zs, oracle_mod, name):
    w = wl.make(name)
    db = _run(zs, w, staged=True)
    out = db.out
    del db
    kc, vc = oracle_staged(oracle_mod, w)
    sel = sample_rows(w, 192, seed=11)
    ref = oracle_rows(oracle_mod, w, kc, vc, sel, MODE)
    ok, err, scale = tolerance_ok(gather_rows(out, w, sel), ref, w.dtype)
    assert ok, f"{name}: max|err|={err:.3e} max|ref|={scale:.3f}"


@pytest.mark.parametrize("splits", [2, 3, 7, 12])
def test_split_keys(zs, oracle_mod, splits):
    w = wl.make("long_ctx", small=True)
    db = _run(zs, w, kv_splits=splits)
    kc, vc = oracle_staged(oracle_mod, w)
    ref = oracle_full(oracle_mod, w, kc, vc, MODE)
    ok, err, _ = tolerance_ok(db.out, ref, w.dtype)
    assert ok, f"splits={splits}: max|err|={err:.3e}"


def test_one_slot_per_block_equals_slot_causal(zs):
    """With one slot per sequence the two verification masks coincide: the
    GPU outputs are bit-identical."""
    session, zb = zs
    w = wl.make("decode_small", small=True, n_slots=1, slot_len=("fixed", 8))
    outs = []
    for mode in (1, 2):
        db = session.upload(w, "cuda", mask_mode=mode)
        db.stage()
        db.attend()
        torch.cuda.synchronize()
        outs.append(db.out.clone())
    assert zb.check_device_error() == 0
    assert torch.equal(outs[0], outs[1])
