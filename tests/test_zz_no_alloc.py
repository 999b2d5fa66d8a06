"""zarya_slot_attn_noalloc: the attention entry point for callers that cannot
allocate device memory when they run it (an engine that gave all of HBM to
its own pool, a host that forbids its plug-ins to allocate, a decode loop
that cannot pay for a synchronising cudaMalloc/cudaFree). Its split-KV scratch
is a fixed array inside the library, so it takes no workspace.

These tests call it through the C ABI and check, on two calls in a row, that
it gives exactly the bytes zarya_slot_attn gives with a workspace (same kernel,
same split plan, and a merge whose order does not depend on arrival), that it
matches the fp64 oracle within the parity tolerance, and that a plan needing
more scratch than the array holds is refused.

The file name sorts last, so pytest collects it after every other test file:
a run that stops at the first failure has then already run all the others.
Each test sets up its own inputs, so the file also passes on its own.
"""
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


def _noalloc(zb, db, out):
    zb.slot_attn_noalloc(db.q, db.k_cache, db.v_cache, db.cache_lens, db.page_table, db.n_slots,
                         db.slot_len, db.mask_mode, out, db.desc)


def _serving_mix_mixed_modes():
    """A paged serving_mix batch (16-token pages, random page permutation)
    with slot lengths 4 and 8 and every mask mode, the slot-independent one
    included, mixed over the sequences."""
    w = wl.make("serving_mix", small=True, B=3, slot_len=("choice", (4, 8)))
    return w, np.array([0, 1, 2], dtype=np.int32)


# More than 3 key splits per tile merge through scratch memory (up to 3
# merge inside a thread-block cluster); these plans need 8.6 to 12.1 MiB.
@pytest.mark.parametrize("name,splits,override", [("decode_small", 9, {"B": 2}),
                                                  ("decode_small", 17, {"B": 1}),
                                                  ("decode_small", 12, {"B": 2}),
                                                  ("serving_mix", 4, None)])
def test_noalloc_matches_workspace_entry_point_twice(zs, oracle_mod, name, splits, override):
    session, zb = zs
    if name == "serving_mix":
        w, modes = _serving_mix_mixed_modes()
        w = w.with_mode(0)
        w.mask_mode[:] = modes
    else:
        w = wl.make(name, **override)
    db = session.upload(w, "cuda", kv_splits=splits)
    assert zb.workspace_size(db.desc) > 0  # the plan really uses scratch
    assert zb.workspace_size(db.desc) <= 16 << 20
    db.stage()
    db.attend()
    ref = db.out.clone()
    kc, vc = oracle_staged(oracle_mod, w)
    expect = oracle_full(oracle_mod, w, kc, vc)
    for call in range(2):
        out = torch.full_like(db.out, float("nan"))
        _noalloc(zb, db, out)
        torch.cuda.synchronize()
        assert zb.check_device_error() == 0
        assert torch.equal(out, ref), f"call {call}: differs from zarya_slot_attn"
        ok, err, _ = tolerance_ok(out, expect, w.dtype)
        assert ok, f"call {call}: max|err| = {err:.3e} against the oracle"


def test_noalloc_second_call_with_other_inputs(zs):
    """The scratch keeps the previous call's contents; a following call with
    a different mask still gives exactly the workspace entry point's bytes."""
    session, zb = zs
    w = wl.make("decode_small", B=2)
    for mode in (0, 1, 2):
        db = session.upload(w, "cuda", kv_splits=10, mask_mode=mode)
        assert zb.workspace_size(db.desc) > 0
        db.stage()
        db.attend()
        ref = db.out.clone()
        out = torch.zeros_like(db.out)
        _noalloc(zb, db, out)
        torch.cuda.synchronize()
        assert zb.check_device_error() == 0
        assert torch.equal(out, ref), f"mode {mode}"


def test_noalloc_refuses_plans_beyond_its_scratch(zs):
    session, zb = zs
    w = wl.make("long_ctx", small=True)
    db = session.upload(w, "cuda", kv_splits=9)
    assert zb.workspace_size(db.desc) > 16 << 20
    out = torch.zeros_like(db.out)
    with pytest.raises(zb.ZaryaError) as e:
        _noalloc(zb, db, out)
    assert e.value.status == zb.ERR_UNSUPPORTED
    # without splits no scratch is needed and the call goes through
    db1 = session.upload(w, "cuda", kv_splits=1)
    db1.stage()
    db1.attend()
    _noalloc(zb, db1, out)
    torch.cuda.synchronize()
    assert zb.check_device_error() == 0
    assert torch.equal(out, db1.out)
