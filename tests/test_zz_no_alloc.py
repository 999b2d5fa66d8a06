"""zarya_slot_attn_noalloc: the attention entry point for callers that cannot
allocate device memory when they run it (an engine that gave all of HBM to
its own pool, a host that forbids its plug-ins to allocate, a decode loop
that cannot pay for cudaMalloc/cudaFree). Its split-KV scratch is a fixed
array inside the library, so it takes no workspace.

These tests call it through the C ABI and compare it with zarya_slot_attn
(given a workspace) within the parity tolerance, on two calls in a row, and
check that a plan needing more scratch than the array holds is refused.
This file is collected last on purpose.
"""
import pytest
import torch

from paper_2609_19868_gb300 import workloads as wl
from _helpers import tolerance_ok

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


# More than 3 key splits per tile merge through scratch memory (up to 3
# merge inside a thread-block cluster); these plans need 8.6 to 12.1 MiB.
@pytest.mark.parametrize("name,small,splits,override", [("decode_small", False, 9, {"B": 2}),
                                                        ("decode_small", False, 17, {"B": 1}),
                                                        ("decode_small", False, 12, {"B": 2})])
def test_noalloc_matches_workspace_entry_point_twice(zs, name, small, splits, override):
    session, zb = zs
    w = wl.make(name, small=small, **override)
    db = session.upload(w, "cuda", kv_splits=splits)
    assert zb.workspace_size(db.desc) > 0  # the plan really uses scratch
    db.stage()
    db.attend()
    ref = db.out.clone()
    for call in range(2):
        out = torch.full_like(db.out, float("nan"))
        _noalloc(zb, db, out)
        torch.cuda.synchronize()
        assert zb.check_device_error() == 0
        ok, err, scale = tolerance_ok(out, ref.double().cpu().numpy(), w.dtype)
        assert ok, f"call {call}: max|err|={err:.3e}"


def test_noalloc_second_call_with_other_inputs(zs):
    """The scratch keeps the previous call's contents; a following call with
    a different mask still matches the workspace entry point."""
    session, zb = zs
    w = wl.make("decode_small", B=2)
    for mode in (0, 1):
        db = session.upload(w, "cuda", kv_splits=10, mask_mode=mode)
        assert zb.workspace_size(db.desc) > 0
        db.stage()
        db.attend()
        ref = db.out.clone()
        out = torch.zeros_like(db.out)
        _noalloc(zb, db, out)
        torch.cuda.synchronize()
        assert zb.check_device_error() == 0
        ok, err, _ = tolerance_ok(out, ref.double().cpu().numpy(), w.dtype)
        assert ok, f"mode {mode}: max|err|={err:.3e}"


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
