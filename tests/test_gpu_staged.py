"""zarya_slot_attn_staged (block K/V staged inside the attention launch) is
bit for bit the same as zarya_kv_append(STAGE) followed by zarya_slot_attn:
same output, same caches, lengths untouched."""
import numpy as np
import pytest
import torch

from paper_2609_19868_gb300 import workloads as wl

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


def _bits(t):
    t = t.detach()
    return t.view(torch.int16) if t.dtype == torch.bfloat16 else t.view(torch.int32)


def _compare(zs, w, mode=None, kv_splits=0):
    session, zb = zs
    a = session.upload(w, "cuda", kv_splits=kv_splits, mask_mode=mode)
    b = session.upload(w, "cuda", kv_splits=kv_splits, mask_mode=mode)
    a.stage()
    a.attend()
    b.stage_and_attend()
    torch.cuda.synchronize()
    assert zb.check_device_error() == 0
    assert not torch.isnan(b.out.float()).any()
    assert torch.equal(_bits(a.out), _bits(b.out))
    assert torch.equal(_bits(a.k_cache), _bits(b.k_cache))
    assert torch.equal(_bits(a.v_cache), _bits(b.v_cache))
    assert np.array_equal(b.cache_lens.cpu().numpy(), w.cache_lens)


@pytest.mark.parametrize("name", wl.ORDER)
def test_staged_equals_stage_then_attend_reduced(zs, name):
    w = wl.make(name, small=True)
    modes = (0, 1) if w.both_modes else (None,)
    for mode in modes:
        _compare(zs, w, mode)


@pytest.mark.parametrize("name", ["decode_small", "ragged_mid", "serving_mix"])
def test_staged_equals_stage_then_attend_full(zs, name):
    _compare(zs, wl.make(name))


@pytest.mark.parametrize("splits", [2, 3, 7, 12])
def test_staged_with_split_keys(zs, splits):
    """Block rows straddling a split boundary are staged by each split that
    reads them (cluster merge up to 3 splits, workspace beyond)."""
    _compare(zs, wl.make("decode_small", B=2), kv_splits=splits)
    _compare(zs, wl.make("long_ctx", small=True), mode=0, kv_splits=splits)


def test_staged_in_a_cuda_graph(zs):
    session, zb = zs
    w = wl.make("decode_small", small=True)
    s = torch.cuda.Stream()
    with torch.cuda.stream(s):
        ref = session.upload(w, "cuda")
        ref.stage(s)
        ref.attend(s)
        db = session.upload(w, "cuda")
        db.stage_and_attend(s)   # warm-up outside the capture
    torch.cuda.synchronize()
    db.out.zero_()
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=s):
        db.stage_and_attend(s)
    g.replay()
    torch.cuda.synchronize()
    assert zb.check_device_error() == 0
    assert torch.equal(_bits(ref.out), _bits(db.out))
