"""Full-size parity in the benchmark's launch configuration, densely.

The benchmark's step runs zarya_slot_attn_staged (the block's K/V staged and
attended in one launch) with the automatic split plan. These tests run that
same call at the full sizes of the configurations and compare against the
fp64 oracle on the same bytes:
  * decode_small: every output, in all three mask modes (the whole step's
    oracle takes about a tenth of a second);
  * ragged_mid, long_ctx (both modes), serving_mix: every (row, head) output
    of the sequence with the longest key range and of the one with the
    shortest, plus 192 sampled (sequence, head, row) outputs.
The staged block rows in the cache are checked bit for bit as well.
"""
import numpy as np
import pytest
import torch

from paper_2609_19868_gb300 import workloads as wl
from _helpers import gather_rows, oracle_full, oracle_rows, oracle_staged, sample_rows, tolerance_ok

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


def _staged(zs, w, mode=None):
    session, zb = zs
    db = session.upload(w, "cuda", mask_mode=mode)
    db.stage_and_attend()
    torch.cuda.synchronize()
    assert zb.check_device_error() == 0
    return db


def _bytes(x):
    """A cache as raw bytes (bit-exact comparison, NaN payloads included)."""
    t = x.detach().cpu() if isinstance(x, torch.Tensor) else torch.from_numpy(np.ascontiguousarray(x))
    return t.contiguous().view(torch.uint8)


def _check_staged_rows(db, kc, vc):
    """The cache after the staged call equals the oracle's staged cache."""
    assert torch.equal(_bytes(db.k_cache), _bytes(kc))
    assert torch.equal(_bytes(db.v_cache), _bytes(vc))


@pytest.mark.parametrize("mode", [0, 1, 2])
def test_decode_small_every_output(zs, oracle_mod, mode):
    w = wl.make("decode_small").with_mode(mode)
    db = _staged(zs, w)
    kc, vc = oracle_staged(oracle_mod, w)
    _check_staged_rows(db, kc, vc)
    ok, err, scale = tolerance_ok(db.out, oracle_full(oracle_mod, w, kc, vc), w.dtype)
    assert ok, f"mode {mode}: max|err|={err:.3e} max|ref|={scale:.3f}"


def _extreme_sequences(w):
    span = w.cache_lens.astype(np.int64) + w.R
    return sorted({int(np.argmax(span)), int(np.argmin(span))})


@pytest.mark.parametrize("name,mode", [("ragged_mid", None), ("long_ctx", 0), ("long_ctx", 1),
                                       ("serving_mix", None)])
def test_longest_and_shortest_sequence_every_output(zs, oracle_mod, name, mode):
    w = wl.make(name)
    if mode is not None:
        w = w.with_mode(mode)
    db = _staged(zs, w)
    out = db.out.cpu()
    assert not torch.isnan(out).any()
    if name != "long_ctx":
        # long_ctx's caches are 1.1 GB each: compare them only where staged
        kc, vc = oracle_staged(oracle_mod, w)
        _check_staged_rows(db, kc, vc)
    else:
        kc, vc = oracle_staged(oracle_mod, w)
        for b in range(w.B):
            lo, hi = int(w.cache_lens[b]), int(w.cache_lens[b] + w.R[b])
            assert torch.equal(_bytes(db.k_cache[b, lo:hi]), _bytes(kc[b, lo:hi]))
            assert torch.equal(_bytes(db.v_cache[b, lo:hi]), _bytes(vc[b, lo:hi]))
    del db
    torch.cuda.empty_cache()
    seqs = _extreme_sequences(w)
    if name == "long_ctx":
        seqs = seqs[-1:]   # every sequence has the same length
    sel = [(b, h, r) for b in seqs for h in range(w.Hq) for r in range(int(w.R[b]))]
    sel += [tuple(x) for x in sample_rows(w, 192, seed=5)]
    sel = np.asarray(sel, dtype=np.int64)
    ref = oracle_rows(oracle_mod, w, kc, vc, sel)
    ok, err, scale = tolerance_ok(gather_rows(out, w, sel), ref, w.dtype)
    assert ok, f"{name} mode={mode} sequences {seqs}: max|err|={err:.3e} max|ref|={scale:.3f}"
