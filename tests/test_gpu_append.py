"""GPU checks of zarya_kv_append (Sec. 5.2 step 7) and of the device error
word. Append must be bit-exact against the oracle; every other cache byte
(including the NaN poison beyond each prefix) must be left alone."""
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
    t = t.detach().cpu()
    if t.dtype == torch.bfloat16:
        return t.view(torch.int16).numpy()
    return t.view(torch.int32).numpy()


def _oracle_stage_commit(oracle, w):
    kc, vc, lens = oracle.kv_append(w.k_new, w.v_new, w.R, w.k_cache, w.v_cache, w.cache_lens,
                                    w.page_table, w.q_row_offsets, page_size=w.page_size,
                                    commit=False)
    assert list(lens) == list(w.cache_lens)
    kc2, vc2, lens2 = oracle.kv_append(w.k_new, w.v_new, w.accept_len, kc, vc, lens,
                                       w.page_table, w.q_row_offsets, page_size=w.page_size,
                                       commit=True)
    return kc, vc, kc2, vc2, lens2


@pytest.mark.parametrize("name,small", [(n, True) for n in wl.ORDER] +
                         [("long_ctx", False), ("serving_mix", False)])
def test_stage_then_commit_bit_exact(zs, oracle_mod, name, small):
    session, zb = zs
    w = wl.make(name, small=small)
    db = session.upload(w, "cuda")
    db.stage()
    torch.cuda.synchronize()
    assert zb.check_device_error() == 0
    kc, vc, kc2, vc2, lens2 = _oracle_stage_commit(oracle_mod, w)
    # staging writes every block row and leaves the lengths alone
    gk, gv = _bits(db.k_cache), _bits(db.v_cache)
    assert np.array_equal(gk, kc.view(gk.dtype))
    assert np.array_equal(gv, vc.view(gv.dtype))
    assert np.array_equal(db.cache_lens.cpu().numpy(), w.cache_lens)
    db.commit()
    torch.cuda.synchronize()
    assert zb.check_device_error() == 0
    gk, gv = _bits(db.k_cache), _bits(db.v_cache)
    assert np.array_equal(gk, kc2.view(gk.dtype))
    assert np.array_equal(gv, vc2.view(gv.dtype))
    assert np.array_equal(db.cache_lens.cpu().numpy(), lens2)


@pytest.mark.parametrize("name,small", [("decode_small", True), ("serving_mix", True),
                                        ("serving_mix", False)])
def test_commit_to_second_array_leaves_lengths_alone(zs, oracle_mod, name, small):
    """zarya_kv_append_commit_to: the same rows as an in-place commit, the
    advanced lengths in new_lens, cache_lens untouched."""
    session, zb = zs
    w = wl.make(name, small=small)
    db = session.upload(w, "cuda")
    db.stage()
    new_lens = torch.full_like(db.cache_lens, -7)
    db.commit(new_lens=new_lens)
    torch.cuda.synchronize()
    assert zb.check_device_error() == 0
    _, _, kc2, vc2, lens2 = _oracle_stage_commit(oracle_mod, w)
    gk, gv = _bits(db.k_cache), _bits(db.v_cache)
    assert np.array_equal(gk, kc2.view(gk.dtype))
    assert np.array_equal(gv, vc2.view(gv.dtype))
    assert np.array_equal(db.cache_lens.cpu().numpy(), w.cache_lens)
    assert np.array_equal(new_lens.cpu().numpy(), lens2)


@pytest.mark.parametrize("name,small", [(n, True) for n in wl.ORDER] +
                         [("long_ctx", False), ("serving_mix", False)])
def test_commit_staged_equals_copy_commit(zs, oracle_mod, name, small):
    """zarya_kv_commit_staged after staging leaves the cache the copy commit
    leaves (the accepted rows are already in place) and the same lengths."""
    session, zb = zs
    w = wl.make(name, small=small)
    db = session.upload(w, "cuda")
    db.stage()
    new_lens = torch.full_like(db.cache_lens, -7)
    db.commit_staged(new_lens=new_lens)
    torch.cuda.synchronize()
    assert zb.check_device_error() == 0
    kc, vc, kc2, vc2, lens2 = _oracle_stage_commit(oracle_mod, w)
    # the oracle's copy commit after staging rewrites rows that are already there
    assert np.array_equal(kc.view(np.uint8), kc2.view(np.uint8))
    gk, gv = _bits(db.k_cache), _bits(db.v_cache)
    assert np.array_equal(gk, kc2.view(gk.dtype))
    assert np.array_equal(gv, vc2.view(gv.dtype))
    assert np.array_equal(new_lens.cpu().numpy(), lens2)
    assert np.array_equal(db.cache_lens.cpu().numpy(), w.cache_lens)
    # in place
    db.commit_staged()
    torch.cuda.synchronize()
    assert zb.check_device_error() == 0
    assert np.array_equal(db.cache_lens.cpu().numpy(), lens2)


def test_commit_staged_checks(zs):
    session, zb = zs
    w = wl.make("decode_small", small=True)
    db = session.upload(w, "cuda")
    new_lens = torch.full_like(db.cache_lens, -7)
    db.accept_len[1] = int(w.R[1]) + 1
    db.commit_staged(new_lens=new_lens)
    assert zb.check_device_error() == 4          # ZARYA_DEVERR_ACCEPT
    got = new_lens.cpu().numpy()
    assert got[1] == -7
    assert all(got[b] == w.cache_lens[b] + w.accept_len[b] for b in range(w.B) if b != 1)
    db = session.upload(w, "cuda")
    db.cache_lens[0] = w.capacity - 2
    db.commit_staged()
    assert zb.check_device_error() == 3          # ZARYA_DEVERR_CAPACITY


def test_commit_to_skips_a_failing_sequence(zs):
    session, zb = zs
    w = wl.make("decode_small", small=True)
    db = session.upload(w, "cuda")
    db.accept_len[1] = int(w.R[1]) + 1
    new_lens = torch.full_like(db.cache_lens, -7)
    db.commit(new_lens=new_lens)
    assert zb.check_device_error() == 4
    got = new_lens.cpu().numpy()
    assert got[1] == -7
    for b in range(w.B):
        if b != 1:
            assert got[b] == w.cache_lens[b] + w.accept_len[b]


def test_commit_of_nothing_is_a_noop(zs):
    session, zb = zs
    w = wl.make("decode_small", small=True)
    db = session.upload(w, "cuda")
    before_k = db.k_cache.clone()
    before_v = db.v_cache.clone()
    db.accept_len.zero_()
    db.commit()
    torch.cuda.synchronize()
    assert zb.check_device_error() == 0
    assert torch.equal(_t(before_k), _t(db.k_cache))
    assert torch.equal(_t(before_v), _t(db.v_cache))
    assert np.array_equal(db.cache_lens.cpu().numpy(), w.cache_lens)


def _t(x):
    return x.view(torch.int16)


def test_accept_beyond_block_sets_error_and_writes_nothing(zs):
    session, zb = zs
    w = wl.make("decode_small", small=True)
    db = session.upload(w, "cuda")
    before = db.k_cache.clone()
    db.accept_len[1] = int(w.R[1]) + 1
    db.accept_len[0] = 0
    db.accept_len[2] = 0
    db.commit()
    assert zb.check_device_error() == 4
    assert torch.equal(_t(before), _t(db.k_cache))
    assert np.array_equal(db.cache_lens.cpu().numpy(), w.cache_lens)


def test_capacity_overflow_sets_error(zs):
    session, zb = zs
    w = wl.make("decode_small", small=True)
    db = session.upload(w, "cuda")
    db.cache_lens[0] = w.capacity - 2
    db.commit()
    assert zb.check_device_error() == 3


def test_bad_page_id_sets_error_without_hanging(zs):
    session, zb = zs
    w = wl.make("serving_mix", small=True)
    db = session.upload(w, "cuda")
    db.stage()
    assert zb.check_device_error() == 0
    db.page_table[2, 0] = w.n_pages + 100
    db.attend()
    assert zb.check_device_error() == 1
    db.page_table[2, 0] = -5
    db.commit()
    code = zb.check_device_error()
    assert code in (0, 1)  # only raised when sequence 2 accepted a token on that page


def test_bad_mask_mode_and_rows_set_errors(zs):
    session, zb = zs
    w = wl.make("decode_small", small=True)
    db = session.upload(w, "cuda")
    db.stage()
    db.mask_mode[1] = 7
    db.attend()
    assert zb.check_device_error() == 6
    db.mask_mode[1] = 1
    db.n_slots[0] = 100  # R_0 no longer matches the row offsets / max_rows
    db.attend()
    assert zb.check_device_error() == 2


def test_fp32_attention_bad_mode_sets_error(zs):
    session, zb = zs
    w = wl.make("tiny_fp32")
    db = session.upload(w, "cuda", mask_mode=0)
    db.stage()
    db.mask_mode[0] = 3
    db.attend()
    assert zb.check_device_error() == 6
