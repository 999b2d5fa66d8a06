"""Pins for the reorder / restore oracle (oracle/reorder.py) against the
definition the paper gives (Sec. 5.1 steps 2 and 4, Sec. 5.2 steps 1 and 8:
masked tokens after unmasked ones; the original order restored afterwards).
Hand-worked examples, and properties checked element by element (a
permutation; visible first; order kept within each group; restore inverts
reorder)."""
import numpy as np
import pytest

from oracle import reorder as ro


def test_hand_example_stable():
    mask = np.array([[0, 1, 0, 1, 1, 0]], dtype=np.uint8)
    tok = np.array([[10, 11, 12, 13, 14, 15]], dtype=np.int32)
    perm, out, nvis = ro.reorder(tok, mask, [6])
    assert perm.tolist() == [[0, 2, 5, 1, 3, 4]]
    assert out.tolist() == [[10, 12, 15, 11, 13, 14]]
    assert nvis.tolist() == [3]
    assert ro.restore(out, perm, [6]).tolist() == tok.tolist()


def test_hand_example_with_key():
    # masked positions 1, 3, 4 with keys 7, 2, 7: order 3 (key 2), 1 (7), 4 (7, later)
    mask = np.array([[0, 1, 0, 1, 1, 0]], dtype=np.uint8)
    key = np.array([[9, 7, 0, 2, 7, 1]], dtype=np.uint32)
    tok = np.arange(6, dtype=np.int32)[None] + 20
    perm, out, nvis = ro.reorder(tok, mask, [6], order_key=key)
    assert perm.tolist() == [[0, 2, 5, 3, 1, 4]]
    assert out.tolist() == [[20, 22, 25, 23, 21, 24]]
    assert nvis.tolist() == [3]


def test_ragged_lengths_and_degenerate_sequences():
    tok = np.arange(24, dtype=np.int32).reshape(4, 6)
    mask = np.array([[1, 1, 1, 1, 0, 0],     # all masked within lens 4
                     [0, 0, 0, 0, 0, 0],     # none masked
                     [1, 0, 1, 0, 1, 0],     # length 0
                     [0, 1, 1, 0, 1, 1]], dtype=np.uint8)
    lens = [4, 6, 0, 5]
    perm, out, nvis = ro.reorder(tok, mask, lens)
    assert perm.tolist() == [[0, 1, 2, 3, -1, -1], [0, 1, 2, 3, 4, 5],
                             [-1] * 6, [0, 3, 1, 2, 4, -1]]
    assert nvis.tolist() == [0, 6, 0, 2]
    # positions past a sequence's length keep their tokens
    assert out[0, 4:].tolist() == [4, 5] and out[2].tolist() == tok[2].tolist()
    assert out[3].tolist() == [18, 21, 19, 20, 22, 23]


def _check_properties(mask, key, n, perm):
    p = [int(x) for x in perm[:n]]
    assert sorted(p) == list(range(n))                    # a permutation of 0..n-1
    nvis = sum(1 for i in range(n) if not mask[i])
    vis, msk = p[:nvis], p[nvis:]
    assert all(not mask[i] for i in vis) and all(mask[i] for i in msk)
    assert all(vis[j] < vis[j + 1] for j in range(len(vis) - 1))   # order kept
    for j in range(len(msk) - 1):
        a, b = msk[j], msk[j + 1]
        if key is None:
            assert a < b
        else:
            assert (int(key[a]), a) < (int(key[b]), b)


@pytest.mark.parametrize("seed", range(6))
def test_random_cases_properties_and_inverse(seed):
    rng = np.random.default_rng(seed)
    B, L = 5, 40
    tok = rng.integers(0, 1000, size=(B, L)).astype(np.int32)
    mask = (rng.random((B, L)) < rng.random()).astype(np.uint8)
    key = rng.integers(0, 8, size=(B, L)).astype(np.uint32)    # small range: many ties
    lens = rng.integers(0, L + 1, size=B)
    for k in (None, key):
        perm, out, nvis = ro.reorder(tok, mask, lens, order_key=k)
        for b in range(B):
            n = int(lens[b])
            _check_properties(mask[b], None if k is None else k[b], n, perm[b])
            assert (perm[b, n:] == -1).all()
            assert nvis[b] == int((mask[b, :n] == 0).sum())
            for i in range(n):
                assert out[b, i] == tok[b, perm[b, i]]
        assert np.array_equal(ro.restore(out, perm, lens), tok)
