"""GPU parity of zarya_reorder / zarya_restore (Sec. 5.1 steps 2 and 4,
Sec. 5.2 steps 1 and 8) with the oracle (oracle/reorder.py): integer work,
so every output is compared bit for bit."""
import numpy as np
import pytest
import torch

from oracle import reorder as ro
from paper_2609_19868_gb300 import _binding as zb

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA GPU")
    from paper_2609_19868_gb300 import build

    build.build()
    zb.load()
    assert zb.check_device_error() == 0


def _masks(rng, B, L, kind):
    if kind == "bernoulli":
        return (rng.random((B, L)) < rng.random((B, 1))).astype(np.uint8)
    if kind == "spans":       # masked spans (infilling): a few contiguous runs per sequence
        m = np.zeros((B, L), dtype=np.uint8)
        for b in range(B):
            for _ in range(rng.integers(1, 5)):
                s = rng.integers(0, L)
                m[b, s:s + rng.integers(1, L // 3 + 2)] = 1
        return m
    if kind == "tail":        # prefix completion: the generation region after the prompt
        m = np.zeros((B, L), dtype=np.uint8)
        for b in range(B):
            m[b, rng.integers(0, L):] = 1
        return m
    if kind == "all":
        return np.ones((B, L), dtype=np.uint8)
    return np.zeros((B, L), dtype=np.uint8)


def _run(tok, mask, lens, key=None):
    dev = lambda a, dt: torch.as_tensor(np.ascontiguousarray(a)).to(dt).cuda()  # noqa: E731
    t = dev(tok, torch.int32)
    m = dev(mask, torch.uint8)
    ln = dev(lens, torch.int32)
    k = None if key is None else dev(key.view(np.int32), torch.int32)
    perm = torch.full_like(t, -7)
    out = torch.full_like(t, -7)
    nv = torch.full((t.shape[0],), -7, dtype=torch.int32, device="cuda")
    zb.reorder(t, m, ln, perm, out, nv, order_key=k)
    back = torch.full_like(t, -7)
    zb.restore(out, perm, ln, back)
    torch.cuda.synchronize()
    err = zb.check_device_error()
    return perm.cpu().numpy(), out.cpu().numpy(), nv.cpu().numpy(), back.cpu().numpy(), err


@pytest.mark.parametrize("kind", ["bernoulli", "spans", "tail", "all", "none"])
@pytest.mark.parametrize("keyed", [False, True])
@pytest.mark.parametrize("L", [37, 1024, 2500, 4096, 5000])
def test_reorder_restore_match_oracle(kind, keyed, L):
    rng = np.random.default_rng(L * 7 + len(kind) + keyed)
    B = 6
    tok = rng.integers(0, 151936, size=(B, L)).astype(np.int32)
    mask = _masks(rng, B, L, kind)
    lens = rng.integers(0, L + 1, size=B).astype(np.int32)
    lens[0], lens[1] = L, 0
    key = rng.integers(0, 50, size=(B, L)).astype(np.uint32) if keyed else None
    perm, out, nv, back, err = _run(tok, mask, lens, key)
    assert err == 0
    rp, rout, rnv = ro.reorder(tok, mask, lens, order_key=key)
    assert np.array_equal(perm, rp)
    assert np.array_equal(out, rout)
    assert np.array_equal(nv, rnv)
    assert np.array_equal(back, tok)
    assert np.array_equal(back, ro.restore(rout, rp, lens))


def test_full_keys_32_bit():
    rng = np.random.default_rng(3)
    B, L = 3, 700
    tok = rng.integers(0, 1000, size=(B, L)).astype(np.int32)
    mask = (rng.random((B, L)) < 0.6).astype(np.uint8)
    key = rng.integers(0, 2 ** 32, size=(B, L), dtype=np.uint64).astype(np.uint32)
    lens = np.array([L, 500, 1], dtype=np.int32)
    perm, out, nv, back, err = _run(tok, mask, lens, key)
    assert err == 0
    rp, rout, rnv = ro.reorder(tok, mask, lens, order_key=key)
    assert np.array_equal(perm, rp) and np.array_equal(out, rout) and np.array_equal(back, tok)


def test_bad_lengths_and_permutation_set_errors():
    tok = torch.arange(12, dtype=torch.int32, device="cuda").view(2, 6)
    m = torch.zeros((2, 6), dtype=torch.uint8, device="cuda")
    lens = torch.tensor([7, 3], dtype=torch.int32, device="cuda")   # 7 > max_len
    perm = torch.empty_like(tok)
    out = torch.empty_like(tok)
    nv = torch.empty(2, dtype=torch.int32, device="cuda")
    zb.reorder(tok, m, lens, perm, out, nv)
    assert zb.check_device_error() == 2          # ZARYA_DEVERR_ROWS
    assert perm[0].tolist() == [-1] * 6 and out[0].tolist() == list(range(6))
    assert perm[1, :3].tolist() == [0, 1, 2] and nv.tolist() == [0, 3]
    bad = torch.tensor([[0, 1, 9, 3, 4, 5], [2, 1, 0, 3, 4, 5]], dtype=torch.int32,
                       device="cuda")
    back = torch.full_like(tok, -1)
    zb.restore(tok, bad, torch.tensor([6, 3], dtype=torch.int32, device="cuda"), back)
    assert zb.check_device_error() == 8          # ZARYA_DEVERR_PERM
    assert back[1].tolist() == [8, 7, 6, 9, 10, 11]
