"""GPU parity of Mode A's mask-budget planning (zarya_mode_a_budget, Sec.
5.1 step 1; integer plans, bit-exact) and of the per-step row sampling
(zarya_sample_rows, Sec. 5.1 step 3) against the oracle (oracle/mode_a.py)."""
import numpy as np
import pytest
import torch

from oracle import mode_a as ma
from oracle import sampling as smp
from paper_2609_19868_gb300 import _binding as zb
from paper_2609_19868_gb300 import workloads as wl

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA GPU")
    from paper_2609_19868_gb300 import build

    build.build()
    zb.load()
    assert zb.check_device_error() == 0


def _budget(n_masked, T, a0, seed, offset, max_steps):
    nm = torch.as_tensor(np.asarray(n_masked, dtype=np.int32)).cuda()
    counts = torch.full((nm.shape[0], max_steps), -7, dtype=torch.int32, device="cuda")
    steps = torch.full((nm.shape[0],), -7, dtype=torch.int32, device="cuda")
    zb.mode_a_budget(nm, T, a0, seed, offset, counts, steps)
    torch.cuda.synchronize()
    return counts.cpu().numpy(), steps.cpu().numpy(), zb.check_device_error()


@pytest.mark.parametrize("T", [0, 1, 3, 16, 64])
@pytest.mark.parametrize("a0", [0.0, 0.25, 0.7, 1.0])
def test_budget_matches_oracle(T, a0):
    rng = np.random.default_rng(T * 10 + int(a0 * 10))
    n = rng.integers(0, 700, size=17).astype(np.int32)
    n[0], n[1] = 0, 1
    max_steps = T + 700
    counts, steps, err = _budget(n, T, a0, 12345, 6, max_steps)
    assert err == 0
    rc, rs = ma.budget(n, T, a0, 12345, 6, max_steps=max_steps)
    assert np.array_equal(steps, rs)
    assert np.array_equal(counts, rc)


def test_budget_seed_and_offset_change_the_plan():
    n = np.full(8, 300, dtype=np.int32)
    a, _, _ = _budget(n, 8, 0.5, 1, 0, 400)
    b, _, _ = _budget(n, 8, 0.5, 2, 0, 400)
    c, _, _ = _budget(n, 8, 0.5, 1, 1, 400)
    assert not np.array_equal(a, b) and not np.array_equal(a, c)
    assert np.array_equal(a, ma.budget(n, 8, 0.5, 1, 0, max_steps=400)[0])


def test_budget_errors():
    counts, steps, err = _budget([5, -1, 9], 0, 0.25, 0, 0, 8)
    assert err == 2                              # ZARYA_DEVERR_ROWS (negative count)
    assert steps.tolist() == [2, 0, 3]
    assert counts[1].tolist() == [0] * 8
    counts, steps, err = _budget([40, 4], 0, 0.25, 0, 0, 5)   # 10 steps > max_steps 5
    assert err == 2
    assert steps.tolist() == [0, 1] and counts[0].tolist() == [0] * 5


@pytest.mark.parametrize("dtype", ["fp32", "bf16"])
@pytest.mark.parametrize("T", [0.0, 1.0])
def test_sample_rows_matches_oracle(dtype, T):
    w = wl.make_sampling("select_tiny", dtype=dtype)
    V = w.V
    epv = 8 if dtype == "bf16" else 4
    stride = (V + epv - 1) // epv * epv
    rows = w.rows
    buf = torch.zeros((rows, stride), dtype=w.draft_logits.dtype, device="cuda")
    buf[:, :V] = w.draft_logits.cuda()
    logits = buf[:, :V]
    # two "sequences" of revealed rows: 5 and the rest
    ro = torch.tensor([0, 5, rows], dtype=torch.int32, device="cuda")
    d = zb.make_sample_desc(batch=2, vocab=V, dtype=zb.BF16 if dtype == "bf16" else zb.FP32,
                            max_slots=1, total_rows=rows, row_stride=stride, temperature=T,
                            slot_threshold=0.9, token_threshold=0.4, seed=77, offset=5,
                            row_offsets=ro)
    tok = torch.full((rows,), -1, dtype=torch.int32, device="cuda")
    prob = torch.full((rows,), float("nan"), device="cuda")
    zb.sample_rows(logits, tok, prob, d)
    torch.cuda.synchronize()
    assert zb.check_device_error() == 0
    x = w.draft_logits.float().numpy()
    rt, rp = ma.sample_rows(x, T, 77, 5)
    tok, prob = tok.cpu().numpy(), prob.cpu().numpy()
    for g in range(rows):
        if tok[g] != rt[g]:
            assert T > 0
            z = x[g].astype(np.float64) / T + smp.gumbel_noise(77, 5, g, V)
            assert z[rt[g]] - z[tok[g]] <= 4e-5 + 2e-6 * abs(z[rt[g]])
        assert abs(prob[g] - smp.row_probability(x[g], int(tok[g]), T)) <= 1e-6 + 1e-4 * prob[g]
