"""Pins for the repetition-penalty oracle (oracle/penalty.py) against its
definition (Sec. 5.1 step 3, Table 2; the penalised sampling of CTRL in its
generate() form: negative logits multiplied, others divided, once per
distinct history token): hand-worked values, the bf16 rounding rule, special
cases, and a brute-force loop over every element."""
import numpy as np
import pytest

from oracle import penalty as pen


def test_hand_example():
    x = np.array([[2.0, -2.0, 0.0, 3.0, -0.5]], dtype=np.float32)
    out, bad = pen.repetition_penalty(x, [0, 1], [0, 5], [0, 1, 1, 4, 9], 2.0)
    assert out.tolist() == [[1.0, -4.0, 0.0, 3.0, -1.0]]
    assert bad                                   # token 9 is outside the vocabulary
    assert x.tolist() == [[2.0, -2.0, 0.0, 3.0, -0.5]]   # the input is left alone


def test_repeated_tokens_count_once():
    x = np.array([[8.0, -8.0]], dtype=np.float32)
    out, bad = pen.repetition_penalty(x, [0, 1], [0, 6], [0, 0, 0, 1, 1, 1], 2.0)
    assert out.tolist() == [[4.0, -16.0]] and not bad


def test_penalty_one_changes_nothing():
    rng = np.random.default_rng(0)
    x = rng.normal(size=(3, 50)).astype(np.float32)
    out, _ = pen.repetition_penalty(x, [0, 3], [0, 20], rng.integers(0, 50, 20), 1.0)
    assert np.array_equal(out, x)


def test_zeros_and_infinities():
    x = np.array([[0.0, -0.0, np.inf, -np.inf]], dtype=np.float32)
    out, _ = pen.repetition_penalty(x, [0, 1], [0, 4], [0, 1, 2, 3], 3.0)
    assert out[0, 0] == 0.0 and not np.signbit(out[0, 0])
    assert out[0, 1] == 0.0 and np.signbit(out[0, 1])     # -0 is not negative: divided
    assert out[0, 2] == np.inf and out[0, 3] == -np.inf


def test_rows_follow_their_own_sequence_and_unowned_rows_stay():
    x = np.ones((5, 4), dtype=np.float32)
    # sequence 0: rows 0-1, history {0}; sequence 1: rows 2-3, history {3}; row 4: none
    out, _ = pen.repetition_penalty(x, [0, 2, 4], [0, 1, 2], [0, 3], 4.0)
    assert out[:2].tolist() == [[0.25, 1, 1, 1]] * 2
    assert out[2:4].tolist() == [[1, 1, 1, 0.25]] * 2
    assert out[4].tolist() == [1, 1, 1, 1]


def test_history_order_does_not_matter():
    rng = np.random.default_rng(1)
    x = rng.normal(scale=3, size=(4, 97)).astype(np.float32)
    h = rng.integers(0, 97, 60)
    a, _ = pen.repetition_penalty(x, [0, 4], [0, 60], h, 1.7)
    b, _ = pen.repetition_penalty(x, [0, 4], [0, 60], h[::-1], 1.7)
    assert np.array_equal(a, b)


@pytest.mark.parametrize("value,expect", [
    (1 + 2.0 ** -8, 1.0),                          # halfway: to the even neighbour (1.0)
    (1 + 3 * 2.0 ** -8, 1 + 2.0 ** -6),            # halfway: to the even neighbour above
    (1 + 2.0 ** -8 + 2.0 ** -20, 1 + 2.0 ** -7),   # above halfway: up
    (1 + 2.0 ** -9, 1.0),                          # below halfway: down
    (-(1 + 2.0 ** -8 + 2.0 ** -20), -(1 + 2.0 ** -7)),
    (3.0, 3.0),                                    # already a bf16 value
])
def test_bf16_rounding_is_to_nearest_even(value, expect):
    assert float(pen.bf16_round(np.float32(value))) == expect


def test_bf16_one_third():
    # 1 / 3 in float32 is 0x3EAAAAAB; its nearest bf16 is 0x3EAB = 0.333984375
    out, _ = pen.repetition_penalty(np.array([[1.0]], np.float32), [0, 1], [0, 1], [0], 3.0,
                                    dtype="bf16")
    assert float(out[0, 0]) == 0.333984375


@pytest.mark.parametrize("dtype", ["fp32", "bf16"])
def test_brute_force_definition(dtype):
    rng = np.random.default_rng(2)
    B, V = 3, 40
    row_offsets = [0, 2, 2, 5]                     # sequence 1 has no rows
    x = rng.normal(scale=2, size=(6, V)).astype(np.float32)
    if dtype == "bf16":
        x = pen.bf16_round(x)
    hist = rng.integers(-2, V + 2, 30)             # some tokens outside the vocabulary
    hist_offsets = [0, 10, 20, 30]
    out, bad = pen.repetition_penalty(x, row_offsets, hist_offsets, hist, 1.3, dtype=dtype)
    p = np.float32(1.3)
    for b in range(B):
        seen = set(int(t) for t in hist[hist_offsets[b]:hist_offsets[b + 1]] if 0 <= t < V)
        for g in range(row_offsets[b], row_offsets[b + 1]):
            for v in range(V):
                xv = x[g, v]
                if v in seen:
                    want = np.float32(xv * p) if xv < 0 else np.float32(xv / p)
                    if dtype == "bf16":
                        want = np.float32(pen.bf16_round(want))
                else:
                    want = xv
                assert out[g, v] == want, (b, g, v)
    assert np.array_equal(out[5], x[5])            # row 5 belongs to no sequence
    assert bad == bool(((hist < 0) | (hist >= V)).any())


def test_bf16_rounding_agrees_with_torch_conversion():
    torch = pytest.importorskip("torch")
    rng = np.random.default_rng(7)
    x = np.concatenate([rng.normal(scale=s, size=4000) for s in (1e-3, 1.0, 1e3, 1e30)])
    x = x.astype(np.float32)
    ours = pen.bf16_round(x)
    lib = torch.from_numpy(x).to(torch.bfloat16).float().numpy()
    assert np.array_equal(ours.view(np.uint32), lib.view(np.uint32))
