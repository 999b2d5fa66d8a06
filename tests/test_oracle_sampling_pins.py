"""Pins for the slot-selection / token-acceptance oracle (oracle/sampling.py)
against what the paper and the mathematics fix (Sec. 5.2 steps 3-6).

None of these checks re-types the oracle's formulas. The random-number
generator is pinned to the published Philox4x32-10 known-answer vectors; the
Gumbel transform to the Gumbel law's moments and CDF; Gumbel-max sampling to
the categorical law softmax(x / T) it must reproduce; probabilities to closed
forms; selection and acceptance to hand-worked cases of the rules the paper
states.
"""
import math
import os

import numpy as np
import pytest

from oracle import sampling as smp

HERE = os.path.dirname(os.path.abspath(__file__))


def _kat():
    rows = []
    with open(os.path.join(HERE, "golden", "philox4x32_10_kat.txt")) as f:
        for line in f:
            line = line.strip()
            if not line or line.startswith("#"):
                continue
            w = [int(t, 16) for t in line.split()]
            rows.append((w[0:4], w[4:6], w[6:10]))
    return rows


@pytest.mark.parametrize("ctr,key,expect", _kat())
def test_philox_known_answers(ctr, key, expect):
    out = smp.philox4x32_10([np.uint32(c) for c in ctr], [np.uint32(k) for k in key])
    assert [int(o) for o in out] == expect


def test_philox_words_layout():
    # word v of a row is output word v % 4 of counter (v // 4, row, offset)
    seed, offset, row = 0x0123456789ABCDEF, (7 << 32) | 9, 5
    w = smp.philox_words(seed, offset, row, 11)
    for v in range(11):
        out = smp.philox4x32_10([np.uint32(v // 4), np.uint32(row), np.uint32(9), np.uint32(7)],
                                [np.uint32(0x89ABCDEF), np.uint32(0x01234567)])
        assert int(w[v]) == int(out[v % 4])


def test_uniform_end_points_and_range():
    u = smp.uniform_from_words(np.array([0, 1, 2 ** 32 - 1], dtype=np.uint32))
    assert u.dtype == np.float32
    assert float(u[0]) == 2.0 ** -33          # the smallest draw is 2^-33, never 0
    assert float(u[1]) == 3 * 2.0 ** -33
    assert float(u[2]) == 1.0                 # fl32(2^32 - 1) = 2^32
    w = smp.philox_words(3, 0, 0, 1 << 16)
    u = smp.uniform_from_words(w)
    assert (u > 0).all() and (u <= 1).all()
    assert abs(float(u.mean()) - 0.5) < 5 * math.sqrt(1 / 12 / u.size)


def test_gumbel_moments_and_cdf():
    scipy_stats = pytest.importorskip("scipy.stats")
    g = np.concatenate([smp.gumbel_noise(11, 0, r, 1 << 14) for r in range(64)])
    n = g.size
    euler_gamma = 0.5772156649015329
    assert abs(g.mean() - euler_gamma) < 5 * math.sqrt(math.pi ** 2 / 6 / n)
    assert abs(g.var() - math.pi ** 2 / 6) < 0.03
    ks = scipy_stats.kstest(g, lambda t: np.exp(-np.exp(-t)))
    assert ks.pvalue > 1e-4


def test_gumbel_end_points():
    g = smp.gumbel_from_uniform(np.array([1.0, 2.0 ** -33]))
    assert g[0] == -np.inf                    # u = 1: E = inf
    # u = 2^-33: E = -log1p(-2^-33) ~ 2^-33, g ~ 33 ln 2
    assert abs(g[1] - 33 * math.log(2)) < 1e-6


@pytest.mark.parametrize("T", [0.7, 1.0, 2.5])
def test_gumbel_max_reproduces_softmax_law(T):
    # Gumbel-max: P(argmax_v x_v / T + g_v = i) = softmax(x / T)_i
    scipy_stats = pytest.importorskip("scipy.stats")
    x = np.array([0.0, 1.0, -0.5, 2.0, 0.3, 1.5])
    n = 12000
    counts = np.zeros(x.size)
    for r in range(n):
        counts[smp.draw_token(x, T, 99, 3, r)] += 1
    e = np.exp(x / T)
    p = e / e.sum()
    chi = scipy_stats.chisquare(counts, n * p)
    assert chi.pvalue > 1e-4
    assert np.abs(counts / n - p).max() < 5 * math.sqrt(0.25 / n)


def test_zero_temperature_is_first_argmax():
    x = np.array([0.5, 3.0, -1.0, 3.0, 2.9])
    assert smp.draw_token(x, 0.0, 0, 0, 0) == 1        # tie at 3.0: first index
    assert smp.draw_token(np.full(7, 2.0), 0.0, 0, 0, 0) == 0
    assert smp._draw_token_fast(x, 0.0, 0, 0, 0) == 1


def test_small_temperature_limit_is_argmax():
    # noise of magnitude <= 33 ln 2 cannot overturn a gap of 1 scaled by 1/T = 1e4
    x = np.array([0.0, -3.0, 1.0, 0.5])
    for r in range(50):
        assert smp.draw_token(x, 1e-4, 5, 0, r) == 2


def test_temperature_scales_logits_not_noise():
    # the draw at T on x equals the draw at T = 1 on x / T (same noise)
    rng = np.random.default_rng(0)
    x = rng.standard_normal(200) * 3
    for r in range(40):
        assert smp.draw_token(x, 0.4, 1, 2, r) == smp.draw_token(x / 0.4, 1.0, 1, 2, r)
        assert smp._draw_token_fast(x, 0.4, 1, 2, r) == smp.draw_token(x, 0.4, 1, 2, r)


def test_noise_depends_on_row_seed_and_offset():
    base = smp.gumbel_noise(1, 0, 0, 64)
    assert not np.array_equal(base, smp.gumbel_noise(1, 0, 1, 64))
    assert not np.array_equal(base, smp.gumbel_noise(2, 0, 0, 64))
    assert not np.array_equal(base, smp.gumbel_noise(1, 1, 0, 64))
    assert np.array_equal(base, smp.gumbel_noise(1, 0, 0, 64))


def test_probability_closed_forms():
    V = 1000
    assert abs(smp.row_probability(np.zeros(V), 17, 0.0) - 1 / V) < 1e-15
    a = 9.0
    x = np.zeros(V)
    x[3] = a
    expect = math.exp(a) / (math.exp(a) + V - 1)
    assert abs(smp.row_probability(x, 3, 0.0) - expect) < 1e-14
    # temperature 2: softmax of x / 2
    expect2 = math.exp(a / 2) / (math.exp(a / 2) + V - 1)
    assert abs(smp.row_probability(x, 3, 2.0) - expect2) < 1e-14
    # shift invariance, including logits far outside exp's range
    assert abs(smp.row_probability(x + 5000.0, 3, 0.0) - expect) < 1e-12


@pytest.mark.parametrize("conf,thr,expect", [
    ([0.95, 0.5, 0.91, 0.2], 0.9, [1, 0, 1, 0]),   # above the threshold
    ([0.3, 0.7, 0.7, 0.1], 0.9, [0, 1, 0, 0]),     # none: most confident, first on ties
    ([0.9, 0.9], 0.9, [1, 0]),                     # equal to the threshold is not above it
    ([0.01], 0.9, [1]),                            # one slot always goes on
    ([0.99, 0.98, 0.97], 0.9, [1, 1, 1]),
    ([0.2, 0.4, 0.3], 0.0, [1, 1, 1]),
])
def test_slot_selection_rule(conf, thr, expect):
    assert smp.select_slots(np.array(conf), thr).astype(int).tolist() == expect


@pytest.mark.parametrize("p,n,L,expect_slots,expect_total", [
    ([0.5, 0.6, 0.3, 0.9, 0.8, 0.8, 0.8, 0.8], 2, 4, [2, 4], 2),
    ([0.5, 0.6, 0.7, 0.9, 0.8, 0.1, 0.8, 0.8], 2, 4, [4, 1], 5),
    ([0.5, 0.6, 0.7, 0.9, 0.8, 0.8, 0.8, 0.8], 2, 4, [4, 4], 8),
    ([0.4, 0.9, 0.9], 1, 3, [0], 0),              # equal to the threshold fails
    ([0.1, 0.9, 0.9, 0.9], 2, 2, [0, 2], 0),
])
def test_acceptance_rule(p, n, L, expect_slots, expect_total):
    sa, total = smp.accept_prefix(np.array(p), n, L, 0.4)
    assert sa.tolist() == expect_slots
    assert total == expect_total


def _peaked(V, peaks, rows):
    """rows x V zeros with x[r, tok] = a for each (r, tok, a) in ``peaks``."""
    x = np.zeros((rows, V))
    for r, tok, a in peaks:
        x[r, tok] = a
    return x


def test_draft_select_worked_example():
    # Two sequences. b = 0: 3 slots x 2 tokens (rows 0-5); b = 1: 2 slots x 3
    # tokens (rows 6-11). V = 50. Row r peaks at token (r + 7) with height a_r,
    # so at T = 0 it draws that token with p = e^a / (e^a + 49).
    V = 50
    heights = [6.0, 1.0, 2.0, 1.0, 5.0, 1.0, 3.0, 1.0, 1.0, 4.0, 1.0, 1.0]
    x = _peaked(V, [(r, r + 7, a) for r, a in enumerate(heights)], 12)
    p = [math.exp(a) / (math.exp(a) + V - 1) for a in heights]
    thr = 0.8
    # confidences: b0 slots -> rows 0, 2, 4 = p(6), p(2), p(5) = .892, .131, .752
    #              b1 slots -> rows 6, 9     = p(3), p(4)     = .291, .527
    out = smp.draft_select(x, [3, 2], [2, 3], temperature=0.0, slot_threshold=thr)
    assert out["draft_tokens"].tolist() == [r + 7 for r in range(12)]
    assert np.allclose(out["draft_prob"], p, rtol=1e-14)
    assert np.allclose(out["slot_conf"], [[p[0], p[2], p[4]], [p[6], p[9], 0.0]], rtol=1e-14)
    # b0: only slot 0 above 0.8; b1: none above, most confident is slot 1
    assert out["slot_selected"].tolist() == [[1, 0, 0], [0, 1, 0]]
    assert out["n_selected"].tolist() == [1, 1]
    # verification block packed densely: b0's slot 0 (2 rows), b1's slot 1 (3 rows)
    assert out["verify_row_offsets"].tolist() == [0, 2, 5]
    assert out["verify_src_rows"].tolist() == [0, 1, 9, 10, 11] + [-1] * 7
    assert out["verify_tokens"].tolist() == [7, 8, 16, 17, 18] + [-1] * 7
    # with a threshold of 0.5 b0 takes slots 0 and 2, b1 slot 1
    out = smp.draft_select(x, [3, 2], [2, 3], temperature=0.0, slot_threshold=0.5)
    assert out["slot_selected"].tolist() == [[1, 0, 1], [0, 1, 0]]
    assert out["verify_row_offsets"].tolist() == [0, 4, 7]
    assert out["verify_src_rows"].tolist() == [0, 1, 4, 5, 9, 10, 11] + [-1] * 5
    assert out["verify_tokens"].tolist() == [7, 8, 11, 12, 16, 17, 18] + [-1] * 5


def test_verify_accept_worked_example():
    # b0 verifies 2 slots of 2 tokens (rows 0-3), b1 one slot of 3 tokens
    # (rows 4-6); two trailing rows belong to no block.
    V = 40
    tokens = np.array([3, 9, 4, 1, 30, 31, 32, -1, -1])
    heights = {0: 2.0, 1: 5.0, 2: 6.0, 3: 1.0, 4: 4.0, 5: 4.5, 6: 0.0}
    x = _peaked(V, [(r, int(tokens[r]), a) for r, a in heights.items()], 9)
    out = smp.verify_accept(x, tokens, [2, 1], [2, 3], temperature=0.0, token_threshold=0.4)
    p = {r: math.exp(a) / (math.exp(a) + V - 1) for r, a in heights.items()}
    # p: row0 .159 (fails), row1 .792, row2 .912, row3 .065; row4 .583, row5 .698, row6 .025
    for r in heights:
        assert abs(out["token_prob"][r] - p[r]) < 1e-14
    assert np.isnan(out["token_prob"][[7, 8]]).all()
    assert out["slot_accept"].tolist() == [[0, 1], [2, 0]]
    assert out["accept_len"].tolist() == [0, 2]
    # the same rows placed at explicit offsets with a gap between the sequences
    xg = np.zeros((11, V))
    xg[0:4], xg[6:9] = x[0:4], x[4:7]
    tg = np.full(11, -1)
    tg[0:4], tg[6:9] = tokens[0:4], tokens[4:7]
    out2 = smp.verify_accept(xg, tg, [2, 1], [2, 3], temperature=0.0, token_threshold=0.4,
                             row_offsets=[0, 6, 9])
    assert out2["accept_len"].tolist() == [0, 2]
    assert out2["slot_accept"].tolist() == [[0, 1], [2, 0]]


def test_verify_of_own_draft_reproduces_draft_probability():
    rng = np.random.default_rng(3)
    x = rng.standard_normal((8, 300)) * 2
    d = smp.draft_select(x, [2], [4], temperature=0.8, slot_threshold=0.0, seed=4, offset=1)
    assert d["verify_src_rows"].tolist() == list(range(8))
    v = smp.verify_accept(x, d["verify_tokens"], [2], [4], temperature=0.8, token_threshold=0.0)
    assert np.allclose(v["token_prob"], d["draft_prob"], rtol=1e-13)
    assert v["accept_len"].tolist() == [8]


def test_sampled_rows_match_full_run():
    rng = np.random.default_rng(5)
    x = rng.standard_normal((12, 257)) * 2
    full = smp.draft_select(x, [2, 1], [4, 4], temperature=1.3, slot_threshold=0.5, seed=9)
    part = smp.draft_select(x, [2, 1], [4, 4], temperature=1.3, slot_threshold=0.5, seed=9,
                            rows=[1, 10], fast=True)
    for r in (1, 10):
        assert part["draft_tokens"][r] == full["draft_tokens"][r]
        assert part["draft_prob"][r] == full["draft_prob"][r]
