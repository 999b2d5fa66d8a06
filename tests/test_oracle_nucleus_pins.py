"""Pins for the top_p oracle (oracle/nucleus.py) against its definition (Sec.
5.1 step 3, Table 2; nucleus sampling: the smallest set of most probable
tokens reaching top_p, boundary ties kept, the draw restricted to it):
hand-worked sets, ties, temperature, reduction to the plain draw, the law of
the draws, renormalised probabilities."""
import math

import numpy as np
import pytest

from oracle import nucleus as nuc
from oracle import sampling as smp

P4 = np.log([0.5, 0.3, 0.15, 0.05])


@pytest.mark.parametrize("top_p,kept", [(0.4, [0]), (0.7, [0, 1]), (0.85, [0, 1, 2]),
                                        (0.99, [0, 1, 2, 3]), (1.0, [0, 1, 2, 3])])
def test_hand_worked_sets(top_p, kept):
    assert np.flatnonzero(nuc.kept_mask(P4, 1.0, top_p)).tolist() == kept


def test_order_of_the_logits_does_not_matter():
    perm = [2, 0, 3, 1]
    m = nuc.kept_mask(P4[perm], 1.0, 0.7)
    assert np.flatnonzero(m).tolist() == [1, 3]         # the tokens of 0.5 and 0.3


def test_boundary_ties_are_kept_together():
    x = np.log([0.4, 0.2, 0.2, 0.2])
    assert nuc.kept_mask(x, 1.0, 0.5).all()             # 0.4 alone is short: all 0.2s join
    assert np.flatnonzero(nuc.kept_mask(x, 1.0, 0.3)).tolist() == [0]


@pytest.mark.parametrize("T,kept", [(0.5, [0, 1]), (2.0, [0, 1, 2]), (0.0, [0, 1])])
def test_temperature_shapes_the_nucleus(T, kept):
    # T = 0.5: softmax(4, 2, 0) = .867 .117 .016; T = 2: softmax(1, .5, 0) = .507 .307 .186;
    # T = 0 reads as softmax(x) = .665 .245 .090
    assert np.flatnonzero(nuc.kept_mask([2.0, 1.0, 0.0], T, 0.9)).tolist() == kept


def test_top_p_one_is_the_plain_draw():
    rng = np.random.default_rng(3)
    for row in range(60):
        x = rng.normal(scale=2, size=50)
        for T in (0.0, 0.8):
            assert nuc.draw_token(x, T, 1.0, 11, 2, row) == smp.draw_token(x, T, 11, 2, row)


def test_greedy_draw_ignores_top_p():
    rng = np.random.default_rng(4)
    for row in range(30):
        x = rng.normal(size=40)
        assert nuc.draw_token(x, 0.0, 0.05, 1, 0, row) == int(np.argmax(x))


def test_draws_stay_in_the_nucleus_with_its_renormalised_law():
    n = 4000
    draws = np.array([nuc.draw_token(P4, 1.0, 0.7, 9, 0, row) for row in range(n)])
    assert set(draws.tolist()) <= {0, 1}
    frac = (draws == 0).mean()                          # 0.5 / 0.8 = 0.625
    assert abs(frac - 0.625) < 4 * math.sqrt(0.625 * 0.375 / n)


def test_renormalised_probabilities():
    assert nuc.row_probability(P4, 1, 1.0, 0.7) == pytest.approx(0.3 / 0.8, rel=1e-12)
    assert nuc.row_probability(P4, 0, 1.0, 0.7) == pytest.approx(0.5 / 0.8, rel=1e-12)
    assert nuc.row_probability(P4, 2, 1.0, 0.7) == 0.0
    assert nuc.row_probability(P4, 3, 1.0, 1.0) == pytest.approx(0.05, rel=1e-12)


@pytest.mark.parametrize("seed", range(4))
def test_threshold_against_every_candidate_value(seed):
    # x* is the largest logit value v whose tokens at or above it hold at least
    # top_p of the mass: checked by trying every distinct value
    rng = np.random.default_rng(seed)
    x = np.round(rng.normal(scale=2, size=300), 1)      # many ties
    for T in (0.0, 0.7):
        p = nuc._probs(x, T)
        for top_p in (0.1, 0.5, 0.8, 0.97):
            vals = np.unique(x)[::-1]
            ok = [v for v in vals if p[x >= v].sum() >= top_p]
            assert nuc.kept_threshold(x, T, top_p) == max(ok)
