"""Pins for the Mode A oracle (oracle/mode_a.py) against the rule the paper
states (Sec. 5.1 step 1: alpha_0 the expected diffusion fraction; T > 0
exactly T diffusion steps then sequential reveals; T = 0 steps of a quarter)
and the mathematics of the binomial draws."""
import math

import numpy as np
import pytest

from oracle import mode_a as ma


@pytest.mark.parametrize("n,expect", [(10, [4, 4, 2]), (4, [4]), (1, [1]), (9, [4, 4, 1]),
                                      (0, [])])
def test_zero_T_quarter_steps(n, expect):
    assert ma.budget_one(n, 0, 0.25, 1, 0, 0) == expect


@pytest.mark.parametrize("seed", range(5))
def test_plan_structure(seed):
    rng = np.random.default_rng(seed)
    for _ in range(30):
        n = int(rng.integers(0, 300))
        T = int(rng.integers(1, 40))
        a0 = float(rng.random())
        seq = int(rng.integers(0, 64))
        c = ma.budget_one(n, T, a0, seed, 7, seq)
        if n == 0:
            assert c == []
            continue
        assert sum(c) == n                                   # every masked token revealed once
        n_diff = ma.binomial(seed, 7, seq, 0, n, a0)
        assert sum(c[:T]) == n_diff and len(c) == T + (n - n_diff)
        assert all(k == 1 for k in c[T:])                    # sequential tail
        assert all(k >= 0 for k in c[:T])


def test_alpha_extremes():
    assert ma.budget_one(50, 5, 0.0, 3, 0, 0) == [0] * 5 + [1] * 50
    c = ma.budget_one(50, 5, 1.0, 3, 0, 0)
    assert sum(c[:5]) == 50 and len(c) == 5


def test_last_diffusion_step_takes_the_rest():
    # p = 1/(T - s) = 1 at s = T - 1: every remaining trial succeeds (u <= 1,
    # and u = 1 happens only for the top 128 of 2^32 draws)
    for seq in range(40):
        c = ma.budget_one(200, 3, 0.6, 11, 0, seq)
        n_diff = ma.binomial(11, 0, seq, 0, 200, 0.6)
        assert sum(c[:3]) == n_diff


def test_diffusion_total_is_binomial():
    scipy_stats = pytest.importorskip("scipy.stats")
    n, a0, m = 40, 0.3, 3000
    draws = np.array([ma.binomial(5, 0, s, 0, n, a0) for s in range(m)])
    assert abs(draws.mean() - n * a0) < 5 * math.sqrt(n * a0 * (1 - a0) / m)
    assert abs(draws.var() - n * a0 * (1 - a0)) < 0.1 * n * a0 * (1 - a0)
    obs = np.bincount(draws, minlength=n + 1)
    exp = scipy_stats.binom.pmf(np.arange(n + 1), n, a0) * m
    keep = exp > 5
    other = m - exp[keep].sum()
    chi = scipy_stats.chisquare(np.append(obs[keep], m - obs[keep].sum()),
                                np.append(exp[keep], other))
    assert chi.pvalue > 1e-4


def test_first_diffusion_step_is_binomial_one_over_T():
    # given r remaining, step 0 of T reveals Binomial(r, 1/T): mean r / T
    T, m = 4, 2000
    ks = []
    for s in range(m):
        r = ma.binomial(9, 0, s, 0, 100, 0.5)
        ks.append((r, ma.budget_one(100, T, 0.5, 9, 0, s)[0]))
    r = np.array([a for a, _ in ks], dtype=float)
    k = np.array([b for _, b in ks], dtype=float)
    assert abs(k.sum() / r.sum() - 1 / T) < 0.01


def test_draws_differ_by_sequence_and_draw_index():
    a = ma.uniforms(1, 0, 0, 0, 64)
    assert not np.array_equal(a, ma.uniforms(1, 0, 1, 0, 64))
    assert not np.array_equal(a, ma.uniforms(1, 0, 0, 1, 64))
    assert not np.array_equal(a, ma.uniforms(1, 1, 0, 0, 64))
    assert np.array_equal(a, ma.uniforms(1, 0, 0, 0, 64))
    assert (a > 0).all() and (a <= 1).all()


def test_batch_plan_padding():
    counts, n_steps = ma.budget([10, 0, 5], 0, 0.25)
    assert counts.tolist() == [[4, 4, 2], [0, 0, 0], [4, 1, 0]]
    assert n_steps.tolist() == [3, 0, 2]


def test_bernoulli_trial_is_strict_at_equality():
    # [u < p]: a trial whose uniform equals p exactly fails
    u = ma.uniforms(4, 0, 0, 0, 8)
    p = float(u[0])
    assert ma.binomial(4, 0, 0, 0, 1, p) == 0
    above = float(np.nextafter(np.float32(p), np.float32(2)))
    assert ma.binomial(4, 0, 0, 0, 1, above) == 1
    # and over several trials the count is the number of uniforms strictly below p
    p = float(np.sort(u)[4])
    assert ma.binomial(4, 0, 0, 0, 8, p) == 4
