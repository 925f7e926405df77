"""Pins of the oracle's drafter entropy and entropy-adaptive lambda (App. F)
against closed forms, a library routine and invariants."""

import math

import numpy as np
import pytest

from oracle import presto_oracle as O


def test_uniform_row_has_entropy_log_v():
    for V in (1, 2, 7, 1000, 151936):
        x = np.full((1, V), 3.25)
        assert abs(O.drafter_entropy(x)[0] - math.log(V)) <= 1e-12 * max(1.0, math.log(V))


def test_single_finite_entry_has_zero_entropy():
    x = np.full((2, 50), -np.inf)
    x[0, 17] = 4.0
    x[1, 0] = -300.0
    np.testing.assert_array_equal(O.drafter_entropy(x), [0.0, 0.0])


def test_two_point_distribution_is_binary_entropy():
    rng = np.random.default_rng(1)
    for _ in range(50):
        a, b = rng.normal(0, 4, 2)
        x = np.full((1, 9), -np.inf)
        x[0, 2], x[0, 6] = a, b
        p = 1.0 / (1.0 + math.exp(b - a))
        want = -(p * math.log(p) + (1 - p) * math.log(1 - p))
        assert abs(O.drafter_entropy(x)[0] - want) <= 1e-12


def test_entropy_matches_scipy_from_probabilities():
    stats = pytest.importorskip("scipy.stats")
    rng = np.random.default_rng(2)
    x = rng.normal(0, 3, size=(6, 4099))
    x[1, ::3] = -np.inf
    ex = np.exp(x - x.max(axis=1, keepdims=True))
    p = ex / ex.sum(axis=1, keepdims=True)
    want = np.array([stats.entropy(row) for row in p])
    np.testing.assert_allclose(O.drafter_entropy(x), want, rtol=1e-10, atol=1e-12)


def test_entropy_invariances_and_bounds():
    rng = np.random.default_rng(3)
    x = rng.normal(0, 2, size=(4, 777))
    H = O.drafter_entropy(x)
    np.testing.assert_allclose(O.drafter_entropy(x + 123.5), H, rtol=1e-12)
    np.testing.assert_allclose(O.drafter_entropy(x[:, rng.permutation(777)]), H, rtol=1e-12)
    assert np.all(H > 0) and np.all(H < math.log(777))
    # sharpening lowers the entropy towards 0, flattening raises it towards log V
    assert np.all(O.drafter_entropy(x * 50) < H) and np.all(O.drafter_entropy(x * 50) < 0.5)
    assert np.all(O.drafter_entropy(x * 1e-3) > H)
    np.testing.assert_allclose(O.drafter_entropy(x * 1e-6), math.log(777), rtol=1e-8)


def test_adaptive_lambda_closed_forms():
    beta, C = 0.6, 1.5
    lam = O.entropy_adaptive_lambda(np.array([0.0, C, 3 * C, 1e12]), beta, C)
    np.testing.assert_allclose(lam, [0.0, beta / 2, 0.75 * beta, beta], rtol=1e-10, atol=0)
    H = np.linspace(0, 12, 200)
    lam = O.entropy_adaptive_lambda(H, beta, C)
    assert np.all(np.diff(lam) > 0) and np.all(lam < beta)
    with pytest.raises(ValueError):
        O.entropy_adaptive_lambda(H, 0.0, C)
    with pytest.raises(ValueError):
        O.entropy_adaptive_lambda(H, beta, 0.0)
