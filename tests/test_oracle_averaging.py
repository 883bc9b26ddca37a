"""Pins of the oracle's eq. 3 (Section III.B step 5, alpha = 1):
V(t) = V_alpha(t) - beta V(t-1), V_alpha the mean of the parallel models'
parameters, V(t-1) the parameters the epoch started from."""
import numpy as np
import pytest

import oracle


def test_worked_example():
    # three models, worked by hand: mean = [4, 5, 6]; beta V(t-1) = [1, -2, 0.05]
    v = oracle.average_models([[1, 2, 3], [4, 5, 6], [7, 8, 9]], [10, -20, 0.5], beta=0.1)
    np.testing.assert_allclose(v, [3.0, 7.0, 5.95], rtol=0, atol=1e-15)


def test_beta_zero_is_the_plain_mean():
    rng = np.random.default_rng(0)
    m = rng.standard_normal((5, 37))
    np.testing.assert_allclose(oracle.average_models(m, rng.standard_normal(37), beta=0.0),
                               np.mean(m, axis=0), rtol=1e-15, atol=1e-15)


def test_single_model_and_paper_constant():
    # one model: V = V_1 - beta V(t-1); with the paper's beta = 1e-6 and a model
    # that did not move, every weight decays by one part in a million
    rng = np.random.default_rng(1)
    prev = rng.standard_normal(50)
    v1 = rng.standard_normal(50)
    np.testing.assert_allclose(oracle.average_models([v1], prev, beta=0.25), v1 - 0.25 * prev, atol=1e-15)
    np.testing.assert_allclose(oracle.average_models([prev, prev], prev, beta=1e-6), prev * (1 - 1e-6),
                               rtol=1e-15, atol=0)


def test_model_order_and_linearity():
    rng = np.random.default_rng(2)
    m = rng.standard_normal((4, 20))
    prev = rng.standard_normal(20)
    a = oracle.average_models(m, prev, beta=0.3)
    b = oracle.average_models(m[[2, 0, 3, 1]], prev, beta=0.3)
    np.testing.assert_allclose(a, b, rtol=1e-15, atol=1e-15)
    # affine in the models: doubling every model doubles the mean part only
    c = oracle.average_models(2 * m, prev, beta=0.3)
    np.testing.assert_allclose(c - a, np.mean(m, axis=0), atol=1e-14)


def test_rejects_mismatched_lengths():
    with pytest.raises(ValueError):
        oracle.average_models([[1.0, 2.0]], [1.0, 2.0, 3.0])
