"""Pins for the oracle's ADADELTA (Zeiler 2012, the paper's ref. [21]; the
update rule of Section III.B step 4): torch CPU's Adadelta (an independent
library implementation of the same algorithm), the closed form of the
squared-gradient average under a constant gradient, the zero-gradient
special case, and the direction of the step."""
import numpy as np
import pytest

import oracle

torch = pytest.importorskip("torch")


@pytest.mark.parametrize("rho,eps,lr", [(0.95, 1e-6, 1.0), (0.9, 1e-4, 0.5), (0.0, 1e-8, 1.0)])
def test_matches_torch_adadelta(rho, eps, lr):
    rng = np.random.default_rng(1)
    n = 257
    x0 = rng.standard_normal(n)
    p = torch.tensor(x0, dtype=torch.float64, requires_grad=True)
    opt = torch.optim.Adadelta([p], lr=lr, rho=rho, eps=eps)
    x, a, b = x0.copy(), np.zeros(n), np.zeros(n)
    for _ in range(7):
        g = rng.standard_normal(n) * rng.uniform(0.01, 10.0)
        p.grad = torch.tensor(g, dtype=torch.float64)
        opt.step()
        x, a, b = oracle.adadelta(x, g, a, b, rho, eps, lr)
        np.testing.assert_allclose(x, p.detach().numpy(), rtol=1e-13, atol=1e-15)
    st = opt.state[p]
    np.testing.assert_allclose(a, st["square_avg"].numpy(), rtol=1e-13)
    np.testing.assert_allclose(b, st["acc_delta"].numpy(), rtol=1e-13, atol=1e-300)


def test_constant_gradient_average_has_closed_form():
    """With g fixed, E[g^2]_t = g^2 (1 - rho^t) from a zero start (geometric sum)."""
    rho, eps = 0.95, 1e-6
    g = np.array([0.3, -2.0, 1e-3])
    x, a, b = np.zeros(3), np.zeros(3), np.zeros(3)
    for t in range(1, 40):
        x, a, b = oracle.adadelta(x, g, a, b, rho, eps)
        np.testing.assert_allclose(a, g * g * (1 - rho ** t), rtol=1e-12)
        assert np.all(np.sign(x) == -np.sign(g))          # steps go against the gradient


def test_zero_gradient_only_decays_the_averages():
    rho = 0.9
    x0 = np.array([1.0, -2.0, 3.0])
    a0, b0 = np.array([0.5, 0.1, 2.0]), np.array([0.2, 0.3, 0.4])
    x, a, b = oracle.adadelta(x0, np.zeros(3), a0, b0, rho, 1e-6)
    assert np.array_equal(x, x0)
    np.testing.assert_allclose(a, rho * a0, rtol=1e-15)
    np.testing.assert_allclose(b, rho * b0, rtol=1e-15)


def test_first_step_size_is_bounded_by_the_unit_correction():
    """From a zero state |dx| = sqrt(eps) / sqrt((1-rho) g^2 + eps) |g|, which
    is below sqrt(eps / (1-rho)) for every g (Zeiler's unit-correction)."""
    rho, eps = 0.95, 1e-6
    g = np.logspace(-6, 6, 25)
    x, a, b = oracle.adadelta(np.zeros_like(g), g, np.zeros_like(g), np.zeros_like(g), rho, eps)
    assert np.all(np.abs(x) < np.sqrt(eps / (1 - rho)) * (1 + 1e-12))
    assert np.all(np.diff(np.abs(x)) >= 0)                 # larger gradients, larger (saturating) steps
