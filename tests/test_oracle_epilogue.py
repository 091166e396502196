"""Pins for the oracle's epilogue references: the two activations against library
special functions and their exact identities, the bf16 rounding against torch, and the
error bounds against an fp32 model of the computation they bound. CPU only."""
import numpy as np
import pytest
import scipy.special as sp
import torch

import oracle


X = np.concatenate([np.linspace(-12, 12, 4801), [-40.0, -20.0, 0.0, 20.0, 40.0]])


def test_gelu_tanh_identities_and_limits():
    g = oracle.gelu_tanh(X)
    # odd part: gelu(x) - gelu(-x) = x exactly in real arithmetic
    assert np.allclose(g - oracle.gelu_tanh(-X), X, rtol=0, atol=1e-13)
    assert oracle.gelu_tanh(0.0) == 0.0
    assert np.allclose(oracle.gelu_tanh([20.0, 40.0]), [20.0, 40.0], rtol=1e-15)
    assert np.all(np.abs(oracle.gelu_tanh([-20.0, -40.0])) < 1e-30)
    # slope 1/2 at 0 (central difference)
    h = 1e-6
    assert abs((oracle.gelu_tanh(h) - oracle.gelu_tanh(-h)) / (2 * h) - 0.5) < 1e-9


def test_gelu_tanh_is_close_to_exact_gelu():
    """The tanh form approximates x * Phi(x) (scipy's erf) to a few 1e-4."""
    exact = X * 0.5 * (1.0 + sp.erf(X / np.sqrt(2.0)))
    err = np.abs(oracle.gelu_tanh(X) - exact)
    assert err.max() < 5e-4 and err.max() > 1e-5   # close, but a different function


def test_silu_against_expit_and_identity():
    s = oracle.silu(X)
    assert np.allclose(s, X * sp.expit(X), rtol=1e-14, atol=1e-300)
    # silu(x) + silu(-x) = x tanh(x / 2)
    assert np.allclose(s + oracle.silu(-X), X * np.tanh(X / 2), rtol=1e-12, atol=1e-13)
    assert oracle.silu(0.0) == 0.0


def test_activation_slopes_below_the_bound_constant():
    """The gated bounds use |act'| <= 1.2 for both activations."""
    x = np.linspace(-30, 30, 600001)
    for f in (oracle.gelu_tanh, oracle.silu):
        d = np.gradient(f(x), x)
        assert np.abs(d).max() < 1.2


def test_bf16_round_matches_torch():
    rng = np.random.default_rng(1)
    v = (rng.standard_normal(10000) * np.exp2(rng.integers(-30, 30, 10000))).astype(np.float32)
    t = torch.from_numpy(v).to(torch.bfloat16).to(torch.float64).numpy()
    assert np.array_equal(oracle.bf16_round(v), t)


@pytest.mark.parametrize("kind", [oracle.EPI_BF16, oracle.EPI_ADD, oracle.EPI_GEGLU, oracle.EPI_SWIGLU])
def test_epilogue_bounds_cover_an_fp32_model(kind):
    """Perturb the exact Y by up to its bound (the matmul's error), evaluate the epilogue
    the way the GPU does (fp32 arithmetic, one bf16 or fp32 rounding at the end) and check
    that the result lies within the epilogue's bound of the fp64 reference."""
    rng = np.random.default_rng(7 + kind)
    M, N = 64, 512
    Y = rng.standard_normal((M, N)) * np.exp2(rng.integers(-6, 6, (M, N)))
    B = 1e-3 * np.abs(Y) * rng.uniform(1, 20, (M, N)) + 1e-6
    acc = (Y + B * rng.uniform(-1, 1, (M, N))).astype(np.float32)
    R = rng.standard_normal((M, N)).astype(np.float32) * 4
    ref, bound = oracle.epilogue_reference(kind, Y, B, R)
    if kind == oracle.EPI_BF16:
        out = oracle.bf16_round(acc)
    elif kind == oracle.EPI_ADD:
        out = (R + acc).astype(np.float64)
    else:
        g, u = acc[:, 0::2], acc[:, 1::2]
        if kind == oracle.EPI_GEGLU:
            c = np.float32(np.sqrt(2.0 / np.pi))
            act = np.float32(0.5) * g * (np.float32(1) + np.tanh(c * (g + np.float32(0.044715) * g * g * g)))
        else:
            with np.errstate(over="ignore"):     # exp(-g) = inf for g << 0 gives act = -0
                act = g / (np.float32(1) + np.exp(-g))
        out = oracle.bf16_round((act * u).astype(np.float32))
    assert np.all(np.abs(out - ref) <= bound)
