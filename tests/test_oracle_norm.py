"""Pins of the oracle's RMSNorm (the step before the gate): against fp64,
exact closed-form cases, and exact invariances of the definition
y = x / sqrt(mean(x^2) + eps) * gamma."""
import numpy as np
import pytest

import oracle


def f64_rmsnorm(x, g, eps):
    x = x.astype(np.float64)
    return x / np.sqrt((x * x).mean(axis=1, keepdims=True) + eps) * g.astype(np.float64)


@pytest.mark.parametrize("H", [256, 4096, 7168])
def test_within_fp32_bound_of_fp64(H):
    rng = np.random.default_rng(H)
    x = (rng.standard_normal((16, H)) * rng.uniform(0.01, 100, (16, 1))).astype(np.float32)
    g = rng.uniform(-2, 2, H).astype(np.float32)
    y = oracle.rmsnorm(x, g, 1e-6)
    ref = f64_rmsnorm(x, g, 1e-6)
    # sum of squares: H/32 + 5 fp32 roundings in sequence; then ~6 more
    bound = (H / 32 + 12) * 2.0 ** -24
    assert np.all(np.abs(y - ref) <= bound * np.abs(ref) + 1e-30)


def test_constant_rows_give_gamma_exactly():
    H = 512
    x = np.full((3, H), 0.5, np.float32)
    x[1] = -0.25
    x[2] = 8.0
    g = np.linspace(-3, 3, H).astype(np.float32)
    y = oracle.rmsnorm(x, g, 0.0)
    assert np.array_equal(y[0], g)
    assert np.array_equal(y[1], -g)
    assert np.array_equal(y[2], g)


def test_power_of_two_scaling_leaves_the_result_unchanged():
    rng = np.random.default_rng(3)
    x = rng.standard_normal((8, 1024)).astype(np.float32)
    g = rng.standard_normal(1024).astype(np.float32)
    y = oracle.rmsnorm(x, g, 0.0)
    for s in (0.25, 4.0, 1024.0):
        assert np.array_equal(oracle.rmsnorm(x * np.float32(s), g, 0.0), y)


def test_pythagorean_row():
    """x = (3, 4, 0, ...), H = 256: mean(x^2) = 25/256 and its root 0.3125 are
    exact, so y = (3, 4) / 0.3125 = (9.6, 12.8) to within the rounding of the
    reciprocal and two products."""
    x = np.zeros((1, 256), np.float32)
    x[0, :2] = (3.0, 4.0)
    y = oracle.rmsnorm(x, np.ones(256, np.float32), 0.0)
    assert abs(y[0, 0] - 9.6) <= 3 * np.spacing(np.float32(9.6))
    assert abs(y[0, 1] - 12.8) <= 3 * np.spacing(np.float32(12.8))
    assert np.all(y[0, 2:] == 0)


def test_zero_row_with_eps_is_zero():
    y = oracle.rmsnorm(np.zeros((2, 256), np.float32), np.ones(256, np.float32), 1e-6)
    assert np.all(y == 0)


def test_bf16_rounding_is_nearest_even():
    v = np.array([1.0, 1.0 + 2.0 ** -8, 1.0 + 3 * 2.0 ** -8, -2.5, 2.0 ** -133, np.inf], np.float32)
    bits = oracle.round_bf16(v)
    assert bits.tolist() == [0x3F80, 0x3F80, 0x3F82, 0xC020, 0x0001, 0x7F80]  # 2^-133: smallest bf16 subnormal
    assert (oracle.round_bf16(np.array([np.nan], np.float32))[0] & 0x7FC0) == 0x7FC0


def test_rejects_bad_arguments():
    with pytest.raises(ValueError):
        oracle.rmsnorm(np.zeros((1, 100), np.float32), np.ones(100, np.float32), 1e-6)
    with pytest.raises(ValueError):
        oracle.rmsnorm(np.zeros((1, 256), np.float32), np.ones(256, np.float32), -1.0)
