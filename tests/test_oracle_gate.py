"""Pins for the MoE Gate part of the oracle: router logits and the pinned
exponential. References: exact integer arithmetic, an fp64 error bound,
Python's math.exp."""
import math

import numpy as np
import pytest

import oracle


def test_logits_exact_on_small_integers():
    # Integer inputs small enough that every partial sum is exact in fp32:
    # the result must equal the int64 dot product whatever the order.
    T, H, E = 5, 512, 7
    h = np.arange(H)
    x = np.stack([((h * (t + 3)) % 7) - 3 for t in range(T)]).astype(np.int64)
    w = np.stack([((h * (e + 1) + e) % 5) - 2 for e in range(E)]).astype(np.int64)
    bias = np.arange(E, dtype=np.int64) - 3
    got = oracle.gate_logits(x.astype(np.float32), w.astype(np.float32), bias.astype(np.float32))
    want = x @ w.T + bias[None, :]
    assert np.array_equal(got.astype(np.int64), want)


def test_logits_single_element_sensitivity():
    # A one-hot x picks exactly one column of W: catches a wrong index or a
    # dropped chunk anywhere in the 8-element / 32-lane decomposition.
    H, E = 768, 3
    rng = np.random.default_rng(1)
    w = rng.integers(-50, 50, size=(E, H)).astype(np.float32)
    for h in [0, 7, 8, 255, 256, 257, 511, 767]:
        x = np.zeros((1, H), np.float32)
        x[0, h] = 1.0
        assert np.array_equal(oracle.gate_logits(x, w)[0], w[:, h])


@pytest.mark.parametrize("H", [256, 4096, 7168])
def test_logits_within_fp32_bound_of_fp64(H):
    rng = np.random.default_rng(H)
    T, E = 16, 9
    x = rng.standard_normal((T, H)).astype(np.float32)
    w = (0.02 * rng.standard_normal((E, H))).astype(np.float32)
    b = rng.standard_normal(E).astype(np.float32)
    got = oracle.gate_logits(x, w, b).astype(np.float64)
    exact = x.astype(np.float64) @ w.astype(np.float64).T + b[None, :]
    # each path: H/32 fused multiply-adds, 5 pairwise additions, 1 bias add
    n = H // 32 + 6
    u = 2.0 ** -24
    gamma = n * u / (1 - n * u)
    mag = np.abs(x.astype(np.float64)) @ np.abs(w.astype(np.float64)).T + np.abs(b)[None, :]
    assert np.all(np.abs(got - exact) <= gamma * mag)


def test_logits_reject_bad_hidden():
    with pytest.raises(ValueError):
        oracle.gate_logits(np.zeros((1, 200), np.float32), np.zeros((2, 200), np.float32))


def test_pexp_against_math_exp():
    xs = np.concatenate([np.linspace(-86, 88, 400001), np.array([0.0, -0.0, 1.0, -1.0, 1e-8, -1e-8])])
    xs = xs.astype(np.float32)
    got = oracle.pexp(xs).astype(np.float64)
    ref = np.array([math.exp(float(v)) for v in xs])
    ulp = np.spacing(ref.astype(np.float32)).astype(np.float64)
    assert np.max(np.abs(got - ref) / ulp) <= 3.0
    assert oracle.pexp(np.array([0.0], np.float32))[0] == 1.0


def test_pexp_clamps_to_normal_range():
    got = oracle.pexp(np.array([-1000.0, -86.0, 88.0, 1000.0], np.float32)).astype(np.float64)
    assert got[0] == got[1] and got[2] == got[3]
    assert np.isfinite(got).all() and (got > np.finfo(np.float32).tiny).all()


def test_sigmoid_against_math():
    ls = np.linspace(-20, 20, 20001).astype(np.float32)
    got = oracle.sigmoid(ls).astype(np.float64)
    ref = np.array([1.0 / (1.0 + math.exp(-float(v))) for v in ls])
    ulp = np.spacing(ref.astype(np.float32)).astype(np.float64)
    assert np.max(np.abs(got - ref) / ulp) <= 4.0
    assert oracle.sigmoid(np.array([0.0], np.float32))[0] == 0.5


def test_pexp_and_sigmoid_propagate_nan():
    """NaN in, NaN out, as for exp (the clamp does not turn NaN into a number)."""
    got = oracle.pexp(np.array([np.nan, -np.nan], np.float32))
    assert np.isnan(got).all()
    assert np.isnan(oracle.sigmoid(np.array([np.nan], np.float32))).all()
    assert oracle.pexp(np.array([np.inf], np.float32))[0] == oracle.pexp(np.array([88.0], np.float32))[0]
