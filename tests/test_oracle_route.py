"""Pins for expert selection and routing weights: brute-force sorting,
scipy's softmax, the hand cases in tests/golden/hand_cases.json and the
defining properties of group-limited selection."""
import json
import math
import os

import numpy as np
import pytest
from scipy.special import softmax

import oracle

GOLDEN = json.load(open(os.path.join(os.path.dirname(__file__), "golden", "hand_cases.json")))


def brute_topk(key_row, k, allowed=None):
    cand = [e for e in range(len(key_row)) if allowed is None or allowed[e]]
    return sorted(cand, key=lambda e: (-float(key_row[e]), e))[:k]


@pytest.mark.parametrize("E,k", [(8, 2), (128, 8), (64, 6), (6, 6), (5, 1)])
def test_softmax_selection_matches_brute_force_with_ties(E, k):
    rng = np.random.default_rng(E * 100 + k)
    logits = rng.integers(-3, 4, size=(200, E)).astype(np.float32)  # many exact ties
    ids, _ = oracle.route(logits, k)
    for t in range(logits.shape[0]):
        assert list(ids[t]) == brute_topk(logits[t], k)


def test_renormalised_weights_are_softmax_over_selected():
    rng = np.random.default_rng(3)
    logits = (1.3 * rng.standard_normal((100, 32))).astype(np.float32)
    ids, w = oracle.route(logits, 4)
    for t in range(100):
        np.testing.assert_allclose(w[t], softmax(logits[t, ids[t]].astype(np.float64)), rtol=1e-13)
    np.testing.assert_allclose(w.sum(1), 1.0, rtol=1e-13)


def test_k_equals_E_gives_full_softmax_and_k1_gives_one():
    rng = np.random.default_rng(4)
    logits = rng.standard_normal((20, 8)).astype(np.float32)
    ids, w = oracle.route(logits, 8)
    for t in range(20):
        full = softmax(logits[t].astype(np.float64))
        np.testing.assert_allclose(w[t], full[ids[t]], rtol=1e-13)
        assert sorted(ids[t]) == list(range(8))
    _, w1 = oracle.route(logits, 1)
    assert np.all(w1 == 1.0)


def test_unnormalised_weights_are_full_softmax_at_selected():
    rng = np.random.default_rng(5)
    logits = rng.standard_normal((30, 16)).astype(np.float32)
    ids, w = oracle.route(logits, 3, renormalize=False, routed_scale=2.0)
    for t in range(30):
        np.testing.assert_allclose(w[t], 2.0 * softmax(logits[t].astype(np.float64))[ids[t]], rtol=1e-13)


def test_hand_case_softmax_ties():
    g = GOLDEN["softmax_ties"]
    ids, w = oracle.route(np.array(g["logits"], np.float32), g["top_k"])
    assert ids.tolist() == g["expected_ids"]
    np.testing.assert_allclose(w, g["expected_w"], rtol=1e-14)


def test_hand_case_sigmoid_grouped():
    g = GOLDEN["sigmoid_grouped"]
    ids, w = oracle.route(np.array(g["logits"], np.float32), g["top_k"], "sigmoid", True, g["n_group"],
                          g["topk_group"], g["routed_scale"], np.array(g["select_bias"], np.float32))
    assert ids.tolist() == g["expected_ids"]
    np.testing.assert_allclose(w, g["expected_w"], rtol=1e-14)


def test_sigmoid_single_group_is_plain_topk_by_biased_score():
    rng = np.random.default_rng(6)
    E, k = 64, 8
    logits = rng.standard_normal((100, E)).astype(np.float32)
    bias = (0.01 * rng.standard_normal(E)).astype(np.float32)
    ids, w = oracle.route(logits, k, "sigmoid", True, 1, 1, 2.5, bias)
    s = oracle.sigmoid(logits)
    q = (s + bias[None, :]).astype(np.float32)
    for t in range(100):
        assert list(ids[t]) == brute_topk(q[t], k)
        sel = s[t, ids[t]].astype(np.float64)
        np.testing.assert_allclose(w[t], 2.5 * sel / sel.sum(), rtol=1e-13)


@pytest.mark.parametrize("E,G,TG,k", [(256, 8, 4, 8), (32, 4, 2, 3), (16, 8, 3, 5)])
def test_sigmoid_grouped_against_sort_based_selection(E, G, TG, k):
    rng = np.random.default_rng(E + G)
    T = 300
    logits = (1.7 * rng.standard_normal((T, E))).astype(np.float32)
    logits[::7, : E // 2] = 0.25  # plant exact ties in every other token's first half
    bias = (0.01 * rng.standard_normal(E)).astype(np.float32)
    ids, w = oracle.route(logits, k, "sigmoid", True, G, TG, 2.5, bias)
    q = (oracle.sigmoid(logits) + bias[None, :]).astype(np.float32)
    gs = E // G
    for t in range(T):
        top2 = np.sort(q[t].reshape(G, gs), axis=1)[:, ::-1][:, :2]
        gscore = (top2[:, 0] + top2[:, 1]).astype(np.float32)
        kept = sorted(range(G), key=lambda g: (-float(gscore[g]), g))[:TG]
        allowed = np.zeros(E, bool)
        for g in kept:
            allowed[g * gs:(g + 1) * gs] = True
        assert list(ids[t]) == brute_topk(q[t], k, allowed)
        assert len({e // gs for e in ids[t]}) <= TG
    np.testing.assert_allclose(w.sum(1), 2.5, rtol=1e-13)


def test_route_rejects_invalid_configurations():
    l = np.zeros((2, 8), np.float32)
    with pytest.raises(ValueError):
        oracle.route(l, 9)
    with pytest.raises(ValueError):
        oracle.route(l, 2, "sigmoid", True, 3, 1)
    with pytest.raises(ValueError):
        oracle.route(l, 5, "sigmoid", True, 4, 2)  # only 4 experts in 2 groups of 2


def _nan_last(v):
    """Sort key of the choice's reading for non-finite scores: NaN counts as -inf."""
    v = float(v)
    return -math.inf if math.isnan(v) else v


def test_nan_scores_rank_as_minus_infinity():
    """Non-finite logits still give valid ids: a NaN key counts as -inf, ties
    (among NaN and -inf keys too) go to the lower index."""
    rng = np.random.default_rng(11)
    E, k = 16, 6
    logits = rng.integers(-2, 3, size=(200, E)).astype(np.float32)
    logits[rng.random((200, E)) < 0.3] = np.nan
    logits[rng.random((200, E)) < 0.1] = -np.inf
    logits[5] = np.nan  # a token whose every logit is NaN
    ids, _ = oracle.route(logits, k)
    for t in range(200):
        assert list(ids[t]) == sorted(range(E), key=lambda e: (-_nan_last(logits[t, e]), e))[:k]
    assert list(ids[5]) == list(range(k))
    # sigmoid, group-limited, NaN selection biases
    bias = np.zeros(E, np.float32)
    bias[[1, 9]] = np.nan
    ids2, _ = oracle.route(logits, 4, "sigmoid", True, 4, 2, 1.0, bias)
    assert ((ids2 >= 0) & (ids2 < E)).all()
    q = (oracle.sigmoid(logits) + bias[None, :]).astype(np.float32)
    for t in range(200):
        key = [_nan_last(v) for v in q[t]]
        gscore = []
        for g in range(4):
            top2 = sorted(key[4 * g:4 * g + 4], reverse=True)[:2]
            s = np.float32(top2[0]) + np.float32(top2[1])
            gscore.append(_nan_last(s))
        kept = sorted(range(4), key=lambda g: (-gscore[g], g))[:2]
        cand = [e for e in range(E) if e // 4 in kept]
        assert list(ids2[t]) == sorted(cand, key=lambda e: (-key[e], e))[:4]
