"""Pins for the MXFP4 weight format (OCP Microscaling v1.0): the oracle's
E2M1 and E8M0 values against the specification's table (a cited fixture),
the dequantised matrix against that table and exact powers of two, and the
input generator's quantiser against a brute-force nearest-grid search."""
import json
import math
import os

import numpy as np

import oracle
import synth

GOLDEN = json.load(open(os.path.join(os.path.dirname(__file__), "golden", "mxfp4_e2m1.json")))
TABLE = np.array([GOLDEN["code_value"][str(c)] for c in range(16)])


def test_e2m1_codes_match_the_specification_table():
    got = np.array([oracle.e2m1_value(c) for c in range(16)])
    assert np.array_equal(got, TABLE)
    assert math.copysign(1.0, oracle.e2m1_value(8)) == -1.0  # negative zero


def test_e8m0_scales_are_powers_of_two():
    for s, v in GOLDEN["e8m0_examples"].items():
        assert oracle.e8m0_value(int(s)) == v
    assert all(oracle.e8m0_value(s) == math.ldexp(1.0, s - 127) for s in range(255))
    assert math.isnan(oracle.e8m0_value(255))


def test_dequant_mxfp4_closed_form():
    rng = np.random.default_rng(3)
    N, K = 5, 96
    codes = rng.integers(0, 16, size=(N, K))
    q = (codes[:, 0::2] | (codes[:, 1::2] << 4)).astype(np.uint8)
    s = rng.integers(100, 140, size=(N, K // 32)).astype(np.uint8)
    ref = TABLE[codes] * np.ldexp(1.0, np.repeat(s.astype(np.int64) - 127, 32, axis=1))
    assert np.array_equal(oracle.dequant_mxfp4(q, s), ref)


def _nearest_even(a):
    grid = [abs(v) for v in TABLE[:8]]
    if a >= 6.0:
        return 7
    d = [abs(a - g) for g in grid]
    best = min(d)
    return min(c for c in range(8) if d[c] == best and (c % 2 == 0 or d.count(best) == 1))


def test_generator_quantises_to_nearest_grid_point():
    seed, tid, sigma, N, K = 7, 3, 0.02, 4, 256
    q, s = synth.mxfp4(seed, tid, sigma, N, K)
    w = synth.normal_f32(seed, tid, sigma, (N * K,)).reshape(N, K)
    for n in range(N):
        for b in range(K // 32):
            blk = w[n, 32 * b:32 * b + 32].astype(np.float64)
            amax = np.max(np.abs(blk))
            assert int(s[0, n, b]) - 127 == math.floor(math.log2(amax)) - 2
            X = math.ldexp(1.0, int(s[0, n, b]) - 127)
            for j in range(32):
                k = 32 * b + j
                code = (q[0, n, k // 2] >> (4 * (k % 2))) & 0xf
                assert code & 7 == _nearest_even(abs(blk[j]) / X)
                assert (code >> 3) == (1 if blk[j] < 0 else 0)
    deq = oracle.dequant_mxfp4(q[0], s[0])
    assert np.max(np.abs(deq - w)) <= np.max(np.abs(w))  # sane magnitude, saturation at 6X bounded
