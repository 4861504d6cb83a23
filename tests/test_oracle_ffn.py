"""Pins for the Fused MoE and Weight Sum parts of the oracle: permutation vs
numpy's stable argsort, weight decoding vs torch's float8 type and the int4
closed form, the expert FFN vs plain Python loops, exact integer arithmetic
and a hand case, the whole layer vs a dense FFN in the cases where MoE
reduces to one."""
import json
import math
import os

import numpy as np
import pytest
import torch

import oracle
import synth

GOLDEN = json.load(open(os.path.join(os.path.dirname(__file__), "golden", "hand_cases.json")))


# ------------------------------------------------------------ permutation

@pytest.mark.parametrize("T,k,E", [(64, 2, 8), (33, 8, 128), (100, 6, 64), (1, 1, 1), (7, 3, 5)])
def test_permute_is_stable_counting_sort(T, k, E):
    rng = np.random.default_rng(T * k + E)
    ids = rng.integers(0, E, size=(T, k)).astype(np.int32)
    counts, offsets, sp, pp = oracle.permute(ids, E)
    flat = ids.ravel()
    assert np.array_equal(counts, np.bincount(flat, minlength=E))
    assert offsets[0] == 0 and np.array_equal(offsets[1:], np.cumsum(counts))
    assert np.array_equal(sp, np.argsort(flat, kind="stable"))
    assert np.array_equal(pp[sp], np.arange(T * k))


def test_permute_all_to_one_expert_and_empty_experts():
    ids = np.full((10, 2), 3, np.int32)
    counts, offsets, sp, pp = oracle.permute(ids, 6)
    assert counts.tolist() == [0, 0, 0, 20, 0, 0]
    assert offsets.tolist() == [0, 0, 0, 0, 20, 20, 20]
    assert sp.tolist() == list(range(20)) and pp.tolist() == list(range(20))


def test_permute_rejects_out_of_range_ids():
    with pytest.raises(ValueError):
        oracle.permute(np.array([[0, 9]], np.int32), 4)


# --------------------------------------------------------- weight formats

def test_e4m3_all_codes_match_torch_float8():
    codes = torch.arange(256, dtype=torch.int32).to(torch.uint8)
    ref = codes.view(torch.float8_e4m3fn).to(torch.float64).numpy()
    got = np.array([oracle.e4m3_value(c) for c in range(256)])
    nan = np.isnan(ref)
    assert np.array_equal(np.isnan(got), nan) and nan.sum() == 2  # 0x7f and 0xff
    assert np.array_equal(got[~nan], ref[~nan])
    assert got[0x7e] == 448.0 and got[0x01] == 2.0 ** -9 and got[0x08] == 2.0 ** -6


def test_fp8_block_dequant_matches_broadcast_scales():
    rng = np.random.default_rng(0)
    N, K = 256, 384
    q = rng.integers(0, 256, size=(N, K)).astype(np.uint8)
    q[(q & 0x7f) == 0x7f] = 0x00  # no NaN codes
    s = rng.uniform(0.5, 2.0, size=(N // 128, K // 128)).astype(np.float32)
    val = torch.from_numpy(q).view(torch.float8_e4m3fn).to(torch.float64).numpy()
    ref = val * np.repeat(np.repeat(s.astype(np.float64), 128, 0), 128, 1)
    assert np.array_equal(oracle.dequant_fp8_b128(q, s), ref)


def test_int4_group_dequant_closed_form():
    rng = np.random.default_rng(1)
    N, K = 3, 256
    vals = rng.integers(-8, 8, size=(N, K))
    packed = ((vals[:, 0::2] & 0xf) | ((vals[:, 1::2] & 0xf) << 4)).astype(np.uint8)
    s = synth.normal_bf16(0, 99, 0.1, (N, K // 128))
    sf = synth.bf16_bits_to_f32(s).astype(np.float64)
    ref = vals * np.repeat(sf, 128, axis=1)
    assert np.array_equal(oracle.dequant_int4_g128(packed, s), ref)
    # all 16 codes in one byte position
    one = np.array([[c | (c << 4) for c in range(16)] + [0] * 48], np.uint8)
    d = oracle.dequant_int4_g128(one, np.array([[0x3f80]], np.uint16))  # scale 1.0
    assert d[0, 0:32:2].tolist() == [0, 1, 2, 3, 4, 5, 6, 7, -8, -7, -6, -5, -4, -3, -2, -1]


# ---------------------------------------------------------------- expert FFN

def numpy_swiglu(x, wg, wu, wd):
    g = x @ wg.T
    u = x @ wu.T
    return (g / (1.0 + np.exp(-g)) * u) @ wd.T


def brute_swiglu(x, wg, wu, wd):
    """The SwiGLU FFN as plain Python loops over the definition's indices
    (independent of any matrix library)."""
    n, H = len(x), len(x[0])
    I = len(wg)
    y = []
    for r in range(n):
        a = []
        for i in range(I):
            g = sum(float(wg[i][h]) * float(x[r][h]) for h in range(H))
            u = sum(float(wu[i][h]) * float(x[r][h]) for h in range(H))
            a.append(g / (1.0 + math.exp(-g)) * u)
        y.append([sum(float(wd[o][i]) * a[i] for i in range(I)) for o in range(H)])
    return np.array(y)


def test_expert_ffn_matches_brute_force_loops():
    rng = np.random.default_rng(2)
    n, H, I = 5, 24, 10  # non-square, so a transposed operand cannot pass
    x = rng.standard_normal((n, H))
    wg, wu = rng.standard_normal((I, H)) * 0.3, rng.standard_normal((I, H)) * 0.3
    wd = rng.standard_normal((H, I)) * 0.3
    np.testing.assert_allclose(oracle.expert_ffn(x, wg, wu, wd), brute_swiglu(x, wg, wu, wd), rtol=1e-12,
                               atol=1e-14)


def test_expert_ffn_is_exact_on_integers():
    """With integer operands and gate values >= 40, silu(g) = g exactly in
    fp64 (exp(-40) < 2^-57), so every output is an integer below 2^53 that
    Python's exact integer arithmetic reproduces."""
    rng = np.random.default_rng(9)
    n, H, I = 4, 12, 7
    x = rng.integers(1, 4, size=(n, H))
    wg = rng.integers(1, 4, size=(I, H))  # g >= 12 * 1 * 1 ... shifted below to >= 40
    wg[:, 0] += 40
    wu = rng.integers(-3, 4, size=(I, H))
    wd = rng.integers(-5, 6, size=(H, I))
    g = [[sum(int(wg[i, h]) * int(x[r, h]) for h in range(H)) for i in range(I)] for r in range(n)]
    assert min(min(row) for row in g) >= 40
    u = [[sum(int(wu[i, h]) * int(x[r, h]) for h in range(H)) for i in range(I)] for r in range(n)]
    y = [[sum(int(wd[o, i]) * g[r][i] * u[r][i] for i in range(I)) for o in range(H)] for r in range(n)]
    got = oracle.expert_ffn(x.astype(np.float64), wg.astype(np.float64), wu.astype(np.float64),
                            wd.astype(np.float64))
    assert got.tolist() == [[float(v) for v in row] for row in y]


def test_expert_ffn_hand_case():
    g = GOLDEN["ffn_h2_i1"]
    y = oracle.expert_ffn(np.array([g["x"]]), np.array(g["w_gate"]), np.array(g["w_up"]),
                          np.array(g["w_down"]))
    np.testing.assert_allclose(y[0], g["expected_y"], rtol=1e-15)
    a = 2.0 / (1.0 + math.exp(-1.0))
    np.testing.assert_allclose(y[0], [a, 3 * a], rtol=1e-15)


def test_combine_matches_einsum():
    rng = np.random.default_rng(3)
    T, k, H = 6, 3, 10
    y = rng.standard_normal((T * k, H))
    w = rng.standard_normal((T, k))
    pp = rng.permutation(T * k).astype(np.int32).reshape(T, k)
    sh = rng.standard_normal((T, H))
    ref = np.einsum("tj,tjh->th", w, y[pp]) + sh
    np.testing.assert_allclose(oracle.combine(y, w, pp, sh), ref, rtol=1e-13)


# -------------------------------------------------------------- whole layer

def _tiny(E, k, seed=11, H=256, I=128, T=24):
    return synth.WORKLOADS[1].replace(T=T, H=H, I=I, E=E, top_k=k, seed=seed)


def test_layer_with_one_expert_is_dense_swiglu():
    wl = _tiny(1, 1)
    inp = synth.make_inputs(wl)
    got = oracle.forward(wl, inp)
    ex = inp["experts"]
    ref = numpy_swiglu(inp["x"].astype(np.float64), ex["w_gate"][0].astype(np.float64),
                       ex["w_up"][0].astype(np.float64), ex["w_down"][0].astype(np.float64))
    assert np.all(got["topk_w"] == 1.0)
    np.testing.assert_allclose(got["out"], ref, rtol=1e-12, atol=1e-15)


def test_layer_with_identical_experts_is_dense_swiglu():
    wl = _tiny(8, 3)
    inp = synth.make_inputs(wl)
    ex = inp["experts"]
    for key in ("w_gate", "w_up", "w_down"):
        ex[key] = np.ascontiguousarray(np.broadcast_to(ex[key][:1], ex[key].shape))
    got = oracle.forward(wl, inp)
    ref = numpy_swiglu(inp["x"].astype(np.float64), ex["w_gate"][0].astype(np.float64),
                       ex["w_up"][0].astype(np.float64), ex["w_down"][0].astype(np.float64))
    np.testing.assert_allclose(got["out"], ref, rtol=1e-12, atol=1e-14)


def test_layer_with_shared_expert_adds_its_dense_output():
    wl = _tiny(4, 2).replace(has_shared=True, I_shared=64, wq="f32")
    inp = synth.make_inputs(wl)
    full = oracle.forward(wl, inp)
    sh = inp["shared"]
    ysh = numpy_swiglu(inp["x"].astype(np.float64), sh["w_gate"][0].astype(np.float64),
                       sh["w_up"][0].astype(np.float64), sh["w_down"][0].astype(np.float64))
    inp2 = dict(inp)
    wl2 = wl.replace(has_shared=False)
    routed = oracle.forward(wl2, inp2)
    np.testing.assert_allclose(full["out"], routed["out"] + ysh, rtol=1e-12, atol=1e-14)


def test_layer_row_subset_equals_full_rows():
    wl = _tiny(8, 2)
    inp = synth.make_inputs(wl)
    full = oracle.forward(wl, inp)
    rows = [0, 5, 23, 7]
    sub = oracle.forward(wl, inp, rows=rows)
    # the fp64 matrix products may sum in another order for another row count:
    # equal up to fp64 rounding, not bit for bit
    np.testing.assert_allclose(sub["out"], full["out"][rows], rtol=1e-13, atol=1e-16)
    np.testing.assert_array_equal(sub["topk_ids"], full["topk_ids"])
