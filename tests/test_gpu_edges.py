"""GPU parity on edge shapes: one token, no tokens, ragged tiles, every token
on one expert, k = E, a single expert, and argument errors."""
import numpy as np
import pytest
import torch

import oracle
import paper_2607_12875_gb300 as gb
import synth
from gpu_helpers import act_np, assert_close, config, to_device, tol_for, wbundle, workspace

pytestmark = pytest.mark.gpu

TINY = synth.WORKLOADS[1]


def run(wl, route, inp=None):
    inp = synth.make_inputs(wl) if inp is None else inp
    dev = to_device(wl, inp)
    cfg = config(wl, route)
    ws = workspace(cfg)
    out = torch.empty((wl.T, wl.H), dtype=dev["x"].dtype, device="cuda")
    ids = torch.empty((max(wl.T, 1), wl.top_k), dtype=torch.int32, device="cuda")
    counts = torch.empty(wl.E, dtype=torch.int32, device="cuda")
    gb.moe_forward(cfg, dev["x"], dev["w_router"], dev["logit_bias"], dev["select_bias"], wbundle(dev["experts"]),
                   wbundle(dev["shared"]), out, ws, topk_ids=ids if wl.T else None,
                   counts=counts if wl.T else None)
    torch.cuda.synchronize()
    return inp, out, ids, counts


def check(wl, route, inp=None):
    inp, out, ids, counts = run(wl, route, inp)
    ref = oracle.forward(wl, inp)
    assert np.array_equal(ids.cpu().numpy()[: wl.T], ref["topk_ids"])
    assert np.array_equal(counts.cpu().numpy(), ref["counts"])
    assert_close(act_np(out), ref["out"], tol_for(wl))
    return ref


@pytest.mark.parametrize("route", ["simt", "stream"])
@pytest.mark.parametrize("act", ["f32", "bf16"])
def test_single_token(route, act):
    wl = TINY.replace(T=1, act=act, wq=act, seed=21)
    check(wl, route)


def test_no_tokens_is_a_noop():
    wl = TINY.replace(T=0)
    cfg = config(wl)
    ws = workspace(cfg)
    dev = to_device(wl, synth.make_inputs(wl.replace(T=1)))
    out = torch.empty((0, wl.H), dtype=torch.float32, device="cuda")
    gb.moe_forward(cfg, dev["x"], dev["w_router"], None, None, wbundle(dev["experts"]), None, out, ws)
    torch.cuda.synchronize()


@pytest.mark.parametrize("route", ["simt", "stream"])
def test_ragged_tiles(route):
    # 37 tokens x top-3 over 5 experts: no expert's row count is a tile multiple
    wl = TINY.replace(T=37, E=5, top_k=3, act="bf16", wq="bf16", seed=22, H=512, I=256)
    check(wl, route)


@pytest.mark.parametrize("route", ["simt", "stream"])
def test_every_token_on_one_expert(route):
    wl = TINY.replace(T=70, E=8, top_k=2, seed=23, act="bf16", wq="bf16")
    inp = synth.make_inputs(wl)
    bias = np.zeros(wl.E, np.float32)
    bias[5] = 1000.0
    inp["logit_bias"] = bias
    ref = check(wl, route, inp)
    assert ref["counts"][5] == wl.T


@pytest.mark.parametrize("route", ["simt", "stream"])
def test_k_equals_E_and_single_expert(route):
    check(TINY.replace(T=9, E=8, top_k=8, seed=24), route)
    check(TINY.replace(T=9, E=1, top_k=1, seed=25), route)


@pytest.mark.parametrize("wq", ["fp8_b128", "int4_g128", "mxfp4"])
@pytest.mark.parametrize("route", ["simt", "stream"])
def test_quantised_weights_small(wq, route):
    wl = TINY.replace(T=24, E=4, top_k=2, act="bf16", wq=wq, H=256, I=256, seed=26)
    check(wl, route)


def test_sigmoid_grouped_small_with_shared():
    wl = TINY.replace(T=40, E=16, top_k=4, act="bf16", wq="fp8_b128", H=256, I=128, seed=27, score="sigmoid",
                      routed_scale=2.5, n_group=4, topk_group=2, has_shared=True, I_shared=256,
                      select_bias_sigma=0.01)
    check(wl, "simt")
    check(wl, "stream")


def test_argument_errors_launch_nothing():
    wl = TINY
    cfg = config(wl)
    ws = workspace(cfg)
    x = torch.zeros((wl.T, wl.H), device="cuda")
    wr = torch.zeros((wl.E, wl.H), device="cuda")
    ids = torch.empty((wl.T, wl.top_k), dtype=torch.int32, device="cuda")
    w = torch.empty((wl.T, wl.top_k), dtype=torch.float32, device="cuda")
    with pytest.raises(gb.GbmoeError) as e:
        gb.moe_route(cfg, x, wr, None, None, ids, w, ws[: gb.workspace_size(cfg) // 4])
    assert e.value.status == gb.EWORKSPACE
    with pytest.raises(gb.GbmoeError) as e:
        gb.moe_route(cfg, x[:, 1:], wr, None, None, ids, w, ws)  # misaligned x
    assert e.value.status == gb.EINVAL


@pytest.mark.parametrize("T,E,k,H,act", [(1100, 20, 3, 512, "bf16"), (1024, 16, 2, 256, "bf16"),
                                         (2049, 256, 8, 768, "bf16"), (1100, 20, 3, 512, "f32"),
                                         (1023, 20, 3, 512, "bf16"), (7, 256, 8, 768, "f32")])
def test_batch_routing_is_bit_exact(T, E, k, H, act):
    # bf16 batches from 1024 tokens take the tiled logits kernel, smaller ones
    # and fp32 the per-warp one; ragged token and expert tiles
    wl = TINY.replace(T=T, E=E, top_k=k, H=H, act=act, wq=act, seed=T + E)
    inp = synth.make_inputs(wl, with_experts=False)
    dev = to_device(wl, dict(inp, experts={}, shared=None))
    cfg = config(wl)
    ws = workspace(cfg)
    ids = torch.empty((T, k), dtype=torch.int32, device="cuda")
    w = torch.empty((T, k), dtype=torch.float32, device="cuda")
    gb.moe_route(cfg, dev["x"], dev["w_router"], None, None, ids, w, ws)
    torch.cuda.synchronize()
    x32 = inp["x"] if act == "f32" else synth.bf16_bits_to_f32(inp["x"])
    g32 = inp["w_router"] if act == "f32" else synth.bf16_bits_to_f32(inp["w_router"])
    ref_ids, ref_w = oracle.route(oracle.gate_logits(x32, g32), k)
    assert np.array_equal(ids.cpu().numpy(), ref_ids)
    np.testing.assert_allclose(w.cpu().numpy(), ref_w, rtol=2e-6, atol=1e-7)


# The streaming kernels let one CTA cover 1, 2 or 4 column groups, as many as
# keep 8 waves of CTAs (two per SM) in the grid. The decode workload itself
# takes 4; these shapes take 2 (64 active experts) and 4 with more rows per
# expert than one pass over the weights holds (16 rows, kNT = 8).
DECODE = synth.WORKLOADS[2]


@pytest.mark.parametrize("T,E,k", [(8, 64, 8), (256, 128, 8)])
def test_streaming_column_groups_per_cta(T, E, k):
    wl = DECODE.replace(T=T, E=E, top_k=k, seed=90 + T)
    assert wl.P <= 16 * wl.E  # streaming route
    inp, out, ids, counts = run(wl, "stream")
    rows = np.unique(np.r_[np.arange(min(T, 24)), np.arange(T - 8, T)]) if T > 32 else None
    ref = oracle.forward(wl, inp, rows=rows)
    assert np.array_equal(ids.cpu().numpy(), ref["topk_ids"])
    assert np.array_equal(counts.cpu().numpy(), ref["counts"])
    got = act_np(out) if rows is None else act_np(out)[ref["rows"]]
    assert_close(got, ref["out"], tol_for(wl))


# The largest expert count and top-k the configuration admits (E = 512,
# top_k = 32), softmax and sigmoid with 32 groups, on every FFN route that
# covers the activation dtype.
@pytest.mark.parametrize("score,act,route", [("softmax", "f32", "stream"), ("softmax", "f32", "simt"),
                                             ("softmax", "bf16", "tc"), ("sigmoid", "bf16", "stream")])
def test_maximum_experts_and_top_k(score, act, route):
    extra = dict(score="sigmoid", routed_scale=2.5, n_group=32, topk_group=4, select_bias_sigma=0.01) \
        if score == "sigmoid" else {}
    wl = TINY.replace(T=40, E=512, top_k=32, H=256, I=128, act=act, wq=act, seed=77, **extra)
    assert gb.check_config(config(wl, route)) == gb.OK
    ref = check(wl, route)
    assert (ref["counts"] > 0).sum() > 200


@pytest.mark.parametrize("route", ["simt", "stream"])
def test_mxfp4_with_fp32_activations(route):
    """MXFP4 weights under fp32 activations (the exact-decode format on the
    fp32 routes, held to the fp32 bound of 1e-5)."""
    wl = TINY.replace(T=30, E=4, top_k=2, act="f32", wq="mxfp4", H=256, I=256, seed=28)
    inp, out, ids, counts = run(wl, route)
    ref = oracle.forward(wl, inp)
    assert np.array_equal(ids.cpu().numpy(), ref["topk_ids"])
    assert_close(act_np(out), ref["out"], 1e-5)


@pytest.mark.parametrize("score", ["softmax", "sigmoid"])
def test_tc_gate_audit_resolves_exact_ties(score):
    """Integer router weights and activations make many logits tie exactly
    (both orders sum them exactly): every such token is flagged by the audit,
    recomputed in the fixed order, and chosen as the oracle chooses (ties to
    the lower expert), on the tensor-core gate."""
    T, H, E, k = 600, 512, 32, 4
    rng = np.random.default_rng(8 if score == "softmax" else 9)
    xi = rng.integers(-2, 3, size=(T, H)).astype(np.float32)
    wi = rng.integers(-1, 2, size=(E, H)).astype(np.float32)
    wi[E // 2:] = wi[: E // 2]  # duplicated router rows: exact ties in every token
    extra = dict(score="sigmoid", n_group=4, topk_group=2) if score == "sigmoid" else {}
    cfg = gb.make_config(T, H, 128, E, k, act="bf16", w="bf16", gate_route="tc", **extra)
    x = torch.from_numpy(xi).cuda().to(torch.bfloat16)
    wr = torch.from_numpy(wi).cuda().to(torch.bfloat16)
    ws = workspace(cfg)
    ids = torch.empty((T, k), dtype=torch.int32, device="cuda")
    w = torch.empty((T, k), dtype=torch.float32, device="cuda")
    gb.moe_route(cfg, x, wr, None, None, ids, w, ws)
    torch.cuda.synchronize()
    ref_ids, ref_w = oracle.route(oracle.gate_logits(xi, wi), k, score, True, extra.get("n_group", 1),
                                  extra.get("topk_group", 1))
    assert np.array_equal(ids.cpu().numpy(), ref_ids)
    np.testing.assert_allclose(w.cpu().numpy(), ref_w, rtol=1e-5, atol=1e-7)
