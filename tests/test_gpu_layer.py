"""GPU parity: every C-ABI call of the layer against the CPU oracle on the
same seeded inputs, for all five workload shapes and every FFN route.
Routing ids, the permutation and the counts must match bit for bit; outputs
within the workload's tolerance (max |gpu - oracle| / max |oracle|)."""
import numpy as np
import pytest
import torch

import oracle
import paper_2607_12875_gb300 as gb
import synth
from gpu_helpers import (act_np, config, rel_err, sample_rows, to_device, tol_for, wbundle, workspace)

pytestmark = pytest.mark.gpu

# sampled-token counts for the big workloads (all tokens for the first two)
SAMPLE = {3: (48, 16), 4: (20, 6), 5: (40, 12)}
ROUTES = {1: ["simt", "stream", "auto"], 2: ["stream", "simt", "auto"], 3: ["simt", "auto"],
          4: ["simt", "auto", "tc_dequant"], 5: ["simt", "auto", "tc"]}

_cache = {}


def case(wid):
    """Host inputs, device inputs and the oracle for workload wid (one cached)."""
    if wid not in _cache:
        _cache.clear()
        torch.cuda.empty_cache()
        wl = synth.WORKLOADS[wid]
        inp = synth.make_inputs(wl)
        dev = to_device(wl, inp)
        # routing for all tokens, expert outputs for the sampled tokens
        x32 = inp["x"] if wl.act == "f32" else synth.bf16_bits_to_f32(inp["x"])
        g32 = inp["w_router"] if wl.act == "f32" else synth.bf16_bits_to_f32(inp["w_router"])
        logits = oracle.gate_logits(x32, g32, inp["logit_bias"])
        ids, _ = oracle.route(logits, wl.top_k, wl.score, wl.renormalize, wl.n_group, wl.topk_group,
                              wl.routed_scale, inp["select_bias"])
        rows = None if wid not in SAMPLE else sample_rows(wl, ids, *SAMPLE[wid], seed=wid)
        ref = oracle.forward(wl, inp, rows=rows)
        _cache[wid] = (wl, inp, dev, ref)
    return _cache[wid]


@pytest.mark.parametrize("wid", [1, 2, 3, 4, 5])
def test_route_is_bit_exact(wid):
    wl, inp, dev, ref = case(wid)
    cfg = config(wl)
    ws = workspace(cfg)
    ids = torch.empty((wl.T, wl.top_k), dtype=torch.int32, device="cuda")
    w = torch.empty((wl.T, wl.top_k), dtype=torch.float32, device="cuda")
    gb.moe_route(cfg, dev["x"], dev["w_router"], dev["logit_bias"], dev["select_bias"], ids, w, ws)
    torch.cuda.synchronize()
    got = ids.cpu().numpy()
    mism = np.argwhere(got != ref["topk_ids"])
    assert mism.size == 0, f"{len(mism)} routing mismatches, first at {mism[:3].tolist()}"
    np.testing.assert_allclose(w.cpu().numpy(), ref["topk_w"], rtol=2e-6, atol=1e-7)


@pytest.mark.parametrize("wid", [1, 2, 3, 4, 5])
def test_permute_is_bit_exact(wid):
    wl, inp, dev, ref = case(wid)
    cfg = config(wl)
    ws = workspace(cfg)
    P, E = wl.P, wl.E
    ids = torch.from_numpy(ref["topk_ids"]).cuda()
    counts = torch.empty(E, dtype=torch.int32, device="cuda")
    offsets = torch.empty(E + 1, dtype=torch.int32, device="cuda")
    sp = torch.empty(P, dtype=torch.int32, device="cuda")
    pp = torch.empty(P, dtype=torch.int32, device="cuda")
    gb.moe_permute(cfg, ids, counts, offsets, sp, pp, ws)
    torch.cuda.synchronize()
    assert np.array_equal(counts.cpu().numpy(), ref["counts"])
    assert np.array_equal(offsets.cpu().numpy(), ref["offsets"])
    assert np.array_equal(sp.cpu().numpy(), ref["sorted_pair"])
    assert np.array_equal(pp.cpu().numpy(), ref["pair_pos"])


def _forward(wl, dev, route, T=None):
    cfg = config(wl, route, T)
    ws = workspace(cfg)
    T = wl.T if T is None else T
    out = torch.empty((T, wl.H), dtype=dev["x"].dtype, device="cuda")
    ids = torch.empty((T, wl.top_k), dtype=torch.int32, device="cuda")
    counts = torch.empty(wl.E, dtype=torch.int32, device="cuda")
    gb.moe_forward(cfg, dev["x"], dev["w_router"], dev["logit_bias"], dev["select_bias"], wbundle(dev["experts"]),
                   wbundle(dev["shared"]), out, ws, topk_ids=ids, counts=counts)
    torch.cuda.synchronize()
    assert gb.moe_device_status(ws) == gb.OK
    return out, ids, counts


@pytest.mark.parametrize("wid,route", [(w, r) for w in [1, 2, 3, 4, 5] for r in ROUTES[w]])
def test_forward_matches_oracle(wid, route):
    wl, inp, dev, ref = case(wid)
    out, ids, counts = _forward(wl, dev, route)
    assert np.array_equal(ids.cpu().numpy(), ref["topk_ids"])
    assert np.array_equal(counts.cpu().numpy(), ref["counts"])
    got = act_np(out)[ref["rows"]]
    err = rel_err(got, ref["out"])
    assert err <= tol_for(wl), f"rel err {err:.3e} > {tol_for(wl):.0e}"


@pytest.mark.parametrize("wid", [1, 2, 4])
def test_grouped_ffn_rows_match_oracle(wid):
    wl, inp, dev, ref = case(wid)
    cfg = config(wl)
    ws = workspace(cfg)
    P = wl.P
    t = lambda a: torch.from_numpy(np.ascontiguousarray(a)).cuda()
    y = torch.empty((P, wl.H), dtype=dev["x"].dtype, device="cuda")
    gb.moe_grouped_ffn(cfg, dev["x"], t(ref["counts"]), t(ref["offsets"]), t(ref["sorted_pair"]),
                       wbundle(dev["experts"]), y, ws)
    torch.cuda.synchronize()
    rows = ref["rows"]
    pos = ref["pair_pos"].reshape(wl.T, wl.top_k)[rows]  # [n, k]
    got = act_np(y)[pos.ravel()].reshape(len(rows), wl.top_k, wl.H)
    err = rel_err(got, ref["y"])
    assert err <= tol_for(wl), f"rel err {err:.3e}"


def test_shared_expert_matches_oracle():
    wl, inp, dev, ref = case(4)
    cfg = config(wl)
    ws = workspace(cfg)
    ysh = torch.empty((wl.T, wl.H), dtype=dev["x"].dtype, device="cuda")
    gb.moe_shared_ffn(cfg, dev["x"], wbundle(dev["shared"]), ysh, ws)
    torch.cuda.synchronize()
    err = rel_err(act_np(ysh)[ref["rows"]], ref["y_shared"])
    assert err <= tol_for(wl), f"rel err {err:.3e}"


@pytest.mark.parametrize("act", ["f32", "bf16"])
def test_combine_matches_oracle(act):
    rng = np.random.default_rng(5)
    T, k, H, E = 37, 3, 512, 8
    cfg = gb.make_config(T, H, 128, E, k, act=act, w="bf16" if act == "bf16" else "f32")
    y = rng.standard_normal((T * k, H)).astype(np.float32)
    ysh = rng.standard_normal((T, H)).astype(np.float32)
    w = rng.random((T, k)).astype(np.float32)
    pp = rng.permutation(T * k).astype(np.int32)
    dt = torch.float32 if act == "f32" else torch.bfloat16
    yd, yshd = torch.from_numpy(y).cuda().to(dt), torch.from_numpy(ysh).cuda().to(dt)
    out = torch.empty((T, H), dtype=dt, device="cuda")
    gb.moe_combine(cfg, yd, torch.from_numpy(w).cuda(), torch.from_numpy(pp).cuda(), yshd, out)
    torch.cuda.synchronize()
    ref = oracle.combine(act_np(yd), w.astype(np.float64), pp.reshape(T, k), act_np(yshd))
    tol = 1e-6 if act == "f32" else 8e-3
    assert rel_err(act_np(out), ref) <= tol


def test_hostio_equals_device_path():
    wl, inp, dev, ref = case(2)
    cfg = config(wl)
    ws = workspace(cfg)
    out_dev, _, _ = _forward(wl, dev, "auto")
    x_host = dev["x"].cpu().pin_memory()
    out_host = torch.empty((wl.T, wl.H), dtype=dev["x"].dtype).pin_memory()
    gb.moe_forward_hostio(cfg, x_host, dev["w_router"], dev["logit_bias"], dev["select_bias"],
                          wbundle(dev["experts"]), None, out_host, ws)
    torch.cuda.synchronize()
    assert torch.equal(out_host, out_dev.cpu())


def test_forward_is_deterministic():
    wl, inp, dev, ref = case(2)
    a, _, _ = _forward(wl, dev, "auto")
    b, _, _ = _forward(wl, dev, "auto")
    assert torch.equal(a, b)
