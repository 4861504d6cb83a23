"""GPU parity: every C-ABI call of the layer against the CPU oracle on the
same seeded inputs, for the five workload shapes, the MXFP4 variant of the
DeepSeek-style layer (workload 6), and every FFN route.
Routing ids, the permutation and the counts must match bit for bit; outputs
within the workload's tolerance, as the infinity-norm relative error
max |gpu - oracle| / max |oracle| and as every row's relative error (floored,
see gpu_helpers.error_report). Every token of every workload is compared, so
every (expert, M tile) and N tile of the full-size launches is checked."""
import numpy as np
import pytest
import torch

import oracle
import paper_2607_12875_gb300 as gb
import synth
from gpu_helpers import (act_np, assert_close, config, rel_err, tiles_covered, to_device, tol_for, wbundle,
                         workspace)

pytestmark = pytest.mark.gpu

ROUTES = {1: ["simt", "stream", "auto"], 2: ["stream", "simt", "auto"], 3: ["simt", "auto", "tc", "tc_pair"],
          4: ["simt", "auto", "tc", "tc_dequant"], 5: ["simt", "auto", "tc", "tc_pair_dequant"],
          6: ["simt", "auto", "tc_dequant", "tc_pair_dequant"]}
ALL_ROUTES = ["auto", "stream", "simt", "tc", "tc_dequant", "tc_fp8", "tc_pair", "tc_pair_dequant"]


@pytest.fixture(scope="module", params=[1, 2, 3, 4, 5, 6])
def wcase(request):
    """Host inputs, device inputs and the full oracle forward of one workload.
    Module scope with parameters: pytest runs all tests of one workload
    together, so each is generated and checked by the oracle once."""
    wid = request.param
    torch.cuda.empty_cache()
    wl = synth.WORKLOADS[wid]
    inp = synth.make_inputs(wl)
    dev = to_device(wl, inp)
    ref = oracle.forward(wl, inp)  # every token
    yield dict(wid=wid, wl=wl, inp=inp, dev=dev, ref=ref)
    del dev
    torch.cuda.empty_cache()


def test_route_is_bit_exact(wcase):
    wl, dev, ref = wcase["wl"], wcase["dev"], wcase["ref"]
    cfg = config(wl)
    ws = workspace(cfg)
    ids = torch.empty((wl.T, wl.top_k), dtype=torch.int32, device="cuda")
    w = torch.empty((wl.T, wl.top_k), dtype=torch.float32, device="cuda")
    gb.moe_route(cfg, dev["x"], dev["w_router"], dev["logit_bias"], dev["select_bias"], ids, w, ws)
    torch.cuda.synchronize()
    got = ids.cpu().numpy()
    mism = np.argwhere(got != ref["topk_ids"])
    assert mism.size == 0, f"{len(mism)} routing mismatches, first at {mism[:3].tolist()}"
    # weights from tensor-core logits (the TC gate) are within ~1e-4 of the fixed-order ones
    rtol = 1e-4 if gb.gate_route(cfg) == "tc" else 2e-6
    np.testing.assert_allclose(w.cpu().numpy(), ref["topk_w"], rtol=rtol, atol=1e-7)


def test_tc_gate_equals_fixed_order_gate(wcase):
    """The tensor-core gate with its audit chooses exactly what the
    fixed-order CUDA-core gate chooses, for every token (bf16 workloads)."""
    wl, dev = wcase["wl"], wcase["dev"]
    if wl.act != "bf16":
        pytest.skip("the tensor-core gate takes bf16 activations")
    res = {}
    for g in ("simt", "tc"):
        cfg = config(wl)
        cfg.gate_route = gb.GATES[g]
        ws = workspace(cfg)
        ids = torch.empty((wl.T, wl.top_k), dtype=torch.int32, device="cuda")
        w = torch.empty((wl.T, wl.top_k), dtype=torch.float32, device="cuda")
        gb.moe_route(cfg, dev["x"], dev["w_router"], dev["logit_bias"], dev["select_bias"], ids, w, ws)
        torch.cuda.synchronize()
        res[g] = (ids.cpu().numpy(), w.cpu().numpy())
    assert np.array_equal(res["tc"][0], res["simt"][0])
    np.testing.assert_allclose(res["tc"][1], res["simt"][1], rtol=1e-4, atol=1e-7)


def test_permute_is_bit_exact(wcase):
    wl, ref = wcase["wl"], wcase["ref"]
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


@pytest.mark.parametrize("route", ALL_ROUTES)
def test_forward_matches_oracle(wcase, route):
    wid, wl, dev, ref = wcase["wid"], wcase["wl"], wcase["dev"], wcase["ref"]
    if route not in ROUTES[wid]:
        pytest.skip(f"route {route} is not exercised on workload {wid}")
    out, ids, counts = _forward(wl, dev, route)
    assert np.array_equal(ids.cpu().numpy(), ref["topk_ids"])
    assert np.array_equal(counts.cpu().numpy(), ref["counts"])
    assert len(ref["rows"]) == wl.T  # every token compared
    if gb.ffn_route(config(wl, route)) in ("tc", "tc_dequant", "tc_fp8", "tc_pair", "tc_pair_dequant"):
        cov, total = tiles_covered(ref["topk_ids"], ref["rows"], ref["counts"], ref["sorted_pair"], ref["offsets"])
        assert cov == total, f"compared tokens reach {cov} of {total} (expert, M tile) pairs"
    assert_close(act_np(out), ref["out"], tol_for(wl), f"workload {wid} route {route}")


def test_grouped_ffn_rows_match_oracle(wcase):
    """Every (token, slot) row of y_pairs against the oracle's expert output."""
    wl, dev, ref = wcase["wl"], wcase["dev"], wcase["ref"]
    cfg = config(wl)
    ws = workspace(cfg)
    P = wl.P
    t = lambda a: torch.from_numpy(np.ascontiguousarray(a)).cuda()
    y = torch.empty((P, wl.H), dtype=dev["x"].dtype, device="cuda")
    gb.moe_grouped_ffn(cfg, dev["x"], t(ref["counts"]), t(ref["offsets"]), t(ref["sorted_pair"]),
                       wbundle(dev["experts"]), y, ws)
    torch.cuda.synchronize()
    got = act_np(y)[ref["pair_pos"]].reshape(wl.T, wl.top_k, wl.H)
    assert_close(got, ref["y"], tol_for(wl), "y_pairs")


def test_shared_expert_matches_oracle(wcase):
    wl, dev, ref = wcase["wl"], wcase["dev"], wcase["ref"]
    if not wl.has_shared:
        pytest.skip("workload has no shared expert")
    cfg = config(wl)
    ws = workspace(cfg)
    ysh = torch.empty((wl.T, wl.H), dtype=dev["x"].dtype, device="cuda")
    gb.moe_shared_ffn(cfg, dev["x"], wbundle(dev["shared"]), ysh, ws)
    torch.cuda.synchronize()
    assert_close(act_np(ysh), ref["y_shared"], tol_for(wl), "shared expert")


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
    wl = synth.WORKLOADS[2]
    dev = to_device(wl, synth.make_inputs(wl))
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
    wl = synth.WORKLOADS[2]
    dev = to_device(wl, synth.make_inputs(wl))
    a, _, _ = _forward(wl, dev, "auto")
    b, _, _ = _forward(wl, dev, "auto")
    assert torch.equal(a, b)


def test_fused_weight_sum_matches_oracle(wcase):
    """The Weight Sum folded into the down GEMM's epilogue (tensor-core FFN
    routes): every token against the oracle, deterministic over two calls, and
    within rounding of the separate combine."""
    wl, dev, ref = wcase["wl"], wcase["dev"], wcase["ref"]
    route = gb.ffn_route(config(wl))
    if route not in ("tc", "tc_dequant", "tc_pair", "tc_pair_dequant"):
        pytest.skip("the fused Weight Sum runs on the bf16 tensor-core routes")
    outs = []
    for comb in ("fused", "fused", "separate"):
        cfg = config(wl)
        cfg.combine_route = gb.COMBINES[comb]
        ws = workspace(cfg)
        out = torch.empty((wl.T, wl.H), dtype=dev["x"].dtype, device="cuda")
        gb.moe_forward(cfg, dev["x"], dev["w_router"], dev["logit_bias"], dev["select_bias"],
                       wbundle(dev["experts"]), wbundle(dev["shared"]), out, ws)
        torch.cuda.synchronize()
        assert gb.moe_device_status(ws) == gb.OK
        outs.append(out)
    assert torch.equal(outs[0], outs[1])
    assert_close(act_np(outs[0]), ref["out"], tol_for(wl), "fused Weight Sum")
    assert_close(act_np(outs[0]), act_np(outs[2]), 2e-2, "fused vs separate")  # two bf16 roundings
