"""GPU parity of the RMSNorm before the gate: bit for bit against the oracle
(it is pinned to the gate's order), and the routing and layer output that
follow from it."""
import numpy as np
import pytest
import torch

import oracle
import paper_2607_12875_gb300 as gb
import synth
from gpu_helpers import act_np, assert_close, config, to_device, tol_for, wbundle, workspace

pytestmark = pytest.mark.gpu


def raw_rows(T, H, seed, act):
    """Rows with very different scales (RMSNorm's job), as stored values:
    bf16 bit patterns, or fp32."""
    rng = np.random.default_rng(seed)
    x = (rng.standard_normal((T, H)) * np.exp(rng.uniform(-6, 6, (T, 1)))).astype(np.float32)
    x[0] = 0.0  # a zero row (eps keeps it finite)
    if act == "bf16":
        return oracle.round_bf16(x)
    return x


def as_f32(a, act):
    return (a.astype(np.uint32) << 16).view(np.float32) if act == "bf16" else a


def to_dev(a, act):
    t = torch.from_numpy(np.ascontiguousarray(a)).cuda()
    return t.view(torch.bfloat16) if act == "bf16" else t


@pytest.mark.parametrize("act", ["bf16", "f32"])
@pytest.mark.parametrize("T,H", [(77, 256), (33, 4096), (129, 7168)])
@pytest.mark.parametrize("eps", [1e-6, 1e-5])
def test_rmsnorm_is_bit_exact(T, H, eps, act):
    x = raw_rows(T, H, T + H, act)
    g = np.random.default_rng(H + 1).uniform(-1.5, 1.5, H).astype(np.float32)
    if act == "bf16":
        g = oracle.round_bf16(g)
    cfg = gb.make_config(T, H, 128, 8, 2, act=act, w=act)
    y = torch.empty((T, H), dtype=torch.bfloat16 if act == "bf16" else torch.float32, device="cuda")
    gb.moe_rmsnorm(cfg, to_dev(x, act), to_dev(g, act), eps, y)
    torch.cuda.synchronize()
    ref = oracle.rmsnorm(as_f32(x, act), as_f32(g[None], act)[0], eps)
    got = y.view(torch.int16).cpu().numpy().view(np.uint16) if act == "bf16" else y.cpu().numpy()
    want = oracle.round_bf16(ref) if act == "bf16" else ref
    mism = np.argwhere(got.view(np.uint32 if act == "f32" else np.uint16) !=
                       want.view(np.uint32 if act == "f32" else np.uint16))
    assert mism.size == 0, f"{len(mism)} mismatches, first at {mism[:3].tolist()}"


def normed_case(wid, T):
    wl = synth.WORKLOADS[wid].replace(T=T)
    inp = synth.make_inputs(wl)
    gamma = oracle.round_bf16(np.random.default_rng(wid).uniform(0.5, 1.5, wl.H).astype(np.float32))
    xn = oracle.round_bf16(oracle.rmsnorm(as_f32(inp["x"], "bf16"), as_f32(gamma[None], "bf16")[0], 1e-6))
    dev = to_device(wl, inp)
    cfg = config(wl)
    x_norm = torch.empty_like(dev["x"])
    gb.moe_rmsnorm(cfg, dev["x"], to_dev(gamma, "bf16"), 1e-6, x_norm)
    return wl, inp, xn, dev, cfg, x_norm


@pytest.mark.parametrize("wid", [3, 4])
def test_routing_after_rmsnorm_is_bit_exact(wid):
    """The workload's x taken as the un-normalised input: RMSNorm then the
    gate (its AUTO route) on the GPU choose exactly what the oracle's RMSNorm
    then gate choose (softmax; sigmoid group-limited)."""
    wl, inp, xn, dev, cfg, x_norm = normed_case(wid, 512)
    ws = workspace(cfg)
    ids = torch.empty((wl.T, wl.top_k), dtype=torch.int32, device="cuda")
    w = torch.empty((wl.T, wl.top_k), dtype=torch.float32, device="cuda")
    gb.moe_route(cfg, x_norm, dev["w_router"], dev["logit_bias"], dev["select_bias"], ids, w, ws)
    torch.cuda.synchronize()
    assert np.array_equal(x_norm.view(torch.int16).cpu().numpy().view(np.uint16), xn)
    logits = oracle.gate_logits(as_f32(xn, "bf16"), as_f32(inp["w_router"], "bf16"), inp["logit_bias"])
    ref_ids, _ = oracle.route(logits, wl.top_k, wl.score, wl.renormalize, wl.n_group, wl.topk_group,
                              wl.routed_scale, inp["select_bias"])
    assert np.array_equal(ids.cpu().numpy(), ref_ids)


def test_layer_after_rmsnorm_matches_the_oracle():
    """RMSNorm then the whole layer (prefill shape, 256 tokens) against the
    oracle's RMSNorm then layer, on a sample of tokens."""
    wl, inp, xn, dev, cfg, x_norm = normed_case(3, 256)
    ws = workspace(cfg)
    out = torch.empty((wl.T, wl.H), dtype=torch.bfloat16, device="cuda")
    ids = torch.empty((wl.T, wl.top_k), dtype=torch.int32, device="cuda")
    gb.moe_forward(cfg, x_norm, dev["w_router"], dev["logit_bias"], dev["select_bias"], wbundle(dev["experts"]),
                   wbundle(dev["shared"]), out, ws, topk_ids=ids)
    torch.cuda.synchronize()
    assert gb.moe_device_status(ws) == gb.OK
    ref = oracle.forward(wl, dict(inp, x=xn), rows=np.arange(0, wl.T, 5))
    assert np.array_equal(ids.cpu().numpy(), ref["topk_ids"])
    assert_close(act_np(out)[ref["rows"]], ref["out"], tol_for(wl))
