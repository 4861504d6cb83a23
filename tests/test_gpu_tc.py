"""GPU parity of the tensor-core (tcgen05) grouped-GEMM routes against the
oracle on small ragged problems (the full-size workloads are compared token
by token in test_gpu_layer.py), and the decode-once route (TC_DEQUANT)
against the in-GEMM decode."""
import os

import numpy as np
import pytest
import torch

import oracle
import paper_2607_12875_gb300 as gb
import synth
from gpu_helpers import act_np, assert_close, config, to_device, tol_for, wbundle, workspace

pytestmark = pytest.mark.gpu

BASE = synth.WORKLOADS[1].replace(act="bf16", wq="bf16")


def forward(wl, dev, route):
    """moe_forward of wl on the given FFN route; returns (out, topk_ids)."""
    cfg = config(wl, route)
    ws = workspace(cfg)
    out = torch.empty((wl.T, wl.H), dtype=torch.bfloat16, device="cuda")
    ids = torch.empty((wl.T, wl.top_k), dtype=torch.int32, device="cuda")
    gb.moe_forward(cfg, dev["x"], dev["w_router"], dev["logit_bias"], dev["select_bias"], wbundle(dev["experts"]),
                   wbundle(dev["shared"]), out, ws, topk_ids=ids)
    torch.cuda.synchronize()
    assert gb.moe_device_status(ws) == gb.OK
    return out, ids


def pair_route(wq):
    """The CTA-pair route of a weight format: pairs multiply bf16 B tiles, so
    quantised weights take the decode-once pair route."""
    return "tc_pair" if wq == "bf16" else "tc_pair_dequant"


@pytest.mark.parametrize("pair", [False, True])
@pytest.mark.parametrize("wq", ["bf16", "fp8_b128", "int4_g128", "mxfp4"])
@pytest.mark.parametrize("T,E,k,H,I", [(200, 4, 2, 512, 256), (1000, 4, 2, 256, 384), (333, 16, 3, 768, 128)])
def test_tc_small_ragged(T, E, k, H, I, wq, pair):
    wl = BASE.replace(T=T, E=E, top_k=k, H=H, I=I, seed=T + E, wq=wq)
    inp = synth.make_inputs(wl)
    dev = to_device(wl, inp)
    out, ids = forward(wl, dev, pair_route(wq) if pair else "tc")
    ref = oracle.forward(wl, inp)
    assert np.array_equal(ids.cpu().numpy(), ref["topk_ids"])
    assert_close(act_np(out), ref["out"], tol_for(wl))


@pytest.mark.parametrize("wq", ["bf16", "int4_g128"])
@pytest.mark.parametrize("T,E,k,H,I", [(1000, 4, 2, 256, 384), (333, 16, 3, 768, 128), (77, 3, 3, 512, 256)])
def test_pair_route_equals_single_cta_route(T, E, k, H, I, wq):
    """A CTA pair's 256-row MMA sums each output element over the same k
    slices in the same order as the one-CTA 128-row MMA, and the decoded
    operands are the same, so the two routes give bit-identical outputs
    (expert tails of 1..255 rows, including pairs whose odd CTA has none)."""
    wl = BASE.replace(T=T, E=E, top_k=k, H=H, I=I, seed=T + 3 * E, wq=wq)
    inp = synth.make_inputs(wl)
    dev = to_device(wl, inp)
    out1, ids1 = forward(wl, dev, "tc" if wq == "bf16" else "tc_dequant")
    out2, ids2 = forward(wl, dev, pair_route(wq))
    assert torch.equal(ids1, ids2)
    assert torch.equal(out1.view(torch.int16), out2.view(torch.int16))


def test_tc_sigmoid_grouped_fp8_with_shared_expert():
    wl = BASE.replace(T=300, E=16, top_k=4, H=512, I=256, wq="fp8_b128", seed=31, score="sigmoid", routed_scale=2.5,
                      n_group=4, topk_group=2, has_shared=True, I_shared=384, select_bias_sigma=0.01)
    inp = synth.make_inputs(wl)
    dev = to_device(wl, inp)
    out, ids = forward(wl, dev, "tc")
    ref = oracle.forward(wl, inp)
    assert np.array_equal(ids.cpu().numpy(), ref["topk_ids"])
    assert_close(act_np(out), ref["out"], tol_for(wl))


@pytest.mark.parametrize("wq", ["fp8_b128", "int4_g128", "mxfp4"])
@pytest.mark.parametrize("T,E,k,H,I", [(200, 4, 2, 512, 256), (333, 16, 3, 768, 128)])
def test_dequant_route_equals_in_gemm_decode(T, E, k, H, I, wq):
    """Decoding the weights once into a bf16 copy gives the GEMM the same bf16
    operands as decoding them inside it, so the outputs are bit-identical."""
    wl = BASE.replace(T=T, E=E, top_k=k, H=H, I=I, seed=T + 2 * E, wq=wq)
    inp = synth.make_inputs(wl)
    dev = to_device(wl, inp)
    out_tc, ids_tc = forward(wl, dev, "tc")
    out_dq, ids_dq = forward(wl, dev, "tc_dequant")
    assert torch.equal(ids_tc, ids_dq)
    assert torch.equal(out_tc.view(torch.int16), out_dq.view(torch.int16))
    out_pq, _ = forward(wl, dev, "tc_pair_dequant")  # the same on CTA pairs
    assert torch.equal(out_tc.view(torch.int16), out_pq.view(torch.int16))
    ref = oracle.forward(wl, inp)
    assert_close(act_np(out_dq), ref["out"], tol_for(wl))


def test_dequant_route_with_shared_expert_and_inactive_experts():
    """Only active experts are decoded; the shared expert has its own copy."""
    wl = BASE.replace(T=60, E=64, top_k=2, H=512, I=256, wq="int4_g128", seed=57, has_shared=True, I_shared=384,
                      zipf=True)
    inp = synth.make_inputs(wl)
    dev = to_device(wl, inp)
    out, ids = forward(wl, dev, "tc_dequant")
    ref = oracle.forward(wl, inp)
    assert (ref["counts"] == 0).any()
    assert np.array_equal(ids.cpu().numpy(), ref["topk_ids"])
    assert_close(act_np(out), ref["out"], tol_for(wl))


def test_auto_route_choice():
    """AUTO: streaming for decode; fp8 weights on the fp8 tensor-core route;
    int4/MXFP4 decoded in the GEMM for few rows per expert, decoded once for
    many; CTA pairs for deep experts (>= 1024 rows each)."""
    assert gb.ffn_route(config(synth.WORKLOADS[2])) == "stream"
    assert gb.ffn_route(config(synth.WORKLOADS[3])) == "tc"
    assert gb.ffn_route(config(synth.WORKLOADS[4])) == "tc_fp8"
    assert gb.ffn_route(config(synth.WORKLOADS[4]), shared=True) == "tc_fp8"
    assert gb.ffn_route(config(synth.WORKLOADS[5])) == "tc_pair_dequant"  # 1536 rows per expert: CTA pairs
    assert gb.ffn_route(config(synth.WORKLOADS[6])) == "tc"
    assert gb.ffn_route(config(synth.WORKLOADS[6]), shared=True) == "tc_pair_dequant"


@pytest.mark.parametrize("pair", [False, True])
@pytest.mark.parametrize("wq", ["bf16", "int4_g128"])
def test_bounded_wait_timeout_is_reported_and_the_next_call_is_clean(wq, pair, monkeypatch):
    """With the tensor-core kernels' wait limit lowered to 0 ns, a wait that
    is not over at once gives up (the first accumulator alone takes tens of
    microseconds): the kernel stops, drains what it issued, frees its TMEM and
    sets the error word, which moe_device_status reports as
    GBMOE_EDEVICE_TIMEOUT. The context stays usable: the next call with the
    normal limit is clean and matches the oracle."""
    wl = BASE.replace(T=333, E=16, top_k=3, H=768, I=128, seed=401, wq=wq)
    inp = synth.make_inputs(wl)
    dev = to_device(wl, inp)
    cfg = config(wl, pair_route(wq) if pair else "tc")
    ws = workspace(cfg)
    out = torch.empty((wl.T, wl.H), dtype=torch.bfloat16, device="cuda")
    args = (cfg, dev["x"], dev["w_router"], dev["logit_bias"], dev["select_bias"], wbundle(dev["experts"]), None,
            out, ws)
    monkeypatch.setenv("GBMOE_TC_WAIT_LIMIT_NS", "0")
    gb.moe_forward(*args)
    assert gb.moe_device_status(ws) == gb.EDEVICE_TIMEOUT
    assert gb.moe_device_status(ws) == gb.OK  # read and cleared
    monkeypatch.delenv("GBMOE_TC_WAIT_LIMIT_NS")
    gb.moe_forward(*args)
    assert gb.moe_device_status(ws) == gb.OK
    ref = oracle.forward(wl, inp)
    assert_close(act_np(out), ref["out"], tol_for(wl))


# fp8 tensor-core route (kind::f8f6f4): fp8 weights as stored, activations
# quantised to e4m3 per 1x128 block; against the oracle with exact
# activations, within the fp8 bound (5e-2) and per row
@pytest.mark.parametrize("T,E,k,H,I", [(200, 4, 2, 512, 256), (1000, 4, 2, 256, 384), (333, 16, 3, 768, 128),
                                       (64, 8, 8, 1024, 512)])
def test_tc_fp8_route_small_ragged(T, E, k, H, I):
    wl = BASE.replace(T=T, E=E, top_k=k, H=H, I=I, seed=T + 3 * E, wq="fp8_b128")
    inp = synth.make_inputs(wl)
    dev = to_device(wl, inp)
    out, ids = forward(wl, dev, "tc_fp8")
    ref = oracle.forward(wl, inp)
    assert np.array_equal(ids.cpu().numpy(), ref["topk_ids"])
    assert_close(act_np(out), ref["out"], tol_for(wl))


def test_tc_fp8_route_with_shared_expert_and_timeout():
    """Sigmoid group routing with a shared expert on the fp8 route; then its
    bounded waits run out under a 0 ns limit and the next call is clean."""
    wl = BASE.replace(T=300, E=16, top_k=4, H=512, I=256, wq="fp8_b128", seed=33, score="sigmoid",
                      routed_scale=2.5, n_group=4, topk_group=2, has_shared=True, I_shared=384,
                      select_bias_sigma=0.01)
    inp = synth.make_inputs(wl)
    dev = to_device(wl, inp)
    out, ids = forward(wl, dev, "tc_fp8")
    ref = oracle.forward(wl, inp)
    assert np.array_equal(ids.cpu().numpy(), ref["topk_ids"])
    assert_close(act_np(out), ref["out"], tol_for(wl))
    cfg = config(wl, "tc_fp8")
    ws = workspace(cfg)
    os.environ["GBMOE_TC_WAIT_LIMIT_NS"] = "0"
    try:
        gb.moe_forward(cfg, dev["x"], dev["w_router"], dev["logit_bias"], dev["select_bias"],
                       wbundle(dev["experts"]), wbundle(dev["shared"]), out, ws)
        assert gb.moe_device_status(ws) == gb.EDEVICE_TIMEOUT
    finally:
        del os.environ["GBMOE_TC_WAIT_LIMIT_NS"]
    out2, _ = forward(wl, dev, "tc_fp8")
    assert_close(act_np(out2), ref["out"], tol_for(wl))



@pytest.mark.parametrize("pair", [False, True])
@pytest.mark.parametrize("wq", ["bf16", "int4_g128"])
def test_fused_weight_sum_small_with_shared_expert(wq, pair):
    """Fused Weight Sum on a ragged problem with a shared expert (its row is
    added by the warp that completes each token), on one-CTA and CTA-pair
    GEMMs."""
    wl = BASE.replace(T=333, E=16, top_k=3, H=768, I=128, seed=211, wq=wq, has_shared=True, I_shared=256)
    inp = synth.make_inputs(wl)
    dev = to_device(wl, inp)
    cfg = config(wl, pair_route(wq) if pair else "tc")
    cfg.combine_route = gb.COMBINE_FUSED
    ws = workspace(cfg)
    out = torch.empty((wl.T, wl.H), dtype=torch.bfloat16, device="cuda")
    gb.moe_forward(cfg, dev["x"], dev["w_router"], dev["logit_bias"], dev["select_bias"], wbundle(dev["experts"]),
                   wbundle(dev["shared"]), out, ws)
    torch.cuda.synchronize()
    assert gb.moe_device_status(ws) == gb.OK
    ref = oracle.forward(wl, inp)
    assert_close(act_np(out), ref["out"], tol_for(wl))
