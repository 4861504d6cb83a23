"""GPU parity of the tensor-core (tcgen05) grouped-GEMM route against the
oracle: small ragged problems first, then the prefill-shaped workload."""
import numpy as np
import pytest
import torch

import oracle
import paper_2607_12875_gb300 as gb
import synth
from gpu_helpers import act_np, config, rel_err, sample_rows, to_device, tol_for, wbundle, workspace

pytestmark = pytest.mark.gpu

BASE = synth.WORKLOADS[1].replace(act="bf16", wq="bf16")


def forward(wl, dev, route):
    cfg = config(wl, route)
    ws = workspace(cfg)
    out = torch.empty((wl.T, wl.H), dtype=torch.bfloat16, device="cuda")
    ids = torch.empty((wl.T, wl.top_k), dtype=torch.int32, device="cuda")
    gb.moe_forward(cfg, dev["x"], dev["w_router"], dev["logit_bias"], dev["select_bias"], wbundle(dev["experts"]),
                   wbundle(dev["shared"]), out, ws, topk_ids=ids)
    torch.cuda.synchronize()
    assert gb.moe_device_status(ws) == gb.OK
    return out, ids


@pytest.mark.parametrize("wq", ["bf16", "fp8_b128", "int4_g128"])
@pytest.mark.parametrize("T,E,k,H,I", [(200, 4, 2, 512, 256), (1000, 4, 2, 256, 384), (333, 16, 3, 768, 128)])
def test_tc_small_ragged(T, E, k, H, I, wq):
    wl = BASE.replace(T=T, E=E, top_k=k, H=H, I=I, seed=T + E, wq=wq)
    inp = synth.make_inputs(wl)
    dev = to_device(wl, inp)
    out, ids = forward(wl, dev, "tc")
    ref = oracle.forward(wl, inp)
    assert np.array_equal(ids.cpu().numpy(), ref["topk_ids"])
    err = rel_err(act_np(out), ref["out"])
    assert err <= tol_for(wl), f"rel err {err:.3e}"


def test_tc_prefill_workload():
    wl = synth.WORKLOADS[3]
    inp = synth.make_inputs(wl)
    dev = to_device(wl, inp)
    out, ids = forward(wl, dev, "tc")
    ids = ids.cpu().numpy()
    rows = sample_rows(wl, ids, 32, 8, seed=7)
    ref = oracle.forward(wl, inp, rows=rows)
    assert np.array_equal(ids, ref["topk_ids"])
    err = rel_err(act_np(out)[rows], ref["out"])
    assert err <= tol_for(wl), f"rel err {err:.3e}"


def test_tc_sigmoid_grouped_fp8_with_shared_expert():
    wl = BASE.replace(T=300, E=16, top_k=4, H=512, I=256, wq="fp8_b128", seed=31, score="sigmoid", routed_scale=2.5,
                      n_group=4, topk_group=2, has_shared=True, I_shared=384, select_bias_sigma=0.01)
    inp = synth.make_inputs(wl)
    dev = to_device(wl, inp)
    out, ids = forward(wl, dev, "tc")
    ref = oracle.forward(wl, inp)
    assert np.array_equal(ids.cpu().numpy(), ref["topk_ids"])
    err = rel_err(act_np(out), ref["out"])
    assert err <= tol_for(wl), f"rel err {err:.3e}"
