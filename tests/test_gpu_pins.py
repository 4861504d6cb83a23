"""GPU pins of the fixed fp32 exponential and sigmoid that decide the
sigmoid-scored expert choice: their bits, read through moe_route, against
the oracle's over a dense sweep of fp32 logits and over special values.

moe_route with fp32 activations, score = sigmoid, renormalize = 0,
routed_scale = 1, top_k = E and one group returns, for every expert, the
weight s = sigmoid(l) of its logit exactly (a product by 1.0). A token whose
x row is c at one position (zero elsewhere) against an all-ones router row
has the logit c exactly in the fixed order (one fused multiply-add by 1.0,
the rest adds of zeros), and logit_bias b_e then makes l = fp32(c + b_e):
the test knows every logit bit for bit without reading the GPU's logits."""
import numpy as np
import pytest
import torch

import oracle
import paper_2607_12875_gb300 as gb
from gpu_helpers import workspace

pytestmark = pytest.mark.gpu

E, H = 32, 256


def route_all(x: torch.Tensor, w_router: torch.Tensor, bias: torch.Tensor):
    T = x.shape[0]
    cfg = gb.make_config(T, H, 128, E, E, score="sigmoid", renormalize=False, n_group=1, topk_group=1,
                         routed_scale=1.0, act="f32", w="f32")
    ws = workspace(cfg)
    ids = torch.empty((T, E), dtype=torch.int32, device="cuda")
    w = torch.empty((T, E), dtype=torch.float32, device="cuda")
    gb.moe_route(cfg, x, w_router, bias, None, ids, w, ws)
    torch.cuda.synchronize()
    return ids.cpu().numpy(), w.cpu().numpy()


def test_pinned_sigmoid_sweep_is_bit_exact():
    T = 1 << 17  # 2^17 tokens x 32 experts = 2^22 logits
    lo, hi = -104.0, 89.0
    c = (lo + (hi - lo) * np.arange(T, dtype=np.float64) / T).astype(np.float32)
    b = ((hi - lo) / T / E * np.arange(E)).astype(np.float32)
    logits = c[:, None] + b[None, :]  # fp32 adds, rounded as the GPU's
    assert logits.dtype == np.float32
    assert len(np.unique(logits)) > 0.99 * T * E
    x = torch.zeros((T, H), dtype=torch.float32, device="cuda")
    x[torch.arange(T, device="cuda"), torch.arange(T, device="cuda") % H] = torch.from_numpy(c).cuda()
    ones = torch.ones((E, H), dtype=torch.float32, device="cuda")
    ids, w = route_all(x, ones, torch.from_numpy(b).cuda())
    ref = oracle.sigmoid(logits)
    got = w[np.arange(T)[:, None], np.argsort(ids, axis=1)]  # weight of expert e in column e
    bad = np.nonzero(got.view(np.uint32) != ref.view(np.uint32))
    assert bad[0].size == 0, (f"{bad[0].size} of {T * E} sigmoid values differ, first logits "
                              f"{logits[bad][:4].tolist()}: gpu {got[bad][:4].tolist()} oracle {ref[bad][:4].tolist()}")
    ref_ids, ref_w = oracle.route(logits, E, "sigmoid", False, 1, 1, 1.0)
    assert np.array_equal(ids, ref_ids)
    assert np.array_equal(w, ref_w.astype(np.float32))


def test_pinned_sigmoid_special_values():
    specials = np.array([0.0, -0.0, 1e-45, -1e-45, 1e-38, -1e-38, 86.0, -86.0, 88.0, -88.0, 88.7, -88.7,
                         104.0, -104.0, np.inf, -np.inf, np.nan, 17.0, 16.635532, -16.635532, 0.5, -0.5,
                         3.4028235e38, -3.4028235e38, 1.0, -1.0, 2.0, -2.0, 15.9, -15.9, 40.0, -40.0],
                        dtype=np.float32)
    assert specials.size == E
    x = torch.zeros((1, H), dtype=torch.float32, device="cuda")
    x[0, 0] = 1.0
    wr = torch.zeros((E, H), dtype=torch.float32, device="cuda")
    wr[:, 0] = torch.from_numpy(specials).cuda()
    ids, w = route_all(x, wr, None)
    logits = (np.float32(0.0) + specials)[None, :]  # one fma by 1.0 onto +0: -0 becomes +0
    ref = oracle.sigmoid(logits)[0]
    got = w[0, np.argsort(ids[0])]
    nan = np.isnan(ref)
    assert np.array_equal(np.isnan(got), nan)
    assert np.array_equal(got[~nan].view(np.uint32), ref[~nan].view(np.uint32))
    ref_ids, _ = oracle.route(logits, E, "sigmoid", False, 1, 1, 1.0)
    assert np.array_equal(ids, ref_ids)  # the NaN logit ranks last (as -inf, lower index first)
