"""GPU checks of pairs whose expert id is out of range: moe_permute drops
them (not counted, pair_pos -1, sorted positions past the last kept pair -1),
and moe_grouped_ffn + moe_combine on those outputs give each token the sum
over its kept slots only. Both permutation paths (one CTA up to 1024 pairs,
three kernels above) are covered."""
import numpy as np
import pytest
import torch

import oracle
import synth
import paper_2607_12875_gb300 as gb
from gpu_helpers import act_np, assert_close, config, to_device, tol_for, wbundle, workspace

pytestmark = pytest.mark.gpu


def expected_permutation(ids: np.ndarray, E: int):
    """The oracle's stable sort with dropped pairs sent to an extra expert E:
    its first offsets[E] sorted positions are the kept pairs in order."""
    flat = ids.ravel().copy()
    keep = (flat >= 0) & (flat < E)
    flat[~keep] = E
    counts, offsets, sp, pp = oracle.permute(flat, E + 1)
    return keep, counts[:E], offsets[:E + 1], sp, pp


def plant_drops(ids: np.ndarray, E: int, seed: int) -> np.ndarray:
    rng = np.random.default_rng(seed)
    out = ids.copy()
    mask = rng.random(out.shape) < 0.07
    out[mask] = rng.choice(np.array([-1, -7, E, E + 3, 1 << 30]), size=int(mask.sum()))
    return out


@pytest.mark.parametrize("T,k,E", [(100, 4, 16), (700, 6, 64)])  # P = 400 (one CTA) and 4200 (three kernels)
def test_permute_drops_out_of_range_ids(T, k, E):
    rng = np.random.default_rng(T)
    ids = plant_drops(rng.integers(0, E, size=(T, k)).astype(np.int32), E, T + 1)
    keep, counts_ref, offsets_ref, sp_ref, pp_ref = expected_permutation(ids, E)
    P, kept = T * k, int(keep.sum())
    assert 0 < kept < P
    cfg = gb.make_config(T, 256, 128, E, k)
    ws = workspace(cfg)
    counts = torch.empty(E, dtype=torch.int32, device="cuda")
    offsets = torch.empty(E + 1, dtype=torch.int32, device="cuda")
    sp = torch.full((P,), 12345, dtype=torch.int32, device="cuda")
    pp = torch.full((P,), 12345, dtype=torch.int32, device="cuda")
    gb.moe_permute(cfg, torch.from_numpy(ids).cuda(), counts, offsets, sp, pp, ws)
    torch.cuda.synchronize()
    assert np.array_equal(counts.cpu().numpy(), counts_ref)
    assert np.array_equal(offsets.cpu().numpy(), offsets_ref) and offsets_ref[E] == kept
    sp, pp = sp.cpu().numpy(), pp.cpu().numpy()
    assert np.array_equal(sp[:kept], sp_ref[:kept])
    assert (sp[kept:] == -1).all()
    assert np.array_equal(pp[keep], pp_ref[keep])
    assert (pp[~keep] == -1).all()


@pytest.mark.parametrize("route", ["tc", "tc_pair", "stream", "simt"])
def test_ffn_and_combine_skip_dropped_pairs(route):
    wl = synth.WORKLOADS[1].replace(T=150, E=8, top_k=3, H=512, I=256, act="bf16", wq="bf16", seed=61)
    inp = synth.make_inputs(wl)
    dev = to_device(wl, inp)
    ref = oracle.forward(wl, inp)
    ids = plant_drops(ref["topk_ids"], wl.E, 5)
    keep = ((ids >= 0) & (ids < wl.E))
    # expected: each token's kept slots, weight times that expert's oracle output
    w_ref = ref["topk_w"] * keep
    out_ref = np.einsum("tj,tjh->th", w_ref, ref["y"] * keep[:, :, None])
    cfg = config(wl, route)
    ws = workspace(cfg)
    T, k, E, P = wl.T, wl.top_k, wl.E, wl.P
    counts = torch.empty(E, dtype=torch.int32, device="cuda")
    offsets = torch.empty(E + 1, dtype=torch.int32, device="cuda")
    sp = torch.empty(P, dtype=torch.int32, device="cuda")
    pp = torch.empty(P, dtype=torch.int32, device="cuda")
    gb.moe_permute(cfg, torch.from_numpy(ids).cuda(), counts, offsets, sp, pp, ws)
    y = torch.empty((P, wl.H), dtype=torch.bfloat16, device="cuda")
    gb.moe_grouped_ffn(cfg, dev["x"], counts, offsets, sp, wbundle(dev["experts"]), y, ws)
    out = torch.empty((T, wl.H), dtype=torch.bfloat16, device="cuda")
    w = torch.from_numpy(ref["topk_w"].astype(np.float32)).cuda()
    gb.moe_combine(cfg, y, w, pp, None, out)
    torch.cuda.synchronize()
    assert_close(act_np(out), out_ref, tol_for(wl), f"route {route} with dropped pairs")
