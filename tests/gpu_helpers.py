"""Shared pieces of the GPU parity tests: moving synth inputs to the device,
building the C-ABI config of a workload, comparing against the oracle."""
from __future__ import annotations

import numpy as np
import torch

import paper_2607_12875_gb300 as gb
import synth

TOL = {"f32": 1e-5, "bf16": 2e-2, "fp8_b128": 5e-2, "int4_g128": 5e-2}


def tol_for(wl) -> float:
    """Output tolerance of a workload: 1e-5 for fp32, 2e-2 for bf16, 5e-2 for fp8/int4 weights."""
    if wl.wq in ("fp8_b128", "int4_g128"):
        return TOL[wl.wq]
    return TOL["f32"] if wl.act == "f32" and wl.wq == "f32" else TOL["bf16"]


def dev_act(a: np.ndarray, act: str, device="cuda") -> torch.Tensor:
    if act == "f32":
        return torch.from_numpy(np.ascontiguousarray(a)).to(device)
    return torch.from_numpy(np.ascontiguousarray(a).view(np.int16)).to(device).view(torch.bfloat16)


def dev_weights(store: dict, wq: str, device="cuda") -> dict:
    out = {}
    for k, v in store.items():
        if k.startswith("w_"):
            if wq == "f32":
                out[k] = torch.from_numpy(v).to(device)
            elif wq == "bf16":
                out[k] = torch.from_numpy(v.view(np.int16)).to(device).view(torch.bfloat16)
            else:
                out[k] = torch.from_numpy(v).to(device)
        else:  # scales
            if wq == "fp8_b128":
                out[k] = torch.from_numpy(v).to(device)
            else:
                out[k] = torch.from_numpy(v.view(np.int16)).to(device).view(torch.bfloat16)
    return out


def to_device(wl, inputs: dict, device="cuda") -> dict:
    d = {
        "x": dev_act(inputs["x"], wl.act, device),
        "w_router": dev_act(inputs["w_router"], wl.act, device),
        "logit_bias": None if inputs["logit_bias"] is None else torch.from_numpy(inputs["logit_bias"]).to(device),
        "select_bias": None if inputs["select_bias"] is None else torch.from_numpy(inputs["select_bias"]).to(device),
        "experts": dev_weights(inputs["experts"], wl.wq, device),
        "shared": dev_weights(inputs["shared"], wl.wq, device) if wl.has_shared else None,
    }
    return d


def wbundle(ws: dict | None):
    if ws is None:
        return None
    return gb.weights(ws["w_gate"], ws["w_up"], ws["w_down"], ws.get("s_gate"), ws.get("s_up"), ws.get("s_down"))


def config(wl, route="auto", T=None):
    return gb.make_config(wl.T if T is None else T, wl.H, wl.I, wl.E, wl.top_k, score=wl.score,
                          renormalize=wl.renormalize, n_group=wl.n_group, topk_group=wl.topk_group,
                          routed_scale=wl.routed_scale, act=wl.act, w=wl.wq, has_shared=wl.has_shared,
                          I_shared=wl.I_shared, ffn_route=route)


def workspace(cfg, device="cuda") -> torch.Tensor:
    n = gb.workspace_size(cfg)
    assert n > 0
    return torch.empty(n, dtype=torch.uint8, device=device)


def act_np(t: torch.Tensor) -> np.ndarray:
    """Device activations -> fp64 numpy."""
    return t.float().cpu().numpy().astype(np.float64)


def rel_err(got: np.ndarray, ref: np.ndarray) -> float:
    """max |got - ref| / max |ref| over the compared rows."""
    return float(np.max(np.abs(got - ref)) / max(np.max(np.abs(ref)), 1e-30))


def sample_rows(wl, ids: np.ndarray, n_random: int, per_extreme: int, seed: int = 0) -> np.ndarray:
    """Seeded token subset: random tokens, the first and last token, and up to
    per_extreme tokens routed to the hottest and to the coldest active expert."""
    rng = np.random.default_rng(seed)
    T = ids.shape[0]
    rows = set(rng.choice(T, size=min(n_random, T), replace=False).tolist()) | {0, T - 1}
    counts = np.bincount(ids.ravel(), minlength=wl.E)
    active = np.nonzero(counts)[0]
    for e in (active[np.argmax(counts[active])], active[np.argmin(counts[active])]):
        toks = np.nonzero((ids == e).any(axis=1))[0]
        rows |= set(rng.choice(toks, size=min(per_extreme, len(toks)), replace=False).tolist())
    return np.array(sorted(rows), dtype=np.int64)
