"""Shared pieces of the GPU parity tests: moving synth inputs to the device,
building the C-ABI config of a workload, comparing against the oracle."""
from __future__ import annotations

import numpy as np
import torch

import paper_2607_12875_gb300 as gb
import synth

TOL = {"f32": 1e-5, "bf16": 2e-2, "fp8_b128": 5e-2, "int4_g128": 5e-2, "mxfp4": 2e-2}


def tol_for(wl) -> float:
    """Output tolerance of a workload: 1e-5 for fp32, 2e-2 for bf16, 5e-2 for
    fp8/int4 weights; MXFP4 weights decode exactly (to bf16 and fp32), so they
    take the bf16 bound."""
    if wl.wq in ("fp8_b128", "int4_g128", "mxfp4"):
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
        else:  # scales: fp32 (fp8), E8M0 bytes (MXFP4), bf16 bits (int4)
            if wq in ("fp8_b128", "mxfp4"):
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


ROW_FLOOR = 0.05  # per-row errors are taken relative to max(|ref row|, ROW_FLOOR * max |ref|)


def error_report(got: np.ndarray, ref: np.ndarray) -> dict:
    """Errors of got against ref over rows (the last axis is a row's elements):
    the infinity-norm relative error (the tolerance metric), per-row relative
    errors max|got_r - ref_r| / max(max|ref_r|, ROW_FLOOR * max|ref|), and the
    largest elementwise relative error with the same floor."""
    got = got.reshape(-1, got.shape[-1])
    ref = ref.reshape(-1, ref.shape[-1])
    gmax = max(float(np.max(np.abs(ref))), 1e-30)
    diff = np.abs(got - ref)
    row_scale = np.maximum(np.max(np.abs(ref), axis=1), ROW_FLOOR * gmax)
    row_err = np.max(diff, axis=1) / row_scale
    elem_err = diff / np.maximum(np.abs(ref), ROW_FLOOR * gmax)
    worst = np.argsort(row_err)[::-1][:3]
    return {"inf": float(np.max(diff) / gmax), "row_max": float(np.max(row_err)),
            "row_median": float(np.median(row_err)), "worst_rows": [(int(r), float(row_err[r])) for r in worst],
            "elem_max": float(np.max(elem_err)), "rows": int(got.shape[0])}


def assert_close(got: np.ndarray, ref: np.ndarray, tol: float, what: str = "output") -> dict:
    """The infinity-norm relative error and every per-row relative error
    within tol; the report (worst rows, elementwise error) is the message."""
    rep = error_report(got, ref)
    assert rep["inf"] <= tol and rep["row_max"] <= tol, f"{what}: {rep} (tol {tol:.0e})"
    return rep


def tiles_covered(ids_rows: np.ndarray, rows: np.ndarray, counts: np.ndarray, sorted_pair: np.ndarray,
                  offsets: np.ndarray, bm: int = 128) -> tuple:
    """(covered, total): how many of the (expert, bm-row tile) pairs of the
    grouped GEMM hold at least one pair of the compared tokens `rows`."""
    k = ids_rows.shape[1]
    want = set(rows.tolist())
    total, covered = 0, 0
    for e in np.nonzero(counts)[0]:
        for m in range(0, int(counts[e]), bm):
            total += 1
            seg = sorted_pair[offsets[e] + m: offsets[e] + min(m + bm, int(counts[e]))] // k
            covered += bool(want.intersection(seg.tolist()))
    return covered, total
