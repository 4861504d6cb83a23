"""Chooses the logit offsets of the skewed-load int4 workload and writes them
to zipf_bias.json.

The workload asks for gate logits offset so that expert load is Zipf-like with
the hottest expert carrying about 20x the tokens of the coldest. Offsets take
the Zipf form b_e = -c * ln(e + 1) (expert 0 hottest); c is found by bisection
on the seeded inputs so that max/min of the per-expert pair counts is 20.

This is input-recipe tuning, not part of the layer: it scores tokens with a
plain fp64 matrix product and numpy's top-k, which may differ from the layer's
fp32 routing on a handful of near-ties. That moves a count by one, not the
ratio. Run: python -m synth.calibrate_zipf
"""
import json
import os

import numpy as np

import synth


def counts_for(logits: np.ndarray, bias: np.ndarray, k: int) -> np.ndarray:
    l = logits + bias[None, :]
    top = np.argsort(-l, axis=1, kind="stable")[:, :k]
    return np.bincount(top.ravel(), minlength=logits.shape[1])


def main(target: float = 20.0) -> None:
    w = synth.WORKLOADS[5]
    x = synth.bf16_bits_to_f32(synth.normal_bf16(w.seed, synth.TID["x"], w.x_sigma, (w.T, w.H)))
    g = synth.bf16_bits_to_f32(synth.normal_bf16(w.seed, synth.TID["w_router"], w.w_sigma, (w.E, w.H)))
    logits = x.astype(np.float64) @ g.astype(np.float64).T
    ln = np.log(np.arange(1, w.E + 1, dtype=np.float64))

    def ratio(c: float) -> float:
        n = counts_for(logits, (-c * ln).astype(np.float32).astype(np.float64), w.top_k)
        return n.max() / max(n.min(), 1)

    lo, hi = 0.0, 4.0
    for _ in range(60):
        mid = 0.5 * (lo + hi)
        if ratio(mid) < target:
            lo = mid
        else:
            hi = mid
    c = hi
    bias = (-c * ln).astype(np.float32)
    n = counts_for(logits, bias.astype(np.float64), w.top_k)
    out = {
        "workload": w.name,
        "E": w.E,
        "c": c,
        "form": "b_e = -c * ln(e + 1), rounded to fp32",
        "max_over_min_count_fp64_scoring": float(n.max() / n.min()),
        "bias_hex": [float(b).hex() for b in bias],
    }
    path = os.path.join(os.path.dirname(os.path.abspath(__file__)), "zipf_bias.json")
    with open(path, "w") as f:
        json.dump(out, f, indent=1)
    print(f"c = {c:.6f}  max/min = {n.max()}/{n.min()} = {n.max() / n.min():.2f}  -> {path}")


if __name__ == "__main__":
    main()
