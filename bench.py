#!/usr/bin/env python
"""MoE layer forward throughput on GB300 (tokens/s), one JSON line.

  python bench.py [--gpus N --steps K --warmup W] [--impl ours|reference] [--workload ID]

A step is one full layer forward (MoE Gate, permutation, expert FFNs,
Weight Sum) over one batch of the workload, through the C ABI (moe_forward)
on inputs already resident in HBM. The headline workload is the decode-shaped
bf16 layer: T=32 tokens, hidden 4096, 128 experts, top-8, intermediate 1536;
the same line carries, under per_config, the same measurements for the
prefill bf16 (T=8192), DeepSeek-style fp8 (T=2048, 256 + 1 experts) and
skewed int4 (T=16384) layers. Every workload's active expert weights (1.1 GB
and up) exceed the 126 MB L2, so no flush is needed between steps. With N
GPUs (torchrun) every rank runs its own replica on its own batch (the layer
has no exchange step here): weak scaling.

--impl reference times the CPU oracle (test infrastructure, plain C) on the
host cores on a bounded token sample of the same workload.
"""
from __future__ import annotations

import argparse
import ctypes
import json
import os
import statistics
import subprocess
import sys
import threading
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import synth  # noqa: E402

METRIC = "MoE layer tokens/sec at 1 GB300; % of HBM (decode) / tensor-core (prefill) roofline"
FALLBACK_PEAKS = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}

# DRAM bytes (dram__bytes_read.sum + dram__bytes_write.sum) of the expert-FFN
# kernels (moe_grouped_ffn's launches) per active expert, from one ncu capture
# of a reduced case with the same H, I, dtypes and rows per expert as the full
# workload (the kernels read each active expert's weights and its rows, so the
# traffic grows with the number of active experts); the bench line reports it
# times this run's active experts. Keyed by (workload, route); absent (null)
# whenever the kernels changed since the counters were taken. Captures
# (python bench.py --workload W --set ... --profile 1 under
# ncu --metrics dram__bytes_read.sum,dram__bytes_write.sum,gpu__time_duration.sum):
#   decode   T=8 E=32 (29 active):    stream gate/up + down            1.0966 GB
#   prefill  T=2048 E=32 (32 active): gate/up GEMM (own row gather) + down GEMM  1.6655 GB
#   fp8      T=512 E=64 (64 active):  quantise, gate/up, quantise, down  3.0185 GB
#   MXFP4    T=512 E=64 (64 active):  gather + gate/up GEMM + down GEMM  1.6565 GB
# (the skewed int4 workload's offsets exist for its full size only, so its
# reduced case differs in I and is not scaled here)
TRAFFIC_PER_ACTIVE_EXPERT: dict = {
    ("decode_bf16_T32_H4096_E128_k8_I1536", "stream"): 1.0966e9 / 29,
    ("prefill_bf16_T8192_H4096_E128_k8_I1536", "tc"): 1.6655e9 / 32,
    ("dsv3_fp8_T2048_H7168_E256s1_k8_I2048", "tc_fp8"): 2.9962e9 / 64,
    ("dsv4_mxfp4_T2048_H7168_E256s1_k8_I2048", "tc"): 1.6565e9 / 64,
}


def peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            d = json.load(f)
        return d, "measured"
    return FALLBACK_PEAKS, "fallback"


# ------------------------------------------------------------------ clocks

class ClockSampler:
    """Samples SM clock and clock-event reasons of this process's GPU during
    the timed region (NVML through ctypes; nvidia-smi if NVML is missing)."""

    REASONS = {0x1: "gpu_idle", 0x2: "applications_clocks_setting", 0x4: "sw_power_cap", 0x8: "hw_slowdown",
               0x10: "sync_boost", 0x20: "sw_thermal_slowdown", 0x40: "hw_thermal_slowdown",
               0x80: "hw_power_brake_slowdown", 0x100: "display_clock_setting"}

    def __init__(self, uuid: str | None, period_s: float = 0.002):
        self.uuid, self.period = uuid, period_s
        self.samples, self.reasons = [], 0
        self.max_mhz = None
        self._stop = threading.Event()
        self._nvml = None
        self._h = None
        try:
            nv = ctypes.CDLL("libnvidia-ml.so.1")
            if nv.nvmlInit_v2() == 0:
                h = ctypes.c_void_p()
                if uuid and nv.nvmlDeviceGetHandleByUUID(uuid.encode(), ctypes.byref(h)) == 0:
                    self._nvml, self._h = nv, h
                    m = ctypes.c_uint()
                    if nv.nvmlDeviceGetMaxClockInfo(h, 1, ctypes.byref(m)) == 0:
                        self.max_mhz = m.value
        except OSError:
            self._nvml = None

    def _run(self):
        nv, h = self._nvml, self._h
        clk, rs = ctypes.c_uint(), ctypes.c_ulonglong()
        fn = getattr(nv, "nvmlDeviceGetCurrentClocksEventReasons", None) or nv.nvmlDeviceGetCurrentClocksThrottleReasons
        while not self._stop.is_set():
            if nv.nvmlDeviceGetClockInfo(h, 1, ctypes.byref(clk)) == 0:
                self.samples.append(clk.value)
            if fn(h, ctypes.byref(rs)) == 0:
                self.reasons |= rs.value
            time.sleep(self.period)

    def __enter__(self):
        if self._nvml is not None:
            self._t = threading.Thread(target=self._run, daemon=True)
            self._t.start()
        else:
            self._proc = subprocess.Popen(
                ["nvidia-smi", "--query-gpu=clocks.sm,clocks.max.sm,clocks_event_reasons.active", "--format=csv,noheader,nounits",
                 "-lms", "100"] + ([f"--id={self.uuid}"] if self.uuid else []),
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        return self

    def __exit__(self, *a):
        if self._nvml is not None:
            self._stop.set()
            self._t.join()
        else:
            self._proc.terminate()
            out, _ = self._proc.communicate(timeout=10)
            for line in out.strip().splitlines():
                try:
                    sm, mx, rs = [v.strip() for v in line.split(",")]
                    self.samples.append(int(sm))
                    self.max_mhz = int(mx)
                    self.reasons |= int(rs, 16)
                except ValueError:
                    pass

    def summary(self):
        reasons = [n for b, n in self.REASONS.items() if self.reasons & b and n != "gpu_idle"]
        return {"sm_mhz": statistics.median(self.samples) if self.samples else None, "sm_max_mhz": self.max_mhz,
                "reasons": reasons, "samples": len(self.samples)}


# --------------------------------------------------------------- workload

def load_workload(wid: int, overrides=()):
    """The workload and its inputs; overrides ("KEY=INT" strings) change its
    shape, e.g. a reduced case for profiling."""
    wl = synth.WORKLOADS[wid]
    if overrides:
        wl = wl.replace(**{k: int(v) for k, v in (o.split("=", 1) for o in overrides)})
    inp = synth.make_inputs(wl)
    return wl, inp


def expert_bytes(wq: str, H: int, I: int) -> int:
    """Bytes of one expert's gate, up and down matrices in storage format wq,
    scales included."""
    per = 3 * H * I
    if wq == "bf16":
        return per * 2
    if wq == "f32":
        return per * 4
    if wq == "fp8_b128":  # e4m3 codes + one fp32 scale per 128x128 block
        return per + 3 * (H // 128) * (I // 128) * 4
    if wq == "mxfp4":  # E2M1 nibbles + one E8M0 byte per 32 along K
        return per // 2 + 3 * (H * I // 32)
    return per // 2 + 3 * (H * I // 128) * 2  # int4 nibbles + one bf16 scale per 128 along K


def algorithmic_weight_bytes(wl, active: int) -> int:
    """Expert weight bytes one layer forward must read: every active expert's
    three matrices (+ scales), plus the shared expert."""
    total = active * expert_bytes(wl.wq, wl.H, wl.I)
    if wl.has_shared:
        total += expert_bytes(wl.wq, wl.H, wl.I_shared)
    return total


def cpu_sample_rows(wl, n_tokens: int, step: int) -> list:
    return [(step * n_tokens + i) % wl.T for i in range(n_tokens)]


def run_reference(args, wl, inp, rank):
    """The oracle on the host cores, a bounded token sample per step."""
    import oracle

    if rank != 0:
        return None
    n_tok = args.ref_tokens
    for s in range(args.warmup):
        oracle.forward(wl, inp, rows=cpu_sample_rows(wl, n_tok, s))
    t0 = time.perf_counter()
    for s in range(args.steps):
        oracle.forward(wl, inp, rows=cpu_sample_rows(wl, n_tok, s))
    dt = time.perf_counter() - t0
    v = n_tok * args.steps / dt
    sample = (f"{n_tok} token(s) per step (expert FFNs of those tokens; router logits, expert choice and "
              f"permutation for all {wl.T} tokens), fp64 C oracle")
    return {"metric": METRIC, "impl": "reference", "value": v, "unit": "tokens/s", "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": dt / args.steps * 1e3,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": workload_config(wl),
            "cpu_baseline": {"value": v, "unit": "tokens/s", "cores": oracle.get_threads(), "kind": "oracle",
                             "sample": sample},
            "e2e": {"value": v, "unit": "tokens/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}


def max_over_ranks(v: float, dist, device) -> float:
    """The largest v over the process group (dist None: v): the slowest replica
    sets the job's time."""
    if dist is None:
        return v
    import torch

    t = torch.tensor([v], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def replica_throughput(tokens_per_step: int, steps: int, world: int, seconds: float) -> float:
    """Whole-job tokens/s of `world` independent replicas that each ran `steps`
    steps of `tokens_per_step` tokens in `seconds` (the max over ranks)."""
    return tokens_per_step * steps * world / seconds


def roofline_entry(alg_bytes: float, flops: float, ms: float, pk: dict, pk_kind: str, extra: dict) -> dict:
    """The bench line's roofline object for one kernel call of `ms` milliseconds
    that must move `alg_bytes` and do `flops`: bound by the slower of the bytes
    over the HBM copy peak and the FLOPs over the bf16 dense peak. A
    tensor-bound entry also gives the fraction of the sustained (power-capped)
    bf16 peak, the denominator for kernels timed inside long runs."""
    t_hbm = alg_bytes / (pk["hbm_gbs"] * 1e9)
    t_tensor = flops / (pk["bf16_tflops"] * 1e12)
    common = {**extra, "algorithmic_bytes": alg_bytes, "algorithmic_flops": flops, "ms_per_launch": ms,
              "roofline_ms": max(t_hbm, t_tensor) * 1e3}
    if t_hbm >= t_tensor:
        achieved = alg_bytes / (ms / 1e3) / 1e9
        return {"bound": "hbm", "achieved": achieved, "peak": pk["hbm_gbs"], "unit": "GB/s",
                "frac": achieved / pk["hbm_gbs"], "peak_kind": f"{pk_kind} HBM copy", **common}
    achieved = flops / (ms / 1e3) / 1e12
    entry = {"bound": "tensor", "achieved": achieved, "peak": pk["bf16_tflops"], "unit": "TFLOP/s",
             "frac": achieved / pk["bf16_tflops"], "peak_kind": f"{pk_kind} bf16 dense burst"}
    sustained = pk.get("bf16_tflops_sustained")
    if sustained:
        entry.update(peak_sustained=sustained, frac_sustained=achieved / sustained)
    return {**entry, **common}


def workload_config(wl):
    return {"workload": wl.name, "T": wl.T, "H": wl.H, "I": wl.I, "E": wl.E, "top_k": wl.top_k,
            "scoring": wl.score, "activations": wl.act, "weights": wl.wq,
            "shared_expert": bool(wl.has_shared), "parallelism": "replicas",
            "l2": "no flush: the active experts' weights read each step exceed the 126 MB L2"}


def launches_per_step(wl, route: str, shared_route) -> int:
    """Kernels this library launches per layer forward: gate logits + expert
    choice, the permutation (one kernel up to 1024 pairs, else three), per FFN
    problem a schedule kernel + 2 GEMM/stream kernels (+ a row gather for the
    routed experts on the CTA-pair routes, whose GEMM does not gather its rows
    itself, + 3 weight-decode passes on the decode-once routes), and the
    combine."""
    def ffn(r, routed):
        if r == "tc_fp8":  # schedule, x quantisation, gate/up GEMM, h quantisation, down GEMM
            return 5
        # the one-CTA bf16 GEMM gathers its own rows; decoding GEMMs and pairs use the gather kernel
        gather = r in ("tc_pair", "tc_pair_dequant") or (r == "tc" and wl.wq != "bf16")
        return 3 + (1 if routed and gather else 0) + (3 if r in ("tc_dequant", "tc_pair_dequant") else 0)

    n = 2 + (1 if wl.P <= 1024 else 3) + ffn(route, True) + 1
    if shared_route is not None:
        n += ffn(shared_route, False)
    return n


def cpu_baseline_entry(wl, inp) -> dict:
    """The oracle on the host cores: the first 32 tokens (full routing of every
    token plus those tokens' expert FFNs and combine), repeated until about
    10 s of work (at most 8 runs)."""
    import oracle

    n_tok = min(wl.T, 32)
    dt, runs = 0.0, 0
    while runs == 0 or (dt < 10.0 and runs < 8):
        t0 = time.perf_counter()
        oracle.forward(wl, inp, rows=list(range(n_tok)))
        dt += time.perf_counter() - t0
        runs += 1
    return {"value": n_tok * runs / dt, "unit": "tokens/s", "cores": oracle.get_threads(), "kind": "oracle",
            "sample": f"first {n_tok} tokens, {runs} runs: full routing of all {wl.T} tokens plus the expert "
                      f"FFNs and combine of the sampled ones ({dt:.1f} s)"}


def measure(args, wid: int, overrides, dist, world: int, rank: int, local: int, with_cpu: bool) -> dict | None:
    """One workload: the layer timed over args.steps forwards (CUDA events on
    the launching stream, clocks sampled meanwhile), the expert FFN timed
    alone for the roofline, the host-buffer entry point end to end, and
    (rank 0, one GPU) the oracle on the host cores. Returns the bench fields
    (None for --profile runs)."""
    import torch

    import paper_2607_12875_gb300 as gb

    wl, inp = load_workload(wid, overrides)
    dev = torch.device("cuda", local)

    def act(a):
        if wl.act == "f32":
            return torch.from_numpy(a).to(dev)
        return torch.from_numpy(np.ascontiguousarray(a).view(np.int16)).to(dev).view(torch.bfloat16)

    def wts(store):
        d = {}
        for k, v in store.items():
            d[k] = torch.from_numpy(v.view(np.int16) if v.dtype == np.uint16 else v).to(dev)
        return gb.weights(d["w_gate"], d["w_up"], d["w_down"], d.get("s_gate"), d.get("s_up"), d.get("s_down")), d

    def barrier():
        if dist is not None:
            dist.barrier()

    x = act(inp["x"])
    wr = act(inp["w_router"])
    lb = None if inp["logit_bias"] is None else torch.from_numpy(inp["logit_bias"]).to(dev)
    sb = None if inp["select_bias"] is None else torch.from_numpy(inp["select_bias"]).to(dev)
    experts, keep1 = wts(inp["experts"])
    shared, keep2 = wts(inp["shared"]) if wl.has_shared else (None, None)
    cfg = gb.make_config(wl.T, wl.H, wl.I, wl.E, wl.top_k, score=wl.score, renormalize=wl.renormalize,
                         n_group=wl.n_group, topk_group=wl.topk_group, routed_scale=wl.routed_scale, act=wl.act,
                         w=wl.wq, has_shared=wl.has_shared, I_shared=wl.I_shared, ffn_route=args.route,
                         gate_route=args.gate, combine_route=args.combine)
    ws = torch.empty(gb.workspace_size(cfg), dtype=torch.uint8, device=dev)
    out = torch.empty((wl.T, wl.H), dtype=x.dtype, device=dev)
    counts = torch.empty(wl.E, dtype=torch.int32, device=dev)
    stream = torch.cuda.current_stream(dev)

    def step():
        gb.moe_forward(cfg, x, wr, lb, sb, experts, shared, out, ws)

    if args.profile:
        for _ in range(args.profile):
            step()
        torch.cuda.synchronize()
        print(f"profile run: {wl.name} {overrides} route={gb.ffn_route(cfg)} status={gb.moe_device_status(ws)}")
        return None

    for _ in range(args.warmup):
        step()
    gb.moe_forward(cfg, x, wr, lb, sb, experts, shared, out, ws, counts=counts)
    torch.cuda.synchronize()
    if gb.moe_device_status(ws) != gb.OK:
        raise RuntimeError("device-side wait timed out during warm-up")
    active = int((counts.cpu() > 0).sum())

    uuid = None
    try:
        uuid = "GPU-" + str(torch.cuda.get_device_properties(dev).uuid)
    except Exception:
        pass
    start, end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    barrier()
    torch.cuda.synchronize()
    with ClockSampler(uuid) as clocks:
        start.record(stream)
        for _ in range(args.steps):
            step()
        end.record(stream)
        torch.cuda.synchronize()
    barrier()
    ms = max_over_ranks(start.elapsed_time(end), dist, dev)
    value = replica_throughput(wl.T, args.steps, world, ms / 1e3)

    # dominant kernel: the expert FFN, timed through its own entry point on the same stream
    P = wl.P
    ids = torch.empty((wl.T, wl.top_k), dtype=torch.int32, device=dev)
    w = torch.empty((wl.T, wl.top_k), dtype=torch.float32, device=dev)
    offs = torch.empty(wl.E + 1, dtype=torch.int32, device=dev)
    sp = torch.empty(P, dtype=torch.int32, device=dev)
    pp = torch.empty(P, dtype=torch.int32, device=dev)
    y = torch.empty((P, wl.H), dtype=x.dtype, device=dev)
    gb.moe_route(cfg, x, wr, lb, sb, ids, w, ws)
    gb.moe_permute(cfg, ids, counts, offs, sp, pp, ws)
    for _ in range(3):
        gb.moe_grouped_ffn(cfg, x, counts, offs, sp, experts, y, ws)
    fs, fe = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    torch.cuda.synchronize()
    fs.record(stream)
    for _ in range(args.steps):
        gb.moe_grouped_ffn(cfg, x, counts, offs, sp, experts, y, ws)
    fe.record(stream)
    torch.cuda.synchronize()
    ffn_ms = fs.elapsed_time(fe) / args.steps
    del y
    pk, pk_kind = peaks()
    route = gb.ffn_route(cfg)
    # the expert FFN's roofline: the slower of its algorithmic weight bytes over
    # HBM bandwidth and its FLOPs over the bf16 tensor peak
    routed_bytes = algorithmic_weight_bytes(wl.replace(has_shared=False), active)
    flops = 6.0 * wl.P * wl.H * wl.I
    kernel = {"stream": "moe_grouped_ffn, weight-streaming route (gate/up + down)",
              "tc": "moe_grouped_ffn, tcgen05 route (gate/up GEMM gathering its rows, with SwiGLU + down GEMM)",
              "tc_dequant": "moe_grouped_ffn, tcgen05 decode-once route (3 weight-decode passes + gate/up GEMM "
                            "gathering its rows, with SwiGLU + down GEMM)",
              "tc_fp8": "moe_grouped_ffn, fp8 tcgen05 route (two-term e4m3 quantisation of the rows + gate/up "
                        "GEMM with per-k-block promotion and SwiGLU + quantisation of h + down GEMM)",
              "tc_pair": "moe_grouped_ffn, tcgen05 CTA-pair route (row gather + gate/up GEMM with SwiGLU + down "
                         "GEMM, cta_group::2 MMAs of 256 rows)",
              "tc_pair_dequant": "moe_grouped_ffn, tcgen05 CTA-pair decode-once route (3 weight-decode passes + "
                                 "row gather + gate/up GEMM with SwiGLU + down GEMM, cta_group::2 MMAs)",
              "simt": "moe_grouped_ffn, CUDA-core route"}[route]
    if route == "tc" and wl.wq != "bf16":  # decoding GEMMs read a gathered copy of x
        kernel = ("moe_grouped_ffn, tcgen05 route (row gather + gate/up GEMM decoding its weight tiles, with "
                  "SwiGLU + down GEMM)")
    tpe = TRAFFIC_PER_ACTIVE_EXPERT.get((wl.name, route))
    extra = {"traffic": None if tpe is None else tpe * active, "kernel": kernel, "active_experts": active,
             "route": route, "gate": gb.gate_route(cfg)}
    roofline = roofline_entry(routed_bytes, flops, ffn_ms, pk, pk_kind, extra)

    # end to end through the public host-buffer entry point
    x_host = x.cpu().pin_memory()
    out_host = torch.empty((wl.T, wl.H), dtype=x.dtype).pin_memory()
    for _ in range(3):
        gb.moe_forward_hostio(cfg, x_host, wr, lb, sb, experts, shared, out_host, ws)
    torch.cuda.synchronize()
    barrier()
    t0 = time.perf_counter()
    for _ in range(args.steps):
        gb.moe_forward_hostio(cfg, x_host, wr, lb, sb, experts, shared, out_host, ws)
        stream.synchronize()
    e2e_s = time.perf_counter() - t0
    barrier()
    e2e_s = max_over_ranks(e2e_s, dist, dev)
    io_bytes = wl.T * wl.H * x.element_size()
    e2e = {"value": replica_throughput(wl.T, args.steps, world, e2e_s), "unit": "tokens/s",
           "h2d_bytes_per_step": io_bytes, "d2h_bytes_per_step": io_bytes}

    per_step = launches_per_step(wl, route, gb.ffn_route(cfg, shared=True) if wl.has_shared else None)
    cpu = cpu_baseline_entry(wl, inp) if with_cpu else None
    del x, wr, lb, sb, experts, shared, keep1, keep2, ws, out, x_host, out_host
    torch.cuda.empty_cache()
    return {"value": value, "ms_per_step": ms / args.steps, "steps": args.steps,
            "dtype": wl.act if wl.wq in ("f32", "bf16") else f"{wl.act}+{wl.wq}",
            "config": workload_config(wl), "clocks": clocks.summary(), "e2e": e2e,
            "gpu_launches": per_step * args.steps, "roofline": roofline, "cpu_baseline": cpu}


# workloads the default run times besides the headline one: prefill bf16,
# DeepSeek-style fp8 and skewed int4 (the other size classes of the layer),
# and the DeepSeek-style layer with MXFP4 experts
PER_CONFIG = (3, 4, 5, 6)


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=200)
    ap.add_argument("--warmup", type=int, default=10)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--workload", type=int, default=2, help="synth.WORKLOADS id of the headline (2 = decode bf16)")
    ap.add_argument("--route", default="auto", choices=["auto", "stream", "simt", "tc", "tc_dequant", "tc_fp8", "tc_pair", "tc_pair_dequant"])
    ap.add_argument("--gate", default="auto", choices=["auto", "simt", "tc"], help="router logits route")
    ap.add_argument("--combine", default="auto", choices=["auto", "separate", "fused"], help="Weight Sum route")
    ap.add_argument("--ref-tokens", type=int, default=1, help="tokens per oracle step (reference arm)")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-per-config", action="store_true",
                    help="time only the headline workload (by default workloads 3, 4 and 5 are timed too)")
    ap.add_argument("--set", action="append", default=[], metavar="KEY=INT",
                    help="override a workload field (reduced cases for profiling), e.g. --set T=2048 --set E=32")
    ap.add_argument("--profile", type=int, default=0, metavar="N",
                    help="run N untimed layer forwards and exit (for ncu captures); prints no bench line")
    args = ap.parse_args()
    if args.warmup < 3 and args.impl == "ours":
        args.warmup = 3

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))

    if args.impl == "reference":
        if rank != 0:
            return
        wl, inp = load_workload(args.workload, args.set)
        print(json.dumps(run_reference(args, wl, inp, rank)))
        return

    import torch

    torch.cuda.set_device(local)
    dist = None
    if world > 1:
        import torch.distributed as dist

        dist.init_process_group("nccl", device_id=torch.device("cuda", local))

    with_cpu = rank == 0 and world == 1 and not args.no_cpu_baseline
    head = measure(args, args.workload, args.set, dist, world, rank, local, with_cpu)
    if head is None:  # --profile
        return
    per_config = {}
    if not args.no_per_config and not args.set and args.route == "auto" and args.gate == "auto" \
            and args.combine == "auto":
        for wid in PER_CONFIG:
            if wid == args.workload:
                continue
            m = measure(args, wid, (), dist, world, rank, local, with_cpu)
            per_config[m["config"]["workload"]] = {"value": m["value"], "unit": "tokens/s", "n_gpus": world, **m}

    if rank == 0:
        line = {"metric": METRIC, "value": head["value"], "unit": "tokens/s", "n_gpus": world,
                "steps": args.steps, "warmup": args.warmup, "ms_per_step": head["ms_per_step"],
                "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": head["dtype"],
                "data": "synthetic (seeded SplitMix64/Irwin-Hall normals; random-init weights)",
                "config": head["config"], "clocks": head["clocks"], "e2e": head["e2e"],
                "gpu_launches": head["gpu_launches"], "roofline": head["roofline"],
                "cpu_baseline": head["cpu_baseline"]}
        if per_config:
            line["per_config"] = per_config
        print(json.dumps(line))
    if dist is not None:
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
