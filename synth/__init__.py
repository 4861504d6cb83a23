"""Seeded synthetic inputs for the MoE layer workloads.

The tensors come from ``synth.c`` (counter-based SplitMix64 streams, Irwin-Hall
normals, fp8/int4 checkpoint storage forms); this module only loads that
library, names the streams and describes the five workloads. It holds none of
the layer's arithmetic and is shared by the oracle side and the GPU side, which
both consume exactly the arrays it returns.
"""
from __future__ import annotations

import ctypes
import dataclasses
import json
import os
import subprocess

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "synth.c")
_LIB_PATH = os.path.join(_HERE, "libsynth.so")
_lib = None

# stream ids of the tensors of one workload
TID = dict(x=1, w_router=2, w_gate=3, w_up=4, w_down=5, select_bias=6,
           sh_gate=7, sh_up=8, sh_down=9)


def build(force: bool = False) -> str:
    """Compiles libsynth.so next to its source (plain C, pthreads)."""
    if force or not os.path.exists(_LIB_PATH) or os.path.getmtime(_LIB_PATH) < os.path.getmtime(_SRC):
        tmp = _LIB_PATH + f".tmp{os.getpid()}"
        subprocess.check_call(["gcc", "-O2", "-fPIC", "-shared", "-pthread", "-o", tmp, _SRC, "-lm"])
        os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def _L():
    global _lib
    if _lib is None:
        build()
        lib = ctypes.CDLL(_LIB_PATH)
        u64, i64, dbl, vp = ctypes.c_uint64, ctypes.c_int64, ctypes.c_double, ctypes.c_void_p
        lib.synth_normal_f32.argtypes = [u64, u64, dbl, u64, i64, vp]
        lib.synth_normal_bf16.argtypes = [u64, u64, dbl, u64, i64, vp]
        lib.synth_fp8_b128.argtypes = [u64, u64, dbl, i64, i64, i64, i64, vp, vp]
        lib.synth_int4_g128.argtypes = [u64, u64, dbl, i64, i64, i64, i64, vp, vp]
        lib.synth_mxfp4.argtypes = [u64, u64, dbl, i64, i64, i64, i64, vp, vp]
        lib.synth_set_threads.argtypes = [ctypes.c_int]
        lib.synth_set_threads(os.cpu_count() or 1)
        _lib = lib
    return _lib


def _ptr(a: np.ndarray) -> int:
    assert a.flags.c_contiguous
    return a.ctypes.data


def normal_f32(seed: int, tid: int, sigma: float, shape, offset: int = 0) -> np.ndarray:
    out = np.empty(shape, dtype=np.float32)
    _L().synth_normal_f32(seed, tid, sigma, offset, out.size, _ptr(out))
    return out


def normal_bf16(seed: int, tid: int, sigma: float, shape, offset: int = 0) -> np.ndarray:
    """bf16 values as raw uint16 bit patterns."""
    out = np.empty(shape, dtype=np.uint16)
    _L().synth_normal_bf16(seed, tid, sigma, offset, out.size, _ptr(out))
    return out


def fp8_b128(seed, tid, sigma, N, K, e0=0, ne=1):
    """Experts [e0, e0+ne) of an [E, N, K] weight as (e4m3 codes [ne,N,K] u8,
    fp32 block scales [ne, N/128, K/128])."""
    q = np.empty((ne, N, K), dtype=np.uint8)
    s = np.empty((ne, N // 128, K // 128), dtype=np.float32)
    if _L().synth_fp8_b128(seed, tid, sigma, e0, ne, N, K, _ptr(q), _ptr(s)) != 0:
        raise ValueError("fp8 128x128 blocks need N and K to be multiples of 128")
    return q, s


def int4_g128(seed, tid, sigma, N, K, e0=0, ne=1):
    """Experts [e0, e0+ne) of an [E, N, K] weight as (packed int4 [ne,N,K/2] u8,
    bf16 group scales [ne, N, K/128] as uint16)."""
    q = np.empty((ne, N, K // 2), dtype=np.uint8)
    s = np.empty((ne, N, K // 128), dtype=np.uint16)
    if _L().synth_int4_g128(seed, tid, sigma, e0, ne, N, K, _ptr(q), _ptr(s)) != 0:
        raise ValueError("int4 groups of 128 need K to be a multiple of 128")
    return q, s


def mxfp4(seed, tid, sigma, N, K, e0=0, ne=1):
    """Experts [e0, e0+ne) of an [E, N, K] weight as MXFP4 (packed E2M1
    [ne, N, K/2] u8, E8M0 block scales [ne, N, K/32] u8)."""
    q = np.empty((ne, N, K // 2), dtype=np.uint8)
    s = np.empty((ne, N, K // 32), dtype=np.uint8)
    if _L().synth_mxfp4(seed, tid, sigma, e0, ne, N, K, _ptr(q), _ptr(s)) != 0:
        raise ValueError("MXFP4 blocks of 32 need K to be a multiple of 32")
    return q, s


def bf16_bits_to_f32(b: np.ndarray) -> np.ndarray:
    """Exact widening of raw bf16 bit patterns to fp32."""
    return (b.astype(np.uint32) << 16).view(np.float32)


# ------------------------------------------------------------- workloads

@dataclasses.dataclass(frozen=True)
class Workload:
    name: str
    T: int
    H: int
    I: int
    E: int
    top_k: int
    act: str            # "f32" | "bf16"   (x, router weight, h, y, out)
    wq: str             # "f32" | "bf16" | "fp8_b128" | "int4_g128" | "mxfp4"  (expert weights)
    seed: int
    score: str = "softmax"      # "softmax" | "sigmoid"
    renormalize: bool = True
    routed_scale: float = 1.0
    n_group: int = 1
    topk_group: int = 1
    has_shared: bool = False
    I_shared: int = 0
    x_sigma: float = 1.0
    w_sigma: float = 0.02
    select_bias_sigma: float = 0.0
    zipf: bool = False

    @property
    def P(self) -> int:
        return self.T * self.top_k

    def replace(self, **kw) -> "Workload":
        return dataclasses.replace(self, **kw)


# The six layer shapes of the benchmark grid. Seeds 0 and 3 are given by the
# workload descriptions; 1, 2, 4 and 5 are chosen here.
WORKLOADS = {
    1: Workload("tiny_f32_T64_H256_E8_k2_I512", 64, 256, 512, 8, 2, "f32", "f32", seed=0),
    2: Workload("decode_bf16_T32_H4096_E128_k8_I1536", 32, 4096, 1536, 128, 8, "bf16", "bf16", seed=1),
    3: Workload("prefill_bf16_T8192_H4096_E128_k8_I1536", 8192, 4096, 1536, 128, 8, "bf16", "bf16", seed=2),
    4: Workload("dsv3_fp8_T2048_H7168_E256s1_k8_I2048", 2048, 7168, 2048, 256, 8, "bf16", "fp8_b128",
                seed=3, score="sigmoid", routed_scale=2.5, n_group=8, topk_group=4,
                has_shared=True, I_shared=2048, select_bias_sigma=0.01),
    5: Workload("skew_int4_T16384_H4096_E64_k6_I2816", 16384, 4096, 2816, 64, 6, "bf16", "int4_g128",
                seed=4, zipf=True),
    # the DeepSeek-style layer of workload 4 with MXFP4 expert weights (the
    # expert format of the DeepSeek reference path, Section 6.2)
    6: Workload("dsv4_mxfp4_T2048_H7168_E256s1_k8_I2048", 2048, 7168, 2048, 256, 8, "bf16", "mxfp4",
                seed=5, score="sigmoid", routed_scale=2.5, n_group=8, topk_group=4,
                has_shared=True, I_shared=2048, select_bias_sigma=0.01),
}


def zipf_logit_bias(E: int) -> np.ndarray:
    """Per-expert logit offsets b_e = -c * ln(e + 1) (expert 0 hottest), stored
    as fp32 values in zipf_bias.json, written by calibrate_zipf.py."""
    with open(os.path.join(_HERE, "zipf_bias.json")) as f:
        d = json.load(f)
    if d["E"] != E:
        raise ValueError(f"zipf_bias.json holds offsets for E={d['E']}, not {E}")
    return np.array([float.fromhex(h) for h in d["bias_hex"]], dtype=np.float64).astype(np.float32)


def _act(seed, tid, sigma, shape, act):
    return normal_f32(seed, tid, sigma, shape) if act == "f32" else normal_bf16(seed, tid, sigma, shape)


def expert_weights(w: Workload, E: int, I: int, tids=("w_gate", "w_up", "w_down"), e0: int = 0,
                   ne: int | None = None) -> dict:
    """Weights of experts [e0, e0+ne): gate/up [ne, I, H], down [ne, H, I] in the
    workload's storage form. Keys w_gate, w_up, w_down (+ s_* when quantised)."""
    ne = E - e0 if ne is None else ne
    H = w.H
    out = {}
    for name, tid in zip(("gate", "up", "down"), tids):
        N, K = (I, H) if name != "down" else (H, I)
        if w.wq in ("f32", "bf16"):
            n = ne * N * K
            off = e0 * N * K
            arr = (normal_f32 if w.wq == "f32" else normal_bf16)(w.seed, TID[tid], w.w_sigma, (n,), off)
            out["w_" + name] = arr.reshape(ne, N, K)
        elif w.wq == "fp8_b128":
            q, s = fp8_b128(w.seed, TID[tid], w.w_sigma, N, K, e0, ne)
            out["w_" + name], out["s_" + name] = q, s
        elif w.wq == "int4_g128":
            q, s = int4_g128(w.seed, TID[tid], w.w_sigma, N, K, e0, ne)
            out["w_" + name], out["s_" + name] = q, s
        elif w.wq == "mxfp4":
            q, s = mxfp4(w.seed, TID[tid], w.w_sigma, N, K, e0, ne)
            out["w_" + name], out["s_" + name] = q, s
        else:
            raise ValueError(w.wq)
    return out


def make_inputs(w: Workload, with_experts: bool = True) -> dict:
    """All input arrays of one workload (numpy, host)."""
    d = {
        "x": _act(w.seed, TID["x"], w.x_sigma, (w.T, w.H), w.act),
        "w_router": _act(w.seed, TID["w_router"], w.w_sigma, (w.E, w.H), w.act),
        "logit_bias": zipf_logit_bias(w.E) if w.zipf else None,
        "select_bias": (normal_f32(w.seed, TID["select_bias"], w.select_bias_sigma, (w.E,))
                        if w.select_bias_sigma > 0 else None),
    }
    if with_experts:
        d["experts"] = expert_weights(w, w.E, w.I)
        if w.has_shared:
            d["shared"] = expert_weights(w, 1, w.I_shared, tids=("sh_gate", "sh_up", "sh_down"))
    return d
