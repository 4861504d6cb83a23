"""CPU oracle for the MoE layer forward (MoE Gate -> Fused MoE -> Weight Sum).

TEST INFRASTRUCTURE: only tests/, the smoke check in __graft_entry__ and the
benchmark's CPU-baseline leg import this package. The product library never
uses it, and it shares no code with the CUDA path. The arithmetic lives in
``oracle.c`` (plain C, fp64 except for the fp32 expert choice), apart from
the expert FFN's matrix products, which are fp64 products from numpy's BLAS
(a library routine used as one step); this module loads the C library and
strings the steps together in the paper's node order.

Every function is pinned in tests/test_oracle_*.py against references that do
not come from this code (brute force, closed forms, library routines, hand
cases).
"""
from __future__ import annotations

import ctypes
import os
import subprocess

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "oracle.c")
_LIB_PATH = os.path.join(_HERE, "liboracle.so")
_lib = None


def build(force: bool = False) -> str:
    """Compiles liboracle.so next to its source. -ffp-contract=off keeps every
    multiply and add a separate rounding unless the source says fmaf."""
    if force or not os.path.exists(_LIB_PATH) or os.path.getmtime(_LIB_PATH) < os.path.getmtime(_SRC):
        tmp = _LIB_PATH + f".tmp{os.getpid()}"
        subprocess.check_call(["gcc", "-O2", "-ffp-contract=off", "-fno-fast-math", "-fPIC", "-shared",
                               "-pthread", "-o", tmp, _SRC, "-lm"])
        os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


class RouteCfg(ctypes.Structure):
    _fields_ = [("T", ctypes.c_int32), ("E", ctypes.c_int32), ("top_k", ctypes.c_int32),
                ("score", ctypes.c_int32), ("renormalize", ctypes.c_int32),
                ("n_group", ctypes.c_int32), ("topk_group", ctypes.c_int32),
                ("routed_scale", ctypes.c_float)]


def _L():
    global _lib
    if _lib is None:
        build()
        lib = ctypes.CDLL(_LIB_PATH)
        i64, i32, vp = ctypes.c_int64, ctypes.c_int32, ctypes.c_void_p
        lib.oracle_set_threads.argtypes = [ctypes.c_int]
        lib.oracle_get_threads.restype = ctypes.c_int
        lib.oracle_gate_logits.argtypes = [i64, i64, i64, vp, vp, vp, vp]
        lib.oracle_gate_logits.restype = ctypes.c_int
        lib.oracle_rmsnorm.argtypes = [i64, i64, vp, vp, ctypes.c_float, vp]
        lib.oracle_rmsnorm.restype = ctypes.c_int
        lib.oracle_pexp.argtypes = [ctypes.c_float]
        lib.oracle_pexp.restype = ctypes.c_float
        lib.oracle_pexp_n.argtypes = [i64, vp, vp]
        lib.oracle_sigmoid_n.argtypes = [i64, vp, vp]
        lib.oracle_route.argtypes = [ctypes.POINTER(RouteCfg), vp, vp, vp, vp]
        lib.oracle_route.restype = ctypes.c_int
        lib.oracle_permute.argtypes = [i64, i32, vp, vp, vp, vp, vp]
        lib.oracle_permute.restype = ctypes.c_int
        lib.oracle_e4m3_value.argtypes = [ctypes.c_uint8]
        lib.oracle_e4m3_value.restype = ctypes.c_double
        lib.oracle_dequant_fp8_b128.argtypes = [i64, i64, vp, vp, vp]
        lib.oracle_dequant_int4_g128.argtypes = [i64, i64, vp, vp, vp]
        lib.oracle_e2m1_value.argtypes = [ctypes.c_uint8]
        lib.oracle_e2m1_value.restype = ctypes.c_double
        lib.oracle_e8m0_value.argtypes = [ctypes.c_uint8]
        lib.oracle_e8m0_value.restype = ctypes.c_double
        lib.oracle_dequant_mxfp4.argtypes = [i64, i64, vp, vp, vp]
        lib.oracle_widen_f32.argtypes = [i64, vp, vp]
        lib.oracle_widen_bf16.argtypes = [i64, vp, vp]
        lib.oracle_combine.argtypes = [i64, i64, i64, vp, vp, vp, vp, vp]
        lib.oracle_set_threads(os.cpu_count() or 1)
        _lib = lib
    return _lib


def set_threads(n: int) -> None:
    _L().oracle_set_threads(int(n))


def get_threads() -> int:
    return _L().oracle_get_threads()


def _p(a):
    if a is None:
        return None
    assert isinstance(a, np.ndarray) and a.flags.c_contiguous, "oracle inputs must be C-contiguous arrays"
    return a.ctypes.data


def _c(a, dtype):
    return None if a is None else np.ascontiguousarray(a, dtype=dtype)


# --------------------------------------------------------------- MoE Gate

def gate_logits(x: np.ndarray, w_router: np.ndarray, logit_bias=None) -> np.ndarray:
    """fp32 router logits [T, E] in the pinned order (see oracle.c)."""
    x = _c(x, np.float32)
    g = _c(w_router, np.float32)
    b = _c(logit_bias, np.float32)
    T, H = x.shape
    E = g.shape[0]
    out = np.empty((T, E), dtype=np.float32)
    if _L().oracle_gate_logits(T, H, E, _p(x), _p(g), _p(b), _p(out)) != 0:
        raise ValueError("gate logits need H % 256 == 0")
    return out


def rmsnorm(x: np.ndarray, gamma: np.ndarray, eps: float) -> np.ndarray:
    """fp32 RMSNorm of the rows of x [T, H] in the pinned order (see
    oracle.c); the caller rounds the result to the activation dtype."""
    x = _c(x, np.float32)
    g = _c(gamma, np.float32)
    T, H = x.shape
    out = np.empty((T, H), dtype=np.float32)
    if _L().oracle_rmsnorm(T, H, _p(x), _p(g), ctypes.c_float(eps), _p(out)) != 0:
        raise ValueError("rmsnorm needs H % 256 == 0 and eps >= 0")
    return out


def round_bf16(v: np.ndarray) -> np.ndarray:
    """Raw bf16 bit patterns (uint16) of fp32 values, rounded to nearest even
    (a NaN stays a quiet NaN)."""
    u = _c(v, np.float32).view(np.uint32).astype(np.uint64)
    nan = (u & 0x7FFFFFFF) > 0x7F800000
    r = ((u + 0x7FFF + ((u >> 16) & 1)) >> 16) & 0xFFFF
    r = np.where(nan, ((u >> 16) | 0x40) & 0xFFFF, r)
    return r.astype(np.uint16)


def pexp(v: np.ndarray) -> np.ndarray:
    v = _c(v, np.float32)
    out = np.empty_like(v)
    _L().oracle_pexp_n(v.size, _p(v), _p(out))
    return out


def sigmoid(v: np.ndarray) -> np.ndarray:
    v = _c(v, np.float32)
    out = np.empty_like(v)
    _L().oracle_sigmoid_n(v.size, _p(v), _p(out))
    return out


def route(logits: np.ndarray, top_k: int, score: str = "softmax", renormalize: bool = True,
          n_group: int = 1, topk_group: int = 1, routed_scale: float = 1.0, select_bias=None):
    """(topk_ids [T, k] int32, topk_w [T, k] fp64) from fp32 logits [T, E]."""
    l = _c(logits, np.float32)
    T, E = l.shape
    cfg = RouteCfg(T, E, top_k, 0 if score == "softmax" else 1, int(bool(renormalize)),
                   n_group, topk_group, routed_scale)
    ids = np.empty((T, top_k), dtype=np.int32)
    w = np.empty((T, top_k), dtype=np.float64)
    sb = _c(select_bias, np.float32)
    if _L().oracle_route(ctypes.byref(cfg), _p(l), _p(sb), _p(ids), _p(w)) != 0:
        raise ValueError("invalid routing configuration")
    return ids, w


# ---------------------------------------------------- Fused MoE: permute

def permute(topk_ids: np.ndarray, E: int):
    """(counts [E], offsets [E+1], sorted_pair [P], pair_pos [P]), all int32."""
    ids = _c(topk_ids, np.int32).reshape(-1)
    P = ids.size
    counts = np.empty(E, np.int32)
    offsets = np.empty(E + 1, np.int32)
    sp = np.empty(P, np.int32)
    pp = np.empty(P, np.int32)
    if _L().oracle_permute(P, E, _p(ids), _p(counts), _p(offsets), _p(sp), _p(pp)) != 0:
        raise ValueError("expert id out of range")
    return counts, offsets, sp, pp


# ------------------------------------------- Fused MoE: stored weights

def e4m3_value(code: int) -> float:
    return _L().oracle_e4m3_value(code)


def dequant_fp8_b128(q: np.ndarray, s: np.ndarray) -> np.ndarray:
    q = _c(q, np.uint8)
    s = _c(s, np.float32)
    N, K = q.shape
    out = np.empty((N, K), np.float64)
    _L().oracle_dequant_fp8_b128(N, K, _p(q), _p(s), _p(out))
    return out


def dequant_int4_g128(q: np.ndarray, s: np.ndarray) -> np.ndarray:
    q = _c(q, np.uint8)
    s = _c(s, np.uint16)
    N, K2 = q.shape
    out = np.empty((N, 2 * K2), np.float64)
    _L().oracle_dequant_int4_g128(N, 2 * K2, _p(q), _p(s), _p(out))
    return out


def e2m1_value(code: int) -> float:
    return _L().oracle_e2m1_value(code)


def e8m0_value(code: int) -> float:
    return _L().oracle_e8m0_value(code)


def dequant_mxfp4(q: np.ndarray, s: np.ndarray) -> np.ndarray:
    q = _c(q, np.uint8)
    s = _c(s, np.uint8)
    N, K2 = q.shape
    out = np.empty((N, 2 * K2), np.float64)
    _L().oracle_dequant_mxfp4(N, 2 * K2, _p(q), _p(s), _p(out))
    return out


def widen(a: np.ndarray, dtype: str) -> np.ndarray:
    """Exact fp64 copy of fp32 values or of raw bf16 bit patterns."""
    if dtype == "f32":
        a = _c(a, np.float32)
        out = np.empty(a.shape, np.float64)
        _L().oracle_widen_f32(a.size, _p(a), _p(out))
    else:
        a = _c(a, np.uint16)
        out = np.empty(a.shape, np.float64)
        _L().oracle_widen_bf16(a.size, _p(a), _p(out))
    return out


def weight_f64(store: dict, name: str, e: int, wq: str) -> np.ndarray:
    """Dequantised fp64 [N, K] matrix ``name`` (gate/up/down) of expert e."""
    q = store["w_" + name][e]
    if wq in ("f32", "bf16"):
        return widen(q, wq)
    if wq == "fp8_b128":
        return dequant_fp8_b128(q, store["s_" + name][e])
    if wq == "int4_g128":
        return dequant_int4_g128(q, store["s_" + name][e])
    if wq == "mxfp4":
        return dequant_mxfp4(q, store["s_" + name][e])
    raise ValueError(wq)


# ------------------------------------------------ Fused MoE: expert FFN

def expert_ffn(x_rows: np.ndarray, w_gate: np.ndarray, w_up: np.ndarray, w_down: np.ndarray) -> np.ndarray:
    """fp64 SwiGLU FFN of one expert on fp64 rows x [n, H] -> y [n, H]:

        g = x Wgate^T,  u = x Wup^T          (Wgate, Wup: [I, H])
        a = silu(g) * u,  silu(z) = z / (1 + exp(-z))
        y = a Wdown^T                        (Wdown: [H, I])

    the gated (SwiGLU) MLP of the MoE models the paper serves (Section 6; the
    paper does not print it). Every product is accumulated in fp64 (numpy's
    BLAS); the order of the fp64 sums is the library's, which moves results
    by ~1e-16 relative, far inside every tolerance the tests use.
    """
    x = _c(x_rows, np.float64)
    wg, wu, wd = (_c(a, np.float64) for a in (w_gate, w_up, w_down))
    g = x @ wg.T
    u = x @ wu.T
    with np.errstate(over="ignore"):  # exp(-g) -> inf for very negative g gives silu = -0
        a = g / (1.0 + np.exp(-g)) * u
    return a @ wd.T


# ----------------------------------------------------------- Weight Sum

def combine(y_pairs: np.ndarray, topk_w: np.ndarray, pair_pos: np.ndarray, y_shared=None) -> np.ndarray:
    y = _c(y_pairs, np.float64)
    w = _c(topk_w, np.float64)
    pp = _c(pair_pos, np.int32).reshape(-1)
    T, k = w.shape
    H = y.shape[1]
    ys = _c(y_shared, np.float64)
    out = np.empty((T, H), np.float64)
    _L().oracle_combine(T, k, H, _p(y), _p(w), _p(pp), _p(ys), _p(out))
    return out


# ------------------------------------------------------------ whole layer

def forward(wl, inputs: dict, rows=None) -> dict:
    """The layer in node order: MoE Gate, permutation, expert FFNs, Weight Sum.

    Routing, weights and the permutation are computed for every token.
    Expert FFNs and the combined output are computed for the tokens ``rows``
    (all tokens when None); ``out`` then holds those tokens' rows, in order.
    ``wl`` is a synth.Workload; ``inputs`` comes from synth.make_inputs.
    """
    x32 = inputs["x"] if wl.act == "f32" else (inputs["x"].astype(np.uint32) << 16).view(np.float32)
    g32 = (inputs["w_router"] if wl.act == "f32"
           else (inputs["w_router"].astype(np.uint32) << 16).view(np.float32))
    logits = gate_logits(x32, g32, inputs.get("logit_bias"))
    ids, w = route(logits, wl.top_k, wl.score, wl.renormalize, wl.n_group, wl.topk_group,
                   wl.routed_scale, inputs.get("select_bias"))
    counts, offsets, sorted_pair, pair_pos = permute(ids, wl.E)
    T, k, H = wl.T, wl.top_k, wl.H
    rows = np.arange(T) if rows is None else np.asarray(rows, dtype=np.int64)
    xr = widen(np.ascontiguousarray(inputs["x"][rows]), wl.act)
    # expert outputs for every (selected row, slot), grouped by expert
    y = np.zeros((len(rows), k, H), np.float64)
    ex = inputs["experts"]
    sel = ids[rows]
    for e in np.unique(sel):
        ri, rj = np.nonzero(sel == e)
        wg = weight_f64(ex, "gate", e, wl.wq)
        wu = weight_f64(ex, "up", e, wl.wq)
        wd = weight_f64(ex, "down", e, wl.wq)
        y[ri, rj] = expert_ffn(xr[ri], wg, wu, wd)
    y_shared = None
    if wl.has_shared:
        sh = inputs["shared"]
        y_shared = expert_ffn(xr, weight_f64(sh, "gate", 0, wl.wq), weight_f64(sh, "up", 0, wl.wq),
                              weight_f64(sh, "down", 0, wl.wq))
    local_pos = np.arange(len(rows) * k, dtype=np.int32).reshape(len(rows), k)
    out = combine(y.reshape(len(rows) * k, H), w[rows], local_pos, y_shared)
    return dict(logits=logits, topk_ids=ids, topk_w=w, counts=counts, offsets=offsets,
                sorted_pair=sorted_pair, pair_pos=pair_pos, rows=rows, y=y, y_shared=y_shared, out=out)
