"""Python binding of libgbmoe.so, the GB300 MoE layer forward (C ABI in
include/gbmoe.h).

Argument marshalling only: every function passes torch tensors' device
pointers and the current CUDA stream to the entry point of the same name and
raises GbmoeError on a non-zero status. All arithmetic runs in the library's
CUDA kernels; there is no fallback. If the library is missing, build it with
``paper_2607_12875_gb300.build.build()`` (needs nvcc).
"""
from __future__ import annotations

import ctypes
import os

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libgbmoe.so")

# status codes, dtypes, scoring and FFN routes (values of include/gbmoe.h)
OK, EINVAL, EUNSUPPORTED, EWORKSPACE, ECUDA, EDEVICE_TIMEOUT = 0, -1, -2, -3, -4, -5
F32, BF16, FP8_E4M3_B128, INT4_G128, MXFP4 = 0, 1, 2, 3, 4
SOFTMAX, SIGMOID = 0, 1
FFN_AUTO, FFN_STREAM, FFN_SIMT, FFN_TC, FFN_TC_DEQUANT, FFN_TC_FP8, FFN_TC_PAIR, FFN_TC_PAIR_DEQUANT = range(8)
GATE_AUTO, GATE_SIMT, GATE_TC = 0, 1, 2
COMBINE_AUTO, COMBINE_SEPARATE, COMBINE_FUSED = 0, 1, 2

DTYPES = {"f32": F32, "bf16": BF16, "fp8_b128": FP8_E4M3_B128, "int4_g128": INT4_G128, "mxfp4": MXFP4}
GATES = {"auto": GATE_AUTO, "simt": GATE_SIMT, "tc": GATE_TC}
COMBINES = {"auto": COMBINE_AUTO, "separate": COMBINE_SEPARATE, "fused": COMBINE_FUSED}
ROUTES = {"auto": FFN_AUTO, "stream": FFN_STREAM, "simt": FFN_SIMT, "tc": FFN_TC, "tc_dequant": FFN_TC_DEQUANT,
          "tc_fp8": FFN_TC_FP8, "tc_pair": FFN_TC_PAIR, "tc_pair_dequant": FFN_TC_PAIR_DEQUANT}

# every function include/gbmoe.h declares
EXPORTS = ("gbmoe_status_string", "gbmoe_check_config", "gbmoe_workspace_size", "gbmoe_ffn_route",
           "gbmoe_gate_route", "moe_route",
           "moe_permute",
           "moe_grouped_ffn", "moe_shared_ffn", "moe_combine", "moe_forward", "moe_forward_hostio",
           "moe_device_status", "moe_permute_noalloc", "gbmoe_last_cuda_error", "moe_rmsnorm")


class GbmoeError(RuntimeError):
    def __init__(self, status: int, call: str):
        self.status = status
        detail = ""
        if status == ECUDA:  # the CUDA error code behind it
            self.cuda_error = lib().gbmoe_last_cuda_error()
            detail = f", cudaError {self.cuda_error}"
        super().__init__(f"{call}: {status_string(status)} ({status}{detail})")


class Config(ctypes.Structure):
    _fields_ = [("T", ctypes.c_int32), ("H", ctypes.c_int32), ("I", ctypes.c_int32), ("E", ctypes.c_int32),
                ("top_k", ctypes.c_int32), ("score", ctypes.c_int32), ("renormalize", ctypes.c_int32),
                ("n_group", ctypes.c_int32), ("topk_group", ctypes.c_int32), ("routed_scale", ctypes.c_float),
                ("act_dtype", ctypes.c_int32), ("w_dtype", ctypes.c_int32), ("has_shared", ctypes.c_int32),
                ("I_shared", ctypes.c_int32), ("ffn_route", ctypes.c_int32), ("gate_route", ctypes.c_int32),
                ("combine_route", ctypes.c_int32)]


class ExpertWeights(ctypes.Structure):
    _fields_ = [("w_gate", ctypes.c_void_p), ("w_up", ctypes.c_void_p), ("w_down", ctypes.c_void_p),
                ("s_gate", ctypes.c_void_p), ("s_up", ctypes.c_void_p), ("s_down", ctypes.c_void_p)]


_lib = None


def lib() -> ctypes.CDLL:
    """The loaded libgbmoe.so (raises if it has not been built)."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError(f"{LIB_PATH} is missing: run paper_2607_12875_gb300.build.build() first")
        L = ctypes.CDLL(LIB_PATH)
        vp, i32p, fp = ctypes.c_void_p, ctypes.POINTER(ctypes.c_int32), ctypes.c_void_p
        cfgp, wp = ctypes.POINTER(Config), ctypes.POINTER(ExpertWeights)
        sz = ctypes.c_size_t
        L.gbmoe_status_string.argtypes = [ctypes.c_int]
        L.gbmoe_status_string.restype = ctypes.c_char_p
        L.gbmoe_last_cuda_error.argtypes = []
        L.gbmoe_last_cuda_error.restype = ctypes.c_int
        L.gbmoe_check_config.argtypes = [cfgp]
        L.gbmoe_workspace_size.argtypes = [cfgp]
        L.gbmoe_workspace_size.restype = sz
        L.gbmoe_ffn_route.argtypes = [cfgp, ctypes.c_int]
        L.gbmoe_gate_route.argtypes = [cfgp]
        L.moe_route.argtypes = [cfgp, vp, vp, fp, fp, vp, vp, vp, sz, vp]
        L.moe_rmsnorm.argtypes = [cfgp, vp, vp, ctypes.c_float, vp, vp]
        L.moe_permute.argtypes = [cfgp, vp, vp, vp, vp, vp, vp, sz, vp]
        L.moe_grouped_ffn.argtypes = [cfgp, vp, vp, vp, vp, wp, vp, vp, sz, vp]
        L.moe_shared_ffn.argtypes = [cfgp, vp, wp, vp, vp, sz, vp]
        L.moe_combine.argtypes = [cfgp, vp, vp, vp, vp, vp, vp]
        L.moe_forward.argtypes = [cfgp, vp, vp, fp, fp, wp, wp, vp, vp, vp, vp, vp, sz, vp]
        L.moe_forward_hostio.argtypes = [cfgp, vp, vp, fp, fp, wp, wp, vp, vp, sz, vp]
        L.moe_device_status.argtypes = [vp, vp, i32p]
        L.moe_permute_noalloc.argtypes = [cfgp, vp, vp, vp, vp, vp, vp]
        _lib = L
    return _lib


def status_string(status: int) -> str:
    return lib().gbmoe_status_string(status).decode()


def make_config(T, H, I, E, top_k, *, score="softmax", renormalize=True, n_group=1, topk_group=1,
                routed_scale=1.0, act="bf16", w="bf16", has_shared=False, I_shared=0, ffn_route="auto",
                gate_route="auto", combine_route="auto") -> Config:
    return Config(T, H, I, E, top_k, SOFTMAX if score == "softmax" else SIGMOID, int(bool(renormalize)), n_group,
                  topk_group, routed_scale, DTYPES[act], DTYPES[w], int(bool(has_shared)), I_shared,
                  ROUTES[ffn_route], GATES[gate_route], COMBINES[combine_route])


def _ptr(t):
    """Device (or host) address of a tensor, or None."""
    if t is None:
        return None
    return t.data_ptr()


def _stream(stream):
    if stream is not None:
        return ctypes.c_void_p(stream)
    import torch
    return ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)


def _check(status: int, call: str) -> None:
    if status != OK:
        raise GbmoeError(status, call)


def weights(w_gate, w_up, w_down, s_gate=None, s_up=None, s_down=None) -> ExpertWeights:
    """Pointer bundle of one set of expert weights (tensors must stay alive)."""
    return ExpertWeights(_ptr(w_gate), _ptr(w_up), _ptr(w_down), _ptr(s_gate), _ptr(s_up), _ptr(s_down))


def gate_route(cfg: Config) -> str:
    """Name of the gate route moe_route runs for cfg ("simt" or "tc")."""
    r = lib().gbmoe_gate_route(ctypes.byref(cfg))
    if r < 0:
        raise GbmoeError(r, "gbmoe_gate_route")
    return {v: k for k, v in GATES.items()}[r]


def check_config(cfg: Config) -> int:
    return lib().gbmoe_check_config(ctypes.byref(cfg))


def workspace_size(cfg: Config) -> int:
    return lib().gbmoe_workspace_size(ctypes.byref(cfg))


def ffn_route(cfg: Config, shared: bool = False) -> str:
    """Name of the FFN route moe_forward runs for cfg ("stream", "simt", "tc", "tc_dequant", "tc_fp8")."""
    r = lib().gbmoe_ffn_route(ctypes.byref(cfg), int(bool(shared)))
    if r < 0:
        raise GbmoeError(r, "gbmoe_ffn_route")
    return {v: k for k, v in ROUTES.items()}[r]


def moe_rmsnorm(cfg, x, gamma, eps, y, stream=None):
    _check(lib().moe_rmsnorm(ctypes.byref(cfg), _ptr(x), _ptr(gamma), float(eps), _ptr(y), _stream(stream)),
           "moe_rmsnorm")


def moe_route(cfg, x, w_router, logit_bias, select_bias, topk_ids, topk_w, ws, stream=None):
    _check(lib().moe_route(ctypes.byref(cfg), _ptr(x), _ptr(w_router), _ptr(logit_bias), _ptr(select_bias),
                           _ptr(topk_ids), _ptr(topk_w), _ptr(ws), ws.numel() * ws.element_size(),
                           _stream(stream)), "moe_route")


def moe_permute(cfg, topk_ids, counts, offsets, sorted_pair, pair_pos, ws, stream=None):
    _check(lib().moe_permute(ctypes.byref(cfg), _ptr(topk_ids), _ptr(counts), _ptr(offsets), _ptr(sorted_pair),
                             _ptr(pair_pos), _ptr(ws), ws.numel() * ws.element_size(), _stream(stream)),
           "moe_permute")


def moe_grouped_ffn(cfg, x, counts, offsets, sorted_pair, experts: ExpertWeights, y_pairs, ws, stream=None):
    _check(lib().moe_grouped_ffn(ctypes.byref(cfg), _ptr(x), _ptr(counts), _ptr(offsets), _ptr(sorted_pair),
                                 ctypes.byref(experts), _ptr(y_pairs), _ptr(ws), ws.numel() * ws.element_size(),
                                 _stream(stream)), "moe_grouped_ffn")


def moe_shared_ffn(cfg, x, shared: ExpertWeights, y_shared, ws, stream=None):
    _check(lib().moe_shared_ffn(ctypes.byref(cfg), _ptr(x), ctypes.byref(shared), _ptr(y_shared), _ptr(ws),
                                ws.numel() * ws.element_size(), _stream(stream)), "moe_shared_ffn")


def moe_combine(cfg, y_pairs, topk_w, pair_pos, y_shared, out, stream=None):
    _check(lib().moe_combine(ctypes.byref(cfg), _ptr(y_pairs), _ptr(topk_w), _ptr(pair_pos), _ptr(y_shared),
                             _ptr(out), _stream(stream)), "moe_combine")


def moe_forward(cfg, x, w_router, logit_bias, select_bias, experts: ExpertWeights, shared, out, ws,
                topk_ids=None, topk_w=None, counts=None, stream=None):
    sh = ctypes.byref(shared) if shared is not None else None
    _check(lib().moe_forward(ctypes.byref(cfg), _ptr(x), _ptr(w_router), _ptr(logit_bias), _ptr(select_bias),
                             ctypes.byref(experts), sh, _ptr(out), _ptr(topk_ids), _ptr(topk_w), _ptr(counts),
                             _ptr(ws), ws.numel() * ws.element_size(), _stream(stream)), "moe_forward")


def moe_forward_hostio(cfg, x_host, w_router, logit_bias, select_bias, experts: ExpertWeights, shared, out_host, ws,
                       stream=None):
    sh = ctypes.byref(shared) if shared is not None else None
    _check(lib().moe_forward_hostio(ctypes.byref(cfg), _ptr(x_host), _ptr(w_router), _ptr(logit_bias),
                                    _ptr(select_bias), ctypes.byref(experts), sh, _ptr(out_host), _ptr(ws),
                                    ws.numel() * ws.element_size(), _stream(stream)), "moe_forward_hostio")


def moe_device_status(ws, stream=None) -> int:
    st = ctypes.c_int32(0)
    _check(lib().moe_device_status(_ptr(ws), _stream(stream), ctypes.byref(st)), "moe_device_status")
    return st.value


def moe_permute_noalloc(cfg, topk_ids, counts, offsets, sorted_pair, pair_pos, stream=None):
    """moe_permute with the library's static scratch instead of a workspace."""
    _check(lib().moe_permute_noalloc(ctypes.byref(cfg), _ptr(topk_ids), _ptr(counts), _ptr(offsets),
                                     _ptr(sorted_pair), _ptr(pair_pos), _stream(stream)), "moe_permute_noalloc")
