"""CPU checks of the C-ABI library: it loads, exports every function the
header declares, and rejects bad arguments on the host (no GPU involved:
every case below returns before any CUDA call)."""
import ctypes
import os
import re

import pytest

import paper_2607_12875_gb300 as gb
import synth

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "gbmoe.h")


def declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return re.findall(r"^[A-Za-z_][\w \t\*]*?\b((?:gbmoe|moe)_\w+)\s*\(", text, flags=re.M)


@pytest.fixture(scope="module")
def lib():
    if not os.path.exists(gb.LIB_PATH):
        from paper_2607_12875_gb300 import build
        build.build()
    return gb.lib()


def test_header_declares_the_layer_entry_points():
    names = declared_functions()
    for n in ("moe_route", "moe_permute", "moe_grouped_ffn", "moe_combine", "moe_forward"):
        assert n in names
    assert set(names) == set(gb.EXPORTS)


def test_library_exports_every_declared_function(lib):
    for name in declared_functions():
        assert hasattr(lib, name), name


def cfg_of(wid, **kw):
    w = synth.WORKLOADS[wid]
    c = gb.make_config(w.T, w.H, w.I, w.E, w.top_k, score=w.score, renormalize=w.renormalize, n_group=w.n_group,
                       topk_group=w.topk_group, routed_scale=w.routed_scale, act=w.act, w=w.wq,
                       has_shared=w.has_shared, I_shared=w.I_shared)
    for k, v in kw.items():
        setattr(c, k, v)
    return c


@pytest.mark.parametrize("wid", [1, 2, 3, 4, 5, 6])
def test_workload_configs_are_valid(lib, wid):
    c = cfg_of(wid)
    assert gb.check_config(c) == gb.OK
    assert gb.workspace_size(c) > 0


@pytest.mark.parametrize("change,status", [
    (dict(H=300), gb.EUNSUPPORTED),
    (dict(H=0), gb.EINVAL),
    (dict(I=100), gb.EUNSUPPORTED),
    (dict(top_k=9), gb.EINVAL),
    (dict(E=1024, top_k=2), gb.EUNSUPPORTED),
    (dict(T=-1), gb.EINVAL),
    (dict(score=7), gb.EINVAL),
    (dict(act_dtype=2), gb.EINVAL),
    (dict(w_dtype=5), gb.EINVAL),
    (dict(ffn_route=9), gb.EINVAL),
    (dict(ffn_route=gb.FFN_TC), gb.EUNSUPPORTED),  # fp32 activations have no tensor-core route
    (dict(ffn_route=gb.FFN_TC_DEQUANT), gb.EUNSUPPORTED),
    (dict(ffn_route=gb.FFN_TC_FP8), gb.EUNSUPPORTED),  # fp8 route needs fp8 weights and bf16 activations
    (dict(ffn_route=gb.FFN_TC_PAIR), gb.EUNSUPPORTED),
    (dict(ffn_route=gb.FFN_TC_PAIR_DEQUANT), gb.EUNSUPPORTED),
    (dict(ffn_route=8), gb.EINVAL),
    (dict(gate_route=3), gb.EINVAL),
    (dict(gate_route=gb.GATE_TC), gb.EUNSUPPORTED),  # the tensor-core gate takes bf16 activations
    (dict(combine_route=3), gb.EINVAL),
])
def test_invalid_configs_are_rejected(lib, change, status):
    c = cfg_of(1, **change)
    assert gb.check_config(c) == status
    assert gb.workspace_size(c) == 0


def test_fp8_configs_keep_scale_offsets_in_32_bits(lib):
    """The fp8 route indexes its scale tensors with 32-bit offsets: a batch
    whose activation scales would reach 2^31 entries is refused (P * H/128 >=
    2^31 at H = 7168 from P = 38.35 M pairs), one just below passes."""
    kb = synth.WORKLOADS[4].H // 128
    limit_pairs = (2 ** 31 - 1) // kb
    below = cfg_of(4, T=limit_pairs // 8)
    above = cfg_of(4, T=limit_pairs // 8 + 1)
    assert below.T * 8 * kb <= 2 ** 31 - 1 < above.T * 8 * kb
    assert gb.check_config(below) == gb.OK
    assert gb.check_config(above) == gb.EUNSUPPORTED
    assert gb.check_config(cfg_of(1, T=limit_pairs)) == gb.OK  # fp32 weights: no such limit


def test_sigmoid_group_rules(lib):
    c = cfg_of(4)
    for ch in (dict(n_group=7), dict(topk_group=9), dict(top_k=200, topk_group=1)):
        bad = cfg_of(4, **ch)
        assert gb.check_config(bad) == gb.EINVAL, ch
    assert gb.check_config(c) == gb.OK
    assert gb.check_config(cfg_of(4, ffn_route=gb.FFN_TC_FP8)) == gb.OK
    assert gb.check_config(cfg_of(5, ffn_route=gb.FFN_TC_FP8)) == gb.EUNSUPPORTED  # int4 weights


class FakePtr:
    """An aligned non-null address the library never dereferences here."""

    def __init__(self, nbytes=1 << 20):
        self.buf = ctypes.create_string_buffer(nbytes + 256)
        self.addr = (ctypes.addressof(self.buf) + 255) & ~255
        self.nbytes = nbytes

    def data_ptr(self):
        return self.addr

    def numel(self):
        return self.nbytes

    def element_size(self):
        return 1


def test_entry_points_reject_bad_arguments_before_launching(lib):
    c = cfg_of(1)
    p = FakePtr()
    small_ws = FakePtr(64)
    with pytest.raises(gb.GbmoeError) as e:
        gb.moe_route(c, None, p, None, None, p, p, p, stream=0)
    assert e.value.status == gb.EINVAL
    with pytest.raises(gb.GbmoeError) as e:
        gb.moe_route(c, p, p, None, None, p, p, small_ws, stream=0)
    assert e.value.status == gb.EWORKSPACE
    with pytest.raises(gb.GbmoeError) as e:
        gb.moe_permute(c, p, None, p, p, p, p, stream=0)
    assert e.value.status == gb.EINVAL
    w = gb.weights(p, None, p)
    with pytest.raises(gb.GbmoeError) as e:
        gb.moe_grouped_ffn(c, p, p, p, p, w, p, p, stream=0)
    assert e.value.status == gb.EINVAL
    with pytest.raises(gb.GbmoeError) as e:
        gb.moe_shared_ffn(c, p, gb.weights(p, p, p), p, p, stream=0)  # config has no shared expert
    assert e.value.status == gb.EINVAL
    c4 = cfg_of(4)
    with pytest.raises(gb.GbmoeError) as e:
        gb.moe_forward(c4, p, p, None, None, gb.weights(p, p, p), gb.weights(p, p, p), p, p, stream=0)  # no fp8 scales
    assert e.value.status == gb.EINVAL
    assert gb.status_string(gb.EDEVICE_TIMEOUT) == "device-side wait timed out"


@pytest.mark.parametrize("wid", [4, 5, 6])
def test_dequant_route_workspace_holds_bf16_weight_copies(lib, wid):
    """Forcing the decode-once route adds one bf16 copy of every expert's
    gate, up and down matrices (and of the shared expert's) to the workspace,
    and drops the sorted copy of x that the in-GEMM decode route reads (the
    bf16 GEMM after the decode pass gathers its rows itself)."""
    wl = synth.WORKLOADS[wid]
    tc = gb.workspace_size(cfg_of(wid, ffn_route=gb.FFN_TC))
    dq = gb.workspace_size(cfg_of(wid, ffn_route=gb.FFN_TC_DEQUANT))
    copies = 3 * wl.E * wl.H * wl.I * 2 + (3 * wl.H * wl.I_shared * 2 if wl.has_shared else 0)
    sorted_x = wl.P * wl.H * 2
    assert copies - sorted_x <= dq - tc <= copies - sorted_x + 3 * 256


def test_forced_stream_route_checks_the_shared_expert_before_launching(lib):
    """With both FFN problems forced onto the streaming route, a shared expert
    whose rows do not fit the streaming kernel's shared memory is refused
    before anything is enqueued (the routed problem alone would fit)."""
    c = cfg_of(4, T=4, ffn_route=gb.FFN_STREAM, I_shared=16384)
    assert gb.check_config(c) == gb.OK
    assert gb.ffn_route(c) == "stream" and gb.ffn_route(c, shared=True) == "stream"
    p = FakePtr()
    ws = FakePtr(gb.workspace_size(c))
    w = gb.weights(p, p, p, p, p, p)
    with pytest.raises(gb.GbmoeError) as e:
        gb.moe_forward(c, p, p, None, None, w, w, p, ws, stream=0)
    assert e.value.status == gb.EUNSUPPORTED
    with pytest.raises(gb.GbmoeError) as e:
        gb.moe_shared_ffn(c, p, w, p, ws, stream=0)
    assert e.value.status == gb.EUNSUPPORTED
    c.I_shared = 2048  # fits: the same call passes the checks (it would launch, so it is not made here)
    assert gb.check_config(c) == gb.OK


def test_last_cuda_error_starts_clear(lib):
    """No CUDA call has failed in this thread: the recorded code is 0, and a
    call that fails on its arguments (not in CUDA) leaves it 0."""
    assert gb.lib().gbmoe_last_cuda_error() == 0
    assert gb.check_config(cfg_of(1, T=-1)) == gb.EINVAL
    assert gb.lib().gbmoe_last_cuda_error() == 0


def test_rmsnorm_rejects_bad_arguments_before_launching(lib):
    """Null, misaligned or overlapping buffers and a negative or non-finite
    eps are refused on the host (nothing reaches the GPU here)."""
    c = cfg_of(1)  # T=64, H=256, fp32 activations: rows of 1 KB
    x, g, y = FakePtr(), FakePtr(), FakePtr()
    for args in [(None, g, 1e-6, y), (x, None, 1e-6, y), (x, g, 1e-6, None), (x, g, -1.0, y),
                 (x, g, float("nan"), y), (x, g, float("inf"), y), (x, g, 1e-6, x)]:
        with pytest.raises(gb.GbmoeError) as e:
            gb.moe_rmsnorm(c, *args, stream=0)
        assert e.value.status == gb.EINVAL

    class Shifted(FakePtr):  # 8 bytes past an aligned address
        def data_ptr(self):
            return self.addr + 8
    with pytest.raises(gb.GbmoeError) as e:
        gb.moe_rmsnorm(c, Shifted(), g, 1e-6, y, stream=0)
    assert e.value.status == gb.EINVAL
    # T = 0: nothing to do, no pointer is needed
    assert lib.moe_rmsnorm(ctypes.byref(cfg_of(1, T=0)), None, None, ctypes.c_float(1e-6), None, None) == gb.OK


def test_sorted_copy_of_x_only_where_a_gemm_reads_it(lib):
    """The one-CTA bf16 GEMM gathers its rows from x, so its workspace holds
    no sorted copy of x; the CTA-pair GEMM and the one-CTA GEMM on quantised
    weights read one (P x H activations)."""
    wl = synth.WORKLOADS[3]
    copy = wl.P * wl.H * 2
    one = gb.workspace_size(cfg_of(3, ffn_route=gb.FFN_TC))
    pair = gb.workspace_size(cfg_of(3, ffn_route=gb.FFN_TC_PAIR))
    assert copy <= pair - one <= copy + 256
    w5 = synth.WORKLOADS[5]
    in_gemm = gb.workspace_size(cfg_of(5, ffn_route=gb.FFN_TC))             # decodes int4 in the GEMM
    dq = gb.workspace_size(cfg_of(5, ffn_route=gb.FFN_TC_DEQUANT))         # bf16 copy, then gathers
    weights_copy = 3 * w5.E * w5.H * w5.I * 2
    assert dq - in_gemm == pytest.approx(weights_copy - w5.P * w5.H * 2, abs=512)


def test_hostio_checks_the_layer_arguments_before_copying(lib):
    """moe_forward_hostio runs moe_forward's own checks (router weights,
    expert weights, scales, routes) before it enqueues the host-to-device
    copy of x: a bad argument returns with nothing enqueued."""
    c = cfg_of(1)
    x_host, out_host, p = FakePtr(), FakePtr(), FakePtr()
    ws = FakePtr(gb.workspace_size(c))
    w = gb.weights(p, p, p)
    with pytest.raises(gb.GbmoeError) as e:
        gb.moe_forward_hostio(c, x_host, None, None, None, w, None, out_host, ws, stream=0)  # no router weights
    assert e.value.status == gb.EINVAL
    with pytest.raises(gb.GbmoeError) as e:
        gb.moe_forward_hostio(c, x_host, p, None, None, gb.weights(p, None, p), None, out_host, ws, stream=0)
    assert e.value.status == gb.EINVAL
    c4 = cfg_of(4, T=16)  # fp8 weights without their scales
    ws4 = FakePtr(gb.workspace_size(c4))
    with pytest.raises(gb.GbmoeError) as e:
        gb.moe_forward_hostio(c4, x_host, p, None, None, gb.weights(p, p, p), gb.weights(p, p, p), out_host, ws4,
                              stream=0)
    assert e.value.status == gb.EINVAL
