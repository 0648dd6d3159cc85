"""Host-side checks of the C ABI (no GPU needed).

The library must load, export every function include/moe.h declares, and
reject bad arguments on the host before any CUDA call.
"""

import ctypes
import os
import re

import pytest

from paper_2603_02376_gb300 import _lib as L
from paper_2603_02376_gb300 import inputs as I

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def lib():
    if not os.path.exists(L.LIB_PATH):
        from paper_2603_02376_gb300 import build
        build.build_library()
    return L.load()


def header_functions():
    src = open(os.path.join(ROOT, "include", "moe.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(moe_[a-z_]+)\s*\(", src)))


def test_header_declares_the_boundary():
    names = header_functions()
    for n in ("moe_gate_topk", "moe_dispatch", "moe_expert_ffn", "moe_combine",
              "moe_layer_forward", "moe_router_logits"):
        assert n in names


def test_library_exports_every_declared_symbol(lib):
    for n in header_functions():
        assert hasattr(lib, n), n
    assert set(header_functions()) <= set(L.EXPORTS) | {"moe_status_string"}


def test_status_strings(lib):
    assert L.status_string(0) == "MOE_OK"
    assert L.status_string(L.MOE_ERR_TIMEOUT) == "MOE_ERR_TIMEOUT"
    assert L.status_string(99) == "MOE_ERR_UNKNOWN"


GOOD = dict(T=128, H=7168, E=256, k=8, I=2048, I_shared=2048, n_groups=8, topk_groups=4,
            gate=1, normalize=1, route_scale=2.5)


@pytest.mark.parametrize("bad", [
    dict(H=100), dict(H=192), dict(I=64), dict(E=0), dict(E=2000), dict(k=0), dict(k=33),
    dict(E=8, k=9, n_groups=1, topk_groups=1), dict(n_groups=7), dict(topk_groups=9),
    dict(topk_groups=0), dict(n_groups=8, topk_groups=1, k=33), dict(gate=2), dict(normalize=3),
    dict(T=-1), dict(I_shared=100), dict(route_scale=float("nan")),
    dict(n_groups=64, E=256),
])
def test_invalid_configs_rejected(lib, bad):
    c = L.config(**{**GOOD, **bad})
    assert L.moe_validate_config(c) == L.MOE_ERR_INVALID_ARG
    assert L.moe_workspace_size(c, L.exec_config()) == 0


def test_group_limit_k_constraint(lib):
    # 8 groups of 32, keep 1 group -> at most 32 experts can be picked
    assert L.moe_validate_config(L.config(**{**GOOD, "topk_groups": 1, "k": 32})) == 0
    c = L.config(**{**GOOD, "E": 64, "topk_groups": 1, "k": 9})  # groups of 8
    assert L.moe_validate_config(c) == L.MOE_ERR_INVALID_ARG


def test_valid_configs_and_workspace(lib):
    for wl in I.WORKLOADS.values():
        c = L.config_of(wl)
        assert L.moe_validate_config(c) == L.MOE_OK
        n = L.moe_workspace_size(c, L.exec_config())
        per_token = wl.k * (2 * wl.H + wl.I) * 2
        assert n >= wl.T * per_token
    c = L.config_of(I.PREFILL)
    seq = L.moe_workspace_size(c, L.exec_config())
    ovl = L.moe_workspace_size(c, L.exec_config(overlap=1, chunk_tokens=512))
    assert ovl > 0 and seq > 0
    assert L.moe_workspace_size(c, L.exec_config(overlap=1, chunk_axis=2)) == 0
    assert L.moe_workspace_size(c, L.exec_config(overlap=1, chunk_tokens=0)) == 0
    assert L.moe_workspace_size(c, L.exec_config(overlap=1, chunk_axis=1, n_expert_chunks=0)) == 0


def test_entry_points_reject_bad_arguments_without_a_gpu(lib):
    c = L.config(**GOOD)
    bad = L.config(**{**GOOD, "H": 100})
    z = ctypes.c_void_p(0)
    p = ctypes.c_void_p(0x1000)       # never dereferenced: validation fails first
    odd = ctypes.c_void_p(0x1002)     # misaligned
    cb = ctypes.byref
    assert lib.moe_router_logits(cb(bad), p, p, p, z, 0, z) == L.MOE_ERR_INVALID_ARG
    assert lib.moe_router_logits(cb(c), z, p, p, z, 0, z) == L.MOE_ERR_INVALID_ARG
    assert lib.moe_router_logits(cb(c), odd, p, p, z, 0, z) == L.MOE_ERR_INVALID_ARG
    assert lib.moe_gate_topk(cb(c), z, z, p, p, z) == L.MOE_ERR_INVALID_ARG
    assert lib.moe_gate_topk(cb(bad), p, z, p, p, z) == L.MOE_ERR_INVALID_ARG
    assert lib.moe_dispatch(cb(c), p, p, p, p, p, p, p, z, 0, z) == L.MOE_ERR_WORKSPACE
    assert lib.moe_dispatch(cb(c), z, p, p, p, p, p, p, p, 1 << 30, z) == L.MOE_ERR_INVALID_ARG
    assert lib.moe_expert_ffn(16, 100, 128, 1, p, p, p, p, p, p, 1 << 20, 0, z) == L.MOE_ERR_INVALID_ARG
    assert lib.moe_expert_ffn(16, 256, 128, 0, p, p, p, p, p, p, 1 << 20, 0, z) == L.MOE_ERR_INVALID_ARG
    assert lib.moe_expert_ffn(16, 256, 128, 1, p, p, p, p, p, z, 0, 0, z) == L.MOE_ERR_WORKSPACE
    assert lib.moe_expert_ffn(16, 256, 128, 1, odd, p, p, p, p, p, 1 << 20, 0, z) == L.MOE_ERR_INVALID_ARG
    assert lib.moe_expert_ffn(16, 256, 128, 1, p, p, p, p, p, p, 1 << 20, 2, z) == L.MOE_ERR_INVALID_ARG
    assert lib.moe_pack_weights(100, 64, p, p, z) == L.MOE_ERR_INVALID_ARG      # rows % 128
    assert lib.moe_pack_weights(128, 96, p, p, z) == L.MOE_ERR_INVALID_ARG      # K % 64
    assert lib.moe_pack_weights(128, 64, p, p, z) == L.MOE_ERR_INVALID_ARG      # W == W_packed
    assert lib.moe_pack_weights(128, 64, p, ctypes.c_void_p(0x1000 + 8192), z) == L.MOE_ERR_INVALID_ARG
    assert lib.moe_pack_weights(0, 64, z, z, z) == L.MOE_OK
    assert lib.moe_combine(cb(c), p, p, p, z, p, 2, z) == L.MOE_ERR_INVALID_ARG
    assert lib.moe_combine(cb(c), p, p, p, z, odd, 0, z) == L.MOE_ERR_INVALID_ARG
    ex = L.exec_config()
    W = L.moe_weights(0x1000, None, 0x1000, 0x1000, 0x1000, 0x1000)
    assert lib.moe_layer_forward(cb(c), cb(ex), cb(W), p, p, None, z, 0, z, z) == L.MOE_ERR_WORKSPACE
    Wn = L.moe_weights(0x1000, None, 0x1000, 0x1000, None, None)  # shared expert missing
    assert lib.moe_layer_forward(cb(c), cb(ex), cb(Wn), p, p, None, p, 1 << 40, z, z) == L.MOE_ERR_INVALID_ARG
    exb = L.exec_config(overlap=3)
    assert lib.moe_layer_forward(cb(c), cb(exb), cb(W), p, p, None, p, 1 << 40, z, z) == L.MOE_ERR_INVALID_ARG
    exc = L.exec_config(fuse_combine=2)
    assert lib.moe_layer_forward(cb(c), cb(exc), cb(W), p, p, None, p, 1 << 40, z, z) == L.MOE_ERR_INVALID_ARG
    assert L.moe_workspace_size(c, exc) == 0


def test_stack_entry_points_reject_bad_arguments_without_a_gpu(lib):
    c = L.config(**GOOD)
    z = ctypes.c_void_p(0)
    p = ctypes.c_void_p(0x1000)
    cb = ctypes.byref
    ex = L.exec_config()
    n1 = L.moe_workspace_size(c, ex)
    ns = L.moe_stack_workspace_size(c, ex)
    assert ns >= n1 + 2 * GOOD["T"] * GOOD["H"] * 2
    assert L.moe_stack_workspace_size(c, L.exec_config(out_fp32=1)) == 0   # bf16 chaining only
    W = (L.moe_weights * 2)(L.moe_weights(0x1000, None, 0x1000, 0x1000, 0x1000, 0x1000),
                           L.moe_weights(0x1000, None, 0x1000, 0x1000, 0x1000, 0x1000))
    S = lib.moe_stack_forward
    assert S(cb(c), cb(ex), W, 0, 1, p, p, p, 1 << 40, z, z) == L.MOE_ERR_INVALID_ARG   # no layers
    assert S(cb(c), cb(ex), W, 2, 2, p, p, p, 1 << 40, z, z) == L.MOE_ERR_INVALID_ARG   # rms_norm
    assert S(cb(c), cb(L.exec_config(out_fp32=1)), W, 2, 1, p, p, p, 1 << 40, z, z) == L.MOE_ERR_INVALID_ARG
    assert S(cb(c), cb(ex), W, 2, 1, p, p, z, 0, z, z) == L.MOE_ERR_WORKSPACE
    assert S(cb(c), cb(ex), None, 2, 1, p, p, p, 1 << 40, z, z) == L.MOE_ERR_INVALID_ARG
    h = ctypes.c_void_p()
    G = lib.moe_graph_create_stack
    assert G(cb(c), cb(ex), W, 2, 1, p, p, p, 1 << 40, z, None) == L.MOE_ERR_INVALID_ARG  # no handle
    assert G(cb(c), cb(ex), W, 0, 1, p, p, p, 1 << 40, z, cb(h)) == L.MOE_ERR_INVALID_ARG
    assert G(cb(c), cb(ex), W, 2, 1, p, p, z, 0, z, cb(h)) == L.MOE_ERR_WORKSPACE
    evs = (ctypes.c_void_p * L.MOE_N_STAGE_EVENTS)()
    ext = L.exec_config()
    ext.stage_events = ctypes.cast(evs, ctypes.POINTER(ctypes.c_void_p))
    assert G(cb(c), cb(ext), W, 2, 1, p, p, p, 1 << 40, z, cb(h)) == L.MOE_ERR_INVALID_ARG  # tracing
    assert h.value is None
    assert lib.moe_graph_launch(None, z) == L.MOE_ERR_INVALID_ARG
    assert lib.moe_graph_kernel_count(None) == 0
    lib.moe_graph_destroy(None)


def test_fused_combine_workspace():
    # fused combine: no y_perm [T*k, H] and no shared y; an fp32 [T, H] accumulator
    # only when the output is bf16 (an fp32 output is the accumulator itself)
    for wl in (I.DECODE, I.PREFILL):
        c = L.config_of(wl)
        plain = L.moe_workspace_size(c, L.exec_config(fuse_gather=0))
        f16 = L.moe_workspace_size(c, L.exec_config(fuse_gather=0, fuse_combine=1))
        f32 = L.moe_workspace_size(c, L.exec_config(fuse_gather=0, fuse_combine=1, out_fp32=1))
        T, H, k = wl.T, wl.H, wl.k
        assert plain - f32 >= T * k * H * 4 + T * H * 4 - T * k * 4 - 4096
        assert f16 - f32 >= T * H * 4


def test_exec_options_validated_on_the_host():
    # dispatch forms 0, 1, 2 are accepted (same workspace for 0 and 2: x_perm is
    # written either by the dispatch kernel or by GEMM1's pack warps); 3 is not;
    # a trace buffer or timeline events need a positive count
    c = L.config_of(I.PREFILL)
    ws0 = L.moe_workspace_size(c, L.exec_config(fuse_gather=0))
    assert ws0 > 0 and L.moe_workspace_size(c, L.exec_config(fuse_gather=2)) == ws0
    assert L.moe_workspace_size(c, L.exec_config(fuse_gather=3)) == 0
    ex = L.exec_config()
    ex.unit_trace, ex.unit_trace_cap = 0x1000, 0
    assert L.moe_workspace_size(c, ex) == 0
    ex = L.exec_config()
    ex.unit_trace_cap = -1
    assert L.moe_workspace_size(c, ex) == 0
    # the traced GEMM: 0 or 1 (GEMM1) or 2 (GEMM2)
    for g, ok in ((0, True), (1, True), (2, True), (3, False), (-1, False)):
        ex = L.exec_config(unit_trace_gemm=g)
        assert (L.moe_workspace_size(c, ex) == ws0 and ws0 > 0) if ok else \
            L.moe_workspace_size(c, ex) == 0, g
    ex = L.exec_config(overlap=1)
    ex.n_pipe_events = -1
    assert L.moe_workspace_size(c, ex) == 0


def test_fp8_entry_points_reject_bad_arguments_without_a_gpu(lib):
    c = L.config(**GOOD)
    z = ctypes.c_void_p(0)
    p = ctypes.c_void_p(0x1000)
    q = ctypes.c_void_p(0x100000)     # a second buffer far from p
    odd = ctypes.c_void_p(0x1008)     # 8-byte aligned only
    cb = ctypes.byref
    Q = lib.moe_quantize_fp8
    assert Q(16, 100, p, q, q, z) == L.MOE_ERR_INVALID_ARG          # K % 16
    assert Q(16, 8, p, q, q, z) == L.MOE_ERR_INVALID_ARG            # K < 16
    assert Q(-1, 128, p, q, q, z) == L.MOE_ERR_INVALID_ARG
    assert Q(16, 128, p, p, q, z) == L.MOE_ERR_INVALID_ARG          # in and out overlap
    assert Q(16, 128, odd, q, q, z) == L.MOE_ERR_INVALID_ARG
    assert Q(16, 128, p, q, z, z) == L.MOE_ERR_INVALID_ARG          # no scale buffer
    assert Q(0, 128, z, z, z, z) == L.MOE_OK
    F = lib.moe_expert_ffn_fp8
    args = [p] * 9                    # x_q .. y_perm; the workspace follows
    assert F(16, 100, 128, 1, *args, q, 1 << 20, z) == L.MOE_ERR_INVALID_ARG
    assert F(16, 256, 96, 1, *args, q, 1 << 20, z) == L.MOE_ERR_INVALID_ARG
    assert F(16, 256, 128, 1, *args, z, 0, z) == L.MOE_ERR_WORKSPACE
    assert F(16, 256, 128, 1, *args, ctypes.c_void_p(0x100010), 1 << 20, z) == L.MOE_ERR_WORKSPACE
    assert F(16, 256, 128, 1, z, *([p] * 8), q, 1 << 20, z) == L.MOE_ERR_INVALID_ARG
    assert F(0, 256, 128, 1, *([z] * 9), z, 0, z) == L.MOE_OK
    n = lib.moe_expert_ffn_fp8_workspace_size(16, 128)
    assert n >= 16 * 128 * 3 + 16 * 4 and n % 256 == 0
    # layer forward: fp8 needs the weight row scales and excludes the packed layout
    ex8 = L.exec_config(fp8=1)
    W = L.moe_weights(0x1000, None, 0x1000, 0x1000, 0x1000, 0x1000, 0)
    assert lib.moe_layer_forward(cb(c), cb(ex8), cb(W), p, p, None, p, 1 << 40, z, z) == L.MOE_ERR_INVALID_ARG
    Wp = L.moe_weights(0x1000, None, 0x1000, 0x1000, 0x1000, 0x1000, 1, 0x1000, 0x1000, 0x1000, 0x1000)
    assert lib.moe_layer_forward(cb(c), cb(ex8), cb(Wp), p, p, None, p, 1 << 40, z, z) == L.MOE_ERR_UNSUPPORTED
    assert lib.moe_layer_forward(cb(c), cb(L.exec_config(fp8=3)), cb(W8 := L.moe_weights(
        0x1000, None, 0x1000, 0x1000, 0x1000, 0x1000, 0, 0x1000, 0x1000, 0x1000, 0x1000)),
        p, p, None, p, 1 << 40, z, z) == L.MOE_ERR_INVALID_ARG                 # no such form
    W8 = L.moe_weights(0x1000, None, 0x1000, 0x1000, 0x1000, 0x1000, 0, 0x1000, 0x1000, 0x1000, 0x1000)
    assert lib.moe_layer_forward(cb(c), cb(ex8), cb(W8), p, p, None, z, 0, z, z) == L.MOE_ERR_WORKSPACE
    # the fp8 layout adds the quantized copies; its x_perm is half the bf16 one,
    # and its row-major x_perm and h have none of the bf16 tile-packed buffers'
    # 16 padding rows per expert (16 for the shared expert's h)
    for wl in (I.DECODE, I.PREFILL):
        cw = L.config_of(wl)
        n16 = L.moe_workspace_size(cw, L.exec_config(fuse_gather=0))
        n8 = L.moe_workspace_size(cw, L.exec_config(fuse_gather=0, fp8=1))
        tk = wl.T * wl.k
        pad = 16 * wl.E * 2 * (wl.H + wl.I) + 16 * 2 * wl.I_shared
        assert n16 >= (tk + 16 * wl.E) * 2 * (wl.H + wl.I)
        assert n8 - n16 >= wl.T * wl.H + tk * wl.I - tk * wl.H - pad - (1 << 16)


def test_fp8_block_entry_points_reject_bad_arguments_without_a_gpu(lib):
    c = L.config(**GOOD)
    z = ctypes.c_void_p(0)
    p = ctypes.c_void_p(0x1000)
    q = ctypes.c_void_p(0x100000)
    odd = ctypes.c_void_p(0x1008)
    cb = ctypes.byref
    QB = lib.moe_quantize_fp8_blocks
    assert QB(16, 100, p, q, q, 16, z) == L.MOE_ERR_INVALID_ARG       # K % 128
    assert QB(16, 64, p, q, q, 16, z) == L.MOE_ERR_INVALID_ARG        # K < 128
    assert QB(16, 256, p, q, q, 1, z) == L.MOE_ERR_INVALID_ARG        # sf_ld < K / 128
    assert QB(16, 128, p, p, q, 16, z) == L.MOE_ERR_INVALID_ARG       # in and out overlap
    assert QB(16, 128, odd, q, q, 16, z) == L.MOE_ERR_INVALID_ARG
    assert QB(16, 128, p, q, z, 16, z) == L.MOE_ERR_INVALID_ARG       # no exponent buffer
    assert QB(0, 128, z, z, z, 1, z) == L.MOE_OK
    QW = lib.moe_quantize_fp8_weight_blocks
    assert QW(100, 128, p, q, q, z) == L.MOE_ERR_INVALID_ARG          # rows % 128
    assert QW(128, 96, p, q, q, z) == L.MOE_ERR_INVALID_ARG           # K % 128
    assert QW(128 * 65536, 128, p, q, q, z) == L.MOE_ERR_INVALID_ARG  # grid rows
    assert QW(128, 128, p, p, q, z) == L.MOE_ERR_INVALID_ARG
    assert QW(0, 128, z, z, z, z) == L.MOE_OK
    F = lib.moe_expert_ffn_fp8_blocks
    a = lambda ld=2, idx=z: [p, p, ld, idx, p, p, p, p, p, p]    # x_q .. y_perm
    assert F(16, 100, 128, 1, *a(), q, 1 << 20, z) == L.MOE_ERR_INVALID_ARG     # H % 128
    assert F(16, 256, 96, 1, *a(), q, 1 << 20, z) == L.MOE_ERR_INVALID_ARG      # I % 128
    assert F(16, 256, 128, 1, *a(ld=1), q, 1 << 20, z) == L.MOE_ERR_INVALID_ARG  # ld < H / 128
    assert F(16, 256, 128, 1, *a(idx=p), ctypes.c_void_p(0x100010), 1 << 20, z) == \
        L.MOE_ERR_WORKSPACE
    assert F(16, 256, 128, 1, *a(), z, 0, z) == L.MOE_ERR_WORKSPACE
    assert F(16, 256, 128, 1, z, *a()[1:], q, 1 << 20, z) == L.MOE_ERR_INVALID_ARG
    assert F(0, 256, 128, 1, z, z, 2, z, z, z, z, z, z, z, z, 0, z) == L.MOE_OK
    n = lib.moe_expert_ffn_fp8_blocks_workspace_size(16, 256)
    assert n >= 16 * 256 * 3 + 2 * 16 and n % 256 == 0
    # layer forward: block scales need whole 128-blocks and the exponent arrays
    W8 = L.moe_weights(0x1000, None, 0x1000, 0x1000, 0x1000, 0x1000, 0, 0x1001, 0x1001, 0x1001,
                       0x1001)                        # byte arrays: any alignment
    exb = L.exec_config(fp8=2)
    assert lib.moe_layer_forward(cb(c), cb(exb), cb(W8), p, p, None, z, 0, z, z) == L.MOE_ERR_WORKSPACE
    Wn = L.moe_weights(0x1000, None, 0x1000, 0x1000, 0x1000, 0x1000, 0, 0x1001, None, 0x1001,
                       0x1001)
    assert lib.moe_layer_forward(cb(c), cb(exb), cb(Wn), p, p, None, z, 0, z, z) == L.MOE_ERR_INVALID_ARG
    # the block layout: per-row scale arrays replaced by exponent bytes, and its
    # row-major e4m3 x_perm and hq without the row-scaled form's tile-packing
    # padding (16 rows per expert, 16 for the shared expert's hq)
    for wl in (I.DECODE, I.PREFILL):
        cw = L.config_of(wl)
        n8 = L.moe_workspace_size(cw, L.exec_config(fuse_gather=0, fp8=1))
        nb = L.moe_workspace_size(cw, L.exec_config(fuse_gather=0, fp8=2))
        tk = wl.T * wl.k
        extra = wl.H // 128 * wl.T + wl.I // 128 * tk + wl.I_shared // 128 * wl.T
        pad = 16 * wl.E * (wl.H + wl.I) + 16 * wl.I_shared
        assert nb - n8 == pytest.approx(extra - 4 * (wl.T + tk + wl.T) - pad, abs=4096)


def test_empty_batch_is_a_no_op(lib):
    c = L.config(**{**GOOD, "T": 0})
    z = ctypes.c_void_p(0)
    cb = ctypes.byref
    assert lib.moe_router_logits(cb(c), z, z, z, z, 0, z) == L.MOE_OK
    assert lib.moe_gate_topk(cb(c), z, z, z, z, z) == L.MOE_OK
    assert lib.moe_combine(cb(c), z, z, z, z, z, 0, z) == L.MOE_OK
    assert lib.moe_expert_ffn(0, 256, 128, 4, z, z, z, z, z, z, 0, 0, z) == L.MOE_OK
    W = L.moe_weights(0x1000, None, 0x1000, 0x1000, 0x1000, 0x1000)
    assert lib.moe_layer_forward(cb(c), cb(L.exec_config()), cb(W), z, z, None, z, 0, z, z) == L.MOE_OK


def test_binding_names_match_header():
    for n in header_functions():
        assert hasattr(L, n), n
