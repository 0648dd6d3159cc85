"""ctypes binding of libmoe.so: the C ABI of include/moe.h, same names.

Argument marshalling only: torch tensors are passed as raw device pointers
(data_ptr) and streams as cudaStream_t handles; every step runs in the
library's CUDA kernels. A non-OK status raises MoeError. Loading fails loudly
when the library has not been built.
"""

from __future__ import annotations

import ctypes
import os

PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(PKG, "libmoe.so")

MOE_OK = 0
MOE_ERR_INVALID_ARG = 1
MOE_ERR_UNSUPPORTED = 2
MOE_ERR_WORKSPACE = 3
MOE_ERR_CUDA = 4
MOE_ERR_TIMEOUT = 5
MOE_ERR_DEVICE_CHECK = 6
MOE_GATE_SOFTMAX = 0
MOE_GATE_SIGMOID = 1

EXPORTS = ("moe_status_string", "moe_validate_config", "moe_workspace_size",
           "moe_router_workspace_size", "moe_dispatch_workspace_size",
           "moe_expert_ffn_workspace_size", "moe_router_logits", "moe_gate_topk", "moe_dispatch",
           "moe_expert_ffn", "moe_combine", "moe_layer_forward", "moe_check_errors",
           "moe_launch_count", "moe_shutdown", "moe_dispatch_noalloc",
           "moe_testing_expert_ffn_stall", "moe_pack_weights", "moe_quantize_fp8",
           "moe_expert_ffn_fp8", "moe_expert_ffn_fp8_workspace_size", "moe_stack_workspace_size",
           "moe_stack_forward", "moe_rms_norm", "moe_graph_create_stack", "moe_graph_launch",
           "moe_graph_kernel_count", "moe_graph_destroy", "moe_quantize_fp8_blocks",
           "moe_quantize_fp8_weight_blocks", "moe_expert_ffn_fp8_blocks",
           "moe_expert_ffn_fp8_blocks_workspace_size", "moe_testing_fail_stage",
           "moe_testing_tiled_chunk")
MOE_DISPATCH_NOALLOC_MAX_ENTRIES = 131072


class MoeError(RuntimeError):
    def __init__(self, status: int, where: str):
        super().__init__(f"{where}: {status_string(status)} ({status})")
        self.status = status


class moe_config(ctypes.Structure):
    _fields_ = [(n, ctypes.c_int32) for n in
                ("T", "H", "E", "k", "I", "I_shared", "n_groups", "topk_groups", "gate",
                 "normalize")] + [("route_scale", ctypes.c_float)]


class moe_exec(ctypes.Structure):
    _fields_ = [(n, ctypes.c_int32) for n in
                ("overlap", "chunk_tokens", "chunk_axis", "n_expert_chunks", "out_fp32",
                 "fuse_gather")] + \
               [("stage_events", ctypes.POINTER(ctypes.c_void_p)), ("fp8", ctypes.c_int32),
                ("fuse_combine", ctypes.c_int32), ("unit_trace", ctypes.c_void_p),
                ("unit_trace_cap", ctypes.c_int32),
                ("pipe_events", ctypes.POINTER(ctypes.c_void_p)), ("n_pipe_events", ctypes.c_int32),
                ("unit_trace_gemm", ctypes.c_int32)]


STAGES = ("start", "router", "gate", "permute", "dispatch", "gemm1", "gemm2", "shared_gemm1",
          "shared_gemm2", "combine")
MOE_N_STAGE_EVENTS = len(STAGES)


class moe_weights(ctypes.Structure):
    _fields_ = [(n, ctypes.c_void_p) for n in ("Wr", "bias", "W13", "W2", "Ws13", "Ws2")] + \
               [("packed", ctypes.c_int32)] + \
               [(n, ctypes.c_void_p) for n in ("W13_scale", "W2_scale", "Ws13_scale",
                                               "Ws2_scale")]


class moe_aux(ctypes.Structure):
    _fields_ = [(n, ctypes.c_void_p) for n in ("logits", "topk_idx", "topk_w", "counts")]


_lib = None


def load(path: str = LIB_PATH) -> ctypes.CDLL:
    """Load libmoe.so (once). Raises if it has not been built."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(path):
        raise RuntimeError(f"{path} is missing: build it with __graft_entry__.build() "
                           "(python -m paper_2603_02376_gb300.build)")
    lib = ctypes.CDLL(path)
    P, I32, SZ, S = ctypes.c_void_p, ctypes.c_int32, ctypes.c_size_t, ctypes.c_int
    cfgp = ctypes.POINTER(moe_config)
    exp = ctypes.POINTER(moe_exec)
    sig = {
        "moe_status_string": (ctypes.c_char_p, [S]),
        "moe_validate_config": (S, [cfgp]),
        "moe_workspace_size": (SZ, [cfgp, exp]),
        "moe_router_workspace_size": (SZ, [cfgp]),
        "moe_dispatch_workspace_size": (SZ, [cfgp]),
        "moe_expert_ffn_workspace_size": (SZ, [I32, I32]),
        "moe_router_logits": (S, [cfgp, P, P, P, P, SZ, P]),
        "moe_gate_topk": (S, [cfgp, P, P, P, P, P]),
        "moe_dispatch": (S, [cfgp, P, P, P, P, P, P, P, P, SZ, P]),
        "moe_dispatch_noalloc": (S, [cfgp, P, P, P, P, P, P, P, P]),
        "moe_expert_ffn": (S, [I32, I32, I32, I32, P, P, P, P, P, P, SZ, I32, P]),
        "moe_pack_weights": (S, [ctypes.c_int64, I32, P, P, P]),
        "moe_quantize_fp8": (S, [ctypes.c_int64, I32, P, P, P, P]),
        "moe_expert_ffn_fp8_workspace_size": (SZ, [I32, I32]),
        "moe_expert_ffn_fp8": (S, [I32, I32, I32, I32, P, P, P, P, P, P, P, P, P, P, SZ, P]),
        "moe_quantize_fp8_blocks": (S, [ctypes.c_int64, I32, P, P, P, ctypes.c_int64, P]),
        "moe_quantize_fp8_weight_blocks": (S, [ctypes.c_int64, I32, P, P, P, P]),
        "moe_expert_ffn_fp8_blocks_workspace_size": (SZ, [I32, I32]),
        "moe_expert_ffn_fp8_blocks": (S, [I32, I32, I32, I32, P, P, ctypes.c_int64, P, P, P, P,
                                          P, P, P, P, SZ, P]),
        "moe_combine": (S, [cfgp, P, P, P, P, P, I32, P]),
        "moe_testing_expert_ffn_stall": (S, [I32, I32, I32, I32, P, P, P, P, P, P, SZ,
                                             ctypes.c_int64, ctypes.c_int64, P]),
        "moe_layer_forward": (S, [cfgp, exp, ctypes.POINTER(moe_weights), P, P,
                                  ctypes.POINTER(moe_aux), P, SZ, P, P]),
        "moe_stack_workspace_size": (SZ, [cfgp, exp]),
        "moe_rms_norm": (S, [ctypes.c_int64, I32, P, P, P]),
        "moe_stack_forward": (S, [cfgp, exp, ctypes.POINTER(moe_weights), I32, I32, P, P, P, SZ,
                                  P, P]),
        "moe_graph_create_stack": (S, [cfgp, exp, ctypes.POINTER(moe_weights), I32, I32, P, P, P,
                                       SZ, P, ctypes.POINTER(ctypes.c_void_p)]),
        "moe_graph_launch": (S, [P, P]),
        "moe_graph_kernel_count": (ctypes.c_uint64, [P]),
        "moe_graph_destroy": (None, [P]),
        "moe_check_errors": (S, [P]),
        "moe_launch_count": (ctypes.c_uint64, []),
        "moe_shutdown": (None, []),
        "moe_testing_fail_stage": (S, [I32]),
        "moe_testing_tiled_chunk": (S, [I32, I32, I32, I32, I32, I32, I32,
                                        ctypes.POINTER(ctypes.c_int64)]),
    }
    for name, (res, args) in sig.items():
        f = getattr(lib, name)
        f.restype = res
        f.argtypes = args
    _lib = lib
    return lib


def status_string(status: int) -> str:
    try:
        return load().moe_status_string(status).decode()
    except Exception:  # the library itself may be what failed to load
        return f"status {status}"


def moe_status_string(status: int) -> str:
    return load().moe_status_string(status).decode()


def _check(status: int, where: str) -> None:
    if status != MOE_OK:
        raise MoeError(status, where)


def _ptr(t):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _stream(stream):
    if stream is None:
        import torch
        stream = torch.cuda.current_stream()
    return ctypes.c_void_p(int(getattr(stream, "cuda_stream", stream)))


def config(T, H, E, k, I, I_shared=0, n_groups=1, topk_groups=1, gate=MOE_GATE_SIGMOID,
           normalize=1, route_scale=1.0) -> moe_config:
    return moe_config(T, H, E, k, I, I_shared, n_groups, topk_groups, gate, normalize,
                      route_scale)


def config_of(wl, T=None) -> moe_config:
    """moe_config of an inputs.Workload (optionally with another token count)."""
    return config(wl.T if T is None else T, wl.H, wl.E, wl.k, wl.I, wl.I_shared, wl.n_groups,
                  wl.topk_groups, wl.gate, wl.normalize, wl.route_scale)


UNIT_TRACE_FIELDS = 5


def exec_config(overlap=0, chunk_tokens=512, chunk_axis=0, n_expert_chunks=8, out_fp32=0,
                fuse_gather=1, stage_events=None, fp8=0, fuse_combine=0, unit_trace=None,
                pipe_events=None, unit_trace_gemm=1):
    """moe_exec; stage_events: a list of MOE_N_STAGE_EVENTS torch.cuda.Event (or None);
    unit_trace: an int64 device tensor [cap, UNIT_TRACE_FIELDS] (or None), filled for
    GEMM1 (unit_trace_gemm 1) or GEMM2 (2); pipe_events: a list of timing
    torch.cuda.Event for a pipelined forward's timeline (or None)."""
    cap = 0 if unit_trace is None else unit_trace.shape[0]
    ex = moe_exec(overlap, chunk_tokens, chunk_axis, n_expert_chunks, out_fp32, fuse_gather, None,
                  int(fp8), int(fuse_combine),
                  None if unit_trace is None else unit_trace.data_ptr(), cap, None, 0,
                  int(unit_trace_gemm))
    if pipe_events:
        arr = (ctypes.c_void_p * len(pipe_events))(*[int(e.cuda_event) for e in pipe_events])
        ex._pipe_keepalive = arr
        ex.pipe_events = ctypes.cast(arr, ctypes.POINTER(ctypes.c_void_p))
        ex.n_pipe_events = len(pipe_events)
    if stage_events is not None:
        arr = (ctypes.c_void_p * MOE_N_STAGE_EVENTS)(*[int(e.cuda_event) for e in stage_events])
        ex._events_keepalive = arr
        ex.stage_events = ctypes.cast(arr, ctypes.POINTER(ctypes.c_void_p))
    return ex


# ---------------------------------------------------------------- entry points

def moe_validate_config(cfg) -> int:
    return load().moe_validate_config(ctypes.byref(cfg))


def moe_workspace_size(cfg, ex) -> int:
    return load().moe_workspace_size(ctypes.byref(cfg), ctypes.byref(ex))


def moe_router_workspace_size(cfg) -> int:
    return load().moe_router_workspace_size(ctypes.byref(cfg))


def moe_dispatch_workspace_size(cfg) -> int:
    return load().moe_dispatch_workspace_size(ctypes.byref(cfg))


def moe_expert_ffn_workspace_size(rows, I) -> int:
    return load().moe_expert_ffn_workspace_size(rows, I)


def moe_router_logits(cfg, x, Wr, logits, ws=None, stream=None) -> None:
    nb = 0 if ws is None else ws.numel() * ws.element_size()
    _check(load().moe_router_logits(ctypes.byref(cfg), _ptr(x), _ptr(Wr), _ptr(logits), _ptr(ws),
                                    nb, _stream(stream)), "moe_router_logits")


def moe_gate_topk(cfg, logits, bias, topk_idx, topk_w, stream=None) -> None:
    _check(load().moe_gate_topk(ctypes.byref(cfg), _ptr(logits), _ptr(bias), _ptr(topk_idx),
                                _ptr(topk_w), _stream(stream)), "moe_gate_topk")


def moe_dispatch(cfg, x, topk_idx, counts, offsets, row_src_token, slot_row, x_perm, ws,
                 stream=None) -> None:
    nb = 0 if ws is None else ws.numel() * ws.element_size()
    _check(load().moe_dispatch(ctypes.byref(cfg), _ptr(x), _ptr(topk_idx), _ptr(counts),
                               _ptr(offsets), _ptr(row_src_token), _ptr(slot_row), _ptr(x_perm),
                               _ptr(ws), nb, _stream(stream)), "moe_dispatch")


def moe_dispatch_noalloc(cfg, x, topk_idx, counts, offsets, row_src_token, slot_row, x_perm,
                         stream=None) -> None:
    """moe_dispatch without a workspace, for callers that cannot allocate device memory."""
    _check(load().moe_dispatch_noalloc(ctypes.byref(cfg), _ptr(x), _ptr(topk_idx), _ptr(counts),
                                       _ptr(offsets), _ptr(row_src_token), _ptr(slot_row),
                                       _ptr(x_perm), _stream(stream)), "moe_dispatch_noalloc")


def moe_expert_ffn(rows, H, I, n_experts, x_perm, offsets, W13, W2, y_perm, ws,
                   stream=None, weights_packed=0) -> None:
    nb = 0 if ws is None else ws.numel() * ws.element_size()
    _check(load().moe_expert_ffn(rows, H, I, n_experts, _ptr(x_perm), _ptr(offsets), _ptr(W13),
                                 _ptr(W2), _ptr(y_perm), _ptr(ws), nb, int(weights_packed),
                                 _stream(stream)),
           "moe_expert_ffn")


def moe_expert_ffn_fp8_workspace_size(rows, I) -> int:
    return load().moe_expert_ffn_fp8_workspace_size(rows, I)


def moe_quantize_fp8(x, out, scale, stream=None) -> None:
    """Per-row e4m3 quantization of a bf16 tensor viewed as [rows, K] (K = its last dim)."""
    K = x.shape[-1]
    rows = x.numel() // K
    _check(load().moe_quantize_fp8(rows, K, _ptr(x), _ptr(out), _ptr(scale), _stream(stream)),
           "moe_quantize_fp8")


def quantize_fp8(x, stream=None):
    """(e4m3 bytes as uint8 of x's shape, fp32 scale per row) of a bf16 tensor."""
    import torch
    K = x.shape[-1]
    q = torch.empty(x.shape, dtype=torch.uint8, device=x.device)
    s = torch.empty(x.numel() // K, dtype=torch.float32, device=x.device)
    moe_quantize_fp8(x, q, s, stream)
    return q, s


def moe_expert_ffn_fp8(rows, H, I, n_experts, x_q, x_scale, x_scale_idx, offsets, W13_q,
                       W13_scale, W2_q, W2_scale, y_perm, ws, stream=None) -> None:
    nb = 0 if ws is None else ws.numel() * ws.element_size()
    _check(load().moe_expert_ffn_fp8(rows, H, I, n_experts, _ptr(x_q), _ptr(x_scale),
                                     _ptr(x_scale_idx), _ptr(offsets), _ptr(W13_q),
                                     _ptr(W13_scale), _ptr(W2_q), _ptr(W2_scale), _ptr(y_perm),
                                     _ptr(ws), nb, _stream(stream)),
           "moe_expert_ffn_fp8")


def moe_quantize_fp8_blocks(x, out, sf, sf_ld, stream=None) -> None:
    """e4m3 quantization of a bf16 tensor viewed as [rows, K] in 1 x 128 blocks;
    UE8M0 exponents to sf[r * sf_ld + c / 128]."""
    K = x.shape[-1]
    rows = x.numel() // K
    _check(load().moe_quantize_fp8_blocks(rows, K, _ptr(x), _ptr(out), _ptr(sf), int(sf_ld),
                                          _stream(stream)), "moe_quantize_fp8_blocks")


def quantize_fp8_blocks(x, stream=None):
    """(e4m3 bytes as uint8 of x's shape, uint8 exponents [rows, K / 128]) of a bf16 tensor."""
    import torch
    K = x.shape[-1]
    rows = x.numel() // K
    q = torch.empty(x.shape, dtype=torch.uint8, device=x.device)
    sf = torch.empty((rows, K // 128), dtype=torch.uint8, device=x.device)
    moe_quantize_fp8_blocks(x, q, sf, K // 128, stream)
    return q, sf


def moe_quantize_fp8_weight_blocks(W, out, sf, stream=None) -> None:
    """e4m3 quantization of a bf16 tensor viewed as [rows, K] in 128 x 128 blocks."""
    K = W.shape[-1]
    rows = W.numel() // K
    _check(load().moe_quantize_fp8_weight_blocks(rows, K, _ptr(W), _ptr(out), _ptr(sf),
                                                 _stream(stream)),
           "moe_quantize_fp8_weight_blocks")


def quantize_fp8_weight_blocks(W, stream=None):
    """(e4m3 bytes as uint8 of W's shape, uint8 exponents [rows / 128, K / 128])."""
    import torch
    K = W.shape[-1]
    rows = W.numel() // K
    q = torch.empty(W.shape, dtype=torch.uint8, device=W.device)
    sf = torch.empty((rows // 128, K // 128), dtype=torch.uint8, device=W.device)
    moe_quantize_fp8_weight_blocks(W, q, sf, stream)
    return q, sf


def moe_expert_ffn_fp8_blocks_workspace_size(rows, I) -> int:
    return load().moe_expert_ffn_fp8_blocks_workspace_size(rows, I)


def moe_expert_ffn_fp8_blocks(rows, H, I, n_experts, x_q, x_sf, x_sf_ld, x_scale_idx, offsets,
                              W13_q, W13_sf, W2_q, W2_sf, y_perm, ws, stream=None) -> None:
    nb = 0 if ws is None else ws.numel() * ws.element_size()
    _check(load().moe_expert_ffn_fp8_blocks(rows, H, I, n_experts, _ptr(x_q), _ptr(x_sf),
                                            int(x_sf_ld), _ptr(x_scale_idx), _ptr(offsets),
                                            _ptr(W13_q), _ptr(W13_sf), _ptr(W2_q), _ptr(W2_sf),
                                            _ptr(y_perm), _ptr(ws), nb, _stream(stream)),
           "moe_expert_ffn_fp8_blocks")


def moe_pack_weights(W, W_packed, stream=None) -> None:
    """Tile-packed copy of a bf16 weight tensor viewed as [rows, K] (K = its last dim)."""
    K = W.shape[-1]
    rows = W.numel() // K
    _check(load().moe_pack_weights(rows, K, _ptr(W), _ptr(W_packed), _stream(stream)),
           "moe_pack_weights")


def pack_weights(W, stream=None):
    """A new tensor holding W (bf16, rows a multiple of 128) in the tile-packed layout."""
    import torch
    out = torch.empty_like(W)
    moe_pack_weights(W, out, stream)
    return out


def moe_testing_expert_ffn_stall(rows, H, I, n_experts, x_perm, offsets, W13, W2, y_perm, ws,
                                 stall_fill, wait_limit_ns, stream=None) -> int:
    """Failure-detection hook: returns the launch status (the timeout shows in moe_check_errors)."""
    nb = 0 if ws is None else ws.numel() * ws.element_size()
    return load().moe_testing_expert_ffn_stall(rows, H, I, n_experts, _ptr(x_perm), _ptr(offsets),
                                               _ptr(W13), _ptr(W2), _ptr(y_perm), _ptr(ws), nb,
                                               int(stall_fill), int(wait_limit_ns),
                                               _stream(stream))


def moe_testing_fail_stage(n: int) -> None:
    """Failure-injection hook: stage call n (0-based) of the forwards that follow fails
    with MOE_ERR_CUDA on the host; -1 turns it off."""
    _check(load().moe_testing_fail_stage(int(n)), "moe_testing_fail_stage")


def moe_testing_tiled_chunk(r, e, off_e, cnt_e, tile, chunks_per_row, c) -> int:
    """16-byte chunk index of chunk c of packed row r (expert e, rows [off_e, off_e + cnt_e))
    in the layer's tile-packed token layout (host computation)."""
    out = ctypes.c_int64()
    _check(load().moe_testing_tiled_chunk(int(r), int(e), int(off_e), int(cnt_e), int(tile),
                                          int(chunks_per_row), int(c), ctypes.byref(out)),
           "moe_testing_tiled_chunk")
    return out.value


def moe_combine(cfg, y_perm, slot_row, topk_w, shared_out, out, out_fp32, stream=None) -> None:
    _check(load().moe_combine(ctypes.byref(cfg), _ptr(y_perm), _ptr(slot_row), _ptr(topk_w),
                              _ptr(shared_out), _ptr(out), int(out_fp32), _stream(stream)),
           "moe_combine")


def weights_struct(Wr, bias, W13, W2, Ws13=None, Ws2=None, packed=0, W13_scale=None,
                   W2_scale=None, Ws13_scale=None, Ws2_scale=None) -> moe_weights:
    p = [None if t is None else t.data_ptr() for t in (Wr, bias, W13, W2, Ws13, Ws2)]
    sc = [None if t is None else t.data_ptr() for t in (W13_scale, W2_scale, Ws13_scale,
                                                         Ws2_scale)]
    return moe_weights(*p, int(packed), *sc)


def aux_struct(logits=None, topk_idx=None, topk_w=None, counts=None) -> moe_aux:
    return moe_aux(*(None if t is None else t.data_ptr()
                     for t in (logits, topk_idx, topk_w, counts)))


def moe_layer_forward(cfg, ex, weights: moe_weights, x, out, aux: moe_aux | None, ws,
                      stream=None, aux_stream=None) -> None:
    nb = 0 if ws is None else ws.numel() * ws.element_size()
    auxp = None if aux is None else ctypes.byref(aux)
    a_s = None if aux_stream is None else _stream(aux_stream)
    _check(load().moe_layer_forward(ctypes.byref(cfg), ctypes.byref(ex), ctypes.byref(weights),
                                    _ptr(x), _ptr(out), auxp, _ptr(ws), nb, _stream(stream), a_s),
           "moe_layer_forward")


def moe_stack_workspace_size(cfg, ex) -> int:
    return load().moe_stack_workspace_size(ctypes.byref(cfg), ctypes.byref(ex))


def moe_rms_norm(x, out, stream=None) -> None:
    """Row-wise unit-gain RMS normalization of a bf16 tensor viewed as [rows, H]."""
    H = x.shape[-1]
    _check(load().moe_rms_norm(x.numel() // H, H, _ptr(x), _ptr(out), _stream(stream)),
           "moe_rms_norm")


def _layers(layers):
    arr = (moe_weights * len(layers))(*layers)
    return arr, len(layers)


def moe_stack_forward(cfg, ex, layers, x, out, ws, stream=None, aux_stream=None,
                      rms_norm=1) -> None:
    """Consecutive layers (a list of moe_weights); bf16 x -> bf16 out."""
    arr, n = _layers(layers)
    nb = 0 if ws is None else ws.numel() * ws.element_size()
    a_s = None if aux_stream is None else _stream(aux_stream)
    _check(load().moe_stack_forward(ctypes.byref(cfg), ctypes.byref(ex), arr, n, int(rms_norm),
                                    _ptr(x), _ptr(out), _ptr(ws), nb, _stream(stream), a_s),
           "moe_stack_forward")


def moe_graph_create_stack(cfg, ex, layers, x, out, ws, rms_norm=1,
                           stream=None) -> ctypes.c_void_p:
    """Handle of an executable CUDA graph of the stack (free with moe_graph_destroy)."""
    arr, n = _layers(layers)
    nb = 0 if ws is None else ws.numel() * ws.element_size()
    h = ctypes.c_void_p()
    _check(load().moe_graph_create_stack(ctypes.byref(cfg), ctypes.byref(ex), arr, n,
                                         int(rms_norm), _ptr(x), _ptr(out), _ptr(ws), nb,
                                         _stream(stream), ctypes.byref(h)),
           "moe_graph_create_stack")
    return h


def moe_graph_launch(graph, stream=None) -> None:
    _check(load().moe_graph_launch(graph, _stream(stream)), "moe_graph_launch")


def moe_graph_kernel_count(graph) -> int:
    return int(load().moe_graph_kernel_count(graph))


def moe_graph_destroy(graph) -> None:
    load().moe_graph_destroy(graph)


class Graph:
    """Owner of a moe_graph_create_stack handle; keeps its tensors alive."""

    def __init__(self, cfg, ex, layers, x, out, ws, rms_norm=1, stream=None):
        self._h = moe_graph_create_stack(cfg, ex, layers, x, out, ws, rms_norm, stream)
        self._keep = (x, out, ws, layers)   # the graph holds these pointers

    @property
    def kernels(self) -> int:
        return moe_graph_kernel_count(self._h)

    def launch(self, stream=None) -> None:
        moe_graph_launch(self._h, stream)

    def close(self) -> None:
        if self._h:
            moe_graph_destroy(self._h)
            self._h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


def moe_check_errors(stream=None) -> None:
    _check(load().moe_check_errors(_stream(stream)), "moe_check_errors")


def moe_launch_count() -> int:
    return int(load().moe_launch_count())


def moe_shutdown() -> None:
    load().moe_shutdown()
