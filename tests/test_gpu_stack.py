"""Layer stacks (the paper's multi-layer study) and their CUDA-graph replay.

* moe_rms_norm (the normalization between stacked layers) equals the
  oracle's bf16-rounded RMS normalization except rare one-ulp flips.
* moe_stack_forward over L layers equals L chained moe_layer_forward calls
  (with moe_rms_norm between them when asked) bit for bit, and every layer of
  the chain matches the oracle run on that layer's input and on the GPU's
  fp32 logits, within the layer bound |err| <= 2e-2 + 1e-2 |ref|.
* A graph made by moe_graph_create_stack replays the stack bit for bit, in
  the sequential and both pipelined modes and in both FP8 forms, also after new
  inputs are written into its x buffer; its kernel count is the eager one.
"""

import numpy as np
import pytest
import torch

from oracle import moe_oracle as O
from paper_2603_02376_gb300 import _lib as L
from paper_2603_02376_gb300 import inputs as I
from tests._support import assert_layer_close, bias32, f64, oracle_cfg

pytestmark = pytest.mark.gpu
DEV = "cuda"

SMALL = I.Workload("small stack layer", T=100, H=256, E=16, k=4, I=128, I_shared=128, n_groups=4,
                   topk_groups=2, gate=I.GATE_SIGMOID, normalize=1, route_scale=2.5)


@pytest.fixture(scope="module", autouse=True)
def lib():
    return L.load()


def small_layers(n, wl=SMALL):
    """n layers with their own weights (seeds 10, 11, ...)."""
    return [I.layer_inputs(wl, seed=10 + l, device=DEV) for l in range(n)]


def wstruct(d):
    return L.weights_struct(d["Wr"], d["bias"], d["W13"], d["W2"], d["Ws13"], d["Ws2"],
                            d.get("packed", 0), d.get("s13"), d.get("s2"), d.get("ss13"),
                            d.get("ss2"))


@pytest.mark.parametrize("rows,H,std", [(100, 256, 1.0), (128, 7168, 0.3), (7, 4096, 20.0)])
def test_rms_norm_matches_the_oracle(rows, H, std):
    x = I.randn((rows, H), std, torch.bfloat16, rows, "x", DEV)
    if rows > 2:
        x[1] = 0                       # an all-zero row stays zero
    y = torch.empty_like(x)
    L.moe_rms_norm(x, y)
    z = x.clone()
    L.moe_rms_norm(z, z)               # in place
    torch.cuda.synchronize()
    assert torch.equal(y, z)
    ref = O.bf16_round(O.rms_normalize(f64(x)))
    got = f64(y)
    # fp32 sum of squares and rsqrt (a few fp32 ulp) before one bf16 rounding: equal
    # to the oracle's bf16 except rare one-ulp rounding flips
    diff = np.abs(got - ref)
    assert (diff <= np.abs(ref) * 2.0 ** -7 + 1e-30).all()
    assert (diff == 0).mean() > 0.99


@pytest.mark.parametrize("rms_norm", [1, 0])
def test_stack_equals_chained_layers_and_the_oracle(rms_norm):
    wl, n = SMALL, 3
    ds = small_layers(n)
    x = I.randn((wl.T, wl.H), 1.0, torch.bfloat16, 5, "x", DEV)
    cfg, ex = L.config_of(wl), L.exec_config()
    ws = torch.empty(L.moe_stack_workspace_size(cfg, ex), dtype=torch.uint8, device=DEV)
    out = torch.empty((wl.T, wl.H), dtype=torch.bfloat16, device=DEV)
    L.moe_stack_forward(cfg, ex, [wstruct(d) for d in ds], x, out, ws, rms_norm=rms_norm)
    L.moe_check_errors()
    # the chain, layer by layer (and the normalization between layers), with the
    # GPU logits of every layer for the oracle
    lws = torch.empty(L.moe_workspace_size(cfg, ex), dtype=torch.uint8, device=DEV)
    h = x
    for l, d in enumerate(ds):
        if l > 0 and rms_norm:
            L.moe_rms_norm(h, h)
        y = torch.empty_like(h)
        logits = torch.empty((wl.T, wl.E), device=DEV)
        idx = torch.empty((wl.T, wl.k), dtype=torch.int32, device=DEV)
        L.moe_layer_forward(cfg, ex, wstruct(d), h, y, L.aux_struct(logits=logits, topk_idx=idx),
                            lws)
        L.moe_check_errors()
        ridx, _ = O.gate_topk(logits.cpu().numpy(), bias32(d["bias"]), oracle_cfg(wl))
        np.testing.assert_array_equal(idx.cpu().numpy(), ridx)
        ref, _ = O.layer_forward(f64(h), f64(d["Wr"]), bias32(d["bias"]), f64(d["W13"]),
                                 f64(d["W2"]), oracle_cfg(wl), f64(d["Ws13"]), f64(d["Ws2"]),
                                 logits=logits.cpu().numpy())
        assert_layer_close(f64(y), ref)
        h = y
    assert torch.equal(out, h)


@pytest.mark.parametrize("mode", [dict(), dict(overlap=1, chunk_axis=0, chunk_tokens=37),
                                  dict(overlap=1, chunk_axis=1, n_expert_chunks=3),
                                  dict(fuse_gather=0), dict(fp8=1), dict(fp8=2)])
def test_graph_replays_the_stack(mode):
    wl, n = SMALL, 3
    ds = small_layers(n)
    if mode.get("fp8"):
        # e4m3 expert weights with row scales (fp8 = 1) or 128 x 128 block exponents
        # (fp8 = 2), quantized on the device
        quant = L.quantize_fp8 if mode["fp8"] == 1 else L.quantize_fp8_weight_blocks
        for d in ds:
            for w_, s_ in (("W13", "s13"), ("W2", "s2"), ("Ws13", "ss13"), ("Ws2", "ss2")):
                d[w_], d[s_] = quant(d[w_])
    cfg, ex = L.config_of(wl), L.exec_config(**mode)
    layers = [wstruct(d) for d in ds]
    ws = torch.empty(L.moe_stack_workspace_size(cfg, ex), dtype=torch.uint8, device=DEV)
    x = I.randn((wl.T, wl.H), 1.0, torch.bfloat16, 6, "x", DEV)
    out = torch.empty((wl.T, wl.H), dtype=torch.bfloat16, device=DEV)
    ref = torch.empty_like(out)
    ws2 = torch.empty_like(ws)
    g = L.Graph(cfg, ex, layers, x, out, ws)
    for seed in (6, 7):
        x.copy_(I.randn((wl.T, wl.H), 1.0, torch.bfloat16, seed, "x", DEV))
        out.zero_()
        n0 = L.moe_launch_count()
        L.moe_stack_forward(cfg, ex, layers, x, ref, ws2)
        eager = L.moe_launch_count() - n0
        g.launch()
        L.moe_check_errors()
        assert torch.equal(out, ref)
        assert g.kernels == eager
    g.close()


def test_graph_of_the_decode_stack():
    """Two DeepSeek-V3 decode layers (own routers, shared expert weights) as one graph."""
    wl = I.DECODE
    d = I.layer_inputs(wl, seed=0, device=DEV)
    d2 = dict(d)
    d2["Wr"] = I.randn((wl.E, wl.H), 0.01, torch.float32, 1, "Wr", DEV)
    d2["bias"] = I.randn((wl.E,), 0.01, torch.float32, 1, "bias", DEV)
    cfg, ex = L.config_of(wl), L.exec_config()
    layers = [wstruct(d), wstruct(d2)]
    ws = torch.empty(L.moe_stack_workspace_size(cfg, ex), dtype=torch.uint8, device=DEV)
    x = d["x"].clone()
    out = torch.empty_like(x)
    ref = torch.empty_like(x)
    g = L.Graph(cfg, ex, layers, x, out, ws)
    out.zero_()
    g.launch()
    L.moe_check_errors()
    L.moe_stack_forward(cfg, ex, layers, x, ref, torch.empty_like(ws))
    L.moe_check_errors()
    assert torch.equal(out, ref)
    assert out.abs().max().item() > 0
    g.close()
    del d, d2
    torch.cuda.empty_cache()
