"""FP8 (e4m3) form of the expert compute against the CPU oracle.

* moe_quantize_fp8: scales and e4m3 bytes bit-exact (both sides divide in
  fp32 and round to nearest even), on token-like and weight-like rows,
  including all-zero rows and rows reaching the subnormal range.
* moe_expert_ffn_fp8, stage by stage on ragged expert segments: GEMM1 + SwiGLU
  h within one bf16 ulp plus the fp32 summation bound of the oracle's fp64 h;
  the quantized h bit-exact given the kernel's own h; GEMM2 within the fp32
  summation bound given that quantized h; end to end against the oracle's own
  chain, where the only extra term is what h's rounding flips change.
* moe_layer_forward with fp8 = 1 on the DeepSeek-V3 decode shape (every token)
  and prefill shape (a sample of 256 tokens): routing bit-exact, output within
  |err| <= 2e-2 + 1e-2 |ref| of the oracle run with the same FP8 expert form.
The expert weights are drawn as stored e4m3 bytes with fp32 row scales; the
oracle reads the bytes through its own decoding of the format.
"""

import numpy as np
import pytest
import torch

from oracle import moe_oracle as O
from paper_2603_02376_gb300 import _lib as L
from paper_2603_02376_gb300 import inputs as I
from tests._support import U32, assert_layer_close, bias32, f64, oracle_cfg, prepare_routing

pytestmark = pytest.mark.gpu
DEV = "cuda"


@pytest.fixture(scope="module", autouse=True)
def lib():
    return L.load()


def e4m3(q) -> np.ndarray:
    """Values of e4m3 bytes held in a uint8 tensor (the oracle's decoding)."""
    return O.e4m3_decode(q.cpu().numpy())


def rand_bf16(shape, seed, std=1.0):
    g = torch.Generator(device=DEV).manual_seed(seed)
    return (torch.randn(shape, generator=g, device=DEV) * std).to(torch.bfloat16)


# ---------------------------------------------------------------- quantization

@pytest.mark.parametrize("rows,K,std", [(1, 16, 1.0), (37, 7168, 1.0), (130, 2048, 0.3),
                                        (256, 7168, 0.02), (5, 4096, 1e-3)])
def test_quantize_fp8_bit_exact(rows, K, std):
    x = rand_bf16((rows, K), rows * 7 + K, std)
    if rows > 2:
        x[1] = 0                                   # all-zero row: scale 1, all codes 0
        x[2, :] = x[2, :] * 1e-3                   # most of the row lands among subnormals
        x[2, 0] = 300.0                            # ... under one large element
    q, s = L.quantize_fp8(x)
    torch.cuda.synchronize()
    q_ref, s_ref = O.quantize_rows_e4m3(f64(x))
    np.testing.assert_array_equal(s.cpu().numpy(), s_ref)
    np.testing.assert_array_equal(e4m3(q), q_ref)
    assert not np.isnan(e4m3(q)).any()


# ---------------------------------------------------------------- grouped FP8 expert FFN

def fp8_ffn_case(counts, H, Iw, seed, rows_extra=3):
    E = len(counts)
    rows = int(sum(counts)) + rows_extra
    offs = np.zeros(E + 1, dtype=np.int32)
    offs[1:] = np.cumsum(counts)
    xp = rand_bf16((rows, H), seed)
    W13, s13 = I.e4m3_codes((E, 2 * Iw, H), seed, "W13q", DEV)
    W2, s2 = I.e4m3_codes((E, H, Iw), seed, "W2q", DEV)
    return rows, offs, xp, W13, s13.view(E, 2 * Iw), W2, s2.view(E, H)


def align256(n):
    return (n + 255) // 256 * 256


@pytest.mark.parametrize("token_scales", [False, True])
@pytest.mark.parametrize("counts,H,Iw", [
    ([5, 0, 17, 1], 256, 128),                          # tiny, ragged, an empty expert
    ([300, 256, 257, 0, 1, 16], 256, 256),              # multi-tile experts, tile edges
    ([4] * 60 + [0, 12, 31, 33], 512, 256),             # decode-like: small token tiles
    ([150, 100, 0, 145, 3], 512, 256),                  # 144-row tiles, experts over two tiles
    ([128, 129, 127, 384, 0, 200], 256, 256),           # 127/128/129-row experts, 128-row tails
    ([128, 129, 16, 144, 273, 0, 60], 384, 128),        # ... 144-row tiles, one GEMM2 tile
    ([130, 111], 7168, 2048),                           # the real layer shape
    ([1, 3, 0, 7], 7168, 2048),                         # decode: few rows per expert
])
def test_expert_ffn_fp8(counts, H, Iw, token_scales):
    rows, offs, xp, W13, s13, W2, s2 = fp8_ffn_case(counts, H, Iw, seed=len(counts) + H)
    E = len(counts)
    if token_scales:
        # packed rows are copies of token rows (a dispatch); scales are kept per token
        n_tok = max(1, rows // 2)
        tok = rand_bf16((n_tok, H), 99 + H)
        src = torch.from_numpy(np.random.default_rng(rows).integers(0, n_tok, rows)
                               .astype(np.int32)).to(DEV)
        xq_tok, sx = L.quantize_fp8(tok)
        xq = xq_tok[src.long()].contiguous()
        xp = tok[src.long()]
        sidx = src
    else:
        xq, sx = L.quantize_fp8(xp)
        sidx = None
    y = torch.full((rows, H), -12345.0, dtype=torch.float32, device=DEV)
    ws = torch.zeros(L.moe_expert_ffn_fp8_workspace_size(rows, Iw), dtype=torch.uint8,
                     device=DEV)
    L.moe_expert_ffn_fp8(rows, H, Iw, E, xq, sx, sidx, torch.from_numpy(offs).to(DEV), W13, s13,
                         W2, s2, y, ws)
    L.moe_check_errors()
    o_hq = align256(rows * Iw * 2)
    o_hs = align256(o_hq + rows * Iw)
    h = ws[:rows * Iw * 2].view(torch.bfloat16).view(rows, Iw)
    hq = ws[o_hq:o_hq + rows * Iw].view(rows, Iw)
    hs = ws[o_hs:o_hs + rows * 4].view(torch.float32)
    n = int(offs[-1])
    xh = f64(xp)
    for e in range(E):
        a, b = int(offs[e]), int(offs[e + 1])
        if b == a:
            continue
        W13e, W2e = e4m3(W13[e]), e4m3(W2[e])
        s13e, s2e = s13[e].cpu().numpy(), s2[e].cpu().numpy()
        # GEMM1 + SwiGLU against the oracle's fp64 chain (it quantizes x itself)
        h_o = O.swiglu_h_fp8(xh[a:b], W13e, s13e)
        xq_o, sx_o = O.quantize_rows_e4m3(xh[a:b])
        gu = O.fp8_linear(xq_o, sx_o, W13e, s13e)
        g, u = gu[:, :Iw], gu[:, Iw:]
        # fp32 sums of exact e4m3 products (K terms), then two fp32 scale products
        mag = O.fp8_linear(np.abs(xq_o), sx_o, np.abs(W13e), s13e)
        dgu = H * U32 * mag + 3 * U32 * np.abs(gu)
        dg, du = dgu[:, :Iw], dgu[:, Iw:]
        sg = 1.0 / (1.0 + np.exp(-g))
        dsilu = np.abs(sg * (1.0 + g * (1.0 - sg))) + dg
        lim = (np.abs(h_o) * 2.0 ** -7 + (dsilu * np.abs(u) * dg + np.abs(O.silu(g)) * du
                                          + dsilu * dg * du) * (1 + 2.0 ** -7)) * 1.0001
        hg = f64(h[a:b])
        diff = np.abs(hg - h_o)
        assert (diff <= lim + 1e-30).all(), f"expert {e}: h outside one ulp + fp32 bound"
        assert (diff == 0).mean() > 0.98, f"expert {e}: too many h rounding flips"
        # quantization of the kernel's own h: bit-exact
        hq_o, hs_o = O.quantize_rows_e4m3(hg)
        np.testing.assert_array_equal(hs[a:b].cpu().numpy(), hs_o)
        np.testing.assert_array_equal(e4m3(hq[a:b]), hq_o)
        # GEMM2 given that quantized h: within the fp32 summation bound
        y_ref = O.fp8_linear(hq_o, hs_o, W2e, s2e)
        bound = Iw * U32 * O.fp8_linear(np.abs(hq_o), hs_o, np.abs(W2e), s2e) \
            + 3 * U32 * np.abs(y_ref)
        yg = f64(y[a:b])
        err = np.abs(yg - y_ref)
        assert (err <= bound + 1e-30).all(), f"expert {e}: GEMM2 max err {err.max():.3e}"
        # end to end against the oracle's own chain: h's rounding flips change the
        # dequantized h (and possibly its row scale); their effect is the only extra term
        y_or = O.swiglu_ffn_fp8(xh[a:b], W13e, s13e, W2e, s2e)
        hq_oo, hs_oo = O.quantize_rows_e4m3(h_o)
        dq = np.abs(hq_o * hs_o[:, None].astype(np.float64) - hq_oo * hs_oo[:, None])
        flip = dq @ (np.abs(W2e) * s2e[:, None].astype(np.float64)).T
        assert (np.abs(yg - y_or) <= bound + flip * 1.0001 + 1e-30).all()
    # rows outside every segment are untouched
    assert (y[n:] == -12345.0).all()


# ---------------------------------------------------------------- the FP8 layer

@pytest.fixture(scope="module")
def fp8_layer():
    """DeepSeek-V3-shaped layer with FP8 experts (11.3 GB of e4m3 bytes), drawn once."""
    wl = I.DECODE
    d = I.layer_inputs(wl, seed=0, device=DEV, with_experts=False)
    d.pop("x")
    d["W13"], d["s13"], d["W2"], d["s2"] = I.fp8_expert_weights(wl, 0, DEV)
    d["Ws13"], d["ss13"], d["Ws2"], d["ss2"] = I.fp8_shared_weights(wl, 0, DEV)
    yield d
    del d
    torch.cuda.empty_cache()


def run_fp8_layer(wl, d, ex):
    cfg = L.config_of(wl)
    T, E, k = wl.T, wl.E, wl.k
    ws = torch.empty(L.moe_workspace_size(cfg, ex), dtype=torch.uint8, device=DEV)
    out = torch.empty((T, wl.H), dtype=torch.float32 if ex.out_fp32 else torch.bfloat16,
                      device=DEV)
    a = dict(logits=torch.empty((T, E), device=DEV),
             topk_idx=torch.empty((T, k), dtype=torch.int32, device=DEV),
             topk_w=torch.empty((T, k), device=DEV),
             counts=torch.empty(E, dtype=torch.int32, device=DEV))
    W = L.weights_struct(d["Wr"], d["bias"], d["W13"], d["W2"], d["Ws13"], d["Ws2"], 0,
                         d["s13"], d["s2"], d["ss13"], d["ss2"])
    L.moe_layer_forward(cfg, ex, W, d["x"], out, L.aux_struct(**a), ws)
    L.moe_check_errors()
    return out, a


def oracle_fp8_tokens(wl, d, toks):
    def expert(e):
        return e4m3(d["W13"][e]), d["s13"][e].cpu().numpy(), e4m3(d["W2"][e]), \
            d["s2"][e].cpu().numpy()

    def shared():
        return e4m3(d["Ws13"]), d["ss13"].cpu().numpy(), e4m3(d["Ws2"]), d["ss2"].cpu().numpy()

    out, idx, _ = O.layer_forward_tokens(f64(d["x"][torch.as_tensor(toks, device=DEV)]),
                                         f64(d["Wr"]), bias32(d["bias"]), expert, oracle_cfg(wl),
                                         shared if wl.I_shared else None, ffn=O.swiglu_ffn_fp8)
    return out, idx


def check_routing_fp8(wl, d, a, toks):
    ridx, _ = O.gate_topk(a["logits"].cpu().numpy(), bias32(d["bias"]), oracle_cfg(wl))
    np.testing.assert_array_equal(a["topk_idx"].cpu().numpy(), ridx)
    np.testing.assert_array_equal(a["counts"].cpu().numpy(),
                                  np.bincount(ridx.reshape(-1), minlength=wl.E))


@pytest.mark.parametrize("T", [150, 8])
def test_layer_fp8_one_tile_gemm2_full(T):
    """Row-scaled FP8 with H = 384: GEMM2 (one 128-feature tile per unit) reads
    the e4m3 copy of h in the tile-packed layout; 144- and 32-row token tiles;
    the packed dispatch, the copy inside GEMM1 and the expert-range pipeline;
    every token against the oracle's FP8 chain."""
    wl = I.Workload("one-tile gemm2 fp8", T=T, H=384, E=12, k=3, I=256, I_shared=256,
                    n_groups=4, topk_groups=2, gate=I.GATE_SIGMOID, normalize=1,
                    route_scale=2.5)
    d = I.layer_inputs(wl, seed=7, device=DEV, with_experts=False)
    d["W13"], d["s13"], d["W2"], d["s2"] = I.fp8_expert_weights(wl, 7, DEV)
    d["Ws13"], d["ss13"], d["Ws2"], d["ss2"] = I.fp8_shared_weights(wl, 7, DEV)
    prepare_routing(wl, d)
    toks = np.arange(wl.T)
    ref, idx = oracle_fp8_tokens(wl, d, toks)
    for ex in (L.exec_config(out_fp32=1, fp8=1, fuse_gather=0),
               L.exec_config(out_fp32=1, fp8=1, fuse_gather=2),
               L.exec_config(out_fp32=1, fp8=1, overlap=1, chunk_axis=1, n_expert_chunks=5)):
        out, a = run_fp8_layer(wl, d, ex)
        check_routing_fp8(wl, d, a, toks)
        assert_layer_close(out, ref)


@pytest.mark.parametrize("H,E,k,T", [(128, 8, 2, 70), (256, 40, 32, 33)])
def test_layer_fp8_copy_in_gemm1_token_major_full(H, E, k, T):
    """Row-scaled FP8 with the e4m3 dispatch copy inside GEMM1 (token-major, the
    shared expert in the launch): rows of 8 and 16 16-byte vectors (H = 128 and
    256 e4m3 bytes), k = 2 and 32; every token against the oracle's FP8 chain."""
    wl = I.Workload("fp8 token-major copy", T=T, H=H, E=E, k=k, I=128, I_shared=128,
                    gate=I.GATE_SIGMOID, normalize=1, route_scale=2.5)
    d = I.layer_inputs(wl, seed=13, device=DEV, with_experts=False)
    d["W13"], d["s13"], d["W2"], d["s2"] = I.fp8_expert_weights(wl, 13, DEV)
    d["Ws13"], d["ss13"], d["Ws2"], d["ss2"] = I.fp8_shared_weights(wl, 13, DEV)
    prepare_routing(wl, d)
    toks = np.arange(wl.T)
    ref, idx = oracle_fp8_tokens(wl, d, toks)
    outs = []
    for ex in (L.exec_config(out_fp32=1, fp8=1, fuse_gather=0),
               L.exec_config(out_fp32=1, fp8=1, fuse_gather=2)):
        out, a = run_fp8_layer(wl, d, ex)
        check_routing_fp8(wl, d, a, toks)
        assert_layer_close(out, ref)
        outs.append(out)
    # the same e4m3 bytes in the same rows as the dispatch kernel's
    assert float((outs[1] - outs[0]).abs().max()) <= 1e-5 * float(np.abs(ref).max())


@pytest.fixture(scope="module")
def fp8_decode(fp8_layer):
    """Decode batch (T=128) on the FP8 layer, routing made well-posed, oracle on every token."""
    wl = I.DECODE
    d = dict(fp8_layer)
    d["x"] = I.randn((wl.T, wl.H), 1.0, torch.bfloat16, 0, "x", DEV)
    prepare_routing(wl, d)
    toks = np.arange(wl.T)
    ref, idx = oracle_fp8_tokens(wl, d, toks)
    return d, toks, ref, idx


@pytest.fixture(scope="module")
def fp8_prefill(fp8_layer):
    """Prefill batch (T=4096, balanced) on the FP8 layer, oracle on 256 sampled tokens."""
    wl = I.PREFILL
    d = dict(fp8_layer)
    d["x"] = I.randn((wl.T, wl.H), 1.0, torch.bfloat16, 0, "x", DEV)
    prepare_routing(wl, d)
    toks = I.sample_tokens(wl.T, 256, 0).numpy()
    ref, idx = oracle_fp8_tokens(wl, d, toks)
    return d, toks, ref, idx


@pytest.mark.parametrize("ex", [dict(out_fp32=1), dict(out_fp32=0), dict(out_fp32=1, fuse_gather=0),
                                dict(out_fp32=1, overlap=1, chunk_axis=1, n_expert_chunks=4),
                                dict(out_fp32=0, fuse_combine=1), dict(out_fp32=1, fuse_gather=2)])
def test_layer_fp8_decode_full(fp8_decode, ex):
    wl = I.DECODE
    d, toks, ref, idx = fp8_decode
    out, a = run_fp8_layer(wl, d, L.exec_config(fp8=1, **ex))
    check_routing_fp8(wl, d, a, toks)
    np.testing.assert_array_equal(np.sort(a["topk_idx"].cpu().numpy(), 1), np.sort(idx, 1))
    assert_layer_close(out, ref)


@pytest.mark.parametrize("ex", [dict(out_fp32=1), dict(out_fp32=1, fuse_gather=0),
                                dict(out_fp32=1, overlap=1, chunk_axis=0, chunk_tokens=512),
                                dict(out_fp32=1, overlap=1, chunk_axis=1, n_expert_chunks=8),
                                dict(out_fp32=1, fuse_combine=1), dict(out_fp32=1, fuse_gather=2)])
def test_layer_fp8_prefill_sampled(fp8_prefill, ex):
    wl = I.PREFILL
    d, toks, ref, idx = fp8_prefill
    out, a = run_fp8_layer(wl, d, L.exec_config(fp8=1, **ex))
    check_routing_fp8(wl, d, a, toks)
    np.testing.assert_array_equal(np.sort(a["topk_idx"].cpu().numpy()[toks], 1), np.sort(idx, 1))
    assert_layer_close(out[torch.as_tensor(toks, device=DEV)], ref)
