"""Block-scaled FP8 form of the expert compute against the CPU oracle.

* moe_quantize_fp8_blocks (1 x 128 activation blocks) and
  moe_quantize_fp8_weight_blocks (128 x 128 weight blocks): UE8M0 exponents
  and e4m3 bytes bit-exact (both sides scale by an exact power of two, then
  round to nearest even), including all-zero blocks, blocks reaching the
  subnormal range and one large element among small ones.
* moe_expert_ffn_fp8_blocks, stage by stage on ragged expert segments (token
  tiles of 32, 144 and 224 rows): GEMM1 + SwiGLU h within one bf16 ulp plus
  the fp32 summation bound of the oracle's fp64 h; the block quantization of
  the kernel's own h bit-exact; GEMM2 within the fp32 summation bound given
  that quantized h; end to end against the oracle's chain, where the only
  extra term is what h's rounding flips change.
* moe_layer_forward with fp8 = 2 on the DeepSeek-V3 decode shape (every
  token), the balanced prefill and the skewed (Zipf) batch (256 sampled tokens
  each): routing bit-exact, output within |err| <= 2e-2 + 1e-2 |ref| of the
  oracle run with the same block-scaled expert form.
Expert weights are drawn as stored e4m3 bytes with UE8M0 block exponents; the
oracle reads both through its own decoding.
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
    return O.e4m3_decode(q.cpu().numpy())


def exps(sf) -> np.ndarray:
    """Block exponents k of UE8M0 bytes (k = byte - 127)."""
    return sf.cpu().numpy().astype(np.int64) - 127


def rand_bf16(shape, seed, std=1.0):
    g = torch.Generator(device=DEV).manual_seed(seed)
    return (torch.randn(shape, generator=g, device=DEV) * std).to(torch.bfloat16)


def align256(n):
    return (n + 255) // 256 * 256


# ---------------------------------------------------------------- quantization

@pytest.mark.parametrize("rows,K,std,ld_extra", [(1, 128, 1.0, 0), (37, 7168, 1.0, 5),
                                                 (130, 2048, 0.3, 0), (256, 7168, 0.02, 0),
                                                 (5, 4096, 1e-3, 3), (3, 384, 50.0, 0)])
def test_quantize_fp8_blocks_bit_exact(rows, K, std, ld_extra):
    x = rand_bf16((rows, K), rows * 11 + K, std)
    if rows > 2:
        x[1, :128] = 0                             # an all-zero block: k = 0, codes 0
        x[2, :] = x[2, :] * 1e-3                   # blocks reaching e4m3 subnormals ...
        x[2, 5] = 300.0                            # ... under one large element
    ld = K // 128 + ld_extra
    q = torch.empty((rows, K), dtype=torch.uint8, device=DEV)
    sf = torch.full((rows, ld), 0xEE, dtype=torch.uint8, device=DEV)
    L.moe_quantize_fp8_blocks(x, q, sf, ld)
    torch.cuda.synchronize()
    q_ref, k_ref = O.quantize_blocks_e4m3(f64(x), 1)
    np.testing.assert_array_equal(exps(sf[:, :K // 128]), k_ref)
    np.testing.assert_array_equal(e4m3(q), q_ref)
    assert (sf[:, K // 128:] == 0xEE).all()        # the stride's slack is untouched
    q2, sf2 = L.quantize_fp8_blocks(x)             # the allocating form: [rows, K / 128]
    assert torch.equal(q2, q) and torch.equal(sf2, sf[:, :K // 128])


@pytest.mark.parametrize("rows,K,std", [(128, 128, 1.0), (256, 7168, 0.02), (4096, 2048, 0.02),
                                        (384, 256, 3.0)])
def test_quantize_fp8_weight_blocks_bit_exact(rows, K, std):
    W = rand_bf16((rows, K), rows + K, std)
    W[:128, 128:] = 0 if K > 128 else W[:128, 128:]   # zero blocks
    W[-1, 0] = 1000.0                                  # one large element in one block
    q, sf = L.quantize_fp8_weight_blocks(W)
    torch.cuda.synchronize()
    q_ref, k_ref = O.quantize_blocks_e4m3(f64(W), 128)
    np.testing.assert_array_equal(exps(sf), k_ref)
    np.testing.assert_array_equal(e4m3(q), q_ref)


# ---------------------------------------------------------------- grouped block-FP8 expert FFN

def block_ffn_case(counts, H, Iw, seed, rows_extra=3):
    E = len(counts)
    rows = int(sum(counts)) + rows_extra
    offs = np.zeros(E + 1, dtype=np.int32)
    offs[1:] = np.cumsum(counts)
    xp = rand_bf16((rows, H), seed)
    W13, k13 = I.e4m3_block_codes((E * 2 * Iw, H), seed, "W13b", DEV)
    W2, k2 = I.e4m3_block_codes((E * H, Iw), seed, "W2b", DEV)
    return rows, offs, xp, W13.view(E, 2 * Iw, H), k13, W2.view(E, H, Iw), k2


@pytest.mark.parametrize("token_scales", [False, True])
@pytest.mark.parametrize("counts,H,Iw", [
    ([5, 0, 17, 1], 256, 128),                          # tiny, ragged, an empty expert (32-row tiles)
    ([300, 256, 257, 0, 1, 16], 256, 256),              # 224-row tiles, experts over two tiles
    ([4] * 60 + [0, 12, 31, 33], 512, 256),             # decode-like: small token tiles
    ([150, 100, 0, 145, 3], 512, 256),                  # 144-row tiles
    ([130, 111], 7168, 2048),                           # the real layer shape
    ([1, 3, 0, 7], 7168, 2048),                         # decode: few rows per expert
])
def test_expert_ffn_fp8_blocks(counts, H, Iw, token_scales):
    rows, offs, xp, W13, k13, W2, k2 = block_ffn_case(counts, H, Iw, seed=len(counts) + H)
    E = len(counts)
    nb13, nb2 = 2 * Iw // 128, H // 128            # weight row blocks per expert
    if token_scales:
        # packed rows are copies of token rows (a dispatch); exponents stay per token
        n_tok = max(1, rows // 2)
        tok = rand_bf16((n_tok, H), 99 + H)
        src = torch.from_numpy(np.random.default_rng(rows).integers(0, n_tok, rows)
                               .astype(np.int32)).to(DEV)
        xq_tok, xsf = L.quantize_fp8_blocks(tok)
        xq = xq_tok[src.long()].contiguous()
        xp = tok[src.long()]
        sidx = src
    else:
        xq, xsf = L.quantize_fp8_blocks(xp)
        sidx = None
    ld = H // 128
    y = torch.full((rows, H), -12345.0, dtype=torch.float32, device=DEV)
    ws = torch.zeros(L.moe_expert_ffn_fp8_blocks_workspace_size(rows, Iw), dtype=torch.uint8,
                     device=DEV)
    L.moe_expert_ffn_fp8_blocks(rows, H, Iw, E, xq, xsf, ld, sidx,
                                torch.from_numpy(offs).to(DEV), W13, k13, W2, k2, y, ws)
    L.moe_check_errors()
    o_hq = align256(rows * Iw * 2)
    o_hs = align256(o_hq + rows * Iw)
    h = ws[:rows * Iw * 2].view(torch.bfloat16).view(rows, Iw)
    hq = ws[o_hq:o_hq + rows * Iw].view(rows, Iw)
    hsf = ws[o_hs:o_hs + (Iw // 128) * rows].view(rows, Iw // 128)
    n = int(offs[-1])
    xh = f64(xp)
    for e in range(E):
        a, b = int(offs[e]), int(offs[e + 1])
        if b == a:
            continue
        W13e, W2e = e4m3(W13[e]), e4m3(W2[e])
        k13e = exps(k13[e * nb13:(e + 1) * nb13])
        k2e = exps(k2[e * nb2:(e + 1) * nb2])
        # GEMM1 + SwiGLU against the oracle's fp64 chain (it quantizes x itself)
        h_o = O.swiglu_h_fp8_blocks(xh[a:b], W13e, k13e)
        xq_o, kx_o = O.quantize_blocks_e4m3(xh[a:b], 1)
        gu = O.fp8_block_linear(xq_o, kx_o, W13e, k13e)
        g, u = gu[:, :Iw], gu[:, Iw:]
        # fp32 sums of exactly scaled e4m3 products (K terms)
        mag = O.fp8_block_linear(np.abs(xq_o), kx_o, np.abs(W13e), k13e)
        dgu = H * U32 * mag + 2 * U32 * np.abs(gu)
        dg, du = dgu[:, :Iw], dgu[:, Iw:]
        sg = 1.0 / (1.0 + np.exp(-g))
        dsilu = np.abs(sg * (1.0 + g * (1.0 - sg))) + dg
        lim = (np.abs(h_o) * 2.0 ** -7 + (dsilu * np.abs(u) * dg + np.abs(O.silu(g)) * du
                                          + dsilu * dg * du) * (1 + 2.0 ** -7)) * 1.0001
        hg = f64(h[a:b])
        diff = np.abs(hg - h_o)
        assert (diff <= lim + 1e-30).all(), f"expert {e}: h outside one ulp + fp32 bound"
        assert (diff == 0).mean() > 0.98, f"expert {e}: too many h rounding flips"
        # block quantization of the kernel's own h: bit-exact
        hq_o, kh_o = O.quantize_blocks_e4m3(hg, 1)
        np.testing.assert_array_equal(exps(hsf[a:b]), kh_o)
        np.testing.assert_array_equal(e4m3(hq[a:b]), hq_o)
        # GEMM2 given that quantized h: within the fp32 summation bound
        y_ref = O.fp8_block_linear(hq_o, kh_o, W2e, k2e)
        bound = Iw * U32 * O.fp8_block_linear(np.abs(hq_o), kh_o, np.abs(W2e), k2e) \
            + 2 * U32 * np.abs(y_ref)
        yg = f64(y[a:b])
        err = np.abs(yg - y_ref)
        assert (err <= bound + 1e-30).all(), f"expert {e}: GEMM2 max err {err.max():.3e}"
        # end to end against the oracle's own chain: h's rounding flips change the
        # dequantized h (and possibly a block exponent); their effect is the only extra term
        y_or = O.swiglu_ffn_fp8_blocks(xh[a:b], W13e, k13e, W2e, k2e)
        hq_oo, kh_oo = O.quantize_blocks_e4m3(h_o, 1)
        dq = np.abs(hq_o * O.block_scales(kh_o, 1) - hq_oo * O.block_scales(kh_oo, 1))
        flip = dq @ np.abs(W2e * O.block_scales(k2e, 128)).T
        assert (np.abs(yg - y_or) <= bound + flip * 1.0001 + 1e-30).all()
    # rows outside every segment are untouched
    assert (y[n:] == -12345.0).all()


# ---------------------------------------------------------------- the block-FP8 layer

@pytest.fixture(scope="module")
def block_layer():
    """DeepSeek-V3-shaped layer with block-scaled FP8 experts (11.3 GB of e4m3 bytes)."""
    wl = I.DECODE
    d = I.layer_inputs(wl, seed=0, device=DEV, with_experts=False)
    d.pop("x")
    d["W13"], d["k13"], d["W2"], d["k2"] = I.fp8_block_expert_weights(wl, 0, DEV)
    d["Ws13"], d["ks13"], d["Ws2"], d["ks2"] = I.fp8_block_shared_weights(wl, 0, DEV)
    yield d
    del d
    torch.cuda.empty_cache()


def run_block_layer(wl, d, ex):
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
                         d["k13"], d["k2"], d["ks13"], d["ks2"])
    L.moe_layer_forward(cfg, ex, W, d["x"], out, L.aux_struct(**a), ws)
    L.moe_check_errors()
    return out, a


def oracle_block_tokens(wl, d, toks):
    def expert(e):
        return e4m3(d["W13"][e]), exps(d["k13"][e]), e4m3(d["W2"][e]), exps(d["k2"][e])

    def shared():
        return e4m3(d["Ws13"]), exps(d["ks13"]), e4m3(d["Ws2"]), exps(d["ks2"])

    out, idx, _ = O.layer_forward_tokens(f64(d["x"][torch.as_tensor(toks, device=DEV)]),
                                         f64(d["Wr"]), bias32(d["bias"]), expert, oracle_cfg(wl),
                                         shared if wl.I_shared else None,
                                         ffn=O.swiglu_ffn_fp8_blocks)
    return out, idx


def check_routing(wl, d, a, toks, idx):
    ridx, _ = O.gate_topk(a["logits"].cpu().numpy(), bias32(d["bias"]), oracle_cfg(wl))
    np.testing.assert_array_equal(a["topk_idx"].cpu().numpy(), ridx)
    np.testing.assert_array_equal(a["counts"].cpu().numpy(),
                                  np.bincount(ridx.reshape(-1), minlength=wl.E))
    np.testing.assert_array_equal(np.sort(ridx[toks], 1), np.sort(idx, 1))


def batch(block_layer, wl, n_sample):
    d = dict(block_layer)
    d["x"] = I.randn((wl.T, wl.H), 1.0, torch.bfloat16, 0, "x", DEV)
    prepare_routing(wl, d)
    toks = np.arange(wl.T) if n_sample is None else I.sample_tokens(wl.T, n_sample, 0).numpy()
    ref, idx = oracle_block_tokens(wl, d, toks)
    return d, toks, ref, idx


@pytest.fixture(scope="module")
def block_decode(block_layer):
    return batch(block_layer, I.DECODE, None)


@pytest.fixture(scope="module")
def block_prefill(block_layer):
    return batch(block_layer, I.PREFILL, 256)


@pytest.fixture(scope="module")
def block_skewed(block_layer):
    return batch(block_layer, I.SKEWED, 256)


@pytest.mark.parametrize("ex", [dict(out_fp32=1), dict(out_fp32=0), dict(out_fp32=1, fuse_gather=0),
                                dict(out_fp32=1, overlap=1, chunk_axis=1, n_expert_chunks=4),
                                dict(out_fp32=0, fuse_combine=1)])
def test_layer_fp8_blocks_decode_full(block_decode, ex):
    wl = I.DECODE
    d, toks, ref, idx = block_decode
    out, a = run_block_layer(wl, d, L.exec_config(fp8=2, **ex))
    check_routing(wl, d, a, toks, idx)
    assert_layer_close(out, ref)


@pytest.mark.parametrize("ex", [dict(out_fp32=1), dict(out_fp32=1, fuse_gather=0),
                                dict(out_fp32=1, overlap=1, chunk_axis=0, chunk_tokens=512),
                                dict(out_fp32=1, overlap=1, chunk_axis=1, n_expert_chunks=8),
                                dict(out_fp32=1, fuse_combine=1)])
def test_layer_fp8_blocks_prefill_sampled(block_prefill, ex):
    wl = I.PREFILL
    d, toks, ref, idx = block_prefill
    out, a = run_block_layer(wl, d, L.exec_config(fp8=2, **ex))
    check_routing(wl, d, a, toks, idx)
    assert_layer_close(out[torch.as_tensor(toks, device=DEV)], ref)


@pytest.mark.parametrize("ex", [dict(out_fp32=1), dict(out_fp32=0, fuse_combine=1)])
def test_layer_fp8_blocks_skewed_sampled(block_skewed, ex):
    """The Zipf batch: hot experts run 224-row token tiles."""
    wl = I.SKEWED
    d, toks, ref, idx = block_skewed
    out, a = run_block_layer(wl, d, L.exec_config(fp8=2, **ex))
    check_routing(wl, d, a, toks, idx)
    assert_layer_close(out[torch.as_tensor(toks, device=DEV)], ref)
