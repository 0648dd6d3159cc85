"""Per-entry-point GPU parity against the CPU oracle, through the C ABI.

Routing indices, counts, offsets and the permutation are compared bit for
bit; floating-point outputs within bounds derived from their arithmetic:
fp32 logits within the worst-case summation bound H*u*sum|x*Wr|; the
SwiGLU activations h equal the oracle's bf16-rounded h except for rare
one-ulp flips; fp32 GEMM2 outputs within the fp32 summation bound of the
fp64 result; combine within (k+1) fp32 roundings (+ bf16 output rounding).
"""

import numpy as np
import pytest
import torch

from oracle import moe_oracle as O
from paper_2603_02376_gb300 import _lib as L
from paper_2603_02376_gb300 import inputs as I
from tests._support import U32, UBF16, f64, logits_bound

pytestmark = pytest.mark.gpu
DEV = "cuda"


@pytest.fixture(scope="module", autouse=True)
def lib():
    return L.load()


def rand_bf16(shape, seed, std=1.0):
    g = torch.Generator(device=DEV).manual_seed(seed)
    return (torch.randn(shape, generator=g, device=DEV) * std).to(torch.bfloat16)


# ---------------------------------------------------------------- router logits

@pytest.mark.parametrize("T,H,E", [(64, 256, 8), (100, 384, 96), (128, 7168, 256), (1, 128, 1000),
                                   (4096, 7168, 256), (300, 384, 128), (1, 7168, 256),
                                   (333, 1024, 384)])
def test_router_logits(T, H, E):
    """With a workspace and E % 128 == 0 the tensor-core path runs (three exact bf16
    planes of Wr); without one the fp32 SIMT kernel does. Both stay within the
    worst-case fp32 summation bound of the fp64 product."""
    cfg = L.config(T, H, E, min(8, E), 128)
    x = rand_bf16((T, H), 1)
    g = torch.Generator(device=DEV).manual_seed(2)
    Wr = torch.randn((E, H), generator=g, device=DEV) * 0.01
    out = torch.full((T, E), float("nan"), device=DEV)
    n = L.moe_router_workspace_size(cfg)
    ws = torch.empty(max(n, 4), dtype=torch.uint8, device=DEV)
    L.moe_router_logits(cfg, x, Wr, out, ws if n else None)
    out2 = torch.full((T, E), float("nan"), device=DEV)
    L.moe_router_logits(cfg, x, Wr, out2, None)   # unsplit path
    torch.cuda.synchronize()
    xh, Wh = f64(x), f64(Wr)
    ref = xh @ Wh.T
    bound = logits_bound(xh, Wh)
    for o in (out, out2):
        err = np.abs(f64(o) - ref)
        assert np.isfinite(err).all()
        assert (err <= bound).all(), f"max err {err.max():.3e}"
    # split-K partials are summed in a fixed order: repeatable bit for bit
    out3 = torch.empty_like(out)
    L.moe_router_logits(cfg, x, Wr, out3, ws if n else None)
    torch.cuda.synchronize()
    assert torch.equal(out, out3)
    if E % 128 == 0:
        # the three bf16 planes left in the workspace add up to Wr (to 2^-26 |w|)
        planes = ws[: 3 * E * H * 2].view(torch.bfloat16).view(3, E, H).to(torch.float64)
        recon = planes.sum(0).cpu().numpy()
        assert (np.abs(recon - Wh) <= 2.0 ** -26 * np.abs(Wh)).all()
        assert (planes[0] == Wr.to(torch.bfloat16).to(torch.float64)).all()


# ---------------------------------------------------------------- gate / top-k

def margin_logits(T, E, cfg, bias, seed):
    """Random fp32 logits, rows redrawn until every routing margin > 1e-3."""
    rng = np.random.default_rng(seed)
    Lg = (rng.standard_normal((T, E)) * 1.2).astype(np.float32)
    for _ in range(200):
        bad = np.nonzero(O.routing_margins(Lg, bias, cfg) <= 1e-3)[0]
        if bad.size == 0:
            return Lg
        Lg[bad] = (rng.standard_normal((bad.size, E)) * 1.2).astype(np.float32)
    raise RuntimeError("could not draw well-separated logits")


@pytest.mark.parametrize("T,E,k,G,KG,gate,norm,scale,with_bias", [
    (64, 8, 2, 1, 1, O.GATE_SOFTMAX, 0, 1.0, False),
    (128, 256, 8, 8, 4, O.GATE_SIGMOID, 1, 2.5, True),
    (1000, 256, 8, 8, 4, O.GATE_SIGMOID, 1, 2.5, True),
    (37, 96, 6, 4, 2, O.GATE_SIGMOID, 1, 1.0, True),
    (50, 1000, 8, 8, 3, O.GATE_SIGMOID, 1, 2.5, True),
    (33, 64, 32, 2, 1, O.GATE_SOFTMAX, 1, 1.0, False),
    (17, 16, 16, 1, 1, O.GATE_SIGMOID, 0, 1.0, True),
    (9, 1, 1, 1, 1, O.GATE_SOFTMAX, 0, 1.0, False),
])
def test_gate_topk_bit_exact(T, E, k, G, KG, gate, norm, scale, with_bias):
    cfg = O.LayerConfig(T=T, H=128, E=E, k=k, I=128, n_groups=G, topk_groups=KG, gate=gate,
                        normalize=norm, route_scale=scale)
    rng = np.random.default_rng(T + E)
    b = (rng.standard_normal(E) * 0.05).astype(np.float32) if with_bias else None
    Lg = margin_logits(T, E, cfg, b, seed=T * 7 + E) if E > k else \
        rng.standard_normal((T, E)).astype(np.float32)
    c = L.config(T, 128, E, k, 128, 0, G, KG, gate, norm, scale)
    logits = torch.from_numpy(Lg).to(DEV)
    bias = None if b is None else torch.from_numpy(b).to(DEV)
    idx = torch.full((T, k), -1, dtype=torch.int32, device=DEV)
    w = torch.full((T, k), float("nan"), device=DEV)
    L.moe_gate_topk(c, logits, bias, idx, w)
    torch.cuda.synchronize()
    ridx, rw = O.gate_topk(Lg, b, cfg)
    np.testing.assert_array_equal(idx.cpu().numpy(), ridx)
    np.testing.assert_allclose(w.cpu().numpy(), rw, rtol=1e-5, atol=1e-7)


# ---------------------------------------------------------------- dispatch (permutation + packing)

def routing(T, E, k, seed, skew=0.0):
    rng = np.random.default_rng(seed)
    p = np.arange(1, E + 1, dtype=np.float64) ** (-skew)
    p /= p.sum()
    return np.stack([rng.choice(E, size=k, replace=False, p=p) for _ in range(T)]).astype(np.int32)


@pytest.mark.parametrize("T,E,k,H,skew", [
    (1, 8, 2, 128, 0.0), (64, 8, 2, 256, 0.0), (300, 16, 4, 128, 0.0), (129, 256, 8, 128, 0.0),
    (4096, 256, 8, 7168, 0.0), (2000, 256, 8, 256, 1.2), (1000, 1000, 8, 128, 0.5),
    (257, 4, 4, 128, 0.0),
])
def test_dispatch_bit_exact(T, E, k, H, skew):
    idx_h = routing(T, E, k, T + E, skew)
    c = L.config(T, H, E, k, 128)
    idx = torch.from_numpy(idx_h).to(DEV)
    x = rand_bf16((T, H), 5)
    counts = torch.full((E,), -1, dtype=torch.int32, device=DEV)
    offsets = torch.full((E + 1,), -1, dtype=torch.int32, device=DEV)
    rst = torch.full((T * k,), -1, dtype=torch.int32, device=DEV)
    slot = torch.full((T * k,), -1, dtype=torch.int32, device=DEV)
    xp = torch.zeros((T * k, H), dtype=torch.bfloat16, device=DEV)
    ws = torch.empty(L.moe_dispatch_workspace_size(c), dtype=torch.uint8, device=DEV)
    L.moe_dispatch(c, x, idx, counts, offsets, rst, slot, xp, ws)
    torch.cuda.synchronize()
    rc, ro, rr, rs = O.permutation(idx_h, E)
    np.testing.assert_array_equal(counts.cpu().numpy(), rc)
    np.testing.assert_array_equal(offsets.cpu().numpy(), ro)
    np.testing.assert_array_equal(rst.cpu().numpy(), rr)
    np.testing.assert_array_equal(slot.cpu().numpy(), rs)
    assert torch.equal(xp, x[torch.from_numpy(rr).long().to(DEV)])   # a pure copy
    # permutation only (x_perm NULL)
    L.moe_dispatch(c, None, idx, counts, offsets, rst, slot, None, ws)
    torch.cuda.synchronize()
    np.testing.assert_array_equal(slot.cpu().numpy(), rs)


# ---------------------------------------------------------------- combine

@pytest.mark.parametrize("T,H,k,E,shared,out_fp32", [
    (64, 256, 2, 8, False, 1), (64, 256, 2, 8, False, 0), (128, 7168, 8, 256, True, 1),
    (333, 384, 8, 64, True, 0), (1, 128, 1, 1, True, 1),
])
def test_combine(T, H, k, E, shared, out_fp32):
    idx_h = routing(T, E, k, 11 * T + k)
    _, _, _, slot_h = O.permutation(idx_h, E)
    c = L.config(T, H, E, k, 128)
    y = rand_bf16((T * k, H), 6).float() * 1.37
    rng = np.random.default_rng(3)
    w_h = rng.uniform(0, 1, (T, k)).astype(np.float32)
    sh = rand_bf16((T, H), 7).float() * 0.71 if shared else None
    out = torch.empty((T, H), dtype=torch.float32 if out_fp32 else torch.bfloat16, device=DEV)
    L.moe_combine(c, y, torch.from_numpy(slot_h).to(DEV), torch.from_numpy(w_h).to(DEV), sh, out,
                  out_fp32)
    torch.cuda.synchronize()
    ref = O.combine(f64(y), slot_h, w_h.astype(np.float64), None if sh is None else f64(sh))
    mag = O.combine(np.abs(f64(y)), slot_h, np.abs(w_h.astype(np.float64)),
                    None if sh is None else np.abs(f64(sh)))
    bound = (k + 1) * U32 * mag + (0 if out_fp32 else UBF16 * np.abs(ref)) + 1e-30
    err = np.abs(f64(out) - ref)
    assert (err <= bound * 1.0001).all(), f"max err {err.max():.3e}"


def test_dispatch_identity_combine_roundtrip():
    """dispatch -> identity experts -> combine with weights 1/k returns x exactly."""
    T, H, E, k = 1000, 7168, 256, 8
    idx_h = routing(T, E, k, 99)
    c = L.config(T, H, E, k, 128)
    x = rand_bf16((T, H), 8)
    idx = torch.from_numpy(idx_h).to(DEV)
    counts = torch.empty(E, dtype=torch.int32, device=DEV)
    offsets = torch.empty(E + 1, dtype=torch.int32, device=DEV)
    rst = torch.empty(T * k, dtype=torch.int32, device=DEV)
    slot = torch.empty(T * k, dtype=torch.int32, device=DEV)
    xp = torch.empty((T * k, H), dtype=torch.bfloat16, device=DEV)
    ws = torch.empty(L.moe_dispatch_workspace_size(c), dtype=torch.uint8, device=DEV)
    L.moe_dispatch(c, x, idx, counts, offsets, rst, slot, xp, ws)
    w = torch.full((T, k), 1.0 / k, device=DEV)
    yp = xp.float()   # identity experts: y = x_perm (fp32 expert outputs)
    out = torch.empty((T, H), dtype=torch.float32, device=DEV)
    L.moe_combine(c, yp, slot, w, None, out, 1)
    outb = torch.empty((T, H), dtype=torch.bfloat16, device=DEV)
    L.moe_combine(c, yp, slot, w, None, outb, 0)
    torch.cuda.synchronize()
    assert torch.equal(out, x.float())
    assert torch.equal(outb, x)
    w1 = torch.ones((T, k), device=DEV)
    L.moe_combine(c, yp, slot, w1, None, out, 1)
    torch.cuda.synchronize()
    assert torch.equal(out, x.float() * k)


# ---------------------------------------------------------------- grouped expert FFN (tcgen05)

def ffn_case(counts, H, Iw, seed, rows_extra=3):
    E = len(counts)
    rows = int(sum(counts)) + rows_extra
    offs = np.zeros(E + 1, dtype=np.int32)
    offs[1:] = np.cumsum(counts)
    xp = rand_bf16((rows, H), seed)
    W13 = rand_bf16((E, 2 * Iw, H), seed + 1, 0.05)
    W2 = rand_bf16((E, H, Iw), seed + 2, 0.05)
    return rows, offs, xp, W13, W2


@pytest.mark.parametrize("rows,K", [(128, 64), (256, 7168), (4096, 2048), (384, 192)])
def test_pack_weights_layout(rows, K):
    """Every 128 x 64 tile becomes one contiguous block, tiles in (row block, k block) order."""
    W = rand_bf16((rows, K), rows + K)
    Wp = torch.empty_like(W)
    L.moe_pack_weights(W, Wp)
    torch.cuda.synchronize()
    # tile order (row block, column block); inside a tile row r's 16-byte chunk j
    # sits at chunk j ^ (r % 8)
    t = W.view(rows // 128, 128, K // 64, 8, 8).permute(0, 2, 1, 3, 4)  # [rb, cb, r, j, 8]
    r = torch.arange(128, device=DEV).view(128, 1)
    j = torch.arange(8, device=DEV).view(1, 8)
    dst = (j ^ (r % 8))                                                     # [r, j]
    ref = torch.empty_like(t)
    ref[:, :, r.expand(128, 8), dst, :] = t
    assert torch.equal(Wp.view_as(ref), ref)


@pytest.mark.parametrize("packed", [0, 1])
@pytest.mark.parametrize("counts,H,Iw", [
    ([5, 0, 17, 1], 256, 128),                          # tiny, ragged, an empty expert
    ([300, 256, 257, 0, 1, 16], 256, 256),              # multi-tile experts, tile edges
    ([4] * 60 + [0, 12, 31, 33], 512, 256),             # decode-like: small token tiles
    ([0, 0, 0, 40], 384, 128),
    ([150, 100, 0, 145, 3], 512, 256),                  # 144-row tiles, experts over two tiles
    # experts of 127/128/129 rows and multi-tile experts with 128-row tails, for
    # 256- and 144-row tiles and one (H % 256 != 0) or two weight tiles per GEMM2 unit
    ([128, 129, 127, 384, 0, 200], 256, 256),
    ([128, 129, 16, 144, 273, 0, 60], 256, 256),
    ([128, 129, 16, 144, 273, 0, 60], 384, 128),
    ([300, 1, 128, 200], 384, 128),
    ([130, 111], 7168, 2048),                           # the real layer shape
    ([1] * 48 + [3, 7], 7168, 2048),                    # decode: few rows per expert
])
def test_expert_ffn(counts, H, Iw, packed):
    rows, offs, xp, W13, W2 = ffn_case(counts, H, Iw, seed=len(counts) + H)
    E = len(counts)
    sentinel = -12345.0
    y = torch.full((rows, H), sentinel, dtype=torch.float32, device=DEV)
    ws = torch.zeros(L.moe_expert_ffn_workspace_size(rows, Iw), dtype=torch.uint8, device=DEV)
    W13g, W2g = (L.pack_weights(W13), L.pack_weights(W2)) if packed else (W13, W2)
    L.moe_expert_ffn(rows, H, Iw, E, xp, torch.from_numpy(offs).to(DEV), W13g, W2g, y, ws,
                     weights_packed=packed)
    L.moe_check_errors()
    h = ws.view(torch.bfloat16).view(rows, Iw)
    n = int(offs[-1])
    xh = f64(xp)
    # oracle, expert by expert (fp64 with bf16-rounded h)
    for e in range(E):
        a, b = int(offs[e]), int(offs[e + 1])
        if b == a:
            continue
        We13, We2 = f64(W13[e]), f64(W2[e])
        g = xh[a:b] @ We13[:Iw].T
        u = xh[a:b] @ We13[Iw:].T
        h_ref = O.bf16_round(O.silu(g) * u)
        hg = f64(h[a:b])
        diff = np.abs(hg - h_ref)
        # one bf16 ulp, plus the fp32 summation error of g and u carried through
        # silu(g) * u (matters only where g or u nearly cancels and h is tiny)
        xa = np.abs(xh[a:b])
        dg = H * 2.0 ** -24 * (xa @ np.abs(We13[:Iw]).T)
        du = H * 2.0 ** -24 * (xa @ np.abs(We13[Iw:]).T)
        sg = 1.0 / (1.0 + np.exp(-g))
        dsilu = np.abs(sg * (1.0 + g * (1.0 - sg))) + dg
        lim = (np.abs(h_ref) * 2.0 ** -7 + (dsilu * np.abs(u) * dg + np.abs(O.silu(g)) * du
                                              + dsilu * dg * du) * (1 + 2.0 ** -7)) * 1.0001
        assert (diff <= lim + 1e-30).all(), f"expert {e}: h outside one ulp + fp32 bound"
        assert (diff == 0).mean() > 0.98, f"expert {e}: too many h rounding flips"
        # GEMM2 given the GPU's own h: fp32 output, within the fp32 summation bound
        y_ref = hg @ We2.T
        acc_bound = Iw * 2.0 ** -24 * (np.abs(hg) @ np.abs(We2).T)
        yg = f64(y[a:b])
        err = np.abs(yg - y_ref)
        assert (err <= acc_bound + 1e-30).all(), f"expert {e}: max err {err.max():.3e}"
        # end to end against the oracle's own h: the h flips above are the only extra term
        y_or = h_ref @ We2.T
        flip = np.abs(hg - h_ref) @ np.abs(We2).T
        assert (np.abs(yg - y_or) <= acc_bound + flip * 1.0001 + 1e-30).all()
    # rows outside every segment are untouched
    assert (y[n:] == sentinel).all()
