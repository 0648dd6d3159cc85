"""Pins for the CPU oracle: closed forms, hand-worked cases, invariants and brute force.

Every check here is computed independently of the oracle's own code path
(pure-Python loops, textbook identities, torch's bf16 conversion, values worked
out by hand in the comments), so that a dropped term, a wrong sign or index or a
transposed operand in the oracle fails at least one of them.
"""

import json
import math
import os

import numpy as np
import pytest
import torch

from oracle import moe_oracle as O
from paper_2603_02376_gb300 import inputs as I

HERE = os.path.dirname(os.path.abspath(__file__))


def cfg_of(wl, **kw):
    d = dict(T=wl.T, H=wl.H, E=wl.E, k=wl.k, I=wl.I, I_shared=wl.I_shared,
             n_groups=wl.n_groups, topk_groups=wl.topk_groups, gate=wl.gate,
             normalize=wl.normalize, route_scale=wl.route_scale)
    d.update(kw)
    return O.LayerConfig(**d)


# ---------------------------------------------------------------- number formats

def test_bf16_round_matches_torch_on_fp32_values():
    g = torch.Generator().manual_seed(1)
    a = torch.randn(100000, generator=g) * torch.exp(torch.randn(100000, generator=g) * 4)
    ref = a.to(torch.bfloat16).to(torch.float64).numpy()
    got = O.bf16_round(a.to(torch.float64).numpy())
    np.testing.assert_array_equal(got, ref)


def test_bf16_round_ties_to_even_by_hand():
    # ulp(1) in bf16 is 2^-7. 1 + 2^-8 is halfway between 1 and 1 + 2^-7 -> even (1).
    # 1 + 3*2^-8 is halfway between 1 + 2^-7 (odd) and 1 + 2^-6 (even) -> 1 + 2^-6.
    vals = [1 + 2**-8, 1 + 3 * 2**-8, -(1 + 2**-8), 3.0, 0.0, 2**-9 * 3]
    exp = [1.0, 1 + 2**-6, -1.0, 3.0, 0.0, 2**-9 * 3]
    np.testing.assert_array_equal(O.bf16_round(vals), exp)


def test_sigmoid_and_silu_closed_forms():
    assert O.sigmoid(0.0) == 0.5
    x = np.linspace(-20, 20, 81)
    np.testing.assert_allclose(O.sigmoid(-x), 1 - O.sigmoid(x), atol=1e-15)
    assert O.silu(0.0) == 0.0
    np.testing.assert_allclose(O.silu(x), x * O.sigmoid(x), rtol=1e-15, atol=1e-300)
    assert abs(O.silu(40.0) - 40.0) < 1e-12
    assert abs(O.silu(-40.0)) < 1e-12
    # silu'(0) = 1/2: symmetric difference quotient
    assert abs((O.silu(1e-6) - O.silu(-1e-6)) / 2e-6 - 0.5) < 1e-9


# ---------------------------------------------------------------- router logits

def test_router_logits_pure_python():
    rng = np.random.default_rng(3)
    x = O.bf16_round(rng.standard_normal((5, 7)))
    Wr = rng.standard_normal((4, 7)).astype(np.float32)
    got = O.router_logits(x, Wr)
    assert got.dtype == np.float32
    for t in range(5):
        for e in range(4):
            s = math.fsum(float(x[t, h]) * float(Wr[e, h]) for h in range(7))
            assert got[t, e] == np.float32(s)


# ---------------------------------------------------------------- gate / top-k

def test_gate_group_limited_hand_worked():
    # All logits 0 -> every sigmoid score is exactly 0.5; selection score = 0.5 + b.
    # Groups of 2: g0 {e0,e1} = 0.78+0.20 = 0.98, g1 {e2,e3} = 0.80+0.50 = 1.30,
    # g2 {e4,e5} = 0.60+0.60 = 1.20, g3 {e6,e7} = 0.30+0.30 = 0.60.
    # Top-2 groups: g1, g2 -> kept experts {2,3,4,5}. Top-2 experts: e2 (0.80), then
    # e4/e5 tie at 0.60 -> lower index e4. (Without groups it would pick e2, e0.)
    # Weights: 0.5/(0.5+0.5) * 2.5 = 1.25 each.
    cfg = O.LayerConfig(T=1, H=1, E=8, k=2, I=1, n_groups=4, topk_groups=2,
                        gate=O.GATE_SIGMOID, normalize=1, route_scale=2.5)
    b = np.array([0.28, -0.30, 0.30, 0.0, 0.10, 0.10, -0.2, -0.2], dtype=np.float32)
    L = np.zeros((1, 8), dtype=np.float32)
    idx, w = O.gate_topk(L, b, cfg)
    assert idx.tolist() == [[2, 4]]
    np.testing.assert_allclose(w, [[1.25, 1.25]], rtol=0, atol=1e-15)
    cfg1 = O.LayerConfig(T=1, H=1, E=8, k=2, I=1, n_groups=1, topk_groups=1,
                         gate=O.GATE_SIGMOID, normalize=1, route_scale=2.5)
    idx1, _ = O.gate_topk(L, b, cfg1)
    assert idx1.tolist() == [[2, 0]]


def test_gate_softmax_hand_worked():
    # L = ln(1..4): softmax = (1,2,3,4)/10. Top-2: e3 (0.4), e2 (0.3); weights not renormalised.
    cfg = O.LayerConfig(T=1, H=1, E=4, k=2, I=1, gate=O.GATE_SOFTMAX, normalize=0, route_scale=1.0)
    L = np.log(np.array([[1, 2, 3, 4]], dtype=np.float64)).astype(np.float32)
    idx, w = O.gate_topk(L, None, cfg)
    assert idx.tolist() == [[3, 2]]
    np.testing.assert_allclose(w, [[0.4, 0.3]], rtol=1e-6)


def brute_gate(L32, bias, cfg):
    """Independent statement of the routing rule with Python loops and math.exp."""
    T, E = L32.shape
    out_idx, out_w = [], []
    for t in range(T):
        Lt = [float(v) for v in L32[t]]
        if cfg.gate == O.GATE_SIGMOID:
            s = [1.0 / (1.0 + math.exp(-v)) for v in Lt]
        else:
            m = max(Lt)
            z = [math.exp(v - m) for v in Lt]
            tot = math.fsum(z)
            s = [v / tot for v in z]
        s32 = [np.float32(v) for v in s]
        sel = [np.float32(s32[e] + (np.float32(bias[e]) if bias is not None else np.float32(0)))
               for e in range(E)]
        G = cfg.n_groups
        gs = E // G
        allowed = set(range(E))
        if G > 1 and cfg.topk_groups < G:
            gscore = []
            for g in range(G):
                mem = sorted(sel[g * gs:(g + 1) * gs], reverse=True)
                gscore.append(np.float32(mem[0] + mem[1]) if gs > 1 else mem[0])
            groups = sorted(range(G), key=lambda g: (-float(gscore[g]), g))[: cfg.topk_groups]
            allowed = {e for g in groups for e in range(g * gs, (g + 1) * gs)}
        chosen = sorted(allowed, key=lambda e: (-float(sel[e]), e))[: cfg.k]
        ws = [s[e] for e in chosen]
        if cfg.normalize:
            tot = math.fsum(ws)
            ws = [v / tot for v in ws]
        out_idx.append(chosen)
        out_w.append([v * cfg.route_scale for v in ws])
    return np.array(out_idx), np.array(out_w)


@pytest.mark.parametrize("E,G,KG,k,gate,norm", [
    (16, 4, 2, 3, O.GATE_SIGMOID, 1),
    (32, 8, 4, 8, O.GATE_SIGMOID, 1),
    (8, 1, 1, 2, O.GATE_SOFTMAX, 0),
    (12, 3, 3, 4, O.GATE_SIGMOID, 1),
    (10, 5, 1, 2, O.GATE_SOFTMAX, 1),
])
def test_gate_matches_brute_force(E, G, KG, k, gate, norm):
    rng = np.random.default_rng(E * 100 + k)
    T = 200
    L = (rng.standard_normal((T, E)) * 1.5).astype(np.float32)
    bias = (rng.standard_normal(E) * 0.05).astype(np.float32)
    cfg = O.LayerConfig(T=T, H=1, E=E, k=k, I=1, n_groups=G, topk_groups=KG, gate=gate,
                        normalize=norm, route_scale=2.5 if norm else 1.0)
    idx, w = O.gate_topk(L, bias, cfg)
    bidx, bw = brute_gate(L, bias, cfg)
    np.testing.assert_array_equal(idx, bidx)
    np.testing.assert_allclose(w, bw, rtol=1e-13)


def test_gate_single_group_is_plain_topk():
    rng = np.random.default_rng(5)
    L = rng.standard_normal((300, 64)).astype(np.float32)
    cfg = O.LayerConfig(T=300, H=1, E=64, k=6, I=1, n_groups=1, topk_groups=1)
    idx, _ = O.gate_topk(L, None, cfg)
    ref = torch.topk(torch.sigmoid(torch.from_numpy(L).double()), 6, dim=1).indices.numpy()
    np.testing.assert_array_equal(idx, ref)


def test_gate_weight_sums():
    rng = np.random.default_rng(6)
    L = rng.standard_normal((100, 32)).astype(np.float32)
    cfg = O.LayerConfig(T=100, H=1, E=32, k=4, I=1, n_groups=4, topk_groups=2, normalize=1,
                        route_scale=2.5)
    _, w = O.gate_topk(L, None, cfg)
    np.testing.assert_allclose(w.sum(1), 2.5, rtol=1e-14)
    cfgs = O.LayerConfig(T=100, H=1, E=32, k=4, I=1, gate=O.GATE_SOFTMAX, normalize=0)
    _, ws = O.gate_topk(L, None, cfgs)
    assert (ws.sum(1) < 1).all() and (ws > 0).all()
    # top-k softmax weights are the k largest probabilities, descending
    assert (np.diff(ws, axis=1) <= 0).all()


def test_routing_margins_brute_force():
    rng = np.random.default_rng(7)
    E, G, KG, k = 16, 4, 2, 3
    L = rng.standard_normal((50, E)).astype(np.float32)
    b = (rng.standard_normal(E) * 0.05).astype(np.float32)
    cfg = O.LayerConfig(T=50, H=1, E=E, k=k, I=1, n_groups=G, topk_groups=KG)
    m = O.routing_margins(L, b, cfg)
    for t in range(50):
        s = [np.float32(np.float32(1 / (1 + math.exp(-float(v)))) + bb) for v, bb in zip(L[t], b)]
        gsc = [np.float32(sorted(s[g * 4:(g + 1) * 4], reverse=True)[0]
                          + sorted(s[g * 4:(g + 1) * 4], reverse=True)[1]) for g in range(G)]
        gs_sorted = sorted([float(v) for v in gsc], reverse=True)
        kept = sorted(range(G), key=lambda g: (-float(gsc[g]), g))[:KG]
        ks = sorted([float(s[e]) for g in kept for e in range(g * 4, g * 4 + 4)], reverse=True)
        ref = min(ks[k - 1] - ks[k], gs_sorted[KG - 1] - gs_sorted[KG])
        assert abs(m[t] - ref) < 1e-12


# ---------------------------------------------------------------- permutation

def test_permutation_hand_worked():
    idx = np.array([[1, 0], [0, 1], [1, 2]])
    counts, offsets, rst, slot_row = O.permutation(idx, 3)
    assert counts.tolist() == [2, 3, 1]
    assert offsets.tolist() == [0, 2, 5, 6]
    assert rst.tolist() == [0, 1, 0, 1, 2, 2]
    assert slot_row.tolist() == [2, 0, 1, 3, 4, 5]


@pytest.mark.parametrize("T,E,k", [(1, 4, 2), (257, 16, 4), (1000, 256, 8), (33, 8, 8)])
def test_permutation_invariants(T, E, k):
    rng = np.random.default_rng(T + E)
    idx = np.stack([rng.permutation(E)[:k] for _ in range(T)])
    counts, offsets, rst, slot_row = O.permutation(idx, E)
    assert counts.sum() == T * k
    assert offsets[0] == 0 and (np.diff(offsets) == counts).all()
    assert sorted(slot_row.tolist()) == list(range(T * k))      # a bijection
    for t in range(T):
        for j in range(k):
            r = slot_row[t * k + j]
            assert rst[r] == t
            e = idx[t, j]
            assert offsets[e] <= r < offsets[e + 1]
    # stability: within an expert, rows are ordered by (t, j)
    for e in range(E):
        seg = [(rst[r], None) for r in range(offsets[e], offsets[e + 1])]
        toks = [s[0] for s in seg]
        assert toks == sorted(toks)
    # each token appears in exactly k rows
    assert np.bincount(rst, minlength=T).tolist() == [k] * T


def test_dispatch_identity_combine_roundtrip():
    rng = np.random.default_rng(8)
    T, H, E, k = 97, 64, 16, 8
    x = O.bf16_round(rng.standard_normal((T, H)))
    idx = np.stack([rng.permutation(E)[:k] for _ in range(T)])
    _, _, rst, slot_row = O.permutation(idx, E)
    xp = O.dispatch(x, rst)
    out = O.combine(xp, slot_row, np.full((T, k), 1.0 / k))
    np.testing.assert_array_equal(out, x)       # exact: x/8 and sums of 8 bf16 values fit fp64
    out1 = O.combine(xp, slot_row, np.ones((T, k)))
    np.testing.assert_array_equal(out1, k * x)


# ---------------------------------------------------------------- SwiGLU experts

def test_swiglu_pure_python():
    rng = np.random.default_rng(9)
    H, Iw, m = 5, 3, 4
    rows = O.bf16_round(rng.standard_normal((m, H)))
    W13 = O.bf16_round(rng.standard_normal((2 * Iw, H)) * 0.5)
    W2 = O.bf16_round(rng.standard_normal((H, Iw)) * 0.5)
    got = O.swiglu_ffn(rows, W13, W2)
    for r in range(m):
        hs = []
        for i in range(Iw):
            g = math.fsum(rows[r, c] * W13[i, c] for c in range(H))
            u = math.fsum(rows[r, c] * W13[Iw + i, c] for c in range(H))
            hv = g / (1 + math.exp(-g)) * u
            hs.append(float(torch.tensor(hv, dtype=torch.float32).to(torch.bfloat16)))
        for c in range(H):
            y = math.fsum(hs[i] * W2[c, i] for i in range(Iw))
            assert abs(got[r, c] - y) < 1e-12 * max(1.0, abs(y))


def test_swiglu_closed_form():
    # Gate row picks x0, up row picks x1: h = silu(x0) * x1; W2 copies h to output 0.
    H, Iw = 2, 1
    W13 = np.array([[1.0, 0.0], [0.0, 1.0]])
    W2 = np.array([[1.0], [0.0]])
    rows = np.array([[2.0, 3.0], [-1.0, 0.5], [0.0, 7.0]])
    got = O.swiglu_ffn(rows, W13, W2)
    exp0 = [O.bf16_round(2 / (1 + math.exp(-2)) * 3), O.bf16_round(-1 / (1 + math.e) * 0.5), 0.0]
    np.testing.assert_array_equal(got[:, 0], exp0)
    np.testing.assert_array_equal(got[:, 1], 0.0)


def dense_layer(x, L32, bias, W13, W2, cfg, Ws13=None, Ws2=None):
    """Brute force: every expert on every token, masked by the dense gate matrix."""
    T = x.shape[0]
    idx, w = brute_gate(L32, bias, cfg)
    G = np.zeros((T, cfg.E))
    for t in range(T):
        for j in range(cfg.k):
            G[t, idx[t, j]] = w[t, j]
    out = np.zeros((T, cfg.H))
    for e in range(cfg.E):
        out += G[:, e:e + 1] * O.swiglu_ffn(x, W13[e], W2[e])
    if Ws13 is not None:
        out += O.swiglu_ffn(x, Ws13, Ws2)
    return out


def _np_inputs(wl, seed=0):
    d = I.layer_inputs(wl, seed=seed, device="cpu")
    f = lambda t: None if t is None else t.to(torch.float64).numpy()
    return {k: f(v) for k, v in d.items()}


def test_layer_matches_dense_brute_force_tiny():
    wl = I.TINY
    cfg = cfg_of(wl)
    d = _np_inputs(wl)
    out, aux = O.layer_forward(d["x"], d["Wr"], None, d["W13"], d["W2"], cfg)
    ref = dense_layer(d["x"], aux["logits"], None, d["W13"], d["W2"], cfg)
    np.testing.assert_allclose(out, ref, rtol=1e-12, atol=1e-12)


def test_layer_matches_dense_brute_force_grouped_shared():
    wl = I.Workload("small grouped", T=40, H=64, E=16, k=4, I=32, I_shared=48, n_groups=4,
                    topk_groups=2, gate=I.GATE_SIGMOID, normalize=1, route_scale=2.5)
    cfg = cfg_of(wl)
    d = _np_inputs(wl, seed=3)
    out, aux = O.layer_forward(d["x"], d["Wr"], d["bias"].astype(np.float32), d["W13"], d["W2"],
                               cfg, d["Ws13"], d["Ws2"])
    ref = dense_layer(d["x"], aux["logits"], d["bias"].astype(np.float32), d["W13"], d["W2"], cfg,
                      d["Ws13"], d["Ws2"])
    np.testing.assert_allclose(out, ref, rtol=1e-12, atol=1e-12)
    assert aux["counts"].sum() == wl.T * wl.k


def test_layer_forward_tokens_equals_full_layer():
    wl = I.Workload("small grouped", T=30, H=64, E=16, k=4, I=32, I_shared=32, n_groups=4,
                    topk_groups=2, gate=I.GATE_SIGMOID, normalize=1, route_scale=2.5)
    cfg = cfg_of(wl)
    d = _np_inputs(wl, seed=4)
    b = d["bias"].astype(np.float32)
    out, _ = O.layer_forward(d["x"], d["Wr"], b, d["W13"], d["W2"], cfg, d["Ws13"], d["Ws2"])
    toks = np.array([0, 3, 7, 29])
    sub, idx, w = O.layer_forward_tokens(d["x"][toks], d["Wr"], b,
                                         lambda e: (d["W13"][e], d["W2"][e]), cfg,
                                         lambda: (d["Ws13"], d["Ws2"]))
    np.testing.assert_allclose(sub, out[toks], rtol=1e-13, atol=1e-13)


# ---------------------------------------------------------------- planted mistakes

@pytest.mark.parametrize("mutation", ["swap_gate_up", "no_bias", "no_normalise", "transpose_w2"])
def test_planted_oracle_mistakes_are_caught(mutation, monkeypatch):
    """Each plausible oracle mistake, planted in the oracle, fails an independent pin."""
    rng = np.random.default_rng(11)
    if mutation in ("no_bias", "no_normalise"):
        E = 16
        L = rng.standard_normal((100, E)).astype(np.float32)
        b = (rng.standard_normal(E) * 0.3).astype(np.float32)
        cfg = O.LayerConfig(T=100, H=1, E=E, k=3, I=1, n_groups=4, topk_groups=2, route_scale=2.5)
        if mutation == "no_bias":
            real = O.selection_scores
            monkeypatch.setattr(O, "selection_scores", lambda L32, b32, c: real(L32, None, c))
        else:
            cfg = O.LayerConfig(**{**cfg.__dict__, "normalize": 0})
        idx, w = O.gate_topk(L, b, cfg)
        bidx, bw = brute_gate(L, b, O.LayerConfig(T=100, H=1, E=E, k=3, I=1, n_groups=4,
                                                  topk_groups=2, route_scale=2.5))
        assert not (np.array_equal(idx, bidx) and np.allclose(w, bw))
        return
    H, Iw, m = 6, 4, 3
    rows = O.bf16_round(rng.standard_normal((m, H)))
    W13 = O.bf16_round(rng.standard_normal((2 * Iw, H)))
    W2 = O.bf16_round(rng.standard_normal((H, Iw)))
    good = O.swiglu_ffn(rows, W13, W2)
    if mutation == "swap_gate_up":
        bad = O.swiglu_ffn(rows, np.concatenate([W13[Iw:], W13[:Iw]]), W2)
    else:
        bad = O.swiglu_ffn(rows, W13, W2.reshape(Iw, H).T)
    assert not np.allclose(good, bad)


# ---------------------------------------------------------------- workloads vs the paper

def test_workload_shapes_match_paper():
    with open(os.path.join(HERE, "golden", "paper_shapes.json")) as f:
        p = json.load(f)
    for wl in (I.DECODE, I.PREFILL, I.SKEWED):
        assert [wl.H, 2 * wl.I] == p["gemm1"]
        assert [wl.I, wl.H] == p["gemm2"]
    assert I.PREFILL.T == p["tokens_per_rank"]


# ---------------------------------------------------------------- FP8 (e4m3) quantization

def test_e4m3_round_matches_torch_inside_the_range():
    g = torch.Generator().manual_seed(4)
    a = torch.randn(200000, generator=g) * torch.exp(torch.randn(200000, generator=g) * 3)
    a = a[a.abs() < 460]                       # torch gives NaN past the range; the oracle saturates
    ref = a.to(torch.float8_e4m3fn).to(torch.float64).numpy()
    np.testing.assert_array_equal(O.e4m3_round(a.to(torch.float64).numpy()), ref)


def test_e4m3_round_by_hand():
    # 3 mantissa bits: between 1 and 2 the grid step is 1/8. 1.0625 is halfway between
    # 1 and 1.125 -> even mantissa (1.0); 1.1875 halfway between 1.125 and 1.25 -> 1.25.
    # 448 is the largest finite value; larger values saturate. Subnormal step 2^-9:
    # 2^-10 is halfway between 0 and 2^-9 -> 0; 3 * 2^-11 -> 2^-9.
    vals = [1.0625, 1.1875, -1.1875, 448.0, 1000.0, -1e9, 2**-10, 3 * 2**-11, 0.0, 240.0, 232.0]
    exp = [1.0, 1.25, -1.25, 448.0, 448.0, -448.0, 0.0, 2**-9, 0.0, 240.0, 224.0]
    np.testing.assert_array_equal(O.e4m3_round(vals), exp)


def test_quantize_rows_closed_form():
    a = np.array([[1.0, -2.0, 0.5], [0.0, 0.0, 0.0], [448.0, 224.0, -112.0]])
    q, s = O.quantize_rows_e4m3(a)
    assert s.dtype == np.float32
    np.testing.assert_array_equal(s, np.float32([2.0 / 448, 1.0, 1.0]))
    # the row maximum maps to +-448 exactly; a zero row stays zero
    assert q[0, 1] == -448.0 and q[2, 0] == 448.0 and (q[1] == 0).all()
    np.testing.assert_array_equal(q[2], [448.0, 224.0, -112.0])
    # dequantized error within half an e4m3 step of the scaled value (relative 2^-4)
    rng = np.random.default_rng(0)
    x = rng.standard_normal((50, 300))
    q, s = O.quantize_rows_e4m3(x)
    deq = q * s[:, None]
    assert (np.abs(deq - x) <= np.abs(x) * 2.0 ** -4 + s[:, None] * 2.0 ** -10 + 1e-12).all()


def test_swiglu_fp8_equals_dequantized_operands():
    # The FP8 form applies the row scales outside the sums; that must equal the same
    # products written with dequantized operands (q * s) inside the sums. Inputs on the
    # e4m3 grid with a row maximum of 448 have scale 1 and quantize to themselves.
    rng = np.random.default_rng(2)
    H, Iw, m = 64, 32, 5
    grid = lambda shape: O.e4m3_round(rng.uniform(-448, 448, shape))
    rows = grid((m, H)); rows[:, 0] = 448.0
    W13 = grid((2 * Iw, H)) / 448.0 / 64.0
    W2 = grid((H, Iw)) / 448.0 / 64.0
    W13q, s13 = O.quantize_rows_e4m3(W13)
    W2q, s2 = O.quantize_rows_e4m3(W2)
    y8 = O.swiglu_ffn_fp8(rows, W13q, s13, W2q, s2)
    # same computation written with the dequantized operands (h re-quantized as in the FP8 form)
    g = rows @ (W13q * s13[:, None].astype(np.float64))[:Iw].T
    u = rows @ (W13q * s13[:, None].astype(np.float64))[Iw:].T
    h = O.bf16_round(O.silu(g) * u)
    hq, sh = O.quantize_rows_e4m3(h)
    y = (hq * sh[:, None].astype(np.float64)) @ (W2q * s2[:, None].astype(np.float64)).T
    np.testing.assert_allclose(y8, y, rtol=1e-12, atol=1e-12)


def test_fp8_linear_by_hand():
    # acc = [[1*3 + 2*4, 1*1 + 2*(-1)]] = [[11, -1]]; scaled by s_a = 0.5 and s_w = (2, 0.25)
    y = O.fp8_linear(np.array([[1.0, 2.0]]), np.array([0.5], np.float32),
                     np.array([[3.0, 4.0], [1.0, -1.0]]), np.array([2.0, 0.25], np.float32))
    np.testing.assert_array_equal(y, [[11.0, -0.125]])


def test_swiglu_h_fp8_row_scale_cancels():
    # Scaling a row by a power of two scales its e4m3 scale alone (same q), so g and u
    # scale with it: h = silu(g) * u for the scaled row follows from the plain one.
    rng = np.random.default_rng(5)
    H, Iw = 32, 16
    rows = O.bf16_round(rng.standard_normal((3, H)))
    W13q, s13 = O.quantize_rows_e4m3(rng.standard_normal((2 * Iw, H)) * 0.05)
    h1 = O.swiglu_h_fp8(rows, W13q, s13)
    xq, sx = O.quantize_rows_e4m3(rows)
    gu = O.fp8_linear(xq, sx, W13q, s13)
    np.testing.assert_array_equal(h1, O.bf16_round(O.silu(gu[:, :Iw]) * gu[:, Iw:]))
    xq4, sx4 = O.quantize_rows_e4m3(rows * 4.0)
    np.testing.assert_array_equal(xq4, xq)
    np.testing.assert_array_equal(sx4, sx * 4)


def test_layer_tokens_fp8_hook_matches_per_expert_calls():
    # the ffn hook of the per-token layer forward: FP8 experts through the same routing
    rng = np.random.default_rng(6)
    cfg = O.LayerConfig(T=6, H=32, E=4, k=2, I=16, gate=O.GATE_SOFTMAX)
    x = O.bf16_round(rng.standard_normal((6, 32)))
    Wr = rng.standard_normal((4, 32)).astype(np.float32) * 0.1
    W13 = [O.quantize_rows_e4m3(rng.standard_normal((32, 32)) * 0.05) for _ in range(4)]
    W2 = [O.quantize_rows_e4m3(rng.standard_normal((32, 16)) * 0.05) for _ in range(4)]
    get = lambda e: (W13[e][0], W13[e][1], W2[e][0], W2[e][1])
    out, idx, w = O.layer_forward_tokens(x, Wr, None, get, cfg, ffn=O.swiglu_ffn_fp8)
    for t in range(6):
        ref = sum(w[t, j] * O.swiglu_ffn_fp8(x[t:t + 1], *get(int(idx[t, j])))[0]
                  for j in range(2))
        np.testing.assert_allclose(out[t], ref, rtol=1e-13, atol=1e-15)


def test_e4m3_decode_every_code():
    codes = np.arange(256, dtype=np.uint8)
    v = O.e4m3_decode(codes)
    ref = torch.from_numpy(codes).view(torch.float8_e4m3fn).to(torch.float64).numpy()
    np.testing.assert_array_equal(v, ref)               # NaN at 0x7f / 0xff on both sides
    # by hand: 1.0, the largest finite, the smallest subnormal, -2.5, -0
    assert O.e4m3_decode([0x38, 0x7E, 0x01, 0xC2, 0x80]).tolist() == [1.0, 448.0, 2.0 ** -9, -2.5, 0.0]
    finite = v[~np.isnan(v)]
    np.testing.assert_array_equal(O.e4m3_round(finite), finite)   # the grid rounds to itself
    assert len(np.unique(finite)) == 253                           # 254 finite codes, +-0 equal


# ------------------------------------------- FP8 with block scales (UE8M0, 1x128 / 128x128)

def test_block_exponent_by_hand():
    # 448 * 2^k >= amax with k minimal: 448 fits at k = 0, 448.5 needs k = 1; 224 = 448 / 2
    # fits at k = -1; 1.0 fits 448 / 256 = 1.75 but not 448 / 512 = 0.875 -> -8; 3.0 fits
    # 3.5 = 448 / 128 but not 1.75 -> -7. An all-zero block takes k = 0; a block far below
    # 448 * 2^-127 is clamped at -127.
    amax = [448.0, 448.5, 224.0, 224.5, 1.0, 3.0, 0.0, 1e-40, 3.3e38]
    assert O.block_exponent(amax).tolist() == [0, 1, -1, 0, -8, -7, 0, -127, 120]


def test_block_exponent_is_the_smallest_fitting_power():
    # brute force: scan k upward until amax <= 448 * 2^k (exact ldexp products)
    rng = np.random.default_rng(11)
    amax = np.ldexp(rng.uniform(1.0, 2.0, 400), rng.integers(-60, 60, 400))
    amax[:8] = [448.0 * 2.0 ** e for e in (-50, -3, 0, 7, 20, 33, 45, 59)]  # exact boundaries
    got = O.block_exponent(amax)
    for a, k in zip(amax.tolist(), got.tolist()):
        kk = -140
        while a > math.ldexp(448.0, kk):
            kk += 1
        assert k == max(kk, -127)


def test_quantize_blocks_by_hand():
    # one activation row of two 128-blocks: block 0 has amax 3 -> k = -7, scaled by 2^7:
    # 3 -> 384 (on the grid: [256, 448) steps 32), -1.5 -> -192 ([128, 256) steps 16),
    # 0.1 -> 12.8 -> 13 ([8, 16) steps 1); block 1 is zero -> k = 0, codes 0.
    row = np.zeros((1, 256))
    row[0, :3] = [3.0, -1.5, 0.1]
    q, k = O.quantize_blocks_e4m3(row, 1)
    assert k.tolist() == [[-7, 0]]
    assert q[0, :4].tolist() == [384.0, -192.0, 13.0, 0.0] and (q[0, 128:] == 0).all()
    # a weight matrix of two 128-row blocks: |v| <= 0.05 -> 2^-13 (448 * 2^-13 = 0.0547,
    # 448 * 2^-14 = 0.0273); a block of 448s -> k = 0 and codes 448
    W = np.full((256, 128), 448.0)
    W[:128] = np.linspace(-0.05, 0.05, 128 * 128).reshape(128, 128)
    q, k = O.quantize_blocks_e4m3(W, 128)
    assert k.tolist() == [[-13], [0]]
    assert (q[128:] == 448.0).all() and np.abs(q[:128]).max() == O.e4m3_round(0.05 * 2 ** 13)


def test_block_quantization_is_local_and_shifts_with_powers_of_two():
    rng = np.random.default_rng(12)
    a = O.bf16_round(rng.standard_normal((4, 384)))
    q, k = O.quantize_blocks_e4m3(a, 1)
    b = a.copy()
    b[2, 128:256] *= 2.0 ** 5                 # one block scaled by a power of two
    qb, kb = O.quantize_blocks_e4m3(b, 1)
    np.testing.assert_array_equal(qb, q)       # same codes everywhere
    dk = kb - k
    assert dk[2, 1] == 5 and np.count_nonzero(dk) == 1
    W = rng.standard_normal((256, 256)) * 0.02
    q, k = O.quantize_blocks_e4m3(W, 128)
    W2 = W.copy()
    W2[0, 0] = 100.0                           # a new maximum in block (0, 0) only
    q2, k2 = O.quantize_blocks_e4m3(W2, 128)
    assert k2[0, 0] > k[0, 0] and (k2.ravel()[1:] == k.ravel()[1:]).all()
    np.testing.assert_array_equal(q2[128:], q[128:])
    np.testing.assert_array_equal(q2[:128, 128:], q[:128, 128:])


def test_quantize_blocks_error_bound():
    # dequantized values within half an e4m3 step: 2^-4 relative, 2^(k-10) absolute
    rng = np.random.default_rng(13)
    a = rng.standard_normal((20, 512)) * np.exp(rng.standard_normal((20, 1)) * 3)
    q, k = O.quantize_blocks_e4m3(a, 1)
    s = np.exp2(np.repeat(k, 128, axis=1).astype(np.float64))
    assert (np.abs(q * s - a) <= np.abs(a) * 2.0 ** -4 + s * 2.0 ** -10).all()
    assert (np.abs(q) <= 448).all()


def test_fp8_block_linear_brute_force():
    # pure-Python sums of q_a * 2^k_a(block) * q_w * 2^k_w(block) over every k
    rng = np.random.default_rng(14)
    m, n, K = 2, 256, 256
    a_q = O.e4m3_round(rng.uniform(-448, 448, (m, K)))
    W_q = O.e4m3_round(rng.uniform(-448, 448, (n, K)))
    k_a = rng.integers(-20, 5, (m, K // 128))
    k_w = rng.integers(-20, 5, (n // 128, K // 128))
    y = O.fp8_block_linear(a_q, k_a, W_q, k_w)
    al, Wl = a_q.tolist(), W_q.tolist()
    for r in range(m):
        for c in range(0, n, 37):
            ref = 0.0
            for kk in range(K):
                ref += math.ldexp(al[r][kk], int(k_a[r][kk // 128])) * \
                    math.ldexp(Wl[c][kk], int(k_w[c // 128][kk // 128]))
            assert y[r, c] == pytest.approx(ref, rel=1e-12, abs=1e-300)


def test_fp8_block_linear_reduces_to_row_scales():
    # with one exponent per row (all its blocks alike) the block form is the per-row form
    rng = np.random.default_rng(15)
    a_q = O.e4m3_round(rng.uniform(-448, 448, (3, 256)))
    W_q = O.e4m3_round(rng.uniform(-448, 448, (128, 256)))
    k_a = np.repeat(rng.integers(-9, 3, (3, 1)), 2, axis=1)
    k_w = np.full((1, 2), -11)
    y = O.fp8_block_linear(a_q, k_a, W_q, k_w)
    ref = O.fp8_linear(a_q, np.exp2(k_a[:, 0]).astype(np.float32), W_q,
                       np.full(128, 2.0 ** -11, np.float32))
    np.testing.assert_allclose(y, ref, rtol=1e-13)


def test_swiglu_fp8_blocks_equals_dequantized_operands():
    # the block form written out: quantize x per 1x128 block, dequantize both operands,
    # two plain products, SwiGLU, bf16 h, h quantized per 1x128 block, third product
    rng = np.random.default_rng(16)
    H, Iw, m = 256, 128, 3
    rows = O.bf16_round(rng.standard_normal((m, H)))
    W13q, k13 = O.quantize_blocks_e4m3(rng.standard_normal((2 * Iw, H)) * 0.05, 128)
    W2q, k2 = O.quantize_blocks_e4m3(rng.standard_normal((H, Iw)) * 0.05, 128)
    y8 = O.swiglu_ffn_fp8_blocks(rows, W13q, k13, W2q, k2)
    xq, kx = O.quantize_blocks_e4m3(rows, 1)
    xd = xq * np.exp2(np.repeat(kx, 128, axis=1))
    W13d = W13q * np.exp2(np.repeat(np.repeat(k13, 128, axis=0), 128, axis=1))
    W2d = W2q * np.exp2(np.repeat(np.repeat(k2, 128, axis=0), 128, axis=1))
    g, u = xd @ W13d[:Iw].T, xd @ W13d[Iw:].T
    h = O.bf16_round(g / (1 + np.exp(-g)) * u)
    hq, kh = O.quantize_blocks_e4m3(h, 1)
    y = (hq * np.exp2(np.repeat(kh, 128, axis=1))) @ W2d.T
    np.testing.assert_allclose(y8, y, rtol=1e-12, atol=1e-14)
    # and close to the unquantized expert (e4m3 keeps ~2^-4 relative per operand)
    ref = O.swiglu_ffn(rows, W13q * np.exp2(np.repeat(np.repeat(k13, 128, 0), 128, 1)), W2d)
    assert np.abs(y8 - ref).max() < 0.15 * np.abs(ref).max()


def test_layer_tokens_fp8_blocks_hook_matches_per_expert_calls():
    rng = np.random.default_rng(17)
    cfg = O.LayerConfig(T=5, H=128, E=3, k=2, I=128, gate=O.GATE_SOFTMAX)
    x = O.bf16_round(rng.standard_normal((5, 128)))
    Wr = rng.standard_normal((3, 128)).astype(np.float32) * 0.1
    W13 = [O.quantize_blocks_e4m3(rng.standard_normal((256, 128)) * 0.05, 128) for _ in range(3)]
    W2 = [O.quantize_blocks_e4m3(rng.standard_normal((128, 128)) * 0.05, 128) for _ in range(3)]
    get = lambda e: (W13[e][0], W13[e][1], W2[e][0], W2[e][1])
    out, idx, w = O.layer_forward_tokens(x, Wr, None, get, cfg, ffn=O.swiglu_ffn_fp8_blocks)
    for t in range(5):
        ref = sum(w[t, j] * O.swiglu_ffn_fp8_blocks(x[t:t + 1], *get(int(idx[t, j])))[0]
                  for j in range(2))
        np.testing.assert_allclose(out[t], ref, rtol=1e-13, atol=1e-15)


def test_rms_normalize_by_hand_and_invariants():
    y = np.array([[3.0, 4.0], [0.0, 0.0], [1e3, -1e3]])
    r = O.rms_normalize(y, eps=0.0 + 1e-30)
    np.testing.assert_allclose(r[0], [3 / math.sqrt(12.5), 4 / math.sqrt(12.5)], rtol=1e-15)
    np.testing.assert_array_equal(O.rms_normalize(y[1:2]), [[0.0, 0.0]])
    np.testing.assert_allclose(r[2], [1.0, -1.0], rtol=1e-15)
    rng = np.random.default_rng(3)
    z = rng.standard_normal((7, 64)) * 5
    n = O.rms_normalize(z, eps=0.0)
    np.testing.assert_allclose(np.mean(n * n, axis=1), 1.0, rtol=1e-13)
    np.testing.assert_allclose(O.rms_normalize(3.5 * z, eps=0.0), n, rtol=1e-13)


def test_stack_forward_chains_layers():
    # one layer = layer_forward; two layers = layer_forward on the bf16 (normalized) output
    rng = np.random.default_rng(8)
    cfg = O.LayerConfig(T=5, H=32, E=4, k=2, I=16, gate=O.GATE_SOFTMAX)
    x = O.bf16_round(rng.standard_normal((5, 32)))
    mk = lambda: dict(Wr=rng.standard_normal((4, 32)).astype(np.float32) * 0.1, bias=None,
                      W13=O.bf16_round(rng.standard_normal((4, 32, 32)) * 0.1),
                      W2=O.bf16_round(rng.standard_normal((4, 32, 16)) * 0.1))
    l0, l1 = mk(), mk()
    y0, _ = O.layer_forward(x, l0["Wr"], None, l0["W13"], l0["W2"], cfg)
    np.testing.assert_array_equal(O.stack_forward(x, [l0], cfg), y0)
    for norm in (False, True):
        h = O.bf16_round(y0)
        if norm:
            h = O.bf16_round(h / np.sqrt(np.mean(h * h, axis=1, keepdims=True) + 1e-6))
        y1, _ = O.layer_forward(h, l1["Wr"], None, l1["W13"], l1["W2"], cfg)
        np.testing.assert_array_equal(O.stack_forward(x, [l0, l1], cfg, norm=norm), y1)
