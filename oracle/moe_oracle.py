"""CPU oracle for the DeepSeek-V3 MoE layer forward (test infrastructure only).

This module is the slow, obviously-correct statement of what the GPU path
computes. Only the test-suite, the smoke check and the CPU-baseline leg of the
benchmark may import it; the product library never calls it and shares no code
with it. Every array here is numpy; floating-point work is fp64 unless a step
states otherwise.

What the layer computes (the paper's DeepSeek-V3 MoE workload, Appendix
"Workload Details" and the host MoE listing of Appendix "Static Analysis
Example"): route each token to k experts, dispatch (pack) the tokens into
per-expert contiguous buffers, run GEMM1 (gate/up projection, H x 2I), SwiGLU,
GEMM2 (down projection, I x H) per expert, then combine the expert outputs back
into token order with the gate weights. The single-GPU form replaces both
AlltoAll exchanges by on-device permutations (the paper's variable-size
per-peer transfers become unpadded per-expert segments). The routing rule is
not restated by the paper; it follows the DeepSeek-V3 layer the paper names:

* sigmoid gating: s = sigmoid(L); a learned bias b is added for *selection
  only* (s' = s + b); experts are split into G contiguous groups, a group's
  score is the sum of its two largest s'; the top K_g groups are kept; the
  top-k experts by s' among kept groups are selected; the weights are the
  unbiased s of the selected experts, normalised to sum 1 and scaled by
  `route_scale`.
* softmax gating (the tiny configuration): p = softmax(L) over all experts;
  the top-k by p are selected; weights are p (not renormalised) times
  `route_scale`.

Readings taken where the paper is silent:
* Decisions (which experts, which groups) are taken on fp32 scores: the
  selection score is fp32(sigmoid(L)) + fp32 bias (one fp32 add); the group
  score is the fp32 sum of the two largest selection scores.
* Ties are broken by lower index (experts and groups). Output slot j = 0..k-1
  lists the selected experts in descending selection score.
* The SwiGLU activation h = silu(g) * u is rounded to bf16 (round to nearest
  even) before GEMM2, because GEMM2 consumes bf16 operands.
* W13 of one expert is [2I, H]: rows 0..I-1 are the gate projection, rows
  I..2I-1 the up projection; W2 is [H, I]. Both are row-major with the
  reduction dimension contiguous.

Parity status: the paper prints no numeric example for the MoE layer, so each
function is pinned by closed forms, invariants and brute force in
tests/test_oracle.py; the absolute values of the full layer are
"parity unpinned" against the paper itself.
"""

from __future__ import annotations

from dataclasses import dataclass

import numpy as np

GATE_SOFTMAX = 0
GATE_SIGMOID = 1


@dataclass(frozen=True)
class LayerConfig:
    """Shapes and routing knobs of one MoE layer.

    T tokens, H hidden, E routed experts, k experts per token, I expert
    intermediate size, I_shared the shared expert's intermediate size (0 = no
    shared expert), n_groups expert groups, topk_groups groups kept, gate
    GATE_SOFTMAX or GATE_SIGMOID, normalize (1 = weights renormalised to sum 1
    before scaling), route_scale the final weight scale.
    """

    T: int
    H: int
    E: int
    k: int
    I: int
    I_shared: int = 0
    n_groups: int = 1
    topk_groups: int = 1
    gate: int = GATE_SIGMOID
    normalize: int = 1
    route_scale: float = 1.0


# ---------------------------------------------------------------------------
# number formats
# ---------------------------------------------------------------------------

def bf16_round(a) -> np.ndarray:
    """Round real values to the nearest bfloat16 value, ties to even.

    bfloat16 keeps 8 significant bits (1 implicit + 7 stored). Writing
    a = m * 2**e with 0.5 <= |m| < 1, the nearest bf16 is rint(m * 2**8) *
    2**(e - 8), where rint rounds half to even. Exact for every finite fp64
    input in the normal bf16 range (the only range the layer produces).
    """
    a = np.asarray(a, dtype=np.float64)
    m, e = np.frexp(a)
    return np.ldexp(np.rint(m * 256.0), e - 8)


def sigmoid(x) -> np.ndarray:
    """Logistic function 1 / (1 + exp(-x)) in fp64."""
    x = np.asarray(x, dtype=np.float64)
    return 1.0 / (1.0 + np.exp(-x))


def silu(x) -> np.ndarray:
    """SiLU (swish) x * sigmoid(x) = x / (1 + exp(-x)) in fp64."""
    x = np.asarray(x, dtype=np.float64)
    return x / (1.0 + np.exp(-x))


# ---------------------------------------------------------------------------
# step 1: router logits
# ---------------------------------------------------------------------------

def router_logits(x, Wr) -> np.ndarray:
    """L[t, e] = sum_h x[t, h] * Wr[e, h], accumulated in fp64, rounded once to fp32.

    x: [T, H] (bf16 values held in any float dtype); Wr: [E, H] fp32.
    Returns fp32 [T, E], the precision the routing decisions are taken in.
    """
    x = np.asarray(x, dtype=np.float64)
    Wr = np.asarray(Wr, dtype=np.float64)
    return (x @ Wr.T).astype(np.float32)


# ---------------------------------------------------------------------------
# step 2: gating and group-limited top-k
# ---------------------------------------------------------------------------

def gate_scores(L32, cfg: LayerConfig):
    """Per-expert gate scores from fp32 logits.

    Returns (score64, score32): the exact score in fp64 (used for weights) and
    the same score rounded to fp32 (used for decisions).
    sigmoid gating: score = sigmoid(L). softmax gating: score = exp(L - max) /
    sum(exp(L - max)) over all E experts of the token.
    """
    L = np.asarray(L32, dtype=np.float64)
    if cfg.gate == GATE_SIGMOID:
        s = sigmoid(L)
    elif cfg.gate == GATE_SOFTMAX:
        z = np.exp(L - L.max(axis=1, keepdims=True))
        s = z / z.sum(axis=1, keepdims=True)
    else:
        raise ValueError("unknown gate")
    return s, s.astype(np.float32)


def selection_scores(L32, bias32, cfg: LayerConfig) -> np.ndarray:
    """fp32 selection score s' = fp32(score) + bias (a single fp32 add); bias None = 0."""
    _, s32 = gate_scores(L32, cfg)
    if bias32 is None:
        return s32
    return (s32 + np.asarray(bias32, dtype=np.float32)[None, :]).astype(np.float32)


def _order_desc(values, axis=-1) -> np.ndarray:
    """Indices that sort `values` descending, ties by lower index (stable)."""
    return np.argsort(-np.asarray(values), axis=axis, kind="stable")


def group_scores(sel32, cfg: LayerConfig) -> np.ndarray:
    """Group score: fp32 sum of the two largest selection scores in each group.

    Groups are contiguous: group g holds experts [g*E/G, (g+1)*E/G). A group of
    one expert scores that expert's selection score.
    """
    T, E = sel32.shape
    G = cfg.n_groups
    gs = E // G
    grouped = sel32.reshape(T, G, gs)
    srt = -np.sort(-grouped, axis=2)            # descending within each group
    if gs == 1:
        return srt[:, :, 0].astype(np.float32)
    return (srt[:, :, 0] + srt[:, :, 1]).astype(np.float32)  # fp32 + fp32


def kept_expert_mask(sel32, cfg: LayerConfig) -> np.ndarray:
    """Boolean [T, E]: experts whose group is among the top `topk_groups` groups."""
    T, E = sel32.shape
    G = cfg.n_groups
    if G <= 1 or cfg.topk_groups >= G:
        return np.ones((T, E), dtype=bool)
    gsc = group_scores(sel32, cfg)
    order = _order_desc(gsc, axis=1)[:, : cfg.topk_groups]
    keep_g = np.zeros((T, G), dtype=bool)
    np.put_along_axis(keep_g, order, True, axis=1)
    return np.repeat(keep_g, E // G, axis=1)


def gate_topk(L32, bias32, cfg: LayerConfig):
    """Route each token: returns (idx [T,k] int32, w [T,k] fp64).

    Selection on fp32 s' restricted to kept groups, descending, ties by lower
    expert index. Weights from the unbiased fp64 score of the chosen experts:
    normalised to sum 1 when cfg.normalize, then multiplied by route_scale.
    """
    L32 = np.asarray(L32, dtype=np.float32)
    s64, _ = gate_scores(L32, cfg)
    sel = selection_scores(L32, bias32, cfg)
    keep = kept_expert_mask(sel, cfg)
    masked = np.where(keep, sel.astype(np.float64), -np.inf)
    idx = _order_desc(masked, axis=1)[:, : cfg.k].astype(np.int32)
    w = np.take_along_axis(s64, idx, axis=1)
    if cfg.normalize:
        w = w / w.sum(axis=1, keepdims=True)
    w = w * cfg.route_scale
    return idx, w


def routing_margins(L32, bias32, cfg: LayerConfig) -> np.ndarray:
    """Per-token decision margin (fp64 view of the fp32 scores).

    min over: (k-th minus (k+1)-th selection score among kept experts) and
    (topk_groups-th minus (topk_groups+1)-th group score). A large margin means
    every routing decision of the token survives fp32 rounding differences.
    """
    sel = selection_scores(L32, bias32, cfg).astype(np.float64)
    keep = kept_expert_mask(sel.astype(np.float32), cfg)
    masked = np.where(keep, sel, -np.inf)
    srt = -np.sort(-masked, axis=1)
    T = sel.shape[0]
    m = np.full(T, np.inf)
    if srt.shape[1] > cfg.k:
        nxt = srt[:, cfg.k]
        gap = np.where(np.isfinite(nxt), srt[:, cfg.k - 1] - nxt, np.inf)
        m = np.minimum(m, gap)
    G = cfg.n_groups
    if 1 < G and cfg.topk_groups < G:
        gsc = -np.sort(-group_scores(sel.astype(np.float32), cfg).astype(np.float64), axis=1)
        m = np.minimum(m, gsc[:, cfg.topk_groups - 1] - gsc[:, cfg.topk_groups])
    return m


# ---------------------------------------------------------------------------
# step 3: histogram, scan and permutation (the on-device "AlltoAll")
# ---------------------------------------------------------------------------

def permutation(idx, E: int):
    """Stable expert-major permutation of the T*k (token, slot) entries.

    counts[e] = number of entries routed to e; offsets = exclusive prefix sum
    (length E+1); the rows of expert e are its entries ordered by (t, j);
    row_src_token[r] = token of row r; slot_row[t*k + j] = row of entry (t, j).
    """
    idx = np.asarray(idx)
    T, k = idx.shape
    flat = idx.reshape(-1).astype(np.int64)
    counts = np.bincount(flat, minlength=E).astype(np.int32)
    offsets = np.zeros(E + 1, dtype=np.int32)
    offsets[1:] = np.cumsum(counts)
    order = np.argsort(flat, kind="stable")     # entries sorted by expert, then t*k+j
    row_src_token = (order // k).astype(np.int32)
    slot_row = np.empty(T * k, dtype=np.int32)
    slot_row[order] = np.arange(T * k, dtype=np.int32)
    return counts, offsets, row_src_token, slot_row


def dispatch(x, row_src_token) -> np.ndarray:
    """x_perm[r] = x[row_src_token[r]] (a pure copy)."""
    return np.asarray(x)[np.asarray(row_src_token)]


# ---------------------------------------------------------------------------
# steps 4-5: expert FFN (GEMM1 + SwiGLU + GEMM2) and the shared expert
# ---------------------------------------------------------------------------

def swiglu_ffn(rows, W13_e, W2_e) -> np.ndarray:
    """One SwiGLU expert on a block of rows, fp64 accumulation.

    rows [m, H]; W13_e [2I, H] (gate rows then up rows); W2_e [H, I].
    g = rows . Wg^T, u = rows . Wu^T, h = bf16(silu(g) * u), y = h . W2^T.
    """
    rows = np.asarray(rows, dtype=np.float64)
    W13_e = np.asarray(W13_e, dtype=np.float64)
    W2_e = np.asarray(W2_e, dtype=np.float64)
    I = W13_e.shape[0] // 2
    g = rows @ W13_e[:I].T
    u = rows @ W13_e[I:].T
    h = bf16_round(silu(g) * u)
    return h @ W2_e.T


def expert_ffn(x_perm, offsets, W13, W2) -> np.ndarray:
    """Grouped expert FFN: y_perm[r] = FFN_e(x_perm[r]) for r in expert e's segment."""
    x_perm = np.asarray(x_perm, dtype=np.float64)
    H = W2[0].shape[0] if len(W2) else x_perm.shape[1]
    y = np.zeros((x_perm.shape[0], H), dtype=np.float64)
    E = len(offsets) - 1
    for e in range(E):
        a, b = int(offsets[e]), int(offsets[e + 1])
        if b > a:
            y[a:b] = swiglu_ffn(x_perm[a:b], W13[e], W2[e])
    return y


# ---------------------------------------------------------------------------
# step 6: combine (the reverse "AlltoAll")
# ---------------------------------------------------------------------------

def combine(y_perm, slot_row, w, shared=None) -> np.ndarray:
    """out[t] = sum_j w[t, j] * y_perm[slot_row[t*k + j]] (+ shared[t]), fp64."""
    w = np.asarray(w, dtype=np.float64)
    T, k = w.shape
    y = np.asarray(y_perm, dtype=np.float64)
    rows = np.asarray(slot_row).reshape(T, k)
    out = np.zeros((T, y.shape[1]), dtype=np.float64)
    for j in range(k):
        out += w[:, j : j + 1] * y[rows[:, j]]
    if shared is not None:
        out += np.asarray(shared, dtype=np.float64)
    return out


# ---------------------------------------------------------------------------
# FP8 expert compute (the paper quantizes tokens before the dispatch and
# dequantizes before GEMM1: int8 in its host listing, "FP8 quantize" in its
# Section 4.3 table). Reading: OCP e4m3 ("E4M3FN": 4 exponent bits, 3 mantissa
# bits, bias 7, largest finite 448, subnormals down to 2^-9), round to nearest
# even, saturating; one fp32 scale per row s = amax / 448 (fp32 division), the
# quantized value e4m3(v / s) with v / s an fp32 division. Per token for x,
# per packed row for h, per output row for the weights. Quantized products
# are exact, the sums are fp64 here; the two row scales multiply the sum.
# ---------------------------------------------------------------------------

E4M3_MAX = 448.0


def e4m3_round(a) -> np.ndarray:
    """Nearest e4m3 value (ties to even), saturating at +-448.

    Normal e4m3 numbers in [2^e, 2^(e+1)) (e = -6..8) are spaced 2^(e-3);
    below 2^-6 the subnormals are spaced 2^-9.
    """
    a = np.asarray(a, dtype=np.float64)
    mag = np.abs(a)
    e = np.floor(np.log2(np.where(mag > 0, mag, 1.0)))
    e = np.clip(e, -6, 8)
    q = np.ldexp(1.0, (e - 3).astype(np.int64))
    r = np.rint(mag / q) * q
    r = np.minimum(r, E4M3_MAX)
    return np.where(mag > 0, np.sign(a) * r, 0.0)


def _e4m3_table() -> np.ndarray:
    """Value of each of the 256 e4m3 bytes (fp64): bit 7 sign, bits 6-3 exponent
    field E, bits 2-0 mantissa field M; E = 0 gives the subnormal M / 8 * 2^-6,
    otherwise (1 + M / 8) * 2^(E - 7); E = 15 with M = 7 is NaN (no infinities)."""
    c = np.arange(256, dtype=np.int64)
    sign = np.where(c & 0x80, -1.0, 1.0)
    E = (c >> 3) & 0xF
    M = c & 0x7
    mag = np.where(E == 0, M / 8.0 * 2.0 ** -6, (1.0 + M / 8.0) * np.exp2(E - 7.0))
    mag = np.where((E == 15) & (M == 7), np.nan, mag)
    return sign * mag


E4M3_VALUES = _e4m3_table()


def e4m3_decode(codes) -> np.ndarray:
    """Values (fp64) of e4m3 bytes: a lookup in the 256-entry table above."""
    return E4M3_VALUES[np.asarray(codes, dtype=np.uint8)]


def quantize_rows_e4m3(a):
    """Per-row e4m3 quantization: returns (q fp64 values on the e4m3 grid, scale fp32 [rows]).

    s = fp32(amax / 448) (1 for an all-zero row); q = e4m3(fp32(v / s)).
    """
    a32 = np.asarray(a, dtype=np.float32)
    amax = np.abs(a32).max(axis=1)
    s = np.where(amax > 0, (amax / np.float32(E4M3_MAX)).astype(np.float32), np.float32(1.0))
    s = s.astype(np.float32)
    v = (a32 / s[:, None]).astype(np.float32)
    return e4m3_round(v), s


def fp8_linear(a_q, s_a, W_q, s_w) -> np.ndarray:
    """Dequantized product of e4m3 operands: (a_q . W_q^T) * s_a[r] * s_w[c] (fp64).

    a_q [m, K], W_q [n, K] on the e4m3 grid; s_a [m], s_w [n] fp32 row scales.
    """
    acc = np.asarray(a_q, dtype=np.float64) @ np.asarray(W_q, dtype=np.float64).T
    return acc * np.asarray(s_a, dtype=np.float64)[:, None] * \
        np.asarray(s_w, dtype=np.float64)[None, :]


def swiglu_h_fp8(rows, W13_q, s13) -> np.ndarray:
    """GEMM1 + SwiGLU of the FP8 form: h = bf16(silu(g) * u), with g | u the
    dequantized product of the per-row quantized rows and W13_q (scales s13)."""
    I = W13_q.shape[0] // 2
    xq, sx = quantize_rows_e4m3(np.asarray(rows, dtype=np.float64))
    gu = fp8_linear(xq, sx, W13_q, s13)
    g, u = gu[:, :I], gu[:, I:]
    return bf16_round(silu(g) * u)


def swiglu_ffn_fp8(rows, W13_q, s13, W2_q, s2):
    """One SwiGLU expert in the FP8 form.

    rows [m, H] (bf16 values); W13_q [2I, H], W2_q [H, I] e4m3 values with
    per-row fp32 scales s13 [2I], s2 [H]. x is quantized per row; g, u =
    (x_q . W_q^T) * s_x * s_w; h = bf16(silu(g) * u) quantized per row;
    y = (h_q . W2_q^T) * s_h * s_2.
    """
    h = swiglu_h_fp8(rows, W13_q, s13)
    hq, sh = quantize_rows_e4m3(h)
    return fp8_linear(hq, sh, W2_q, s2)


# ---------------------------------------------------------------------------
# FP8 with block scales: DeepSeek-V3's fine-grained form of the quantize step,
# one scale per 1 x 128 block of an activation row (x per token, h per packed
# row) and one per 128 x 128 block of a weight matrix. Reading: the scales are
# powers of two 2^k stored as UE8M0 exponent bytes k + 127 (the block-scale
# format a tensor core applies by itself); a block's k is the smallest integer
# with amax <= 448 * 2^k (k = 0 for an all-zero block), clamped to [-127, 127];
# its values are e4m3(v * 2^-k), an exact scaling then one rounding to nearest
# even, saturating. A product sums, block by block, q_a * q_w * 2^(k_a + k_w).
# ---------------------------------------------------------------------------

FP8_BLOCK = 128


def block_exponent(amax) -> np.ndarray:
    """k = min{integer k : amax <= 448 * 2^k} (0 where amax == 0), clamped to [-127, 127]."""
    amax = np.asarray(amax, dtype=np.float64)
    safe = np.where(amax > 0, amax, E4M3_MAX)
    k = np.ceil(np.log2(safe / E4M3_MAX))
    # settle the rounding of log2 against the definition (448 * 2^k is exact)
    k = np.where(safe > E4M3_MAX * np.exp2(k), k + 1, k)
    k = np.where(safe <= E4M3_MAX * np.exp2(k - 1), k - 1, k)
    return np.clip(k, -127, 127).astype(np.int64)


def quantize_blocks_e4m3(a, rows_per_block: int):
    """Block e4m3 quantization of a [m, K] matrix in blocks of rows_per_block x 128.

    Returns (q fp64 [m, K] on the e4m3 grid, k int64 [m / rows_per_block, K / 128]).
    rows_per_block = 1 for activations, 128 for weights; m and K must divide.
    """
    a = np.asarray(a, dtype=np.float64)
    m, K = a.shape
    rb, cb = rows_per_block, FP8_BLOCK
    assert m % rb == 0 and K % cb == 0
    amax = np.abs(a).reshape(m // rb, rb, K // cb, cb).max(axis=(1, 3))
    k = block_exponent(amax)
    return e4m3_round(a * block_scales(-k, rb)), k


def block_scales(k, rows_per_block: int) -> np.ndarray:
    """2^k of every element: the block exponents k [m / rb, K / 128] spread over their blocks."""
    k = np.asarray(k, dtype=np.int64)
    return np.exp2(np.repeat(np.repeat(k, rows_per_block, axis=0), FP8_BLOCK, axis=1).astype(np.float64))


def fp8_block_linear(a_q, k_a, W_q, k_w) -> np.ndarray:
    """Product of block-scaled e4m3 operands (fp64): dequantize, then a_deq . W_deq^T.

    a_q [m, K] with 1 x 128 block exponents k_a [m, K/128]; W_q [n, K] with
    128 x 128 block exponents k_w [n/128, K/128].
    """
    a = np.asarray(a_q, dtype=np.float64) * block_scales(k_a, 1)
    W = np.asarray(W_q, dtype=np.float64) * block_scales(k_w, FP8_BLOCK)
    return a @ W.T


def swiglu_h_fp8_blocks(rows, W13_q, k13) -> np.ndarray:
    """GEMM1 + SwiGLU of the block-scaled FP8 form: x quantized per 1 x 128 block,
    g | u = fp8_block_linear(x_q, W13_q), h = bf16(silu(g) * u)."""
    I = W13_q.shape[0] // 2
    xq, kx = quantize_blocks_e4m3(rows, 1)
    gu = fp8_block_linear(xq, kx, W13_q, k13)
    return bf16_round(silu(gu[:, :I]) * gu[:, I:])


def swiglu_ffn_fp8_blocks(rows, W13_q, k13, W2_q, k2):
    """One SwiGLU expert in the block-scaled FP8 form.

    rows [m, H] (bf16 values); W13_q [2I, H], W2_q [H, I] on the e4m3 grid with
    128 x 128 block exponents k13 [2I/128, H/128], k2 [H/128, I/128]. h (bf16)
    is quantized per 1 x 128 block before GEMM2.
    """
    h = swiglu_h_fp8_blocks(rows, W13_q, k13)
    hq, kh = quantize_blocks_e4m3(h, 1)
    return fp8_block_linear(hq, kh, W2_q, k2)


# ---------------------------------------------------------------------------
# the whole layer
# ---------------------------------------------------------------------------

def layer_forward(x, Wr, bias, W13, W2, cfg: LayerConfig, Ws13=None, Ws2=None, logits=None):
    """Full layer forward over all T tokens, in the paper's stage order.

    route -> dispatch -> expert FFN -> combine (+ shared expert). `logits`
    (fp32 [T, E]) may be supplied to route on given logits. Returns (out fp64
    [T, H], aux dict with logits, idx, w, counts, offsets, row_src_token,
    slot_row, y_perm).
    """
    x = np.asarray(x, dtype=np.float64)
    L32 = router_logits(x, Wr) if logits is None else np.asarray(logits, dtype=np.float32)
    idx, w = gate_topk(L32, bias, cfg)
    counts, offsets, rst, slot_row = permutation(idx, cfg.E)
    x_perm = dispatch(x, rst)
    y_perm = expert_ffn(x_perm, offsets, W13, W2)
    shared = None
    if cfg.I_shared and Ws13 is not None:
        shared = swiglu_ffn(x, Ws13, Ws2)
    out = combine(y_perm, slot_row, w, shared)
    aux = dict(logits=L32, idx=idx, w=w, counts=counts, offsets=offsets,
               row_src_token=rst, slot_row=slot_row, y_perm=y_perm, shared=shared)
    return out, aux


def rms_normalize(y, eps: float = 1e-6) -> np.ndarray:
    """Per-row RMS normalization y / sqrt(mean(y^2) + eps) (fp64), the unit-gain
    form of the RMSNorm a DeepSeek-V3 block applies in front of its MoE."""
    y = np.asarray(y, dtype=np.float64)
    return y / np.sqrt(np.mean(y * y, axis=1, keepdims=True) + eps)


def stack_forward(x, layers, cfg: LayerConfig, norm: bool = True):
    """Consecutive layers (the paper's multi-layer study, Section 4.3): layer l + 1
    reads layer l's output rounded to bf16 (then, with norm, RMS-normalized and
    rounded to bf16 again); returns the last layer's fp64 output.
    layers: a list of dicts with Wr, bias, W13, W2, Ws13, Ws2."""
    h = np.asarray(x, dtype=np.float64)
    out = None
    for n, w in enumerate(layers):
        if n > 0:
            h = bf16_round(out)
            if norm:
                h = bf16_round(rms_normalize(h))
        out, _ = layer_forward(h, w["Wr"], w["bias"], w["W13"], w["W2"], cfg, w.get("Ws13"),
                               w.get("Ws2"))
    return out


def layer_forward_tokens(x_rows, Wr, bias, get_expert, cfg: LayerConfig, get_shared=None,
                         ffn=swiglu_ffn):
    """Layer output for a sample of tokens, one token at a time.

    Routing is independent per token, so a token's output needs only its own
    row. x_rows [n, H]; get_expert(e) -> the expert's weight arguments of
    `ffn` after the rows ((W13_e, W2_e) for swiglu_ffn; (W13_q, s13, W2_q, s2)
    for swiglu_ffn_fp8); get_shared() -> the shared expert's, or None.
    Experts are visited once each, with all sampled rows routed to them.
    Returns (out fp64 [n, H], idx [n, k], w [n, k]).
    """
    x_rows = np.asarray(x_rows, dtype=np.float64)
    L32 = router_logits(x_rows, Wr)
    idx, w = gate_topk(L32, bias, cfg)
    n = x_rows.shape[0]
    out = np.zeros((n, cfg.H), dtype=np.float64)
    for e in np.unique(idx):
        who, slot = np.nonzero(idx == e)
        y = ffn(x_rows[who], *get_expert(int(e)))
        out[who] += w[who, slot][:, None] * y
    if get_shared is not None and cfg.I_shared:
        out += ffn(x_rows, *get_shared())
    return out, idx, w
