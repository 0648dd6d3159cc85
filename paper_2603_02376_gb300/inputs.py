"""Seeded synthetic inputs for the MoE layer workloads.

This module only draws random numbers and lays them out; it holds none of the
layer's arithmetic, so both the CUDA path and the CPU oracle can be fed from it
without sharing any computation. Routing-dependent adjustments (balancing the
per-expert load, Zipf-skewing it, resampling tokens whose routing decision is
within a margin) take the router as a callable supplied by the caller.

Workloads (DeepSeek-V3-shaped, the layer of the paper's MoE workload: GEMM1
7168 x 4096 and GEMM2 2048 x 7168, Appendix "Workload Details"):

* tiny:    T=64, H=256, E=8, k=2, I=128, softmax gating, no shared expert.
* decode:  T=128, H=7168, E=256 (+1 shared, I=I_s=2048), sigmoid gating with
           bias, 8 groups / 4 kept, top-8, normalised weights x 2.5.
* prefill: T=4096, same layer, per-expert load within +-10 % of the mean.
* skewed:  T=8192, same layer, bias drawn so expert popularity follows a
           Zipf(1.2) ranking calibrated to a hottest expert ~15x the mean load.
* dispatch sweep: H=7168, E=256, k=8, uniform random distinct experts per
           token, T in {1024, 4096, 16384, 65536}.

Distributions: activations N(0, 1) bf16; expert and shared weights
N(0, 0.02^2) bf16; router weights N(0, 0.01^2) fp32; bias N(0, 0.01^2) fp32.
Each tensor draws from its own torch.Generator seeded from (seed, tensor id).
"""

from __future__ import annotations

import math
from dataclasses import dataclass, replace

import torch

GATE_SOFTMAX = 0
GATE_SIGMOID = 1


@dataclass(frozen=True)
class Workload:
    """Shape and routing knobs of a workload, plus how its inputs are drawn."""

    name: str
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
    has_bias: bool = True
    balance: str = "none"          # "none" | "balanced" | "zipf"
    zipf_s: float = 1.2
    zipf_hot_ratio: float = 15.0
    balance_tol: float = 0.10


TINY = Workload("tiny T=64 H=256 E=8 k=2 I=128 softmax", T=64, H=256, E=8, k=2, I=128,
                I_shared=0, n_groups=1, topk_groups=1, gate=GATE_SOFTMAX, normalize=0,
                route_scale=1.0, has_bias=False)
DECODE = Workload("deepseek-v3 decode T=128 H=7168 E=256+1 k=8 I=2048", T=128, H=7168, E=256,
                  k=8, I=2048, I_shared=2048, n_groups=8, topk_groups=4, gate=GATE_SIGMOID,
                  normalize=1, route_scale=2.5, has_bias=True)
PREFILL = replace(DECODE, name="deepseek-v3 prefill T=4096 balanced", T=4096, balance="balanced")
SKEWED = replace(DECODE, name="deepseek-v3 skewed prefill T=8192 zipf1.2", T=8192, balance="zipf")
# The decode shape with 32 experts (4 per group), 2.8 GB of weights: small enough
# for multi-pass profiler captures, still far larger than L2.
DECODE_E32 = replace(DECODE, name="deepseek-v3 decode shape, 32 experts, T=16", T=16, E=32)
# The prefill shape (128 rows per expert) with 32 experts, for profiler captures.
PREFILL_E32 = replace(PREFILL, name="deepseek-v3 prefill shape, 32 experts, T=512", T=512, E=32)
# The skewed (Zipf) batch with 32 experts: ~512 rows per expert in 256-row
# token tiles, hot experts over several tiles, for profiler captures.
SKEWED_E32 = replace(SKEWED, name="deepseek-v3 skewed shape, 32 experts, T=2048", T=2048, E=32)
WORKLOADS = {"tiny": TINY, "decode": DECODE, "prefill": PREFILL, "skewed": SKEWED,
             "decode_e32": DECODE_E32, "prefill_e32": PREFILL_E32, "skewed_e32": SKEWED_E32}
DISPATCH_SWEEP_T = (1024, 4096, 16384, 65536)

_SUB = {"x": 1, "Wr": 2, "bias": 3, "W13": 4, "W2": 5, "Ws13": 6, "Ws2": 7,
        "resample": 8, "zipf": 9, "sample": 10, "route": 11, "W13q": 12, "W2q": 13,
        "Ws13q": 14, "Ws2q": 15, "W13b": 16, "W2b": 17, "Ws13b": 18, "Ws2b": 19}


def generator(seed: int, what: str, device, extra: int = 0) -> torch.Generator:
    """A torch.Generator for one tensor: seeded from (seed, tensor id, extra)."""
    g = torch.Generator(device=device)
    g.manual_seed(int(seed) * 1_000_003 + _SUB[what] * 10_007 + int(extra))
    return g


def randn(shape, std, dtype, seed, what, device, extra=0):
    """N(0, std^2) samples drawn in fp32 and rounded once to `dtype`."""
    g = generator(seed, what, device, extra)
    t = torch.randn(shape, generator=g, device=device, dtype=torch.float32)
    if std != 1.0:
        t.mul_(std)
    return t.to(dtype)


def expert_weights(wl: Workload, seed: int, device, experts=None):
    """Routed-expert weights W13 [E, 2I, H] and W2 [E, H, I], bf16.

    Drawn expert by expert (one generator per expert and matrix) so any
    subset can be regenerated alone; `experts` restricts to a list.
    """
    es = range(wl.E) if experts is None else experts
    W13 = torch.empty((len(es), 2 * wl.I, wl.H), dtype=torch.bfloat16, device=device)
    W2 = torch.empty((len(es), wl.H, wl.I), dtype=torch.bfloat16, device=device)
    for n, e in enumerate(es):
        W13[n] = randn((2 * wl.I, wl.H), 0.02, torch.bfloat16, seed, "W13", device, extra=e)
        W2[n] = randn((wl.H, wl.I), 0.02, torch.bfloat16, seed, "W2", device, extra=e)
    return W13, W2


# FP8 expert weights are drawn in their stored form: e4m3 bytes plus one fp32
# scale per row, as an FP8 checkpoint holds them. Bytes: a random sign and a
# magnitude code uniform over 0x30..0x7E (values 0.5 .. 448, ten binades, no
# NaN code); row scales 2^-14 * U[1, 2), so the weights span about +-0.05 like
# the N(0, 0.02^2) bf16 ones.
E4M3_CODE_LO, E4M3_CODE_HI = 0x30, 0x7E


def e4m3_codes(shape, seed, what, device, extra=0):
    """(uint8 e4m3 bytes of `shape`, fp32 scales [prod(shape[:-1])]) for one weight matrix."""
    g = generator(seed, what, device, extra)
    mag = torch.randint(E4M3_CODE_LO, E4M3_CODE_HI + 1, shape, generator=g, device=device,
                        dtype=torch.int32)
    sgn = torch.randint(0, 2, shape, generator=g, device=device, dtype=torch.int32)
    codes = (mag + 128 * sgn).to(torch.uint8)
    rows = codes.numel() // shape[-1]
    scale = (torch.rand(rows, generator=g, device=device, dtype=torch.float32) + 1.0) * 2.0 ** -14
    return codes, scale


def fp8_expert_weights(wl: Workload, seed: int, device, experts=None):
    """FP8 routed-expert weights: W13 bytes [E, 2I, H] with scales [E, 2I], W2 bytes
    [E, H, I] with scales [E, H]; drawn expert by expert like expert_weights."""
    es = range(wl.E) if experts is None else experts
    W13 = torch.empty((len(es), 2 * wl.I, wl.H), dtype=torch.uint8, device=device)
    W2 = torch.empty((len(es), wl.H, wl.I), dtype=torch.uint8, device=device)
    s13 = torch.empty((len(es), 2 * wl.I), dtype=torch.float32, device=device)
    s2 = torch.empty((len(es), wl.H), dtype=torch.float32, device=device)
    for n, e in enumerate(es):
        W13[n], s13[n] = e4m3_codes((2 * wl.I, wl.H), seed, "W13q", device, extra=e)
        W2[n], s2[n] = e4m3_codes((wl.H, wl.I), seed, "W2q", device, extra=e)
    return W13, s13, W2, s2


# Block-scaled FP8 weights in stored form: the same e4m3 bytes, and one UE8M0
# exponent byte per 128 x 128 block (scale 2^(byte - 127)), drawn from
# {127 - 14, 127 - 13}: weights within about +-0.05 again.
def e4m3_block_codes(shape, seed, what, device, extra=0):
    """(uint8 e4m3 bytes of `shape` [rows, cols], uint8 exponents [rows/128, cols/128])."""
    g = generator(seed, what, device, extra)
    rows, cols = shape
    mag = torch.randint(E4M3_CODE_LO, E4M3_CODE_HI + 1, shape, generator=g, device=device,
                        dtype=torch.int32)
    sgn = torch.randint(0, 2, shape, generator=g, device=device, dtype=torch.int32)
    codes = (mag + 128 * sgn).to(torch.uint8)
    exps = torch.randint(127 - 14, 127 - 12, (rows // 128, cols // 128), generator=g,
                         device=device, dtype=torch.int32).to(torch.uint8)
    return codes, exps


def fp8_block_expert_weights(wl: Workload, seed: int, device, experts=None):
    """Block-scaled FP8 routed-expert weights: W13 bytes [E, 2I, H] with exponents
    [E, 2I/128, H/128], W2 bytes [E, H, I] with exponents [E, H/128, I/128]."""
    es = range(wl.E) if experts is None else experts
    W13 = torch.empty((len(es), 2 * wl.I, wl.H), dtype=torch.uint8, device=device)
    W2 = torch.empty((len(es), wl.H, wl.I), dtype=torch.uint8, device=device)
    k13 = torch.empty((len(es), 2 * wl.I // 128, wl.H // 128), dtype=torch.uint8, device=device)
    k2 = torch.empty((len(es), wl.H // 128, wl.I // 128), dtype=torch.uint8, device=device)
    for n, e in enumerate(es):
        W13[n], k13[n] = e4m3_block_codes((2 * wl.I, wl.H), seed, "W13b", device, extra=e)
        W2[n], k2[n] = e4m3_block_codes((wl.H, wl.I), seed, "W2b", device, extra=e)
    return W13, k13, W2, k2


def fp8_block_shared_weights(wl: Workload, seed: int, device):
    """Block-scaled FP8 shared-expert weights (Ws13, its exponents, Ws2, its exponents)."""
    if not wl.I_shared:
        return None, None, None, None
    Ws13, k13 = e4m3_block_codes((2 * wl.I_shared, wl.H), seed, "Ws13b", device)
    Ws2, k2 = e4m3_block_codes((wl.H, wl.I_shared), seed, "Ws2b", device)
    return Ws13, k13, Ws2, k2


def fp8_shared_weights(wl: Workload, seed: int, device):
    """FP8 shared-expert weights (Ws13, Ws13 scales, Ws2, Ws2 scales), or four Nones."""
    if not wl.I_shared:
        return None, None, None, None
    Ws13, ss13 = e4m3_codes((2 * wl.I_shared, wl.H), seed, "Ws13q", device)
    Ws2, ss2 = e4m3_codes((wl.H, wl.I_shared), seed, "Ws2q", device)
    return Ws13, ss13, Ws2, ss2


def layer_inputs(wl: Workload, seed: int = 0, device="cpu", with_experts=True):
    """All tensors of one layer: dict with x, Wr, bias, W13, W2, Ws13, Ws2.

    bias is None without bias; Ws13/Ws2 are None without a shared expert.
    """
    d = {}
    d["x"] = randn((wl.T, wl.H), 1.0, torch.bfloat16, seed, "x", device)
    d["Wr"] = randn((wl.E, wl.H), 0.01, torch.float32, seed, "Wr", device)
    d["bias"] = randn((wl.E,), 0.01, torch.float32, seed, "bias", device) if wl.has_bias else None
    if with_experts:
        d["W13"], d["W2"] = expert_weights(wl, seed, device)
    if wl.I_shared:
        d["Ws13"] = randn((2 * wl.I_shared, wl.H), 0.02, torch.bfloat16, seed, "Ws13", device)
        d["Ws2"] = randn((wl.H, wl.I_shared), 0.02, torch.bfloat16, seed, "Ws2", device)
    else:
        d["Ws13"] = d["Ws2"] = None
    return d


def resample_rows(x: torch.Tensor, rows, seed: int, attempt: int) -> None:
    """Redraw rows of x in place from N(0, 1), one generator per (row, attempt)."""
    for t in list(rows):
        x[int(t)] = randn((x.shape[1],), 1.0, x.dtype, seed, "resample", x.device,
                          extra=int(t) * 997 + int(attempt))


def resample_until_margin(x, margins_fn, seed: int, min_margin: float = 1e-3, max_rounds: int = 64):
    """Redraw rows of x whose routing margin is below `min_margin`.

    margins_fn(x) -> per-token margins (any array-like of length T); it is the
    caller's router. Returns the number of rounds used; raises if rows still
    fail after max_rounds.
    """
    for attempt in range(max_rounds):
        m = torch.as_tensor(margins_fn(x)).reshape(-1)
        bad = torch.nonzero(m <= min_margin).reshape(-1).tolist()
        if not bad:
            return attempt
        resample_rows(x, bad, seed, attempt)
    raise RuntimeError("margin resampling did not converge")


def zipf_ranks(E: int, seed: int) -> torch.Tensor:
    """Popularity rank r_e in 1..E of each expert (a seeded permutation)."""
    g = generator(seed, "zipf", "cpu")
    perm = torch.randperm(E, generator=g)
    r = torch.empty(E, dtype=torch.float64)
    r[perm] = torch.arange(1, E + 1, dtype=torch.float64)
    return r


def zipf_bias(E: int, s: float, beta: float, seed: int) -> torch.Tensor:
    """Selection bias b_e = beta * (-s * ln r_e): a Zipf(s)-shaped preference."""
    r = zipf_ranks(E, seed)
    return (beta * (-s * torch.log(r))).to(torch.float32)


def calibrate_zipf(counts_fn, wl: Workload, seed: int, iters: int = 30):
    """Bisection on beta so that max(count)/mean(count) ~ wl.zipf_hot_ratio.

    counts_fn(bias fp32 [E] cpu) -> per-expert counts of the routed tokens.
    Returns (bias, counts).
    """
    mean = wl.T * wl.k / wl.E
    lo, hi = 0.0, 1.0
    best = None
    for _ in range(iters):
        beta = 0.5 * (lo + hi)
        b = zipf_bias(wl.E, wl.zipf_s, beta, seed)
        c = torch.as_tensor(counts_fn(b)).to(torch.float64)
        ratio = float(c.max()) / mean
        best = (b, c)
        if abs(ratio - wl.zipf_hot_ratio) < 0.25:
            break
        if ratio < wl.zipf_hot_ratio:
            lo = beta
        else:
            hi = beta
    return best


def calibrate_balanced(counts_fn, wl: Workload, bias0: torch.Tensor, iters: int = 400,
                       gamma: float = 2e-3):
    """Sign-step bias updates until every expert's load is within +-tol of the mean.

    counts_fn(bias) -> counts. b_e -= gamma * sign(load_e - mean) with a
    slowly shrinking gamma. Returns (bias, counts).
    """
    mean = wl.T * wl.k / wl.E
    b = bias0.clone().to(torch.float32).cpu()
    c = None
    for it in range(iters):
        c = torch.as_tensor(counts_fn(b)).to(torch.float64)
        dev = (c - mean) / mean
        if float(dev.abs().max()) <= wl.balance_tol:
            return b, c
        b = b - gamma * torch.sign(dev).to(torch.float32)
        if it % 50 == 49:
            gamma *= 0.7
    return b, c


def sample_tokens(T: int, n: int, seed: int) -> torch.Tensor:
    """n distinct token indices drawn uniformly without replacement (sorted)."""
    g = generator(seed, "sample", "cpu")
    n = min(n, T)
    return torch.sort(torch.randperm(T, generator=g)[:n]).values


def uniform_routing(T: int, E: int, k: int, seed: int, device="cpu"):
    """Uniform random routing with k distinct experts per token (dispatch sweep).

    Returns idx [T, k] int32 and w [T, k] fp32 drawn from U(0, 1).
    """
    g = generator(seed, "route", device)
    keys = torch.rand((T, E), generator=g, device=device)
    idx = torch.topk(keys, k, dim=1).indices.to(torch.int32)
    w = torch.rand((T, k), generator=g, device=device)
    return idx, w


def bf16_bytes(*shape) -> int:
    """Bytes of a bf16 tensor of the given shape."""
    return 2 * math.prod(shape)
