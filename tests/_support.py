"""Helpers shared by the GPU parity tests (inputs, oracle glue, tolerances)."""

from __future__ import annotations

import numpy as np
import torch

from oracle import moe_oracle as O
from paper_2603_02376_gb300 import inputs as I

U32 = 2.0 ** -24   # fp32 unit roundoff
UBF16 = 2.0 ** -8  # bf16 unit roundoff (8 significant bits)


def f64(t) -> np.ndarray:
    return t.detach().to(torch.float64).cpu().numpy()


def oracle_cfg(wl, T=None) -> O.LayerConfig:
    return O.LayerConfig(T=wl.T if T is None else T, H=wl.H, E=wl.E, k=wl.k, I=wl.I,
                         I_shared=wl.I_shared, n_groups=wl.n_groups, topk_groups=wl.topk_groups,
                         gate=wl.gate, normalize=wl.normalize, route_scale=wl.route_scale)


def bias32(b):
    return None if b is None else b.detach().cpu().numpy().astype(np.float32)


def prepare_routing(wl, d, seed=0, min_margin=1e-3):
    """Make the workload's routing well-posed on the oracle's side.

    Calibrates the bias for the balanced / Zipf workloads with the oracle
    gate, then redraws token rows whose decision margin is <= min_margin.
    Mutates d["x"] (device) and d["bias"]; returns a dict of realised stats.
    """
    cfg = oracle_cfg(wl)
    Wr = f64(d["Wr"])
    xh = f64(d["x"])
    L = O.router_logits(xh, Wr)

    def counts_of(b):
        idx, _ = O.gate_topk(L, b.numpy().astype(np.float32), cfg)
        return np.bincount(idx.reshape(-1), minlength=wl.E)

    stats = {}
    mean = wl.T * wl.k / wl.E
    rounds = 0
    # Calibrating the bias moves margins and redrawing rows moves loads: alternate
    # until both hold (the Zipf workload only needs its hot ratio, not a band).
    for outer in range(12):
        if wl.balance == "balanced":
            b, c = I.calibrate_balanced(counts_of, wl, d["bias"].cpu(),
                                        gamma=2e-3 if outer == 0 else 3e-4)
            d["bias"] = b.to(d["x"].device)
        elif wl.balance == "zipf" and outer == 0:
            b, c = I.calibrate_zipf(counts_of, wl, seed)
            d["bias"] = b.to(d["x"].device)
        b32 = bias32(d["bias"])
        for attempt in range(64):
            m = O.routing_margins(L, b32, cfg)
            bad = np.nonzero(m <= min_margin)[0]
            if bad.size == 0:
                break
            I.resample_rows(d["x"], bad.tolist(), seed, 1000 * outer + attempt)
            L[bad] = O.router_logits(f64(d["x"][torch.as_tensor(bad, device=d["x"].device)]), Wr)
            rounds += 1
        else:
            raise RuntimeError("margin resampling did not converge")
        idx, _ = O.gate_topk(L, b32, cfg)
        cnt = np.bincount(idx.reshape(-1), minlength=wl.E)
        # redrawing low-margin rows after balancing costs about 1-2 % of load spread
        if wl.balance != "balanced" or np.abs(cnt / mean - 1).max() <= wl.balance_tol + 0.02:
            break
    stats.update(resample_rounds=rounds, max_over_mean=float(cnt.max() / mean),
                 min_over_mean=float(cnt.min() / mean), oracle_logits=L)
    return stats


def logits_bound(x, Wr) -> np.ndarray:
    """Worst-case fp32 summation error bound H * u * sum_h |x_h Wr_eh| per logit."""
    S = np.abs(x) @ np.abs(Wr).T
    return x.shape[1] * U32 * S + 1e-30


def assert_layer_close(got, ref, atol=2e-2, rtol=1e-2):
    """The layer tolerance, |got - ref| <= atol + rtol * |ref| elementwise, and
    for an fp32 output (a torch float32 tensor) also max|got - ref| <= atol:
    the strict absolute bound, reachable when no bf16 rounding of the output
    sits between the fp32 accumulation and the comparison. A bf16 output is
    held to the allclose form only (half a bf16 ulp of |y| >= 8 is 0.031 > atol).
    Returns (max|err|, ||err|| / ||ref||)."""
    strict = isinstance(got, torch.Tensor) and got.dtype == torch.float32
    got = f64(got) if isinstance(got, torch.Tensor) else np.asarray(got, dtype=np.float64)
    err = np.abs(got - ref)
    lim = atol + rtol * np.abs(ref)
    bad = err > lim
    rel = np.linalg.norm(got - ref) / max(np.linalg.norm(ref), 1e-30)
    what = "fp32 output" if strict else "output"
    assert not bad.any(), (f"{what}: {bad.sum()} of {bad.size} elements out of tolerance; "
                           f"max|err| {err.max():.3e}, rel-fro {rel:.3e}")
    if strict:
        assert err.max() <= atol, (f"fp32 output: max|err| {err.max():.3e} > {atol} absolute; "
                                   f"rel-fro {rel:.3e}")
    return float(err.max()), float(rel)
