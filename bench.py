#!/usr/bin/env python3
"""Benchmark of the DeepSeek-V3 MoE layer forward on GB300.

One step = one full layer forward (router -> gate/top-k -> permutation ->
dispatch -> grouped GEMM1+SwiGLU -> grouped GEMM2 -> shared expert ->
combine) over one batch of synthetic tokens, through the library's C ABI.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--workload skewed]
    python bench.py --impl reference ...     # the CPU oracle, timed on host cores

The default workload is the largest single-GPU configuration: the skewed
(Zipf 1.2, hottest expert ~15x the mean load) DeepSeek-V3 prefill batch of
T=8192 tokens. decode (T=128) and prefill (T=4096, balanced) are flags.

Prints one JSON line (rank 0). With N > 1 (torchrun) every rank runs an
independent replica of the layer on its own tokens (no collective on the data
path); the barrier and max-over-ranks timing use a gloo process group.
"""

from __future__ import annotations

import argparse
import datetime as _dt
import hashlib
import json
import os
import statistics
import subprocess
import sys
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import numpy as np  # noqa: E402
import torch  # noqa: E402

from paper_2603_02376_gb300 import inputs as I  # noqa: E402

METRIC = "MoE layer tokens/sec on 1 GB300; grouped-GEMM % bf16 peak; dispatch/combine % HBM BW"
FALLBACK_HBM_GBS = 6800.0
FALLBACK_BF16_TFLOPS = 1900.0
NOMINAL_HBM_GBS = 8000.0        # GB300 HBM3e, nominal (context beside the measured copy peak)
NOMINAL_BF16_TFLOPS = 2250.0    # GB300 dense bf16, nominal
TRAFFIC_FILE = os.path.join(ROOT, "profiles", "traffic.json")
L2_BYTES = 129 * 1000 * 1000    # GB300 L2
GEMM_SOURCES = ("paper_2603_02376_gb300/csrc/gemm_tc.cu", "paper_2603_02376_gb300/csrc/common.cuh")


def parse():
    p = argparse.ArgumentParser(description=__doc__.splitlines()[0])
    p.add_argument("--gpus", type=int, default=1)
    p.add_argument("--steps", type=int, default=200)
    p.add_argument("--warmup", type=int, default=10)
    p.add_argument("--impl", choices=("ours", "reference"), default="ours")
    p.add_argument("--workload", choices=tuple(I.WORKLOADS), default="skewed")
    p.add_argument("--mode", choices=("seq", "overlap-tokens", "overlap-experts"), default="seq")
    p.add_argument("--chunk-tokens", type=int, default=512)
    p.add_argument("--expert-chunks", type=int, default=8)
    p.add_argument("--dispatch", choices=("auto", "packed", "gather4", "gemm1"), default="auto",
                   help="packed: a dispatch kernel packs x_perm before GEMM1; gather4: for "
                        "decode-sized batches GEMM1's operand loads gather the token rows "
                        "(TMA gather4), no x_perm; gemm1: the dispatch copy runs inside the "
                        "GEMM1 launch (pack warps, hidden behind the shared expert's units); "
                        "auto (default): gemm1 above 24 rows per expert (measured 0.8-1 %% "
                        "faster at prefill and on the skewed batch), packed below (gemm1 and "
                        "gather4 measured slower at decode)")
    p.add_argument("--pack", choices=("auto", "yes", "no"), default="auto",
                   help="tile-pack the expert weights at load (auto: yes for bf16, "
                        "no for fp8, which has no packed form)")
    p.add_argument("--precision", choices=("bf16", "fp8", "fp8-block"), default="bf16",
                   help="expert GEMM operands: bf16; e4m3 with per-row scales; or e4m3 with "
                        "UE8M0 block scales (1x128 tokens and h, 128x128 weights). Weights "
                        "are quantized once at load, tokens and h inside each step")
    p.add_argument("--fuse-combine", action="store_true",
                   help="fuse the gate-weighted combine into GEMM2's epilogue (fp32 reductions)")
    p.add_argument("--layers", type=int, default=1,
                   help="time a stack of this many consecutive layers replayed as one CUDA "
                        "graph (each layer its own router; expert weights shared)")
    p.add_argument("--sweep", action="store_true",
                   help="the dispatch + combine data-movement sweep instead of a layer: identity "
                        "experts, H=7168, E=256, top-8 uniform routing, T in 1024..65536; one JSON "
                        "line with the HBM GB/s of the permutation, dispatch and combine kernels")
    p.add_argument("--sweep-t", default=None,
                   help="comma-separated token counts of the sweep (default: 1024,4096,16384,65536)")
    p.add_argument("--unit-trace", action="store_true",
                   help="after the timed run, one more forward with GEMM1's per-unit trace "
                        "(moe_exec.unit_trace) of GEMM1 and of GEMM2; adds gemm1_units and "
                        "gemm2_units summaries to the JSON line")
    p.add_argument("--no-cpu-baseline", action="store_true")
    p.add_argument("--cpu-tokens", type=int, default=None,
                   help="oracle sample size (tokens); default 128, or 8 with --precision "
                        "fp8-block, whose oracle dequantizes each touched expert in full")
    p.add_argument("--cpu-one-core-tokens", type=int, default=4,
                   help="tokens of the single-core oracle timing (a child process with one "
                        "BLAS thread); 0 skips it")
    p.add_argument("--oracle-one-core", default=None, help=argparse.SUPPRESS)
    return p.parse_args()


# ---------------------------------------------------------------- distributed plumbing

def dist_env():
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return rank, world, local


def barrier(world):
    if world > 1:
        torch.distributed.barrier()


def max_over_ranks(v: float, world: int) -> float:
    if world == 1:
        return v
    t = torch.tensor([v], dtype=torch.float64)
    torch.distributed.all_reduce(t, op=torch.distributed.ReduceOp.MAX)
    return float(t.item())


# ---------------------------------------------------------------- measured peaks, clocks

def peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            m = json.load(f)
        return float(m["hbm_gbs"]), float(m["bf16_tflops"]), float(m.get(
            "bf16_tflops_sustained", m["bf16_tflops"])), "measured"
    except Exception:
        return FALLBACK_HBM_GBS, FALLBACK_BF16_TFLOPS, 1700.0, "fallback"


class ClockSampler:
    """nvidia-smi clock/throttle samples; only those inside the timed window count."""

    FIELDS = ("timestamp,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")
    NAMES = ("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap")

    def __init__(self, device_index: int):
        self.proc = None
        self.lines = []
        sel = []
        try:
            uuid = str(torch.cuda.get_device_properties(device_index).uuid)
            sel = ["-i", uuid if uuid.startswith("GPU-") else "GPU-" + uuid]
        except Exception:
            sel = ["-i", str(device_index)]
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", *sel, "--query-gpu=" + self.FIELDS, "--format=csv,noheader",
                 "-lms", "100"], stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except Exception:
            self.proc = None

    def stop(self):
        if self.proc is None:
            return
        self.proc.terminate()
        try:
            out, _ = self.proc.communicate(timeout=5)
        except Exception:
            self.proc.kill()
            out, _ = self.proc.communicate()
        self.lines = [l for l in out.splitlines() if l.strip()]

    def summary(self, t0: _dt.datetime, t1: _dt.datetime):
        rows = []
        for l in self.lines:
            f = [x.strip() for x in l.split(",")]
            if len(f) < 9:
                continue
            try:
                ts = _dt.datetime.strptime(f[0], "%Y/%m/%d %H:%M:%S.%f")
                rows.append((ts, float(f[1].split()[0]), float(f[2].split()[0]), f[5:9]))
            except Exception:
                continue
        inside = [r for r in rows if t0 <= r[0] <= t1]
        window = "timed"
        if not inside and rows:  # very short timed region: nearest samples (same workload)
            rows.sort(key=lambda r: abs((r[0] - t0).total_seconds()))
            inside, window = rows[:3], "adjacent"
        if not inside:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": [], "samples": 0}
        reasons = sorted({n for r in inside for n, v in zip(self.NAMES, r[3]) if v == "Active"})
        return {"sm_mhz": statistics.median(r[1] for r in inside),
                "sm_max_mhz": max(r[2] for r in inside), "reasons": reasons,
                "samples": len(inside), "window": window}


# ---------------------------------------------------------------- workload set-up

def build_inputs(wl, device, rank):
    d = I.layer_inputs(wl, seed=0, device=device)
    if rank:
        d["x"] = I.randn((wl.T, wl.H), 1.0, torch.bfloat16, rank, "x", device)
    return d


def gpu_counts_fn(L, wl, d, device):
    """Per-expert counts of the GPU routing for a given bias (used to calibrate the bias)."""
    cfg = L.config_of(wl)
    logits = torch.empty((wl.T, wl.E), device=device)
    idx = torch.empty((wl.T, wl.k), dtype=torch.int32, device=device)
    w = torch.empty((wl.T, wl.k), device=device)
    L.moe_router_logits(cfg, d["x"], d["Wr"], logits, None)

    def counts(b):
        L.moe_gate_topk(cfg, logits, b.to(device), idx, w)
        return torch.bincount(idx.reshape(-1).long(), minlength=wl.E).cpu()

    return counts


def calibrate(L, wl, d, device):
    if wl.balance == "balanced":
        b, _ = I.calibrate_balanced(gpu_counts_fn(L, wl, d, device), wl, d["bias"].cpu())
        d["bias"] = b.to(device)
    elif wl.balance == "zipf":
        b, _ = I.calibrate_zipf(gpu_counts_fn(L, wl, d, device), wl, 0)
        d["bias"] = b.to(device)


def scale_bytes(rows, n, fp8):
    """Bytes of the scales of a [rows, n] activation: one fp32 per row (fp8 = 1)
    or one UE8M0 byte per 1 x 128 block (fp8 = 2)."""
    return 0 if not fp8 else rows * 4 if fp8 == 1 else rows * (n // 128)


def algorithmic(wl, touched, fused_gather=True, fp8=0, fused_combine=False, pack_in_gemm1=False):
    """Algorithmic bytes and flops of each stage for one forward.

    GEMM1's token operand is counted as R*H*eb either way (packed rows read, or
    the same rows gathered from x); a fused dispatch has no copy of its own.
    With the copy inside GEMM1 (pack_in_gemm1) its bytes move to the GEMM1 stage.
    FP8 (eb = 1; fp8 = 1 row scales, 2 block scales): the dispatch stage also
    quantizes x (bf16 read, e4m3 + scales written) and the GEMM1 stage also
    quantizes h (bf16 read, e4m3 + scales); the GEMMs read the scales of their
    operands (weights: one fp32 per row, or one byte per 128 x 128 block).
    Fused combine: GEMM2 reduces into the fp32 [T, H] accumulator (counted once)
    instead of writing y_perm; the accumulator is cleared at the start (counted
    in the router stage) and converted to the bf16 output in the combine stage.
    """
    T, H, E, k, Iw, Is = wl.T, wl.H, wl.E, wl.k, wl.I, wl.I_shared
    R = T * k
    eb = 1 if fp8 else 2
    sb = lambda rows, n: scale_bytes(rows, n, fp8)
    # weight scales of a [rows, n] matrix: fp32 per row, or a byte per 128 x 128 block
    wsb = lambda rows, n: 0 if not fp8 else rows * 4 if fp8 == 1 else (rows // 128) * (n // 128)
    qx = T * H * 3 + sb(T, H) if fp8 else 0               # x -> e4m3 rows + scales
    qh = lambda rows, n: rows * n * 3 + sb(rows, n) if fp8 else 0   # h -> e4m3
    b = {
        "router": T * H * 2 + E * H * 4 + T * E * 4,
        "gate": T * E * 4 + T * k * 8,
        "permute": T * k * 4 * 3,
        "dispatch": qx + (0 if fused_gather else T * H * eb + R * H * eb),
        "gemm1": touched * (2 * Iw * H * eb + wsb(2 * Iw, H)) + R * H * eb + sb(R, H)
        + R * Iw * 2 + qh(R, Iw),
        "gemm2": touched * (H * Iw * eb + wsb(H, Iw)) + R * Iw * eb + sb(R, Iw) + R * H * 4,
        "shared_gemm1": (2 * Is * H * eb + wsb(2 * Is, H) + T * H * eb + sb(T, H) + T * Is * 2
                         + qh(T, Is)) if Is else 0,
        "shared_gemm2": (H * Is * eb + wsb(H, Is) + T * Is * eb + sb(T, Is) + T * H * 4)
        if Is else 0,
        "combine": R * H * 4 + (T * H * 4 if Is else 0) + T * H * 2 + R * 8,
    }
    if pack_in_gemm1 and not fused_gather:
        b["gemm1"] += T * H * eb + R * H * eb
        b["dispatch"] -= T * H * eb + R * H * eb
    if fused_combine:
        b["router"] += T * H * 4
        b["gemm2"] += T * H * 4 - R * H * 4
        if Is:  # the shared expert adds into the same accumulator: no y of its own
            b["shared_gemm2"] -= T * H * 4
        b["combine"] = T * H * 4 + T * H * 2
    f = {"router": 2 * T * E * H, "gemm1": 2 * R * H * 2 * Iw, "gemm2": 2 * R * Iw * H,
         "shared_gemm1": 2 * T * H * 2 * Is, "shared_gemm2": 2 * T * Is * H}
    if Is and Is == Iw:  # the library runs the shared expert inside the routed GEMM launches
        for d_ in (b, f):
            d_["gemm1"] += d_.pop("shared_gemm1")
            d_["gemm2"] += d_.pop("shared_gemm2")
    return b, f


def source_sha():
    """Hash of the GEMM kernel sources' code: `//` comments and blank lines are
    left out (the sources hold no `//` inside string literals), so a captured
    traffic figure stays attached to the code it was measured on."""
    h = hashlib.sha256()
    for p in GEMM_SOURCES:
        with open(os.path.join(ROOT, p), encoding="utf-8") as f:
            for line in f:
                code = line.split("//", 1)[0].rstrip()
                if code:
                    h.update(code.encode() + b"\n")
    return h.hexdigest()[:16]


def traffic_key(workload, fp8=0, pack_in_gemm1=False):
    """Key of a GEMM1 traffic capture: the workload, the operand form, and whether
    the launch also carried the dispatch copy (its pack warps' bytes)."""
    return (workload + {0: "", 1: " fp8", 2: " fp8-block"}[int(fp8)]
            + (" +dispatch in GEMM1" if pack_in_gemm1 else ""))


def measured_traffic(workload, fp8=0, kernel_bytes=None, pack_in_gemm1=False):
    """ncu DRAM bytes per GEMM1 launch, if captured for the current kernel source.

    The bf16 entry holds the bytes of the full launch; the FP8 entry holds the
    measured traffic / algorithmic ratio, applied to this run's GEMM1 kernel bytes.
    """
    try:
        with open(TRAFFIC_FILE) as f:
            t = json.load(f)
        e = t.get(traffic_key(workload, fp8, pack_in_gemm1))
        if e and e.get("source_sha") == source_sha():
            if "dram_bytes_per_launch" in e:
                return float(e["dram_bytes_per_launch"])
            if kernel_bytes is not None:
                return float(e["traffic_over_algorithmic"]) * kernel_bytes
    except Exception:
        pass
    return None


def kernel_roofline(bytes_, flops, t_s, hbm_gbs, tf_sust, tf_burst, src, dtype):
    """Roofline of one kernel: its bound is whichever of bytes / (measured copy
    bandwidth) and flops / (measured sustained dense peak of its dtype) takes
    longer; achieved and peak are in that bound's unit and frac = achieved /
    peak (= that time / the measured time). Both sides are also given against
    the measured and the nominal denominators."""
    t_b = bytes_ / (hbm_gbs * 1e9)
    t_f = flops / (tf_sust * 1e12)
    gbs, tfs = bytes_ / t_s / 1e9, flops / t_s / 1e12
    nominal_tf = NOMINAL_BF16_TFLOPS * (2.0 if dtype == "e4m3" else 1.0)
    hbm_side = {"achieved_GBs": round(gbs, 1), "frac_measured_copy": round(gbs / hbm_gbs, 4),
                "frac_nominal_8TBs": round(gbs / NOMINAL_HBM_GBS, 4)}
    tensor_side = {"achieved_TFLOPs": round(tfs, 1),
                   "frac_measured_sustained": round(tfs / tf_sust, 4),
                   "frac_measured_burst": round(tfs / tf_burst, 4),
                   "frac_nominal": round(tfs / nominal_tf, 4)}
    if t_f > t_b:
        r = {"bound": "tensor", "achieved": round(tfs, 1), "peak": round(tf_sust, 1),
             "unit": "TFLOP/s", "frac": round(tfs / tf_sust, 4),
             "peak_source": f"{dtype} dense, sustained ({'bf16_tflops_sustained' if dtype == 'bf16' else '2 x bf16_tflops_sustained'} of {src})"}
    else:
        r = {"bound": "hbm", "achieved": round(gbs, 1), "peak": hbm_gbs, "unit": "GB/s",
             "frac": round(gbs / hbm_gbs, 4), "peak_source": f"hbm_gbs of {src}"}
    r.update({"t_bytes_ms": round(t_b * 1e3, 4), "t_flops_ms": round(t_f * 1e3, 4),
              "t_measured_ms": round(t_s * 1e3, 4), "hbm": hbm_side, "tensor": tensor_side})
    return r


def unit_trace_summary(rec, H, fp8=0, flops_per_row=None):
    """Summary of a GEMM's per-unit trace records [n, 5] (int64): per token-row bin
    of the routed units (and the shared expert's), the units' count and median
    times: wait = handed out -> first stage ready, mma = first stage ready ->
    accumulator complete, epilogue = accumulator complete -> stored; and the
    unit's tensor rate while its MMAs ran (flops_per_row * m; GEMM1's default
    2 * 2 * 128 * H: gate and up of 128 features)."""
    fpr = 2 * 2 * 128 * H if flops_per_row is None else flops_per_row
    rec = np.asarray(rec, dtype=np.int64)
    rec = rec[(rec[:, 3] > 0) & (rec[:, 1] > 0)]
    if len(rec) == 0:
        return None
    t = (rec[:, :4] - rec[:, 0].min()) / 1e3  # us
    meta = rec[:, 4]
    m = (meta >> 16) & 0xFFFF
    grp = ((meta >> 32) & 0xFFFF) >= 1024
    wait, mma, epi = t[:, 1] - t[:, 0], t[:, 2] - t[:, 1], t[:, 3] - t[:, 2]
    tfs = fpr * m / np.maximum(mma, 1e-3) / 1e6   # TFLOP/s per SM
    out = {"units": int(len(rec)), "span_us": round(float(t[:, 3].max()), 1),
           "sms": int(len(np.unique(meta & 0xFFFF)))}
    bins = {}
    for lo, hi in ((0, 32), (32, 64), (64, 128), (128, 192), (192, 256)):
        sel = (m > lo) & (m <= hi) & ~grp
        if sel.any():
            bins[f"routed m {lo + 1}-{hi}"] = sel
    if grp.any():
        bins["shared"] = grp
    for name, sel in bins.items():
        out[name] = {"n": int(sel.sum()), "wait_us": round(float(np.median(wait[sel])), 2),
                     "mma_us": round(float(np.median(mma[sel])), 2),
                     "epilogue_us": round(float(np.median(epi[sel])), 2),
                     "TFLOPs_per_SM": round(float(np.median(tfs[sel])), 3)}
    return out


# ---------------------------------------------------------------- CPU oracle leg

def cpu_model() -> str:
    """The host CPU's model name (lscpu, else /proc/cpuinfo, else the machine type)."""
    try:
        out = subprocess.run(["lscpu"], capture_output=True, text=True, timeout=10).stdout
        for line in out.splitlines():
            if line.split(":")[0].strip() == "Model name":
                return line.split(":", 1)[1].strip()
    except Exception:
        pass
    try:
        with open("/proc/cpuinfo") as f:
            for line in f:
                if line.lower().startswith("model name"):
                    return line.split(":", 1)[1].strip()
    except Exception:
        pass
    import platform
    return platform.machine()


def oracle_cfg(wl, n):
    from oracle import moe_oracle as O
    return O.LayerConfig(T=n, H=wl.H, E=wl.E, k=wl.k, I=wl.I, I_shared=wl.I_shared,
                         n_groups=wl.n_groups, topk_groups=wl.topk_groups, gate=wl.gate,
                         normalize=wl.normalize, route_scale=wl.route_scale)


def time_oracle(wl, xr, Wr, b, host_of, shared, f8=None):
    """Time the oracle's layer on token rows xr (fp64 [n, H]).

    host_of(experts) -> {e: host tensors of expert e}, built before the clock
    starts (host copies of the touched experts: bf16 W13, W2, or the FP8 forms'
    codes and scales); shared likewise for the shared expert (or None)."""
    from oracle import moe_oracle as O

    cfg = oracle_cfg(wl, len(xr))
    idx, _ = O.gate_topk(O.router_logits(xr, Wr), b, cfg)
    host = host_of(sorted(int(e) for e in np.unique(idx)))
    if f8:
        blk = f8.get("block", False)

        def conv(t, i):
            if i % 2 == 0:
                return O.e4m3_decode(t.numpy())
            return t.numpy().astype(np.int64) - 127 if blk else t.numpy()

        ffn = O.swiglu_ffn_fp8_blocks if blk else O.swiglu_ffn_fp8
    else:
        conv = lambda t, i: t.to(torch.float64).numpy()
        ffn = O.swiglu_ffn

    def get_expert(e):
        return tuple(conv(t, i) for i, t in enumerate(host[e]))

    get_shared = (lambda: tuple(conv(t, i) for i, t in enumerate(shared))) if shared else None
    t0 = time.perf_counter()
    O.layer_forward_tokens(xr, Wr, b, get_expert, cfg, get_shared, ffn=ffn)
    dt = time.perf_counter() - t0
    return len(xr) / dt, dt, len(host)


def oracle_tokens_per_s(wl, d, tokens):
    """Time the CPU oracle on a sample of tokens; weights come from host copies.

    With d["fp8"] the oracle runs the FP8 expert form on the e4m3 weights."""
    tok = torch.as_tensor(tokens, device=d["x"].device)
    xr = d["x"][tok].to(torch.float64).cpu().numpy()
    Wr = d["Wr"].cpu().numpy()
    b = None if d["bias"] is None else d["bias"].cpu().numpy()
    f8 = d.get("fp8")
    if f8:
        # (codes, scales) pairs: e4m3 bytes, then fp32 row scales or UE8M0 block exponents
        host_of = lambda es: {e: tuple(f8[n][e].cpu() for n in ("W13", "s13", "W2", "s2"))
                              for e in es}
        shared = tuple(f8[n].cpu() for n in ("Ws13", "ss13", "Ws2", "ss2")) \
            if wl.I_shared else None
    else:
        host_of = lambda es: {e: (d["W13"][e].cpu(), d["W2"][e].cpu()) for e in es}
        shared = (d["Ws13"].cpu(), d["Ws2"].cpu()) if wl.I_shared else None
    return time_oracle(wl, xr, Wr, b, host_of, shared, f8)


def oracle_one_core_child(path):
    """Child-process body of the single-core timing (BLAS limited to one thread
    by the parent through the environment). Reads the sampled token rows, Wr and
    the bias from `path`; the touched experts' bf16 weights are drawn here on the
    CPU with the workload's distributions (same shapes and work as the device
    draw; the oracle's time does not depend on the values). Prints one JSON line."""
    torch.set_num_threads(1)
    z = np.load(path)
    wl = I.WORKLOADS[str(z["workload"])]
    b = z["bias"] if z["bias"].size else None

    def host_of(es):
        return {e: (I.randn((2 * wl.I, wl.H), 0.02, torch.bfloat16, 0, "W13", "cpu", extra=e),
                    I.randn((wl.H, wl.I), 0.02, torch.bfloat16, 0, "W2", "cpu", extra=e))
                for e in es}

    shared = (I.randn((2 * wl.I_shared, wl.H), 0.02, torch.bfloat16, 0, "Ws13", "cpu"),
              I.randn((wl.H, wl.I_shared), 0.02, torch.bfloat16, 0, "Ws2", "cpu")) \
        if wl.I_shared else None
    v, dt, ne = time_oracle(wl, z["x"], z["Wr"], b, host_of, shared)
    print(json.dumps({"value": v, "seconds": dt, "experts": ne, "tokens": int(len(z["x"]))}))


def oracle_one_core(wl, d, n_tokens, seed=2):
    """The oracle on one core: a child process with every BLAS / OpenMP pool at
    one thread, timing n_tokens sampled tokens of the batch (bf16 form only)."""
    import tempfile
    toks = I.sample_tokens(wl.T, n_tokens, seed)
    xr = d["x"][toks.to(d["x"].device)].to(torch.float64).cpu().numpy()
    b = np.zeros(0, np.float32) if d["bias"] is None else d["bias"].cpu().numpy()
    env = dict(os.environ, OMP_NUM_THREADS="1", OPENBLAS_NUM_THREADS="1", MKL_NUM_THREADS="1")
    with tempfile.TemporaryDirectory() as td:
        path = os.path.join(td, "sample.npz")
        name = next(k_ for k_, v in I.WORKLOADS.items() if v == wl)
        np.savez(path, x=xr, Wr=d["Wr"].cpu().numpy(), bias=b, workload=name)
        r = subprocess.run([sys.executable, os.path.abspath(__file__), "--oracle-one-core", path],
                           capture_output=True, text=True, env=env, timeout=600)
    if r.returncode != 0:
        return {"error": (r.stderr.strip().splitlines() or ["child failed"])[-1][:200]}
    o = json.loads(r.stdout.strip().splitlines()[-1])
    return {"value": o["value"], "unit": "tokens/s", "cores": 1,
            "sample": f"{o['tokens']} sampled tokens ({o['experts']} experts touched), "
                      f"{o['seconds']:.1f} s, one BLAS thread; the touched experts' weights "
                      f"drawn on the host with the workload's distributions"}


def cpu_baseline(wl, d, n_tokens, seed=1, one_core_tokens=0):
    toks = I.sample_tokens(wl.T, n_tokens, seed).numpy()
    v, dt, ne = oracle_tokens_per_s(wl, d, toks)
    form = ("block-scaled FP8 expert form, " if d["fp8"].get("block") else
            "FP8 expert form, ") if d.get("fp8") else ""
    sampled = len(toks) < wl.T
    r = {"value": v, "unit": "tokens/s", "cores": os.cpu_count(), "kind": "oracle",
         "cpu_model": cpu_model(),
         "sample": f"{'sampled: ' if sampled else ''}{len(toks)} of the {wl.T} tokens "
                   f"({ne} experts touched), {form}numpy fp64 oracle, {dt:.1f} s; "
                   f"BLAS threads = host cores"}
    if one_core_tokens and not d.get("fp8"):
        r["one_core"] = oracle_one_core(wl, d, one_core_tokens)
    return r


# ---------------------------------------------------------------- main arms

REF_TIMED_S = 90.0  # the reference arm's timed steps together take about this long


def run_reference(args, wl, rank, world, device):
    if rank != 0:
        return
    d = build_inputs(wl, device, 0)
    from paper_2603_02376_gb300 import _lib as L
    if wl.balance != "none":
        L.load()
        calibrate(L, wl, d, device)
    # per-step sample: a first untimed call measures the oracle's cost per token,
    # then each timed step takes as many tokens as keep the K steps near REF_TIMED_S
    n_max = max(1, (args.cpu_tokens or 128) // 2)
    v0, _, _ = oracle_tokens_per_s(wl, d, I.sample_tokens(wl.T, min(8, n_max), 99).numpy())
    n = int(max(1, min(n_max, REF_TIMED_S * v0 / max(args.steps, 1))))
    for s in range(args.warmup):
        oracle_tokens_per_s(wl, d, I.sample_tokens(wl.T, n, 100 + s).numpy())
    times = []
    for s in range(args.steps):
        v, dt, _ = oracle_tokens_per_s(wl, d, I.sample_tokens(wl.T, n, 1000 + s).numpy())
        times.append(dt)
    tot = sum(times)
    value = n * args.steps / tot
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": "tokens/s",
        "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": 1e3 * tot / args.steps, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": config_of(wl, args),
        "cpu_baseline": {"value": value, "unit": "tokens/s", "cores": os.cpu_count(),
                         "kind": "oracle", "cpu_model": cpu_model(),
                         "sample": f"sampled: {n} tokens per step of the {wl.T}-token batch, "
                                   f"numpy fp64"},
        "e2e": {"value": value, "unit": "tokens/s", "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


def packs(args, wl):
    """Whether the run uses tile-packed expert weights (bf16 only; auto = yes: the
    GEMMs fetch each packed weight tile with one bulk copy, measured as fast or
    faster at every batch size)."""
    if args.precision != "bf16":
        return False
    return args.pack in ("auto", "yes")


def dispatch_flag(args, wl):
    """moe_exec.fuse_gather of the run: 0 packed, 1 gather4, 2 copy inside GEMM1."""
    if args.dispatch == "auto":
        return 2 if wl.T * wl.k > 24 * wl.E else 0
    return {"packed": 0, "gather4": 1, "gemm1": 2}[args.dispatch]


def dispatch_label(args, wl):
    f = dispatch_flag(args, wl)
    if f == 1 and wl.T * wl.k <= 24 * wl.E:
        return "fused into GEMM1 (TMA gather4)"
    tiled = args.mode != "overlap-tokens" and args.precision != "fp8-block"
    rows = " in the tile-packed row layout" if tiled else ""
    if f == 2 and args.mode == "seq" and args.precision != "fp8-block":
        return ("inside the GEMM1 launch (pack warps write x_perm" + rows
                + " behind the shared expert)")
    if tiled:
        return "packed x_perm in the tile-packed row layout (dispatch kernel)"
    return "packed x_perm (dispatch kernel)"


def config_of(wl, args):
    return {"workload": wl.name, "T": wl.T, "H": wl.H, "E": wl.E, "k": wl.k, "I": wl.I,
            "I_shared": wl.I_shared, "gating": ("sigmoid+bias, 8 groups keep 4, top-8, x2.5"
                                                if wl.gate == 1 else "softmax top-k"),
            "mode": args.mode, "dispatch": dispatch_label(args, wl),
            "weights": "tile-packed at load (moe_pack_weights)" if packs(args, wl) else "row-major",
            "precision": {"bf16": "bf16 expert GEMMs",
                          "fp8": "e4m3 expert GEMMs, per-row fp32 scales (weights quantized "
                                 "at load)",
                          "fp8-block": "e4m3 expert GEMMs, UE8M0 block scales: 1x128 "
                                       "activations, 128x128 weights (quantized at load), "
                                       "applied by tcgen05 kind::mxf8f6f4"}[args.precision],
            "combine": "fused into GEMM2's epilogue (fp32 reductions)" if args.fuse_combine
            else "y_perm + combine kernel",
            "global_batch": wl.T * args.gpus,
            "l2": "inputs larger than L2: the expert weights streamed per step exceed 129 MB",
            "parallelism": f"replicas{args.gpus}"}


def run_ours(args, wl, rank, world, local, device):
    from paper_2603_02376_gb300 import _lib as L
    L.load()
    d = build_inputs(wl, device, rank)
    calibrate(L, wl, d, device)
    cfg = L.config_of(wl)
    mode = dict(seq=dict(), **{"overlap-tokens": dict(overlap=1, chunk_axis=0,
                                                      chunk_tokens=args.chunk_tokens),
                               "overlap-experts": dict(overlap=1, chunk_axis=1,
                                                       n_expert_chunks=args.expert_chunks)})[
        args.mode]
    fuse = dispatch_flag(args, wl)
    # the library gathers in GEMM1 only for decode-sized batches (<= 24 rows per expert)
    fused = fuse == 1 and wl.T * wl.k <= 24 * wl.E
    fusable = wl.T * wl.k <= 24 * wl.E  # the library would fuse the dispatch on request
    # the dispatch copy inside GEMM1: sequential forwards, bf16 or row-scaled e4m3
    in_gemm1_ok = args.mode == "seq" and args.precision != "fp8-block"
    in_gemm1 = fuse == 2 and in_gemm1_ok
    fp8 = {"bf16": 0, "fp8": 1, "fp8-block": 2}[args.precision]
    fc = 1 if args.fuse_combine else 0
    ex = L.exec_config(fuse_gather=fuse, fp8=fp8, fuse_combine=fc, **mode)
    # one workspace serves the timed mode and the sequential stats / stage-event passes
    ws = torch.empty(max(L.moe_workspace_size(cfg, ex),
                         L.moe_workspace_size(cfg, L.exec_config(fuse_gather=fuse, fp8=fp8)),
                         L.moe_workspace_size(cfg, L.exec_config(fuse_gather=0, fp8=fp8))),
                     dtype=torch.uint8, device=device)
    out = torch.empty((wl.T, wl.H), dtype=torch.bfloat16, device=device)
    # a stream of its own: the default stream's handle is NULL, which the C ABI
    # reads as "no aux stream given" (the library's own pack stream), so the
    # one-stream comparison of the pipelined modes needs a non-default stream
    stream = torch.cuda.Stream()
    torch.cuda.synchronize()
    # the layer runs on tile-packed copies (a load-time layout transform, not part
    # of the timed step); the row-major tensors stay for the CPU oracle
    run_w = {k_: d.get(k_) for k_ in ("W13", "W2", "Ws13", "Ws2")}
    packed = packs(args, wl)
    if packed:
        run_w = {k_: (None if v is None else L.pack_weights(v)) for k_, v in run_w.items()}
        torch.cuda.synchronize()
    if fp8:
        # e4m3 copies of the expert weights with per-row scales (fp8 = 1, kept per
        # expert as [E, rows]) or 128 x 128 block exponents (fp8 = 2, kept per
        # expert as [E, rows/128, cols/128]): a
        # load-time step like the packing above; the bf16 tensors are dropped (the
        # oracle leg reads the e4m3 bytes)
        f8 = {"block": fp8 == 2}
        for n, sn in (("W13", "s13"), ("W2", "s2"), ("Ws13", "ss13"), ("Ws2", "ss2")):
            if d.get(n) is None:
                f8[n] = f8[sn] = None
            elif fp8 == 1:
                f8[n], f8[sn] = L.quantize_fp8(d[n])
                if d[n].dim() == 3:  # row scales per expert: [E, rows]
                    f8[sn] = f8[sn].view(d[n].shape[0], -1)
            else:
                f8[n], f8[sn] = L.quantize_fp8_weight_blocks(d[n])
                if d[n].dim() == 3:
                    f8[sn] = f8[sn].view(d[n].shape[0], -1, f8[sn].shape[-1])
        torch.cuda.synchronize()
        d["fp8"] = f8
        for n in ("W13", "W2", "Ws13", "Ws2"):
            d[n] = None
        run_w = None
        torch.cuda.empty_cache()
        W = L.weights_struct(d["Wr"], d["bias"], f8["W13"], f8["W2"], f8["Ws13"], f8["Ws2"], 0,
                             f8["s13"], f8["s2"], f8["ss13"], f8["ss2"])
    else:
        W = L.weights_struct(d["Wr"], d["bias"], run_w["W13"], run_w["W2"], run_w["Ws13"],
                             run_w["Ws2"], 1 if packed else 0)

    if args.layers > 1:
        return run_stack(args, wl, rank, world, local, device, L, cfg, ex, W, d)

    def step():
        L.moe_layer_forward(cfg, ex, W, d["x"], out, None, ws, stream)

    # routing statistics of this batch (touched experts set the GEMM weight bytes)
    counts = torch.empty(wl.E, dtype=torch.int32, device=device)
    L.moe_layer_forward(cfg, L.exec_config(fuse_gather=fuse, fp8=fp8), W, d["x"], out,
                        L.aux_struct(counts=counts), ws, stream)
    L.moe_check_errors(stream)
    cnt = counts.cpu()
    touched = int((cnt > 0).sum())

    for _ in range(args.warmup):
        step()
    torch.cuda.synchronize()
    L.moe_check_errors(stream)

    # --- device-resident timing
    sampler = ClockSampler(local)
    time.sleep(0.3)
    barrier(world)
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    n0 = L.moe_launch_count()
    w0 = _dt.datetime.now()
    e0.record(stream)
    for _ in range(args.steps):
        step()
    e1.record(stream)
    torch.cuda.synchronize()
    w1 = _dt.datetime.now()
    barrier(world)
    launches = L.moe_launch_count() - n0
    ms = max_over_ranks(e0.elapsed_time(e1), world)
    time.sleep(0.25)
    sampler.stop()
    clocks = sampler.summary(w0, w1)
    L.moe_check_errors(stream)
    value = wl.T * world * args.steps / (ms / 1e3)

    # --- per-stage timing (sequential forward with stage events, same stream)
    K2 = min(args.steps, 50)

    def traced(fuse_flag):
        evs = [[torch.cuda.Event(enable_timing=True) for _ in L.STAGES] for _ in range(K2)]
        for row in evs:          # torch creates the CUDA event at its first record
            for e in row:
                e.record(stream)
        torch.cuda.synchronize()
        for i in range(K2):
            exs = L.exec_config(fuse_gather=fuse_flag, stage_events=evs[i], fp8=fp8,
                                fuse_combine=fc)
            L.moe_layer_forward(cfg, exs, W, d["x"], out, None, ws, stream)
        torch.cuda.synchronize()
        return {L.STAGES[j]: statistics.mean(evs[i][j - 1].elapsed_time(evs[i][j])
                                             for i in range(K2))
                for j in range(1, len(L.STAGES))}

    stage_ms = traced(fuse)
    dispatch_fusion = None
    # the packed dispatch against the dispatch fused into GEMM1 (same batch): the
    # copy inside the GEMM1 launch at every size, TMA gather4 at decode sizes;
    # hidden_frac = 1 - (GEMM1 fused - GEMM1 packed) / dispatch kernel
    if in_gemm1_ok and args.layers == 1:
        pk_ms = stage_ms if fuse == 0 else traced(0)
        dispatch_fusion = {"active": {0: "packed", 1: "gather4" if fused else "packed",
                                      2: "gemm1"}[fuse],
                           "dispatch_ms_packed": round(pk_ms["dispatch"], 4),
                           "gemm1_ms_packed": round(pk_ms["gemm1"], 4),
                           "layer_ms_packed": round(sum(pk_ms.values()), 4)}
        forms = [("gemm1", 2)] + ([("gather4", 1)] if fusable else [])
        for name, flag in forms:
            fz_ms = stage_ms if fuse == flag else traced(flag)
            extra = fz_ms["gemm1"] + fz_ms["dispatch"] - pk_ms["gemm1"]
            dispatch_fusion[f"gemm1_ms_{name}"] = round(fz_ms["gemm1"], 4)
            dispatch_fusion[f"layer_ms_{name}"] = round(sum(fz_ms.values()), 4)
            dispatch_fusion[f"hidden_frac_{name}"] = round(1.0 - extra / pk_ms["dispatch"], 3) \
                if pk_ms["dispatch"] > 0 else None

    # --- end to end through the C ABI with host buffers: every step copies its
    # input batch in from pinned host memory and its output back out, on two
    # copy streams with double-buffered device tensors, so that step i + 1's
    # input and step i's output move while the layers run (a serving loop); the
    # timed region spans the first copy in to the last copy out
    xh = d["x"].cpu().pin_memory()
    oh = [torch.empty((wl.T, wl.H), dtype=torch.bfloat16).pin_memory() for _ in range(2)]
    xd = [torch.empty_like(d["x"]) for _ in range(2)]
    od = [out, torch.empty_like(out)]
    s_in, s_out = torch.cuda.Stream(), torch.cuda.Stream()

    def e2e_run(n, t0=None, t1=None):
        ev_in = [torch.cuda.Event() for _ in range(2)]
        ev_fwd = [torch.cuda.Event() for _ in range(2)]
        ev_out = [torch.cuda.Event() for _ in range(2)]
        s_in.wait_stream(stream)
        s_out.wait_stream(stream)
        if t0 is not None:
            t0.record(s_in)
        with torch.cuda.stream(s_in):
            xd[0].copy_(xh, non_blocking=True)
        ev_in[0].record(s_in)
        for i in range(n):
            b = i % 2
            stream.wait_event(ev_in[b])
            if i >= 2:
                stream.wait_event(ev_out[b])  # step i - 2's output has left od[b]
            L.moe_layer_forward(cfg, ex, W, xd[b], od[b], None, ws, stream)
            ev_fwd[b].record(stream)
            if i + 1 < n:  # next step's input, once step i - 1 has read that buffer
                nb = (i + 1) % 2
                if i >= 1:
                    s_in.wait_event(ev_fwd[nb])
                with torch.cuda.stream(s_in):
                    xd[nb].copy_(xh, non_blocking=True)
                ev_in[nb].record(s_in)
            s_out.wait_event(ev_fwd[b])
            with torch.cuda.stream(s_out):
                oh[b].copy_(od[b], non_blocking=True)
            ev_out[b].record(s_out)
        if t1 is not None:
            t1.record(s_out)

    e2e_run(min(3, args.warmup))
    barrier(world)
    torch.cuda.synchronize()
    f0, f1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e2e_run(args.steps, f0, f1)
    torch.cuda.synchronize()
    barrier(world)
    e2e_ms = max_over_ranks(f0.elapsed_time(f1), world)
    e2e_value = wl.T * world * args.steps / (e2e_ms / 1e3)
    assert torch.equal(oh[(args.steps - 1) % 2], od[(args.steps - 1) % 2].cpu())

    # --- two-stream overlap: the same chunking on one stream, and the pack work alone
    overlap = None
    if ex.overlap:
        barrier(world)
        torch.cuda.synchronize()
        g0, g1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        g0.record(stream)
        for _ in range(args.steps):
            L.moe_layer_forward(cfg, ex, W, d["x"], out, None, ws, stream, aux_stream=stream)
        g1.record(stream)
        torch.cuda.synchronize()
        t_single = max_over_ranks(g0.elapsed_time(g1), world) / args.steps
        t_ovl = ms / args.steps
        # the pipelined modes pack on the pack stream with the gather kernel, not
        # inside GEMM1: their pack work is that of the sequential forward with
        # the packed dispatch
        pk_ms = stage_ms if fuse != 2 else traced(0)
        t_pack = sum(pk_ms[k] for k in ("router", "gate", "permute", "dispatch"))
        overlap = {"ms_two_streams": round(t_ovl, 4), "ms_same_chunks_one_stream": round(t_single, 4),
                   "ms_pack_work": round(t_pack, 4),
                   "hidden_frac": round((t_single - t_ovl) / t_pack, 3) if t_pack > 0 else None,
                   "ms_sequential_unchunked": round(sum(stage_ms.values()), 4),
                   "timeline": pipeline_timeline(L, cfg, ex, W, d["x"], out, ws, stream, wl, args)}

    hbm, tf_burst, tf_sust, src = peaks()
    b, f = algorithmic(wl, touched, fused, fp8, bool(fc), pack_in_gemm1=in_gemm1)
    g1 = stage_ms["gemm1"] / 1e3
    # GEMM1's own bytes (the FP8 GEMM1 stage also holds the h quantization)
    R = wl.T * wl.k
    qh = (R * wl.I * 3 + scale_bytes(R, wl.I, fp8)
          + (wl.T * wl.I_shared * 3 + scale_bytes(wl.T, wl.I_shared, fp8)
             if wl.I_shared == wl.I else 0)) if fp8 else 0
    traffic = measured_traffic(wl.name, fp8, b["gemm1"] - qh, pack_in_gemm1=in_gemm1)
    pk = 2.0 if fp8 else 1.0   # e4m3 dense peak = the measured bf16 peak x the nominal 2x
    stages = {}
    for s_, t in stage_ms.items():
        e = {"ms": round(t, 4)}
        if b.get(s_):
            e["GB/s"] = round(b[s_] / (t / 1e3) / 1e9, 1)
            e["frac_hbm"] = round(b[s_] / (t / 1e3) / 1e9 / hbm, 3)
            e["frac_hbm_nominal"] = round(b[s_] / (t / 1e3) / 1e9 / NOMINAL_HBM_GBS, 3)
        if f.get(s_):
            e["TFLOP/s"] = round(f[s_] / (t / 1e3) / 1e12, 2)
            e["frac_fp8" if fp8 else "frac_bf16"] = round(
                f[s_] / (t / 1e3) / 1e12 / (pk * tf_sust), 4)
        stages[s_] = e
    roofline = kernel_roofline(b["gemm1"], f["gemm1"], g1, hbm, tf_sust * pk, tf_burst * pk,
                               src, "e4m3" if fp8 else "bf16")
    roofline.update({
        "kernel": {0: "grouped GEMM1 + SwiGLU (tcgen05), routed + shared",
                   1: "grouped GEMM1 + SwiGLU (tcgen05 kind::f8f6f4) and the h "
                      "quantization, routed + shared",
                   2: "grouped GEMM1 + SwiGLU (tcgen05 kind::mxf8f6f4 block_scale) "
                      "and the h block quantization, routed + shared"}[fp8],
        "traffic": traffic, "algorithmic_bytes": b["gemm1"], "algorithmic_flops": f["gemm1"],
        "touched_experts": touched,
        "note": ("the grouped GEMM1 launch also runs the shared expert's GEMM1; its bytes and "
                 "flops are included") if wl.I_shared == wl.I else ""})

    line = {
        "metric": METRIC, "value": value, "unit": "tokens/s", "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms / args.steps,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
        "dtype": "e4m3" if fp8 else "bf16",
        "data": "synthetic (seeded N(0,1) activations, N(0,0.02^2) bf16 weights"
                + ({1: ", quantized to e4m3 at load)",
                    2: ", quantized to e4m3 in 128x128 blocks at load)"}.get(fp8, ")")),
        "config": config_of(wl, args),
        "e2e": {"value": e2e_value, "unit": "tokens/s", "h2d_bytes_per_step": wl.T * wl.H * 2,
                "d2h_bytes_per_step": wl.T * wl.H * 2,
                "copies": "pinned host <-> device every step, on two copy streams, "
                          "double-buffered (overlapping the neighbouring steps' layers)"},
        "gpu_launches": launches,
        "roofline": roofline,
        "clocks": clocks,
        "stages": stages,
        "denominators": {"frac_hbm": f"measured copy {hbm} GB/s ({src}; read + write bytes)",
                         "frac_hbm_nominal": f"nominal {NOMINAL_HBM_GBS:.0f} GB/s",
                         "frac_bf16 / frac_fp8": f"measured sustained dense "
                                                 f"{tf_sust} TFLOP/s (x2 for e4m3)"},
        "routing": {"max_over_mean": round(float(cnt.max()) * wl.E / (wl.T * wl.k), 3),
                    "touched_experts": touched},
    }
    # the whole layer against its roofline: max(bytes / BW, flops / P) over the
    # measured step time, with the measured peaks and with the nominal ones
    # (8 TB/s; 2.25 PFLOP/s bf16, twice that for e4m3)
    B, F = float(sum(b.values())), float(sum(f.values()))
    t_step = ms / args.steps / 1e3
    tb, tfb, tfs = B / (hbm * 1e9), F / (pk * tf_burst * 1e12), F / (pk * tf_sust * 1e12)
    line["layer_roofline"] = {
        "bytes": B, "flops": F, "t_bytes_ms": round(tb * 1e3, 4),
        "t_flops_ms_burst": round(tfb * 1e3, 4), "t_flops_ms_sustained": round(tfs * 1e3, 4),
        "frac_measured_peaks": round(max(tb, tfs) / t_step, 4),
        "frac_nominal_peaks": round(max(B / (NOMINAL_HBM_GBS * 1e9),
                                        F / (pk * NOMINAL_BF16_TFLOPS * 1e12)) / t_step, 4),
        "bound": "hbm" if tb >= tfs else "tensor"}
    if args.unit_trace and not ex.overlap:
        # one extra forward per traced GEMM; GEMM2's units cover 256 output
        # features (128 when H is not a multiple of 256) over K = I
        feat2 = 256 if wl.H % 256 == 0 else 128
        for gemm, key, fpr in ((1, "gemm1_units", 2 * 2 * 128 * wl.H),
                               (2, "gemm2_units", 2 * feat2 * wl.I)):
            rt = torch.zeros((1 << 17, L.UNIT_TRACE_FIELDS), dtype=torch.int64, device=device)
            L.moe_layer_forward(cfg, L.exec_config(fuse_gather=fuse, fp8=fp8, fuse_combine=fc,
                                                   unit_trace=rt, unit_trace_gemm=gemm),
                                W, d["x"], out, None, ws, stream)
            torch.cuda.synchronize()
            line[key] = unit_trace_summary(rt.cpu().numpy(), wl.H, fp8, fpr)
    if overlap:
        line["overlap"] = overlap
    if dispatch_fusion:
        line["dispatch_fusion"] = dispatch_fusion
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        n_cpu = args.cpu_tokens or (8 if args.precision == "fp8-block" else 128)
        line["cpu_baseline"] = cpu_baseline(wl, d, n_cpu,
                                            one_core_tokens=args.cpu_one_core_tokens)
    if rank == 0:
        print(json.dumps(line), flush=True)


def pipeline_timeline(L, cfg, ex, W, x, out, ws, stream, wl, args):
    """One pipelined forward with moe_exec.pipe_events: when each launch boundary
    of both streams was reached, in ms after the first event (the order is the
    one include/moe.h documents)."""
    n = -(-wl.T // min(wl.T, args.chunk_tokens)) if ex.chunk_axis == 0 else args.expert_chunks
    if ex.chunk_axis == 0:
        labels = [f"pack: chunk {i} {w}" for i in range(n) for w in ("begins", "packed")]
        comp = [f"compute: chunk {i} GEMMs {w}" for i in range(n) for w in ("begin", "end")]
    else:
        labels = ["pack: routing begins", "pack: routed"] + [f"pack: range {i} gathered"
                                                             for i in range(n)]
        comp = [f"compute: range {i} GEMMs {w}" for i in range(n) for w in ("begin", "end")]
    labels += ["compute: shared expert begins", "compute: shared expert ends"] + comp
    evs = [torch.cuda.Event(enable_timing=True) for _ in labels]
    for e in evs:   # torch creates the CUDA event at its first record
        e.record(stream)
    torch.cuda.synchronize()
    ext = L.exec_config(overlap=1, chunk_axis=ex.chunk_axis, chunk_tokens=ex.chunk_tokens,
                        n_expert_chunks=ex.n_expert_chunks, fuse_gather=ex.fuse_gather,
                        fp8=ex.fp8, fuse_combine=ex.fuse_combine, pipe_events=evs)
    L.moe_layer_forward(cfg, ext, W, x, out, None, ws, stream)
    torch.cuda.synchronize()
    return sorted(((lab, round(evs[0].elapsed_time(e), 4)) for lab, e in zip(labels, evs)),
                  key=lambda r: r[1])


def run_stack(args, wl, rank, world, local, device, L, cfg, ex, W, d):
    """The paper's multi-layer study: L consecutive layers (layer l + 1 reads layer l's
    bf16 output) captured once into a CUDA graph; each step is one graph launch.

    Layer l has its own router weights (seeded by l); the expert weights are shared by
    all layers (a distinct copy per layer would not fit 16 layers in HBM, and each
    layer still streams its 22.5 GB of expert weights from HBM: L2 is 129 MB).
    """
    nl = args.layers
    layers = [W]
    keep = []
    for l in range(1, nl):
        Wr = I.randn((wl.E, wl.H), 0.01, torch.float32, l, "Wr", device)
        keep.append(Wr)
        wl_ = L.moe_weights.from_buffer_copy(W)
        wl_.Wr = Wr.data_ptr()
        layers.append(wl_)
    ws = torch.empty(L.moe_stack_workspace_size(cfg, ex), dtype=torch.uint8, device=device)
    x = d["x"].clone()
    out = torch.empty_like(x)
    stream = torch.cuda.current_stream()
    g = L.Graph(cfg, ex, layers, x, out, ws, stream=stream)
    for _ in range(args.warmup):
        g.launch(stream)
    torch.cuda.synchronize()
    L.moe_check_errors(stream)
    sampler = ClockSampler(local)
    time.sleep(0.3)
    barrier(world)
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    w0 = _dt.datetime.now()
    e0.record(stream)
    for _ in range(args.steps):
        g.launch(stream)
    e1.record(stream)
    torch.cuda.synchronize()
    w1 = _dt.datetime.now()
    barrier(world)
    ms = max_over_ranks(e0.elapsed_time(e1), world)
    time.sleep(0.25)
    sampler.stop()
    L.moe_check_errors(stream)
    line = {
        "metric": METRIC + f" (stack of {nl} layers, one CUDA graph)",
        "value": wl.T * world * args.steps / (ms / 1e3), "unit": "tokens/s", "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms / args.steps,
        "ms_per_layer": ms / args.steps / nl, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "bf16" if args.precision == "bf16" else "e4m3",
        "data": "synthetic (seeded N(0,1) activations, N(0,0.02^2) bf16 weights)",
        "config": dict(config_of(wl, args), layers=nl, graph=True,
                       between_layers="unit-gain RMS normalization (moe_rms_norm)"),
        "gpu_launches": g.kernels * args.steps,
        "clocks": sampler.summary(w0, w1),
    }
    g.close()
    if rank == 0:
        print(json.dumps(line), flush=True)


def run_sweep(args, rank, world, local, device):
    """Dispatch + combine of uniform top-8 routing at T = 1024 .. 65536 (identity experts).

    Per T: the permutation alone (moe_dispatch without x_perm), the permutation and
    the row copy (moe_dispatch with x_perm; the copy's time is the difference), and
    moe_combine of fp32 rows into a bf16 output, each timed with CUDA events around
    `steps` launches, a buffer larger than L2 written before each launch whose
    input would fit in L2 (the combine's y_perm never does). Algorithmic
    bytes: copy T*H*2 read + T*k*H*2 written; combine T*k*H*4 read + T*H*2 written
    (+ 8 bytes of slot row and weight per entry).
    """
    from paper_2603_02376_gb300 import _lib as L
    L.load()
    H, E, k = 7168, 256, 8
    hbm, _, _, src = peaks()
    stream = torch.cuda.current_stream()
    flush = torch.empty(256 << 20, dtype=torch.uint8, device=device)
    n0 = L.moe_launch_count()
    rows, w0 = [], _dt.datetime.now()
    sampler = ClockSampler(local)

    def timed(fn, flush_l2=True):
        # all launches enqueued ahead (one synchronisation at the end), so each
        # timed kernel is already queued behind its L2 flush when its start
        # event fires: the events bracket the kernel, not the host's launch.
        # flush_l2=False where the kernel's input alone exceeds L2.
        n = args.warmup + args.steps
        ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
              for _ in range(n)]
        for i in range(n):
            if flush_l2:
                flush.fill_(i & 0xFF)
            ev[i][0].record(stream)
            fn()
            ev[i][1].record(stream)
        torch.cuda.synchronize()
        return sum(ev[i][0].elapsed_time(ev[i][1]) for i in range(args.warmup, n)) / args.steps

    sweep_t = tuple(int(v) for v in args.sweep_t.split(",")) if args.sweep_t else \
        I.DISPATCH_SWEEP_T
    for T in sweep_t:
        c = L.config(T, H, E, k, 2048)
        idx, w = I.uniform_routing(T, E, k, seed=rank, device=device)
        x = I.randn((T, H), 1.0, torch.bfloat16, rank, "x", device)
        counts = torch.empty(E, dtype=torch.int32, device=device)
        offsets = torch.empty(E + 1, dtype=torch.int32, device=device)
        rst = torch.empty(T * k, dtype=torch.int32, device=device)
        slot = torch.empty(T * k, dtype=torch.int32, device=device)
        xp = torch.empty((T * k, H), dtype=torch.bfloat16, device=device)
        ws = torch.empty(L.moe_dispatch_workspace_size(c), dtype=torch.uint8, device=device)
        perm_ms = timed(lambda: L.moe_dispatch(c, x, idx, counts, offsets, rst, slot, None, ws,
                                               stream))
        disp_ms = timed(lambda: L.moe_dispatch(c, x, idx, counts, offsets, rst, slot, xp, ws,
                                               stream))
        yp = xp.float()
        del xp
        out = torch.empty((T, H), dtype=torch.bfloat16, device=device)
        # y_perm (T*k*H*4 B, 235 MB at T = 1024) exceeds L2 by itself
        comb_ms = timed(lambda: L.moe_combine(c, yp, slot, w, None, out, 0, stream),
                        flush_l2=yp.numel() * 4 <= L2_BYTES)
        L.moe_check_errors(stream)
        copy_ms = max(disp_ms - perm_ms, 1e-6)
        copy_b = T * H * 2 + T * k * H * 2
        comb_b = T * k * H * 4 + T * H * 2 + T * k * 8
        rows.append({"T": T, "permutation_ms": round(perm_ms, 4),
                     "dispatch_copy_ms": round(copy_ms, 4),
                     "dispatch_copy_GBs": round(copy_b / copy_ms / 1e6, 1),
                     "dispatch_copy_frac_hbm": round(copy_b / copy_ms / 1e6 / hbm, 3),
                     "combine_ms": round(comb_ms, 4),
                     "combine_GBs": round(comb_b / comb_ms / 1e6, 1),
                     "combine_frac_hbm": round(comb_b / comb_ms / 1e6 / hbm, 3)})
        del yp, out, x
        torch.cuda.empty_cache()
    w1 = _dt.datetime.now()
    sampler.stop()
    big = rows[-1]
    line = {
        "metric": "dispatch / combine HBM GB/s, identity experts (H=7168, E=256, top-8 uniform)",
        "value": big["combine_GBs"], "unit": "GB/s", "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": big["combine_ms"], "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "bf16 rows, fp32 combine",
        "data": "synthetic (seeded N(0,1) rows, uniform routing)",
        "config": {"workload": "dispatch+combine sweep", "H": H, "E": E, "k": k,
                   "T": list(sweep_t),
                   "l2": "a 256 MB buffer is written before each timed permutation and "
                         "dispatch launch (their input x fits in L2 up to T = 8192); none "
                         "before the combine, whose input y_perm (T*k*H*4 B, 235 MB at "
                         "T = 1024) exceeds the 129 MB L2 by itself"},
        "peak": hbm, "peak_source": f"hbm_gbs of {src}", "sweep": rows,
        "gpu_launches": L.moe_launch_count() - n0,
        "clocks": sampler.summary(w0, w1),
    }
    if rank == 0:
        print(json.dumps(line), flush=True)


def main():
    args = parse()
    if args.oracle_one_core:  # child of the CPU baseline's single-core leg: no GPU
        oracle_one_core_child(args.oracle_one_core)
        return
    rank, world, local = dist_env()
    if world > 1:
        torch.distributed.init_process_group("gloo")
    torch.cuda.set_device(local)
    device = torch.device("cuda", local)
    wl = I.WORKLOADS[args.workload]
    if args.sweep and args.impl != "reference":
        run_sweep(args, rank, world, local, device)
    elif args.impl == "reference":
        run_reference(args, wl, rank, world, device)
    else:
        run_ours(args, wl, rank, world, local, device)
    if world > 1:
        torch.distributed.destroy_process_group()


if __name__ == "__main__":
    main()
