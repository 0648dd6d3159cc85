"""Host logic of bench.py and of the input generator (no GPU).

* algorithmic(): the per-stage bytes and flops of the tiny layer, worked out by
  hand in the comments, for bf16 and for the block-scaled FP8 form;
* the traffic captures' source hash: unchanged by comment edits, changed by a
  code edit; a capture keyed to another hash is not used;
* the block-scaled FP8 weight generator: shapes, exponent range, no NaN code;
* the per-kernel roofline: its bound is the longer of bytes / bandwidth and
  flops / peak, with fractions against the measured and nominal peaks;
* the CPU baseline's single-core leg (a child process with one BLAS thread).
"""

import json
import os
import shutil

import pytest
import torch

import bench
from paper_2603_02376_gb300 import inputs as I


def test_algorithmic_bytes_of_the_tiny_layer_by_hand():
    # T=64, H=256, E=8, k=2 (R=128 packed rows), I=128, no shared expert, 8 experts touched
    b, f = bench.algorithmic(I.TINY, 8, fused_gather=False, fp8=0)
    assert b["router"] == 64 * 256 * 2 + 8 * 256 * 4 + 64 * 8 * 4 == 43008
    assert b["gate"] == 64 * 8 * 4 + 64 * 2 * 8 == 3072
    assert b["permute"] == 128 * 12 == 1536
    assert b["dispatch"] == 64 * 256 * 2 + 128 * 256 * 2 == 98304        # x read, x_perm written
    # W13 of 8 experts (8 x 2*128*256 bf16), x_perm read, h written
    assert b["gemm1"] == 8 * 131072 + 65536 + 32768 == 1146880
    # W2 of 8 experts, h read, y_perm written in fp32
    assert b["gemm2"] == 8 * 65536 + 32768 + 131072 == 688128
    assert b["shared_gemm1"] == 0 and b["shared_gemm2"] == 0
    # y_perm read, bf16 out written, slot row + weight per entry
    assert b["combine"] == 131072 + 32768 + 1024 == 164864
    assert f["router"] == 2 * 64 * 8 * 256
    assert f["gemm1"] == 2 * 128 * 256 * 256 and f["gemm2"] == 2 * 128 * 128 * 256
    # a fused dispatch has no copy of its own (GEMM1 gathers the same rows)
    bf, _ = bench.algorithmic(I.TINY, 8, fused_gather=True, fp8=0)
    assert bf["dispatch"] == 0 and bf["gemm1"] == b["gemm1"]


def test_algorithmic_bytes_of_the_block_scaled_form_by_hand():
    b, _ = bench.algorithmic(I.TINY, 8, fused_gather=True, fp8=2)
    # x -> e4m3 (bf16 read + byte written) and one exponent per 128 values of a row
    assert b["dispatch"] == 64 * 256 * 3 + 64 * 2 == 49280
    # W13 bytes plus one exponent per 128x128 block (2 x 2 per expert), x_q rows and
    # their exponents, h written in bf16, then h quantized (bf16 read, byte + exponent)
    assert b["gemm1"] == 8 * (65536 + 4) + 32768 + 256 + 32768 + (128 * 128 * 3 + 128) == 639392
    assert bench.scale_bytes(10, 7168, 1) == 40 and bench.scale_bytes(10, 7168, 2) == 560
    assert bench.scale_bytes(10, 7168, 0) == 0


def _copy_sources(dst):
    for p in bench.GEMM_SOURCES:
        os.makedirs(os.path.join(dst, os.path.dirname(p)), exist_ok=True)
        shutil.copy(os.path.join(bench.ROOT, p), os.path.join(dst, p))


def test_source_hash_follows_code_not_comments(tmp_path, monkeypatch):
    _copy_sources(tmp_path)
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    h0 = bench.source_sha()
    src = os.path.join(tmp_path, bench.GEMM_SOURCES[0])
    text = open(src).read()
    open(src, "w").write("// a new comment line\n\n" + text.replace("\n", "  // trailing\n", 3))
    assert bench.source_sha() == h0
    open(src, "w").write(text.replace("constexpr int BM = 128;", "constexpr int BM = 64;", 1))
    assert bench.source_sha() != h0


def test_traffic_capture_of_another_source_is_not_used(tmp_path, monkeypatch):
    key = I.DECODE.name
    f = tmp_path / "traffic.json"
    monkeypatch.setattr(bench, "TRAFFIC_FILE", str(f))
    f.write_text(json.dumps({key: {"source_sha": "0" * 16, "dram_bytes_per_launch": 123}}))
    assert bench.measured_traffic(key, 0) is None
    f.write_text(json.dumps({key: {"source_sha": bench.source_sha(), "dram_bytes_per_launch": 123}}))
    assert bench.measured_traffic(key, 0) == 123.0
    assert bench.measured_traffic(key, 2) is None          # no block-scaled entry
    assert bench.measured_traffic(key, 0, pack_in_gemm1=True) is None   # another launch form


def test_block_scaled_weight_generator():
    codes, exps = I.e4m3_block_codes((256, 384), 0, "W13b", "cpu", extra=3)
    assert codes.shape == (256, 384) and codes.dtype == torch.uint8
    assert exps.shape == (2, 3) and exps.dtype == torch.uint8
    assert set(exps.unique().tolist()) <= {113, 114}
    mag = codes & 0x7F
    assert int(mag.min()) >= I.E4M3_CODE_LO and int(mag.max()) <= I.E4M3_CODE_HI  # no NaN code
    again = I.e4m3_block_codes((256, 384), 0, "W13b", "cpu", extra=3)
    assert torch.equal(again[0], codes) and torch.equal(again[1], exps)   # seeded
    wl = I.Workload("t", T=4, H=256, E=2, k=1, I=128, I_shared=128, n_groups=1, topk_groups=1,
                    gate=I.GATE_SOFTMAX, normalize=0, route_scale=1.0)
    W13, k13, W2, k2 = I.fp8_block_expert_weights(wl, 0, "cpu")
    assert W13.shape == (2, 256, 256) and k13.shape == (2, 2, 2)
    assert W2.shape == (2, 256, 128) and k2.shape == (2, 2, 1)
    Ws13, ks13, Ws2, ks2 = I.fp8_block_shared_weights(wl, 0, "cpu")
    assert Ws13.shape == (256, 256) and ks13.shape == (2, 2) and ks2.shape == (2, 1)


def test_kernel_roofline_takes_the_longer_bound():
    # 16.45 GB and 4.33 TFLOP in 3.9 ms against 6776 GB/s and 1699.8 TFLOP/s sustained:
    # the bytes need 2.43 ms, the flops 2.55 ms, so the kernel is tensor-bound
    r = bench.kernel_roofline(16.45e9, 4.33e12, 3.9e-3, 6776.3, 1699.8, 1910.6, "measured", "bf16")
    assert r["bound"] == "tensor" and r["unit"] == "TFLOP/s"
    assert r["achieved"] == pytest.approx(4.33e12 / 3.9e-3 / 1e12, rel=1e-3)
    assert r["frac"] == pytest.approx(4.33e12 / 3.9e-3 / 1e12 / 1699.8, abs=1e-4)
    assert r["frac"] == pytest.approx(r["t_flops_ms"] / r["t_measured_ms"], abs=1e-3)
    assert r["hbm"]["frac_nominal_8TBs"] == pytest.approx(16.45e9 / 3.9e-3 / 1e9 / 8000, abs=1e-4)
    # decode: 14.7 GB and 0.1 TFLOP in 1.96 ms is bandwidth-bound
    d = bench.kernel_roofline(14.7e9, 0.1e12, 1.96e-3, 6776.3, 1699.8, 1910.6, "measured", "bf16")
    assert d["bound"] == "hbm" and d["unit"] == "GB/s" and d["peak"] == 6776.3
    assert d["frac"] == pytest.approx(14.7e9 / 1.96e-3 / 1e9 / 6776.3, abs=1e-4)
    # e4m3 takes twice the bf16 peak (the caller scales it) and names its own dtype
    e = bench.kernel_roofline(8.4e9, 4.33e12, 2.3e-3, 6776.3, 2 * 1699.8, 2 * 1910.6, "measured",
                              "e4m3")
    assert e["tensor"]["frac_nominal"] == pytest.approx(4.33e12 / 2.3e-3 / 1e12 / 4500, abs=1e-4)


def test_oracle_single_core_leg_runs_in_a_child():
    d = I.layer_inputs(I.TINY, seed=0, device="cpu")
    r = bench.oracle_one_core(I.TINY, d, 4)
    assert "error" not in r, r
    assert r["cores"] == 1 and r["value"] > 0 and r["sample"].startswith("4 sampled tokens")


if __name__ == "__main__":
    pytest.main([__file__, "-q"])
