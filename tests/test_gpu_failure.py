"""Failure detection on the GPU without a fault, a trap or a hang.

Every barrier wait in the grouped GEMM is bounded. A testing entry point runs
the grouped expert FFN with one producer fill of CTA 0 never issued -- a
barrier that nothing will complete -- and a short wait limit. The kernel must
give up, latch MOE_ERR_TIMEOUT, wait (bounded) for its own copies and MMAs,
free its tensor memory and return within a few limits; moe_check_errors()
must report the timeout once; and the same context must then run the normal
path correctly.
"""

import time

import numpy as np
import pytest
import torch

from paper_2603_02376_gb300 import _lib as L

pytestmark = pytest.mark.gpu
DEV = "cuda"


def _case(counts, H, Iw, seed):
    g = torch.Generator(device=DEV).manual_seed(seed)
    E = len(counts)
    rows = int(sum(counts))
    offs = torch.tensor(np.concatenate([[0], np.cumsum(counts)]), dtype=torch.int32, device=DEV)
    xp = (torch.randn((rows, H), generator=g, device=DEV)).to(torch.bfloat16)
    W13 = (torch.randn((E, 2 * Iw, H), generator=g, device=DEV) * 0.05).to(torch.bfloat16)
    W2 = (torch.randn((E, H, Iw), generator=g, device=DEV) * 0.05).to(torch.bfloat16)
    return rows, offs, xp, W13, W2


@pytest.mark.parametrize("counts,stall_fill", [([40, 3, 0, 17], 3), ([300, 200], 0),
                                               ([4] * 64, 5)])
def test_stalled_wait_times_out_and_context_survives(counts, stall_fill):
    L.load()
    H, Iw = 512, 256
    rows, offs, xp, W13, W2 = _case(counts, H, Iw, seed=len(counts))
    E = len(counts)
    y = torch.zeros((rows, H), dtype=torch.float32, device=DEV)
    ws = torch.zeros(L.moe_expert_ffn_workspace_size(rows, Iw), dtype=torch.uint8, device=DEV)
    L.moe_check_errors()                       # start from a clear error word
    limit_ns = 100_000_000                     # 0.1 s per wait
    t0 = time.time()
    st = L.moe_testing_expert_ffn_stall(rows, H, Iw, E, xp, offs, W13, W2, y, ws, stall_fill,
                                        limit_ns)
    assert st == L.MOE_OK                      # the launches themselves succeed
    with pytest.raises(L.MoeError) as exc:
        L.moe_check_errors()                   # synchronises: the kernels have returned
    assert exc.value.status == L.MOE_ERR_TIMEOUT
    assert time.time() - t0 < 10.0             # a few 0.1 s limits, not a hang
    L.moe_check_errors()                       # the error word was cleared: reported once

    # the same context runs the normal path correctly afterwards
    y2 = torch.zeros_like(y)
    L.moe_expert_ffn(rows, H, Iw, E, xp, offs, W13, W2, y2, ws)
    L.moe_check_errors()
    e0 = int(offs[1].item())
    if e0 > 0:
        xh = xp[:e0].double()
        g = xh @ W13[0, :Iw].double().T
        u = xh @ W13[0, Iw:].double().T
        h = (g / (1 + torch.exp(-g)) * u).to(torch.bfloat16).double()
        ref = h @ W2[0].double().T
        err = (y2[:e0].double() - ref).abs().max().item()
        assert err <= 1e-3 * ref.abs().max().item() + 1e-3


@pytest.mark.parametrize("axis", [0, 1])
def test_pipelined_forward_failing_after_the_fork_joins_its_pack_stream(axis):
    """A pipelined forward that fails after forking its pack stream must still
    make the caller's stream wait for the pack stream's work before returning.

    The failure is injected on the host (moe_testing_fail_stage): the second
    stage call fails with MOE_ERR_CUDA, after the first one has put routing and
    packing work on the pack stream. Eagerly, the error comes back and the same
    stream then runs a correct forward. Under CUDA-graph capture, ending the
    capture succeeds only if every stream forked from the capturing stream was
    joined back into it; the captured graph is never launched."""
    from paper_2603_02376_gb300 import inputs as I

    L.load()
    wl = I.TINY
    d = I.layer_inputs(wl, seed=0, device=DEV)
    cfg = L.config_of(wl)
    ex = L.exec_config(overlap=1, chunk_axis=axis, chunk_tokens=16, n_expert_chunks=4)
    W = L.weights_struct(d["Wr"], d["bias"], d["W13"], d["W2"], d["Ws13"], d["Ws2"])
    ws = torch.zeros(L.moe_workspace_size(cfg, ex), dtype=torch.uint8, device=DEV)
    out = torch.zeros((wl.T, wl.H), dtype=torch.bfloat16, device=DEV)
    s = torch.cuda.Stream()
    L.moe_check_errors()

    L.moe_testing_fail_stage(1)
    with pytest.raises(L.MoeError) as exc:
        L.moe_layer_forward(cfg, ex, W, d["x"], out, None, ws, s)
    assert exc.value.status == L.MOE_ERR_CUDA
    L.moe_layer_forward(cfg, ex, W, d["x"], out, None, ws, s)   # injector is off again
    ws2 = torch.zeros_like(ws)
    ref = torch.zeros_like(out)
    L.moe_layer_forward(cfg, ex, W, d["x"], ref, None, ws2, s)  # a fresh workspace
    L.moe_check_errors(s)
    assert torch.equal(out, ref)

    g = torch.cuda.CUDAGraph()
    L.moe_testing_fail_stage(1)
    with torch.cuda.stream(s):
        g.capture_begin()
        try:
            with pytest.raises(L.MoeError):
                L.moe_layer_forward(cfg, ex, W, d["x"], out, None, ws, s)
        finally:
            g.capture_end()   # raises if the pack stream was left forked
    L.moe_testing_fail_stage(-1)
    del g
    torch.cuda.synchronize()
