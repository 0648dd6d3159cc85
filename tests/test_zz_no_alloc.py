"""moe_dispatch_noalloc: the dispatch for callers that cannot allocate device memory.

Some callers (a plugin inside a framework that owns all device memory, a
serving loop with a fixed memory plan, a latency-critical path where an
allocation may synchronise the device) can pass no workspace. This checks,
through the C ABI, that the allocation-free variant gives exactly what the
workspace-taking moe_dispatch gives, on two calls in a row (the second one
reuses the library's scratch array as the first left it), that repeated
calls leave the device's free memory unchanged, and that inputs larger than
its fixed scratch are refused.
"""

import ctypes

import numpy as np
import pytest
import torch

from paper_2603_02376_gb300 import _lib as L

pytestmark = pytest.mark.gpu
DEV = "cuda"


def _routing(T, E, k, seed):
    rng = np.random.default_rng(seed)
    return np.stack([rng.permutation(E)[:k] for _ in range(T)]).astype(np.int32)


def _outputs(T, E, k, H):
    return dict(counts=torch.full((E,), -1, dtype=torch.int32, device=DEV),
                offsets=torch.full((E + 1,), -1, dtype=torch.int32, device=DEV),
                rst=torch.full((T * k,), -1, dtype=torch.int32, device=DEV),
                slot=torch.full((T * k,), -1, dtype=torch.int32, device=DEV),
                xp=torch.zeros((T * k, H), dtype=torch.bfloat16, device=DEV))


def test_dispatch_noalloc_matches_dispatch_twice():
    L.load()
    for call, (T, E, k, H) in enumerate([(4096, 256, 8, 7168), (777, 64, 6, 256)]):
        cfg = L.config(T, H, E, k, 128, 0, 1, 1)
        g = torch.Generator(device=DEV).manual_seed(call)
        x = torch.randn((T, H), generator=g, device=DEV).to(torch.bfloat16)
        idx = torch.from_numpy(_routing(T, E, k, 10 + call)).to(DEV)
        ref = _outputs(T, E, k, H)
        ws = torch.empty(L.moe_dispatch_workspace_size(cfg), dtype=torch.uint8, device=DEV)
        L.moe_dispatch(cfg, x, idx, ref["counts"], ref["offsets"], ref["rst"], ref["slot"],
                       ref["xp"], ws)
        got = _outputs(T, E, k, H)
        L.moe_dispatch_noalloc(cfg, x, idx, got["counts"], got["offsets"], got["rst"],
                               got["slot"], got["xp"])
        L.moe_check_errors()
        for name in ref:   # integer and copy outputs: bit for bit
            assert torch.equal(got[name], ref[name]), f"call {call}: {name} differs"


def test_dispatch_noalloc_leaves_free_device_memory_unchanged():
    L.load()
    T, E, k, H = 2048, 256, 8, 512
    cfg = L.config(T, H, E, k, 128, 0, 1, 1)
    g = torch.Generator(device=DEV).manual_seed(7)
    x = torch.randn((T, H), generator=g, device=DEV).to(torch.bfloat16)
    idx = torch.from_numpy(_routing(T, E, k, 99)).to(DEV)
    out = _outputs(T, E, k, H)
    args = (cfg, x, idx, out["counts"], out["offsets"], out["rst"], out["slot"], out["xp"])
    L.moe_dispatch_noalloc(*args)   # the first call on the device finds the scratch array
    torch.cuda.synchronize()
    free0 = torch.cuda.mem_get_info()[0]
    for _ in range(3):
        L.moe_dispatch_noalloc(*args)
    torch.cuda.synchronize()
    assert torch.cuda.mem_get_info()[0] == free0
    L.moe_check_errors()


def test_dispatch_noalloc_rejects_inputs_beyond_its_scratch():
    L.load()
    E = 256
    T = (L.MOE_DISPATCH_NOALLOC_MAX_ENTRIES // E) * 128   # one chunk too many
    cfg = L.config(T, 128, E, 8, 128)
    p = ctypes.c_void_p(0x1000)
    st = L.load().moe_dispatch_noalloc(ctypes.byref(cfg), p, p, p, p, p, p, None, None)
    assert st == L.MOE_ERR_UNSUPPORTED
