"""The tile-packed token-row layout, checked on the host (no GPU needed).

The layer keeps its bf16 and row-scaled e4m3 token operands (x_perm, and
GEMM2's h or hq) as blocks the expert GEMMs load with one bulk copy per
stage. moe_testing_tiled_chunk runs the address function the kernels use.
These tests check its properties against the layout's definition: every chunk
of every packed row lands in a distinct 16-byte slot of the buffer of
rows + 16 E rows; a tile's k-block is one contiguous block of n_pad x 8
chunks, with n_pad the tile's rows rounded up to 16; inside it, row i's chunk
j sits at i * 8 + (j xor (i mod 8)), the 128-byte swizzle of the MMA's
K-major operand (the order the tile-packed weights use); and the block of
(tile, k-block) follows the tile's blocks in k order.
"""

import os

import numpy as np
import pytest

from paper_2603_02376_gb300 import _lib as L


@pytest.fixture(scope="module")
def lib():
    if not os.path.exists(L.LIB_PATH):
        from paper_2603_02376_gb300 import build
        build.build_library()
    return L.load()


def layout(counts, tile, cpr):
    """Chunk index of every (packed row, chunk) through the library, with the
    row's expert, tile, row in tile and the tile's padded row count."""
    offs = np.concatenate([[0], np.cumsum(counts)]).astype(int)
    rows = []
    for e, cnt in enumerate(counts):
        for r in range(offs[e], offs[e] + cnt):
            idx = [L.moe_testing_tiled_chunk(r, e, offs[e], cnt, tile, cpr, c) for c in range(cpr)]
            l = r - offs[e]
            t, i = divmod(l, tile)
            m = min(tile, cnt - t * tile)
            rows.append((e, t, i, (m + 15) // 16 * 16, idx))
    return offs, rows


CASES = [
    ([5, 0, 17, 1], 32, 16),                  # ragged, an empty expert
    ([300, 256, 257, 0, 1, 16], 256, 8),      # tile edges: 256 + 44, 256 + 1
    ([128, 129, 16, 144, 273, 0, 60], 144, 16),
    ([0, 0, 40], 144, 24),                    # leading empty experts
    ([64, 33, 7], 32, 8),
]


@pytest.mark.parametrize("counts,tile,cpr", CASES)
def test_chunks_are_distinct_and_inside_the_padded_buffer(lib, counts, tile, cpr):
    offs, rows = layout(counts, tile, cpr)
    allidx = np.array([i for *_, idx in rows for i in idx])
    assert len(np.unique(allidx)) == len(allidx), "two chunks share a slot"
    assert allidx.min() >= 0
    assert allidx.max() < (offs[-1] + 16 * len(counts)) * cpr, "outside rows + 16 E rows"


@pytest.mark.parametrize("counts,tile,cpr", CASES)
def test_each_tile_block_is_contiguous_and_swizzled(lib, counts, tile, cpr):
    offs, rows = layout(counts, tile, cpr)
    blocks = {}
    for e, t, i, n_pad, idx in rows:
        for kb in range(cpr // 8):
            blocks.setdefault((e, t, kb, n_pad), []).append((i, idx[8 * kb: 8 * kb + 8]))
    for (e, t, kb, n_pad), members in blocks.items():
        base = min(min(c) for _, c in members) - min(i for i, _ in members) * 8
        # the block is n_pad x 8 chunks long; row i's chunk j at i * 8 + (j ^ (i % 8))
        for i, chunks in members:
            for j, c in enumerate(chunks):
                assert c - base == i * 8 + (j ^ (i % 8)), (e, t, kb, i, j)
        assert max(max(c) for _, c in members) < base + n_pad * 8
        if kb > 0:
            prev = blocks[(e, t, kb - 1, n_pad)]
            prev_base = min(min(c) for _, c in prev) - min(i for i, _ in prev) * 8
            assert base == prev_base + n_pad * 8, "k-blocks of a tile are not consecutive"


@pytest.mark.parametrize("counts,tile,cpr", CASES)
def test_tiles_start_at_the_padded_row(lib, counts, tile, cpr):
    """Tile t of expert e starts at padded row off[e] + 16 e + t * tile, and its
    rows (rounded up to 16) end before the next expert's first tile."""
    offs, rows = layout(counts, tile, cpr)
    for e, t, i, n_pad, idx in rows:
        if i == 0:
            assert min(idx) == (offs[e] + 16 * e + t * tile) * cpr
            end = (offs[e] + 16 * e + t * tile + n_pad) * cpr
            assert end <= (offs[e + 1] + 16 * (e + 1)) * cpr


def test_bad_arguments_are_refused(lib):
    import ctypes
    out = ctypes.c_int64()
    f = lib.moe_testing_tiled_chunk
    assert f(5, 0, 0, 5, 32, 8, 0, ctypes.byref(out)) == L.MOE_ERR_INVALID_ARG   # r past the expert
    assert f(0, 0, 0, 5, 24, 8, 0, ctypes.byref(out)) == L.MOE_ERR_INVALID_ARG   # tile % 16
    assert f(0, 0, 0, 5, 32, 12, 0, ctypes.byref(out)) == L.MOE_ERR_INVALID_ARG  # chunks % 8
    assert f(0, 0, 0, 5, 32, 8, 8, ctypes.byref(out)) == L.MOE_ERR_INVALID_ARG   # c >= chunks
    assert f(0, -1, 0, 5, 32, 8, 0, ctypes.byref(out)) == L.MOE_ERR_INVALID_ARG  # e < 0
    assert f(0, 0, 0, 5, 32, 8, 0, None) == L.MOE_ERR_INVALID_ARG                # no output
    assert f(3, 1, 2, 4, 32, 8, 5, ctypes.byref(out)) == L.MOE_OK
