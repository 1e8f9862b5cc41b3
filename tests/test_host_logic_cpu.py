"""Host-side integer logic of the kernels, checked exhaustively on the CPU."""
import numpy as np


def test_cube_index_reciprocal_division_is_exact():
    """The sparse kernel finds a cube's coordinates as floor((a + 0.5) * fl(1/d)) in fp32 instead of
    an integer division a / d.  That equals a / d for every block id a and divisor d the library
    accepts (at most 7008 blocks), checked here for all pairs in fp32 arithmetic."""
    a = np.arange(7008, dtype=np.int64)
    af = a.astype(np.float32) + np.float32(0.5)
    for d in range(1, 7009):
        r = np.float32(1.0 / d)                       # the host's fp64 reciprocal rounded to fp32
        q = np.floor(af * r).astype(np.int64)         # fp32 product, truncated
        assert np.array_equal(q, a // d), d


def test_cube_slots_match_the_oracle_block_ids(oracle, tmp_path):
    """The kernels' cube indexing (cube_origin, cube_token in csrc/common.cuh, compiled for the host)
    against the oracle's independent block numbering on grids with ragged edge cubes: every token sits
    in exactly one slot, the slot's block is the oracle's block of that token, and slot
    i = 16 dt + 4 dx + dy holds the token at offset (dt, dx, dy) from the cube's corner."""
    import os
    import shutil
    import subprocess

    from paper_2609_06712_gb300 import configs

    nvcc = shutil.which("nvcc") or "/usr/local/cuda/bin/nvcc"
    if not os.path.exists(nvcc):
        import pytest
        pytest.skip("nvcc not available")
    here = os.path.dirname(os.path.abspath(__file__))
    exe = str(tmp_path / "cube_index")
    subprocess.check_call([nvcc, "-std=c++17", "-gencode", "arch=compute_103a,code=sm_103a", "-o", exe,
                           os.path.join(here, "cube_index_harness.cu")])
    for T, Hh, Ww in [(5, 9, 13), (4, 8, 12), (1, 3, 2), (7, 1, 1), (3, 17, 4), (21, 30, 52)]:
        out = subprocess.check_output([exe, str(T), str(Hh), str(Ww)], text=True)
        tab = np.array([[int(v) for v in line.split()] for line in out.splitlines()], dtype=np.int64)
        cfg = configs.get("tiny", T=T, Hh=Hh, Ww=Ww, block_geometry="cube")
        ids = oracle.block_of(cfg)
        N = T * Hh * Ww
        assert tab.shape == (-(-T // 4) * -(-Hh // 4) * -(-Ww // 4), 64)
        blocks, slots = np.nonzero(tab >= 0)
        toks = tab[blocks, slots]
        assert np.array_equal(np.sort(toks), np.arange(N))
        assert np.array_equal(ids[toks], blocks)
        t, x, y = toks // (Hh * Ww), (toks // Ww) % Hh, toks % Ww
        assert np.array_equal(slots, 16 * (t % 4) + 4 * (x % 4) + (y % 4))
