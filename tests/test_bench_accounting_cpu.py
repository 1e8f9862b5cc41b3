"""The bench's work accounting (CPU only): block sizes, the sparse FLOPs counted from
the mask, the low-rank FLOPs and the summary's bytes.

They are checked against independent counts: the oracle's block ids (numpy
bincount), a brute-force loop over a random mask, the dense closed form
4 B H L^2 d_h (App. D) when every block is kept, and the layer sizes of the
Wan2.1-14B 720p layer (75600 tokens, 1182 blocks, the last of 16 tokens)."""
import os

import numpy as np
import pytest
import torch

import bench
from paper_2609_06712_gb300 import configs


@pytest.mark.parametrize("name", ["tiny", "wan13b_480p", "wan14b_720p", "wan14b_720p_long"])
def test_chunk_block_sizes(name):
    cfg = configs.get(name)
    sizes = bench.block_sizes(cfg)
    N = cfg["N"]
    assert len(sizes) == -(-N // 64) and sum(sizes) == N
    assert all(s == 64 for s in sizes[:-1]) and 1 <= sizes[-1] <= 64


def test_720p_layer_sizes():
    sizes = bench.block_sizes(configs.get("wan14b_720p"))
    assert len(sizes) == 1182 and sizes[-1] == 16


@pytest.mark.parametrize("grid", [(5, 9, 13), (4, 8, 12), (1, 3, 2), (21, 45, 80)])
def test_cube_block_sizes_match_the_oracle_block_ids(oracle, grid):
    T, Hh, Ww = grid
    cfg = configs.get("tiny", T=T, Hh=Hh, Ww=Ww, block_geometry="cube")
    sizes = bench.block_sizes(cfg)
    if T * Hh * Ww <= 20000:
        ids = oracle.block_of(cfg)
        assert sizes == np.bincount(ids, minlength=len(sizes)).tolist()
    cubes = -(-T // 4) * -(-Hh // 4) * -(-Ww // 4)
    assert len(sizes) == cubes and sum(sizes) == T * Hh * Ww and max(sizes) <= 64


def test_sparse_flops_equal_a_brute_force_count():
    rng = np.random.default_rng(5)
    cfg = configs.get("tiny", T=3, Hh=7, Ww=11)             # 231 tokens: blocks of 64, 64, 64, 39
    sizes = bench.block_sizes(cfg)
    nB, n_keep, B, H = len(sizes), 2, 2, 3
    kv = np.stack([np.sort(rng.choice(nB, n_keep, replace=False)) for _ in range(B * H * nB)])
    kv = kv.reshape(B, H, nB, n_keep).astype(np.int32)
    want = 0
    for b in range(B):
        for h in range(H):
            for i in range(nB):
                for j in kv[b, h, i]:
                    want += 4 * 128 * sizes[i] * sizes[j]     # QK^T and PV, 2 flops per multiply-add
    assert bench.sparse_flops_from_mask(torch.from_numpy(kv), sizes) == float(want)


def test_every_block_kept_is_the_dense_closed_form():
    cfg = configs.get("wan14b_720p")
    sizes = bench.block_sizes(cfg)
    nB, H = len(sizes), cfg["H"]
    kv = torch.arange(nB, dtype=torch.int32).expand(1, H, nB, nB)
    dense = 4.0 * 1 * H * cfg["N"] ** 2 * 128
    assert bench.sparse_flops_from_mask(kv, sizes) == dense
    assert dense == pytest.approx(117.05e12, rel=1e-4)


def test_lowrank_flops_and_summary_bytes_at_720p():
    B, H, N, r = 1, 40, 75600, 32
    # App. D: 8 B H L d_h r; half of it is the summary, half the readout (~49.5 GFLOP each)
    assert bench.lowrank_flops(B, H, N, 128, r) == pytest.approx(2 * 49.54e9, rel=1e-3)
    # the summary reads k and v once in bf16: 2 B H N d_h 2 bytes
    assert bench.summary_bytes(B, H, N, 128) == pytest.approx(1.548e9, rel=1e-3)


def test_accounting_uses_the_printed_complexity_formulas():
    """App. D's coefficients (tests/golden/paper_constants.json): C_sparse = 4 B H L^2 (1-S) d_h,
    C_lowrank = 8 B H L d_h r, and with C_fusion = 2 B H L d_h the overhead
    eta = (C_lowrank + C_fusion) / C_sparse = (2r + 0.5) / (L (1 - S))."""
    import json
    import os
    gold = json.load(open(os.path.join(os.path.dirname(__file__), "golden", "paper_constants.json")))["flops"]
    B, H, L, d, r = 1, 40, 75600, 128, 32
    assert bench.lowrank_flops(B, H, L, d, r) == gold["lowrank_coeff"] * B * H * L * d * r
    sizes = bench.block_sizes(configs.get("wan14b_720p"))
    nB = len(sizes)
    kv = torch.arange(nB, dtype=torch.int32).expand(B, H, nB, nB)
    assert bench.sparse_flops_from_mask(kv, sizes) == gold["sparse_coeff"] * B * H * L ** 2 * d
    for keep in (0.05, 0.1, 0.2):
        S = 1.0 - keep
        c_sparse = gold["sparse_coeff"] * B * H * L ** 2 * (1 - S) * d
        eta = (bench.lowrank_flops(B, H, L, d, r) + gold["fusion_coeff"] * B * H * L * d) / c_sparse
        assert eta == pytest.approx((gold["eta_r_coeff"] * r + gold["eta_const"]) / (L * (1 - S)), rel=1e-12)


def test_sparse_traffic_follows_the_committed_capture(tmp_path, monkeypatch):
    """roofline.traffic comes from the committed ncu summary only while the kernel's sources are the
    ones that capture was taken on: a summary recording the sources' own hash gives its figure, one
    recording another hash, or lacking the two fields, gives None (the bench then reports
    traffic: null).  The committed summary carries both fields."""
    import hashlib
    text = open(bench.SPARSE_PROFILE).read()
    assert "traffic_bytes_per_head_token: " in text and "kernel_sources_sha256: " in text
    h = hashlib.sha256()
    for f in bench.SPARSE_SOURCES:
        h.update(open(os.path.join(bench.ROOT, "paper_2609_06712_gb300", "csrc", f), "rb").read())
    current = tmp_path / "current.md"
    current.write_text("notes\ntraffic_bytes_per_head_token: 996.5\nkernel_sources_sha256: " + h.hexdigest() + "\n")
    monkeypatch.setattr(bench, "SPARSE_PROFILE", str(current))
    assert bench.sparse_traffic_per_head_token() == 996.5
    stale = tmp_path / "stale.md"
    stale.write_text("traffic_bytes_per_head_token: 996.5\nkernel_sources_sha256: " + "0" * 64 + "\n")
    monkeypatch.setattr(bench, "SPARSE_PROFILE", str(stale))
    assert bench.sparse_traffic_per_head_token() is None
    bare = tmp_path / "bare.md"
    bare.write_text("kernel_sources_sha256: " + h.hexdigest() + "\n")
    monkeypatch.setattr(bench, "SPARSE_PROFILE", str(bare))
    assert bench.sparse_traffic_per_head_token() is None


def test_sparse_flops_with_128_token_query_chunks():
    """With 128-token query chunks each mask row weighs its chunk's size: brute force over a random
    mask on a ragged 585-token layer (query chunks 128 x 4 + 73, key blocks 64 x 9 ... 9)."""
    cfg = configs.get("tiny", T=5, Hh=9, Ww=13, H=2)
    ks, qs = bench.block_sizes(cfg), bench.block_sizes(cfg, 128)
    assert sum(ks) == sum(qs) == 585 and len(qs) == 5 and qs[-1] == 73
    rng = np.random.default_rng(3)
    kv = torch.from_numpy(np.sort(np.stack([[rng.choice(len(ks), 3, replace=False) for _ in qs]
                                            for _ in range(2)])[None], axis=-1).astype(np.int32))
    want = 0.0
    for h in range(2):
        for i, qsz in enumerate(qs):
            want += 4 * 128 * qsz * sum(ks[j] for j in kv[0, h, i].tolist())
    assert bench.sparse_flops_from_mask(kv, ks, qsizes=qs) == want
