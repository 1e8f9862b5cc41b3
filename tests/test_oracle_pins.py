"""Pins of the fp64 oracle to facts outside itself (CPU only).

Each test checks the oracle against something the paper or the mathematics
fixes: closed forms, exact identities the paper proves, special cases that
reduce to a library routine (torch SDPA, torch rms_norm, torch silu), brute
force on tiny inputs, and invariants.  See the per-test docstrings for the
passage each one follows.
"""
import itertools
import json
import math
import os

import numpy as np
import pytest
import torch

from paper_2609_06712_gb300 import configs, inputs

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")


def small_cfg(**kw):
    """A small ragged layer: 3 x 5 x 7 grid = 105 tokens -> blocks of 64 and 41."""
    c = configs.get("tiny")
    c.update(T=3, Hh=5, Ww=7, H=2, r=16, keep=0.5, seed=11)
    c.update(kw)
    c["N"] = c["T"] * c["Hh"] * c["Ww"]
    return c


def draw(cfg, dtype=torch.float32):
    x = inputs.make_inputs(cfg, dtype=dtype)
    return {n: (None if t is None else t.float().numpy()) for n, t in x.items()}


# ---------------------------------------------------------------- RoPE --------

def rot_matrix(O, cfg, npairs, pos, dim):
    return np.stack([O.rotate(cfg, npairs, pos, e) for e in np.eye(dim)], axis=1)


def test_rope_orthogonal_and_group_property(oracle):
    """Sec. 3 (R(p) orthogonal) and App. B (R_r(p)^T R_r(q) = R_r(q - p), R(0) = I)."""
    O = oracle
    cfg = configs.get("tiny")
    rng = np.random.default_rng(0)
    for npairs in (8, 16, 32, 64):
        dim = 2 * npairs
        for _ in range(3):
            p = rng.integers(-40, 90, size=3).astype(float)
            q = rng.integers(-40, 90, size=3).astype(float)
            Rp = rot_matrix(O, cfg, npairs, p, dim)
            Rq = rot_matrix(O, cfg, npairs, q, dim)
            Rqp = rot_matrix(O, cfg, npairs, q - p, dim)
            np.testing.assert_allclose(Rp.T @ Rp, np.eye(dim), atol=1e-13)
            np.testing.assert_allclose(Rp.T @ Rq, Rqp, atol=1e-12)
        np.testing.assert_allclose(rot_matrix(O, cfg, npairs, np.zeros(3), dim), np.eye(dim), atol=0)


def test_rope_closed_forms(oracle):
    """Sec. 3 / Sec. 4.2 with the 44/42/42 split and theta = 10^4: the first pair of
    each axis turns by exactly its position (frequency theta^0 = 1), frequencies
    fall geometrically by theta^(-2/d_axis) within an axis, and the pair ->
    axis assignment follows the native ordering t | x | y."""
    O = oracle
    cfg = configs.get("tiny")
    pos = np.array([3.0, 5.0, 7.0])
    assert O.pair_angle(cfg, 0, pos) == 3.0           # first temporal pair
    assert O.pair_angle(cfg, 22, pos) == 5.0          # first height pair
    assert O.pair_angle(cfg, 43, pos) == 7.0          # first width pair
    for m in range(1, 22):
        ratio = O.pair_angle(cfg, m, pos) / O.pair_angle(cfg, m - 1, pos)
        assert ratio == pytest.approx(10000.0 ** (-2.0 / 44.0), rel=1e-14)
    for m in range(23, 43):
        ratio = O.pair_angle(cfg, m, pos) / O.pair_angle(cfg, m - 1, pos)
        assert ratio == pytest.approx(10000.0 ** (-2.0 / 42.0), rel=1e-14)
    # the truncated schedule at r = 32 is purely temporal: moving x, y does nothing
    assert all(O.pair_angle(cfg, m, [3, 0, 0]) == O.pair_angle(cfg, m, pos) for m in range(16))


def test_rope_is_complex_multiplication(oracle):
    """Sec. 4.5: RoPE acts on adjacent (even, odd) coordinate pairs; each pair is the
    complex number x + iy multiplied by exp(i angle) (a counter-clockwise turn)."""
    O = oracle
    cfg = configs.get("tiny")
    rng = np.random.default_rng(1)
    x = rng.standard_normal(128)
    pos = np.array([2.0, 9.0, 4.0])
    got = O.rotate(cfg, 64, pos, x)
    ang = np.array([O.pair_angle(cfg, m, pos) for m in range(64)])
    z = (x[0::2] + 1j * x[1::2]) * np.exp(1j * ang)
    np.testing.assert_allclose(got[0::2], z.real, atol=1e-14)
    np.testing.assert_allclose(got[1::2], z.imag, atol=1e-14)
    # coordinates past the truncation are untouched
    got_r = O.rotate(cfg, 8, pos, x)
    np.testing.assert_array_equal(got_r[16:], x[16:])
    np.testing.assert_allclose(got_r[:16], got[:16], atol=0)


def test_positions_t_major(oracle):
    """Sec. 3 notation: p = (t, x, y), L = T H W; flattening is t-major."""
    O = oracle
    cfg = small_cfg()
    for n in (0, 1, 6, 7, 34, 35, 36, 104):
        t, x, y = np.unravel_index(n, (cfg["T"], cfg["Hh"], cfg["Ww"]))
        np.testing.assert_array_equal(O.position(cfg, n), [t, x, y])
    cfg2 = small_cfg(pos_offset=(2, -1, 5))
    np.testing.assert_array_equal(O.position(cfg2, 36), np.array([1, 0, 1]) + [2, -1, 5])


# ---------------------------------------------------------------- mask --------

def test_num_keep_rounding(oracle):
    """n_keep = clamp(floor(keep * nKB + 0.5), 1, nKB) at the layer shapes."""
    O = oracle
    assert O.num_keep(configs.get("tiny")) == 2
    assert O.num_keep(configs.get("wan13b_480p")) == 51
    assert O.num_keep(configs.get("wan14b_720p")) == 118
    assert O.num_keep(configs.get("wan14b_720p_long")) == 231
    assert O.num_blocks(configs.get("wan14b_720p")) == 1182
    assert O.num_keep(small_cfg(keep=0.0)) == 1
    assert O.num_keep(small_cfg(keep=1.0)) == 2


def test_mask_is_the_best_subset_by_brute_force(oracle):
    """Top-k by exhaustive search: on distinct scores, the kept set is the unique
    n_keep-subset with the largest score sum."""
    O = oracle
    cfg = configs.get("tiny")
    x = draw(cfg)
    idx, scores, gap, tau = O.block_mask(cfg, x["q"], x["k"])
    nb, nk = scores.shape[-1], idx.shape[-1]
    for h in range(cfg["H"]):
        for i in range(nb):
            s = scores[0, h, i]
            best = max(itertools.combinations(range(nb), nk), key=lambda S: sum(s[list(S)]))
            assert list(best) == list(idx[0, h, i])
            srt = np.sort(s)[::-1]
            assert gap[0, h, i] == pytest.approx(srt[nk - 1] - srt[nk], abs=1e-15)


def wide_range(cfg, seed):
    """q, k with per-token magnitudes spread over six decades (10^-3 .. 10^3): pooled sums that
    cancel and round, the hard case for the fp32 evaluation of the block scores."""
    rng = np.random.default_rng(seed)
    shape = (cfg["B"], cfg["H"], cfg["N"], 128)
    scale = 10.0 ** rng.uniform(-3, 3, size=shape[:3] + (1,))
    return {n: (rng.standard_normal(shape) * scale).astype(np.float32) for n in ("q", "k")}


@pytest.mark.parametrize("geometry", ["flat", "cube"])
@pytest.mark.parametrize("dist", ["normal", "rmsnorm", "wide"])
def test_fp32_decision_within_the_near_tie_bound(oracle, dist, geometry):
    """The block mask is an fp32 decision.  tau / 2 is a rigorous bound on how far the
    oracle's fp32 evaluation of a score sits from the fp64 one (first-order error analysis of the
    rotation, the pairwise pooling, the division, the fma chain and the scale); checked at every
    (i, j) on three input distributions and both block geometries.  Rows with gap > tau then keep the
    same blocks in fp32 and in fp64.  The bound stays meaningful: below 1e-3 of the largest score."""
    O = oracle
    cfg = small_cfg(T=4, Hh=9, Ww=10, dist="rmsnorm" if dist == "rmsnorm" else "normal",
                    block_geometry=geometry)            # 360 tokens: 6 ragged chunks / 6 ragged cubes
    x = wide_range(cfg, 5) if dist == "wide" else draw(cfg)
    idx, s64, gap, tau = O.block_mask(cfg, x["q"], x["k"])
    idx32, s32 = O.block_mask_f32(cfg, x["q"], x["k"])
    bound = tau / 2
    assert (bound > 0).all() and bound.max() <= 1e-3 * np.abs(s64).max()
    err = np.abs(s32 - s64)
    assert (err <= bound[..., None]).all(), float((err / bound[..., None]).max())
    assert (err > 0).any()                              # fp32 really rounds here
    far = gap > tau
    assert far.any() and (idx32[far] == idx[far]).all()


def test_fp32_pooling_is_pairwise_in_slot_order(oracle):
    """The fp32 block mean is the pairwise sum (Higham, Accuracy and Stability of Numerical Algorithms,
    Sec. 4.2) of the block's slots in slot order, divided once by the token count; closed forms where
    the order decides the rounding.  Coordinate 0 of pair 0 (temporal, angle t = 0 in the first frame)
    is not rotated and every other coordinate is 0; the key block's mean in coordinate 0 is 1 (chunks)
    or 1/4 (cubes), so the score is the fp32 product of the pooled query value, that mean and
    fl(1/sqrt(128))."""
    O = oracle
    scale = np.float32(1.0 / math.sqrt(128.0))
    # chunks: 64 tokens of frame 0, token 0 holds 2^24 and tokens 1..63 hold 1.  Pairwise: the first
    # pair rounds 2^24 + 1 to 2^24 (ties to even) and every later level is exact, 2^24 + 62; the
    # sequential sum would lose all 63 ones and the exact sum is 2^24 + 63.
    cfg = small_cfg(T=2, Hh=8, Ww=8, H=1, keep=0.5)
    q = np.zeros((1, 1, cfg["N"], 128), np.float32)
    k = np.zeros_like(q)
    q[0, 0, :64, 0] = 1.0
    q[0, 0, 0, 0] = 2.0 ** 24
    k[0, 0, :, 0] = 1.0
    _, s32 = O.block_mask_f32(cfg, q, k)
    assert s32[0, 0, 0, 0] == np.float32(np.float32(2.0 ** 24 + 62) / np.float32(64)) * scale
    assert s32[0, 0, 0, 0] == np.float32(262144.96875) * scale
    assert np.float32(262144.0) * scale != np.float32(262144.96875) * scale
    # cubes: a 4 x 4 x 8 grid holds two cubes; in cube 0, (dx, dy) = (0, 0) holds 2^24, (0, 1) holds 1,
    # (1, 0) holds 2 (frame 0).  Slot 16 dt + 4 dx + dy: the pair (slot 0, slot 1) rounds 2^24 + 1 to
    # 2^24, the 2 joins at the third level exactly: 2^24 + 2.  With dx and dy swapped in the slot
    # number the pair would hold 2^24 + 2 and the 1 would round the total to 2^24 + 4.
    cfg = small_cfg(T=4, Hh=4, Ww=8, H=1, keep=0.5, block_geometry="cube")
    q = np.zeros((1, 1, cfg["N"], 128), np.float32)
    k = np.zeros_like(q)
    tok = lambda t, xx, y: (t * 4 + xx) * 8 + y
    q[0, 0, tok(0, 0, 0), 0] = 2.0 ** 24
    q[0, 0, tok(0, 0, 1), 0] = 1.0
    q[0, 0, tok(0, 1, 0), 0] = 2.0
    for xx in range(4):
        for y in range(4):
            k[0, 0, tok(0, xx, y), 0] = 1.0        # cube 0's key mean in coordinate 0: 16 / 64 = 1/4 exactly
    _, s32 = O.block_mask_f32(cfg, q, k)
    assert s32[0, 0, 0, 0] == np.float32(262144.03125 / 4) * scale     # (2^24 + 2) / 64, times 1/4
    assert np.float32(262144.0625 / 4) * scale != np.float32(262144.03125 / 4) * scale


def test_fp32_pooling_of_128_token_query_chunks(oracle):
    """A 128-token query chunk pools its 128 slots pairwise in slot order -- the top node of the two
    64-slot trees -- and divides once by its token count.  Frame 0 only (coordinate 0 of pair 0 is
    not rotated), every other coordinate 0, key block 0's mean in coordinate 0 is 1."""
    O = oracle
    scale = np.float32(1.0 / math.sqrt(128.0))
    # 128 tokens of frame 0: token 0 holds 2^24, tokens 1..127 hold 1.  The first 64-slot tree gives
    # 2^24 + 62 (its first pair rounds 2^24 + 1 to 2^24), the second 64 exactly, the top node
    # 2^24 + 126 (even, exact); divided by 128: 131072.984375, exact.  The sequential sum would keep
    # 2^24 (131072) and the exact sum 2^24 + 127 would round differently.
    cfg = small_cfg(T=2, Hh=8, Ww=16, H=1, keep=0.5, qblock=128)
    assert O.num_qblocks(cfg) == 2 and O.num_blocks(cfg) == 4
    q = np.zeros((1, 1, cfg["N"], 128), np.float32)
    k = np.zeros_like(q)
    q[0, 0, :128, 0] = 1.0
    q[0, 0, 0, 0] = 2.0 ** 24
    k[0, 0, :64, 0] = 1.0
    _, s32 = O.block_mask_f32(cfg, q, k)
    assert s32[0, 0, 0, 0] == np.float32(np.float32(2.0 ** 24 + 126) / np.float32(128)) * scale
    assert s32[0, 0, 0, 0] == np.float32(131072.984375) * scale
    assert np.float32(131072.0) * scale != np.float32(131072.984375) * scale
    # a ragged last chunk: 128 + 73 tokens in one frame; chunk 1 holds 73 tokens of value 1, so its
    # pooled value is 73 / 73 = 1 (a divisor of 128 would give 0.5703125)
    cfg = small_cfg(T=1, Hh=3, Ww=67, H=1, keep=0.5, qblock=128)
    assert cfg["N"] == 201 and O.num_qblocks(cfg) == 2
    q = np.zeros((1, 1, 201, 128), np.float32)
    k = np.zeros_like(q)
    q[0, 0, 128:, 0] = 1.0
    k[0, 0, :64, 0] = 1.0
    _, s32 = O.block_mask_f32(cfg, q, k)
    assert s32[0, 0, 1, 0] == np.float32(1.0) * scale


def test_fp32_decision_ties_and_brute_force(oracle):
    """The fp32 decision keeps, per row, the n_keep-subset with the largest fp32 score sum (brute
    force over all subsets on the tiny layer, whose fp32 scores are distinct), and breaks an exact
    tie toward the lower block: an all-zero query row keeps block 0."""
    O = oracle
    cfg = configs.get("tiny")
    x = draw(cfg)
    idx32, s32 = O.block_mask_f32(cfg, x["q"], x["k"])
    nb, nk = s32.shape[-1], idx32.shape[-1]
    for h in range(cfg["H"]):
        for i in range(nb):
            s = s32[0, h, i]
            assert len(set(s.tolist())) == nb
            best = max(itertools.combinations(range(nb), nk), key=lambda S: sum(s[list(S)]))
            assert list(best) == list(idx32[0, h, i])
    cfg = small_cfg(keep=0.5)                               # two blocks, n_keep = 1
    q = np.zeros((1, cfg["H"], cfg["N"], 128), np.float32)
    k = draw(cfg)["k"]
    idx32, s32 = O.block_mask_f32(cfg, q, k)
    assert (s32 == 0).all() and (idx32 == 0).all()


def test_mask_closed_form_single_token(oracle):
    """Pooling divides by the block's own token count (the ragged last block too);
    ties go to the lower key block.  q and k are zero except one token whose
    position is moved to the origin (R = I), so every score is known."""
    O = oracle
    cfg = small_cfg(keep=0.5)          # 2 blocks of 64 and 41 tokens, n_keep = 1
    n = 70                             # a token of the partial block
    t, xx, y = np.unravel_index(n, (cfg["T"], cfg["Hh"], cfg["Ww"]))
    cfg["pos_offset"] = (-int(t), -int(xx), -int(y))
    q = np.zeros((1, cfg["H"], cfg["N"], 128), np.float32)
    k = np.zeros_like(q)
    a = np.linspace(-1, 1, 128).astype(np.float32)
    q[0, :, n] = a
    k[0, :, n] = a
    idx, scores, gap, tau = O.block_mask(cfg, q, k)
    expect = float(a.astype(np.float64) @ a.astype(np.float64)) / 41 ** 2 / math.sqrt(128)
    assert scores[0, 0, 1, 1] == pytest.approx(expect, rel=1e-14)
    assert scores[0, 0, 0, 0] == 0 and scores[0, 0, 0, 1] == 0
    assert idx[0, 0, 1, 0] == 1        # the one positive score wins
    assert idx[0, 0, 0, 0] == 0        # all-zero row: the tie goes to block 0
    # a negative pooled score loses to the zero score of the other block
    k[0, :, n] = -a
    idx, scores, _, _ = O.block_mask(cfg, q, k)
    assert scores[0, 0, 1, 1] == pytest.approx(-expect, rel=1e-14)
    assert idx[0, 0, 1, 0] == 0
    # pooling acts on the ROTATED vectors: a query token and a key token at
    # different positions score a^T R(p_k - p_q) b (Eq. shiftinv)
    cfg["pos_offset"] = (0, 0, 0)
    nq, nk = 10, 100                   # blocks 0 (64 tokens) and 1 (41 tokens)
    q[:] = 0
    k[:] = 0
    b = np.cos(np.arange(128)).astype(np.float32)
    q[0, :, nq] = a
    k[0, :, nk] = b
    _, scores, _, _ = O.block_mask(cfg, q, k)
    rel = O.position(cfg, nk) - O.position(cfg, nq)
    expect = float(a.astype(np.float64) @ O.rotate(cfg, 64, rel, b)) / (64 * 41) / math.sqrt(128)
    assert scores[0, 0, 0, 1] == pytest.approx(expect, rel=1e-12)
    assert abs(expect - float(a @ b) / (64 * 41) / math.sqrt(128)) > 1e-3 * abs(expect)


def test_mask_keep_all_and_shift_invariance(oracle):
    """keep = 1 keeps every block in order; the pooled scores depend only on relative
    positions (Eq. shiftinv: each block mean turns by the same R(delta))."""
    O = oracle
    cfg = small_cfg(keep=1.0)
    x = draw(cfg)
    idx, _, _, _ = O.block_mask(cfg, x["q"], x["k"])
    assert (idx == np.arange(2)).all()
    cfg = configs.get("tiny")
    x = draw(cfg)
    _, s0, _, _ = O.block_mask(cfg, x["q"], x["k"])
    _, s1, _, _ = O.block_mask(dict(cfg, pos_offset=(5, -3, 11)), x["q"], x["k"])
    np.testing.assert_allclose(s1, s0, atol=1e-13)


# ---------------------------------------------------------------- sparse ------

def sdpa64(qr, kr, v, mask=None):
    t = lambda a: torch.from_numpy(np.ascontiguousarray(a, dtype=np.float64))
    return torch.nn.functional.scaled_dot_product_attention(
        t(qr), t(kr), t(v), attn_mask=None if mask is None else torch.from_numpy(mask)).numpy()


@pytest.mark.parametrize("grid", [(4, 16, 16), (3, 5, 7)])
def test_sparse_keep_all_is_dense_sdpa(oracle, grid):
    """T4: at keep ratio 1 the block-sparse branch is dense softmax attention
    softmax(Q K^T / sqrt d_h) V (Sec. 3), here torch's fp64 SDPA."""
    O = oracle
    cfg = small_cfg(T=grid[0], Hh=grid[1], Ww=grid[2], keep=1.0)
    x = draw(cfg)
    qr, kr = O.rope_full(cfg, x["q"]), O.rope_full(cfg, x["k"])
    idx, _, _, _ = O.block_mask(cfg, x["q"], x["k"])
    got = O.sparse_attn(cfg, qr, kr, x["v"], idx)
    np.testing.assert_allclose(got, sdpa64(qr, kr, x["v"]), rtol=1e-11, atol=1e-12)


def test_sparse_with_mask_is_masked_sdpa(oracle):
    """The sparse branch with a block mask equals SDPA with the equivalent boolean
    token mask; query rows of the ragged block use only real keys."""
    O = oracle
    cfg = small_cfg(T=4, Hh=9, Ww=10, keep=0.34)     # 360 tokens: 6 blocks, last has 40
    x = draw(cfg)
    qr, kr = O.rope_full(cfg, x["q"]), O.rope_full(cfg, x["k"])
    idx, _, _, _ = O.block_mask(cfg, x["q"], x["k"])
    N, bs = cfg["N"], cfg["block"]
    mask = np.zeros((1, cfg["H"], N, N), dtype=bool)
    for h in range(cfg["H"]):
        for i in range(idx.shape[2]):
            for j in idx[0, h, i]:
                mask[0, h, i * bs:(i + 1) * bs, j * bs:(j + 1) * bs] = True
    got = O.sparse_attn(cfg, qr, kr, x["v"], idx)
    np.testing.assert_allclose(got, sdpa64(qr, kr, x["v"], mask), rtol=1e-11, atol=1e-12)
    sel = O.sparse_attn(cfg, qr, kr, x["v"], idx, qblocks=[1, 5])
    np.testing.assert_array_equal(sel[:, :, 64:128], got[:, :, 64:128])
    assert np.isnan(sel[:, :, :64]).all()


# ---------------------------------------------------------------- cube blocks -

def cube_ids(T, Hh, Ww):
    """Cube of every token by numpy: (t // 4, x // 4, y // 4), numbered t-major over the cube grid."""
    t, x, y = np.meshgrid(np.arange(T), np.arange(Hh), np.arange(Ww), indexing="ij")
    nx, ny = -(-Hh // 4), -(-Ww // 4)
    return (((t // 4) * nx + x // 4) * ny + y // 4).reshape(-1)


def test_cube_blocks_partition_the_grid(oracle):
    """Cube geometry: every token lies in exactly one 4 x 4 x 4 cube of the latent grid, the cube
    count is the product of the per-axis cube counts, and an edge cube holds the product of its
    per-axis extents min(4, extent - 4 c)."""
    O = oracle
    cfg = small_cfg(T=5, Hh=9, Ww=13, block_geometry="cube")
    ids = O.block_of(cfg)
    np.testing.assert_array_equal(ids, cube_ids(5, 9, 13))
    assert O.num_blocks(cfg) == 2 * 3 * 4
    ext = lambda n: [min(4, n - 4 * c) for c in range(-(-n // 4))]
    want = np.array([a * b * c for a in ext(5) for b in ext(9) for c in ext(13)])
    np.testing.assert_array_equal(np.bincount(ids, minlength=24), want)
    assert O.num_keep(dict(cfg, keep=0.25)) == 6


def test_cube_pooled_scores_by_numpy(oracle):
    """Cube geometry: the block scores are the means of the rotated q / k over each cube's real
    tokens (numpy bincount over the cube ids), dotted and scaled by 1/sqrt(d_h)."""
    O = oracle
    cfg = small_cfg(T=5, Hh=9, Ww=13, block_geometry="cube", keep=0.25)
    x = draw(cfg)
    _, scores, _, _ = O.block_mask(cfg, x["q"], x["k"])
    ids = cube_ids(5, 9, 13)
    cnt = np.bincount(ids)
    for h in range(cfg["H"]):
        qr, kr = O.rope_full(cfg, x["q"])[0, h], O.rope_full(cfg, x["k"])[0, h]
        qb = np.stack([np.bincount(ids, weights=qr[:, d]) for d in range(128)], axis=1) / cnt[:, None]
        kb = np.stack([np.bincount(ids, weights=kr[:, d]) for d in range(128)], axis=1) / cnt[:, None]
        np.testing.assert_allclose(scores[0, h], qb @ kb.T / math.sqrt(128), rtol=1e-11, atol=1e-13)


def test_cube_keep_all_is_dense_and_mask_is_shift_invariant(oracle):
    """Cube geometry at keep = 1 is dense attention (torch fp64 SDPA) whatever the tiling; the cube
    scores, like the chunk scores, depend only on relative positions (Eq. shiftinv)."""
    O = oracle
    cfg = small_cfg(T=5, Hh=6, Ww=7, block_geometry="cube", keep=1.0)
    x = draw(cfg)
    qr, kr = O.rope_full(cfg, x["q"]), O.rope_full(cfg, x["k"])
    idx, _, _, _ = O.block_mask(cfg, x["q"], x["k"])
    assert (idx == np.arange(O.num_blocks(cfg))).all()
    got = O.sparse_attn(cfg, qr, kr, x["v"], idx)
    np.testing.assert_allclose(got, sdpa64(qr, kr, x["v"]), rtol=1e-11, atol=1e-12)
    cfg = dict(cfg, keep=0.3)
    _, s0, _, _ = O.block_mask(cfg, x["q"], x["k"])
    _, s1, _, _ = O.block_mask(dict(cfg, pos_offset=(5, -3, 11)), x["q"], x["k"])
    np.testing.assert_allclose(s1, s0, atol=1e-13)


def test_cube_sparse_equals_chunks_of_the_cube_ordered_sequence(oracle):
    """On a grid of whole cubes, sorting the tokens by cube turns every cube into one contiguous
    64-token chunk: the cube-geometry sparse branch equals the chunk-geometry branch run on the
    permuted q^r, k^r, v with the same block mask, permuted back."""
    O = oracle
    cfg = small_cfg(T=4, Hh=8, Ww=12, block_geometry="cube", keep=0.5)
    x = draw(cfg)
    qr, kr, v = O.rope_full(cfg, x["q"]), O.rope_full(cfg, x["k"]), x["v"]
    nb = O.num_blocks(cfg)
    assert nb == 6
    rng = np.random.default_rng(5)
    idx = np.sort(np.stack([[rng.choice(nb, 3, replace=False) for _ in range(nb)]
                            for _ in range(cfg["H"])]), axis=-1)[None].astype(np.int32)
    got = O.sparse_attn(cfg, qr, kr, v, idx)
    perm = np.argsort(cube_ids(4, 8, 12), kind="stable")
    flat = dict(cfg, block_geometry="flat")
    pf = O.sparse_attn(flat, qr[:, :, perm], kr[:, :, perm], v[:, :, perm], idx)
    back = np.empty_like(pf)
    back[:, :, perm] = pf
    np.testing.assert_allclose(got, back, rtol=1e-13, atol=1e-14)
    # a random cube mask differs from the chunk mask on the unpermuted sequence
    assert np.abs(got - O.sparse_attn(flat, qr, kr, v, idx)).max() > 1e-3


# ---------------------------------------------------------------- low-rank ----

def test_summary_form_equals_explicit_quadratic_form(oracle):
    """T2 / Prop. exact, Step 2: q~_p^T C equals sum_q (q~_p . k~_q) v_q."""
    O = oracle
    cfg = small_cfg(T=2, Hh=6, Ww=9, r=32)
    x = draw(cfg)
    C, z = O.lowrank_summary(cfg, x["k"], x["v"], x["P_k"])
    y = O.lowrank_readout(cfg, x["q"], x["P_q"], C)
    y2 = O.lowrank_explicit(cfg, x["q"], x["k"], x["v"], x["P_q"], x["P_k"])
    np.testing.assert_allclose(y, y2, rtol=1e-10, atol=1e-10)
    kt = O.lowrank_features(cfg, x["k"], x["P_k"])
    np.testing.assert_allclose(z, kt.sum(axis=2), rtol=1e-12, atol=1e-12)


@pytest.mark.parametrize("r", [16, 64])
def test_even_odd_split_evaluation_equals_interleaved(oracle, r):
    """T3 / Sec. 4.5: P's rows taken as the even rows then the odd rows, SiLU applied to both halves,
    element i of the first half rotated with element i of the second half by pair i's angle, and the
    result put back in interleaved order, is the oracle's interleaved feature vector (numpy matmuls;
    r = 64 spans temporal and height pairs)."""
    O = oracle
    cfg = small_cfg(r=r, T=2, Hh=3, Ww=4)
    x = draw(cfg)
    want = O.lowrank_features(cfg, x["k"], x["P_k"])
    P, k = x["P_k"].astype(np.float64), x["k"].astype(np.float64)
    got = np.empty_like(want)
    for n in range(cfg["N"]):
        pos = O.position(cfg, n)
        ang = np.array([O.pair_angle(cfg, m, pos) for m in range(r // 2)])
        for h in range(cfg["H"]):
            ue, uo = P[h, 0::2] @ k[0, h, n], P[h, 1::2] @ k[0, h, n]
            ae, ao = ue / (1 + np.exp(-ue)), uo / (1 + np.exp(-uo))
            got[0, h, n, 0::2] = ae * np.cos(ang) - ao * np.sin(ang)
            got[0, h, n, 1::2] = ae * np.sin(ang) + ao * np.cos(ang)
    np.testing.assert_allclose(got, want, rtol=1e-12, atol=1e-13)


def test_features_identity_projection_reduces_to_silu_then_rope(oracle):
    """With r = d_h and P = I the feature map of Eq. (qklr) is R(p) SiLU(x): torch's
    SiLU, then the full RoPE; the inside variant is SiLU(R(p) x)."""
    O = oracle
    cfg = small_cfg(r=128)
    x = draw(cfg)
    P = np.broadcast_to(np.eye(128, dtype=np.float32), (cfg["H"], 128, 128)).copy()
    silu = torch.nn.functional.silu(torch.from_numpy(x["k"]).double()).numpy()
    got = O.lowrank_features(cfg, x["k"], P)
    want = np.stack([np.stack([O.rotate(cfg, 64, O.position(cfg, n), silu[0, h, n])
                               for n in range(cfg["N"])]) for h in range(cfg["H"])])[None]
    np.testing.assert_allclose(got, want, rtol=1e-13, atol=1e-14)
    inside = O.lowrank_features(cfg, x["k"], P, rope_mode=O.ROPE_INSIDE)
    want_in = torch.nn.functional.silu(torch.from_numpy(O.rope_full(cfg, x["k"]))).numpy()
    np.testing.assert_allclose(inside, want_in, rtol=1e-13, atol=1e-14)
    none = O.lowrank_features(cfg, x["k"], P, rope_mode=O.ROPE_NONE)
    np.testing.assert_allclose(none, silu, rtol=1e-13, atol=1e-14)


def test_projection_is_a_matmul(oracle):
    """With RoPE removed the feature map is SiLU(x P^T) (torch matmul + silu)."""
    O = oracle
    cfg = small_cfg(r=48)
    x = draw(cfg)
    got = O.lowrank_features(cfg, x["q"], x["P_q"], rope_mode=O.ROPE_NONE)
    q = torch.from_numpy(x["q"]).double()
    P = torch.from_numpy(x["P_q"]).double()
    want = torch.nn.functional.silu(torch.einsum("bhnd,hrd->bhnr", q, P)).numpy()
    np.testing.assert_allclose(got, want, rtol=1e-12, atol=1e-13)


ACTS = ["silu", "identity", "tanh", "relu", "gelu"]


def test_activation_pins(oracle):
    """The feature maps of the activation ablation (Tab. abl_activation) against closed forms:
    phi(x) - phi(-x) = x for SiLU (sigma(x) + sigma(-x) = 1), ReLU and GELU (Phi(x) + Phi(-x) = 1);
    SiLU(ln 3) = (3/4) ln 3; tanh odd, tanh(ln 2) = 3/5 and tanh(x) = 2 sigma(2x) - 1 with
    sigma(2x) = SiLU(2x) / 2x; GELU(1) = Phi(1) from the normal table and x Phi(x) on a grid
    (scipy's ndtr, an implementation independent of the C library's erf)."""
    O = oracle
    xs = np.linspace(-6.0, 6.0, 49)
    phi = {n: np.array([O.activation(n, v) for v in xs]) for n in ACTS}
    for n in ("silu", "relu", "gelu"):
        np.testing.assert_allclose(phi[n] - phi[n][::-1], xs, rtol=0, atol=1e-14)
    np.testing.assert_array_equal(phi["identity"], xs)
    np.testing.assert_array_equal(phi["relu"], np.where(xs > 0, xs, 0.0))
    assert O.activation("silu", math.log(3.0)) == pytest.approx(0.75 * math.log(3.0), abs=1e-15)
    np.testing.assert_allclose(phi["tanh"], -phi["tanh"][::-1], rtol=0, atol=1e-16)
    assert O.activation("tanh", math.log(2.0)) == pytest.approx(0.6, abs=1e-15)
    nz = xs != 0
    sig2 = np.array([O.activation("silu", 2 * v) / (2 * v) for v in xs[nz]])
    np.testing.assert_allclose(phi["tanh"][nz], 2 * sig2 - 1, rtol=0, atol=1e-14)
    assert O.activation("gelu", 1.0) == pytest.approx(0.8413447460685429, abs=1e-15)
    special = pytest.importorskip("scipy.special")
    np.testing.assert_allclose(phi["gelu"], xs * special.ndtr(xs), rtol=1e-14, atol=1e-15)


def closed_form_act(name):
    special = pytest.importorskip("scipy.special")
    return {"silu": lambda a: a / (1.0 + np.exp(-a)), "identity": lambda a: a, "tanh": np.tanh,
            "relu": lambda a: np.maximum(a, 0.0), "gelu": lambda a: a * special.ndtr(a)}[name]


@pytest.mark.parametrize("act", ACTS)
def test_features_apply_the_chosen_activation(oracle, act):
    """With r = d_h and P = I the features of Eq. (qklr) are R(p) phi(x) (outside), phi(R(p) x)
    (inside) and phi(x) (none), for every feature map of Tab. abl_activation."""
    O = oracle
    cfg = small_cfg(r=128, lowrank_act=act)
    x = draw(cfg)
    phi = closed_form_act(act)
    P = np.broadcast_to(np.eye(128, dtype=np.float32), (cfg["H"], 128, 128)).copy()
    k = x["k"].astype(np.float64)
    none = O.lowrank_features(cfg, x["k"], P, rope_mode=O.ROPE_NONE)
    np.testing.assert_allclose(none, phi(k), rtol=1e-13, atol=1e-14)
    inside = O.lowrank_features(cfg, x["k"], P, rope_mode=O.ROPE_INSIDE)
    np.testing.assert_allclose(inside, phi(O.rope_full(cfg, x["k"])), rtol=1e-13, atol=1e-14)
    outside = O.lowrank_features(cfg, x["k"], P)
    pk = phi(k)
    want = np.stack([np.stack([O.rotate(cfg, 64, O.position(cfg, n), pk[0, h, n])
                               for n in range(cfg["N"])]) for h in range(cfg["H"])])[None]
    np.testing.assert_allclose(outside, want, rtol=1e-13, atol=1e-14)


def test_identity_activation_is_rotary_linear_attention(oracle):
    """Identity feature map, r = d_h, P = I: the summary form is plain (unnormalised) linear
    attention on the fully rotated q and k, y = R q (R k)^T V (numpy matmuls); and the inside
    placement equals the outside one, since a rotation commutes with the identity."""
    O = oracle
    cfg = small_cfg(r=128, lowrank_act="identity")
    x = draw(cfg)
    P = np.broadcast_to(np.eye(128, dtype=np.float32), (cfg["H"], 128, 128)).copy()
    C, _ = O.lowrank_summary(cfg, x["k"], x["v"], P)
    y = O.lowrank_readout(cfg, x["q"], P, C)
    qr, kr = O.rope_full(cfg, x["q"]), O.rope_full(cfg, x["k"])
    want = qr @ np.swapaxes(kr, -1, -2) @ x["v"].astype(np.float64)
    np.testing.assert_allclose(y, want, rtol=1e-10, atol=1e-9)
    Ci, _ = O.lowrank_summary(cfg, x["k"], x["v"], P, rope_mode=O.ROPE_INSIDE)
    np.testing.assert_allclose(Ci, C, rtol=1e-12, atol=1e-11)


def shift_residual(O, cfg, x, rope_mode, delta):
    a = O.forward(cfg, x["q"], x["k"], x["v"], x["P_q"], x["P_k"], x["gate"], rope_mode=rope_mode)
    b = O.forward(dict(cfg, pos_offset=delta), x["q"], x["k"], x["v"], x["P_q"], x["P_k"],
                  x["gate"], rope_mode=rope_mode)
    assert (a["kv_idx"] == b["kv_idx"]).all()
    return np.linalg.norm(a["o"] - b["o"]) / np.linalg.norm(a["o"])


def test_module_shift_invariance_outside_vs_inside(oracle):
    """T5 / T6 (Eq. shiftinv, Prop. exact vs Prop. inside, Sec. 5.2 shift test): with
    RoPE outside SiLU the whole module is invariant under a uniform shift of all
    positions; with RoPE inside it is not; with no RoPE the low-rank branch is
    position-blind.  The shift moves t, the only axis the r = 16 schedule sees."""
    O = oracle
    cfg = small_cfg(T=4, Hh=6, Ww=8, r=16, keep=0.25)
    x = draw(cfg)
    x["gate"] = np.full((1, cfg["N"]), 0.9, np.float32)   # make the low-rank branch matter
    out = shift_residual(O, cfg, x, O.ROPE_OUTSIDE, (7, 3, -2))
    ins = shift_residual(O, cfg, x, O.ROPE_INSIDE, (7, 3, -2))
    non = shift_residual(O, cfg, x, O.ROPE_NONE, (7, 3, -2))
    assert out < 1e-12
    assert non < 1e-12
    assert ins > 1e-3


@pytest.mark.parametrize("act", ["identity", "tanh", "relu", "gelu"])
def test_shift_invariance_for_every_activation(oracle, act):
    """T5 for each feature map of Tab. abl_activation: with RoPE outside the activation the
    module is shift-invariant whatever phi is (Prop. exact needs only a pointwise map before the
    rotation); inside, a nonlinear phi breaks it (Prop. inside) while the identity does not."""
    O = oracle
    cfg = small_cfg(T=4, Hh=6, Ww=8, r=16, keep=0.25, lowrank_act=act)
    x = draw(cfg)
    x["gate"] = np.full((1, cfg["N"]), 0.9, np.float32)
    assert shift_residual(O, cfg, x, O.ROPE_OUTSIDE, (7, 3, -2)) < 1e-12
    ins = shift_residual(O, cfg, x, O.ROPE_INSIDE, (7, 3, -2))
    assert ins < 1e-12 if act == "identity" else ins > 1e-3


def test_truncation_bound(oracle):
    """T7 / Prop. truncation-bound: for full-dimensional position-free features,
    |Phi^T R(q-p) Psi - Phi_<=r^T R_r(q-p) Psi_<=r| <= ||Phi_>r|| ||Psi_>r||,
    with equality to zero at r = d_h."""
    O = oracle
    cfg = configs.get("tiny")
    rng = np.random.default_rng(3)
    for _ in range(20):
        phi, psi = rng.standard_normal(128), rng.standard_normal(128)
        d = rng.integers(-20, 20, size=3).astype(float)
        full = phi @ O.rotate(cfg, 64, d, psi)
        for r in (16, 32, 64, 128):
            tr = phi[:r] @ O.rotate(cfg, r // 2, d, psi[:r].copy())[:r]
            bound = np.linalg.norm(phi[r:]) * np.linalg.norm(psi[r:])
            assert abs(full - tr) <= bound + 1e-12
            if r == 128:
                assert abs(full - tr) < 1e-12


# ---------------------------------------------------------------- fusion ------

def test_fusion_identities(oracle):
    """T8 / Eq. (gate): g = 0 gives O = O^s exactly; O is affine in g with slope
    r_p O^lr, r_p = sqrt(mean O^s^2 + eps), and O^lr = RMSNorm(y) is torch's
    rms_norm of the readout; O^s = 0 leaves g sqrt(eps) O^lr."""
    O = oracle
    cfg = small_cfg(T=2, Hh=6, Ww=9, r=32)
    x = draw(cfg)
    C, _ = O.lowrank_summary(cfg, x["k"], x["v"], x["P_k"])
    rng = np.random.default_rng(4)
    o_s = (0.05 * rng.standard_normal(x["q"].shape)).astype(np.float32)
    N = cfg["N"]
    g0, g1, gh = (np.full((1, N), g, np.float32) for g in (0.0, 1.0, 0.5))
    o0 = O.lowrank_apply(cfg, x["q"], x["P_q"], C, g0, o_s)
    o1 = O.lowrank_apply(cfg, x["q"], x["P_q"], C, g1, o_s)
    oh = O.lowrank_apply(cfg, x["q"], x["P_q"], C, gh, o_s)
    np.testing.assert_allclose(o0, o_s.astype(np.float64), rtol=1e-15, atol=0)
    np.testing.assert_allclose(oh, 0.5 * (o0 + o1), rtol=1e-13, atol=1e-15)
    y = torch.from_numpy(O.lowrank_readout(cfg, x["q"], x["P_q"], C))
    olr = torch.nn.functional.rms_norm(y, (128,), eps=float(np.float32(1e-6))).numpy()
    osd = torch.from_numpy(o_s).double()
    rp = torch.sqrt(osd.pow(2).mean(-1, keepdim=True) + float(np.float32(1e-6))).numpy()
    np.testing.assert_allclose(o1 - o0, rp * olr, rtol=1e-11, atol=1e-14)
    zero = O.lowrank_apply(cfg, x["q"], x["P_q"], C, gh, np.zeros_like(o_s))
    np.testing.assert_allclose(zero, 0.5 * math.sqrt(float(np.float32(1e-6))) * olr, rtol=1e-11)


def test_default_gate_is_one_eighth(oracle):
    """Tab. (hyper) initialises the gate bias at -1.946, i.e. -ln 7 to 3 decimals, so the
    default gate sigmoid(b_g) is 1/8; gate = NULL must use it."""
    with open(os.path.join(GOLDEN, "paper_constants.json")) as f:
        gold = json.load(f)
    b = gold["gate_bias_init"]["value"]
    assert b == pytest.approx(-math.log(7.0), abs=5e-4)
    O = oracle
    cfg = small_cfg(T=1, Hh=8, Ww=8, r=16)
    x = draw(cfg)
    C, _ = O.lowrank_summary(cfg, x["k"], x["v"], x["P_k"])
    o_s = np.full(x["q"].shape, 0.1, np.float32)
    g = np.full((1, cfg["N"]), 1.0 / (1.0 + math.exp(-np.float32(b))), np.float32)
    a = O.lowrank_apply(cfg, x["q"], x["P_q"], C, None, o_s)
    bb = O.lowrank_apply(cfg, x["q"], x["P_q"], C, g, o_s)
    np.testing.assert_allclose(a, bb, rtol=1e-7)


# ------------------------------------------------------------------ token gate (Sec. fusion)


def test_gate_pins(oracle):
    """g = sigmoid(X w_g + b_g): with zero input the gate is sigmoid(b_g), 1/8 at the paper's initial bias;
    flipping the signs of w_g and b_g gives 1 - g; the logit is additive in X and moves by delta * w_d when
    one input feature moves by delta."""
    import json
    O = oracle
    b0 = json.load(open(os.path.join(os.path.dirname(__file__), "golden", "paper_constants.json")))[
        "gate_bias_init"]["value"]
    rng = np.random.default_rng(7)
    B, N, D = 2, 37, 96
    # multiples of 1/8 and 1/64: every product and the sums below are exact in fp32 and fp64
    X = (rng.integers(-16, 17, (B, N, D)) / 8.0).astype(np.float32)
    X2 = (rng.integers(-16, 17, (B, N, D)) / 8.0).astype(np.float32)
    w = (rng.integers(-8, 9, D) / 64.0).astype(np.float32)
    logit = lambda g: np.log(g / (1.0 - g))
    g = O.gate(X, w, b0)
    assert ((g > 0) & (g < 1)).all()
    assert np.abs(O.gate(np.zeros_like(X), w, b0) - 0.125).max() < 1e-4
    assert np.allclose(O.gate(X, -w, -b0), 1.0 - g, rtol=0, atol=1e-14)
    assert np.allclose(logit(O.gate(X + X2, w, b0)), logit(g) + logit(O.gate(X2, w, b0)) - b0, rtol=0, atol=1e-9)
    for d in (0, 41, D - 1):
        Xd = X.copy()
        Xd[:, :, d] += 0.5
        assert np.allclose(logit(O.gate(Xd, w, b0)) - logit(g), 0.5 * float(w[d]), rtol=0, atol=1e-9)


# ---------------------------------------------------------------- 128-token query blocks

def test_query_blocks_of_128_tokens(oracle):
    """qblock = 128 (the b_q = 128 / b_kv = 64 tiling of the block-sparse attentions the paper builds
    on): the query blocks are 128-token chunks, the last one ragged, and the key blocks stay 64-token
    chunks; unset, both are the 64-token chunks.  Cube geometry takes no query-block size."""
    O = oracle
    cfg = small_cfg(T=4, Hh=9, Ww=10, qblock=128)       # 360 tokens: query blocks 128, 128, 104
    assert O.num_qblocks(cfg) == 3 and O.num_blocks(cfg) == 6
    assert np.array_equal(O.qblock_of(cfg), np.arange(360) // 128)
    assert np.array_equal(O.block_of(cfg), np.arange(360) // 64)
    base = small_cfg(T=4, Hh=9, Ww=10)
    assert O.num_qblocks(base) == 6 and np.array_equal(O.qblock_of(base), np.arange(360) // 64)
    with pytest.raises(ValueError):
        O.make_config(small_cfg(T=4, Hh=8, Ww=8, qblock=128, block_geometry="cube"))


def test_query_block_scores_are_count_weighted_chunk_scores(oracle):
    """A 128-token query block's pooled mean is the count-weighted mean of its two 64-token halves'
    means, and the score is linear in q_bar, so its score row is the count-weighted mean of the two
    halves' rows (ragged tail: 104 = 64 + 40 tokens).  Its kept set is its n_keep best key blocks,
    ties to the lower id, ascending."""
    O = oracle
    cfg = small_cfg(T=4, Hh=9, Ww=10, keep=0.34)
    x = draw(cfg)
    _, s64, _, _ = O.block_mask(cfg, x["q"], x["k"])
    idx, s128, _, _ = O.block_mask(dict(cfg, qblock=128), x["q"], x["k"])
    assert idx.shape == (1, cfg["H"], 3, 2) and s128.shape == (1, cfg["H"], 3, 6)
    cnt = np.bincount(np.arange(cfg["N"]) // 64).astype(np.float64)
    for I in range(3):
        a, b = 2 * I, 2 * I + 1
        want = (cnt[a] * s64[:, :, a] + cnt[b] * s64[:, :, b]) / (cnt[a] + cnt[b])
        np.testing.assert_allclose(s128[:, :, I], want, rtol=1e-12, atol=1e-14)
    for h in range(cfg["H"]):
        for I in range(3):
            order = sorted(range(6), key=lambda j: (-s128[0, h, I, j], j))
            assert list(idx[0, h, I]) == sorted(order[:2])


def test_query_block_sparse_branch_shares_the_mask_row(oracle):
    """Every query of a 128-token block attends to that block's kept key blocks: the sparse branch
    equals, bit for bit, the 64-token-chunk branch under the mask whose rows 2I and 2I + 1 are row I;
    query-block selection and the full forward follow the 128-token blocks; keep = 1 is dense SDPA."""
    O = oracle
    cfg = small_cfg(T=4, Hh=9, Ww=10, keep=0.34, dist="normal_gate")
    c128 = dict(cfg, qblock=128)
    x = draw(cfg)
    qr, kr = O.rope_full(cfg, x["q"]), O.rope_full(cfg, x["k"])
    idx, _, _, _ = O.block_mask(c128, x["q"], x["k"])
    got = O.sparse_attn(c128, qr, kr, x["v"], idx)
    dup = np.ascontiguousarray(np.repeat(idx, 2, axis=2)[:, :, :6])
    np.testing.assert_array_equal(got, O.sparse_attn(cfg, qr, kr, x["v"], dup))
    sel = O.sparse_attn(c128, qr, kr, x["v"], idx, qblocks=[1])
    np.testing.assert_array_equal(sel[:, :, 128:256], got[:, :, 128:256])
    assert np.isnan(sel[:, :, :128]).all() and np.isnan(sel[:, :, 256:]).all()
    fw = O.forward(c128, x["q"], x["k"], x["v"], x["P_q"], x["P_k"], x["gate"])
    np.testing.assert_array_equal(fw["kv_idx"], idx)
    np.testing.assert_array_equal(fw["o_s"], got)
    fs = O.forward(c128, x["q"], x["k"], x["v"], x["P_q"], x["P_k"], x["gate"], qblocks=[2])
    np.testing.assert_array_equal(fs["o"][:, :, 256:], fw["o"][:, :, 256:])
    assert np.isnan(fs["o"][:, :, :256]).all()
    full = dict(c128, keep=1.0)
    idx1, _, _, _ = O.block_mask(full, x["q"], x["k"])
    np.testing.assert_allclose(O.sparse_attn(full, qr, kr, x["v"], idx1), sdpa64(qr, kr, x["v"]),
                               rtol=1e-11, atol=1e-12)


def test_out_proj_pins(oracle):
    """Output projection (Alg. 1, last step): the heads concatenated per token in head order, times
    W_o^T, plus the bias.  Pinned by a numpy matmul of the concatenation on small integer inputs
    (exact in fp64) with a rectangular W_o, by the head selection (W_o's identity block at head h
    returns head h's rows), and by O = 0 giving the bias."""
    O = oracle
    rng = np.random.default_rng(7)
    B, H, N, dh, dm = 2, 3, 5, 4, 7
    Oh = rng.integers(-3, 4, size=(B, H, N, dh)).astype(np.float64)
    W = rng.integers(-2, 3, size=(dm, H * dh)).astype(np.float32)
    b = rng.integers(-5, 6, size=dm).astype(np.float32)
    cat = np.concatenate([Oh[:, h] for h in range(H)], axis=-1)          # [B, N, H*dh]
    assert (O.out_proj(Oh, W, b) == cat @ W.T.astype(np.float64) + b).all()
    assert (O.out_proj(Oh, W) == cat @ W.T.astype(np.float64)).all()
    for h in range(H):
        Wh = np.zeros((dh, H * dh), np.float32)
        Wh[:, h * dh:(h + 1) * dh] = np.eye(dh)
        assert (O.out_proj(Oh, Wh) == Oh[:, h]).all()
    assert (O.out_proj(np.zeros_like(Oh), W, b) == np.broadcast_to(b, (B, N, dm))).all()
    part = O.out_proj(Oh, W, b, rows=[1, 3])
    assert np.isnan(part[:, [0, 2, 4]]).all() and (part[:, [1, 3]] == (cat @ W.T.astype(np.float64) + b)[:, [1, 3]]).all()
