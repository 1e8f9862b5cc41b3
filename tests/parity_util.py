"""Helpers shared by the GPU parity tests: run the CUDA path through the C ABI,
compare against the oracle with the stated tolerances."""
import numpy as np
import torch

# Output tolerances: bf16 storage -> max-abs 2e-2 and relative L2 5e-3; fp32
# validation mode -> relative L2 1e-5.
BF16_MAX_ABS = 2e-2
BF16_REL_L2 = 5e-3
F32_REL_L2 = 1e-5


def rel_l2(a, b):
    a = np.asarray(a, np.float64)
    b = np.asarray(b, np.float64)
    return float(np.linalg.norm(a - b) / max(np.linalg.norm(b), 1e-300))


def assert_close(got, want, dtype_is_bf16, what, unit_rms=False):
    """rel-L2 and max-abs bars.  For the module's outputs (O, O^s: entries of
    order one or below) max-abs is absolute.  unit_rms=True measures max-abs in
    units of the reference's RMS, for fp32 intermediates whose entries are sums
    over the sequence (C, z: magnitude ~ sqrt(N))."""
    got = np.asarray(got, np.float64)
    want = np.asarray(want, np.float64)
    assert got.shape == want.shape, (what, got.shape, want.shape)
    assert np.isfinite(got).all(), f"{what}: non-finite values"
    rl = rel_l2(got, want)
    ma = float(np.abs(got - want).max()) if got.size else 0.0
    if unit_rms:
        ma /= max(float(np.sqrt(np.mean(want ** 2))), 1e-300)
    if dtype_is_bf16:
        assert rl <= BF16_REL_L2 and ma <= BF16_MAX_ABS, f"{what}: rel-L2 {rl:.3e}, max-abs {ma:.3e}"
    else:
        assert rl <= F32_REL_L2, f"{what}: rel-L2 {rl:.3e}"
    return rl, ma


# Gradients (backward pass) in bf16: rel-L2 as for the outputs, max-abs in units
# of the reference's largest magnitude -- gradient entries spread to ~10x their
# RMS, and one bf16 rounding of the largest is 2^-9 of it; the bar allows about
# five roundings' worth along the chain (rotated copies, O^s, the gradient).
BF16_GRAD_MAX_REL = 1e-2


def assert_close_grad(got, want, dtype_is_bf16, what):
    got = np.asarray(got, np.float64)
    want = np.asarray(want, np.float64)
    assert got.shape == want.shape, (what, got.shape, want.shape)
    assert np.isfinite(got).all(), f"{what}: non-finite values"
    rl = rel_l2(got, want)
    if dtype_is_bf16:
        ma = float(np.abs(got - want).max()) / max(float(np.abs(want).max()), 1e-300)
        assert rl <= BF16_REL_L2 and ma <= BF16_GRAD_MAX_REL, f"{what}: rel-L2 {rl:.3e}, max-abs/max {ma:.3e}"
    else:
        assert rl <= F32_REL_L2, f"{what}: rel-L2 {rl:.3e}"
    return rl


# Mask parity counts per checked layer, printed in the session summary (conftest):
# (label, rows, near-tie rows, rows where the fp32 decision differs from the fp64
# definition, rows where the GPU differs from the fp32 decision).
MASK_STATS = []


def check_mask(cfg, h, gpu_idx, label):
    """Mask parity.  Keeping the n_keep best blocks turns floating point into
    integers, so the block mask is an fp32 decision with every rounding fixed
    (the oracle's block_mask_f32 states the evaluation); the GPU mask must equal
    the oracle's fp32 decision on EVERY row, bit for bit.  That decision is in
    turn checked against the fp64 definition: equal on every row whose fp64
    gap (n_keep-th minus (n_keep+1)-th score) exceeds tau, the rigorous bound on
    the fp32 evaluation error; on the remaining near-tie rows a valid top-n_keep
    of the fp64 scores within tau.  Returns the fp64 (idx, scores, gap, tau)."""
    from oracle import oracle as O
    gpu_idx = np.asarray(gpu_idx)
    f32_idx, _ = O.block_mask_f32(cfg, h["q"], h["k"])
    idx, scores, gap, tau = O.block_mask(cfg, h["q"], h["k"])
    nB = scores.shape[-1]
    near = gap <= tau
    gpu_ne = (gpu_idx != f32_idx).any(axis=-1)
    f32_ne = (f32_idx != idx).any(axis=-1)
    rows = int(near.size)
    counts = (label, rows, int(near.sum()), int(f32_ne.sum()), int(gpu_ne.sum()))
    MASK_STATS.append(counts)
    msg = (f"{label}: {rows} rows, near-tie {counts[2]} ({100.0 * counts[2] / rows:.2f} %), "
           f"fp32 decision != fp64 definition {counts[3]}, GPU != fp32 decision {counts[4]}")
    assert not gpu_ne.any(), f"{msg}; first GPU difference at {np.argwhere(gpu_ne)[0]}"
    bad = f32_ne & ~near
    assert not bad.any(), f"{msg}; fp32 decision differs on a row with gap > tau at {np.argwhere(bad)[0]}"
    for b, hh, i in np.argwhere(f32_ne):
        row = f32_idx[b, hh, i]
        assert (np.diff(row) > 0).all() and row[0] >= 0 and row[-1] < nB, f"{msg}: invalid mask row"
        s = scores[b, hh, i]
        kept = np.zeros(nB, bool)
        kept[row] = True
        if (~kept).any():
            assert s[kept].min() >= s[~kept].max() - tau[b, hh, i], f"{msg}: mask row is not a top-k within tau"
    return idx, scores, gap, tau


def to_np(t):
    return t.detach().float().cpu().numpy()


def dev(x, device="cuda"):
    return None if x is None else x.to(device).contiguous()


def rows_of_blocks(blocks, block, N):
    rows = np.zeros(N, bool)
    for i in blocks:
        rows[i * block:(i + 1) * block] = True
    return rows
