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


def check_mask(gpu_idx, orc_idx, scores, gap, tau, nB):
    """Mask parity.  Rows whose oracle gap (n_keep-th minus (n_keep+1)-th score)
    exceeds the fp32 error bound tau must match bit for bit.  On the remaining
    near-tie rows more than one kept set is a correct fp32 answer: the GPU row
    must be a valid top-n_keep (ascending, distinct, in range, and no kept score
    below an unkept one by more than tau).  Returns the boolean [B,H,nQB] map of
    rows where the GPU mask equals the oracle's."""
    gpu_idx = np.asarray(gpu_idx)
    near = gap <= tau
    equal = (gpu_idx == orc_idx).all(axis=-1)
    bad = ~equal & ~near
    assert not bad.any(), f"{int(bad.sum())} non-near-tie mask rows differ, first at {np.argwhere(bad)[0]}"
    for b, h, i in np.argwhere(~equal):
        row = gpu_idx[b, h, i]
        assert (np.diff(row) > 0).all() and row[0] >= 0 and row[-1] < nB, "invalid mask row"
        s = scores[b, h, i]
        kept = np.zeros(nB, bool)
        kept[row] = True
        if (~kept).any():
            assert s[kept].min() >= s[~kept].max() - tau[b, h, i], "mask row is not a top-k"
    return equal


def to_np(t):
    return t.detach().float().cpu().numpy()


def dev(x, device="cuda"):
    return None if x is None else x.to(device).contiguous()


def rows_of_blocks(blocks, block, N):
    rows = np.zeros(N, bool)
    for i in blocks:
        rows[i * block:(i + 1) * block] = True
    return rows
