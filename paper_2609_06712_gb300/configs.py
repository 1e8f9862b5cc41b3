"""Named layer shapes: Wan2.1-style video DiT attention layers.

Each entry is a plain dict of sizes and draw parameters -- no arithmetic of the
method.  ``keep`` is the fraction of key blocks kept per query block (90 %
sparsity -> 0.10).  The token grid is T x Hh x Ww latent frames / rows / cols.
"""

D_H = 128
BLOCK = 64
SPLIT = (44, 42, 42)   # d_t, d_x, d_y of the 3D RoPE
THETA = 10000.0

_BASE = dict(d_h=D_H, block=BLOCK, rope_split=SPLIT, rope_theta=THETA,
             eps_lr=1e-6, eps_fuse=1e-6, gate_bias=-1.946, pos_offset=(0, 0, 0))


def _cfg(name, B, H, T, Hh, Ww, keep, r, seed, dist, **kw):
    c = dict(_BASE)
    c.update(name=name, B=B, H=H, T=T, Hh=Hh, Ww=Ww, N=T * Hh * Ww, keep=keep, r=r,
             seed=seed, dist=dist)
    c.update(kw)
    return c


CONFIGS = {
    # tiny correctness case: 4x16x16 grid, 2 heads, 2 of 16 key blocks kept, r = 16
    "tiny": _cfg("tiny", 1, 2, 4, 16, 16, 0.125, 16, 0, "normal"),
    # Wan2.1-1.3B layer, 480p / 81 frames (21 x 30 x 52 latents), per-head RMS-normalised q, k
    "wan13b_480p": _cfg("wan13b_480p", 1, 12, 21, 30, 52, 0.10, 32, 1, "rmsnorm"),
    # Wan2.1-14B layer, 480p, RMS-normalised q, k with a per-channel gain ~ U(0.5, 1.5)
    "wan14b_480p": _cfg("wan14b_480p", 1, 40, 21, 30, 52, 0.10, 32, 2, "rmsnorm_gain"),
    # headline: Wan2.1-14B layer at 720p / 81 frames (21 x 45 x 80 latents)
    "wan14b_720p": _cfg("wan14b_720p", 1, 40, 21, 45, 80, 0.10, 32, 3, "normal_gate"),
    # long video: 161 frames (41 x 45 x 80 latents)
    "wan14b_720p_long": _cfg("wan14b_720p_long", 1, 40, 41, 45, 80, 0.10, 32, 5, "normal_gate"),
}

# rank x sparsity sweep at the 720p shape
SWEEP_R = (16, 32, 64, 128)
SWEEP_KEEP = (0.20, 0.10, 0.05)


def sweep_config(r: int, keep: float) -> dict:
    c = dict(CONFIGS["wan14b_720p"])
    c.update(name=f"wan14b_720p_r{r}_keep{keep}", r=r, keep=keep, seed=4)
    return c


def get(name: str, **overrides) -> dict:
    c = dict(CONFIGS[name])
    c.update(overrides)
    c["N"] = c["T"] * c["Hh"] * c["Ww"]
    return c
