"""Seeded synthetic inputs shaped like Wan2.1 attention layers.

This module is shared by the CUDA path's tests / bench and by the oracle's
tests.  It draws random numbers and nothing else: none of the method's
arithmetic lives here.  Draw order is fixed: q, k, v, P_q, P_k, per-channel
gain, gate; all draws are fp32 from one ``torch.Generator`` and are rounded
once to the storage dtype.

Distributions (``cfg["dist"]``):
  normal        q, k, v ~ N(0, 1); gate = None (the module uses sigmoid(gate_bias))
  rmsnorm       x ~ N(0, 1) then each token rescaled to unit RMS over d_h (a
                stand-in for the backbone's norm_q / norm_k); v ~ N(0, 1)
  rmsnorm_gain  as rmsnorm, then times a per-head per-channel gain ~ U(0.5, 1.5)
  normal_gate   as normal, plus a per-token gate sigmoid(-1.946 + 0.5 N(0, 1)),
                a stand-in for the upstream gate sigmoid(X W_g + b_g)
P_q, P_k ~ N(0, 1/d_h), shape [H][r][d_h].
"""
from __future__ import annotations

import torch


def _unit_rms(x: torch.Tensor) -> torch.Tensor:
    return x * torch.rsqrt(x.pow(2).mean(dim=-1, keepdim=True))


def make_inputs(cfg: dict, dtype: torch.dtype = torch.bfloat16, device="cpu", seed=None,
                with_gate=None) -> dict:
    """Returns dict(q, k, v, P_q, P_k, gate) on ``device``.

    Draws happen on ``device`` with a generator of that device seeded with
    ``seed`` (default cfg["seed"]); CPU draws are the ones the parity tests use.
    """
    B, H, N, dh, r = cfg["B"], cfg["H"], cfg["N"], cfg.get("d_h", 128), cfg["r"]
    dist = cfg.get("dist", "normal")
    g = torch.Generator(device=device)
    g.manual_seed(cfg["seed"] if seed is None else seed)
    f32 = dict(dtype=torch.float32, device=device, generator=g)
    shape = (B, H, N, dh)
    q = torch.randn(shape, **f32)
    k = torch.randn(shape, **f32)
    v = torch.randn(shape, **f32)
    P_q = torch.randn((H, r, dh), **f32) * (1.0 / dh) ** 0.5
    P_k = torch.randn((H, r, dh), **f32) * (1.0 / dh) ** 0.5
    if dist in ("rmsnorm", "rmsnorm_gain"):
        q = _unit_rms(q)
        k = _unit_rms(k)
    if dist == "rmsnorm_gain":
        gain_q = 0.5 + torch.rand((H, 1, dh), **f32)
        gain_k = 0.5 + torch.rand((H, 1, dh), **f32)
        q = q * gain_q
        k = k * gain_k
    gate = None
    if with_gate is None:
        with_gate = dist == "normal_gate"
    if with_gate:
        gate = torch.sigmoid(-1.946 + 0.5 * torch.randn((B, N), **f32))
    out = dict(q=q.to(dtype), k=k.to(dtype), v=v.to(dtype), P_q=P_q.to(dtype), P_k=P_k.to(dtype),
               gate=gate)
    return out


def make_gate_inputs(B: int, N: int, d_model: int, dtype: torch.dtype = torch.bfloat16, device="cpu",
                     seed: int = 0) -> dict:
    """Inputs of the token gate g = sigmoid(X w_g + b_g): the attention block's input hidden states
    X ~ N(0, 1) [B][N][d_model] (a stand-in for the normalised block input), w_g ~ N(0, 1/d_model)
    (so the logit is ~N(0, 1) around the bias) and the paper's initial bias b_g = -1.946."""
    g = torch.Generator(device=device)
    g.manual_seed(seed)
    f32 = dict(dtype=torch.float32, device=device, generator=g)
    X = torch.randn((B, N, d_model), **f32)
    w = torch.randn((d_model,), **f32) * (1.0 / d_model) ** 0.5
    return dict(X=X.to(dtype), w_g=w.to(dtype), b_g=-1.946)
