"""Pins of the oracle's backward pass (CPU only).

The gradients are checked against the oracle's own forward pass, which is
pinned separately: directional central differences with Richardson
extrapolation, for every input (q, k, v, P_q, P_k, gate) and several feature
maps and RoPE placements; phi' against differences of phi; and the sparse
branch's gradient at keep = 1 against torch's fp64 autograd of SDPA on the
rotated inputs, rotated back (R(p)^T = R(-p))."""
import math

import numpy as np
import pytest
import torch

from paper_2609_06712_gb300 import configs, inputs


def small_cfg(**kw):
    c = configs.get("tiny")
    c.update(T=2, Hh=5, Ww=7, H=2, r=16, keep=0.5, seed=61, dist="normal_gate")
    c.update(kw)
    c["N"] = c["T"] * c["Hh"] * c["Ww"]
    return c


def draw(cfg):
    x = inputs.make_inputs(cfg, dtype=torch.float32)
    return {n: (None if t is None else t.float().numpy()) for n, t in x.items()}


ACTS = ["silu", "identity", "tanh", "relu", "gelu"]


def test_activation_derivatives(oracle):
    """phi' against fp64 central differences of phi (away from ReLU's kink), and closed forms:
    SiLU'(0) = 1/2, tanh'(0) = 1, GELU'(0) = 1/2, ReLU' a step."""
    O = oracle
    xs = np.array([-3.1, -1.2, -0.4, 0.3, 0.9, 2.6])
    h = 1e-5
    for n in ACTS:
        fd = np.array([(O.activation(n, x + h) - O.activation(n, x - h)) / (2 * h) for x in xs])
        got = np.array([O.activation_grad(n, x) for x in xs])
        np.testing.assert_allclose(got, fd, rtol=1e-8, atol=1e-9, err_msg=n)
    assert O.activation_grad("silu", 0.0) == pytest.approx(0.5, abs=1e-15)
    assert O.activation_grad("tanh", 0.0) == 1.0
    assert O.activation_grad("gelu", 0.0) == pytest.approx(0.5, abs=1e-15)
    assert O.activation_grad("relu", -0.5) == 0.0 and O.activation_grad("relu", 0.5) == 1.0


def loss(O, cfg, x, mask, rope_mode, dO):
    r = O.forward(cfg, x["q"], x["k"], x["v"], x["P_q"], x["P_k"], x["gate"], mask_override=mask,
                  rope_mode=rope_mode)
    return float(np.sum(r["o"] * dO))


def directional(O, cfg, x, mask, rope_mode, dO, name, delta, h):
    """Central differences L(x + s) - L(x - s') along delta, Richardson-extrapolated over the steps h
    and h / 2.  Returns the extrapolated difference and the matching combination of the actual
    float32 steps (s + s'), which the gradient is dotted with."""
    def central(step):
        xp, xm = dict(x), dict(x)
        xp[name] = (x[name] + step * delta).astype(np.float32)
        xm[name] = (x[name] - step * delta).astype(np.float32)
        diff = loss(O, cfg, xp, mask, rope_mode, dO) - loss(O, cfg, xm, mask, rope_mode, dO)
        return diff, xp[name].astype(np.float64) - xm[name]
    f1, s1 = central(h)
    f2, s2 = central(h / 2)
    return (4 * f2 - f1) / 3, (4 * s2 - s1) / 3


# (feature map, RoPE placement, block geometry); the cube case has ragged edge cubes
# (5 x 5 x 7 tokens: 2 x 2 x 2 cubes, 4 of 8 kept); "q128" takes 128-token query blocks
# against 64-token key blocks (3 x 7 x 11 tokens: query blocks of 128 and 103, 2 of 4 kept)
CASES = [("silu", 0, "flat"), ("gelu", 1, "flat"), ("tanh", 2, "flat"), ("identity", 0, "flat"),
         ("silu", 1, "flat"), ("silu", 0, "cube"), ("silu", 0, "q128")]


@pytest.mark.parametrize("act,rope_mode,geometry", CASES)
def test_gradients_match_central_differences(oracle, act, rope_mode, geometry):
    """Each gradient of L = sum(dO * O) dotted with a random direction equals the directional
    derivative of the (pinned) forward pass under the same fixed mask."""
    O = oracle
    if geometry == "flat":
        cfg = small_cfg(lowrank_act=act)
    elif geometry == "cube":
        cfg = small_cfg(lowrank_act=act, T=5, block_geometry="cube")
    else:
        cfg = small_cfg(lowrank_act=act, T=3, Hh=7, Ww=11, qblock=128)
    x = draw(cfg)
    rng = np.random.default_rng(7)
    dO = rng.standard_normal((1, cfg["H"], cfg["N"], 128)).astype(np.float32)
    mask, _, _, _ = O.block_mask(cfg, x["q"], x["k"])
    g = O.backward(cfg, x["q"], x["k"], x["v"], x["P_q"], x["P_k"], x["gate"], mask, dO, rope_mode=rope_mode)
    grads = {"q": g["dq"], "k": g["dk"], "v": g["dv"], "P_q": g["dP_q"], "P_k": g["dP_k"], "gate": g["dgate"]}
    for name, grad in grads.items():
        delta = rng.choice([-1.0, 1.0], size=x[name].shape)
        # step: 2^-8 of the input's RMS, a power of two so that x +- h is exact in float32
        h = 2.0 ** (round(math.log2(float(np.sqrt(np.mean(x[name].astype(np.float64) ** 2))))) - 8)
        want, step = directional(O, cfg, x, mask, rope_mode, dO, name, delta, h)
        got = float(np.sum(grad * step))
        scale = float(np.sum(np.abs(grad * step)))    # the terms the directional sum cancels
        assert abs(got - want) <= 3e-6 * scale + 1e-12, (name, got, want, scale)


def test_constant_gate_gradient(oracle):
    """gate = NULL uses the constant g = sigmoid(b_g); dgate is still dL/dg_p, equal to the
    gradient at an explicit gate array holding that constant."""
    O = oracle
    cfg = small_cfg(dist="normal")
    x = draw(cfg)
    assert x["gate"] is None
    dO = np.random.default_rng(3).standard_normal((1, cfg["H"], cfg["N"], 128)).astype(np.float32)
    mask, _, _, _ = O.block_mask(cfg, x["q"], x["k"])
    a = O.backward(cfg, x["q"], x["k"], x["v"], x["P_q"], x["P_k"], None, mask, dO)
    gconst = np.full((1, cfg["N"]), 1.0 / (1.0 + math.exp(1.946)), np.float32)
    b = O.backward(cfg, x["q"], x["k"], x["v"], x["P_q"], x["P_k"], gconst, mask, dO)
    for n in a:
        # the constant is sigmoid(b_g) in fp64 against its float32 copy in the array
        np.testing.assert_allclose(a[n], b[n], rtol=1e-6, atol=1e-7 * np.abs(b[n]).max())


def test_sparse_gradient_is_sdpa_autograd_at_zero_gate(oracle):
    """With g = 0 the module is the sparse branch: P_q, P_k get no gradient, and at keep = 1 the
    gradients of q, k, v are torch's fp64 autograd of dense SDPA on R(p) q, R(p) k, rotated back."""
    O = oracle
    cfg = small_cfg(keep=1.0, dist="normal")
    x = draw(cfg)
    zero = np.zeros((1, cfg["N"]), np.float32)
    dO = np.random.default_rng(4).standard_normal((1, cfg["H"], cfg["N"], 128)).astype(np.float32)
    mask, _, _, _ = O.block_mask(cfg, x["q"], x["k"])
    g = O.backward(cfg, x["q"], x["k"], x["v"], x["P_q"], x["P_k"], zero, mask, dO)
    assert np.abs(g["dP_q"]).max() == 0 and np.abs(g["dP_k"]).max() == 0
    qr = torch.tensor(O.rope_full(cfg, x["q"]), requires_grad=True)
    kr = torch.tensor(O.rope_full(cfg, x["k"]), requires_grad=True)
    v = torch.tensor(x["v"].astype(np.float64), requires_grad=True)
    o = torch.nn.functional.scaled_dot_product_attention(qr, kr, v)
    (o * torch.from_numpy(dO)).sum().backward()
    back = lambda t: np.stack([np.stack([O.rotate(cfg, 64, -O.position(cfg, n), t[0, h, n])
                                         for n in range(cfg["N"])]) for h in range(cfg["H"])])[None]
    np.testing.assert_allclose(g["dq"], back(qr.grad.numpy()), rtol=1e-9, atol=1e-11)
    np.testing.assert_allclose(g["dk"], back(kr.grad.numpy()), rtol=1e-9, atol=1e-11)
    np.testing.assert_allclose(g["dv"], v.grad.numpy(), rtol=1e-9, atol=1e-11)
