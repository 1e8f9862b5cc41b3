"""Token gate g = sigmoid(X w_g + b_g) (Sec. fusion) on the GPU vs the fp64 oracle.

Tolerance: the kernel accumulates the d_model products in fp32 in some order,
so its logit is within gamma_{D+2} * sum_d |x_d w_d| of the exact one
(gamma_n = n u / (1 - n u), u = 2^-24); the sigmoid's slope is at most 1/4,
and the fp32 sigmoid itself adds a few ulp of g.
"""
import numpy as np
import pytest
import torch

from oracle import oracle as O
from paper_2609_06712_gb300 import inputs

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def rl():
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    from paper_2609_06712_gb300 import build
    build.build()
    from paper_2609_06712_gb300 import rola
    O.build()
    return rola


CASES = [
    ("small_ragged", 2, 333, 96),
    ("wan13b_480p", 1, 32760, 1536),      # d_model = 12 heads x 128
    ("wan14b_720p", 1, 75600, 5120),      # d_model = 40 heads x 128
]


@pytest.mark.parametrize("name,B,N,D", CASES, ids=[c[0] for c in CASES])
@pytest.mark.parametrize("dname,tdt", [("bf16", torch.bfloat16), ("fp32", torch.float32)])
def test_gate_matches_oracle(rl, name, B, N, D, dname, tdt):
    x = inputs.make_gate_inputs(B, N, D, dtype=tdt, seed=B * 1000 + D)
    c = rl.make_config({"B": B, "H": 1, "N": N, "T": 1, "Hh": 1, "Ww": N, "keep": 0.1, "r": 16},
                       rl.ROLA_BF16 if dname == "bf16" else rl.ROLA_FP32)
    g = torch.empty((B, N), dtype=torch.float32, device="cuda")
    rl.gate(c, x["X"].cuda(), x["w_g"].cuda(), x["b_g"], g)
    torch.cuda.synchronize()
    Xh, wh = x["X"].float().numpy(), x["w_g"].float().numpy()
    want = O.gate(Xh, wh, x["b_g"])
    u = 2.0 ** -24
    gamma = (D + 2) * u / (1 - (D + 2) * u)
    bound = 0.25 * gamma * (np.abs(Xh) * np.abs(wh)).sum(axis=-1) + 8 * u
    err = np.abs(g.cpu().numpy().astype(np.float64) - want)
    assert (err <= bound).all(), f"max err {err.max():.3e}, worst ratio {(err / bound).max():.3f}"
