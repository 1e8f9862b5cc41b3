"""The backward pass (rola_forward_train + rola_backward) vs the fp64 oracle's
backward under the same mask: dq, dk, dv, dP_q, dP_k and dgate, bf16 and fp32,
on layers with ragged tails, several feature maps and RoPE placements; the
saved log-sum-exp against its definition; and the autograd wrapper."""
import numpy as np
import pytest
import torch

from oracle import oracle as O
from paper_2609_06712_gb300 import configs, inputs
from parity_util import assert_close_grad, dev, to_np

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def rl():
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    from paper_2609_06712_gb300 import build
    build.build()
    from paper_2609_06712_gb300 import rola
    O.build()
    return rola


def layer(**kw):
    c = configs.get("tiny")
    c.update(kw)
    c["N"] = c["T"] * c["Hh"] * c["Ww"]
    return c


CASES = {
    "ragged_585_r32": layer(T=5, Hh=9, Ww=13, H=2, r=32, keep=0.3, seed=71, dist="normal_gate"),
    "r16_keep1": layer(T=2, Hh=8, Ww=12, H=2, r=16, keep=1.0, seed=72),
    "gelu_inside_r64": layer(T=3, Hh=7, Ww=11, H=2, r=64, keep=0.4, seed=73, dist="normal_gate",
                             lowrank_act="gelu", lowrank_rope=1),
    "tanh_none_b2": layer(T=3, Hh=6, Ww=8, B=2, H=2, r=32, keep=0.5, seed=74, dist="normal_gate",
                          lowrank_act="tanh", lowrank_rope=2),
    "r128": layer(T=2, Hh=8, Ww=12, H=2, r=128, keep=0.3, seed=78, dist="normal_gate"),
    # a rank that is not a multiple of 16 (the bf16 kernels run at 32 with zero rows of P)
    "r24": layer(T=2, Hh=8, Ww=12, H=2, r=24, keep=0.3, seed=76, dist="normal_gate"),
    # one kept block of eight: half tiles on both sides, and key blocks no query block kept
    "keep1of8": layer(T=2, Hh=16, Ww=16, H=2, r=32, keep=0.125, seed=77, dist="normal_gate"),
    # 4 x 4 x 4 cube blocks: ragged edge cubes, and a grid of whole cubes
    "cube_5x9x13": layer(T=5, Hh=9, Ww=13, H=2, r=32, keep=0.3, seed=79, dist="normal_gate", block_geometry="cube"),
    "cube_4x8x12": layer(T=4, Hh=8, Ww=12, H=2, r=16, keep=0.5, seed=80, block_geometry="cube"),
    # latent frames of the 480p layers: 74 blocks (the last of 8 tokens), 15 kept
    "frames_3x30x52": layer(T=3, Hh=30, Ww=52, H=2, r=32, keep=0.2, seed=75, dist="normal_gate"),
}
DTYPES = [("bf16", torch.bfloat16), ("fp32", torch.float32)]


def draw(cfg, dtype):
    x = inputs.make_inputs(cfg, dtype=dtype)
    return x, {k: (None if v is None else v.float().numpy()) for k, v in x.items()}


def run_train(rl, cfg, x, dname, dO):
    c = rl.make_config(cfg, rl.ROLA_BF16 if dname == "bf16" else rl.ROLA_FP32)
    B, H, N = cfg["B"], cfg["H"], cfg["N"]
    q, k, v = dev(x["q"]), dev(x["k"]), dev(x["v"])
    Pq, Pk, g = dev(x["P_q"]), dev(x["P_k"]), dev(x["gate"])
    ws = rl.workspace(c)
    o, o_s = torch.empty_like(q), torch.empty_like(q)
    kv = torch.empty((B, H, rl.num_blocks(c), rl.num_keep(c)), dtype=torch.int32, device="cuda")
    lse = torch.empty((B, H, N), dtype=torch.float32, device="cuda")
    C = torch.empty((B, H, cfg["r"], 128), dtype=torch.float32, device="cuda")
    rl.forward_train(c, q, k, v, Pq, Pk, g, o, kv, o_s, lse, C, ws)
    grads = {"dq": torch.empty_like(q), "dk": torch.empty_like(k), "dv": torch.empty_like(v),
             "dP_q": torch.empty(Pq.shape, dtype=torch.float32, device="cuda"),
             "dP_k": torch.empty(Pk.shape, dtype=torch.float32, device="cuda"),
             "dgate": torch.empty((B, N), dtype=torch.float32, device="cuda")}
    bws = rl.backward_workspace(c)
    rl.backward(c, q, k, v, Pq, Pk, g, kv, o_s, lse, C, dev(dO), grads["dq"], grads["dk"], grads["dv"],
                grads["dP_q"], grads["dP_k"], grads["dgate"], bws)
    torch.cuda.synchronize()
    assert rl.get_device_status(ws) == rl.ROLA_OK and rl.get_device_status(bws) == rl.ROLA_OK
    return dict(o=o, o_s=o_s, kv=kv, lse=lse, C=C), grads


@pytest.mark.parametrize("case", sorted(CASES))
@pytest.mark.parametrize("dname,tdt", DTYPES)
def test_backward(rl, case, dname, tdt):
    cfg = CASES[case]
    x, h = draw(cfg, tdt)
    g = torch.Generator().manual_seed(cfg["seed"] + 500)
    dO = torch.randn(x["q"].shape, generator=g).to(tdt)
    fw, grads = run_train(rl, cfg, x, dname, dO)
    kv = fw["kv"].cpu().numpy()
    want = O.backward(cfg, h["q"], h["k"], h["v"], h["P_q"], h["P_k"], h["gate"], kv, dO.float().numpy(),
                      rope_mode=cfg.get("lowrank_rope", 0))
    for name in ("dq", "dk", "dv", "dP_q", "dP_k", "dgate"):
        assert_close_grad(to_np(grads[name]), want[name], dname == "bf16", f"{name}[{case},{dname}]")


@pytest.mark.parametrize("dname,tdt", DTYPES)
def test_saved_lse_is_the_log_sum_exp(rl, dname, tdt):
    """lse_p = log sum_j exp(q^r_p . k^r_j / sqrt d) over the kept keys (numpy, from the oracle's q^r, k^r)."""
    cfg = CASES["ragged_585_r32"]
    x, h = draw(cfg, tdt)
    fw, _ = run_train(rl, cfg, x, dname, torch.zeros(x["q"].shape, dtype=tdt))
    qr, kr = O.rope_full(cfg, h["q"]), O.rope_full(cfg, h["k"])
    kv = fw["kv"].cpu().numpy()
    N = cfg["N"]
    want = np.empty((1, cfg["H"], N))
    for hh in range(cfg["H"]):
        for i in range(kv.shape[2]):
            keys = np.concatenate([np.arange(j * 64, min(j * 64 + 64, N)) for j in kv[0, hh, i]])
            rows = np.arange(i * 64, min(i * 64 + 64, N))
            sc = qr[0, hh, rows] @ kr[0, hh, keys].T / np.sqrt(128.0)
            mx = sc.max(axis=1, keepdims=True)
            want[0, hh, rows] = (mx + np.log(np.exp(sc - mx).sum(axis=1, keepdims=True)))[:, 0]
    got = to_np(fw["lse"])
    tol = 2e-3 if dname == "bf16" else 1e-5
    assert np.abs(got - want).max() <= tol * np.abs(want).max(), np.abs(got - want).max()


def test_autograd_wrapper_matches_the_entry_points(rl):
    cfg = CASES["ragged_585_r32"]
    x, _ = draw(cfg, torch.float32)
    c = rl.make_config(cfg, rl.ROLA_FP32)
    leaves = {n: dev(x[n]).requires_grad_() for n in ("q", "k", "v", "P_q", "P_k", "gate")}
    o = rl.RoLAFunction.apply(c, *(leaves[n] for n in ("q", "k", "v", "P_q", "P_k", "gate")))
    g = torch.Generator().manual_seed(9)
    dO = torch.randn(o.shape, generator=g).cuda()
    o.backward(dO)
    fw, grads = run_train(rl, cfg, x, "fp32", dO.cpu())
    assert torch.equal(o.detach(), fw["o"])
    for n, gname in (("q", "dq"), ("k", "dk"), ("v", "dv"), ("P_q", "dP_q"), ("P_k", "dP_k"), ("gate", "dgate")):
        assert torch.equal(leaves[n].grad, grads[gname]), n


def test_backward_is_deterministic(rl):
    cfg = CASES["tanh_none_b2"]
    x, _ = draw(cfg, torch.bfloat16)
    dO = torch.randn(x["q"].shape, generator=torch.Generator().manual_seed(3)).to(torch.bfloat16)
    _, a = run_train(rl, cfg, x, "bf16", dO)
    _, b = run_train(rl, cfg, x, "bf16", dO)
    for n in a:
        assert torch.equal(a[n], b[n]), n
