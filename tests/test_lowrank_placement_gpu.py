"""The three placements of the truncated RoPE in the low-rank features (the
orderings of the paper's RoPE-placement study, Tab. mechanism): outside SiLU
(Eq. qklr), inside SiLU (Prop. inside) and none.  CUDA path vs the fp64 oracle
in each placement, per kernel and for the module, bf16 and fp32; and the
property that singles out the outside placement: a uniform shift of every
position leaves the low-rank readout unchanged outside SiLU (Eq. shiftinv,
Prop. exact) and changes it inside (Prop. inside)."""
import numpy as np
import pytest
import torch

from oracle import oracle as O
from paper_2609_06712_gb300 import configs, inputs
from parity_util import assert_close, check_mask, dev, to_np

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
    "ragged_585_r64": layer(T=5, Hh=9, Ww=13, H=2, r=64, keep=0.3, seed=22),
    "r48_gate": layer(T=3, Hh=10, Ww=20, H=2, r=48, keep=0.2, seed=24, dist="normal_gate"),
    "r128": layer(T=2, Hh=12, Ww=16, H=2, r=128, keep=0.25, seed=27),
    "r8": layer(T=3, Hh=7, Ww=11, H=2, r=8, keep=0.25, seed=28),
}
MODES = {"inside": (1, O.ROPE_INSIDE), "none": (2, O.ROPE_NONE)}
DTYPES = [("bf16", torch.bfloat16), ("fp32", torch.float32)]


def draw(cfg, dtype):
    x = inputs.make_inputs(cfg, dtype=dtype)
    return x, {k: (None if v is None else v.float().numpy()) for k, v in x.items()}


def config(rl, cfg, dname, lr_mode):
    return rl.make_config(dict(cfg, lowrank_rope=lr_mode), rl.ROLA_BF16 if dname == "bf16" else rl.ROLA_FP32)


@pytest.mark.parametrize("case", sorted(CASES))
@pytest.mark.parametrize("mode", sorted(MODES))
@pytest.mark.parametrize("dname,tdt", DTYPES)
def test_summary_and_apply(rl, case, mode, dname, tdt):
    cfg = CASES[case]
    lr_mode, o_mode = MODES[mode]
    x, h = draw(cfg, tdt)
    c = config(rl, cfg, dname, lr_mode)
    ws = rl.workspace(c)
    C = torch.empty((cfg["B"], cfg["H"], cfg["r"], 128), dtype=torch.float32, device="cuda")
    z = torch.empty((cfg["B"], cfg["H"], cfg["r"]), dtype=torch.float32, device="cuda")
    rl.lowrank_summary(c, dev(x["k"]), dev(x["v"]), dev(x["P_k"]), C, z, ws)
    torch.cuda.synchronize()
    Cw, zw = O.lowrank_summary(cfg, h["k"], h["v"], h["P_k"], rope_mode=o_mode)
    assert_close(to_np(C), Cw, dname == "bf16", f"C[{case},{mode},{dname}]", unit_rms=True)
    assert_close(to_np(z), zw, dname == "bf16", f"z[{case},{mode},{dname}]", unit_rms=True)
    g = torch.Generator().manual_seed(cfg["seed"] + 1000)
    o_s = (0.02 * torch.randn(x["q"].shape, generator=g)).to(tdt)
    C32 = torch.from_numpy(Cw.astype(np.float32))
    o = torch.empty_like(dev(o_s))
    rl.lowrank_apply(c, dev(x["q"]), dev(x["P_q"]), dev(C32), dev(x["gate"]), dev(o_s), o, ws)
    torch.cuda.synchronize()
    want = O.lowrank_apply(cfg, h["q"], h["P_q"], C32.double().numpy(), h["gate"], o_s.float().numpy(),
                           rope_mode=o_mode)
    assert_close(to_np(o), want, dname == "bf16", f"O[{case},{mode},{dname}]")


@pytest.mark.parametrize("mode", sorted(MODES))
@pytest.mark.parametrize("dname,tdt", DTYPES)
def test_forward(rl, mode, dname, tdt):
    cfg = CASES["ragged_585_r64"]
    lr_mode, o_mode = MODES[mode]
    x, h = draw(cfg, tdt)
    c = config(rl, cfg, dname, lr_mode)
    ws = rl.workspace(c)
    nB, nk = rl.num_blocks(c), rl.num_keep(c)
    out = torch.empty_like(dev(x["q"]))
    kv = torch.empty((cfg["B"], cfg["H"], nB, nk), dtype=torch.int32, device="cuda")
    rl.forward(c, dev(x["q"]), dev(x["k"]), dev(x["v"]), dev(x["P_q"]), dev(x["P_k"]), dev(x["gate"]), out, kv, ws)
    torch.cuda.synchronize()
    assert rl.get_device_status(ws) == rl.ROLA_OK
    # the GPU's mask (the mask does not depend on the low-rank placement) is handed to the oracle
    res = O.forward(cfg, h["q"], h["k"], h["v"], h["P_q"], h["P_k"], h["gate"], mask_override=kv.cpu().numpy(),
                    rope_mode=o_mode)
    check_mask(cfg, h, kv.cpu().numpy(), f"forward {mode} {dname}")
    assert_close(to_np(out), res["o"], dname == "bf16", f"O[forward,{mode},{dname}]")


def readout(rl, cfg, x, lr_mode, offset):
    """Low-rank readout of the fused output (O^s = 0 in, so O = g sqrt(eps) O^lr), fp32."""
    c = rl.make_config(dict(cfg, lowrank_rope=lr_mode, pos_offset=offset), rl.ROLA_FP32)
    ws = rl.workspace(c)
    C = torch.empty((cfg["B"], cfg["H"], cfg["r"], 128), dtype=torch.float32, device="cuda")
    rl.lowrank_summary(c, dev(x["k"]), dev(x["v"]), dev(x["P_k"]), C, None, ws)
    o_s = torch.zeros_like(dev(x["q"]))
    o = torch.empty_like(o_s)
    rl.lowrank_apply(c, dev(x["q"]), dev(x["P_q"]), C, None, o_s, o, ws)
    torch.cuda.synchronize()
    return to_np(o)


def test_uniform_shift_leaves_only_the_outside_readout_unchanged(rl):
    cfg = CASES["r128"]
    x, _ = draw(cfg, torch.float32)
    shift = (3, -2, 5)
    rel = {}
    for mode, lr_mode in [("outside", 0), ("inside", 1), ("none", 2)]:
        a = readout(rl, cfg, x, lr_mode, (0, 0, 0))
        b = readout(rl, cfg, x, lr_mode, shift)
        rel[mode] = float(np.linalg.norm(b - a) / np.linalg.norm(a))
    assert rel["outside"] < 1e-4, rel       # Eq. (shiftinv) carried through the summary: rounding only
    assert rel["none"] < 1e-6, rel          # position-blind
    assert rel["inside"] > 1e-2, rel        # Prop. inside: absolute position leaks into C
