"""The sparse branch with 4 x 4 x 4 cube blocks of the latent grid (the
ROLA_BLOCK_CUBE geometry) vs the fp64 oracle in the same geometry: the block
mask (bit for bit against the oracle's fp32 decision on every row), the sparse branch and the
module, bf16 and fp32, on grids with whole cubes, ragged edge cubes and a
single partial cube; and the 720p layer at full size on sampled query cubes."""
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


def layer(name=None, **kw):
    c = configs.get(name or "tiny")
    c.update(kw, block_geometry="cube")
    c["N"] = c["T"] * c["Hh"] * c["Ww"]
    return c


CASES = {
    "ragged_5x9x13": layer(T=5, Hh=9, Ww=13, H=2, r=32, keep=0.3, seed=41, dist="normal_gate"),
    "whole_4x8x12": layer(T=4, Hh=8, Ww=12, H=2, r=16, keep=0.5, seed=42),
    "frames_3x30x52": layer(T=3, Hh=30, Ww=52, H=2, r=32, keep=0.2, seed=43),
    "one_partial_cube": layer(T=1, Hh=1, Ww=3, H=2, r=16, keep=0.5, seed=44),
}
DTYPES = [("bf16", torch.bfloat16), ("fp32", torch.float32)]


def draw(cfg, dtype):
    x = inputs.make_inputs(cfg, dtype=dtype)
    return x, {k: (None if v is None else v.float().numpy()) for k, v in x.items()}


def config(rl, cfg, dname):
    return rl.make_config(cfg, rl.ROLA_BF16 if dname == "bf16" else rl.ROLA_FP32)


@pytest.mark.parametrize("case", sorted(CASES))
@pytest.mark.parametrize("dname,tdt", DTYPES)
def test_block_mask(rl, case, dname, tdt):
    cfg = CASES[case]
    x, h = draw(cfg, tdt)
    c = config(rl, cfg, dname)
    ws = rl.workspace(c)
    nB, nk = rl.num_blocks(c), rl.num_keep(c)
    assert nB == O.num_blocks(cfg) and nk == O.num_keep(cfg)
    kv = torch.empty((cfg["B"], cfg["H"], nB, nk), dtype=torch.int32, device="cuda")
    rl.block_mask(c, dev(x["q"]), dev(x["k"]), kv, ws)
    torch.cuda.synchronize()
    check_mask(cfg, h, kv.cpu().numpy(), f"mask cube {case} {dname}")


@pytest.mark.parametrize("case", sorted(CASES))
@pytest.mark.parametrize("dname,tdt", DTYPES)
def test_sparse_attn(rl, case, dname, tdt):
    cfg = CASES[case]
    x, h = draw(cfg, tdt)
    c = config(rl, cfg, dname)
    ws = rl.workspace(c)
    idx, _, _, _ = O.block_mask(cfg, h["q"], h["k"])
    o_s = torch.full_like(dev(x["q"]), float("nan"))
    rl.sparse_attn(c, dev(x["q"]), dev(x["k"]), dev(x["v"]), torch.from_numpy(idx).cuda(), o_s, ws)
    torch.cuda.synchronize()
    assert rl.get_device_status(ws) == rl.ROLA_OK
    want = O.sparse_attn(cfg, O.rope_full(cfg, h["q"]), O.rope_full(cfg, h["k"]), h["v"], idx)
    assert_close(to_np(o_s), want, dname == "bf16", f"O^s[{case},{dname}]")     # every token written


def run_forward(rl, cfg, x, dname):
    c = config(rl, cfg, dname)
    ws = rl.workspace(c)
    nB, nk = rl.num_blocks(c), rl.num_keep(c)
    out = torch.empty_like(dev(x["q"]))
    kv = torch.empty((cfg["B"], cfg["H"], nB, nk), dtype=torch.int32, device="cuda")
    rl.forward(c, dev(x["q"]), dev(x["k"]), dev(x["v"]), dev(x["P_q"]), dev(x["P_k"]), dev(x["gate"]), out, kv, ws)
    torch.cuda.synchronize()
    assert rl.get_device_status(ws) == rl.ROLA_OK
    return out, kv


def compare_forward(cfg, h, out, kv, dname, qblocks=None):
    """The mask (bit for bit against the oracle's fp32 decision, every row), then O on every token
    of the selected query cubes, the oracle running the module under the GPU's mask."""
    kvn = kv.cpu().numpy()
    check_mask(cfg, h, kvn, f"forward cube {cfg['name']} {dname}")
    res = O.forward(cfg, h["q"], h["k"], h["v"], h["P_q"], h["P_k"], h["gate"], mask_override=kvn, qblocks=qblocks)
    nB = kvn.shape[2]
    blocks = range(nB) if qblocks is None else qblocks
    rows = np.isin(O.block_of(cfg), list(blocks))
    got = to_np(out)
    for b in range(cfg["B"]):
        for hh in range(cfg["H"]):
            assert_close(got[b, hh, rows], res["o"][b, hh, rows], dname == "bf16",
                         f"O[{cfg['name']},cube,{dname},b{b},h{hh}]")
    return res


@pytest.mark.parametrize("case", sorted(CASES))
@pytest.mark.parametrize("dname,tdt", DTYPES)
def test_forward(rl, case, dname, tdt):
    cfg = CASES[case]
    x, h = draw(cfg, tdt)
    out, kv = run_forward(rl, cfg, x, dname)
    compare_forward(cfg, h, out, kv, dname)


def test_forward_720p_cubes_sampled(rl):
    """The Wan2.1-14B 720p layer (21 x 45 x 80 latents: 6 x 12 x 20 = 1440 cubes, 144 kept) at full
    size in bf16: the mask in full, O on sampled query cubes of every head, including the first
    cube and the last (a 1 x 1 x 4 corner of the grid)."""
    cfg = configs.get("wan14b_720p")
    cfg["block_geometry"] = "cube"
    x, h = draw(cfg, torch.bfloat16)
    out, kv = run_forward(rl, cfg, x, "bf16")
    nB = kv.shape[2]
    assert nB == 1440 and kv.shape[3] == 144
    rng = np.random.default_rng(cfg["seed"])
    blocks = sorted({0, nB - 1, *rng.choice(np.arange(1, nB - 1), size=14, replace=False).tolist()})
    compare_forward(cfg, h, out, kv, "bf16", qblocks=blocks)
