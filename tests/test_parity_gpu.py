"""CUDA path vs the fp64 oracle, element by element, through the C ABI.

Per kernel (mask, sparse branch, summary, apply) and for the whole module, in
bf16 and in the fp32 validation mode, on small layers that still span many
blocks and a ragged tail, and on the Wan2.1 layer shapes with sampled query
blocks.  Inputs come from the shared seeded generator; expected values come
from the oracle only.
"""
import numpy as np
import pytest
import torch

from oracle import oracle as O
from paper_2609_06712_gb300 import configs, inputs
from parity_util import assert_close, check_mask, dev, rows_of_blocks, to_np

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
    c.update(kw)
    c["N"] = c["T"] * c["Hh"] * c["Ww"]
    return c


SMALL = {
    "tiny": layer(),
    "ragged_105": layer(T=3, Hh=5, Ww=7, H=3, r=16, keep=0.5, seed=21),
    "ragged_585_r64": layer(T=5, Hh=9, Ww=13, H=2, r=64, keep=0.3, seed=22),
    "r128_keep1": layer(T=2, Hh=12, Ww=16, H=2, r=128, keep=1.0, seed=23),
    "r48_gate": layer(T=3, Hh=10, Ww=20, H=2, r=48, keep=0.2, seed=24, dist="normal_gate"),
    "rmsnorm_gain_b2": layer(T=4, Hh=8, Ww=9, B=2, H=2, r=32, keep=0.25, seed=25, dist="rmsnorm_gain"),
    "offset": layer(T=3, Hh=8, Ww=8, H=2, r=32, keep=0.25, seed=26, pos_offset=(5, -3, 7)),
    # ranks that are not multiples of 16 (the paper's sweep starts at r = 8)
    "r8_ragged": layer(T=3, Hh=7, Ww=11, H=2, r=8, keep=0.25, seed=28),
    "r24": layer(T=2, Hh=8, Ww=12, H=2, r=24, keep=0.3, seed=29, dist="normal_gate"),
    # the whole sequence is one partial block (40 tokens): one query block, one kept key block, a half tile
    "one_partial_block": layer(T=1, Hh=5, Ww=8, H=2, r=16, keep=0.5, seed=30),
}


def draw(cfg, dtype):
    x = inputs.make_inputs(cfg, dtype=dtype)
    host = {k: (None if v is None else v.float().numpy()) for k, v in x.items()}
    return x, host


def dtype_cases():
    return [("bf16", torch.bfloat16), ("fp32", torch.float32)]


def rola_dtype(rl, name):
    return rl.ROLA_BF16 if name == "bf16" else rl.ROLA_FP32


# ------------------------------------------------------------------ per kernel


@pytest.mark.parametrize("case", sorted(SMALL))
@pytest.mark.parametrize("dname,tdt", dtype_cases())
def test_block_mask(rl, case, dname, tdt):
    cfg = SMALL[case]
    x, h = draw(cfg, tdt)
    c = rl.make_config(cfg, rola_dtype(rl, dname))
    ws = rl.workspace(c)
    nB, nk = rl.num_blocks(c), rl.num_keep(c)
    kv = torch.empty((cfg["B"], cfg["H"], nB, nk), dtype=torch.int32, device="cuda")
    rl.block_mask(c, dev(x["q"]), dev(x["k"]), kv, ws)
    torch.cuda.synchronize()
    check_mask(cfg, h, kv.cpu().numpy(), f"mask {case} {dname}")


@pytest.mark.parametrize("case", sorted(SMALL))
@pytest.mark.parametrize("dname,tdt", dtype_cases())
def test_sparse_attn(rl, case, dname, tdt):
    cfg = SMALL[case]
    x, h = draw(cfg, tdt)
    c = rl.make_config(cfg, rola_dtype(rl, dname))
    ws = rl.workspace(c)
    idx, _, _, _ = O.block_mask(cfg, h["q"], h["k"])
    o_s = torch.empty_like(dev(x["q"]))
    rl.sparse_attn(c, dev(x["q"]), dev(x["k"]), dev(x["v"]), torch.from_numpy(idx).cuda(), o_s, ws)
    torch.cuda.synchronize()
    want = O.sparse_attn(cfg, O.rope_full(cfg, h["q"]), O.rope_full(cfg, h["k"]), h["v"], idx)
    assert_close(to_np(o_s), want, dname == "bf16", f"O^s[{case},{dname}]")


@pytest.mark.parametrize("case", sorted(SMALL))
@pytest.mark.parametrize("dname,tdt", dtype_cases())
def test_lowrank_summary(rl, case, dname, tdt):
    cfg = SMALL[case]
    x, h = draw(cfg, tdt)
    c = rl.make_config(cfg, rola_dtype(rl, dname))
    ws = rl.workspace(c)
    B, H, r = cfg["B"], cfg["H"], cfg["r"]
    C = torch.empty((B, H, r, 128), dtype=torch.float32, device="cuda")
    z = torch.empty((B, H, r), dtype=torch.float32, device="cuda")
    rl.lowrank_summary(c, dev(x["k"]), dev(x["v"]), dev(x["P_k"]), C, z, ws)
    torch.cuda.synchronize()
    Cw, zw = O.lowrank_summary(cfg, h["k"], h["v"], h["P_k"])
    assert_close(to_np(C), Cw, dname == "bf16", f"C[{case},{dname}]", unit_rms=True)
    assert_close(to_np(z), zw, dname == "bf16", f"z[{case},{dname}]", unit_rms=True)


@pytest.mark.parametrize("case", sorted(SMALL))
@pytest.mark.parametrize("dname,tdt", dtype_cases())
def test_lowrank_apply(rl, case, dname, tdt):
    cfg = SMALL[case]
    x, h = draw(cfg, tdt)
    c = rl.make_config(cfg, rola_dtype(rl, dname))
    ws = rl.workspace(c)
    Cw, _ = O.lowrank_summary(cfg, h["k"], h["v"], h["P_k"])
    # O^s stand-in: attention-sized values, stored in the layer dtype
    g = torch.Generator().manual_seed(cfg["seed"] + 1000)
    o_s = (0.02 * torch.randn(x["q"].shape, generator=g)).to(tdt)
    C32 = torch.from_numpy(Cw.astype(np.float32))
    o = torch.empty_like(dev(o_s))
    rl.lowrank_apply(c, dev(x["q"]), dev(x["P_q"]), dev(C32), dev(x["gate"]), dev(o_s), o, ws)
    torch.cuda.synchronize()
    want = O.lowrank_apply(cfg, h["q"], h["P_q"], C32.double().numpy(), h["gate"], o_s.float().numpy())
    assert_close(to_np(o), want, dname == "bf16", f"O[{case},{dname}]")
    # in place: o aliases o_s
    o_s_dev = dev(o_s)
    rl.lowrank_apply(c, dev(x["q"]), dev(x["P_q"]), dev(C32), dev(x["gate"]), o_s_dev, o_s_dev, ws)
    torch.cuda.synchronize()
    assert torch.equal(o_s_dev, o)


# ------------------------------------------------------------------ module


def run_forward(rl, cfg, x, dname, o=None):
    c = rl.make_config(cfg, rola_dtype(rl, dname))
    ws = rl.workspace(c)
    nB, nk = rl.num_blocks(c), rl.num_keep(c)
    q = dev(x["q"])
    out = torch.empty_like(q) if o is None else o
    kv = torch.empty((cfg["B"], cfg["H"], nB, nk), dtype=torch.int32, device="cuda")
    rl.forward(c, q, dev(x["k"]), dev(x["v"]), dev(x["P_q"]), dev(x["P_k"]), dev(x["gate"]), out, kv, ws)
    assert rl.get_device_status(ws) == rl.ROLA_OK
    return out, kv


def compare_forward(cfg, x, h, out, kv, dname, qblocks=None, label=None):
    """The mask (bit for bit against the oracle's fp32 decision, every row), then O on every
    token of the selected query blocks, the oracle running the module under the GPU's mask."""
    kvn = kv.cpu().numpy()
    check_mask(cfg, h, kvn, f"forward {label or cfg['name']} r{cfg['r']} keep{cfg['keep']} {dname}")
    res = O.forward(cfg, h["q"], h["k"], h["v"], h["P_q"], h["P_k"], h["gate"], mask_override=kvn,
                    qblocks=qblocks)
    nB = kvn.shape[2]
    blocks = range(nB) if qblocks is None else qblocks
    rows = rows_of_blocks(blocks, cfg["block"], cfg["N"])
    got = to_np(out)
    for b in range(cfg["B"]):
        for hh in range(cfg["H"]):
            assert_close(got[b, hh, rows], res["o"][b, hh, rows], dname == "bf16",
                         f"O[{cfg['name']},{dname},b{b},h{hh}]")
    return res


@pytest.mark.parametrize("case", sorted(SMALL))
@pytest.mark.parametrize("dname,tdt", dtype_cases())
def test_forward_small(rl, case, dname, tdt):
    cfg = SMALL[case]
    x, h = draw(cfg, tdt)
    out, kv = run_forward(rl, cfg, x, dname)
    torch.cuda.synchronize()
    compare_forward(cfg, x, h, out, kv, dname, label=case)


@pytest.mark.parametrize("case", ["tiny", "ragged_585_r64", "rmsnorm_gain_b2"])
def test_fused_prepass_matches_separate_entry_points(rl, case):
    """In bf16 the forward pass rotates, pools and summarises in one pass over
    q, k, v; its mask must be the one rola_block_mask returns, bit for bit, and
    its output the one the separate entry points compose to."""
    cfg = SMALL[case]
    x, h = draw(cfg, torch.bfloat16)
    out, kv = run_forward(rl, cfg, x, "bf16")
    c = rl.make_config(cfg, rl.ROLA_BF16)
    ws = rl.workspace(c)
    kv2 = torch.empty_like(kv)
    rl.block_mask(c, dev(x["q"]), dev(x["k"]), kv2, ws)
    C = torch.empty((cfg["B"], cfg["H"], cfg["r"], 128), dtype=torch.float32, device="cuda")
    rl.lowrank_summary(c, dev(x["k"]), dev(x["v"]), dev(x["P_k"]), C, None, ws)
    o_s = torch.empty_like(out)
    rl.sparse_attn(c, dev(x["q"]), dev(x["k"]), dev(x["v"]), kv2, o_s, ws)
    o = torch.empty_like(out)
    rl.lowrank_apply(c, dev(x["q"]), dev(x["P_q"]), C, dev(x["gate"]), o_s, o, ws)
    torch.cuda.synchronize()
    assert torch.equal(kv, kv2)
    assert torch.equal(out, o)


def test_forward_is_deterministic_and_stays_in_bounds(rl):
    """Two runs are bitwise equal; bytes around the output are never written."""
    cfg = SMALL["ragged_585_r64"]
    x, _ = draw(cfg, torch.bfloat16)
    n = x["q"].numel()
    pad = 4096
    canvas = torch.full((n + 2 * pad,), 7.25, dtype=torch.bfloat16, device="cuda")
    o1 = canvas[pad:pad + n].view(x["q"].shape)
    _, kv1 = run_forward(rl, cfg, x, "bf16", o=o1)
    o2, kv2 = run_forward(rl, cfg, x, "bf16")
    torch.cuda.synchronize()
    assert torch.equal(o1, o2) and torch.equal(kv1, kv2)
    assert (canvas[:pad] == 7.25).all() and (canvas[pad + n:] == 7.25).all()


def test_shift_invariance_on_gpu(rl):
    """Eq. (shiftinv): a uniform shift of all positions leaves the GPU output unchanged
    up to fp32 table rounding (outputs match the unshifted oracle)."""
    cfg = SMALL["offset"]
    x, h = draw(cfg, torch.bfloat16)
    out, kv = run_forward(rl, cfg, x, "bf16")
    base = dict(cfg, pos_offset=(0, 0, 0))
    out0, kv0 = run_forward(rl, base, x, "bf16")
    torch.cuda.synchronize()
    assert torch.equal(kv, kv0)
    assert_close(to_np(out), to_np(out0), True, "shifted vs unshifted")


def test_gate_zero_returns_sparse_branch(rl):
    """Eq. (gate) with g = 0 gives O = O^s."""
    cfg = SMALL["tiny"]
    x, h = draw(cfg, torch.float32)
    x["gate"] = torch.zeros((cfg["B"], cfg["N"]))
    out, kv = run_forward(rl, cfg, x, "fp32")
    c = rl.make_config(cfg, rl.ROLA_FP32)
    ws = rl.workspace(c)
    o_s = torch.empty_like(out)
    rl.sparse_attn(c, dev(x["q"]), dev(x["k"]), dev(x["v"]), kv, o_s, ws)
    torch.cuda.synchronize()
    assert torch.equal(out, o_s)


# ------------------------------------------------------------------ layer shapes


def sample_blocks(nB, n=32, seed=0):
    rng = np.random.default_rng(seed)
    mid = rng.choice(np.arange(1, nB - 1), size=min(n - 2, nB - 2), replace=False)
    return sorted({0, nB - 1, *mid.tolist()})


LAYERS = [
    ("wan13b_480p", None, None, 32),
    ("wan14b_480p", None, None, 32),
    ("wan14b_720p", None, None, 32),
    ("wan14b_720p_long", None, None, 16),
    # rank x sparsity sweep at the 720p shape
    ("wan14b_720p", 16, 0.20, 8),
    ("wan14b_720p", 64, 0.05, 8),
    ("wan14b_720p", 128, 0.10, 8),
    ("wan14b_720p", 128, 0.20, 8),
]


@pytest.mark.parametrize("name,r,keep,nsample", LAYERS,
                         ids=[f"{n}-r{r}-keep{k}" if r else n for n, r, k, _ in LAYERS])
def test_forward_layer_shapes_sampled(rl, name, r, keep, nsample):
    """The Wan2.1 layer shapes at full size, in the launch configuration the bench
    times: the mask and C in full, O on sampled query blocks of every head
    (including the first and the ragged last block)."""
    cfg = configs.get(name) if r is None else configs.sweep_config(r, keep)
    x, h = draw(cfg, torch.bfloat16)
    out, kv = run_forward(rl, cfg, x, "bf16")
    torch.cuda.synchronize()
    nB = (cfg["N"] + 63) // 64
    blocks = sample_blocks(nB, nsample, seed=cfg["seed"])
    res = compare_forward(cfg, x, h, out, kv, "bf16", qblocks=blocks)
    c = rl.make_config(cfg)
    ws = rl.workspace(c)
    # the fused pre-pass and the stand-alone rotate + pool give the same mask, bit for bit, in full
    kv2 = torch.empty_like(kv)
    rl.block_mask(c, dev(x["q"]), dev(x["k"]), kv2, ws)
    torch.cuda.synchronize()
    assert torch.equal(kv, kv2)
    # the summary in full
    C = torch.empty((cfg["B"], cfg["H"], cfg["r"], 128), dtype=torch.float32, device="cuda")
    rl.lowrank_summary(c, dev(x["k"]), dev(x["v"]), dev(x["P_k"]), C, None, ws)
    torch.cuda.synchronize()
    assert_close(to_np(C), res["C"], True, f"C[{cfg['name']}]", unit_rms=True)


# ------------------------------------------------------------------ 128-token query blocks

QBLOCK = {
    # 585 tokens: query chunks of 128, 128, 128, 128, 73 against key blocks of 64 (the last of 9)
    "q128_ragged_585": layer(T=5, Hh=9, Ww=13, H=2, r=32, keep=0.3, seed=71, qblock=128),
    # 448 tokens: query chunks of 128 x 3 and 64 (an odd number of key blocks, 7)
    "q128_odd_448": layer(T=4, Hh=8, Ww=14, H=3, r=16, keep=0.4, seed=72, qblock=128, dist="normal_gate"),
}


@pytest.mark.parametrize("case", sorted(QBLOCK))
@pytest.mark.parametrize("dname,tdt", dtype_cases())
def test_block_mask_query_blocks_of_128(rl, case, dname, tdt):
    """128-token query chunks against 64-token key blocks: the mask (one row per query chunk) bit for bit
    against the oracle's fp32 decision, every row."""
    cfg = QBLOCK[case]
    x, h = draw(cfg, tdt)
    c = rl.make_config(cfg, rola_dtype(rl, dname))
    ws = rl.workspace(c)
    nQ, nk = rl.num_query_blocks(c), rl.num_keep(c)
    assert nQ == O.num_qblocks(cfg) == -(-cfg["N"] // 128) and rl.num_blocks(c) == O.num_blocks(cfg)
    kv = torch.empty((cfg["B"], cfg["H"], nQ, nk), dtype=torch.int32, device="cuda")
    rl.block_mask(c, dev(x["q"]), dev(x["k"]), kv, ws)
    torch.cuda.synchronize()
    check_mask(cfg, h, kv.cpu().numpy(), f"mask {case} {dname}")


@pytest.mark.parametrize("case", sorted(QBLOCK))
@pytest.mark.parametrize("dname,tdt", dtype_cases())
def test_forward_query_blocks_of_128(rl, case, dname, tdt):
    """The module with 128-token query blocks: the fused forward's mask bit for bit, then O on every token
    against the oracle's forward (qblock = 128) under the GPU's mask."""
    cfg = QBLOCK[case]
    x, h = draw(cfg, tdt)
    c = rl.make_config(cfg, rola_dtype(rl, dname))
    ws = rl.workspace(c)
    out = torch.empty_like(dev(x["q"]))
    kv = torch.empty((cfg["B"], cfg["H"], rl.num_query_blocks(c), rl.num_keep(c)), dtype=torch.int32, device="cuda")
    rl.forward(c, dev(x["q"]), dev(x["k"]), dev(x["v"]), dev(x["P_q"]), dev(x["P_k"]), dev(x["gate"]), out, kv, ws)
    torch.cuda.synchronize()
    assert rl.get_device_status(ws) == rl.ROLA_OK
    kvn = kv.cpu().numpy()
    check_mask(cfg, h, kvn, f"forward {case} {dname}")
    res = O.forward(cfg, h["q"], h["k"], h["v"], h["P_q"], h["P_k"], h["gate"], mask_override=kvn)
    assert_close(to_np(out), res["o"], dname == "bf16", f"O[{case},{dname}]")


def test_forward_query_blocks_of_128_720p_sampled(rl):
    """The Wan2.1-14B 720p layer with 128-token query chunks (591 of them, 118 of 1182 key blocks kept
    each): the mask in full, O on sampled query chunks of every head (the first and the ragged last)."""
    cfg = configs.get("wan14b_720p", qblock=128)
    x, h = draw(cfg, torch.bfloat16)
    c = rl.make_config(cfg)
    ws = rl.workspace(c)
    nQ = rl.num_query_blocks(c)
    assert nQ == 591
    out = torch.empty_like(dev(x["q"]))
    kv = torch.empty((1, cfg["H"], nQ, rl.num_keep(c)), dtype=torch.int32, device="cuda")
    rl.forward(c, dev(x["q"]), dev(x["k"]), dev(x["v"]), dev(x["P_q"]), dev(x["P_k"]), dev(x["gate"]), out, kv, ws)
    torch.cuda.synchronize()
    kvn = kv.cpu().numpy()
    check_mask(cfg, h, kvn, "forward wan14b_720p qblock128 bf16")
    chunks = sample_blocks(nQ, 16, seed=cfg["seed"])
    res = O.forward(cfg, h["q"], h["k"], h["v"], h["P_q"], h["P_k"], h["gate"], mask_override=kvn, qblocks=chunks)
    rows = rows_of_blocks(chunks, 128, cfg["N"])
    got = to_np(out)
    for hh in range(cfg["H"]):
        assert_close(got[0, hh, rows], res["o"][0, hh, rows], True, f"O[720p q128,h{hh}]")


def test_training_refuses_query_blocks_of_128(rl):
    """The backward pass is built for 64-token query blocks only; the training entry points refuse 128."""
    cfg = QBLOCK["q128_ragged_585"]
    c = rl.make_config(cfg)
    L = rl.library()
    import ctypes
    P = ctypes.c_void_p(0x10000)
    w = ctypes.c_void_p(0x100000)
    st = L.rola_forward_train(ctypes.byref(c), P, P, P, P, P, None, P, P, P, P, P, w, 1 << 30, None)
    assert st == rl.ROLA_ERR_UNSUPPORTED
