"""The output projection (Alg. 1, last step) and the whole attention block vs the fp64 oracle,
through the C ABI.

rola_out_proj: Y = concat_h(O) W_o^T (+ b_o), bf16 on the tcgen05 GEMM and fp32 in the validation
mode, on a small layer with a ragged token tile and a ragged feature tile (every output checked), and
at the Wan2.1 model widths (1.3B: 12 heads, d_model 1536; 14B: 40 heads, d_model 5120) at full
sequence length in the launch configuration the bench times, on sampled token rows that include the
first tile and the ragged last one.  rola_attention_block: gate -> module -> projection against the
oracle's chain of the same three steps under the GPU's mask.
"""
import numpy as np
import pytest
import torch

from oracle import oracle as O
from paper_2609_06712_gb300 import configs, inputs
from parity_util import assert_close, check_mask, to_np

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def rl():
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    from paper_2609_06712_gb300 import build
    build.build()
    from paper_2609_06712_gb300 import rola
    O.build()
    return rola


def proj_inputs(B, H, N, d_model, dtype, seed, bias=True):
    """O ~ N(0, 0.3^2) (the module's output scale), W_o ~ N(0, 1/(H*128)) in the nn.Linear layout,
    b_o ~ N(0, 0.1^2), all seeded; O and W_o rounded once to the storage dtype."""
    g = torch.Generator().manual_seed(seed)
    Oh = (0.3 * torch.randn((B, H, N, 128), generator=g)).to(dtype)
    W = (torch.randn((d_model, H * 128), generator=g) / (H * 128) ** 0.5).to(dtype)
    b = (0.1 * torch.randn((d_model,), generator=g)) if bias else None
    return Oh, W, b


def run_proj(rl, cfg, Oh, W, b, dtype):
    c = rl.make_config(cfg, rl.ROLA_BF16 if dtype == torch.bfloat16 else rl.ROLA_FP32)
    ws = torch.empty(256, dtype=torch.uint8, device="cuda")
    Y = torch.full((cfg["B"], cfg["N"], W.shape[0]), float("nan"), dtype=dtype, device="cuda")
    rl.out_proj(c, Oh.cuda(), W.cuda(), None if b is None else b.cuda(), Y, ws)
    torch.cuda.synchronize()
    assert rl.get_device_status(ws) == rl.ROLA_OK
    return Y


@pytest.mark.parametrize("bias", [True, False])
@pytest.mark.parametrize("dname,dtype", [("bf16", torch.bfloat16), ("fp32", torch.float32)])
def test_out_proj_small_ragged(rl, dname, dtype, bias):
    """B = 2, 3 heads, 200 tokens (a full 128-token tile and one of 72), d_model = 320 (a full
    256-feature tile and one of 64): every output element against the oracle."""
    cfg = configs.get("tiny", T=2, Hh=10, Ww=10, B=2, H=3)
    Oh, W, b = proj_inputs(2, 3, 200, 320, dtype, seed=61, bias=bias)
    Y = run_proj(rl, cfg, Oh, W, b, dtype)
    want = O.out_proj(Oh.float().numpy(), W.float().numpy(), None if b is None else b.numpy())
    assert_close(to_np(Y), want, dname == "bf16", f"Y[{dname},bias={bias}]")


def sample_rows(N, n=48, seed=0):
    rng = np.random.default_rng(seed)
    last = (N - 1) // 128 * 128
    rows = {0, 1, 127, 128, N - 1, last, *range(last, N, max(1, (N - last) // 8))}
    rows |= set(rng.choice(N, size=n - len(rows), replace=False).tolist())
    return sorted(rows)


@pytest.mark.parametrize("name,d_model", [("wan13b_480p", 1536), ("wan14b_720p", 5120)])
def test_out_proj_model_width(rl, name, d_model):
    """The Wan2.1 layer widths at full sequence length (bf16), sampled token rows, all features."""
    cfg = configs.get(name)
    B, H, N = cfg["B"], cfg["H"], cfg["N"]
    assert H * 128 == d_model
    Oh, W, b = proj_inputs(B, H, N, d_model, torch.bfloat16, seed=62)
    Y = run_proj(rl, cfg, Oh, W, b, torch.bfloat16)
    rows = sample_rows(N, seed=cfg["seed"])
    want = O.out_proj(Oh.float().numpy(), W.float().numpy(), b.numpy(), rows=rows)
    got = to_np(Y)
    assert_close(got[:, rows], want[:, rows], True, f"Y[{name}]")
    assert np.isfinite(got).all()                        # every row written


@pytest.mark.parametrize("dname,dtype", [("bf16", torch.bfloat16), ("fp32", torch.float32)])
def test_attention_block(rl, dname, dtype):
    """Gate from the block input X, the module, the output projection in one call, against the
    oracle's gate, module (under the GPU's mask, itself checked bit for bit) and projection."""
    cfg = configs.get("tiny", T=3, Hh=9, Ww=13, H=2, r=32, keep=0.3, seed=63)
    B, H, N = cfg["B"], cfg["H"], cfg["N"]
    d_model = 256
    x = inputs.make_inputs(cfg, dtype=dtype)
    xg = inputs.make_gate_inputs(B, N, d_model, dtype=dtype, seed=64)
    _, W, b = proj_inputs(B, H, 1, d_model, dtype, seed=65)
    h = {k: (None if v is None else v.float().numpy()) for k, v in x.items()}
    c = rl.make_config(cfg, rl.ROLA_BF16 if dtype == torch.bfloat16 else rl.ROLA_FP32)
    ws = rl.workspace(c)
    d = {k: (None if v is None else v.cuda()) for k, v in x.items()}
    gate = torch.empty((B, N), dtype=torch.float32, device="cuda")
    o = torch.empty_like(d["q"])
    Y = torch.empty((B, N, d_model), dtype=dtype, device="cuda")
    kv = torch.empty((B, H, rl.num_blocks(c), rl.num_keep(c)), dtype=torch.int32, device="cuda")
    rl.attention_block(c, xg["X"].cuda(), xg["w_g"].cuda(), xg["b_g"], d["q"], d["k"], d["v"], d["P_q"], d["P_k"],
                       W.cuda(), b.cuda(), gate, o, Y, kv, ws)
    torch.cuda.synchronize()
    assert rl.get_device_status(ws) == rl.ROLA_OK
    g_want = O.gate(xg["X"].float().numpy(), xg["w_g"].float().numpy(), xg["b_g"])
    assert_close(to_np(gate), g_want, False if dname == "fp32" else True, f"gate[{dname}]")
    kvn = kv.cpu().numpy()
    check_mask(cfg, h, kvn, f"block {dname}")
    res = O.forward(cfg, h["q"], h["k"], h["v"], h["P_q"], h["P_k"], g_want, mask_override=kvn)
    assert_close(to_np(o), res["o"], dname == "bf16", f"O[block,{dname}]")
    want = O.out_proj(res["o"], W.float().numpy(), b.numpy())
    assert_close(to_np(Y), want, dname == "bf16", f"Y[block,{dname}]")
