"""Guard canaries: no entry point writes outside the buffers it is given (every
output of every entry point, the workspace-free summary and the token gate
included).

compute-sanitizer is closed on this machine, so every output and workspace is
placed inside a larger buffer whose margins (8 KB on each side) hold a fixed
bit pattern; after the calls the margins must still hold it.  The layers have
ragged tails (a last block of 39 tokens; edge cubes) where an unmasked store
would land past the end.  Collected last: a run that stops at the first
failure has run everything else.
"""
import ctypes

import numpy as np
import pytest
import torch

from paper_2609_06712_gb300 import configs, inputs

pytestmark = pytest.mark.gpu

PAD = 8192                                  # guard bytes per side (a multiple of 256: alignment kept)
RAW = {1: (torch.uint8, 0xA5), 2: (torch.int16, 0x5A5A), 4: (torch.int32, 0x5A5A5A5A)}


class Guarded:
    """A tensor of `shape` and `dtype` with PAD bytes of pattern before and after it."""

    def __init__(self, shape, dtype):
        es = torch.empty((), dtype=dtype).element_size()
        raw, self.pat = RAW[es]
        self.n, self.p = int(np.prod(shape)), PAD // es
        self.buf = torch.full((self.n + 2 * self.p,), self.pat, dtype=raw, device="cuda")
        self.t = self.buf[self.p:self.p + self.n].view(dtype).view(shape)

    def intact(self):
        return bool((self.buf[:self.p] == self.pat).all()) and bool((self.buf[self.p + self.n:] == self.pat).all())


@pytest.fixture(scope="module")
def rl():
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    from paper_2609_06712_gb300 import build
    build.build()
    from paper_2609_06712_gb300 import rola
    return rola


LAYERS = {
    # 231 tokens: blocks of 64, 64, 64, 39
    "ragged_231": configs.get("tiny", T=3, Hh=7, Ww=11, H=2, r=16, keep=0.5, seed=91, dist="normal_gate"),
    # 585 tokens in 2 x 3 x 4 cubes, ragged in every axis
    "cube_5x9x13": configs.get("tiny", T=5, Hh=9, Ww=13, H=2, r=32, keep=0.3, seed=92, dist="normal_gate",
                               block_geometry="cube"),
}
DTYPES = [("bf16", torch.bfloat16), ("fp32", torch.float32)]


@pytest.mark.parametrize("layer", sorted(LAYERS))
@pytest.mark.parametrize("dname,tdt", DTYPES)
def test_no_store_outside_the_given_buffers(rl, layer, dname, tdt):
    cfg = LAYERS[layer]
    c = rl.make_config(cfg, rl.ROLA_BF16 if dname == "bf16" else rl.ROLA_FP32)
    B, H, N, r = cfg["B"], cfg["H"], cfg["N"], cfg["r"]
    x = {n: (None if t is None else t.cuda()) for n, t in inputs.make_inputs(cfg, dtype=tdt).items()}
    q, k, v, Pq, Pk, g = x["q"], x["k"], x["v"], x["P_q"], x["P_k"], x["gate"]
    row = (B, H, N, 128)
    kvs = (B, H, rl.num_blocks(c), rl.num_keep(c))
    guards = []

    def G(shape, dtype):
        t = Guarded(shape, dtype)
        guards.append(t)
        return t.t

    ws = G((rl.workspace_bytes(c),), torch.uint8)
    kv = G(kvs, torch.int32)
    rl.block_mask(c, q, k, kv, ws)
    C, z = G((B, H, r, 128), torch.float32), G((B, H, r), torch.float32)
    rl.lowrank_summary(c, k, v, Pk, C, z, ws)
    o_s = G(row, tdt)
    rl.sparse_attn(c, q, k, v, kv, o_s, ws)
    rl.lowrank_apply(c, q, Pq, C, g, o_s, G(row, tdt), ws)
    rl.forward(c, q, k, v, Pq, Pk, g, G(row, tdt), G(kvs, torch.int32), ws)
    kv2, o_s2 = G(kvs, torch.int32), G(row, tdt)
    lse, C2 = G((B, H, N), torch.float32), G((B, H, r, 128), torch.float32)
    rl.forward_train(c, q, k, v, Pq, Pk, g, G(row, tdt), kv2, o_s2, lse, C2, ws)
    dO = torch.randn(row, generator=torch.Generator().manual_seed(3)).to(tdt).cuda()
    bws = G((rl.library().rola_backward_workspace_bytes(ctypes.byref(c)),), torch.uint8)
    rl.backward(c, q, k, v, Pq, Pk, g, kv2, o_s2, lse, C2, dO, G(row, tdt), G(row, tdt), G(row, tdt),
                G(Pq.shape, torch.float32), G(Pk.shape, torch.float32),
                G((B, N), torch.float32) if g is not None else None, bws)
    # the summary without a workspace (its scratch is the library's own array)
    Cs, zs = G((B, H, r, 128), torch.float32), G((B, H, r), torch.float32)
    st = rl.library().rola_lowrank_summary_static(
        ctypes.byref(c), ctypes.c_void_p(k.data_ptr()), ctypes.c_void_p(v.data_ptr()), ctypes.c_void_p(Pk.data_ptr()),
        ctypes.c_void_p(Cs.data_ptr()), ctypes.c_void_p(zs.data_ptr()),
        ctypes.c_void_p(torch.cuda.current_stream().cuda_stream))
    assert st == rl.ROLA_OK
    # the token gate from a block input of d_model = 8 * 40 (a ragged last warp tile)
    xg = inputs.make_gate_inputs(B, N, 320, dtype=tdt, device="cuda", seed=5)
    rl.gate(c, xg["X"], xg["w_g"], xg["b_g"], G((B, N), torch.float32))
    torch.cuda.synchronize()
    assert rl.get_device_status(ws) == rl.ROLA_OK and rl.get_device_status(bws) == rl.ROLA_OK
    bad = [i for i, t in enumerate(guards) if not t.intact()]
    assert not bad, f"margins overwritten around buffers {bad} of {len(guards)}"
