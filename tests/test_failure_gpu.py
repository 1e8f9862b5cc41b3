"""Failure detection without a GPU fault.

Every wait of the bf16 sparse kernel on an mbarrier is bounded.  The
ROLA_DEBUG_SKIP_FIRST_K_COPY test hook makes each CTA skip its first K copy (a
barrier that nothing will complete), so the waits run out after
cfg.wait_limit_ms; the kernel records ROLA_ERR_TIMEOUT in the workspace status
word, drains what it issued, releases its TMEM and returns.  The host reads the
status, and the same CUDA context then runs a normal call whose output matches
the oracle.
"""
import numpy as np
import pytest
import torch

from oracle import oracle as O
from paper_2609_06712_gb300 import configs, inputs
from parity_util import assert_close, to_np

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def rl():
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    from paper_2609_06712_gb300 import build
    build.build()
    from paper_2609_06712_gb300 import rola
    O.build()
    return rola


def test_timeout_is_reported_and_context_survives(rl):
    cfg = configs.get("tiny")
    x = inputs.make_inputs(cfg, dtype=torch.bfloat16)
    h = {k: (None if v is None else v.float().numpy()) for k, v in x.items()}
    d = {k: (None if v is None else v.cuda()) for k, v in x.items()}
    idx, _, _, _ = O.block_mask(cfg, h["q"], h["k"])
    kv = torch.from_numpy(idx).cuda()

    bad = rl.make_config(cfg)
    bad.debug_flags = rl.ROLA_DEBUG_SKIP_FIRST_K_COPY
    bad.wait_limit_ms = 50
    ws = rl.workspace(bad)
    o_s = torch.zeros_like(d["q"])
    rl.sparse_attn(bad, d["q"], d["k"], d["v"], kv, o_s, ws)      # the launch itself succeeds
    assert rl.get_device_status(ws) == rl.ROLA_ERR_TIMEOUT

    good = rl.make_config(cfg)
    ws2 = rl.workspace(good)
    rl.sparse_attn(good, d["q"], d["k"], d["v"], kv, o_s, ws2)
    assert rl.get_device_status(ws2) == rl.ROLA_OK
    want = O.sparse_attn(cfg, O.rope_full(cfg, h["q"]), O.rope_full(cfg, h["k"]), h["v"], idx)
    assert_close(to_np(o_s), want, True, "O^s after a timed-out call")


def test_backward_timeout_is_reported_and_context_survives(rl):
    """The same hook in the two tcgen05 backward kernels (their first K pair, their first Q / dO
    pair): rola_backward reports ROLA_ERR_TIMEOUT, and a normal backward afterwards returns the
    gradients of a backward run before it, bit for bit."""
    cfg = configs.get("tiny")
    x = inputs.make_inputs(cfg, dtype=torch.bfloat16)
    d = {k: (None if v is None else v.cuda()) for k, v in x.items()}
    good = rl.make_config(cfg)
    B, H, N = cfg["B"], cfg["H"], cfg["N"]
    ws = rl.workspace(good)
    o, o_s = torch.empty_like(d["q"]), torch.empty_like(d["q"])
    kv = torch.empty((B, H, rl.num_blocks(good), rl.num_keep(good)), dtype=torch.int32, device="cuda")
    lse = torch.empty((B, H, N), dtype=torch.float32, device="cuda")
    C = torch.empty((B, H, cfg["r"], 128), dtype=torch.float32, device="cuda")
    rl.forward_train(good, d["q"], d["k"], d["v"], d["P_q"], d["P_k"], d["gate"], o, kv, o_s, lse, C, ws)
    dO = torch.randn(d["q"].shape, generator=torch.Generator().manual_seed(2)).to(torch.bfloat16).cuda()

    def backward(c):
        g = [torch.zeros_like(d["q"]) for _ in range(3)] + [torch.zeros(d["P_q"].shape, device="cuda")
                                                             for _ in range(2)]
        bws = rl.backward_workspace(c)
        rl.backward(c, d["q"], d["k"], d["v"], d["P_q"], d["P_k"], d["gate"], kv, o_s, lse, C, dO, *g, None, bws)
        return g, rl.get_device_status(bws)

    ref, st = backward(good)
    assert st == rl.ROLA_OK
    bad = rl.make_config(cfg)
    bad.debug_flags = rl.ROLA_DEBUG_SKIP_FIRST_K_COPY
    bad.wait_limit_ms = 50
    _, st = backward(bad)
    assert st == rl.ROLA_ERR_TIMEOUT
    again, st = backward(good)
    assert st == rl.ROLA_OK
    for a, b in zip(ref, again):
        assert torch.equal(a, b)

