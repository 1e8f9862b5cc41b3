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
