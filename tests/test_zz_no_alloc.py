"""rola_lowrank_summary_static: the summary for callers that cannot allocate.

Some callers cannot give the library device scratch (a plugin whose host
framework owns the allocator, a runtime that forbids allocation while
serving).  This entry point keeps its scratch in a static device array inside
the library.  The GPU tests check it against the workspace-based
rola_lowrank_summary, through the C ABI, on two calls in a row (the second
call reuses the array the first one left behind), also on a layer too large
for the regular split (the reduced-capacity path); against the fp64 oracle;
and on a call whose bounded waits run out (C and z come back NaN, and the
next call recovers).  This file is collected
next to last (before the guard canaries), so a run that stops at the first
failure has run the parity tests first.
"""
import ctypes

import numpy as np
import pytest
import torch

from oracle import oracle as O
from paper_2609_06712_gb300 import configs, inputs
from parity_util import assert_close


@pytest.fixture(scope="module")
def rl():
    from paper_2609_06712_gb300 import build
    build.build()
    from paper_2609_06712_gb300 import rola
    return rola


def test_static_summary_rejects_layers_beyond_its_array(rl):
    """A layer whose one-split scratch exceeds the 16 MiB array is refused before any launch."""
    c = rl.make_config(configs.get("wan14b_720p", H=400, r=128))   # 400 heads x 66 KB partial > 16 MiB
    P = ctypes.c_void_p(0x10000)
    st = rl.library().rola_lowrank_summary_static(ctypes.byref(c), P, P, P, P, None, None)
    assert st == rl.ROLA_ERR_UNSUPPORTED
    c = rl.make_config(configs.get("tiny"))
    st = rl.library().rola_lowrank_summary_static(ctypes.byref(c), P, P, P, ctypes.c_void_p(0), None, None)
    assert st == rl.ROLA_ERR_INVALID_ARG


def static_call(rl, c, x, C, z):
    L = rl.library()
    stream = ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    return L.rola_lowrank_summary_static(ctypes.byref(c), ctypes.c_void_p(x["k"].data_ptr()),
                                         ctypes.c_void_p(x["v"].data_ptr()), ctypes.c_void_p(x["P_k"].data_ptr()),
                                         ctypes.c_void_p(C.data_ptr()),
                                         ctypes.c_void_p(z.data_ptr()) if z is not None else None, stream)


# The 720p grid cut to 2 frames (7200 tokens) with 120 heads and r = 128: a partial slot is
# 4 * (128 * 128 + 128) = 66048 bytes, so the 16 MiB array holds 253 slots -- fewer than the
# 152 CTAs + 119 extra slots of the regular bf16 split and the regular fp32 splits of 120 heads:
# both dtypes take the reduced-capacity path.
REDUCED = dict(T=2, H=120, r=128)


@pytest.mark.gpu
@pytest.mark.parametrize("name,dtype", [("wan13b_480p", torch.bfloat16), ("tiny", torch.float32),
                                        ("reduced", torch.bfloat16), ("reduced", torch.float32)])
def test_static_summary_matches_workspace_summary(rl, name, dtype):
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    cfg = configs.get("wan14b_720p", **REDUCED) if name == "reduced" else configs.get(name)
    x = {k: (None if v is None else v.cuda()) for k, v in inputs.make_inputs(cfg, dtype=dtype).items()}
    c = rl.make_config(cfg, rl.ROLA_BF16 if dtype == torch.bfloat16 else rl.ROLA_FP32)
    B, H, r = cfg["B"], cfg["H"], cfg["r"]
    C_ref = torch.empty((B, H, r, 128), dtype=torch.float32, device="cuda")
    z_ref = torch.empty((B, H, r), dtype=torch.float32, device="cuda")
    ws = rl.workspace(c)
    rl.lowrank_summary(c, x["k"], x["v"], x["P_k"], C_ref, z_ref, ws)
    L = rl.library()
    for call in range(2):
        C = torch.full((B, H, r, 128), float("nan"), dtype=torch.float32, device="cuda")
        z = torch.full((B, H, r), float("nan"), dtype=torch.float32, device="cuda")
        st = static_call(rl, c, x, C, z)
        assert st == rl.ROLA_OK, L.rola_status_string(st)
        torch.cuda.synchronize()
        bf16 = dtype == torch.bfloat16
        assert_close(C.cpu().numpy(), C_ref.cpu().numpy(), bf16, f"static C, call {call}", unit_rms=True)
        assert_close(z.cpu().numpy(), z_ref.cpu().numpy(), bf16, f"static z, call {call}", unit_rms=True)


@pytest.mark.gpu
@pytest.mark.parametrize("dtype", [torch.bfloat16, torch.float32])
def test_static_summary_matches_the_oracle(rl, dtype):
    """The static summary against the fp64 oracle (Eq. ctx), not only against the workspace
    summary, on a ragged layer that takes the reduced-capacity path in neither dtype."""
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    cfg = configs.get("tiny", T=5, Hh=9, Ww=13, H=3, r=48, seed=31)
    xh = inputs.make_inputs(cfg, dtype=dtype)
    x = {k: (None if v is None else v.cuda()) for k, v in xh.items()}
    c = rl.make_config(cfg, rl.ROLA_BF16 if dtype == torch.bfloat16 else rl.ROLA_FP32)
    C = torch.empty((1, 3, 48, 128), dtype=torch.float32, device="cuda")
    z = torch.empty((1, 3, 48), dtype=torch.float32, device="cuda")
    assert static_call(rl, c, x, C, z) == rl.ROLA_OK
    torch.cuda.synchronize()
    Cw, zw = O.lowrank_summary(cfg, xh["k"].float().numpy(), xh["v"].float().numpy(), xh["P_k"].float().numpy())
    bf16 = dtype == torch.bfloat16
    assert_close(C.cpu().numpy(), Cw, bf16, "static C vs oracle", unit_rms=True)
    assert_close(z.cpu().numpy(), zw, bf16, "static z vs oracle", unit_rms=True)


@pytest.mark.gpu
def test_static_summary_timeout_gives_nan_and_the_next_call_recovers(rl):
    """With no workspace there is no status word to read: when a bounded wait of the bf16 kernel
    runs out (the test hook skips each CTA's first load; waits limited to 50 ms), C and z come
    back NaN.  The next normal call clears the shared array's status and matches the workspace
    summary again."""
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    cfg = configs.get("tiny")
    x = {k: (None if v is None else v.cuda()) for k, v in inputs.make_inputs(cfg, dtype=torch.bfloat16).items()}
    B, H, r = cfg["B"], cfg["H"], cfg["r"]
    bad = rl.make_config(cfg)
    bad.debug_flags = rl.ROLA_DEBUG_SKIP_FIRST_K_COPY
    bad.wait_limit_ms = 50
    C = torch.zeros((B, H, r, 128), dtype=torch.float32, device="cuda")
    z = torch.zeros((B, H, r), dtype=torch.float32, device="cuda")
    assert static_call(rl, bad, x, C, z) == rl.ROLA_OK          # the launches themselves succeed
    torch.cuda.synchronize()
    assert torch.isnan(C).all() and torch.isnan(z).all()
    good = rl.make_config(cfg)
    C_ref = torch.empty_like(C)
    z_ref = torch.empty_like(z)
    rl.lowrank_summary(good, x["k"], x["v"], x["P_k"], C_ref, z_ref, rl.workspace(good))
    assert static_call(rl, good, x, C, z) == rl.ROLA_OK
    torch.cuda.synchronize()
    assert_close(C.cpu().numpy(), C_ref.cpu().numpy(), True, "static C after a timed-out call", unit_rms=True)
    assert_close(z.cpu().numpy(), z_ref.cpu().numpy(), True, "static z after a timed-out call", unit_rms=True)
