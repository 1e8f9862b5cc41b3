"""rola_lowrank_summary_static: the summary for callers that cannot allocate.

Some callers cannot give the library device scratch (a plugin whose host
framework owns the allocator, a runtime that forbids allocation while
serving).  This entry point keeps its scratch in a static device array inside
the library.  The GPU test checks it against the workspace-based
rola_lowrank_summary, through the C ABI, on two calls in a row (the second
call reuses the array the first one left behind).  This file is collected
next to last (before the guard canaries), so a run that stops at the first
failure has run the parity tests first.
"""
import ctypes

import numpy as np
import pytest
import torch

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


@pytest.mark.gpu
@pytest.mark.parametrize("name,dtype", [("wan13b_480p", torch.bfloat16), ("tiny", torch.float32)])
def test_static_summary_matches_workspace_summary(rl, name, dtype):
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    cfg = configs.get(name)
    x = {k: (None if v is None else v.cuda()) for k, v in inputs.make_inputs(cfg, dtype=dtype).items()}
    c = rl.make_config(cfg, rl.ROLA_BF16 if dtype == torch.bfloat16 else rl.ROLA_FP32)
    B, H, r = cfg["B"], cfg["H"], cfg["r"]
    C_ref = torch.empty((B, H, r, 128), dtype=torch.float32, device="cuda")
    z_ref = torch.empty((B, H, r), dtype=torch.float32, device="cuda")
    ws = rl.workspace(c)
    rl.lowrank_summary(c, x["k"], x["v"], x["P_k"], C_ref, z_ref, ws)
    L = rl.library()
    stream = ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    for call in range(2):
        C = torch.full((B, H, r, 128), float("nan"), dtype=torch.float32, device="cuda")
        z = torch.full((B, H, r), float("nan"), dtype=torch.float32, device="cuda")
        st = L.rola_lowrank_summary_static(ctypes.byref(c), ctypes.c_void_p(x["k"].data_ptr()),
                                           ctypes.c_void_p(x["v"].data_ptr()), ctypes.c_void_p(x["P_k"].data_ptr()),
                                           ctypes.c_void_p(C.data_ptr()), ctypes.c_void_p(z.data_ptr()), stream)
        assert st == rl.ROLA_OK, L.rola_status_string(st)
        torch.cuda.synchronize()
        bf16 = dtype == torch.bfloat16
        assert_close(C.cpu().numpy(), C_ref.cpu().numpy(), bf16, f"static C, call {call}", unit_rms=True)
        assert_close(z.cpu().numpy(), z_ref.cpu().numpy(), bf16, f"static z, call {call}", unit_rms=True)
