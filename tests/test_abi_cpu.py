"""The C ABI library on a machine without a GPU: it builds, loads, exports every
entry point include/rola.h declares, and its host-side validation returns the
documented status codes before touching the device."""
import ctypes
import os
import re
import subprocess

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "rola.h")


@pytest.fixture(scope="module")
def rl():
    from paper_2609_06712_gb300 import build
    build.build()
    from paper_2609_06712_gb300 import rola
    return rola


def declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(rola_[a-z0-9_]+)\s*\(", text)))


def test_exports_every_declared_entry_point(rl):
    names = declared_functions()
    assert {"rola_block_mask", "rola_sparse_attn", "rola_lowrank_summary", "rola_lowrank_apply",
            "rola_forward"} <= set(names)
    out = subprocess.run(["nm", "-D", "--defined-only", rl.LIB_PATH], capture_output=True, text=True,
                         check=True).stdout
    exported = set(line.split()[-1] for line in out.splitlines() if line.strip())
    missing = [n for n in names if n not in exported]
    assert not missing, missing
    for n in names:
        getattr(rl.library(), n)


def test_config_struct_layout_matches_the_header(rl, tmp_path):
    """The binding's RolaConfig has the size and field offsets that a C compiler gives rola_config_t."""
    fields = [f[0] for f in rl.RolaConfig._fields_]
    prog = tmp_path / "layout.c"
    body = "".join(f'    printf("%s %zu\\n", "{n}", offsetof(rola_config_t, {n}));\n' for n in fields)
    prog.write_text('#include <stdio.h>\n#include <stddef.h>\n#include "rola.h"\nint main(void) {\n'
                    '    printf("sizeof %zu\\n", sizeof(rola_config_t));\n' + body + "    return 0;\n}\n")
    exe = tmp_path / "layout"
    inc = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))), "include")
    subprocess.run(["gcc", "-std=c99", "-I", inc, str(prog), "-o", str(exe)], check=True)
    got = dict(line.split() for line in subprocess.run([str(exe)], capture_output=True, text=True,
                                                       check=True).stdout.splitlines())
    assert int(got["sizeof"]) == ctypes.sizeof(rl.RolaConfig)
    for n in fields:
        assert int(got[n]) == getattr(rl.RolaConfig, n).offset, n


def cfg_tiny(rl, **kw):
    from paper_2609_06712_gb300 import configs
    c = rl.make_config(configs.get("tiny"))
    for k, v in kw.items():
        setattr(c, k, v)
    return c


def test_defaults_and_sizes(rl):
    c = rl.RolaConfig()
    assert rl.library().rola_config_init(ctypes.byref(c)) == rl.ROLA_OK
    assert (c.d_h, c.block, list(c.rope_split), c.rope_theta) == (128, 64, [44, 42, 42], 10000.0)
    assert c.gate_bias == pytest.approx(-1.946) and c.eps_lr == pytest.approx(1e-6)
    assert c.lowrank_act == rl.ROLA_LOWRANK_ACT_SILU and c.block_geometry == rl.ROLA_BLOCK_FLAT
    assert c.lowrank_rope == rl.ROLA_LOWRANK_ROPE_OUTSIDE and c.wait_limit_ms == 0 and c.debug_flags == 0
    from paper_2609_06712_gb300 import configs
    for name, nb, nk in [("tiny", 16, 2), ("wan13b_480p", 512, 51), ("wan14b_720p", 1182, 118),
                         ("wan14b_720p_long", 2307, 231)]:
        cc = rl.make_config(configs.get(name))
        assert rl.num_blocks(cc) == nb and rl.num_keep(cc) == nk
        assert rl.workspace_bytes(cc) > 0


def call_all(rl, c, ws_bytes=1 << 30, ptr=0x10000, ws=0x100000):
    """Every compute entry point with dummy (never dereferenced) pointers."""
    L = rl.library()
    P = ctypes.c_void_p
    p, w = P(ptr), P(ws)
    b = ctypes.byref(c)
    return [
        L.rola_block_mask(b, p, p, p, w, ws_bytes, None),
        L.rola_sparse_attn(b, p, p, p, p, p, w, ws_bytes, None),
        L.rola_lowrank_summary(b, p, p, p, p, None, w, ws_bytes, None),
        L.rola_lowrank_apply(b, p, p, p, None, p, p, w, ws_bytes, None),
        L.rola_forward(b, p, p, p, p, p, None, p, None, w, ws_bytes, None),
        L.rola_out_proj(b, p, p, None, 256, p, w, ws_bytes, None),
        L.rola_attention_block(b, p, p, -1.946, 256, p, p, p, p, p, p, None, p, p, p, None, w, ws_bytes, None),
    ]


@pytest.mark.parametrize("field,value,code", [
    ("N", 1000, 1),            # N != T*Hh*Ww
    ("B", 0, 1),
    ("d_h", 64, 2),            # valid shape, not built
    ("block", 128, 2),
    ("r", 12, 2),              # even but not a multiple of 8
    ("r", 15, 1),
    ("r", 256, 1),             # r > d_h
    ("keep_ratio", 1.5, 1),
    ("keep_ratio", float("nan"), 1),
    ("rope_theta", 0.0, 1),
    ("eps_lr", -1.0, 1),
    ("dtype", 7, 1),
    ("wait_limit_ms", -1, 1),
    ("wait_limit_ms", 60001, 1),
    ("debug_flags", 2, 1),
    ("lowrank_rope", 3, 1),
    ("lowrank_rope", -1, 1),
    ("lowrank_act", 5, 1),
    ("lowrank_act", -1, 1),
    ("block_geometry", 2, 1),
    ("block_geometry", -1, 1),
])
def test_invalid_config_is_rejected_before_launch(rl, field, value, code):
    c = cfg_tiny(rl, **{field: value})
    assert all(s == code for s in call_all(rl, c)), call_all(rl, c)
    assert rl.workspace_bytes(c) == 0 and rl.num_keep(c) == 0


def test_kept_block_count_limit(rl):
    """B*H*nB*n_keep must stay below 2^31: the sparse kernel counts a CTA's kept blocks in 32 bits."""
    N = 5793 * 64                                    # nB = 5793; 64 * 5793^2 just exceeds 2^31
    big = cfg_tiny(rl, H=64, N=N, T=1, Hh=1, Ww=N, keep_ratio=1.0)
    assert all(s == rl.ROLA_ERR_UNSUPPORTED for s in call_all(rl, big))
    assert rl.workspace_bytes(big) == 0
    half = cfg_tiny(rl, H=64, N=N, T=1, Hh=1, Ww=N, keep_ratio=0.5)
    assert rl.num_keep(half) == 2897 and rl.workspace_bytes(half) > 0


def test_cube_geometry_sizes(rl):
    """Cube geometry: nB is the cube count of the latent grid, n_keep rounds on it, and the
    workspace grows by the padded cube-ordered copies (q^r, k^r and v)."""
    from oracle import oracle as O
    from paper_2609_06712_gb300 import configs
    for T, Hh, Ww in [(5, 9, 13), (21, 45, 80), (1, 1, 3), (4, 16, 16)]:
        cfg = dict(configs.get("tiny"), T=T, Hh=Hh, Ww=Ww, N=T * Hh * Ww, keep=0.1)
        flat = rl.make_config(cfg)
        cube = rl.make_config(dict(cfg, block_geometry="cube"))
        nb = -(-T // 4) * -(-Hh // 4) * -(-Ww // 4)
        assert rl.num_blocks(cube) == nb == O.num_blocks(dict(cfg, block_geometry="cube"))
        assert rl.num_keep(cube) == O.num_keep(dict(cfg, block_geometry="cube"))
        assert rl.workspace_bytes(cube) > rl.workspace_bytes(flat) or nb * 64 == T * Hh * Ww
    # more blocks than the top-k kernel holds
    big = rl.make_config(dict(configs.get("tiny"), T=1, Hh=1, Ww=7009 * 64, N=7009 * 64, keep=0.01))
    assert rl.num_blocks(big) == 0 and rl.workspace_bytes(big) == 0


def test_rope_split_must_sum_to_head_dim(rl):
    c = cfg_tiny(rl)
    c.rope_split[:] = [44, 42, 40]
    assert all(s == rl.ROLA_ERR_INVALID_ARG for s in call_all(rl, c))
    c.rope_split[:] = [43, 43, 42]
    assert all(s == rl.ROLA_ERR_INVALID_ARG for s in call_all(rl, c))


def test_null_and_misaligned_pointers(rl):
    c = cfg_tiny(rl)
    assert all(s == rl.ROLA_ERR_INVALID_ARG for s in call_all(rl, c, ptr=0))
    assert all(s == rl.ROLA_ERR_INVALID_ARG for s in call_all(rl, c, ptr=0x10008))


def test_workspace_checks(rl):
    c = cfg_tiny(rl)
    need = rl.workspace_bytes(c)
    short = call_all(rl, c, ws_bytes=need - 1)
    del short[5]                       # rola_out_proj needs only the 256-byte status word
    assert all(s == rl.ROLA_ERR_WORKSPACE for s in short)
    assert all(s == rl.ROLA_ERR_WORKSPACE for s in call_all(rl, c, ws=0x100080))   # not 256-aligned
    assert all(s == rl.ROLA_ERR_WORKSPACE for s in call_all(rl, c, ws=0))


def test_status_strings(rl):
    L = rl.library()
    for code in range(6):
        assert L.rola_status_string(code).decode().startswith("ROLA_")
    assert b"unknown" in L.rola_status_string(42)


def test_training_entry_points_are_checked_before_launch(rl):
    """rola_forward_train and rola_backward reject bad arguments before any launch: an invalid
    config, missing saved tensors, a short or misaligned workspace."""
    L = rl.library()
    P = ctypes.c_void_p
    p, w = P(0x10000), P(0x100000)
    c = cfg_tiny(rl)
    bad = cfg_tiny(rl, r=15)
    cube = cfg_tiny(rl, block_geometry=rl.ROLA_BLOCK_CUBE)
    need = L.rola_backward_workspace_bytes(ctypes.byref(c))
    assert need > rl.workspace_bytes(c) and L.rola_backward_workspace_bytes(ctypes.byref(cube)) > need
    assert L.rola_backward_workspace_bytes(ctypes.byref(bad)) == 0

    def bwd(cfg, ptr=p, ws=w, ws_bytes=1 << 40):
        return L.rola_backward(ctypes.byref(cfg), *([ptr] * 17), ws, ws_bytes, None)

    assert bwd(bad) == rl.ROLA_ERR_INVALID_ARG
    assert bwd(c, ptr=P(0)) == rl.ROLA_ERR_INVALID_ARG
    assert bwd(c, ptr=P(0x10008)) == rl.ROLA_ERR_INVALID_ARG
    assert bwd(c, ws_bytes=need - 1) == rl.ROLA_ERR_WORKSPACE
    assert bwd(c, ws=P(0x100080)) == rl.ROLA_ERR_WORKSPACE

    def fwd(cfg, o_s=p, lse=p, C=p, kv=p, ws_bytes=1 << 40):
        return L.rola_forward_train(ctypes.byref(cfg), p, p, p, p, p, None, P(0x20000), kv, o_s, lse, C, w,
                                    ws_bytes, None)

    assert fwd(bad) == rl.ROLA_ERR_INVALID_ARG
    for missing in ({"o_s": None}, {"lse": None}, {"C": None}, {"kv": None}):
        assert fwd(c, **missing) == rl.ROLA_ERR_INVALID_ARG
    assert fwd(c, o_s=P(0x20000)) == rl.ROLA_ERR_INVALID_ARG           # o_s may not alias o
    assert fwd(c, ws_bytes=rl.workspace_bytes(c) - 1) == rl.ROLA_ERR_WORKSPACE


def test_gate_arguments_are_checked_before_launch(rl):
    """Every call here is rejected by validation, so no kernel is launched on the dummy pointers."""
    L = rl.library()
    c = rl.make_config({"B": 1, "H": 2, "N": 1024, "T": 4, "Hh": 16, "Ww": 16, "keep": 0.125, "r": 16})
    P = ctypes.c_void_p
    ok, mis = P(0x10000), P(0x10004)
    b = ctypes.byref(c)
    for d_model in (0, 4, 12, -8):
        assert L.rola_gate(b, ok, ok, -1.946, d_model, ok, None) == rl.ROLA_ERR_INVALID_ARG
    assert L.rola_gate(b, None, ok, -1.946, 128, ok, None) == rl.ROLA_ERR_INVALID_ARG
    assert L.rola_gate(b, mis, ok, -1.946, 128, ok, None) == rl.ROLA_ERR_INVALID_ARG
    assert L.rola_gate(b, ok, ok, float("nan"), 128, ok, None) == rl.ROLA_ERR_INVALID_ARG
    c.N = 1000                                   # N != T * Hh * Ww
    assert L.rola_gate(b, ok, ok, -1.946, 128, ok, None) == rl.ROLA_ERR_INVALID_ARG


def test_out_proj_arguments_are_checked_before_launch(rl):
    """rola_out_proj: d_model a positive multiple of 64, 16-byte aligned operands, and a 256-byte
    aligned status word of at least 256 bytes -- each refused before any launch."""
    L = rl.library()
    P = ctypes.c_void_p
    c = cfg_tiny(rl)
    b, p, w = ctypes.byref(c), P(0x10000), P(0x100000)
    assert L.rola_out_proj(b, p, p, None, 96, p, w, 4096, None) == rl.ROLA_ERR_INVALID_ARG
    assert L.rola_out_proj(b, p, p, None, 0, p, w, 4096, None) == rl.ROLA_ERR_INVALID_ARG
    assert L.rola_out_proj(b, P(0x10008), p, None, 128, p, w, 4096, None) == rl.ROLA_ERR_INVALID_ARG
    assert L.rola_out_proj(b, p, p, ctypes.cast(P(0x10004), ctypes.POINTER(ctypes.c_float)), 128, p, w, 4096,
                           None) == rl.ROLA_ERR_INVALID_ARG
    assert L.rola_out_proj(b, None, p, None, 128, p, w, 4096, None) == rl.ROLA_ERR_INVALID_ARG
    assert L.rola_out_proj(b, p, p, None, 128, p, w, 128, None) == rl.ROLA_ERR_WORKSPACE
    assert L.rola_out_proj(b, p, p, None, 128, p, P(0x100010), 4096, None) == rl.ROLA_ERR_WORKSPACE
    assert L.rola_out_proj(b, p, p, None, 128, p, None, 4096, None) == rl.ROLA_ERR_WORKSPACE
