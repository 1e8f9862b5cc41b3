"""fp64 CPU oracle for the RoLA hybrid attention module -- TEST INFRASTRUCTURE.

Only ``tests/``, ``__graft_entry__.smoke()`` and ``bench.py``'s CPU-baseline
leg may import this module.  It wraps ``rola_oracle.c`` (plain C, fp64,
OpenMP) through ctypes and takes / returns numpy arrays.  It imports nothing
from the CUDA library and the CUDA library imports nothing from it.

Each wrapper names the passage of the paper it follows; the C file states the
steps.  Configuration is a plain dict with the keys of ``OracleConfig`` below.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "rola_oracle.c")
_LIB = os.path.join(_HERE, "liboracle.so")
_lock = threading.Lock()
_lib = None


def build(force: bool = False) -> str:
    """Compile rola_oracle.c into liboracle.so with gcc (-O2, OpenMP, no fast-math, and no
    contraction of a * b + c into an fma, so each expression rounds as written on every host)."""
    if force or not os.path.exists(_LIB) or os.path.getmtime(_LIB) < os.path.getmtime(_SRC):
        tmp = _LIB + f".tmp{os.getpid()}"
        subprocess.check_call(["gcc", "-O2", "-fopenmp", "-fPIC", "-shared", "-std=c99", "-ffp-contract=off",
                               "-o", tmp, _SRC, "-lm"])
        os.replace(tmp, _LIB)
    return _LIB


class OracleConfig(ctypes.Structure):
    _fields_ = [
        ("B", ctypes.c_int32), ("H", ctypes.c_int32), ("N", ctypes.c_int32), ("dh", ctypes.c_int32),
        ("T", ctypes.c_int32), ("Hh", ctypes.c_int32), ("Ww", ctypes.c_int32),
        ("pos_offset", ctypes.c_int32 * 3),
        ("split", ctypes.c_int32 * 3),
        ("theta", ctypes.c_double),
        ("block", ctypes.c_int32),
        ("keep", ctypes.c_double),
        ("r", ctypes.c_int32),
        ("eps_lr", ctypes.c_double), ("eps_f", ctypes.c_double),
        ("gate_bias", ctypes.c_double),
        ("rope_mode", ctypes.c_int32),
        ("act", ctypes.c_int32),
        ("geometry", ctypes.c_int32),
        ("qblock", ctypes.c_int32),
    ]


ROPE_OUTSIDE, ROPE_INSIDE, ROPE_NONE = 0, 1, 2
# feature maps of the activation ablation (Tab. abl_activation), by the name a config dict uses
ACTIVATIONS = {"silu": 0, "identity": 1, "tanh": 2, "relu": 3, "gelu": 4}
# block geometries: contiguous 64-token chunks, or 4 x 4 x 4 cubes of the latent grid
GEOMETRIES = {"flat": 0, "cube": 1}


def _get():
    global _lib
    with _lock:
        if _lib is None:
            # ORACLE_LIB points the pins at a deliberately broken copy (mutation test)
            path = os.environ.get("ORACLE_LIB") or build()
            lib = ctypes.CDLL(path)
            P = ctypes.c_void_p
            cfgp = ctypes.POINTER(OracleConfig)
            lib.orc_num_blocks.argtypes = [cfgp]
            lib.orc_num_keep.argtypes = [cfgp]
            lib.orc_block_of.argtypes = [cfgp, ctypes.c_int]
            lib.orc_num_qblocks.argtypes = [cfgp]
            lib.orc_qblock_of.argtypes = [cfgp, ctypes.c_int]
            lib.orc_position.argtypes = [cfgp, ctypes.c_int, P]
            lib.orc_pair_angle.argtypes = [cfgp, ctypes.c_int, P]
            lib.orc_pair_angle.restype = ctypes.c_double
            lib.orc_activation.argtypes = [cfgp, ctypes.c_double]
            lib.orc_activation.restype = ctypes.c_double
            lib.orc_activation_grad.argtypes = [cfgp, ctypes.c_double]
            lib.orc_activation_grad.restype = ctypes.c_double
            lib.orc_backward.argtypes = [cfgp] + [P] * 14
            lib.orc_rotate.argtypes = [cfgp, ctypes.c_int, P, P, P, ctypes.c_int]
            lib.orc_lowrank_features.argtypes = [cfgp, P, P, P]
            lib.orc_lowrank_summary.argtypes = [cfgp, P, P, P, P, P]
            lib.orc_lowrank_apply.argtypes = [cfgp, P, P, P, P, P, P, P]
            lib.orc_lowrank_readout.argtypes = [cfgp, P, P, P, P]
            lib.orc_lowrank_explicit.argtypes = [cfgp, P, P, P, P, P, P]
            lib.orc_rope_full.argtypes = [cfgp, P, P]
            lib.orc_block_mask.argtypes = [cfgp, P, P, P, P, P, P]
            lib.orc_block_mask_f32.argtypes = [cfgp, P, P, P, P]
            lib.orc_sparse_attn.argtypes = [cfgp, P, P, P, P, ctypes.c_int, P, P]
            lib.orc_forward.argtypes = [cfgp, P, P, P, P, P, P, P, P, P, P, P, P, P]
            lib.orc_gate.argtypes = [ctypes.c_int, ctypes.c_int, ctypes.c_int, P, P, ctypes.c_double, P]
            lib.orc_out_proj.argtypes = [ctypes.c_int] * 5 + [P] * 5
            _lib = lib
    return _lib


def make_config(cfg: dict, rope_mode: int = ROPE_OUTSIDE) -> OracleConfig:
    """Oracle configuration from a plain dict (the keys the tests use)."""
    c = OracleConfig()
    c.B, c.H, c.N, c.dh = cfg["B"], cfg["H"], cfg["N"], cfg.get("d_h", 128)
    c.T, c.Hh, c.Ww = cfg["T"], cfg["Hh"], cfg["Ww"]
    c.pos_offset[:] = list(cfg.get("pos_offset", (0, 0, 0)))
    c.split[:] = list(cfg.get("rope_split", (44, 42, 42)))
    c.theta = float(cfg.get("rope_theta", 10000.0))
    c.block = cfg.get("block", 64)
    # the keep ratio crosses the C ABI as a float32; the oracle rounds the same value
    c.keep = float(np.float32(cfg["keep"]))
    c.r = cfg["r"]
    c.eps_lr = float(np.float32(cfg.get("eps_lr", 1e-6)))
    c.eps_f = float(np.float32(cfg.get("eps_fuse", 1e-6)))
    c.gate_bias = float(np.float32(cfg.get("gate_bias", -1.946)))
    c.rope_mode = rope_mode
    c.act = ACTIVATIONS[cfg.get("lowrank_act", "silu")]
    c.geometry = GEOMETRIES[cfg.get("block_geometry", "flat")]
    # query-block size of the contiguous geometry (0: the key blocks' size)
    c.qblock = int(cfg.get("qblock", 0))
    if c.qblock < 0 or (c.qblock and c.geometry != GEOMETRIES["flat"]):
        raise ValueError("qblock is a size of contiguous query blocks (flat geometry only)")
    return c


def _f32(a):
    a = np.ascontiguousarray(a, dtype=np.float32)
    return a, a.ctypes.data


def _ptr(a):
    return None if a is None else a.ctypes.data


def activation(name: str, x: float) -> float:
    """The feature map phi of Eq. (qklr) (Tab. abl_activation), one fp64 value."""
    c = make_config({"B": 1, "H": 1, "N": 1, "T": 1, "Hh": 1, "Ww": 1, "keep": 1.0, "r": 2,
                     "lowrank_act": name})
    return _get().orc_activation(ctypes.byref(c), float(x))


def activation_grad(name: str, x: float) -> float:
    """phi'(x) of the feature map, one fp64 value (the backward pass's derivative)."""
    c = make_config({"B": 1, "H": 1, "N": 1, "T": 1, "Hh": 1, "Ww": 1, "keep": 1.0, "r": 2,
                     "lowrank_act": name})
    return _get().orc_activation_grad(ctypes.byref(c), float(x))


def backward(cfg: dict, q, k, v, Pq, Pk, gate, kv_idx, dO, rope_mode: int = ROPE_OUTSIDE) -> dict:
    """Gradients of sum(dO * O) through the forward pass under the mask kv_idx: dq, dk, dv
    [B,H,N,dh], dP_q, dP_k [H,r,dh] (summed over the batch) and dgate [B,N] (summed over heads)."""
    c = make_config(cfg, rope_mode)
    q, qp = _f32(q)
    k, kp = _f32(k)
    v, vp = _f32(v)
    Pq, Pqp = _f32(Pq)
    Pk, Pkp = _f32(Pk)
    g = None if gate is None else np.ascontiguousarray(gate, dtype=np.float32)
    idx = np.ascontiguousarray(kv_idx, dtype=np.int32)
    dO, dOp = _f32(dO)
    shape = (c.B, c.H, c.N, c.dh)
    out = {"dq": np.empty(shape), "dk": np.empty(shape), "dv": np.empty(shape),
           "dP_q": np.empty((c.H, c.r, c.dh)), "dP_k": np.empty((c.H, c.r, c.dh)), "dgate": np.empty((c.B, c.N))}
    _get().orc_backward(ctypes.byref(c), qp, kp, vp, Pqp, Pkp, _ptr(g), idx.ctypes.data, dOp,
                        *(out[n].ctypes.data for n in ("dq", "dk", "dv", "dP_q", "dP_k", "dgate")))
    return out


def num_blocks(cfg: dict) -> int:
    c = make_config(cfg)
    return _get().orc_num_blocks(ctypes.byref(c))


def num_keep(cfg: dict) -> int:
    c = make_config(cfg)
    return _get().orc_num_keep(ctypes.byref(c))


def num_qblocks(cfg: dict) -> int:
    """Query blocks: chunks of cfg["qblock"] tokens if set, else the key blocks."""
    c = make_config(cfg)
    return _get().orc_num_qblocks(ctypes.byref(c))


def qblock_of(cfg: dict) -> np.ndarray:
    """Query-block id of every token [N]."""
    c = make_config(cfg)
    lib = _get()
    return np.array([lib.orc_qblock_of(ctypes.byref(c), n) for n in range(c.N)], dtype=np.int64)


def block_of(cfg: dict) -> np.ndarray:
    """Block id of every token [N]: its 64-token chunk, or its 4 x 4 x 4 cube (t-major cube numbering)."""
    c = make_config(cfg)
    lib = _get()
    return np.array([lib.orc_block_of(ctypes.byref(c), n) for n in range(c.N)], dtype=np.int64)


def position(cfg: dict, n: int) -> np.ndarray:
    """(t, x, y) of flattened token n, Sec. 3 notation (t-major)."""
    c = make_config(cfg)
    out = np.zeros(3)
    _get().orc_position(ctypes.byref(c), n, out.ctypes.data)
    return out


def pair_angle(cfg: dict, m: int, pos) -> float:
    c = make_config(cfg)
    p = np.ascontiguousarray(pos, dtype=np.float64)
    return _get().orc_pair_angle(ctypes.byref(c), m, p.ctypes.data)


def rotate(cfg: dict, npairs: int, pos, x) -> np.ndarray:
    """R(pos) on the first 2*npairs coordinates of x (Sec. 3, Sec. 4.2)."""
    c = make_config(cfg)
    p = np.ascontiguousarray(pos, dtype=np.float64)
    xi = np.ascontiguousarray(x, dtype=np.float64)
    out = np.empty_like(xi)
    _get().orc_rotate(ctypes.byref(c), npairs, p.ctypes.data, xi.ctypes.data, out.ctypes.data, xi.size)
    return out


def lowrank_features(cfg: dict, x, P, rope_mode: int = ROPE_OUTSIDE) -> np.ndarray:
    """Eq. (qklr) features [B,H,N,r] (or the inside / no-RoPE ablations)."""
    c = make_config(cfg, rope_mode)
    x, xp = _f32(x)
    P, Pp = _f32(P)
    out = np.empty((c.B, c.H, c.N, c.r))
    _get().orc_lowrank_features(ctypes.byref(c), xp, Pp, out.ctypes.data)
    return out


def lowrank_summary(cfg: dict, k, v, Pk, rope_mode: int = ROPE_OUTSIDE):
    """Eq. (ctx): C = sum_q k~_q v_q^T [B,H,r,dh] and z = sum_q k~_q [B,H,r]."""
    c = make_config(cfg, rope_mode)
    k, kp = _f32(k)
    v, vp = _f32(v)
    Pk, Pkp = _f32(Pk)
    C = np.empty((c.B, c.H, c.r, c.dh))
    z = np.empty((c.B, c.H, c.r))
    _get().orc_lowrank_summary(ctypes.byref(c), kp, vp, Pkp, C.ctypes.data, z.ctypes.data)
    return C, z


def _sel(cfg: dict, qblocks):
    if qblocks is None:
        return None
    sel = np.zeros(num_qblocks(cfg), dtype=np.uint8)
    sel[np.asarray(qblocks, dtype=np.int64)] = 1
    return sel


def lowrank_apply(cfg: dict, q, Pq, C, gate, o_s, qblocks=None, rope_mode: int = ROPE_OUTSIDE):
    """Eq. (ctx) readout + RMSNorm, then Eq. (gate) fusion with O^s -> O [B,H,N,dh].

    Rows outside ``qblocks`` (query-block ids) are left as NaN."""
    c = make_config(cfg, rope_mode)
    q, qp = _f32(q)
    Pq, Pqp = _f32(Pq)
    C = np.ascontiguousarray(C, dtype=np.float64)
    g = None if gate is None else np.ascontiguousarray(gate, dtype=np.float32)
    o_s, osp = _f32(o_s)
    sel = _sel(cfg, qblocks)
    o = np.full((c.B, c.H, c.N, c.dh), np.nan)
    _get().orc_lowrank_apply(ctypes.byref(c), qp, Pqp, C.ctypes.data, _ptr(g), osp, _ptr(sel), o.ctypes.data)
    return o


def lowrank_readout(cfg: dict, q, Pq, C, rope_mode: int = ROPE_OUTSIDE) -> np.ndarray:
    """Pre-RMSNorm readout y_p = q~_p^T C [B,H,N,dh]."""
    c = make_config(cfg, rope_mode)
    q, qp = _f32(q)
    Pq, Pqp = _f32(Pq)
    C = np.ascontiguousarray(C, dtype=np.float64)
    y = np.empty((c.B, c.H, c.N, c.dh))
    _get().orc_lowrank_readout(ctypes.byref(c), qp, Pqp, C.ctypes.data, y.ctypes.data)
    return y


def gate(X, w, b: float) -> np.ndarray:
    """Token gate g = sigmoid(X w_g + b_g) of the gated fusion (Sec. fusion); X [B][N][D], w [D] -> [B][N]."""
    X, Xp = _f32(X)
    w, wp = _f32(w)
    B, N, D = X.shape
    assert w.shape == (D,)
    g = np.empty((B, N))
    _get().orc_gate(B, N, D, Xp, wp, float(b), g.ctypes.data)
    return g


def out_proj(O, W, bias=None, rows=None) -> np.ndarray:
    """Output projection of the block (Alg. 1, last step): the heads of O [B][H][N][dh] concatenated
    per token (head-major), times W^T, W [d_model][H*dh] (+ bias [d_model]) -> Y [B][N][d_model].
    ``rows``: token indices to compute (the other rows are NaN); None computes every token."""
    O = np.ascontiguousarray(O, dtype=np.float64)
    W, Wp = _f32(W)
    B, H, N, dh = O.shape
    d_model = W.shape[0]
    assert W.shape == (d_model, H * dh)
    b = None if bias is None else np.ascontiguousarray(bias, dtype=np.float32)
    sel = None
    if rows is not None:
        sel = np.zeros(N, dtype=np.uint8)
        sel[np.asarray(rows, dtype=np.int64)] = 1
    Y = np.full((B, N, d_model), np.nan)
    _get().orc_out_proj(B, N, H, dh, d_model, O.ctypes.data, Wp, _ptr(b), _ptr(sel), Y.ctypes.data)
    return Y


def lowrank_explicit(cfg: dict, q, k, v, Pq, Pk, rope_mode: int = ROPE_OUTSIDE) -> np.ndarray:
    """Explicit O(N^2) pre-RMSNorm form sum_q (q~_p . k~_q) v_q (Prop. exact)."""
    c = make_config(cfg, rope_mode)
    q, qp = _f32(q)
    k, kp = _f32(k)
    v, vp = _f32(v)
    Pq, Pqp = _f32(Pq)
    Pk, Pkp = _f32(Pk)
    y = np.empty((c.B, c.H, c.N, c.dh))
    _get().orc_lowrank_explicit(ctypes.byref(c), qp, kp, vp, Pqp, Pkp, y.ctypes.data)
    return y


def rope_full(cfg: dict, x) -> np.ndarray:
    """Full 3D RoPE R(p) x of every token (Alg. 1, sparse-branch input)."""
    c = make_config(cfg)
    x, xp = _f32(x)
    out = np.empty((c.B, c.H, c.N, c.dh))
    _get().orc_rope_full(ctypes.byref(c), xp, out.ctypes.data)
    return out


def block_mask(cfg: dict, q, k):
    """Pooled-score top-n_keep block mask.

    Returns (kv_idx int32 [B,H,nQB,n_keep] ascending, scores [B,H,nQB,nKB],
    gap [B,H,nQB], tau [B,H,nQB]); rows with gap <= tau are near-tie rows."""
    c = make_config(cfg)
    q, qp = _f32(q)
    k, kp = _f32(k)
    nb, nq, nk = num_blocks(cfg), num_qblocks(cfg), num_keep(cfg)
    idx = np.empty((c.B, c.H, nq, nk), dtype=np.int32)
    scores = np.empty((c.B, c.H, nq, nb))
    gap = np.empty((c.B, c.H, nq))
    tau = np.empty((c.B, c.H, nq))
    _get().orc_block_mask(ctypes.byref(c), qp, kp, idx.ctypes.data, scores.ctypes.data,
                          gap.ctypes.data, tau.ctypes.data)
    return idx, scores, gap, tau


def block_mask_f32(cfg: dict, q, k):
    """The block mask as an fp32 decision (the precision of the CUDA path), every rounding fixed:
    fp32 (cos, sin) table, fma rotation, pairwise pooling over the block's slots, one divide,
    ascending-d fma chain, one scale product, ties to the lower block.

    Returns (kv_idx int32 [B,H,nQB,n_keep] ascending, fp32 scores [B,H,nQB,nKB] as float64)."""
    c = make_config(cfg)
    q, qp = _f32(q)
    k, kp = _f32(k)
    nb, nq, nk = num_blocks(cfg), num_qblocks(cfg), num_keep(cfg)
    idx = np.empty((c.B, c.H, nq, nk), dtype=np.int32)
    scores = np.empty((c.B, c.H, nq, nb))
    _get().orc_block_mask_f32(ctypes.byref(c), qp, kp, idx.ctypes.data, scores.ctypes.data)
    return idx, scores


def sparse_attn(cfg: dict, qr, kr, v, kv_idx, qblocks=None) -> np.ndarray:
    """Block-sparse softmax attention over the kept key blocks.

    qr, kr: already-rotated q / k (float64); rows outside ``qblocks`` are NaN."""
    c = make_config(cfg)
    qr = np.ascontiguousarray(qr, dtype=np.float64)
    kr = np.ascontiguousarray(kr, dtype=np.float64)
    v, vp = _f32(v)
    kv = np.ascontiguousarray(kv_idx, dtype=np.int32)
    sel = _sel(cfg, qblocks)
    o = np.full((c.B, c.H, c.N, c.dh), np.nan)
    _get().orc_sparse_attn(ctypes.byref(c), qr.ctypes.data, kr.ctypes.data, vp, kv.ctypes.data,
                           kv.shape[-1], _ptr(sel), o.ctypes.data)
    return o


def forward(cfg: dict, q, k, v, Pq, Pk, gate=None, mask_override=None, qblocks=None,
            rope_mode: int = ROPE_OUTSIDE):
    """Alg. 1 per-head steps (RoPE, sparse branch, low-rank branch, fusion).

    Returns dict(o, kv_idx, o_s, C, z); rows outside ``qblocks`` are NaN in o / o_s."""
    c = make_config(cfg, rope_mode)
    q, qp = _f32(q)
    k, kp = _f32(k)
    v, vp = _f32(v)
    Pq, Pqp = _f32(Pq)
    Pk, Pkp = _f32(Pk)
    g = None if gate is None else np.ascontiguousarray(gate, dtype=np.float32)
    nq, nk = num_qblocks(cfg), num_keep(cfg)
    mo = None if mask_override is None else np.ascontiguousarray(mask_override, dtype=np.int32)
    sel = _sel(cfg, qblocks)
    shape = (c.B, c.H, c.N, c.dh)
    o = np.full(shape, np.nan)
    idx = np.empty((c.B, c.H, nq, nk), dtype=np.int32)
    o_s = np.empty(shape)
    C = np.empty((c.B, c.H, c.r, c.dh))
    z = np.empty((c.B, c.H, c.r))
    _get().orc_forward(ctypes.byref(c), qp, kp, vp, Pqp, Pkp, _ptr(g), _ptr(mo), _ptr(sel),
                       o.ctypes.data, idx.ctypes.data, o_s.ctypes.data, C.ctypes.data, z.ctypes.data)
    if sel is not None:
        rows = sel.astype(bool)[qblock_of(cfg)]
        o_s[:, :, ~rows, :] = np.nan
    return dict(o=o, kv_idx=idx, o_s=o_s, C=C, z=z)
