"""Thin Python binding of the C ABI in include/rola.h.

Argument marshalling only: every step of the module runs in the CUDA kernels
of librola.so.  Torch tensors supply device memory and the current stream.
Importing this module loads librola.so and raises if it is missing -- there is
no CPU fallback.
"""
from __future__ import annotations

import ctypes
import os

import torch

_PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_PKG, "librola.so")

ROLA_OK, ROLA_ERR_INVALID_ARG, ROLA_ERR_UNSUPPORTED, ROLA_ERR_WORKSPACE, ROLA_ERR_CUDA, ROLA_ERR_TIMEOUT = range(6)
ROLA_BF16, ROLA_FP32 = 0, 1


class RolaConfig(ctypes.Structure):
    """Mirror of rola_config_t."""
    _fields_ = [
        ("B", ctypes.c_int32), ("H", ctypes.c_int32), ("N", ctypes.c_int32), ("d_h", ctypes.c_int32),
        ("T", ctypes.c_int32), ("Hh", ctypes.c_int32), ("Ww", ctypes.c_int32),
        ("pos_offset", ctypes.c_int32 * 3),
        ("rope_split", ctypes.c_int32 * 3),
        ("rope_theta", ctypes.c_double),
        ("block", ctypes.c_int32),
        ("keep_ratio", ctypes.c_float),
        ("r", ctypes.c_int32),
        ("eps_lr", ctypes.c_float),
        ("eps_fuse", ctypes.c_float),
        ("gate_bias", ctypes.c_float),
        ("dtype", ctypes.c_int32),
        ("wait_limit_ms", ctypes.c_int32),
        ("debug_flags", ctypes.c_int32),
        ("lowrank_rope", ctypes.c_int32),
        ("lowrank_act", ctypes.c_int32),
        ("block_geometry", ctypes.c_int32),
        ("query_block", ctypes.c_int32),
    ]


ROLA_DEBUG_SKIP_FIRST_K_COPY = 1
# rola_lowrank_rope_t: where the truncated RoPE sits in the low-rank features
ROLA_LOWRANK_ROPE_OUTSIDE, ROLA_LOWRANK_ROPE_INSIDE, ROLA_LOWRANK_ROPE_NONE = 0, 1, 2
# rola_lowrank_act_t: the feature map of the low-rank features, and the names a config dict uses
(ROLA_LOWRANK_ACT_SILU, ROLA_LOWRANK_ACT_IDENTITY, ROLA_LOWRANK_ACT_TANH, ROLA_LOWRANK_ACT_RELU,
 ROLA_LOWRANK_ACT_GELU) = 0, 1, 2, 3, 4
LOWRANK_ACTS = {"silu": ROLA_LOWRANK_ACT_SILU, "identity": ROLA_LOWRANK_ACT_IDENTITY,
                "tanh": ROLA_LOWRANK_ACT_TANH, "relu": ROLA_LOWRANK_ACT_RELU, "gelu": ROLA_LOWRANK_ACT_GELU}
# rola_block_geometry_t: contiguous 64-token chunks, or 4 x 4 x 4 cubes of the latent grid
ROLA_BLOCK_FLAT, ROLA_BLOCK_CUBE = 0, 1
BLOCK_GEOMETRIES = {"flat": ROLA_BLOCK_FLAT, "cube": ROLA_BLOCK_CUBE}


class RolaError(RuntimeError):
    def __init__(self, status: int, where: str):
        self.status = status
        super().__init__(f"{where}: {_lib.rola_status_string(status).decode()}")


def _load():
    if not os.path.exists(LIB_PATH):
        raise ImportError(f"{LIB_PATH} is missing: build it with paper_2609_06712_gb300.build.build() "
                          "(the RoLA module has no CPU fallback)")
    lib = ctypes.CDLL(LIB_PATH)
    P, S = ctypes.c_void_p, ctypes.c_size_t
    cfgp = ctypes.POINTER(RolaConfig)
    st = ctypes.c_int
    sig = {
        "rola_config_init": (st, [cfgp]),
        "rola_num_blocks": (ctypes.c_int32, [cfgp]),
        "rola_num_keep": (ctypes.c_int32, [cfgp]),
        "rola_num_query_blocks": (ctypes.c_int32, [cfgp]),
        "rola_workspace_bytes": (S, [cfgp]),
        "rola_block_mask": (st, [cfgp, P, P, P, P, S, P]),
        "rola_sparse_attn": (st, [cfgp, P, P, P, P, P, P, S, P]),
        "rola_lowrank_summary": (st, [cfgp, P, P, P, P, P, P, S, P]),
        "rola_lowrank_summary_static": (st, [cfgp, P, P, P, P, P, P]),
        "rola_lowrank_apply": (st, [cfgp, P, P, P, P, P, P, P, S, P]),
        "rola_forward": (st, [cfgp, P, P, P, P, P, P, P, P, P, S, P]),
        "rola_forward_timed": (st, [cfgp, P, P, P, P, P, P, P, P, P, S, P, P]),
        "rola_forward_train": (st, [cfgp, P, P, P, P, P, P, P, P, P, P, P, P, S, P]),
        "rola_backward_workspace_bytes": (S, [cfgp]),
        "rola_backward": (st, [cfgp] + [P] * 18 + [S, P]),
        "rola_gate": (st, [cfgp, P, P, ctypes.c_float, ctypes.c_int32, P, P]),
        "rola_out_proj": (st, [cfgp, P, P, P, ctypes.c_int32, P, P, S, P]),
        "rola_attention_block": (st, [cfgp, P, P, ctypes.c_float, ctypes.c_int32] + [P] * 12 + [S, P]),
        "rola_get_device_status": (st, [P, P]),
        "rola_status_string": (ctypes.c_char_p, [st]),
    }
    for name, (res, args) in sig.items():
        fn = getattr(lib, name)
        fn.restype = res
        fn.argtypes = args
    return lib


_lib = _load()


def library():
    """The loaded ctypes library (for tests that call the ABI directly)."""
    return _lib


def make_config(cfg: dict, dtype: int = ROLA_BF16) -> RolaConfig:
    """rola_config_t from a plain dict of layer sizes (see configs.py)."""
    c = RolaConfig()
    _lib.rola_config_init(ctypes.byref(c))
    c.B, c.H, c.N = cfg["B"], cfg["H"], cfg["N"]
    c.d_h = cfg.get("d_h", 128)
    c.T, c.Hh, c.Ww = cfg["T"], cfg["Hh"], cfg["Ww"]
    c.pos_offset[:] = list(cfg.get("pos_offset", (0, 0, 0)))
    c.rope_split[:] = list(cfg.get("rope_split", (44, 42, 42)))
    c.rope_theta = float(cfg.get("rope_theta", 10000.0))
    c.block = cfg.get("block", 64)
    c.keep_ratio = float(cfg["keep"])
    c.r = cfg["r"]
    c.eps_lr = float(cfg.get("eps_lr", 1e-6))
    c.eps_fuse = float(cfg.get("eps_fuse", 1e-6))
    c.gate_bias = float(cfg.get("gate_bias", -1.946))
    c.dtype = dtype
    c.lowrank_rope = int(cfg.get("lowrank_rope", ROLA_LOWRANK_ROPE_OUTSIDE))
    act = cfg.get("lowrank_act", "silu")
    c.lowrank_act = LOWRANK_ACTS[act] if isinstance(act, str) else int(act)
    geom = cfg.get("block_geometry", "flat")
    c.block_geometry = BLOCK_GEOMETRIES[geom] if isinstance(geom, str) else int(geom)
    c.query_block = int(cfg.get("qblock", 0))
    return c


def _p(t):
    if t is None:
        return None
    if not (t.is_cuda and t.is_contiguous()):
        raise ValueError("RoLA tensors must be contiguous CUDA tensors")
    return ctypes.c_void_p(t.data_ptr())


def _stream(stream=None):
    s = torch.cuda.current_stream() if stream is None else stream
    return ctypes.c_void_p(s.cuda_stream)


def _check(status: int, where: str):
    if status != ROLA_OK:
        raise RolaError(status, where)


def num_blocks(c: RolaConfig) -> int:
    return _lib.rola_num_blocks(ctypes.byref(c))


def num_query_blocks(c: RolaConfig) -> int:
    """Rows of kv_idx: 128-token query chunks when c.query_block is 128, else the key blocks."""
    return _lib.rola_num_query_blocks(ctypes.byref(c))


def num_keep(c: RolaConfig) -> int:
    return _lib.rola_num_keep(ctypes.byref(c))


def workspace_bytes(c: RolaConfig) -> int:
    return _lib.rola_workspace_bytes(ctypes.byref(c))


def workspace(c: RolaConfig, device="cuda") -> torch.Tensor:
    """A workspace tensor of rola_workspace_bytes(c) bytes (torch allocations are 256-byte aligned)."""
    n = workspace_bytes(c)
    if n == 0:
        raise RolaError(ROLA_ERR_INVALID_ARG, "rola_workspace_bytes")
    return torch.empty(n, dtype=torch.uint8, device=device)


def block_mask(c, q, k, kv_idx, ws, stream=None):
    _check(_lib.rola_block_mask(ctypes.byref(c), _p(q), _p(k), _p(kv_idx), _p(ws), ws.numel(), _stream(stream)),
           "rola_block_mask")


def sparse_attn(c, q, k, v, kv_idx, o_s, ws, stream=None):
    _check(_lib.rola_sparse_attn(ctypes.byref(c), _p(q), _p(k), _p(v), _p(kv_idx), _p(o_s), _p(ws), ws.numel(),
                                 _stream(stream)), "rola_sparse_attn")


def lowrank_summary(c, k, v, P_k, C, z, ws, stream=None):
    _check(_lib.rola_lowrank_summary(ctypes.byref(c), _p(k), _p(v), _p(P_k), _p(C), _p(z), _p(ws), ws.numel(),
                                     _stream(stream)), "rola_lowrank_summary")


def lowrank_summary_static(c, k, v, P_k, C, z, stream=None):
    """The summary with no workspace: scratch lives in the library's static device array."""
    _check(_lib.rola_lowrank_summary_static(ctypes.byref(c), _p(k), _p(v), _p(P_k), _p(C), _p(z),
                                            _stream(stream)), "rola_lowrank_summary_static")


def lowrank_apply(c, q, P_q, C, gate, o_s, o, ws, stream=None):
    _check(_lib.rola_lowrank_apply(ctypes.byref(c), _p(q), _p(P_q), _p(C), _p(gate), _p(o_s), _p(o), _p(ws),
                                   ws.numel(), _stream(stream)), "rola_lowrank_apply")


def forward(c, q, k, v, P_q, P_k, gate, o, kv_idx_out, ws, stream=None):
    _check(_lib.rola_forward(ctypes.byref(c), _p(q), _p(k), _p(v), _p(P_q), _p(P_k), _p(gate), _p(o),
                             _p(kv_idx_out), _p(ws), ws.numel(), _stream(stream)), "rola_forward")


def forward_train(c, q, k, v, P_q, P_k, gate, o, kv_idx_out, o_s, lse, C, ws, stream=None):
    """rola_forward keeping O^s, the per-row log-sum-exp and C for backward()."""
    _check(_lib.rola_forward_train(ctypes.byref(c), _p(q), _p(k), _p(v), _p(P_q), _p(P_k), _p(gate), _p(o),
                                   _p(kv_idx_out), _p(o_s), _p(lse), _p(C), _p(ws), ws.numel(), _stream(stream)),
           "rola_forward_train")


def backward_workspace(c: RolaConfig, device="cuda") -> torch.Tensor:
    n = _lib.rola_backward_workspace_bytes(ctypes.byref(c))
    if n == 0:
        raise RolaError(ROLA_ERR_UNSUPPORTED, "rola_backward_workspace_bytes")
    return torch.empty(n, dtype=torch.uint8, device=device)


def backward(c, q, k, v, P_q, P_k, gate, kv_idx, o_s, lse, C, dO, dq, dk, dv, dP_q, dP_k, dgate, ws, stream=None):
    _check(_lib.rola_backward(ctypes.byref(c), _p(q), _p(k), _p(v), _p(P_q), _p(P_k), _p(gate), _p(kv_idx),
                              _p(o_s), _p(lse), _p(C), _p(dO), _p(dq), _p(dk), _p(dv), _p(dP_q), _p(dP_k),
                              _p(dgate), _p(ws), ws.numel(), _stream(stream)), "rola_backward")


def gate(c, X, w_g, b_g: float, gate_out, stream=None):
    """Token gate g = sigmoid(X w_g + b_g) into gate_out (fp32 [B][N]); X [B][N][d_model]."""
    _check(_lib.rola_gate(ctypes.byref(c), _p(X), _p(w_g), float(b_g), int(X.shape[-1]), _p(gate_out),
                          _stream(stream)), "rola_gate")


def out_proj(c, O, W_o, b_o, Y, ws, stream=None):
    """Y = concat_h(O) W_o^T (+ b_o): O [B][H][N][128], W_o [d_model][H*128], b_o fp32 [d_model] or
    None, Y [B][N][d_model] (the block's output projection)."""
    _check(_lib.rola_out_proj(ctypes.byref(c), _p(O), _p(W_o), _p(b_o), int(W_o.shape[0]), _p(Y), _p(ws),
                              ws.numel(), _stream(stream)), "rola_out_proj")


def attention_block(c, X, w_g, b_g: float, q, k, v, P_q, P_k, W_o, b_o, gate, o, Y, kv_idx_out, ws, stream=None):
    """The block after the QKV projection: gate from X, the RoLA module, the output projection."""
    _check(_lib.rola_attention_block(ctypes.byref(c), _p(X), _p(w_g), float(b_g), int(X.shape[-1]), _p(q), _p(k),
                                     _p(v), _p(P_q), _p(P_k), _p(W_o), _p(b_o), _p(gate), _p(o), _p(Y),
                                     _p(kv_idx_out), _p(ws), ws.numel(), _stream(stream)), "rola_attention_block")


def forward_timed(c, q, k, v, P_q, P_k, gate, o, kv_idx_out, ws, events, stream=None):
    """rola_forward recording 5 stage events (torch.cuda.Event, already created)."""
    arr = (ctypes.c_void_p * 5)(*[ctypes.c_void_p(e.cuda_event) for e in events])
    _check(_lib.rola_forward_timed(ctypes.byref(c), _p(q), _p(k), _p(v), _p(P_q), _p(P_k), _p(gate), _p(o),
                                   _p(kv_idx_out), _p(ws), ws.numel(), _stream(stream), arr),
           "rola_forward_timed")


def get_device_status(ws, stream=None) -> int:
    return _lib.rola_get_device_status(_p(ws), _stream(stream))


class RoLAAttention:
    """Convenience wrapper: owns the workspace for one layer shape and runs rola_forward.

    ``__call__(q, k, v, P_q, P_k, gate=None)`` returns (o, kv_idx) as new tensors."""

    def __init__(self, cfg: dict, dtype: int = ROLA_BF16, device="cuda"):
        self.cfg = make_config(cfg, dtype)
        self.ws = workspace(self.cfg, device)
        self.nB = num_blocks(self.cfg)
        self.n_keep = num_keep(self.cfg)

    def __call__(self, q, k, v, P_q, P_k, gate=None, out=None, kv_idx=None, stream=None):
        c = self.cfg
        if out is None:
            out = torch.empty_like(q)
        if kv_idx is None:
            kv_idx = torch.empty((c.B, c.H, self.nB, self.n_keep), dtype=torch.int32, device=q.device)
        forward(c, q, k, v, P_q, P_k, gate, out, kv_idx, self.ws, stream)
        return out, kv_idx


class RoLAFunction(torch.autograd.Function):
    """The module as a differentiable torch op on this library's kernels:
    rola_forward_train in forward, rola_backward in backward (torch allocates the
    buffers and casts the fp32 P gradients to P's dtype; it computes nothing else).

    ``RoLAFunction.apply(c, q, k, v, P_q, P_k, gate)`` returns O; ``gate`` may be None."""

    @staticmethod
    def forward(ctx, c, q, k, v, P_q, P_k, gate):
        B, H, N = c.B, c.H, c.N
        dev = q.device
        ws = workspace(c, dev)
        o = torch.empty_like(q)
        o_s = torch.empty_like(q)
        kv = torch.empty((B, H, num_blocks(c), num_keep(c)), dtype=torch.int32, device=dev)
        lse = torch.empty((B, H, N), dtype=torch.float32, device=dev)
        C = torch.empty((B, H, c.r, 128), dtype=torch.float32, device=dev)
        forward_train(c, q, k, v, P_q, P_k, gate, o, kv, o_s, lse, C, ws)
        ctx.c = c
        ctx.has_gate = gate is not None
        ctx.save_for_backward(q, k, v, P_q, P_k, gate if gate is not None else torch.empty(0, device=dev),
                              kv, o_s, lse, C)
        return o

    @staticmethod
    def backward(ctx, dO):
        q, k, v, P_q, P_k, gate, kv, o_s, lse, C = ctx.saved_tensors
        c = ctx.c
        gate = gate if ctx.has_gate else None
        dO = dO.contiguous()
        dq, dk, dv = torch.empty_like(q), torch.empty_like(k), torch.empty_like(v)
        dP_q = torch.empty(P_q.shape, dtype=torch.float32, device=q.device)
        dP_k = torch.empty(P_k.shape, dtype=torch.float32, device=q.device)
        dgate = torch.empty((c.B, c.N), dtype=torch.float32, device=q.device) if ctx.has_gate else None
        ws = backward_workspace(c, q.device)
        backward(c, q, k, v, P_q, P_k, gate, kv, o_s, lse, C, dO, dq, dk, dv, dP_q, dP_k, dgate, ws)
        return None, dq, dk, dv, dP_q.to(P_q.dtype), dP_k.to(P_k.dtype), dgate

