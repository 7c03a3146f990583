"""ctypes front end of the fp32 C++ oracle (flglm_oracle32.cpp).

TEST INFRASTRUCTURE ONLY: only tests/, __graft_entry__.smoke() and bench.py's CPU legs
use it.  It marshals numpy arrays; every step of the arithmetic runs in the C++ source.
"""
from __future__ import annotations

import ctypes as C
from typing import List, Sequence

import numpy as np

from . import build as _build


class _Shape(C.Structure):
    _fields_ = [("hidden", C.c_int32), ("n_heads", C.c_int32), ("head_dim", C.c_int32),
                ("ffn_hidden", C.c_int32), ("rotary_dim", C.c_int32), ("rope_base", C.c_float),
                ("ln_eps", C.c_float), ("alpha", C.c_float), ("residual_from_ln", C.c_int32)]


_LIB = None


def lib():
    global _LIB
    if _LIB is None:
        L = C.CDLL(_build.build())
        L.flo_threads.restype = C.c_int
        L.flo_server_fwd_bwd.restype = C.c_int
        L.flo_server_fwd_bwd.argtypes = [C.POINTER(_Shape), C.c_int32, C.POINTER(C.c_void_p),
                                         C.POINTER(C.c_void_p), C.c_int32, C.c_void_p, C.c_void_p, C.c_void_p,
                                         C.c_void_p, C.c_void_p]
        L.flo_server_fwd_bwd_ext.restype = C.c_int
        L.flo_server_fwd_bwd_ext.argtypes = [C.POINTER(_Shape), C.c_int32, C.POINTER(C.c_void_p),
                                             C.POINTER(C.c_void_p), C.c_int32, C.c_void_p, C.c_void_p, C.c_void_p,
                                             C.c_int32, C.POINTER(C.c_void_p), C.POINTER(C.c_void_p), C.c_void_p,
                                             C.c_void_p, C.c_void_p, C.c_void_p]
        L.flo_client_round.restype = C.c_int
        L.flo_client_round.argtypes = [C.POINTER(_Shape), C.c_int32, C.c_int32, C.c_int32, C.c_void_p, C.c_void_p,
                                       C.c_void_p, C.c_void_p, C.c_int32, C.c_void_p, C.POINTER(C.c_void_p),
                                       C.POINTER(C.c_void_p), C.c_void_p, C.c_void_p, C.c_void_p, C.c_void_p,
                                       C.POINTER(C.c_void_p), C.POINTER(C.c_void_p), C.POINTER(C.c_void_p),
                                       C.c_void_p, C.c_void_p]
        L.flo_adamw.restype = C.c_int
        L.flo_adamw.argtypes = [C.c_int64, C.c_void_p, C.c_void_p, C.c_void_p, C.c_void_p, C.c_int32,
                                C.c_float, C.c_float, C.c_float, C.c_float, C.c_float]
        _LIB = L
    return _LIB


def threads() -> int:
    return int(lib().flo_threads())


def _f32(a) -> np.ndarray:
    a = np.ascontiguousarray(a, np.float32)
    return a


def shape_of(cfg) -> _Shape:
    return _Shape(cfg.hidden, cfg.n_heads, cfg.head_dim, cfg.ffn_hidden, cfg.rdim, cfg.rope_base, cfg.ln_eps,
                  cfg.residual_alpha, cfg.residual_from_ln)


def server_fwd_bwd(cfg, params: Sequence[Sequence[np.ndarray]], grads: List[List[np.ndarray]],
                   cu_seqlens: Sequence[int], x: np.ndarray, dy: np.ndarray, context_lens=None, mask_pos=None,
                   prefixes=None, prefix_grads=None):
    """Packed tokens x [T, H] through the blocks (params[b] = the 12 fp32 tensors of block b)
    and dy [T, H] back; returns (y, dx) [T, H] fp32 and adds the weight gradients into
    `grads` (fp32 arrays, same shapes as params, updated in place).  context_lens /
    mask_pos (one per segment): GLM segments; prefixes[b] = (prefix keys, prefix values)
    [Lp, H] of block b, whose gradients are added into prefix_grads[b] (fp32, in place)."""
    nb = len(params)
    ps = [[_f32(p) for p in blk] for blk in params]
    for blk in grads:
        for g in blk:
            if g.dtype != np.float32 or not g.flags.c_contiguous:
                raise ValueError("grads must be contiguous float32 arrays")
    pp = (C.c_void_p * (12 * nb))(*[p.ctypes.data for blk in ps for p in blk[:12]])
    gp = (C.c_void_p * (12 * nb))(*[g.ctypes.data for blk in grads for g in blk[:12]])
    cu = np.ascontiguousarray(cu_seqlens, np.int32)
    x = _f32(x)
    dy = _f32(dy)
    y = np.empty_like(x)
    dx = np.empty_like(x)
    sh = shape_of(cfg)
    ctx = None if context_lens is None else np.ascontiguousarray(context_lens, np.int32)
    mp = None if mask_pos is None else np.ascontiguousarray(mask_pos, np.int32)
    Lp, pre, pg = 0, None, None
    if prefixes is not None:
        pf = [[_f32(p) for p in blk] for blk in prefixes]
        for blk in prefix_grads:
            for g in blk:
                if g.dtype != np.float32 or not g.flags.c_contiguous:
                    raise ValueError("prefix_grads must be contiguous float32 arrays")
        Lp = pf[0][0].shape[0]
        pre = (C.c_void_p * (2 * nb))(*[p.ctypes.data for blk in pf for p in blk[:2]])
        pg = (C.c_void_p * (2 * nb))(*[g.ctypes.data for blk in prefix_grads for g in blk[:2]])
    rc = lib().flo_server_fwd_bwd_ext(C.byref(sh), nb, pp, gp, len(cu) - 1, cu.ctypes.data,
                                      None if ctx is None else ctx.ctypes.data, None if mp is None else mp.ctypes.data,
                                      Lp, pre, pg, x.ctypes.data, dy.ctypes.data, y.ctypes.data, dx.ctypes.data)
    if rc != 0:
        raise ValueError(f"flo_server_fwd_bwd: bad arguments (rc {rc})")
    return y, dx


def client_round(cfg, params: dict, tokens: np.ndarray, labels: np.ndarray, context_lens=None, mask_pos=None):
    """One client's round of §3.1 with the server's blocks left out: tokens / labels int32
    [b, L]; params as synthetic.init_client (parts bottom, top, embed, head, final_ln).
    Returns (loss, grads) with grads a dict of fp32 arrays shaped like params."""
    ps = {k: [_f32(p) for p in v] for k, v in params.items()}
    gs = {k: [np.zeros(p.shape, np.float32) for p in v] for k, v in ps.items()}
    tok = np.ascontiguousarray(tokens, np.int32)
    lab = np.ascontiguousarray(labels, np.int32)
    b, L = tok.shape
    nblk = len(ps["bottom"])
    arr = lambda xs: (C.c_void_p * len(xs))(*[x.ctypes.data for x in xs])  # noqa: E731
    ctx = None if context_lens is None else np.ascontiguousarray(context_lens, np.int32)
    mp = None if mask_pos is None else np.ascontiguousarray(mask_pos, np.int32)
    loss = np.zeros(1, np.float32)
    sh = shape_of(cfg)
    rc = lib().flo_client_round(C.byref(sh), cfg.vocab, b, L, tok.ctypes.data, lab.ctypes.data,
                                None if ctx is None else ctx.ctypes.data, None if mp is None else mp.ctypes.data,
                                cfg.prefix_len if nblk > 12 else 0, ps["embed"][0].ctypes.data, arr(ps["bottom"]),
                                arr(ps["top"]), ps["final_ln"][0].ctypes.data, ps["final_ln"][1].ctypes.data,
                                ps["head"][0].ctypes.data, gs["embed"][0].ctypes.data, arr(gs["bottom"]),
                                arr(gs["top"]), arr(gs["final_ln"]), gs["head"][0].ctypes.data, loss.ctypes.data)
    if rc != 0:
        raise ValueError(f"flo_client_round: bad arguments (rc {rc})")
    return float(loss[0]), gs


def adamw(w: np.ndarray, g: np.ndarray, m: np.ndarray, v: np.ndarray, t: int, lr: float, beta1: float,
          beta2: float, eps: float, wd: float):
    """In-place AdamW step t on fp32 arrays w, m, v with gradient g."""
    for a in (w, m, v):
        if a.dtype != np.float32 or not a.flags.c_contiguous:
            raise ValueError("w, m, v must be contiguous float32 arrays")
    g = _f32(g)
    rc = lib().flo_adamw(w.size, w.ctypes.data, g.ctypes.data, m.ctypes.data, v.ctypes.data, t, lr, beta1, beta2,
                         eps, wd)
    if rc != 0:
        raise ValueError("flo_adamw: bad arguments")
