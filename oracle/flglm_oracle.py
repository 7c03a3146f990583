"""fp64 CPU oracle of the FL-GLM server block stack under client-batching.

TEST INFRASTRUCTURE ONLY.  Nothing in the product path may import or run this
module: only ``tests/``, ``__graft_entry__.smoke()`` and the ``cpu_baseline`` /
``--impl reference`` legs of ``bench.py`` use it.  It shares no code with the CUDA
library; the only shared module is ``synthetic`` (seeded inputs, no arithmetic of
the method).

What it computes (plain definitions, in the paper's order, float64 throughout):

* §3.1 (Model Split): the server holds blocks 1..N-2 and maps the smashed data
  h_0 of each client to h_{N-2} = Block_(1,N-2)(h_0); the client sends back the
  gradient of its loss w.r.t. h_{N-2} and the server back-propagates it and updates
  its own parameters (the split-learning protocol the introduction describes for
  FedBERT, which FL-GLM keeps).
* §3.3 (Parallel Acceleration, client-batch): the M clients' {seqlength, batch,
  hidden} tensors are stacked into one server batch.  Stacking is not averaging,
  so each client row is an independent causal segment: packed results equal the
  per-client results (the batching invariant tested on this module).
* The block internals are not printed in the paper (§3.1 only says each block is
  a transformer layer of multi-head self-attention and an FFN; §4.1.4 gives 28
  layers, hidden 4096, 32 heads).  The reading taken is the ChatGLM-6B block:
      a = LN1(x); qkv = a Wqkv^T + bqkv; q,k <- RoPE; o = causal softmax(q k^T/sqrt(d_h)) v
      h = alpha * a + (o Wd^T + bd)        (residual_from_ln = 1; alpha*x with 0)
      m = LN2(h); y = alpha * m + (gelu(m W1^T + b1) W2^T + b2)   (alpha*h with 0)
  with the softmax scale 1/sqrt(d_h) of App. A (P-tuning v2 equations).
* The optimizer of §4.1.4 (Adam, without weight decay) in the decoupled AdamW form
  with bias correction; the decay rate is a parameter that defaults to 0.
* §3.1 client parts: h_0 = Block_0(Embedding(x)) at the bottom; at the top
  y' = Linear(Block_{N-1}(h_{N-2})) and the cross-entropy loss.  Reading: the
  ChatGLM-6B top, a final LayerNorm before the bias-free LM head, the loss the mean
  over the answer tokens that carry a target.  Clients and server parameters are
  averaged at the end of a period (§3.3).
* §4.1.1 casts every task as GLM blank infilling: a context with a mask token [M]
  (a cloze question, or [M] appended after the text for summarisation) and an answer
  span generated after it.  Optional per-segment GLM structure (context length c and
  [M] position): the context attends bidirectionally within itself, the span causally
  to the context and to its own earlier tokens; positions are two-dimensional (the
  span takes the position of [M] and block positions 1, 2, ...), the second position
  rotating the second half of each head.  Without it (c = 0) a segment is plainly
  causal with positions 0..L-1.

The backward is the exact chain rule of the forward, written out by hand.
"""
from __future__ import annotations

import math
from dataclasses import dataclass
from typing import List, Optional, Sequence

import numpy as np

import synthetic as syn

F64 = np.float64

# ----------------------------------------------------------------------------- packing
# §3.3 client-batch: each client sends {seqlength, batch, hidden}; the server stacks them.


@dataclass
class Packing:
    cu_seqlens: np.ndarray   # int32 [S + 1], segment s = tokens [cu[s], cu[s+1])
    pos: np.ndarray          # int32 [T], position of each token inside its own segment
    seg_client: np.ndarray   # int32 [S], client that owns segment s
    seg_row: np.ndarray      # int32 [S], row of that client's batch
    ctx: Optional[np.ndarray] = None    # int32 [S], GLM context length (0: plain causal segment)
    pos2: Optional[np.ndarray] = None   # int32 [T], GLM block position (rotates the second half)

    @property
    def T(self) -> int:
        return int(self.cu_seqlens[-1])

    @property
    def S(self) -> int:
        return len(self.cu_seqlens) - 1


def glm_positions(L: int, c: int, mask_pos: int):
    """GLM's two position streams of one segment of length L with context length c and
    the mask token at mask_pos (< c): context token t has (t, 0); span token t >= c has
    (mask_pos, t - c + 1).  c = 0 is a plain causal segment: (t, 0)."""
    p1 = np.arange(L, dtype=np.int32)
    p2 = np.zeros(L, np.int32)
    if c > 0:
        if not 0 <= mask_pos < c <= L:
            raise ValueError("GLM segment: need 0 <= mask_pos < context_len <= L")
        p1[c:] = mask_pos
        p2[c:] = np.arange(1, L - c + 1)
    elif c < 0:
        raise ValueError("GLM segment: negative context length")
    return p1, p2


def make_packing(seq_lens: Sequence[int], client_batch: int, context_lens: Optional[Sequence[int]] = None,
                 mask_pos: Optional[Sequence[int]] = None) -> Packing:
    """Segments in client-major, then row-major order: client k row r is segment k*b + r.
    context_lens / mask_pos (one per segment; mask_pos defaults to the last context token,
    the summarisation layout of §4.1.1) give every segment the GLM blank-infilling structure."""
    cu = [0]
    pos, pos2, segc, segr = [], [], [], []
    for k, L in enumerate(seq_lens):
        for r in range(client_batch):
            s = len(segc)
            cu.append(cu[-1] + L)
            if context_lens is None:
                pos.extend(range(L))
            else:
                c = int(context_lens[s])
                mp = int(mask_pos[s]) if mask_pos is not None else c - 1
                p1, p2 = glm_positions(L, c, mp)
                pos.extend(p1)
                pos2.extend(p2)
            segc.append(k)
            segr.append(r)
    ctx = None if context_lens is None else np.array(context_lens, np.int32)
    return Packing(np.array(cu, np.int32), np.array(pos, np.int32),
                   np.array(segc, np.int32), np.array(segr, np.int32),
                   ctx, None if context_lens is None else np.array(pos2, np.int32))


def pack(client_tensors: Sequence[np.ndarray]) -> np.ndarray:
    """Concatenate K tensors [b, L_k, H] into X[T, H] (segment = one client row)."""
    H = client_tensors[0].shape[-1]
    return np.concatenate([t.reshape(-1, H) for t in client_tensors], axis=0)


def unpack(X: np.ndarray, seq_lens: Sequence[int], client_batch: int) -> List[np.ndarray]:
    out, t0 = [], 0
    H = X.shape[-1]
    for L in seq_lens:
        n = client_batch * L
        out.append(X[t0:t0 + n].reshape(client_batch, L, H))
        t0 += n
    return out


# ----------------------------------------------------------------------------- LayerNorm


def layer_norm_fwd(x: np.ndarray, gamma: np.ndarray, beta: np.ndarray, eps: float):
    """Row LayerNorm with the biased variance over the hidden dim."""
    mu = x.mean(axis=-1)
    xc = x - mu[:, None]
    var = (xc * xc).mean(axis=-1)
    rstd = 1.0 / np.sqrt(var + eps)
    xhat = xc * rstd[:, None]
    return xhat * gamma[None, :] + beta[None, :], mu, rstd


def layer_norm_bwd(dy: np.ndarray, x: np.ndarray, mu: np.ndarray, rstd: np.ndarray, gamma: np.ndarray):
    """dx = rstd * (g - mean(g) - xhat * mean(g * xhat)), g = gamma * dy; dgamma, dbeta summed over rows."""
    xhat = (x - mu[:, None]) * rstd[:, None]
    g = dy * gamma[None, :]
    dx = rstd[:, None] * (g - g.mean(axis=-1, keepdims=True) - xhat * (g * xhat).mean(axis=-1, keepdims=True))
    dgamma = (dy * xhat).sum(axis=0)
    dbeta = dy.sum(axis=0)
    return dx, dgamma, dbeta


# ----------------------------------------------------------------------------- RoPE


def rope_cos_sin(pos: np.ndarray, rotary_dim: int, base: float):
    """Angles p * base^(-2i/rotary_dim), i < rotary_dim/2, one per rotated pair."""
    half = rotary_dim // 2
    inv_freq = base ** (-(2.0 * np.arange(half, dtype=F64)) / rotary_dim)
    ang = pos.astype(F64)[:, None] * inv_freq[None, :]
    return np.cos(ang), np.sin(ang)


def rope_rotate(x: np.ndarray, cos: np.ndarray, sin: np.ndarray, rotary_dim: int, inverse: bool = False):
    """Rotate-half pairing (i, i + rotary_dim/2) inside dims [0, rotary_dim) of every head;
    dims [rotary_dim, head_dim) pass through.  x: [T, nh, hd]."""
    half = rotary_dim // 2
    s = -sin if inverse else sin
    c = cos[:, None, :]
    s = s[:, None, :]
    out = x.copy()
    x1 = x[..., :half]
    x2 = x[..., half:rotary_dim]
    out[..., :half] = x1 * c - x2 * s
    out[..., half:rotary_dim] = x2 * c + x1 * s
    return out


def rope_2d(x: np.ndarray, pk: "Packing", rotary_dim: int, base: float, inverse: bool = False):
    """Rotary encoding of every head of x [T, nh, hd]: dims [0, rotary_dim) by the first
    position; with GLM positions, dims [rotary_dim, 2 rotary_dim) by the block position,
    same frequencies and pairing (ChatGLM's 2D rotary, rotary_dim = hd / 2)."""
    cos, sin = rope_cos_sin(pk.pos, rotary_dim, base)
    out = rope_rotate(x, cos, sin, rotary_dim, inverse)
    if pk.pos2 is not None:
        if 2 * rotary_dim != x.shape[-1]:
            raise ValueError("2D rotary needs rotary_dim = head_dim / 2")
        cos2, sin2 = rope_cos_sin(pk.pos2, rotary_dim, base)
        out[..., rotary_dim:] = rope_rotate(out[..., rotary_dim:], cos2, sin2, rotary_dim, inverse)
    return out


# ----------------------------------------------------------------------------- attention


def _keys_values(k, v, pk, pv, a, b, h):
    """Keys and values one segment's queries see: the prefix (P-tuning v2, App. A:
    K' = [prefix_key : key], V' = [prefix_value : value]) then the segment's own."""
    if pk is None:
        return k[a:b, h], v[a:b, h], 0
    return np.concatenate([pk[:, h], k[a:b, h]]), np.concatenate([pv[:, h], v[a:b, h]]), pk.shape[0]


def _mask(L: int, Lp: int, c: int = 0):
    """Query t sees every prefix key and the keys u of its own segment with u <= t or, in a
    GLM segment with context length c, u < c (the context is seen by every token)."""
    t = np.arange(L)[:, None]
    u = np.arange(L)[None, :]
    own = (u <= t) | (u < c)
    return np.concatenate([np.ones((L, Lp), bool), own], axis=1)


def _ctx(ctx, s):
    return 0 if ctx is None else int(ctx[s])


def attention_fwd(q: np.ndarray, k: np.ndarray, v: np.ndarray, cu_seqlens: np.ndarray, pk=None, pv=None,
                  ctx=None):
    """Per segment, per head: O = softmax(Q K'^T / sqrt(d_h) + mask) V' (App. A), K' and V'
    the optional prefix followed by the segment's own keys (causal; with a GLM context
    length ctx[s], the context is bidirectional).
    Returns O [T, nh, hd] and the row log-sum-exp LSE [nh, T] of the scaled scores."""
    T, nh, hd = q.shape
    scale = 1.0 / math.sqrt(hd)
    o = np.zeros_like(q)
    lse = np.zeros((nh, T), F64)
    for s in range(len(cu_seqlens) - 1):
        a, b = int(cu_seqlens[s]), int(cu_seqlens[s + 1])
        L = b - a
        if L == 0:
            continue
        for h in range(nh):
            kk, vv, Lp = _keys_values(k, v, pk, pv, a, b, h)
            S = (q[a:b, h] @ kk.T) * scale
            S = np.where(_mask(L, Lp, _ctx(ctx, s)), S, -np.inf)
            m = S.max(axis=-1)
            P = np.exp(S - m[:, None])
            l = P.sum(axis=-1)
            P /= l[:, None]
            o[a:b, h] = P @ vv
            lse[h, a:b] = m + np.log(l)
    return o, lse


def attention_bwd(do: np.ndarray, q: np.ndarray, k: np.ndarray, v: np.ndarray, cu_seqlens: np.ndarray,
                  pk=None, pv=None, ctx=None):
    """Chain rule of attention_fwd: dV' = P^T dO, dP = dO V'^T, dS = P (dP - rowsum(dP P)),
    dQ = dS K' / sqrt(d_h), dK' = dS^T Q / sqrt(d_h).  With a prefix, its gradients are
    summed over every segment (the prefix is shared) and returned as dpk, dpv."""
    T, nh, hd = q.shape
    scale = 1.0 / math.sqrt(hd)
    dq = np.zeros_like(q)
    dk = np.zeros_like(k)
    dv = np.zeros_like(v)
    dpk = None if pk is None else np.zeros_like(pk)
    dpv = None if pv is None else np.zeros_like(pv)
    for s in range(len(cu_seqlens) - 1):
        a, b = int(cu_seqlens[s]), int(cu_seqlens[s + 1])
        L = b - a
        if L == 0:
            continue
        for h in range(nh):
            kk, vv, Lp = _keys_values(k, v, pk, pv, a, b, h)
            S = (q[a:b, h] @ kk.T) * scale
            S = np.where(_mask(L, Lp, _ctx(ctx, s)), S, -np.inf)
            P = np.exp(S - S.max(axis=-1, keepdims=True))
            P /= P.sum(axis=-1, keepdims=True)
            dP = do[a:b, h] @ vv.T
            dS = P * (dP - (dP * P).sum(axis=-1, keepdims=True))
            dvv = P.T @ do[a:b, h]
            dkk = (dS.T @ q[a:b, h]) * scale
            dq[a:b, h] = (dS @ kk) * scale
            dv[a:b, h] = dvv[Lp:]
            dk[a:b, h] = dkk[Lp:]
            if Lp:
                dpk[:, h] += dkk[:Lp]
                dpv[:, h] += dvv[:Lp]
    if pk is None:
        return dq, dk, dv
    return dq, dk, dv, dpk, dpv


# ----------------------------------------------------------------------------- GeLU (tanh form)

_C = math.sqrt(2.0 / math.pi)
_A = 0.044715


def gelu(u: np.ndarray) -> np.ndarray:
    return 0.5 * u * (1.0 + np.tanh(_C * (u + _A * u ** 3)))


def gelu_grad(u: np.ndarray) -> np.ndarray:
    t = np.tanh(_C * (u + _A * u ** 3))
    return 0.5 * (1.0 + t) + 0.5 * u * (1.0 - t * t) * _C * (1.0 + 3.0 * _A * u * u)


# ----------------------------------------------------------------------------- one block


@dataclass
class BlockShape:
    hidden: int
    n_heads: int
    head_dim: int
    ffn_hidden: int
    rotary_dim: int
    rope_base: float
    ln_eps: float
    alpha: float
    residual_from_ln: int

    @staticmethod
    def of(cfg: syn.ServerConfig) -> "BlockShape":
        return BlockShape(cfg.hidden, cfg.n_heads, cfg.head_dim, cfg.ffn_hidden, cfg.rdim,
                          cfg.rope_base, cfg.ln_eps, cfg.residual_alpha, cfg.residual_from_ln)


def block_fwd(P: Sequence[np.ndarray], x: np.ndarray, pk: Packing, sh: BlockShape, prefix=None):
    """One server block over the packed tokens x [T, H]; returns y and the saved values.
    prefix: optional (prefix_key, prefix_value), each [L_p, H], seen by every query (App. A);
    the prefix keys enter the scores as they are (no rotary rotation)."""
    Wqkv, bqkv, Wd, bd, W1, b1, W2, b2, g1, be1, g2, be2 = P
    T, H = x.shape
    nh, hd = sh.n_heads, sh.head_dim
    a, mu1, rs1 = layer_norm_fwd(x, g1, be1, sh.ln_eps)
    qkv = a @ Wqkv.T + bqkv[None, :]                         # [T, 3H]: q | k | v, each [nh, hd]
    q = qkv[:, 0:H].reshape(T, nh, hd)
    k = qkv[:, H:2 * H].reshape(T, nh, hd)
    v = qkv[:, 2 * H:3 * H].reshape(T, nh, hd)
    qr = rope_2d(q, pk, sh.rotary_dim, sh.rope_base)
    kr = rope_2d(k, pk, sh.rotary_dim, sh.rope_base)
    ppk = ppv = None
    if prefix is not None:
        ppk = np.asarray(prefix[0], F64).reshape(-1, nh, hd)
        ppv = np.asarray(prefix[1], F64).reshape(-1, nh, hd)
    o, lse = attention_fwd(qr, kr, v, pk.cu_seqlens, ppk, ppv, pk.ctx)
    o = o.reshape(T, H)
    res1 = a if sh.residual_from_ln else x
    h = sh.alpha * res1 + (o @ Wd.T + bd[None, :])
    m, mu2, rs2 = layer_norm_fwd(h, g2, be2, sh.ln_eps)
    u = m @ W1.T + b1[None, :]
    g = gelu(u)
    res2 = m if sh.residual_from_ln else h
    y = sh.alpha * res2 + (g @ W2.T + b2[None, :])
    saved = dict(x=x, a=a, mu1=mu1, rs1=rs1, qr=qr, kr=kr, v=v, o=o, lse=lse, h=h, m=m,
                 mu2=mu2, rs2=rs2, u=u, g=g, ppk=ppk, ppv=ppv)
    return y, saved


def block_bwd(P: Sequence[np.ndarray], sv: dict, dy: np.ndarray, pk: Packing, sh: BlockShape):
    """Exact chain rule of block_fwd.  Returns dx and the 12 parameter gradients (summed over T),
    followed by the prefix key and value gradients [L_p, H] when the block has a prefix."""
    Wqkv, bqkv, Wd, bd, W1, b1, W2, b2, g1, be1, g2, be2 = P
    T, H = dy.shape
    nh, hd = sh.n_heads, sh.head_dim
    al = sh.alpha
    # FFN down: y = alpha*res2 + g W2^T + b2
    dW2 = dy.T @ sv["g"]
    db2 = dy.sum(axis=0)
    dg = dy @ W2
    du = dg * gelu_grad(sv["u"])
    dW1 = du.T @ sv["m"]
    db1 = du.sum(axis=0)
    dm = du @ W1
    if sh.residual_from_ln:
        dm = dm + al * dy
    dh, dg2, dbe2 = layer_norm_bwd(dm, sv["h"], sv["mu2"], sv["rs2"], g2)
    if not sh.residual_from_ln:
        dh = dh + al * dy
    # attention output projection: h = alpha*res1 + o Wd^T + bd
    dWd = dh.T @ sv["o"]
    dbd = dh.sum(axis=0)
    do = (dh @ Wd).reshape(T, nh, hd)
    res = attention_bwd(do, sv["qr"], sv["kr"], sv["v"], pk.cu_seqlens, sv["ppk"], sv["ppv"], pk.ctx)
    dqr, dkr, dv = res[:3]
    dq = rope_2d(dqr, pk, sh.rotary_dim, sh.rope_base, inverse=True)
    dk = rope_2d(dkr, pk, sh.rotary_dim, sh.rope_base, inverse=True)
    dqkv = np.concatenate([dq.reshape(T, H), dk.reshape(T, H), dv.reshape(T, H)], axis=1)
    dWqkv = dqkv.T @ sv["a"]
    dbqkv = dqkv.sum(axis=0)
    da = dqkv @ Wqkv
    if sh.residual_from_ln:
        da = da + al * dh
    dx, dg1, dbe1 = layer_norm_bwd(da, sv["x"], sv["mu1"], sv["rs1"], g1)
    if not sh.residual_from_ln:
        dx = dx + al * dh
    grads = [dWqkv, dbqkv, dWd, dbd, dW1, db1, dW2, db2, dg1, dbe1, dg2, dbe2]
    if sv["ppk"] is not None:
        grads += [res[3].reshape(-1, H), res[4].reshape(-1, H)]
    return dx, grads


# ----------------------------------------------------------------------------- stack + server


def stack_fwd(params: Sequence[Sequence[np.ndarray]], x: np.ndarray, pk: Packing, sh: BlockShape, prefixes=None):
    saved = []
    for b, P in enumerate(params):
        x, sv = block_fwd(P, x, pk, sh, None if prefixes is None else prefixes[b])
        saved.append(sv)
    return x, saved


def stack_bwd(params, saved, dy, pk: Packing, sh: BlockShape):
    grads = [None] * len(params)
    for b in range(len(params) - 1, -1, -1):
        dy, grads[b] = block_bwd(params[b], saved[b], dy, pk, sh)
    return dy, grads


def adamw_update(w, g, m, v, t: int, lr: float, beta1: float, beta2: float, eps: float, wd: float):
    """Decoupled-weight-decay Adam with bias correction (step t >= 1).  Returns new w, m, v."""
    m = beta1 * m + (1.0 - beta1) * g
    v = beta2 * v + (1.0 - beta2) * g * g
    mhat = m / (1.0 - beta1 ** t)
    vhat = v / (1.0 - beta2 ** t)
    w = w - lr * (mhat / (np.sqrt(vhat) + eps) + wd * w)
    return w, m, v


class OracleServer:
    """The server's protocol on the oracle: forward(client states) -> output states,
    backward(output-state grads) -> input-state grads (+ accumulated weight grads),
    step(lr) -> AdamW update that clears the grads.  With cfg.prefix_len > 0 every block
    carries P-tuning v2 prefix keys and values (tensors 12 and 13 of the block); with
    cfg.freeze_base the step updates only those (App. A: the model is frozen and only the
    prefix is trained)."""

    def __init__(self, cfg: syn.ServerConfig, params: Optional[List[List[np.ndarray]]] = None, prefixes=None):
        self.cfg = cfg
        self.sh = BlockShape.of(cfg)
        if params is None:
            params = syn.init_params(cfg)
        if cfg.prefix_len and prefixes is None:
            prefixes = [syn.init_prefix(cfg, b) for b in range(cfg.n_blocks)]
        self.params = [[np.asarray(p, F64).copy() for p in blk] for blk in params]
        if cfg.prefix_len:
            for blk, pre in zip(self.params, prefixes):
                blk.extend(np.asarray(p, F64).copy() for p in pre)
        self.grads = [[np.zeros_like(p) for p in blk] for blk in self.params]
        self.m = [[np.zeros_like(p) for p in blk] for blk in self.params]
        self.v = [[np.zeros_like(p) for p in blk] for blk in self.params]
        self.t = 0
        self._pending = None

    def forward(self, client_states: Sequence[np.ndarray], context_lens=None, mask_pos=None) -> List[np.ndarray]:
        """context_lens / mask_pos: optional GLM structure, one entry per segment
        (client-major, then row)."""
        seq_lens = [s.shape[1] for s in client_states]
        b = client_states[0].shape[0]
        pk = make_packing(seq_lens, b, context_lens, mask_pos)
        X = pack([np.asarray(s, F64) for s in client_states])
        base = [blk[:12] for blk in self.params]
        pre = [blk[12:14] for blk in self.params] if self.cfg.prefix_len else None
        Y, saved = stack_fwd(base, X, pk, self.sh, pre)
        self._pending = (seq_lens, b, pk, saved)
        return unpack(Y, seq_lens, b)

    def backward(self, grad_out: Sequence[np.ndarray]) -> List[np.ndarray]:
        if self._pending is None:
            raise RuntimeError("backward without a pending forward")
        seq_lens, b, pk, saved = self._pending
        dY = pack([np.asarray(g, F64) for g in grad_out])
        dX, grads = stack_bwd([blk[:12] for blk in self.params], saved, dY, pk, self.sh)
        for gb, acc in zip(grads, self.grads):
            for i in range(len(gb)):
                acc[i] += gb[i]
        self._pending = None
        return unpack(dX, seq_lens, b)

    def step(self, lr: float):
        c = self.cfg
        self.t += 1
        trained = range(12, 14) if c.freeze_base else range(len(self.params[0]))
        for bi in range(len(self.params)):
            for i in trained:
                w, m, v = adamw_update(self.params[bi][i], self.grads[bi][i], self.m[bi][i], self.v[bi][i],
                                       self.t, lr, c.adam_beta1, c.adam_beta2, c.adam_eps, c.weight_decay)
                self.params[bi][i], self.m[bi][i], self.v[bi][i] = w, m, v
            self.grads[bi] = [np.zeros_like(g) for g in self.grads[bi]]



def average_params(servers: Sequence["OracleServer"]):
    """§3.3 server-hierarchical strategy: at the end of a training period every replica's
    parameters are replaced by the arithmetic mean over the replicas; optimizer moments and
    step counts stay with each replica."""
    n = len(servers)
    for b in range(len(servers[0].params)):
        for t in range(len(servers[0].params[b])):
            mean = sum(s.params[b][t] for s in servers) / n
            for s in servers:
                s.params[b][t] = mean.copy()


# ----------------------------------------------------------------------------- client parts (§3.1)


def embedding_fwd(E: np.ndarray, tokens: np.ndarray) -> np.ndarray:
    """Rows of the embedding table for the token ids."""
    return E[tokens]


def embedding_bwd(dX: np.ndarray, tokens: np.ndarray, vocab: int) -> np.ndarray:
    """Gradient of the table: each row receives the sum of the gradients of its occurrences."""
    dE = np.zeros((vocab, dX.shape[1]), F64)
    np.add.at(dE, tokens, dX)
    return dE


def cross_entropy(logits: np.ndarray, labels: np.ndarray):
    """Mean over the rows with a target (label >= 0) of -log softmax(logits)[label], and its
    gradient w.r.t. the logits (zero on rows without a target).  No target: loss 0."""
    valid = labels >= 0
    n = int(valid.sum())
    m = logits.max(axis=-1, keepdims=True)
    lse = m[:, 0] + np.log(np.exp(logits - m).sum(axis=-1))
    d = np.exp(logits - lse[:, None])
    rows = np.nonzero(valid)[0]
    loss = float((lse[rows] - logits[rows, labels[rows]]).sum() / max(n, 1))
    d[rows, labels[rows]] -= 1.0
    d[~valid] = 0.0
    return loss, d / max(n, 1)


CLIENT_PARTS = ("bottom", "top", "embed", "head", "final_ln")


class OracleClient:
    """One client of §3.1: bottom = Embedding + Block_0, top = Block_{N-1} + final LayerNorm +
    LM head + cross-entropy.  Protocol: bottom_forward(tokens) -> h_0 (to the server);
    top_forward_backward(h_{N-2}, labels) -> loss and the gradient w.r.t. h_{N-2} (to the
    server); bottom_backward(gradient w.r.t. h_0); step(lr).  Both blocks see the segment
    structure (GLM context, positions) of the bottom call and, with prefix_len, carry their
    own P-tuning v2 prefixes; with freeze_base only those prefixes are trained."""

    def __init__(self, cfg: syn.ServerConfig, params=None):
        self.cfg = cfg
        self.sh = BlockShape.of(cfg)
        p = syn.init_client(cfg) if params is None else params
        self.params = {k: [np.asarray(x, F64).copy() for x in p[k]] for k in CLIENT_PARTS}
        self.grads = {k: [np.zeros_like(x) for x in v] for k, v in self.params.items()}
        self.m = {k: [np.zeros_like(x) for x in v] for k, v in self.params.items()}
        self.v = {k: [np.zeros_like(x) for x in v] for k, v in self.params.items()}
        self.t = 0
        self._pk = None
        self._bottom = None

    def _block(self, name):
        blk = self.params[name]
        return blk[:12], (blk[12:14] if self.cfg.prefix_len else None)

    def _accumulate(self, name, grads):
        for acc, g in zip(self.grads[name], grads):
            acc += g

    def bottom_forward(self, tokens: np.ndarray, context_lens=None, mask_pos=None) -> np.ndarray:
        b, L = tokens.shape
        pk = make_packing([L], b, context_lens, mask_pos)
        x = embedding_fwd(self.params["embed"][0], tokens.reshape(-1))
        P, pre = self._block("bottom")
        y, sv = block_fwd(P, x, pk, self.sh, pre)
        self._pk = pk
        self._bottom = (tokens.reshape(-1), sv)
        return y.reshape(b, L, -1)

    def top_forward_backward(self, h: np.ndarray, labels: np.ndarray):
        b, L, H = h.shape
        pk = self._pk
        P, pre = self._block("top")
        y, sv = block_fwd(P, h.reshape(-1, H), pk, self.sh, pre)
        g, be = self.params["final_ln"]
        z, mu, rs = layer_norm_fwd(y, g, be, self.sh.ln_eps)
        W = self.params["head"][0]
        logits = z @ W.T
        loss, dlog = cross_entropy(logits, labels.reshape(-1))
        self._accumulate("head", [dlog.T @ z])
        dz = dlog @ W
        dy, dg, dbe = layer_norm_bwd(dz, y, mu, rs, g)
        self._accumulate("final_ln", [dg, dbe])
        dx, gb = block_bwd(P, sv, dy, pk, self.sh)
        self._accumulate("top", gb)
        return loss, dx.reshape(b, L, H)

    def bottom_backward(self, grad_h0: np.ndarray):
        tokens, sv = self._bottom
        P, _ = self._block("bottom")
        H = grad_h0.shape[-1]
        dx, gb = block_bwd(P, sv, grad_h0.reshape(-1, H), self._pk, self.sh)
        self._accumulate("bottom", gb)
        self._accumulate("embed", [embedding_bwd(dx, tokens, self.cfg.vocab)])
        self._bottom = None

    def trained(self):
        """(part, tensor index) of every trained tensor."""
        if self.cfg.freeze_base:
            return [(k, i) for k in ("bottom", "top") for i in (12, 13)]
        return [(k, i) for k in CLIENT_PARTS for i in range(len(self.params[k]))]

    def step(self, lr: float):
        c = self.cfg
        self.t += 1
        for k, i in self.trained():
            w, m, v = adamw_update(self.params[k][i], self.grads[k][i], self.m[k][i], self.v[k][i], self.t, lr,
                                   c.adam_beta1, c.adam_beta2, c.adam_eps, c.weight_decay)
            self.params[k][i], self.m[k][i], self.v[k][i] = w, m, v
        self.grads = {k: [np.zeros_like(x) for x in v] for k, v in self.params.items()}


def average_clients(clients: Sequence[OracleClient]):
    """§3.3: at the end of a period the client-side parameters are replaced by their mean
    over the clients (moments and step counts stay local)."""
    n = len(clients)
    for k in CLIENT_PARTS:
        for i in range(len(clients[0].params[k])):
            mean = sum(c.params[k][i] for c in clients) / n
            for c in clients:
                c.params[k][i] = mean.copy()
