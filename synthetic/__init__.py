"""Seeded synthetic inputs for the FL-GLM server block stack.

This module is the one piece shared by the fp64 oracle (``oracle/``) and the GPU
path (tests, ``bench.py``).  It holds none of the method's arithmetic: only

* a counter-based random generator (SplitMix64, Steele, Lea & Flood, OOPSLA 2014,
  with Vigna's published output mix) and the Box-Muller transform (Box & Muller,
  1958) built on it;
* the round-to-nearest-even narrowing float32 -> bfloat16 of the inputs the
  clients send (bf16 is the activation type of the server, §3.1 of the paper
  sends "smashed data" h_0 of shape {seqlength, batch, hidden});
* the workload table: the five server configurations the build is measured on.

Generator definition (the CUDA library implements the same definition on the
device for ``fl_server_create(cfg, seed)``; both sides are written independently
from this text):

    GOLDEN        = 0x9E3779B97F4A7C15
    mix64(z)      : z ^= z >> 30; z *= 0xBF58476D1CE4E5B9;
                    z ^= z >> 27; z *= 0x94D049BB133111EB; z ^= z >> 31
    key(seed,tag) = mix64(mix64(seed + GOLDEN) ^ tag)        (mod 2^64)
    tag           = purpose << 56 | block << 40 | tensor << 32 | client
    raw(key, i)   = mix64(key + (i + 1) * GOLDEN)            (the i-th SplitMix64 output)
    U(key, i)     = ((raw(key, i) >> 11) + 1) * 2^-53         in (0, 1]
    normal element i of a tensor (pair j = i // 2, computed in double):
        r = sqrt(-2 ln U(key, 2j));  phi = 2 pi U(key, 2j + 1)
        z = r cos(phi) if i is even else r sin(phi)
        value = float32(mean + std * z)   (bf16 inputs: then narrowed RNE to bf16)
    (the weight init uses std = the fp32 value of init_std, which is what the C ABI's
    float field carries)
    ragged length k (seed 7 in the ragged workload):
        L_k = 64 + raw(key(seed, LENGTHS), k) mod 961        in [64, 1024]
    GLM blank-infilling structure of segment s (length L >= 2; workloads with glm = 1):
        key  = key(seed, GLM, client = s)
        span = 1 + raw(key, 0) mod max(1, L // 4)           answer tokens, at most L/4
        c    = L - span                                      context length
        [M]  = c - 1 if raw(key, 1) is even (summarisation: [M] ends the context),
               else raw(key, 1) >> 1 mod c                   (cloze: [M] inside it)
      (L = 1: c = 1, [M] = 0)
    client parts (one client model, the same initial values for every client):
        block 0 (bottom) tensor t: key(seed, CLIENT, block 0, t); block N-1 (top): block 1;
        embedding [V, H]: key(seed, CLIENT, block 2, 0); LM head [V, H]: block 3;
        final LayerNorm gamma = 1, beta = 0; N(0, init_std) like the server's weights
    client k's token ids: raw(key(seed, TOKENS, client = k), i) mod V, i over [b, L];
    labels (next-token targets of the answer span): label[t] = token[t + 1] when
        t + 1 >= c (c = the segment's GLM context length, 0 without GLM) and t + 1 < L,
        else -1 (ignored)
"""
from __future__ import annotations

import math
from dataclasses import dataclass, field, replace
from typing import Dict, List, Optional

import numpy as np

GOLDEN = 0x9E3779B97F4A7C15
M1 = 0xBF58476D1CE4E5B9
M2 = 0x94D049BB133111EB
MASK64 = (1 << 64) - 1

# stream purposes
P_WEIGHTS = 1
P_STATES = 2
P_GRADS = 3
P_LENGTHS = 4
P_GLM = 5
P_CLIENT = 6
P_TOKENS = 7
# client-side tensors outside the two blocks (block ids of the CLIENT streams)
CB_BOTTOM, CB_TOP, CB_EMBED, CB_HEAD = 0, 1, 2, 3
CHATGLM6B_VOCAB = 130528

# per-block parameter tensors, in arena order (the C library uses the same ids)
TENSOR_NAMES = ("w_qkv", "b_qkv", "w_dense", "b_dense", "w_up", "b_up",
                "w_down", "b_down", "ln1_gamma", "ln1_beta", "ln2_gamma", "ln2_beta")
T_WQKV, T_BQKV, T_WD, T_BD, T_W1, T_B1, T_W2, T_B2, T_G1, T_BE1, T_G2, T_BE2 = range(12)


def _mix64_int(z: int) -> int:
    z &= MASK64
    z ^= z >> 30
    z = (z * M1) & MASK64
    z ^= z >> 27
    z = (z * M2) & MASK64
    z ^= z >> 31
    return z


def stream_key(seed: int, purpose: int, block: int = 0, tensor: int = 0, client: int = 0) -> int:
    """Key of one counter-based stream, see the module docstring."""
    if not (0 <= purpose < 256 and 0 <= block < 65536 and 0 <= tensor < 256 and 0 <= client < 2**32):
        raise ValueError("stream tag field out of range")
    tag = (purpose << 56) | (block << 40) | (tensor << 32) | client
    return _mix64_int(_mix64_int((seed + GOLDEN) & MASK64) ^ tag)


def _mix64_vec(z: np.ndarray) -> np.ndarray:
    z = z ^ (z >> np.uint64(30))
    z = z * np.uint64(M1)
    z = z ^ (z >> np.uint64(27))
    z = z * np.uint64(M2)
    return z ^ (z >> np.uint64(31))


def raw_u64(key: int, start: int, n: int) -> np.ndarray:
    """raw(key, i) for i in [start, start + n)."""
    with np.errstate(over="ignore"):
        i = np.arange(start + 1, start + n + 1, dtype=np.uint64)
        z = np.uint64(key) + i * np.uint64(GOLDEN)
        return _mix64_vec(z)


def uniform(key: int, start: int, n: int) -> np.ndarray:
    x = raw_u64(key, start, n)
    return ((x >> np.uint64(11)).astype(np.float64) + 1.0) * (2.0 ** -53)


def normal_f64(key: int, n: int, mean: float, std: float, start: int = 0) -> np.ndarray:
    """Elements [start, start + n) of a normal stream, in double."""
    if n == 0:
        return np.zeros(0, np.float64)
    j0 = start // 2
    j1 = (start + n + 1) // 2
    u = uniform(key, 2 * j0, 2 * (j1 - j0))
    u1 = u[0::2]
    u2 = u[1::2]
    r = np.sqrt(-2.0 * np.log(u1))
    phi = 2.0 * math.pi * u2
    z = np.empty(2 * (j1 - j0), np.float64)
    z[0::2] = r * np.cos(phi)
    z[1::2] = r * np.sin(phi)
    off = start - 2 * j0
    return mean + std * z[off:off + n]


def normal_f32(key: int, n: int, mean: float, std: float, start: int = 0) -> np.ndarray:
    """float32(normal_f64(...)), produced in chunks so that large tensors need no
    float64 temporaries of their full size."""
    out = np.empty(n, np.float32)
    chunk = 1 << 22
    for a in range(0, n, chunk):
        b = min(n, a + chunk)
        out[a:b] = normal_f64(key, b - a, mean, std, start + a)
    return out


def f32_to_bf16_bits(x: np.ndarray) -> np.ndarray:
    """Round-to-nearest-even float32 -> bfloat16, returned as uint16 bit patterns."""
    b = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32)
    rounding = ((b >> np.uint32(16)) & np.uint32(1)) + np.uint32(0x7FFF)
    with np.errstate(over="ignore"):
        return ((b + rounding) >> np.uint32(16)).astype(np.uint16)


def bf16_bits_to_f32(h: np.ndarray) -> np.ndarray:
    return (np.ascontiguousarray(h, dtype=np.uint16).astype(np.uint32) << np.uint32(16)).view(np.float32)


def bf16_bits_to_f64(h: np.ndarray) -> np.ndarray:
    return bf16_bits_to_f32(h).astype(np.float64)


# ----------------------------------------------------------------------------- workloads


@dataclass(frozen=True)
class ServerConfig:
    """Shape of the server block stack plus the client workload of one call."""
    name: str
    n_blocks: int
    hidden: int
    n_heads: int
    head_dim: int
    ffn_hidden: int
    residual_alpha: float
    client_batch: int
    seq_lens: tuple            # per client
    rotary_dim: int = 0        # 0 -> head_dim // 2
    rope_base: float = 10000.0
    ln_eps: float = 1e-5
    residual_from_ln: int = 1  # 1: GLM block (residual taken from the LN output)
    init_std: float = 0.02
    adam_beta1: float = 0.9
    adam_beta2: float = 0.999
    adam_eps: float = 1e-8
    weight_decay: float = 0.0
    lr: float = 1e-4
    seed: int = 0
    state_std: float = 1.0
    grad_std: float = 1e-3
    prefix_len: int = 0        # P-tuning v2 prefix keys/values per block (0: none)
    freeze_base: int = 0       # 1: only the prefixes are trained (P-tuning v2)
    glm: int = 0               # 1: every segment carries a GLM blank-infilling structure
    vocab: int = CHATGLM6B_VOCAB   # client embedding / LM head rows

    @property
    def K(self) -> int:
        return len(self.seq_lens)

    @property
    def rdim(self) -> int:
        return self.rotary_dim if self.rotary_dim else self.head_dim // 2

    @property
    def segment_lengths(self) -> List[int]:
        out = []
        for L in self.seq_lens:
            out.extend([L] * self.client_batch)
        return out

    @property
    def tokens(self) -> int:
        return self.client_batch * int(sum(self.seq_lens))

    def with_(self, **kw) -> "ServerConfig":
        return replace(self, **kw)


def param_shapes(cfg: ServerConfig) -> List[tuple]:
    H, F = cfg.hidden, cfg.ffn_hidden
    return [(3 * H, H), (3 * H,), (H, H), (H,), (F, H), (F,), (H, F), (H,), (H,), (H,), (H,), (H,)]


# prefix tensors of a block (P-tuning v2): keys then values, [prefix_len, hidden] each,
# head j at columns j*head_dim (ids follow the 12 block tensors)
T_PK, T_PV = 12, 13


def prefix_shapes(cfg: ServerConfig) -> List[tuple]:
    return [(cfg.prefix_len, cfg.hidden), (cfg.prefix_len, cfg.hidden)]


def init_prefix(cfg: ServerConfig, block: int, seed: Optional[int] = None) -> List[np.ndarray]:
    """Initial fp32 prefix keys and values of a block: N(0, init_std), streams (seed, 1, block, 12|13)."""
    seed = cfg.seed if seed is None else seed
    out = []
    for t, shp in zip((T_PK, T_PV), prefix_shapes(cfg)):
        n = int(np.prod(shp))
        out.append(normal_f32(stream_key(seed, P_WEIGHTS, block, t), n, 0.0, float(np.float32(cfg.init_std))).reshape(shp))
    return out


def params_per_block(cfg: ServerConfig) -> int:
    return int(sum(int(np.prod(s)) for s in param_shapes(cfg)))


def ragged_lengths(seed: int, K: int, lo: int = 64, hi: int = 1024) -> tuple:
    x = raw_u64(stream_key(seed, P_LENGTHS), 0, K)
    return tuple(int(lo + int(v) % (hi - lo + 1)) for v in x)


def init_tensor(cfg: ServerConfig, block: int, tensor: int, seed: Optional[int] = None,
                purpose: int = P_WEIGHTS) -> np.ndarray:
    """Initial fp32 master value of one parameter tensor: N(0, init_std) for weights and
    biases, gamma = 1, beta = 0 for the LayerNorms."""
    seed = cfg.seed if seed is None else seed
    shape = param_shapes(cfg)[tensor]
    n = int(np.prod(shape))
    if tensor in (T_G1, T_G2):
        return np.ones(shape, np.float32)
    if tensor in (T_BE1, T_BE2):
        return np.zeros(shape, np.float32)
    key = stream_key(seed, purpose, block, tensor)
    return normal_f32(key, n, 0.0, float(np.float32(cfg.init_std))).reshape(shape)


def init_client(cfg: ServerConfig, seed: Optional[int] = None) -> Dict[str, list]:
    """Initial client model (see the module docstring): the two blocks (12 tensors each, plus
    the prefix keys/values with prefix_len), embedding, final LayerNorm and LM head."""
    seed = cfg.seed if seed is None else seed
    std = float(np.float32(cfg.init_std))
    out = {}
    for name, blk in (("bottom", CB_BOTTOM), ("top", CB_TOP)):
        ts = [init_tensor(cfg, blk, t, seed, P_CLIENT) for t in range(12)]
        if cfg.prefix_len:
            for t, shp in zip((T_PK, T_PV), prefix_shapes(cfg)):
                ts.append(normal_f32(stream_key(seed, P_CLIENT, blk, t), int(np.prod(shp)), 0.0, std).reshape(shp))
        out[name] = ts
    V, H = cfg.vocab, cfg.hidden
    out["embed"] = [normal_f32(stream_key(seed, P_CLIENT, CB_EMBED, 0), V * H, 0.0, std).reshape(V, H)]
    out["head"] = [normal_f32(stream_key(seed, P_CLIENT, CB_HEAD, 0), V * H, 0.0, std).reshape(V, H)]
    out["final_ln"] = [np.ones(H, np.float32), np.zeros(H, np.float32)]
    return out


def client_tokens(cfg: ServerConfig, k: int, seed: Optional[int] = None) -> np.ndarray:
    """Client k's token ids, int32 [client_batch, L_k], uniform over the vocabulary."""
    seed = cfg.seed if seed is None else seed
    L = cfg.seq_lens[k]
    x = raw_u64(stream_key(seed, P_TOKENS, 0, 0, k), 0, cfg.client_batch * L)
    return (x % np.uint64(cfg.vocab)).astype(np.int32).reshape(cfg.client_batch, L)


def client_labels(tokens: np.ndarray, context_lens: Optional[List[int]] = None) -> np.ndarray:
    """Next-token targets of the answer span of each row (-1: no target)."""
    b, L = tokens.shape
    lab = np.full((b, L), -1, np.int32)
    for r in range(b):
        c = 0 if context_lens is None else int(context_lens[r])
        for t in range(L - 1):
            if t + 1 >= c:
                lab[r, t] = tokens[r, t + 1]
    return lab


def init_params(cfg: ServerConfig, seed: Optional[int] = None) -> List[List[np.ndarray]]:
    return [[init_tensor(cfg, b, t, seed) for t in range(12)] for b in range(cfg.n_blocks)]


def client_tensor_bits(cfg: ServerConfig, purpose: int, k: int, seed: Optional[int] = None) -> np.ndarray:
    """Client k's bf16 tensor [client_batch, L_k, H] (uint16 bit patterns): hidden states
    N(0, state_std) for P_STATES, output-state gradients N(0, grad_std) for P_GRADS."""
    seed = cfg.seed if seed is None else seed
    std = cfg.state_std if purpose == P_STATES else cfg.grad_std
    L = cfg.seq_lens[k]
    n = cfg.client_batch * L * cfg.hidden
    v = normal_f32(stream_key(seed, purpose, 0, 0, k), n, 0.0, std)
    return f32_to_bf16_bits(v).reshape(cfg.client_batch, L, cfg.hidden)


def client_states(cfg: ServerConfig, seed: Optional[int] = None) -> List[np.ndarray]:
    return [client_tensor_bits(cfg, P_STATES, k, seed) for k in range(cfg.K)]


def client_grads(cfg: ServerConfig, seed: Optional[int] = None) -> List[np.ndarray]:
    return [client_tensor_bits(cfg, P_GRADS, k, seed) for k in range(cfg.K)]


def glm_structure(cfg: ServerConfig, seed: Optional[int] = None):
    """Per-segment (context length, [M] position) of a GLM workload, segments in
    client-major then row order; see the module docstring for the recipe."""
    seed = cfg.seed if seed is None else seed
    ctx, mpos = [], []
    for s, L in enumerate(cfg.segment_lengths):
        if L < 2:
            ctx.append(1)
            mpos.append(0)
            continue
        x0, x1 = (int(v) for v in raw_u64(stream_key(seed, P_GLM, 0, 0, s), 0, 2))
        c = L - (1 + x0 % max(1, L // 4))
        ctx.append(c)
        mpos.append(c - 1 if x1 % 2 == 0 else (x1 >> 1) % c)
    return ctx, mpos


def _glm(name, n_blocks, K, b, seq_lens, **kw) -> ServerConfig:
    return ServerConfig(name=name, n_blocks=n_blocks, hidden=4096, n_heads=32, head_dim=128,
                        ffn_hidden=16384, residual_alpha=math.sqrt(56.0), client_batch=b,
                        seq_lens=tuple(seq_lens), **kw)


CONFIGS: Dict[str, ServerConfig] = {
    # 1 block, H=256, 4 heads x 64, FFN 1024, alpha = sqrt(2*2), K=2 x b2 x L64
    "tiny": ServerConfig(name="tiny", n_blocks=1, hidden=256, n_heads=4, head_dim=64, ffn_hidden=1024,
                         residual_alpha=2.0, client_batch=2, seq_lens=(64, 64)),
    # one ChatGLM-6B-shaped block, K=4 x b1 x L512
    "block6b": _glm("block6b", 1, 4, 1, (512,) * 4),
    # 26 blocks, K=8 x b4 x L256
    "stack26": _glm("stack26", 26, 8, 4, (256,) * 8),
    # 26 blocks, K=16 x b1, L ~ U[64, 1024] drawn with seed 7
    "ragged26": _glm("ragged26", 26, 16, 1, ragged_lengths(7, 16)),
}


def sweep_config(K: int) -> ServerConfig:
    """26-block stack, per-client batch 2 x seq 512, K clients in one call."""
    return _glm(f"sweep26_K{K}", 26, K, 2, (512,) * K)


SWEEP_KS = (1, 2, 4, 8, 16, 32)
