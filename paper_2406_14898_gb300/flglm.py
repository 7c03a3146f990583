"""Python binding of libflglm.so (ctypes; argument marshalling only).

Every function here forwards to the C ABI of ``include/flglm.h`` and
``include/flglm_kernels.h`` with the same name; all arithmetic runs in the CUDA
library.  Tensors may be passed as anything with ``data_ptr()`` (torch CUDA
tensors) or as raw integer device addresses.  There is no fallback: if the
library is missing or fails to load, every call raises.
"""
from __future__ import annotations

import ctypes as C
import os
from typing import Optional, Sequence

_PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_PKG, "libflglm.so")

FL_OK = 0
ERRORS = {-1: "FL_ERR_INVALID_ARG", -2: "FL_ERR_CAPACITY", -3: "FL_ERR_STATE", -4: "FL_ERR_OOM",
          -5: "FL_ERR_CUDA", -6: "FL_ERR_TIMEOUT", -7: "FL_ERR_UNSUPPORTED"}

(FL_T_WQKV, FL_T_BQKV, FL_T_WDENSE, FL_T_BDENSE, FL_T_WUP, FL_T_BUP, FL_T_WDOWN, FL_T_BDOWN,
 FL_T_LN1_G, FL_T_LN1_B, FL_T_LN2_G, FL_T_LN2_B) = range(12)
FL_T_BLOCK_COUNT = 12
FL_T_PREFIX_K, FL_T_PREFIX_V = 12, 13
FL_T_COUNT = 14
(FL_EPI_STORE, FL_EPI_BIAS_GELU, FL_EPI_BIAS_RESID, FL_EPI_BIAS_ROPE, FL_EPI_GELU_BWD, FL_EPI_RESID,
 FL_EPI_ACCUM_F32, FL_EPI_STORE_F32, FL_EPI_ADAMW) = range(9)
FL_TILE_AUTO, FL_TILE_128x128, FL_TILE_128x256, FL_TILE_256x256_PAIR = range(4)
FL_GEMM_MAX_BATCH = 4
PROF_CLASSES = ("gemm", "attention", "layernorm", "adamw", "other")
FL_DT_BF16, FL_DT_F32 = 0, 1


class FlError(RuntimeError):
    def __init__(self, code: int, msg: str):
        super().__init__(f"{ERRORS.get(code, code)}: {msg}")
        self.code = code


class fl_server_cfg(C.Structure):
    _fields_ = [("n_blocks", C.c_int32), ("hidden", C.c_int32), ("n_heads", C.c_int32), ("head_dim", C.c_int32),
                ("ffn_hidden", C.c_int32), ("rotary_dim", C.c_int32), ("rope_base", C.c_float),
                ("ln_eps", C.c_float), ("residual_alpha", C.c_float), ("residual_from_ln", C.c_int32),
                ("client_batch", C.c_int32), ("max_tokens", C.c_int32), ("max_seq_len", C.c_int32),
                ("recompute", C.c_int32), ("init_std", C.c_float), ("adam_beta1", C.c_float),
                ("adam_beta2", C.c_float), ("adam_eps", C.c_float), ("weight_decay", C.c_float),
                ("prefix_len", C.c_int32), ("freeze_base", C.c_int32), ("fused_step_min_tokens", C.c_int32),
                ("n_replicas", C.c_int32)]


class fl_client_cfg(C.Structure):
    _fields_ = [("block", fl_server_cfg), ("vocab", C.c_int32)]


FL_CP_BOTTOM, FL_CP_TOP, FL_CP_EMBED, FL_CP_HEAD, FL_CP_FINAL_LN = range(5)


class fl_gemm_args(C.Structure):
    _fields_ = [("M", C.c_int32), ("N", C.c_int32), ("K", C.c_int32),
                ("A", C.c_void_p), ("lda", C.c_int64), ("a_mn_major", C.c_int32),
                ("B", C.c_void_p), ("ldb", C.c_int64), ("b_mn_major", C.c_int32),
                ("D", C.c_void_p), ("ldd", C.c_int64), ("epilogue", C.c_int32),
                ("bias", C.c_void_p), ("aux", C.c_void_p), ("ld_aux", C.c_int64), ("alpha", C.c_float),
                ("aux_out", C.c_void_p), ("ld_aux_out", C.c_int64), ("pos", C.c_void_p),
                ("rope_tab", C.c_void_p), ("n_heads", C.c_int32), ("head_dim", C.c_int32),
                ("rotary_dim", C.c_int32), ("aux_dtype", C.c_int32), ("d_dtype", C.c_int32),
                ("ln_mean", C.c_void_p), ("ln_rstd", C.c_void_p), ("ln_gamma", C.c_void_p),
                ("ln_beta", C.c_void_p), ("adam_m", C.c_void_p), ("adam_v", C.c_void_p),
                ("lr", C.c_float), ("beta1", C.c_float), ("beta2", C.c_float), ("eps", C.c_float),
                ("weight_decay", C.c_float), ("inv_bc1", C.c_float), ("inv_bc2", C.c_float),
                ("pos2", C.c_void_p), ("tile", C.c_int32), ("colsum", C.c_void_p),
                ("batch", C.c_int32), ("a_bstride", C.c_int64), ("b_bstride", C.c_int64),
                ("d_bstride", C.c_int64), ("aux_bstride", C.c_int64), ("aux_out_bstride", C.c_int64),
                ("bias_bstride", C.c_int64), ("row_bstride", C.c_int64), ("lnp_bstride", C.c_int64),
                ("adam_bstride", C.c_int64)]


_P = C.c_void_p
_I32 = C.c_int32
_I64 = C.c_int64
_F = C.c_float
_SIGS = {
    "fl_server_cfg_default": (None, [C.POINTER(fl_server_cfg)]),
    "fl_server_create": (C.c_int, [C.POINTER(fl_server_cfg), C.c_uint64, C.POINTER(_P)]),
    "fl_server_forward": (C.c_int, [_P, C.POINTER(_P), C.POINTER(_I32), _I32, C.POINTER(_P)]),
    "fl_server_forward_glm": (C.c_int, [_P, C.POINTER(_P), C.POINTER(_I32), _I32, _P, _P, C.POINTER(_P)]),
    "fl_server_backward": (C.c_int, [_P, C.POINTER(_P), C.POINTER(_P)]),
    "fl_server_step": (C.c_int, [_P, _F]),
    "fl_server_backward_step": (C.c_int, [_P, C.POINTER(_P), C.POINTER(_P), _F]),
    "fl_server_destroy": (C.c_int, [_P]),
    "fl_server_set_stream": (C.c_int, [_P, _P]),
    "fl_server_sync": (C.c_int, [_P]),
    "fl_server_tensor_numel": (_I64, [_P, _I32]),
    "fl_server_get_param": (C.c_int, [_P, _I32, _I32, _P, C.c_size_t]),
    "fl_server_set_param": (C.c_int, [_P, _I32, _I32, _P, C.c_size_t]),
    "fl_server_get_grad": (C.c_int, [_P, _I32, _I32, _P, C.c_size_t]),
    "fl_server_get_adam_moments": (C.c_int, [_P, _I32, _I32, _P, _P, C.c_size_t]),
    "fl_server_average": (C.c_int, [C.POINTER(_P), _I32]),
    "fl_server_param_arena": (C.c_int, [_P, C.POINTER(_P), C.POINTER(_I64)]),
    "fl_server_refresh_working_copy": (C.c_int, [_P]),
    "fl_server_average_finish": (C.c_int, [_P, _I32]),
    "fl_server_average_replicas": (C.c_int, [_P]),
    "fl_server_get_replica_param": (C.c_int, [_P, _I32, _I32, _I32, _P, C.c_size_t]),
    "fl_server_profile": (C.c_int, [_P, C.c_int]),
    "fl_server_profile_read": (C.c_int, [_P, C.POINTER(C.c_double), C.POINTER(_I64), _I32]),
    "fl_server_launch_count": (_I64, [_P]),
    "fl_server_last_error": (C.c_char_p, [_P]),
    "fl_k_gemm": (C.c_int, [C.POINTER(fl_gemm_args), _P, _P]),
    "fl_k_gemm_multi": (C.c_int, [C.POINTER(fl_gemm_args), _I32, _P, _P]),
    "fl_k_layernorm_fwd": (C.c_int, [_I32, _I32, _P, _I32, _P, _P, _F, _P, _P, _P, _P]),
    "fl_k_layernorm_bwd_workspace": (C.c_size_t, [_I32, _I32]),
    "fl_k_layernorm_bwd": (C.c_int, [_I32, _I32, _P, _P, _I32, _P, _P, _P, _P, _F, _P, _P, _P, _P, _P, _P]),
    "fl_k_layernorm_bwd_noalloc": (C.c_int, [_I32, _I32, _P, _P, _P, _P, _P, _P, _F, _P, _P, _P, _P]),
    "fl_k_attention_tiles": (_I32, [_P, _I32]),
    "fl_k_attention_fwd": (C.c_int, [_I32, _I32, _I32, _P, _P, _P, _I32, _P, _P, _P, _P, _P, _I32, _P, _P]),
    "fl_k_attention_bwd": (C.c_int, [_I32, _I32, _I32, _P, _P, _P, _P, _P, _P, _I32, _P, _P, _P, _I32, _P,
                                     _P, _P, _I32, _P, _P, _P, _P, _P, _P]),
    "fl_k_adamw": (C.c_int, [_I64, _P, _P, _P, _P, _P, _F, _F, _F, _F, _F, _F, _F, _P]),
    "fl_k_colsum": (C.c_int, [_I32, _I32, _P, _P, _P]),
    "fl_k_pack_clients": (C.c_int, [_I32, C.POINTER(_P), C.POINTER(_I64), _P, _I32, _P]),
    "fl_k_embedding_gather": (C.c_int, [_I32, _I32, _P, _P, _I32, _P, _P, _P]),
    "fl_k_embedding_scatter_add": (C.c_int, [_I32, _I32, _P, _I32, _P, _P, _P]),
    "fl_k_cross_entropy": (C.c_int, [_I32, _I32, _I64, _P, _P, _P, _P, _P, _P, _P, _P]),
    "fl_client_cfg_default": (None, [C.POINTER(fl_client_cfg)]),
    "fl_client_create": (C.c_int, [C.POINTER(fl_client_cfg), C.c_uint64, C.POINTER(_P)]),
    "fl_client_destroy": (C.c_int, [_P]),
    "fl_client_set_stream": (C.c_int, [_P, _P]),
    "fl_client_sync": (C.c_int, [_P]),
    "fl_client_bottom_forward": (C.c_int, [_P, _P, _I32, _P, _P, _P]),
    "fl_client_top_forward_backward": (C.c_int, [_P, _P, _P, _P, _P]),
    "fl_client_bottom_backward": (C.c_int, [_P, _P]),
    "fl_client_step": (C.c_int, [_P, _F]),
    "fl_client_tensor_numel": (_I64, [_P, _I32, _I32]),
    "fl_client_get_param": (C.c_int, [_P, _I32, _I32, _P, C.c_size_t]),
    "fl_client_set_param": (C.c_int, [_P, _I32, _I32, _P, C.c_size_t]),
    "fl_client_get_grad": (C.c_int, [_P, _I32, _I32, _P, C.c_size_t]),
    "fl_client_average": (C.c_int, [C.POINTER(_P), _I32]),
    "fl_client_launch_count": (_I64, [_P]),
    "fl_client_last_error": (C.c_char_p, [_P]),
}

_lib = None


def lib() -> C.CDLL:
    """Loads libflglm.so (raises if it is missing: there is no CPU fallback)."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError(f"{LIB_PATH} is not built; run `python -m paper_2406_14898_gb300.build`")
        L = C.CDLL(LIB_PATH)
        for name, (res, args) in _SIGS.items():
            f = getattr(L, name)
            f.restype = res
            f.argtypes = args
        _lib = L
    return _lib


def ptr(x) -> Optional[int]:
    if x is None:
        return None
    if isinstance(x, int):
        return x
    return int(x.data_ptr())


def stream_ptr(stream) -> Optional[int]:
    if stream is None:
        return None
    if isinstance(stream, int):
        return stream
    return int(stream.cuda_stream)


def check(rc: int, h=None):
    if rc != FL_OK:
        msg = lib().fl_server_last_error(h)
        raise FlError(rc, msg.decode() if msg else "")


def _parr(xs) -> "C.Array":
    return (C.c_void_p * len(xs))(*[ptr(x) for x in xs])


def make_cfg(c, max_tokens: int, max_seq_len: int = 0, recompute: int = 0,
             fused_step_min_tokens: int = 0, n_replicas: int = 0) -> fl_server_cfg:
    """fl_server_cfg from a workload description with the attributes of
    ``synthetic.ServerConfig`` (n_blocks, hidden, ... , weight_decay); ``recompute``
    keeps one block's activations and recomputes the rest in the backward;
    ``fused_step_min_tokens`` as in fl_server_cfg (0: the library's crossover);
    ``n_replicas`` > 1 holds that many server replicas in the handle (§3.3)."""
    cfg = fl_server_cfg()
    lib().fl_server_cfg_default(C.byref(cfg))
    cfg.n_blocks = c.n_blocks
    cfg.hidden = c.hidden
    cfg.n_heads = c.n_heads
    cfg.head_dim = c.head_dim
    cfg.ffn_hidden = c.ffn_hidden
    cfg.rotary_dim = c.rdim
    cfg.rope_base = c.rope_base
    cfg.ln_eps = c.ln_eps
    cfg.residual_alpha = c.residual_alpha
    cfg.residual_from_ln = c.residual_from_ln
    cfg.client_batch = c.client_batch
    cfg.max_tokens = max_tokens
    cfg.max_seq_len = max_seq_len
    cfg.recompute = recompute
    cfg.init_std = c.init_std
    cfg.adam_beta1 = c.adam_beta1
    cfg.adam_beta2 = c.adam_beta2
    cfg.adam_eps = c.adam_eps
    cfg.weight_decay = c.weight_decay
    cfg.prefix_len = getattr(c, "prefix_len", 0)
    cfg.freeze_base = getattr(c, "freeze_base", 0)
    cfg.fused_step_min_tokens = fused_step_min_tokens
    cfg.n_replicas = n_replicas
    return cfg


class Server:
    """Owns one fl_server handle.  Methods mirror fl_server_* one to one."""

    def __init__(self, cfg: fl_server_cfg, seed: int, stream=None):
        self.h = C.c_void_p()
        rc = lib().fl_server_create(C.byref(cfg), seed, C.byref(self.h))
        check(rc, None)
        self.cfg = cfg
        if stream is not None:
            self.set_stream(stream)

    def close(self):
        if self.h:
            lib().fl_server_destroy(self.h)
            self.h = C.c_void_p()

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def set_stream(self, stream):
        check(lib().fl_server_set_stream(self.h, stream_ptr(stream)), self.h)

    def forward(self, client_states: Sequence, seq_lens: Sequence[int], out_states: Sequence,
                context_lens: Optional[Sequence[int]] = None, mask_pos: Optional[Sequence[int]] = None):
        """context_lens / mask_pos (one per segment, client-major): GLM blank-infilling
        segments through fl_server_forward_glm."""
        K = len(client_states)
        lens = (C.c_int32 * K)(*seq_lens)
        if context_lens is None:
            check(lib().fl_server_forward(self.h, _parr(client_states), lens, K, _parr(out_states)), self.h)
            return
        ctx = (C.c_int32 * len(context_lens))(*context_lens)
        mp = None if mask_pos is None else (C.c_int32 * len(mask_pos))(*mask_pos)
        check(lib().fl_server_forward_glm(self.h, _parr(client_states), lens, K, C.cast(ctx, _P),
                                          None if mp is None else C.cast(mp, _P), _parr(out_states)), self.h)

    def backward(self, grad_out: Sequence, grad_in: Sequence):
        check(lib().fl_server_backward(self.h, _parr(grad_out), _parr(grad_in)), self.h)

    def step(self, lr: float):
        check(lib().fl_server_step(self.h, lr), self.h)

    def backward_step(self, grad_out: Sequence, grad_in: Sequence, lr: float):
        check(lib().fl_server_backward_step(self.h, _parr(grad_out), _parr(grad_in), lr), self.h)

    def sync(self):
        check(lib().fl_server_sync(self.h), self.h)

    def numel(self, tensor_id: int) -> int:
        return int(lib().fl_server_tensor_numel(self.h, tensor_id))

    def _get(self, fn, block, tensor_id):
        import numpy as np
        out = np.empty(self.numel(tensor_id), np.float32)
        check(fn(self.h, block, tensor_id, out.ctypes.data, out.size), self.h)
        return out

    def get_param(self, block: int, tensor_id: int):
        return self._get(lib().fl_server_get_param, block, tensor_id)

    def get_replica_param(self, replica: int, block: int, tensor_id: int):
        import numpy as np
        out = np.empty(self.numel(tensor_id), np.float32)
        check(lib().fl_server_get_replica_param(self.h, replica, block, tensor_id, out.ctypes.data, out.size), self.h)
        return out

    def get_grad(self, block: int, tensor_id: int):
        return self._get(lib().fl_server_get_grad, block, tensor_id)

    def get_adam_moments(self, block: int, tensor_id: int):
        import numpy as np
        n = self.numel(tensor_id)
        m = np.empty(n, np.float32)
        v = np.empty(n, np.float32)
        check(lib().fl_server_get_adam_moments(self.h, block, tensor_id, m.ctypes.data, v.ctypes.data, n), self.h)
        return m, v

    def set_param(self, block: int, tensor_id: int, values):
        import numpy as np
        a = np.ascontiguousarray(values, np.float32).reshape(-1)
        check(lib().fl_server_set_param(self.h, block, tensor_id, a.ctypes.data, a.size), self.h)

    def param_arena(self):
        """(device address, element count) of the fp32 master-weight arena."""
        p = C.c_void_p()
        n = C.c_int64()
        check(lib().fl_server_param_arena(self.h, C.byref(p), C.byref(n)), self.h)
        return int(p.value), int(n.value)

    def refresh_working_copy(self):
        check(lib().fl_server_refresh_working_copy(self.h), self.h)

    def average_finish(self, n_replicas: int):
        check(lib().fl_server_average_finish(self.h, n_replicas), self.h)

    def average_replicas(self):
        """The §3.3 period-end average of the replicas held in this handle."""
        check(lib().fl_server_average_replicas(self.h), self.h)

    def profile(self, enable: bool):
        check(lib().fl_server_profile(self.h, 1 if enable else 0), self.h)

    def profile_read(self) -> dict:
        n = len(PROF_CLASSES)
        ms = (C.c_double * n)()
        cnt = (C.c_int64 * n)()
        check(lib().fl_server_profile_read(self.h, ms, cnt, n), self.h)
        return {PROF_CLASSES[i]: (float(ms[i]), int(cnt[i])) for i in range(n)}

    def launch_count(self) -> int:
        return int(lib().fl_server_launch_count(self.h))


def fl_server_average(replicas: Sequence["Server"]):
    """Averages the replicas' parameters in place (the server-hierarchical strategy)."""
    arr = (C.c_void_p * len(replicas))(*[r.h.value for r in replicas])
    check(lib().fl_server_average(arr, len(replicas)), replicas[0].h if replicas else None)


def make_client_cfg(c, max_tokens: int, max_seq_len: int = 0) -> fl_client_cfg:
    """fl_client_cfg from a workload description (block fields as make_cfg, plus vocab)."""
    cfg = fl_client_cfg()
    lib().fl_client_cfg_default(C.byref(cfg))
    cfg.block = make_cfg(c, max_tokens, max_seq_len)
    cfg.block.n_blocks = 1
    cfg.vocab = c.vocab
    return cfg


def check_client(rc: int, h):
    if rc != FL_OK:
        msg = lib().fl_client_last_error(h)
        raise FlError(rc, msg.decode() if msg else "")


class Client:
    """Owns one fl_client handle (the client parts of §3.1).  Methods mirror fl_client_*."""

    def __init__(self, cfg: fl_client_cfg, seed: int, stream=None):
        self.h = C.c_void_p()
        rc = lib().fl_client_create(C.byref(cfg), seed, C.byref(self.h))
        check_client(rc, None)
        self.cfg = cfg
        if stream is not None:
            self.set_stream(stream)

    def close(self):
        if self.h:
            lib().fl_client_destroy(self.h)
            self.h = C.c_void_p()

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def set_stream(self, stream):
        check_client(lib().fl_client_set_stream(self.h, stream_ptr(stream)), self.h)

    def sync(self):
        check_client(lib().fl_client_sync(self.h), self.h)

    def bottom_forward(self, tokens, seq_len: int, h0, context_lens=None, mask_pos=None):
        ctx = None if context_lens is None else (C.c_int32 * len(context_lens))(*context_lens)
        mp = None if mask_pos is None else (C.c_int32 * len(mask_pos))(*mask_pos)
        check_client(lib().fl_client_bottom_forward(self.h, ptr(tokens), seq_len,
                                                    None if ctx is None else C.cast(ctx, _P),
                                                    None if mp is None else C.cast(mp, _P), ptr(h0)), self.h)

    def top_forward_backward(self, h, labels, loss, grad_h):
        check_client(lib().fl_client_top_forward_backward(self.h, ptr(h), ptr(labels), ptr(loss), ptr(grad_h)),
                     self.h)

    def bottom_backward(self, grad_h0):
        check_client(lib().fl_client_bottom_backward(self.h, ptr(grad_h0)), self.h)

    def step(self, lr: float):
        check_client(lib().fl_client_step(self.h, lr), self.h)

    def numel(self, part: int, tensor: int) -> int:
        return int(lib().fl_client_tensor_numel(self.h, part, tensor))

    def _get(self, fn, part, tensor):
        import numpy as np
        out = np.empty(self.numel(part, tensor), np.float32)
        check_client(fn(self.h, part, tensor, out.ctypes.data, out.size), self.h)
        return out

    def get_param(self, part: int, tensor: int):
        return self._get(lib().fl_client_get_param, part, tensor)

    def get_grad(self, part: int, tensor: int):
        return self._get(lib().fl_client_get_grad, part, tensor)

    def set_param(self, part: int, tensor: int, values):
        import numpy as np
        a = np.ascontiguousarray(values, np.float32).reshape(-1)
        check_client(lib().fl_client_set_param(self.h, part, tensor, a.ctypes.data, a.size), self.h)

    def launch_count(self) -> int:
        return int(lib().fl_client_launch_count(self.h))


def fl_client_average(clients: Sequence["Client"]):
    """Averages the clients' parameters in place (end of a training period, §3.3)."""
    arr = (C.c_void_p * len(clients))(*[c.h.value for c in clients])
    check_client(lib().fl_client_average(arr, len(clients)), clients[0].h if clients else None)


# ----------------------------------------------------------------------------- kernel-level calls

def fl_k_gemm(args: fl_gemm_args, status=None, stream=None):
    check(lib().fl_k_gemm(C.byref(args), ptr(status), stream_ptr(stream)))


def fl_k_gemm_multi(args: Sequence[fl_gemm_args], status=None, stream=None):
    arr = (fl_gemm_args * len(args))(*args)
    check(lib().fl_k_gemm_multi(arr, len(args), ptr(status), stream_ptr(stream)))


def gemm(M, N, K, A, lda, a_mn, B, ldb, b_mn, D, ldd, status=None, stream=None, **kw):
    """One fl_k_gemm call; arguments as gemm_args."""
    fl_k_gemm(gemm_args(M, N, K, A, lda, a_mn, B, ldb, b_mn, D, ldd, **kw), status, stream)


def gemm_args(M, N, K, A, lda, a_mn, B, ldb, b_mn, D, ldd, epilogue=FL_EPI_STORE, bias=None, aux=None, ld_aux=0,
              alpha=0.0, aux_out=None, ld_aux_out=0, pos=None, rope_tab=None, n_heads=0, head_dim=0, rotary_dim=0,
              aux_dtype=FL_DT_BF16, d_dtype=FL_DT_BF16, ln_mean=None, ln_rstd=None, ln_gamma=None, ln_beta=None,
              pos2=None, tile=0, colsum=None, batch=1, bstrides=None, **fields) -> fl_gemm_args:
    """bstrides: {"a": .., "b": .., "d": .., "aux": .., "aux_out": .., "bias": .., "row": .., "lnp": ..,
    "adam": ..} element strides between the problems of a batched launch; `fields` sets any
    other fl_gemm_args field by name (tensors as device pointers)."""
    a = fl_gemm_args(M, N, K, ptr(A), lda, a_mn, ptr(B), ldb, b_mn, ptr(D), ldd, epilogue, ptr(bias), ptr(aux),
                     ld_aux, alpha, ptr(aux_out), ld_aux_out, ptr(pos), ptr(rope_tab), n_heads, head_dim, rotary_dim,
                     aux_dtype, d_dtype, ptr(ln_mean), ptr(ln_rstd), ptr(ln_gamma), ptr(ln_beta))
    a.pos2 = ptr(pos2)
    a.tile = tile
    a.colsum = ptr(colsum)
    a.batch = batch
    for k, v in (bstrides or {}).items():
        setattr(a, f"{k}_bstride", int(v))
    for k, v in fields.items():
        setattr(a, k, v if isinstance(v, (int, float)) else ptr(v))
    return a


def fl_k_layernorm_fwd(T, H, x, gamma, beta, eps, y, mean, rstd, x_dtype=FL_DT_BF16, stream=None):
    check(lib().fl_k_layernorm_fwd(T, H, ptr(x), x_dtype, ptr(gamma), ptr(beta), eps, ptr(y), ptr(mean), ptr(rstd),
                                   stream_ptr(stream)))


def fl_k_layernorm_bwd_workspace(T, H) -> int:
    return int(lib().fl_k_layernorm_bwd_workspace(T, H))


def fl_k_layernorm_bwd(T, H, dy, x, mean, rstd, gamma, resid, resid_alpha, dx_bf16, dgamma, dbeta, workspace,
                       io_dtype=FL_DT_BF16, dx_f32=None, stream=None):
    check(lib().fl_k_layernorm_bwd(T, H, ptr(dy), ptr(x), io_dtype, ptr(mean), ptr(rstd), ptr(gamma), ptr(resid),
                                   resid_alpha, ptr(dx_bf16), ptr(dx_f32), ptr(dgamma), ptr(dbeta), ptr(workspace),
                                   stream_ptr(stream)))


def fl_k_layernorm_bwd_noalloc(T, H, dy, x, mean, rstd, gamma, resid, resid_alpha, dx, dgamma, dbeta, stream=None):
    check(lib().fl_k_layernorm_bwd_noalloc(T, H, ptr(dy), ptr(x), ptr(mean), ptr(rstd), ptr(gamma), ptr(resid),
                                           resid_alpha, ptr(dx), ptr(dgamma), ptr(dbeta), stream_ptr(stream)))


def fl_k_attention_tiles(cu_host) -> int:
    import numpy as np
    a = np.ascontiguousarray(cu_host, np.int32)
    return int(lib().fl_k_attention_tiles(a.ctypes.data, a.size - 1))


def fl_k_attention_fwd(T, n_heads, head_dim, qkv, cu_host, cu_dev, tile_ws, o, lse, prefix_k=None, prefix_v=None,
                       prefix_len=0, context_lens=None, stream=None):
    import numpy as np
    a = np.ascontiguousarray(cu_host, np.int32)
    check(lib().fl_k_attention_fwd(T, n_heads, head_dim, ptr(qkv), a.ctypes.data, ptr(cu_dev), a.size - 1,
                                   ptr(tile_ws), ptr(o), ptr(lse), ptr(prefix_k), ptr(prefix_v), prefix_len,
                                   ptr(context_lens), stream_ptr(stream)))


def fl_k_attention_bwd(T, n_heads, head_dim, qkv, o, lse, dout, cu_host, cu_dev, tile_ws, delta_ws, rope_tab,
                       rotary_dim, dqkv, prefix_k=None, prefix_v=None, prefix_len=0, dprefix_k=None, dprefix_v=None,
                       context_lens=None, positions=None, block_positions=None, stream=None):
    import numpy as np
    a = np.ascontiguousarray(cu_host, np.int32)
    check(lib().fl_k_attention_bwd(T, n_heads, head_dim, ptr(qkv), ptr(o), ptr(lse), ptr(dout), a.ctypes.data,
                                   ptr(cu_dev), a.size - 1, ptr(tile_ws), ptr(delta_ws), ptr(rope_tab), rotary_dim,
                                   ptr(dqkv), ptr(prefix_k), ptr(prefix_v), prefix_len, ptr(dprefix_k),
                                   ptr(dprefix_v), ptr(context_lens), ptr(positions), ptr(block_positions),
                                   stream_ptr(stream)))


def fl_k_embedding_gather(T, H, tokens, table, vocab, out, status, stream=None):
    check(lib().fl_k_embedding_gather(T, H, ptr(tokens), ptr(table), vocab, ptr(out), ptr(status), stream_ptr(stream)))


def fl_k_embedding_scatter_add(T, H, tokens, vocab, dx, dtable, stream=None):
    check(lib().fl_k_embedding_scatter_add(T, H, ptr(tokens), vocab, ptr(dx), ptr(dtable), stream_ptr(stream)))


def fl_k_cross_entropy(T, vocab, ld, logits, labels, row_loss, dlogits, loss, count, status, stream=None):
    check(lib().fl_k_cross_entropy(T, vocab, ld, ptr(logits), ptr(labels), ptr(row_loss), ptr(dlogits), ptr(loss),
                                   ptr(count), ptr(status), stream_ptr(stream)))


def fl_k_adamw(n, w, g, m, v, w_bf16, lr, beta1, beta2, eps, weight_decay, bc1, bc2, stream=None):
    check(lib().fl_k_adamw(n, ptr(w), ptr(g), ptr(m), ptr(v), ptr(w_bf16), lr, beta1, beta2, eps, weight_decay,
                           bc1, bc2, stream_ptr(stream)))


def fl_k_colsum(T, N, x, out, stream=None):
    check(lib().fl_k_colsum(T, N, ptr(x), ptr(out), stream_ptr(stream)))


def fl_k_pack_clients(clients: Sequence, nbytes: Sequence[int], packed, scatter: bool, stream=None):
    K = len(clients)
    b = (C.c_int64 * K)(*nbytes)
    check(lib().fl_k_pack_clients(K, _parr(clients), b, ptr(packed), 1 if scatter else 0, stream_ptr(stream)))
