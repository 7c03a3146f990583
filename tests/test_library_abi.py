"""CPU-side checks of the C ABI: the library loads without a GPU, exports every
function that include/*.h declares, and the host-side validation answers with the
documented error codes (no compute call is made)."""
import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def declared_functions():
    names = set()
    for h in ("flglm.h", "flglm_kernels.h", "flglm_client.h"):
        with open(os.path.join(ROOT, "include", h)) as fh:
            src = fh.read()
        src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
        for m in re.finditer(r"\b(fl_[a-z0-9_]+)\s*\(", src):
            names.add(m.group(1))
    return sorted(names)


@pytest.fixture(scope="module")
def F():
    from paper_2406_14898_gb300 import build, flglm
    build.build()
    flglm.lib()
    return flglm


def test_every_declared_symbol_is_exported(F):
    names = declared_functions()
    assert len(names) >= 25
    L = F.lib()
    missing = [n for n in names if not hasattr(L, n)]
    assert not missing, missing
    # and the binding covers them all with the same names
    assert set(names) <= set(F._SIGS), set(names) - set(F._SIGS)


def test_cfg_default_and_validation(F):
    cfg = F.fl_server_cfg()
    F.lib().fl_server_cfg_default(ctypes.byref(cfg))
    assert (cfg.n_blocks, cfg.hidden, cfg.n_heads, cfg.head_dim, cfg.ffn_hidden) == (26, 4096, 32, 128, 16384)
    assert abs(cfg.residual_alpha - 56 ** 0.5) < 1e-6
    h = ctypes.c_void_p()
    bad = F.fl_server_cfg()
    F.lib().fl_server_cfg_default(ctypes.byref(bad))
    bad.head_dim = 96
    bad.n_heads = 4096 // 96
    assert F.lib().fl_server_create(ctypes.byref(bad), 0, ctypes.byref(h)) in (-1, -7)
    assert not h.value
    bad.head_dim = 128
    bad.n_heads = 32
    bad.rotary_dim = 32
    assert F.lib().fl_server_create(ctypes.byref(bad), 0, ctypes.byref(h)) == -7
    assert b"rotary" in F.lib().fl_server_last_error(None)
    assert F.lib().fl_server_create(None, 0, ctypes.byref(h)) == -1
    assert F.lib().fl_server_forward(None, None, None, 1, None) == -1
    assert F.lib().fl_server_destroy(None) == 0
    cfg = F.fl_server_cfg()
    F.lib().fl_server_cfg_default(ctypes.byref(cfg))
    assert cfg.fused_step_min_tokens == 0
    cfg.fused_step_min_tokens = -1
    assert F.lib().fl_server_create(ctypes.byref(cfg), 0, ctypes.byref(h)) == -1
    assert not h.value and b"fused_step_min_tokens" in F.lib().fl_server_last_error(None)
    # client handles: defaults, validation before any device work
    cc = F.fl_client_cfg()
    F.lib().fl_client_cfg_default(ctypes.byref(cc))
    assert cc.vocab == 130528 and cc.block.hidden == 4096
    cc.vocab = 0
    assert F.lib().fl_client_create(ctypes.byref(cc), 0, ctypes.byref(h)) == -1
    assert not h.value and b"vocab" in F.lib().fl_client_last_error(None)
    assert F.lib().fl_client_bottom_forward(None, None, 1, None, None, None) == -1
    assert F.lib().fl_client_destroy(None) == 0


def no_gpu_here():
    """The checks below pass made-up device addresses: they run only where no GPU exists, so
    that a check that regressed could never launch a kernel on them."""
    import torch
    if torch.cuda.is_available():
        pytest.skip("made-up device addresses: CPU-only check")


def test_kernel_entry_points_validate_before_launch(F):
    no_gpu_here()
    L = F.lib()
    a = F.fl_gemm_args()
    assert L.fl_k_gemm(ctypes.byref(a), None, None) == -1          # null operands
    # tile shape checks come before any device call (addresses are never dereferenced)
    a = F.fl_gemm_args(8, 384, 64, 0x10000, 64, 0, 0x20000, 64, 0, 0x30000, 384, F.FL_EPI_STORE)
    a.tile = 7
    assert L.fl_k_gemm(ctypes.byref(a), None, None) == -1
    a.tile = F.FL_TILE_128x256                                      # N % 256 != 0
    assert L.fl_k_gemm(ctypes.byref(a), None, None) == -7
    a.tile = F.FL_TILE_256x256_PAIR
    assert L.fl_k_gemm(ctypes.byref(a), None, None) == -7
    a.tile = F.FL_TILE_AUTO
    a.colsum = 0x40000                                              # only with FL_EPI_GELU_BWD
    assert L.fl_k_gemm(ctypes.byref(a), None, None) == -7
    assert L.fl_k_layernorm_fwd(4, 300, None, 0, None, None, 1e-5, None, None, None, None) == -7
    assert L.fl_k_adamw(6, None, None, None, None, None, 1e-3, .9, .999, 1e-8, 0, .1, .001, None) == -1


def test_kernel_entry_points_check_alignment(F):
    """Every pointer a kernel reads or writes with vector accesses is checked for the width
    it is accessed with; a misaligned one is refused (INVALID_ARG) before any CUDA call."""
    no_gpu_here()
    L = F.lib()
    A = [0x100000 * (i + 1) for i in range(16)]          # made-up, 16-byte aligned, never dereferenced
    odd = lambda p, b=4: p + b                           # noqa: E731
    CUDA = -5  # aligned arguments pass the checks and fail at the first CUDA call (no device here)
    # LayerNorm forward: x, gamma, beta, y
    args = [4, 256, A[0], 0, A[1], A[2], 1e-5, A[3], A[4], A[5], None]
    assert L.fl_k_layernorm_fwd(*args) == CUDA
    for i in (2, 4, 5, 7):
        bad = list(args)
        bad[i] = odd(bad[i], 8)
        assert L.fl_k_layernorm_fwd(*bad) == -1, i
    # LayerNorm backward: dy, x, gamma, resid, dx_bf16, dx_f32, workspace
    args = [4, 256, A[0], A[1], 0, A[2], A[3], A[4], A[5], 1.0, A[6], A[7], A[8], A[9], A[10], None]
    assert L.fl_k_layernorm_bwd(*args) == CUDA
    for i in (2, 3, 7, 8, 10, 11, 14):
        bad = list(args)
        bad[i] = odd(bad[i], 8)
        assert L.fl_k_layernorm_bwd(*bad) == -1, i
    args = [4, 256, A[0], A[1], A[2], A[3], A[4], A[5], 1.0, A[6], A[7], A[8], None]
    assert L.fl_k_layernorm_bwd_noalloc(*args) == CUDA
    for i in (2, 3, 6, 7, 9):
        bad = list(args)
        bad[i] = odd(bad[i], 8)
        assert L.fl_k_layernorm_bwd_noalloc(*bad) == -1, i
    # column sums, AdamW (w, g, m, v 16-byte, the bf16 copy 8-byte)
    assert L.fl_k_colsum(4, 256, A[0], A[1], None) == CUDA
    assert L.fl_k_colsum(4, 256, odd(A[0], 8), A[1], None) == -1
    assert L.fl_k_adamw(8, A[0], A[1], A[2], A[3], A[4], 1e-3, .9, .999, 1e-8, 0., .1, .001, None) == CUDA
    for i in (1, 2, 3, 4):
        bad = [8, A[0], A[1], A[2], A[3], A[4], 1e-3, .9, .999, 1e-8, 0., .1, .001, None]
        bad[i] = odd(bad[i])
        assert L.fl_k_adamw(*bad) == -1, i
    assert L.fl_k_adamw(8, A[0], A[1], A[2], A[3], odd(A[4]), 1e-3, .9, .999, 1e-8, 0., .1, .001, None) == -1
    # embedding table / output rows (16-byte), scatter operands (4-byte)
    assert L.fl_k_embedding_gather(4, 256, A[0], A[1], 10, A[2], A[3], None) == CUDA
    assert L.fl_k_embedding_scatter_add(4, 256, A[0], 10, A[1], A[2], None) == CUDA
    assert L.fl_k_embedding_gather(4, 256, A[0], odd(A[1], 8), 10, A[2], A[3], None) == -1
    assert L.fl_k_embedding_gather(4, 256, A[0], A[1], 10, odd(A[2], 8), A[3], None) == -1
    assert L.fl_k_embedding_scatter_add(4, 256, A[0], 10, odd(A[1], 2), A[2], None) == -1
    # attention: o (forward); o, dout, dqkv and the prefix gradients (backward)
    cu = (ctypes.c_int32 * 2)(0, 4)
    assert L.fl_k_attention_fwd(4, 2, 128, A[0], cu, A[1], 1, A[2], A[3], A[4], None, None, 0, None, None) == CUDA
    assert L.fl_k_attention_fwd(4, 2, 128, A[0], cu, A[1], 1, A[2], odd(A[3], 8), A[4], None, None, 0, None,
                                None) == -1
    bwd = [4, 2, 128, A[0], A[1], A[2], A[3], cu, A[4], 1, A[5], A[6], None, 64, A[7], A[8], A[9], 4, A[10],
           A[11], None, None, None, None]
    assert L.fl_k_attention_bwd(*bwd) == CUDA
    for i in (4, 6, 14, 18, 19):
        bad = list(bwd)
        bad[i] = odd(bad[i], 8)
        assert L.fl_k_attention_bwd(*bad) == -1, i
    # GEMM: the rotary table is read as (cos, sin) pairs
    a = F.fl_gemm_args(8, 384, 64, A[0], 64, 0, A[1], 64, 0, A[2], 384, F.FL_EPI_STORE)
    a.rope_tab = A[3]
    assert L.fl_k_gemm(ctypes.byref(a), None, None) == CUDA
    a.rope_tab = odd(A[3])
    assert L.fl_k_gemm(ctypes.byref(a), None, None) == -1
