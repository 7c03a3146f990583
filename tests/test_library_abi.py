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
        src = open(os.path.join(ROOT, "include", h)).read()
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


def test_kernel_entry_points_validate_before_launch(F):
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
