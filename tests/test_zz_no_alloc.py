"""The allocation-free LayerNorm backward (fl_k_layernorm_bwd_noalloc) against the
workspace-taking entry point (fl_k_layernorm_bwd), GPU only.

The no-alloc variant is for callers that cannot call cudaMalloc (a plug-in whose host
framework owns all device memory, a loop that cannot afford cudaMalloc's device
synchronisation, a fully reserved memory budget): its scratch is a fixed array inside
the library.  Two calls in a row with different inputs check that the second call does
not depend on what the first left in the shared array.  This file is collected last so
that a run that stops at the first failure has already run every other test.
"""
import ctypes

import numpy as np
import pytest
import torch

from tests._gpu import dev_bf16, dev_f32, f64, flglm, need_gpu, rel_inf, rnd_bf16_f64

pytestmark = pytest.mark.gpu


def _inputs(rng, T, H):
    x = rnd_bf16_f64(rng, (T, H), 2.0)
    g = (1 + 0.2 * rng.standard_normal(H)).astype(np.float32)
    b = (0.2 * rng.standard_normal(H)).astype(np.float32)
    dy = rnd_bf16_f64(rng, (T, H))
    res = rnd_bf16_f64(rng, (T, H))
    return x, g, b, dy, res


def test_noalloc_layernorm_bwd_matches_workspace_variant():
    need_gpu()
    F = flglm()
    L = F.lib()
    rng = np.random.default_rng(123)
    for T, H, use_res in ((300, 4096, False), (77, 4096, True), (1000, 256, True)):
        x, g, b, dy, res = _inputs(rng, T, H)
        dx_, dg_, db_, ddy, dres = dev_bf16(x), dev_f32(g), dev_f32(b), dev_bf16(dy), dev_bf16(res)
        y = torch.empty((T, H), dtype=torch.bfloat16, device="cuda")
        mean = torch.empty(T, dtype=torch.float32, device="cuda")
        rstd = torch.empty(T, dtype=torch.float32, device="cuda")
        F.fl_k_layernorm_fwd(T, H, dx_, dg_, db_, 1e-5, y, mean, rstd)
        # existing entry point with a caller-provided workspace
        ws = torch.empty(F.fl_k_layernorm_bwd_workspace(T, H) // 4 + 64, dtype=torch.float32, device="cuda")
        dx_ref = torch.empty((T, H), dtype=torch.bfloat16, device="cuda")
        dgam_ref = torch.zeros(H, dtype=torch.float32, device="cuda")
        dbet_ref = torch.zeros(H, dtype=torch.float32, device="cuda")
        F.fl_k_layernorm_bwd(T, H, ddy, dx_, mean, rstd, dg_, dres if use_res else None, 2.5, dx_ref, dgam_ref,
                             dbet_ref, ws, io_dtype=F.FL_DT_BF16)
        # the allocation-free entry point, called through the C ABI
        dx_na = torch.full((T, H), float("nan"), dtype=torch.bfloat16, device="cuda")
        dgam_na = torch.zeros(H, dtype=torch.float32, device="cuda")
        dbet_na = torch.zeros(H, dtype=torch.float32, device="cuda")
        rc = L.fl_k_layernorm_bwd_noalloc(T, H, ddy.data_ptr(), dx_.data_ptr(), mean.data_ptr(), rstd.data_ptr(),
                                          dg_.data_ptr(), dres.data_ptr() if use_res else None, ctypes.c_float(2.5),
                                          dx_na.data_ptr(), dgam_na.data_ptr(), dbet_na.data_ptr(), None)
        assert rc == 0, L.fl_server_last_error(None)
        torch.cuda.synchronize()
        assert rel_inf(f64(dx_na), f64(dx_ref)) < 1e-2
        assert rel_inf(f64(dgam_na), f64(dgam_ref)) < 1e-4
        assert rel_inf(f64(dbet_na), f64(dbet_ref)) < 1e-4


def test_noalloc_layernorm_bwd_rejects_oversized_hidden():
    """H above the fixed array's 4096 columns is refused before any launch.  The buffers
    are real and sized for H = 8192, so that even a launch that slipped past the check
    would stay inside memory the test owns."""
    need_gpu()
    F = flglm()
    L = F.lib()
    T, H = 4, 8192
    bf = [torch.zeros((T, H), dtype=torch.bfloat16, device="cuda") for _ in range(4)]  # dy, x, resid, dx
    rows = [torch.ones(T, dtype=torch.float32, device="cuda") for _ in range(2)]         # mean, rstd
    cols = [torch.zeros(H, dtype=torch.float32, device="cuda") for _ in range(3)]        # gamma, dgamma, dbeta
    dy, x, res, dx = bf
    mean, rstd = rows
    gamma, dgam, dbet = cols
    rc = L.fl_k_layernorm_bwd_noalloc(T, H, dy.data_ptr(), x.data_ptr(), mean.data_ptr(), rstd.data_ptr(),
                                      gamma.data_ptr(), res.data_ptr(), ctypes.c_float(0.0), dx.data_ptr(),
                                      dgam.data_ptr(), dbet.data_ptr(), None)
    assert rc == -2
    assert b"4096" in L.fl_server_last_error(None)
    rc = L.fl_k_layernorm_bwd_noalloc(-1, 256, dy.data_ptr(), x.data_ptr(), mean.data_ptr(), rstd.data_ptr(),
                                      gamma.data_ptr(), res.data_ptr(), ctypes.c_float(0.0), dx.data_ptr(),
                                      dgam.data_ptr(), dbet.data_ptr(), None)
    assert rc == -1
    assert b"negative" in L.fl_server_last_error(None)
    torch.cuda.synchronize()
    assert not dgam.any() and not dbet.any() and not dx.view(torch.int16).any()
