"""Activation recompute (cfg.recompute = 1) on the GPU: one block's activations are kept
and each block's forward runs again before its backward.  Every kernel that produces the
activations is deterministic, so from the same state the results must be the same bits
as with every activation kept; the bias, LayerNorm and prefix gradients are summed with
fp32 atomics, so for those only the rounding may differ.  (Over several steps two runs
drift apart either way: those rounding differences flip bf16 roundings of activations.)
GPU only."""
import numpy as np
import pytest
import torch

import synthetic as syn
from oracle import flglm_oracle as O
from tests._gpu import bits, dev_bf16_from_bits, f64, flglm, need_gpu, rel_inf
from tests.test_gpu_server import GRAD_TOL, OUT_TOL, check_updated_weights

pytestmark = pytest.mark.gpu

MATRICES = (0, 2, 4, 6)  # Wqkv, Wdense, Wup, Wdown: weight-gradient GEMMs, no atomics


@pytest.fixture(scope="module")
def F():
    need_gpu()
    return flglm()


def glm_kwargs(cfg):
    if not cfg.glm:
        return {}
    ctx, mp = syn.glm_structure(cfg)
    return {"context_lens": ctx, "mask_pos": mp}


def run(F, cfg, recompute, fused):
    """One forward and one backward (fused: backward + AdamW step) from the seeded state."""
    srv = F.Server(F.make_cfg(cfg, cfg.tokens, max(cfg.seq_lens), recompute=recompute, fused_step_min_tokens=1),
                   cfg.seed)
    states = [dev_bf16_from_bits(s) for s in syn.client_states(cfg)]
    grads = [dev_bf16_from_bits(g) for g in syn.client_grads(cfg)]
    outs = [torch.empty_like(s) for s in states]
    gins = [torch.empty_like(s) for s in states]
    srv.forward(states, cfg.seq_lens, outs, **glm_kwargs(cfg))
    if fused:
        srv.backward_step(grads, gins, 1e-3)
    else:
        srv.backward(grads, gins)
    srv.sync()
    n_t = 14 if cfg.prefix_len else 12
    get = srv.get_param if fused else srv.get_grad
    res = {"outs": [bits(o) for o in outs], "gins": [bits(g) for g in gins],
           "tensors": [[get(b, t) for t in range(n_t)] for b in range(cfg.n_blocks)]}
    srv.close()
    return res


def compare(cfg, kept, rec, n_t):
    """Outputs, input gradients and the weight matrices' gradients (or updated weights)
    bit for bit; the vectors summed with atomics to rounding.  After a step a vector
    element whose gradient is pure rounding noise (the key bias on unrotated dims) may
    move by +-lr either way, so for the updated vectors a few elements may differ more."""
    for k in range(cfg.K):
        np.testing.assert_array_equal(rec["outs"][k], kept["outs"][k])
        np.testing.assert_array_equal(rec["gins"][k], kept["gins"][k])
    for b in range(cfg.n_blocks):
        for t in range(n_t):
            xk, xr = kept["tensors"][b][t], rec["tensors"][b][t]
            if t in MATRICES:
                np.testing.assert_array_equal(xr.view(np.uint32), xk.view(np.uint32), err_msg=f"{b} {t}")
            else:
                far = np.abs(xr.astype(np.float64) - xk) > 1e-5 * np.abs(xk).max()
                assert far.mean() < 0.01, (b, t, far.sum())


@pytest.mark.parametrize("fused", [False, True], ids=["backward", "backward_step"])
@pytest.mark.parametrize("mode", ["causal", "glm_prefix"])
def test_recompute_bit_identical(F, mode, fused):
    """One pass from the same seeded state with and without recompute.  With the fused
    backward + step the weight matrices are updated inside the GEMM epilogue while the
    recomputed forward of the next lower block still reads its own, not yet updated,
    weights."""
    if mode == "causal":
        cfg = syn.CONFIGS["tiny"].with_(n_blocks=3, client_batch=2, seq_lens=(1, 64, 130, 17))
    else:
        cfg = syn.CONFIGS["tiny"].with_(n_blocks=3, client_batch=1, seq_lens=(64, 90, 33), prefix_len=20, glm=1)
    n_t = 14 if cfg.prefix_len else 12
    compare(cfg, run(F, cfg, 0, fused), run(F, cfg, 1, fused), n_t)


def test_recompute_oracle_parity(F):
    """Outputs, input and weight gradients and the weights after one AdamW step of a
    recomputing server against the fp64 oracle."""
    cfg = syn.CONFIGS["tiny"].with_(n_blocks=2, client_batch=1, seq_lens=(5, 64, 100))
    srv = F.Server(F.make_cfg(cfg, cfg.tokens, max(cfg.seq_lens), recompute=1), cfg.seed)
    states, grads = syn.client_states(cfg), syn.client_grads(cfg)
    st = [dev_bf16_from_bits(s) for s in states]
    outs = [torch.empty_like(s) for s in st]
    gi = [torch.empty_like(s) for s in st]
    srv.forward(st, cfg.seq_lens, outs)
    srv.backward([dev_bf16_from_bits(g) for g in grads], gi)
    srv.sync()
    ref = O.OracleServer(cfg, syn.init_params(cfg))
    ro = ref.forward([syn.bf16_bits_to_f64(s) for s in states])
    rg = ref.backward([syn.bf16_bits_to_f64(g) for g in grads])
    for k in range(cfg.K):
        assert rel_inf(f64(outs[k]), ro[k]) < OUT_TOL, k
        assert rel_inf(f64(gi[k]), rg[k]) < GRAD_TOL, k
    w0 = [[p.reshape(-1).copy() for p in blk] for blk in ref.params]
    gref = [[g.reshape(-1).copy() for g in blk] for blk in ref.grads]
    for b in range(cfg.n_blocks):
        for t in range(12):
            assert rel_inf(srv.get_grad(b, t), gref[b][t]) < GRAD_TOL, (b, t)
    srv.step(cfg.lr)
    srv.sync()
    ref.step(cfg.lr)
    for b in range(cfg.n_blocks):
        for t in range(12):
            check_updated_weights(srv.get_param(b, t), ref.params[b][t].reshape(-1), w0[b][t], gref[b][t],
                                  cfg.lr, (b, t))
    srv.close()


def test_recompute_bit_identical_6b_shapes(F):
    """Two ChatGLM-6B-shaped blocks (H 4096, 32 x 128, F 16384), K = 4 x 512 tokens: the
    tcgen05 GEMM and attention kernels recomputing at full width."""
    cfg = syn.CONFIGS["block6b"].with_(n_blocks=2)
    compare(cfg, run(F, cfg, 0, False), run(F, cfg, 1, False), 12)
