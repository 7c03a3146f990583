"""P-tuning v2 on the server (App. A; the paper's own training setting, §4.1.4): learnable
prefix keys/values per block, with the block weights trained as well or frozen (GPU only)."""
import numpy as np
import pytest
import torch

import synthetic as syn
from oracle import flglm_oracle as O
from tests._gpu import dev_bf16_from_bits, f64, flglm, need_gpu, rel_inf
from tests.test_gpu_server import GRAD_TOL, OUT_TOL, check_updated_weights

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def F():
    need_gpu()
    return flglm()


def test_prefix_init_matches_generator(F):
    cfg = syn.CONFIGS["tiny"].with_(prefix_len=16)
    srv = F.Server(F.make_cfg(cfg, cfg.tokens, fused_step_min_tokens=1), cfg.seed)
    want = syn.init_prefix(cfg, 0)
    for j, t in enumerate((F.FL_T_PREFIX_K, F.FL_T_PREFIX_V)):
        got = srv.get_param(0, t)
        ulps = np.abs(got.view(np.int32).astype(np.int64) - want[j].reshape(-1).view(np.int32).astype(np.int64))
        assert ulps.max() <= 1
    srv.close()


@pytest.mark.parametrize("freeze", [0, 1], ids=["full", "frozen_base"])
@pytest.mark.parametrize("fused", [False, True], ids=["step", "backward_step"])
def test_ptuning_parity(F, freeze, fused):
    cfg = syn.CONFIGS["tiny"].with_(n_blocks=2, client_batch=1, seq_lens=(64, 17, 90), prefix_len=20,
                                    freeze_base=freeze, lr=1e-3)
    params = syn.init_params(cfg)
    prefixes = [syn.init_prefix(cfg, b) for b in range(cfg.n_blocks)]
    srv = F.Server(F.make_cfg(cfg, cfg.tokens, fused_step_min_tokens=1), cfg.seed)
    for b in range(cfg.n_blocks):
        for t in range(12):
            srv.set_param(b, t, params[b][t])
        srv.set_param(b, F.FL_T_PREFIX_K, prefixes[b][0])
        srv.set_param(b, F.FL_T_PREFIX_V, prefixes[b][1])
    states, grads = syn.client_states(cfg), syn.client_grads(cfg)
    st = [dev_bf16_from_bits(s) for s in states]
    outs = [torch.empty_like(s) for s in st]
    gi = [torch.empty_like(s) for s in st]
    srv.forward(st, cfg.seq_lens, outs)
    go = [dev_bf16_from_bits(g) for g in grads]
    ref = O.OracleServer(cfg, params, prefixes)
    ro = ref.forward([syn.bf16_bits_to_f64(s) for s in states])
    rg = ref.backward([syn.bf16_bits_to_f64(g) for g in grads])
    gref = [[g.reshape(-1).copy() for g in blk] for blk in ref.grads]
    if fused:
        srv.backward_step(go, gi, cfg.lr)
    else:
        srv.backward(go, gi)
        srv.sync()
        for b in range(cfg.n_blocks):   # prefix gradients (and block gradients when trained)
            for t in (range(14) if not freeze else (12, 13)):
                assert rel_inf(srv.get_grad(b, t), gref[b][t]) < GRAD_TOL, (b, t)
        srv.step(cfg.lr)
    srv.sync()
    for k in range(cfg.K):
        assert rel_inf(f64(outs[k]), ro[k]) < OUT_TOL
        assert rel_inf(f64(gi[k]), rg[k]) < GRAD_TOL
    ref.step(cfg.lr)
    for b in range(cfg.n_blocks):
        for t in range(14):
            w0 = (params[b][t] if t < 12 else prefixes[b][t - 12]).reshape(-1)
            w = srv.get_param(b, t)
            if freeze and t < 12:
                np.testing.assert_array_equal(w, w0)   # the frozen base does not move
            else:
                check_updated_weights(w, ref.params[b][t].reshape(-1), w0, gref[b][t], cfg.lr, (b, t))
    srv.close()
