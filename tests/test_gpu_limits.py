"""Limits of one server call on the GPU: the largest number of segments a call packs
(1024), one past it, and one long segment, each against the fp64 oracle (GPU only)."""
import numpy as np
import pytest
import torch

import synthetic as syn
from oracle import flglm_oracle as O
from tests._gpu import dev_bf16_from_bits, f64, flglm, need_gpu, rel_inf
from tests.test_gpu_server import GRAD_TOL, OUT_TOL

pytestmark = pytest.mark.gpu

MAX_SEGS = 1024  # segments (client rows) one call packs


@pytest.fixture(scope="module")
def F():
    need_gpu()
    return flglm()


def parity(F, cfg, check_wgrad=True):
    params = syn.init_params(cfg)
    srv = F.Server(F.make_cfg(cfg, cfg.tokens, max(cfg.seq_lens)), cfg.seed)
    states, grads = syn.client_states(cfg), syn.client_grads(cfg)
    st = [dev_bf16_from_bits(s) for s in states]
    outs = [torch.empty_like(s) for s in st]
    srv.forward(st, cfg.seq_lens, outs)
    gi = [torch.empty_like(s) for s in st]
    srv.backward([dev_bf16_from_bits(g) for g in grads], gi)
    srv.sync()
    ref = O.OracleServer(cfg, params)
    ro = ref.forward([syn.bf16_bits_to_f64(s) for s in states])
    rg = ref.backward([syn.bf16_bits_to_f64(g) for g in grads])
    # all clients together: one norm over the packed batch
    got_o = np.concatenate([f64(o).reshape(-1, cfg.hidden) for o in outs])
    got_g = np.concatenate([f64(g).reshape(-1, cfg.hidden) for g in gi])
    want_o = np.concatenate([o.reshape(-1, cfg.hidden) for o in ro])
    want_g = np.concatenate([g.reshape(-1, cfg.hidden) for g in rg])
    assert rel_inf(got_o, want_o) < OUT_TOL
    assert rel_inf(got_g, want_g) < GRAD_TOL
    # per client as well (the smallest segments included)
    for k in range(cfg.K):
        assert rel_inf(f64(outs[k]), ro[k]) < OUT_TOL, k
    if check_wgrad:
        for t in range(12):
            assert rel_inf(srv.get_grad(0, t), ref.grads[0][t].reshape(-1)) < GRAD_TOL, t
    srv.close()


def test_max_segments_parity(F):
    """1024 clients of 1 to 8 tokens in one call: the packing, tile list and metadata at
    their segment limit."""
    rng = np.random.default_rng(11)
    lens = tuple(int(x) for x in rng.integers(1, 9, size=MAX_SEGS))
    cfg = syn.CONFIGS["tiny"].with_(n_blocks=1, client_batch=1, seq_lens=lens)
    parity(F, cfg)


def test_one_past_the_segment_limit(F):
    cfg = syn.CONFIGS["tiny"].with_(n_blocks=1, client_batch=1, seq_lens=(1,) * (MAX_SEGS + 1))
    srv = F.Server(F.make_cfg(cfg, cfg.tokens, 8), cfg.seed)
    st = [torch.zeros((1, 1, cfg.hidden), dtype=torch.bfloat16, device="cuda") for _ in range(MAX_SEGS + 1)]
    with pytest.raises(F.FlError) as ei:
        srv.forward(st, cfg.seq_lens, st)
    assert ei.value.code == -2          # FL_ERR_CAPACITY
    # two rows per client: 513 clients are 1026 segments
    cfg2 = cfg.with_(client_batch=2, seq_lens=(1,) * 513)
    srv2 = F.Server(F.make_cfg(cfg2, cfg2.tokens, 8), cfg.seed)
    st2 = [torch.zeros((2, 1, cfg.hidden), dtype=torch.bfloat16, device="cuda") for _ in range(513)]
    with pytest.raises(F.FlError) as ei:
        srv2.forward(st2, cfg2.seq_lens, st2)
    assert ei.value.code == -2
    # the handles stay usable: a call within the limits goes through
    srv.forward(st[:3], (1, 1, 1), st[:3])
    srv.backward(st[:3], st[:3])
    srv.sync()
    srv.close()
    srv2.close()


def test_long_segment_parity(F):
    """One 2048-token segment (32 query tiles, the longest causal rows) next to a 1-token
    one."""
    cfg = syn.CONFIGS["tiny"].with_(n_blocks=1, client_batch=1, seq_lens=(2048, 1))
    parity(F, cfg)
