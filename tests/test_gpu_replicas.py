"""Server-hierarchical replicas held in one handle (cfg.n_replicas, §3.3): a call's clients
split in order into equal-token groups, group r trained by replica r, the block GEMMs of all
replicas batched into one launch.  Checked against the same replicas run as separate
handles (one per group) and against the fp64 oracle running the §3.3 schedule.  GPU only."""
import numpy as np
import pytest
import torch

import synthetic as syn
from oracle import flglm_oracle as O
from tests._gpu import dev_bf16_from_bits, f64, flglm, need_gpu, rel_inf

pytestmark = pytest.mark.gpu

MATRICES = (syn.T_WQKV, syn.T_WD, syn.T_W1, syn.T_W2)


@pytest.fixture(scope="module")
def F():
    need_gpu()
    return flglm()


def _bits_equal(a, b):
    return torch.equal(a.view(torch.int16), b.view(torch.int16))


# (name, replicas, per-client sequence lengths, rows per client, GLM segments, fused step, recompute)
CASES = [
    ("R2_ragged", 2, (64, 40, 50, 54), 2, 0, 0, 0),
    ("R2_glm_fused", 2, (64, 40, 50, 54), 1, 1, 1, 0),
    ("R2_recompute", 2, (33, 31, 60, 4), 2, 0, 0, 1),
    ("R3", 3, (72, 72, 72), 2, 0, 0, 0),
    ("R4_fused", 4, (40, 24, 30, 34, 10, 54, 63, 1), 1, 0, 1, 0),
]


def _setup(F, R, seq_lens, b, glm, fused, recompute):
    cfg = syn.CONFIGS["tiny"].with_(n_blocks=2, client_batch=b, seq_lens=seq_lens, glm=glm)
    K = len(seq_lens)
    kr = K // R
    groups = [cfg.with_(seq_lens=seq_lens[r * kr:(r + 1) * kr]) for r in range(R)]
    Lmax = max(seq_lens)
    bat = F.Server(F.make_cfg(cfg, cfg.tokens, Lmax, recompute, fused, n_replicas=R), cfg.seed)
    sep = [F.Server(F.make_cfg(g, g.tokens, Lmax, recompute, fused), cfg.seed) for g in groups]
    ctx = syn.glm_structure(cfg) if glm else None
    return cfg, groups, kr, bat, sep, ctx


def _run(srv, st, lens, go, lr, ctx=None):
    """One training step (forward, backward + AdamW) of srv on clients st; returns the
    outputs and the input gradients."""
    outs = [torch.empty_like(s) for s in st]
    gin = [torch.empty_like(s) for s in st]
    if ctx is None:
        srv.forward(st, lens, outs)
    else:
        srv.forward(st, lens, outs, context_lens=ctx[0], mask_pos=ctx[1])
    srv.backward_step(go, gin, lr)
    srv.sync()
    return outs, gin


def _step_all(bat, sep, st, go, cfg, groups, kr, ctx, lr):
    b = cfg.client_batch
    ob, gb = _run(bat, st, cfg.seq_lens, go, lr, ctx)
    os_, gs = [], []
    for r, (srv, g) in enumerate(zip(sep, groups)):
        c_r = None
        if ctx is not None:
            lo, hi = r * kr * b, (r + 1) * kr * b  # segments of group r
            c_r = (ctx[0][lo:hi], ctx[1][lo:hi])
        o, gi = _run(srv, st[r * kr:(r + 1) * kr], g.seq_lens, go[r * kr:(r + 1) * kr], lr, c_r)
        os_ += o
        gs += gi
    return ob, gb, os_, gs


@pytest.mark.parametrize("case", CASES, ids=[c[0] for c in CASES])
def test_replicas_match_separate_handles(F, case):
    """First step: outputs, input gradients and updated weight matrices bit-identical to
    separate handles (batched GEMM problems are computed exactly as single ones); the bias
    and LayerNorm vectors within rounding of their atomically summed gradients (AdamW's
    first step moves each element by about lr * sign(g)).  After averaging both ways and a
    second step, the outputs agree to rounding."""
    _, R, seq_lens, b, glm, fused, recompute = case
    cfg, groups, kr, bat, sep, ctx = _setup(F, R, seq_lens, b, glm, fused, recompute)
    lr = 1e-4
    st = [dev_bf16_from_bits(s) for s in syn.client_states(cfg)]
    go = [dev_bf16_from_bits(g) for g in syn.client_grads(cfg)]
    ob, gb, os_, gs = _step_all(bat, sep, st, go, cfg, groups, kr, ctx, lr)
    for k in range(cfg.K):
        assert _bits_equal(ob[k], os_[k]), k
        assert _bits_equal(gb[k], gs[k]), k
    for r in range(R):
        for blk in range(cfg.n_blocks):
            for t in range(12):
                w_b = bat.get_replica_param(r, blk, t)
                w_s = sep[r].get_param(blk, t)
                if t in MATRICES:
                    np.testing.assert_array_equal(w_b, w_s, err_msg=f"replica {r} block {blk} tensor {t}")
                else:
                    d = np.abs(w_b.astype(np.float64) - w_s)
                    assert d.max() <= 2.05 * lr and d.mean() < 0.1 * lr, (r, blk, t, d.max() / lr, d.mean() / lr)
    # replicas differ after training on different clients
    assert not np.array_equal(bat.get_replica_param(0, 0, syn.T_W1), bat.get_replica_param(R - 1, 0, syn.T_W1))
    # period-end average: every replica holds the fp32 mean summed in replica order
    before = [[bat.get_replica_param(r, blk, t) for blk in range(cfg.n_blocks) for t in range(12)] for r in range(R)]
    bat.average_replicas()
    F.fl_server_average(sep)
    inv = np.float32(1.0) / np.float32(R)
    i = 0
    for blk in range(cfg.n_blocks):
        for t in range(12):
            s = before[0][i].copy()
            for r in range(1, R):
                s = s + before[r][i]
            want = s * inv
            for r in range(R):
                np.testing.assert_array_equal(bat.get_replica_param(r, blk, t), want)
            if t in MATRICES:
                np.testing.assert_array_equal(want, sep[0].get_param(blk, t))
            i += 1
    # a second period starts from the averaged weights
    ob, gb, os_, gs = _step_all(bat, sep, st, go, cfg, groups, kr, ctx, lr)
    for k in range(cfg.K):
        assert rel_inf(f64(ob[k]), f64(os_[k])) < 1e-3, k
        assert rel_inf(f64(gb[k]), f64(gs[k])) < 1e-2, k
    bat.close()
    for s in sep:
        s.close()


def test_replica_errors(F):
    cfg = syn.CONFIGS["tiny"].with_(n_blocks=1, client_batch=1, seq_lens=(64, 40, 50, 54))
    srv = F.Server(F.make_cfg(cfg, cfg.tokens, n_replicas=2), cfg.seed)
    st = [dev_bf16_from_bits(s) for s in syn.client_states(cfg)]
    outs = [torch.empty_like(s) for s in st]
    with pytest.raises(F.FlError, match="multiple of n_replicas"):
        srv.forward(st[:3], cfg.seq_lens[:3], outs[:3])
    with pytest.raises(F.FlError, match="tokens"):  # groups of 104 and 104 - 10 tokens
        srv.forward(st, (64, 40, 50, 44), outs)
    with pytest.raises(F.FlError):
        srv.get_replica_param(2, 0, syn.T_WQKV)
    with pytest.raises(F.FlError):
        srv.get_replica_param(-1, 0, syn.T_WQKV)
    # nothing is pending after the refused calls: a valid call runs
    srv.forward(st, cfg.seq_lens, outs)
    srv.backward([torch.zeros_like(s) for s in st], [torch.empty_like(s) for s in st])
    srv.sync()
    srv.close()
    with pytest.raises(F.FlError):  # more replicas than one batched GEMM launch holds
        F.Server(F.make_cfg(cfg, cfg.tokens, n_replicas=F.FL_GEMM_MAX_BATCH + 1), cfg.seed)
    with pytest.raises(F.FlError, match="prefix"):
        F.Server(F.make_cfg(cfg.with_(prefix_len=8), cfg.tokens, n_replicas=2), cfg.seed)
    ccfg = F.make_client_cfg(cfg, cfg.tokens)
    ccfg.block.n_replicas = 2
    with pytest.raises(F.FlError):
        F.Client(ccfg, cfg.seed)


def test_batched_replicas_period_matches_oracle(F):
    """Two replicas in one handle, each trained two steps on its own client, then averaged;
    against the oracle run of the same schedule (as for separate handles)."""
    from paper_2406_14898_gb300.hierarchical import BatchedReplicas
    cfg = syn.CONFIGS["tiny"].with_(n_blocks=2, client_batch=1, seq_lens=(64, 64))
    lr, steps = 1e-3, 2
    states = syn.client_states(cfg)
    grads = syn.client_grads(cfg)
    one = [cfg.with_(seq_lens=(L,)) for L in cfg.seq_lens]
    hs = BatchedReplicas(F.make_cfg(cfg, cfg.tokens, max(cfg.seq_lens)), cfg.seed, 2)
    st = [dev_bf16_from_bits(s) for s in states]
    go = [dev_bf16_from_bits(g) for g in grads]
    outs = [torch.empty_like(s) for s in st]
    gin = [torch.empty_like(s) for s in st]
    for _ in range(steps):
        hs.step(st, cfg.seq_lens, outs, go, gin, lr)
    hs.average()
    hs.sync()
    params = syn.init_params(cfg)
    reps = [O.OracleServer(one[k], params) for k in range(cfg.K)]
    for _ in range(steps):
        for k, r in enumerate(reps):
            r.forward([syn.bf16_bits_to_f64(states[k])])
            r.backward([syn.bf16_bits_to_f64(grads[k])])
            r.step(lr)
    O.average_params(reps)
    # the key bias on the un-rotated half of each head has a zero gradient in exact
    # arithmetic (it shifts a whole score row): its update sign is rounding noise
    H, hd = cfg.hidden, cfg.head_dim
    keep_bqkv = np.ones(3 * H, bool)
    for h in range(cfg.n_heads):
        keep_bqkv[H + h * hd + hd // 2:H + (h + 1) * hd] = False
    for b in range(cfg.n_blocks):
        for t in range(12):
            w = hs.get_param(0, b, t).astype(np.float64)
            np.testing.assert_array_equal(w, hs.get_param(1, b, t))
            w0 = params[b][t].reshape(-1).astype(np.float64)
            dref = reps[0].params[b][t].reshape(-1) - w0
            err = np.abs((w - w0) - dref)
            if t == syn.T_BQKV:
                err = err[keep_bqkv]
            assert np.mean(err) < 0.1 * lr, (b, t, np.mean(err) / lr)
    # the averaged replicas' outputs for both clients (one call, one client per replica)
    hs.server.forward(st, cfg.seq_lens, outs)
    hs.server.backward(go, gin)
    hs.sync()
    for k in range(cfg.K):
        ref_out = reps[k].forward([syn.bf16_bits_to_f64(states[k])])
        assert rel_inf(f64(outs[k]), ref_out[0]) < 2e-2
    hs.close()
