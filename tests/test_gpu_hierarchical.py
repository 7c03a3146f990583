"""Server-hierarchical strategy (§3.3) on the GPU: one replica per client, parameters
averaged at the end of the period, against the fp64 oracle doing the same (GPU only)."""
import numpy as np
import pytest
import torch

import synthetic as syn
from oracle import flglm_oracle as O
from tests._gpu import dev_bf16_from_bits, f64, flglm, need_gpu, rel_inf

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def F():
    need_gpu()
    return flglm()


def test_average_is_the_mean(F):
    """fl_server_average writes the fp32 mean (summed in replica order) into every replica."""
    cfg = syn.CONFIGS["tiny"].with_(n_blocks=2)
    reps = [F.Server(F.make_cfg(cfg, cfg.tokens), seed) for seed in (1, 2, 3)]
    before = [[r.get_param(b, t) for t in range(12) for b in range(2)] for r in reps]
    F.fl_server_average(reps)
    after = [[r.get_param(b, t) for t in range(12) for b in range(2)] for r in reps]
    inv = np.float32(1.0) / np.float32(3.0)
    for i in range(len(before[0])):
        want = ((before[0][i] + before[1][i]) + before[2][i]) * inv
        for r in range(3):
            np.testing.assert_array_equal(after[r][i], want)
    with pytest.raises(F.FlError):
        F.fl_server_average([reps[0], reps[0]])
    for r in reps:
        r.close()


def test_average_finish_matches_average(F):
    """The cross-process form: a replica whose arena holds the sum of two replicas' weights
    (what an all-reduce leaves), finished by fl_server_average_finish(2), has the bits
    fl_server_average gives, fp32 master and bf16 working copy (checked through a forward)."""
    from paper_2406_14898_gb300.hierarchical import arena_tensor
    cfg = syn.CONFIGS["tiny"].with_(n_blocks=2)
    a, b, c = (F.Server(F.make_cfg(cfg, cfg.tokens), seed) for seed in (4, 5, 6))
    wa, wb, wc = arena_tensor(a), arena_tensor(b), arena_tensor(c)
    torch.cuda.synchronize()
    wc.copy_(wa + wb)
    torch.cuda.synchronize()
    c.average_finish(2)
    F.fl_server_average([a, b])
    c.sync()
    torch.testing.assert_close(wc, wa, rtol=0, atol=0)
    st = [dev_bf16_from_bits(s) for s in syn.client_states(cfg)]
    outs = {}
    for name, srv in (("a", a), ("c", c)):
        o = [torch.empty_like(x) for x in st]
        srv.forward(st, cfg.seq_lens, o)
        srv.backward([torch.zeros_like(x) for x in st], [torch.empty_like(x) for x in st])
        srv.sync()
        outs[name] = o
    for x, y in zip(outs["a"], outs["c"]):
        assert torch.equal(x.view(torch.int16), y.view(torch.int16))
    with pytest.raises(F.FlError):
        c.average_finish(0)
    for s_ in (a, b, c):
        s_.close()


def test_hierarchical_period_matches_oracle(F):
    """Two replicas, each trained two steps on its own client, then averaged; the averaged
    server's outputs for both clients match the oracle run of the same schedule."""
    from paper_2406_14898_gb300.hierarchical import HierarchicalServers
    cfg = syn.CONFIGS["tiny"].with_(n_blocks=2, client_batch=1, seq_lens=(64, 40))
    lr, steps = 1e-3, 2
    states = syn.client_states(cfg)
    grads = syn.client_grads(cfg)
    one = [cfg.with_(seq_lens=(L,)) for L in cfg.seq_lens]
    hs = HierarchicalServers(F.make_cfg(one[0], max(cfg.seq_lens)), cfg.seed, cfg.K)
    st = [dev_bf16_from_bits(s) for s in states]
    go = [dev_bf16_from_bits(g) for g in grads]
    outs = [torch.empty_like(s) for s in st]
    gin = [torch.empty_like(s) for s in st]
    for _ in range(steps):
        hs.step(st, cfg.seq_lens, outs, go, gin, lr)
    hs.average()
    hs.sync()
    # oracle: the same schedule
    params = syn.init_params(cfg)
    reps = [O.OracleServer(one[k], params) for k in range(cfg.K)]
    for _ in range(steps):
        for k, r in enumerate(reps):
            r.forward([syn.bf16_bits_to_f64(states[k])])
            r.backward([syn.bf16_bits_to_f64(grads[k])])
            r.step(lr)
    O.average_params(reps)
    # parameters: mean update agrees (Adam's early steps are about lr * sign(g)).  The key
    # bias on the un-rotated half of each head only shifts a whole score row, which softmax
    # ignores: its gradient is zero in exact arithmetic and its update sign is rounding
    # noise on both sides, so those elements are left out.
    H, hd = cfg.hidden, cfg.head_dim
    keep_bqkv = np.ones(3 * H, bool)
    for h in range(cfg.n_heads):
        keep_bqkv[H + h * hd + hd // 2:H + (h + 1) * hd] = False
    for b in range(cfg.n_blocks):
        for t in range(12):
            w = hs.replicas[0].get_param(b, t).astype(np.float64)
            np.testing.assert_array_equal(w, hs.replicas[1].get_param(b, t))
            w0 = params[b][t].reshape(-1).astype(np.float64)
            dref = reps[0].params[b][t].reshape(-1) - w0
            err = np.abs((w - w0) - dref)
            if t == syn.T_BQKV:
                err = err[keep_bqkv]
            assert np.mean(err) < 0.1 * lr, (b, t, np.mean(err) / lr)
    # outputs of the averaged replicas for each client
    for k in range(cfg.K):
        srv = hs.replicas[k]
        srv.forward([st[k]], [cfg.seq_lens[k]], [outs[k]])
        srv.backward([go[k]], [gin[k]])
        srv.sync()
        ref_out = reps[k].forward([syn.bf16_bits_to_f64(states[k])])
        assert rel_inf(f64(outs[k]), ref_out[0]) < 2e-2
    hs.close()
