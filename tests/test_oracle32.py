"""The fp32 C++ oracle (oracle/flglm_oracle32.cpp) against what fixes it independently of
itself: the pinned fp64 oracle (an independent implementation of the same definitions),
the zero-weight closed form, the batching invariant of §3.3, causality and segment
isolation, and the first-step closed form of AdamW (CPU only)."""
import numpy as np
import pytest

import synthetic as syn
from oracle import flglm_oracle as O
from oracle import oracle32 as O32


def _rel(a, b):
    a = np.asarray(a, np.float64)
    b = np.asarray(b, np.float64)
    return float(np.abs(a - b).max() / max(np.abs(b).max(), 1e-30))


def _inputs(cfg):
    states = syn.client_states(cfg)
    grads = syn.client_grads(cfg)
    x = np.concatenate([syn.bf16_bits_to_f64(s).reshape(-1, cfg.hidden) for s in states])
    dy = np.concatenate([syn.bf16_bits_to_f64(g).reshape(-1, cfg.hidden) for g in grads])
    cu = np.concatenate([[0], np.cumsum([L for L in cfg.seq_lens for _ in range(cfg.client_batch)])])
    return states, grads, x, dy, cu


def _run32(cfg, params, cu, x, dy):
    g = [[np.zeros(p.shape, np.float32) for p in blk] for blk in params]
    y, dx = O32.server_fwd_bwd(cfg, params, g, cu, x, dy)
    return y, dx, g


@pytest.mark.parametrize("rfl", [1, 0], ids=["glm_block", "pre_ln"])
def test_matches_fp64_oracle(rfl):
    """Two blocks over ragged segments (64, 37 and a 1-token one), both residual readings:
    outputs, input gradients and every weight gradient within fp32 rounding of the fp64
    oracle."""
    cfg = syn.CONFIGS["tiny"].with_(n_blocks=2, client_batch=1, seq_lens=(64, 37, 1), residual_from_ln=rfl,
                                    residual_alpha=2.0 if rfl else 1.0)
    params = syn.init_params(cfg)
    states, grads, x, dy, cu = _inputs(cfg)
    ref = O.OracleServer(cfg, params)
    ro = np.concatenate([r.reshape(-1, cfg.hidden) for r in ref.forward([syn.bf16_bits_to_f64(s) for s in states])])
    rg = np.concatenate([r.reshape(-1, cfg.hidden) for r in ref.backward([syn.bf16_bits_to_f64(g) for g in grads])])
    y, dx, g = _run32(cfg, params, cu, x, dy)
    assert _rel(y, ro) < 1e-5
    assert _rel(dx, rg) < 1e-5
    for b in range(cfg.n_blocks):
        for t in range(12):
            assert _rel(g[b][t], ref.grads[b][t]) < 1e-5, (b, syn.TENSOR_NAMES[t])


def test_matches_fp64_oracle_head_dim_128():
    """One block with 128-dim heads (the ChatGLM-6B head size) at a small hidden size."""
    cfg = syn.CONFIGS["tiny"].with_(hidden=256, n_heads=2, head_dim=128, ffn_hidden=1024, client_batch=2,
                                    seq_lens=(40, 17))
    params = syn.init_params(cfg)
    states, grads, x, dy, cu = _inputs(cfg)
    ref = O.OracleServer(cfg, params)
    ro = np.concatenate([r.reshape(-1, cfg.hidden) for r in ref.forward([syn.bf16_bits_to_f64(s) for s in states])])
    rg = np.concatenate([r.reshape(-1, cfg.hidden) for r in ref.backward([syn.bf16_bits_to_f64(g) for g in grads])])
    y, dx, g = _run32(cfg, params, cu, x, dy)
    assert _rel(y, ro) < 1e-5 and _rel(dx, rg) < 1e-5
    assert max(_rel(g[0][t], ref.grads[0][t]) for t in range(12)) < 1e-5


def test_zero_weights_closed_form():
    """Wd = W1 = W2 = 0 and zero biases, gamma = 1, beta = 0: y = alpha LN(alpha LN(x))."""
    cfg = syn.CONFIGS["tiny"].with_(client_batch=1, seq_lens=(9, 4))
    params = syn.init_params(cfg)
    for t in (syn.T_WD, syn.T_BD, syn.T_W1, syn.T_B1, syn.T_W2, syn.T_B2):
        params[0][t][:] = 0
    _, _, x, dy, cu = _inputs(cfg)
    y, _, _ = _run32(cfg, params, cu, x, dy)

    def ln(v):
        v = v - v.mean(axis=1, keepdims=True)
        return v / np.sqrt((v * v).mean(axis=1, keepdims=True) + cfg.ln_eps)
    a = cfg.residual_alpha
    assert _rel(y, a * ln(a * ln(x))) < 1e-5


def test_batching_invariant_and_isolation():
    """Packed segments equal each segment run alone bit for bit (row-independent loops,
    sums in a fixed order); weight gradients equal the sum of the per-segment runs within
    fp32 rounding; changing a later token or another segment leaves an output bit-identical."""
    cfg = syn.CONFIGS["tiny"].with_(client_batch=1, seq_lens=(20, 11, 5))
    params = syn.init_params(cfg)
    _, _, x, dy, cu = _inputs(cfg)
    y, dx, g = _run32(cfg, params, cu, x, dy)
    gsum = [np.zeros(p.shape, np.float64) for p in params[0]]
    for s in range(3):
        a, b = cu[s], cu[s + 1]
        ys, dxs, gs = _run32(cfg, params, [0, b - a], x[a:b], dy[a:b])
        np.testing.assert_array_equal(ys, y[a:b])
        np.testing.assert_array_equal(dxs, dx[a:b])
        for t in range(12):
            gsum[t] += gs[0][t]
    for t in range(12):
        assert _rel(g[0][t], gsum[t]) < 1e-5
    x2 = x.copy()
    rng = np.random.default_rng(5)   # not a constant shift, which LayerNorm removes exactly
    x2[cu[1] - 1] += rng.standard_normal(cfg.hidden)          # last token of segment 0
    x2[cu[2]:cu[3]] += rng.standard_normal((cu[3] - cu[2], cfg.hidden))  # all of segment 2
    y2, _, _ = _run32(cfg, params, cu, x2, dy)
    np.testing.assert_array_equal(y2[:cu[1] - 1], y[:cu[1] - 1])
    np.testing.assert_array_equal(y2[cu[1]:cu[2]], y[cu[1]:cu[2]])
    assert not np.array_equal(y2[cu[1] - 1], y[cu[1] - 1])


def test_adamw_first_step_and_fp64():
    """First step (zero moments, no decay): w1 = w0 - lr g / (|g| + eps) within fp32
    rounding; five steps against the fp64 AdamW."""
    rng = np.random.default_rng(3)
    n = 1000
    w0 = rng.standard_normal(n).astype(np.float32)
    g = (1e-3 * rng.standard_normal(n)).astype(np.float32)
    w, m, v = w0.copy(), np.zeros(n, np.float32), np.zeros(n, np.float32)
    O32.adamw(w, g, m, v, 1, 1e-2, 0.9, 0.999, 1e-8, 0.0)
    want = w0.astype(np.float64) - 1e-2 * g / (np.abs(g.astype(np.float64)) + 1e-8)
    assert np.abs(w - want).max() < 1e-6
    w64, m64, v64 = w0.astype(np.float64), np.zeros(n), np.zeros(n)
    w, m, v = w0.copy(), np.zeros(n, np.float32), np.zeros(n, np.float32)
    for t in range(1, 6):
        gt = (1e-3 * rng.standard_normal(n)).astype(np.float32)
        O32.adamw(w, gt, m, v, t, 1e-3, 0.9, 0.999, 1e-8, 0.01)
        w64, m64, v64 = O.adamw_update(w64, gt.astype(np.float64), m64, v64, t, 1e-3, 0.9, 0.999, 1e-8, 0.01)
    assert np.abs(w - w64).max() < 1e-6
    assert _rel(m, m64) < 1e-5


def test_bad_arguments():
    cfg = syn.CONFIGS["tiny"].with_(client_batch=1, seq_lens=(4,))
    params = syn.init_params(cfg)
    x = np.zeros((4, cfg.hidden), np.float32)
    with pytest.raises(ValueError):
        _run32(cfg, params, [0, 3, 2, 4], x, x)
    with pytest.raises(ValueError):
        O32.adamw(np.zeros(2, np.float32), np.zeros(2, np.float32), np.zeros(2, np.float32),
                  np.zeros(2, np.float32), 0, 1e-3, 0.9, 0.999, 1e-8, 0.0)


def _fp64(cfg, params, states, grads, prefixes=None, ctx=None, mp=None):
    ref = O.OracleServer(cfg, params, prefixes)
    ro = ref.forward([syn.bf16_bits_to_f64(s) for s in states], ctx, mp)
    rg = ref.backward([syn.bf16_bits_to_f64(g) for g in grads])
    cat = lambda rs: np.concatenate([r.reshape(-1, cfg.hidden) for r in rs])  # noqa: E731
    return cat(ro), cat(rg), ref.grads


@pytest.mark.parametrize("rfl,Lp,glm", [(1, 0, True), (0, 0, True), (1, 3, False), (1, 3, True), (0, 2, True)],
                         ids=["glm", "glm_pre_ln", "prefix", "prefix_glm", "prefix_glm_pre_ln"])
def test_glm_and_prefix_match_fp64_oracle(rfl, Lp, glm):
    """§4.1.1 GLM segments (bidirectional context, causal span, 2D positions) and App. A
    P-tuning prefixes, two blocks over ragged segments: outputs, input gradients, the 12
    weight gradients and the prefix key / value gradients within fp32 rounding of the fp64
    oracle."""
    cfg = syn.CONFIGS["tiny"].with_(n_blocks=2, client_batch=1, seq_lens=(13, 9, 5, 1), residual_from_ln=rfl,
                                    residual_alpha=2.0 if rfl else 1.0, prefix_len=Lp)
    params = syn.init_params(cfg)
    rng = np.random.default_rng(40 + Lp)
    prefixes = [[(0.5 * rng.standard_normal((Lp, cfg.hidden))) for _ in range(2)] for _ in range(cfg.n_blocks)] \
        if Lp else None
    ctx, mp = ([6, 0, 5, 1], [2, 0, 4, 0]) if glm else (None, None)
    states, grads, x, dy, cu = _inputs(cfg)
    ro, rg, rgrads = _fp64(cfg, params, states, grads, prefixes, ctx, mp)
    g = [[np.zeros(p.shape, np.float32) for p in blk] for blk in params]
    pg = [[np.zeros((Lp, cfg.hidden), np.float32) for _ in range(2)] for _ in range(cfg.n_blocks)] if Lp else None
    y, dx = O32.server_fwd_bwd(cfg, params, g, cu, x, dy, ctx, mp, prefixes, pg)
    assert _rel(y, ro) < 1e-5
    assert _rel(dx, rg) < 1e-5
    for b in range(cfg.n_blocks):
        for t in range(12):
            assert _rel(g[b][t], rgrads[b][t]) < 1e-5, (b, syn.TENSOR_NAMES[t])
        for j in range(2 if Lp else 0):
            assert _rel(pg[b][j], rgrads[b][12 + j]) < 1e-5, (b, "prefix", j)


def test_glm_and_prefix_batching_invariant():
    """§3.3 stacking with GLM segments and a shared prefix: packed outputs and input
    gradients equal each segment run alone bit for bit; weight and prefix gradients are the
    sum of the per-segment runs within fp32 rounding."""
    cfg = syn.CONFIGS["tiny"].with_(n_blocks=2, client_batch=1, seq_lens=(11, 6, 3), prefix_len=2)
    params = syn.init_params(cfg)
    rng = np.random.default_rng(44)
    prefixes = [[(0.5 * rng.standard_normal((2, cfg.hidden))) for _ in range(2)] for _ in range(cfg.n_blocks)]
    ctx, mp = [4, 0, 3], [1, 0, 2]
    states, grads, x, dy, cu = _inputs(cfg)
    g = [[np.zeros(p.shape, np.float32) for p in blk] for blk in params]
    pg = [[np.zeros((2, cfg.hidden), np.float32) for _ in range(2)] for _ in range(cfg.n_blocks)]
    y, dx = O32.server_fwd_bwd(cfg, params, g, cu, x, dy, ctx, mp, prefixes, pg)
    gs = [[np.zeros(p.shape, np.float64) for p in blk] for blk in params]
    pgs = [[np.zeros((2, cfg.hidden), np.float64) for _ in range(2)] for _ in range(cfg.n_blocks)]
    for s in range(len(cfg.seq_lens)):
        a, b = cu[s], cu[s + 1]
        g1 = [[np.zeros(p.shape, np.float32) for p in blk] for blk in params]
        pg1 = [[np.zeros((2, cfg.hidden), np.float32) for _ in range(2)] for _ in range(cfg.n_blocks)]
        y1, dx1 = O32.server_fwd_bwd(cfg, params, g1, [0, b - a], x[a:b], dy[a:b], [ctx[s]], [mp[s]], prefixes, pg1)
        np.testing.assert_array_equal(y1, y[a:b])
        np.testing.assert_array_equal(dx1, dx[a:b])
        for bb in range(cfg.n_blocks):
            for t in range(12):
                gs[bb][t] += g1[bb][t]
            for j in range(2):
                pgs[bb][j] += pg1[bb][j]
    for bb in range(cfg.n_blocks):
        for t in range(12):
            assert _rel(g[bb][t], gs[bb][t]) < 1e-5
        for j in range(2):
            assert _rel(pg[bb][j], pgs[bb][j]) < 1e-5


def test_glm_and_prefix_bad_arguments():
    cfg = syn.CONFIGS["tiny"].with_(n_blocks=1, client_batch=1, seq_lens=(4,))
    params = syn.init_params(cfg)
    x = np.zeros((4, cfg.hidden), np.float32)
    g = [[np.zeros(p.shape, np.float32) for p in blk] for blk in params]
    for ctx, mp in (([5], [0]), ([3], [3]), ([-1], [0])):   # context past the segment, [M] outside it, negative
        with pytest.raises(ValueError):
            O32.server_fwd_bwd(cfg, params, g, [0, 4], x, x, ctx, mp)


@pytest.mark.parametrize("Lp,glm", [(0, False), (2, True)], ids=["plain", "prefix_glm"])
def test_client_round_matches_fp64_oracle(Lp, glm):
    """§3.1 client parts in fp32 (Embedding + Block_0, Block_{N-1} + final LayerNorm + LM
    head + cross-entropy; the server's blocks left out): the loss and every client
    parameter's gradient within fp32 rounding of the fp64 oracle client, with repeated
    tokens, rows without a target, and optionally GLM segments with P-tuning prefixes."""
    cfg = syn.CONFIGS["tiny"].with_(n_blocks=1, client_batch=2, seq_lens=(9,), vocab=37, prefix_len=Lp)
    params = syn.init_client(cfg)
    rng = np.random.default_rng(50 + Lp)
    tok = rng.integers(0, cfg.vocab, size=(2, 9)).astype(np.int32)
    lab = rng.integers(0, cfg.vocab, size=(2, 9)).astype(np.int32)
    lab[0, :4] = -1
    ctx, mp = ([5, 3], [2, 0]) if glm else (None, None)
    loss32, g32 = O32.client_round(cfg, params, tok, lab, ctx, mp)
    c = O.OracleClient(cfg, params)
    h0 = c.bottom_forward(tok, ctx, mp)
    loss, gh = c.top_forward_backward(h0, lab)
    c.bottom_backward(gh)
    assert abs(loss32 - loss) <= 1e-6 * abs(loss)
    for k in O.CLIENT_PARTS:
        for i, (a, b) in enumerate(zip(g32[k], c.grads[k])):
            assert _rel(a, b) < 1e-5, (k, i)


def test_client_round_no_target_and_bad_ids():
    """No target at all: zero loss and zero gradients; a token id outside the vocabulary or a
    label >= vocab is refused."""
    cfg = syn.CONFIGS["tiny"].with_(n_blocks=1, client_batch=1, seq_lens=(4,), vocab=11)
    params = syn.init_client(cfg)
    tok = np.array([[1, 2, 3, 1]], np.int32)
    loss, g = O32.client_round(cfg, params, tok, np.full((1, 4), -1, np.int32))
    assert loss == 0.0
    assert all(not a.any() for v in g.values() for a in v)
    with pytest.raises(ValueError):
        O32.client_round(cfg, params, np.array([[1, 2, 11, 0]], np.int32), np.zeros((1, 4), np.int32))
    with pytest.raises(ValueError):
        O32.client_round(cfg, params, tok, np.array([[0, 11, 0, 0]], np.int32))
