"""Pins of the fp64 oracle to facts other than itself (CPU only).

Each pin is chosen so that a plausible slip in the oracle (a dropped term, a sign,
a wrong index or operand order) fails at least one of them:

* finite differences pin every backward formula against the forward;
* library routines that special cases reduce to (torch's LayerNorm, causal SDPA,
  tanh-GeLU and AdamW, all in float64) pin the forward primitives;
* closed forms (zero-weight block, first AdamW step, single-token attention,
  constant keys) and invariants (client-batching, causality, segment isolation,
  RoPE norm and relative-position properties, LayerNorm row statistics) pin the
  composition the paper fixes: §3.3 stacks clients without mixing them.
"""
import math
import os

import numpy as np
import pytest
import torch

import synthetic as syn
from oracle import flglm_oracle as O

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


# ----------------------------------------------------------------------------- helpers

def tiny_cfg(residual_from_ln=1, n_blocks=2, seq_lens=(3, 5), b=1, alpha=2.0):
    return syn.ServerConfig(name="fd", n_blocks=n_blocks, hidden=16, n_heads=2, head_dim=8,
                            ffn_hidden=32, residual_alpha=alpha, client_batch=b, seq_lens=tuple(seq_lens),
                            residual_from_ln=residual_from_ln)


def random_params(cfg, rng, std=0.3):
    """Large random weights and non-trivial LayerNorm affine parameters so that every
    term of the block contributes measurably to the finite differences."""
    out = []
    for _ in range(cfg.n_blocks):
        blk = []
        for t, shp in enumerate(syn.param_shapes(cfg)):
            if t in (syn.T_G1, syn.T_G2):
                blk.append(1.0 + 0.3 * rng.standard_normal(shp))
            elif t in (syn.T_BE1, syn.T_BE2):
                blk.append(0.3 * rng.standard_normal(shp))
            else:
                blk.append(std * rng.standard_normal(shp))
        out.append(blk)
    return out


def run_stack(cfg, params, X, pk):
    sh = O.BlockShape.of(cfg)
    return O.stack_fwd(params, X, pk, sh)


def loss_and_grads(cfg, params, X, pk, dY):
    sh = O.BlockShape.of(cfg)
    Y, saved = O.stack_fwd(params, X, pk, sh)
    dX, grads = O.stack_bwd(params, saved, dY, pk, sh)
    return float((Y * dY).sum()), dX, grads


# ----------------------------------------------------------------------------- generator pins

def test_splitmix64_published_vector():
    with open(os.path.join(GOLDEN, "splitmix64_seed1234567.txt")) as fh:
        vals = [int(l) for l in fh if l.strip() and not l.startswith("#")]
    got = [int(v) for v in syn.raw_u64(1234567, 0, 5)]
    assert got == vals


def test_normal_stream_statistics_and_offsets():
    key = syn.stream_key(0, syn.P_WEIGHTS, 3, 2)
    z = syn.normal_f64(key, 200001, 0.0, 1.0)
    assert abs(z.mean()) < 0.01 and abs(z.std() - 1.0) < 0.01
    # counter-based: any window equals the slice of the full stream
    for start, n in [(0, 7), (1, 6), (13, 100), (99999, 3)]:
        np.testing.assert_array_equal(syn.normal_f64(key, n, 0.0, 1.0, start), z[start:start + n])


def test_bf16_rounding_is_rne():
    x = np.array([1.0, 1.0 + 2 ** -8, 1.0 + 3 * 2 ** -8, -2.5, 1.0 + 2 ** -9, 3.0e38], np.float32)
    got = syn.bf16_bits_to_f32(syn.f32_to_bf16_bits(x))
    want = torch.tensor(x).to(torch.bfloat16).float().numpy()
    np.testing.assert_array_equal(got, want)


def test_ragged_lengths_range_and_seed():
    L = syn.ragged_lengths(7, 16)
    assert len(L) == 16 and all(64 <= l <= 1024 for l in L)
    assert syn.CONFIGS["ragged26"].seq_lens == L
    assert len(set(L)) > 8


# ----------------------------------------------------------------------------- packing

def test_pack_unpack_roundtrip_and_metadata():
    rng = np.random.default_rng(1)
    seq = (3, 1, 4)
    b = 2
    ts = [rng.standard_normal((b, L, 5)) for L in seq]
    pk = O.make_packing(seq, b)
    assert list(pk.cu_seqlens) == [0, 3, 6, 7, 8, 12, 16]
    assert list(pk.pos) == [0, 1, 2, 0, 1, 2, 0, 0, 0, 1, 2, 3, 0, 1, 2, 3]
    assert list(pk.seg_client) == [0, 0, 1, 1, 2, 2]
    X = O.pack(ts)
    np.testing.assert_array_equal(X[6], ts[1][0, 0])
    np.testing.assert_array_equal(X[12:16], ts[2][1])
    for a, c in zip(O.unpack(X, seq, b), ts):
        np.testing.assert_array_equal(a, c)


# ----------------------------------------------------------------------------- forward primitives vs library routines

def test_layer_norm_matches_torch_and_row_stats():
    rng = np.random.default_rng(2)
    x = 3.0 * rng.standard_normal((7, 33)) + 1.5
    g = rng.standard_normal(33)
    be = rng.standard_normal(33)
    y, mu, rs = O.layer_norm_fwd(x, g, be, 1e-5)
    ref = torch.nn.functional.layer_norm(torch.tensor(x), (33,), torch.tensor(g), torch.tensor(be), 1e-5).numpy()
    np.testing.assert_allclose(y, ref, rtol=0, atol=1e-12)
    # gamma = 1, beta = 0: zero row mean, variance sigma^2 / (sigma^2 + eps)
    y1, _, _ = O.layer_norm_fwd(x, np.ones(33), np.zeros(33), 1e-5)
    assert np.abs(y1.mean(axis=1)).max() < 1e-12
    var = x.var(axis=1)
    np.testing.assert_allclose(y1.var(axis=1), var / (var + 1e-5), rtol=1e-12)


def test_gelu_matches_torch_tanh_form():
    u = np.linspace(-8, 8, 1001)
    ref = torch.nn.functional.gelu(torch.tensor(u), approximate="tanh").numpy()
    np.testing.assert_allclose(O.gelu(u), ref, rtol=0, atol=1e-14)
    # derivative against torch autograd
    tu = torch.tensor(u, requires_grad=True)
    torch.nn.functional.gelu(tu, approximate="tanh").sum().backward()
    np.testing.assert_allclose(O.gelu_grad(u), tu.grad.numpy(), rtol=0, atol=1e-13)


def test_attention_matches_torch_sdpa_per_segment():
    rng = np.random.default_rng(3)
    seq = [5, 1, 9]
    cu = np.cumsum([0] + seq).astype(np.int32)
    T, nh, hd = cu[-1], 3, 8
    q, k, v = (rng.standard_normal((T, nh, hd)) for _ in range(3))
    o, lse = O.attention_fwd(q, k, v, cu)
    for s in range(len(seq)):
        a, b = cu[s], cu[s + 1]
        tq = torch.tensor(q[a:b]).transpose(0, 1)
        tk = torch.tensor(k[a:b]).transpose(0, 1)
        tv = torch.tensor(v[a:b]).transpose(0, 1)
        ref = torch.nn.functional.scaled_dot_product_attention(tq, tk, tv, is_causal=True).transpose(0, 1).numpy()
        np.testing.assert_allclose(o[a:b], ref, rtol=0, atol=1e-12)
        # LSE against torch.logsumexp of the masked, scaled scores
        S = torch.einsum("hid,hjd->hij", tq, tk) / math.sqrt(hd)
        S = S.masked_fill(~torch.ones(b - a, b - a, dtype=torch.bool).tril(), float("-inf"))
        np.testing.assert_allclose(lse[:, a:b], torch.logsumexp(S, -1).numpy(), rtol=0, atol=1e-12)


def test_attention_brute_force_global_mask():
    """The packed form equals one dense softmax over all T keys with a block-diagonal
    causal mask (brute force over the whole packed batch)."""
    rng = np.random.default_rng(4)
    seq = [4, 6, 2]
    cu = np.cumsum([0] + seq).astype(np.int32)
    T, nh, hd = cu[-1], 2, 4
    q, k, v = (rng.standard_normal((T, nh, hd)) for _ in range(3))
    o, _ = O.attention_fwd(q, k, v, cu)
    seg = np.repeat(np.arange(len(seq)), seq)
    for h in range(nh):
        for t in range(T):
            w = np.array([math.exp(float(q[t, h] @ k[u, h]) / math.sqrt(hd)) if (seg[u] == seg[t] and u <= t) else 0.0
                          for u in range(T)])
            np.testing.assert_allclose(o[t, h], (w[:, None] * v[:, h]).sum(0) / w.sum(), rtol=0, atol=1e-12)


def test_attention_special_cases():
    rng = np.random.default_rng(5)
    # L = 1: output equals v exactly
    q, k, v = (rng.standard_normal((1, 2, 8)) for _ in range(3))
    o, lse = O.attention_fwd(q, k, v, np.array([0, 1], np.int32))
    np.testing.assert_array_equal(o, v)
    # all keys equal: every row is the running mean of v
    L = 6
    q = rng.standard_normal((L, 1, 4))
    k = np.tile(rng.standard_normal((1, 1, 4)), (L, 1, 1))
    v = rng.standard_normal((L, 1, 4))
    o, _ = O.attention_fwd(q, k, v, np.array([0, L], np.int32))
    want = np.cumsum(v[:, 0], axis=0) / np.arange(1, L + 1)[:, None]
    np.testing.assert_allclose(o[:, 0], want, rtol=0, atol=1e-13)


def test_rope_properties():
    rng = np.random.default_rng(6)
    hd, rd, base = 16, 8, 10000.0
    pos = np.arange(12, dtype=np.int32)
    cos, sin = O.rope_cos_sin(pos, rd, base)
    x = rng.standard_normal((12, 2, hd))
    xr = O.rope_rotate(x, cos, sin, rd)
    # p = 0 is the identity; dims beyond the rotary dims pass through
    np.testing.assert_array_equal(xr[0], x[0])
    np.testing.assert_array_equal(xr[..., rd:], x[..., rd:])
    # norm preserved; inverse undoes the rotation
    np.testing.assert_allclose(np.linalg.norm(xr, axis=-1), np.linalg.norm(x, axis=-1), rtol=1e-13)
    np.testing.assert_allclose(O.rope_rotate(xr, cos, sin, rd, inverse=True), x, atol=1e-13)
    # complex-number form: pair (i, i + rd/2) is z = x_i + j x_{i+rd/2}, rotated by e^{j p theta_i}
    theta = base ** (-2.0 * np.arange(rd // 2) / rd)
    z = (x[..., :rd // 2] + 1j * x[..., rd // 2:rd]) * np.exp(1j * pos[:, None, None] * theta[None, None, :])
    np.testing.assert_allclose(xr[..., :rd // 2], z.real, atol=1e-13)
    np.testing.assert_allclose(xr[..., rd // 2:rd], z.imag, atol=1e-13)
    # q . k depends only on the position difference
    q = rng.standard_normal((1, 1, hd))
    kk = rng.standard_normal((1, 1, hd))
    def dot(p, pp):
        c1, s1 = O.rope_cos_sin(np.array([p]), rd, base)
        c2, s2 = O.rope_cos_sin(np.array([pp]), rd, base)
        return float((O.rope_rotate(q, c1, s1, rd) * O.rope_rotate(kk, c2, s2, rd)).sum())
    assert abs(dot(7, 3) - dot(11, 7)) < 1e-12
    assert abs(dot(5, 0) - dot(9, 4)) < 1e-12


# ----------------------------------------------------------------------------- block closed form

@pytest.mark.parametrize("rfl", [1, 0])
def test_zero_weight_block_closed_form(rfl):
    cfg = tiny_cfg(residual_from_ln=rfl, n_blocks=1, seq_lens=(4, 3))
    rng = np.random.default_rng(7)
    P = [np.zeros(s) for s in syn.param_shapes(cfg)]
    P[syn.T_G1][:] = 1.0
    P[syn.T_G2][:] = 1.0
    pk = O.make_packing(cfg.seq_lens, 1)
    x = 2.0 * rng.standard_normal((pk.T, cfg.hidden)) + 0.5
    y, _ = run_stack(cfg, [P], x, pk)
    al, eps = cfg.residual_alpha, cfg.ln_eps

    def ln(z):
        zc = z - z.mean(1, keepdims=True)
        return zc / np.sqrt((zc * zc).mean(1, keepdims=True) + eps)
    if rfl:
        want = al * ln(al * ln(x))
    else:
        want = al * al * x   # attention and FFN branches are exactly zero
    np.testing.assert_allclose(y, want, rtol=1e-12, atol=1e-12)


# ----------------------------------------------------------------------------- finite differences

@pytest.mark.parametrize("rfl", [1, 0])
def test_finite_difference_gradients(rfl):
    cfg = tiny_cfg(residual_from_ln=rfl, n_blocks=2, seq_lens=(3, 5), b=1)
    rng = np.random.default_rng(10 + rfl)
    params = random_params(cfg, rng)
    pk = O.make_packing(cfg.seq_lens, cfg.client_batch)
    X = rng.standard_normal((pk.T, cfg.hidden))
    dY = rng.standard_normal((pk.T, cfg.hidden))
    _, dX, grads = loss_and_grads(cfg, params, X, pk, dY)

    def f(params_, X_):
        Y, _ = run_stack(cfg, params_, X_, pk)
        return float((Y * dY).sum())

    h = 1e-5

    def check(an, perturb, n_samples, idx_rng):
        flat = an.reshape(-1)
        scale = max(np.abs(flat).max(), 1e-8)
        idx = idx_rng.choice(flat.size, size=min(n_samples, flat.size), replace=False)
        for i in idx:
            fp = perturb(i, +h)
            fm = perturb(i, -h)
            fd = (fp - fm) / (2 * h)
            assert abs(fd - flat[i]) <= 1e-6 * scale, (i, fd, flat[i], scale)

    irng = np.random.default_rng(99)

    def pert_x(i, d):
        Xp = X.copy()
        Xp.reshape(-1)[i] += d
        return f(params, Xp)
    check(dX, pert_x, 60, irng)

    for b in range(cfg.n_blocks):
        for t in range(12):
            def pert_p(i, d, b=b, t=t):
                pp = [[p.copy() if (bb == b and tt == t) else p for tt, p in enumerate(blk)]
                      for bb, blk in enumerate(params)]
                pp[b][t].reshape(-1)[i] += d
                return f(pp, X)
            check(grads[b][t], pert_p, 25, irng)


# ----------------------------------------------------------------------------- client-batching invariant

@pytest.mark.parametrize("rfl", [1, 0])
def test_client_batching_invariant(rfl):
    """§3.3 stacks clients: packed results equal each client run alone; weight
    gradients equal the sum of the per-client runs."""
    cfg = tiny_cfg(residual_from_ln=rfl, n_blocks=2, seq_lens=(3, 7, 1), b=2)
    rng = np.random.default_rng(20)
    params = random_params(cfg, rng, std=0.2)
    states = [rng.standard_normal((cfg.client_batch, L, cfg.hidden)) for L in cfg.seq_lens]
    gouts = [rng.standard_normal((cfg.client_batch, L, cfg.hidden)) for L in cfg.seq_lens]
    srv = O.OracleServer(cfg, params)
    outs = srv.forward(states)
    gins = srv.backward(gouts)
    gsum = [[np.zeros_like(p) for p in blk] for blk in srv.params]
    for k in range(cfg.K):
        for r in range(cfg.client_batch):
            c1 = cfg.with_(seq_lens=(cfg.seq_lens[k],), client_batch=1)
            s1 = O.OracleServer(c1, params)
            o1 = s1.forward([states[k][r:r + 1]])
            g1 = s1.backward([gouts[k][r:r + 1]])
            np.testing.assert_allclose(o1[0][0], outs[k][r], rtol=0, atol=1e-12)
            np.testing.assert_allclose(g1[0][0], gins[k][r], rtol=0, atol=1e-12)
            for b in range(cfg.n_blocks):
                for t in range(12):
                    gsum[b][t] += s1.grads[b][t]
    for b in range(cfg.n_blocks):
        for t in range(12):
            np.testing.assert_allclose(srv.grads[b][t], gsum[b][t], rtol=1e-10, atol=1e-12)


def test_causality_and_segment_isolation():
    cfg = tiny_cfg(n_blocks=2, seq_lens=(6, 5), b=1)
    rng = np.random.default_rng(21)
    params = random_params(cfg, rng)
    pk = O.make_packing(cfg.seq_lens, 1)
    X = rng.standard_normal((pk.T, cfg.hidden))
    Y, _ = run_stack(cfg, params, X, pk)
    # a later token of the same segment
    Xp = X.copy()
    Xp[4] += 3.0 * rng.standard_normal(cfg.hidden)   # not a constant shift: LN would remove that
    Yp, _ = run_stack(cfg, params, Xp, pk)
    np.testing.assert_array_equal(Yp[:4], Y[:4])
    assert np.abs(Yp[4:6] - Y[4:6]).max() > 1e-3
    np.testing.assert_array_equal(Yp[6:], Y[6:])
    # any token of the other segment
    Xq = X.copy()
    Xq[7] -= 2.0 * rng.standard_normal(cfg.hidden)
    Yq, _ = run_stack(cfg, params, Xq, pk)
    np.testing.assert_array_equal(Yq[:6], Y[:6])


# ----------------------------------------------------------------------------- AdamW

def test_adamw_first_step_closed_form():
    rng = np.random.default_rng(30)
    w = rng.standard_normal(1000)
    g = rng.standard_normal(1000) * 1e-3
    for wd in (0.0, 0.01):
        w1, m1, v1 = O.adamw_update(w, g, np.zeros_like(w), np.zeros_like(w), 1, 1e-4, 0.9, 0.999, 1e-8, wd)
        np.testing.assert_allclose(w1, w - 1e-4 * (g / (np.abs(g) + 1e-8) + wd * w), rtol=0, atol=1e-15)
        np.testing.assert_allclose(m1, 0.1 * g, rtol=1e-14)
        np.testing.assert_allclose(v1, 0.001 * g * g, rtol=1e-14)


def test_adamw_matches_torch_over_steps():
    rng = np.random.default_rng(31)
    w0 = rng.standard_normal(257)
    tw = torch.tensor(w0.copy(), requires_grad=True)
    opt = torch.optim.AdamW([tw], lr=3e-3, betas=(0.9, 0.999), eps=1e-8, weight_decay=0.05)
    w, m, v = w0.copy(), np.zeros(257), np.zeros(257)
    for t in range(1, 6):
        g = rng.standard_normal(257)
        tw.grad = torch.tensor(g)
        opt.step()
        w, m, v = O.adamw_update(w, g, m, v, t, 3e-3, 0.9, 0.999, 1e-8, 0.05)
        np.testing.assert_allclose(w, tw.detach().numpy(), rtol=0, atol=1e-13)


def test_server_protocol_state_and_accumulation():
    """forward/backward pairs without a step accumulate (serial mode, §3.3); step clears."""
    cfg = tiny_cfg(n_blocks=1, seq_lens=(3, 2), b=1)
    rng = np.random.default_rng(40)
    params = random_params(cfg, rng, std=0.2)
    st = [rng.standard_normal((1, L, cfg.hidden)) for L in cfg.seq_lens]
    gr = [rng.standard_normal((1, L, cfg.hidden)) for L in cfg.seq_lens]
    srv = O.OracleServer(cfg, params)
    with pytest.raises(RuntimeError):
        srv.backward(gr)
    # serial: one client at a time, then one step
    ser = O.OracleServer(cfg, params)
    for k in range(cfg.K):
        ser.forward([st[k]])
        ser.backward([gr[k]])
    srv.forward(st)
    srv.backward(gr)
    for t in range(12):
        np.testing.assert_allclose(ser.grads[0][t], srv.grads[0][t], rtol=1e-10, atol=1e-12)
    srv.step(1e-3)
    assert all(not g.any() for g in srv.grads[0])
    assert srv.t == 1


def test_replica_averaging():
    """Averaging is the arithmetic mean; identical replicas are unchanged; training K
    replicas on the same client for one step and averaging equals one replica's step."""
    cfg = tiny_cfg(n_blocks=1, seq_lens=(3,), b=1)
    rng = np.random.default_rng(50)
    params = random_params(cfg, rng, std=0.2)
    a = O.OracleServer(cfg, params)
    b = O.OracleServer(cfg, params)
    c = O.OracleServer(cfg, params)
    for t in range(12):
        b.params[0][t] = b.params[0][t] + 1.0
        c.params[0][t] = c.params[0][t] - 4.0
    O.average_params([a, b, c])
    for t in range(12):
        np.testing.assert_allclose(a.params[0][t], np.asarray(params[0][t]) - 1.0, rtol=0, atol=1e-12)
        np.testing.assert_array_equal(a.params[0][t], c.params[0][t])
    st = [rng.standard_normal((1, 3, cfg.hidden))]
    gr = [rng.standard_normal((1, 3, cfg.hidden))]
    reps = [O.OracleServer(cfg, params) for _ in range(3)]
    for r in reps:
        r.forward(st)
        r.backward(gr)
        r.step(1e-3)
    O.average_params(reps)
    for t in range(12):
        np.testing.assert_allclose(reps[0].params[0][t], reps[1].params[0][t], rtol=0, atol=0)


# ----------------------------------------------------------------------------- P-tuning v2 prefix (App. A)

def test_prefix_attention_matches_torch_sdpa():
    """Each query sees every prefix key and its own causal keys: one SDPA call per segment
    with an explicit boolean mask over [prefix ; segment]."""
    rng = np.random.default_rng(60)
    seq = [5, 1, 9]
    cu = np.cumsum([0] + seq).astype(np.int32)
    T, nh, hd, Lp = cu[-1], 2, 8, 3
    q, k, v = (rng.standard_normal((T, nh, hd)) for _ in range(3))
    pk, pv = (rng.standard_normal((Lp, nh, hd)) for _ in range(2))
    o, lse = O.attention_fwd(q, k, v, cu, pk, pv)
    for s in range(len(seq)):
        a, b = cu[s], cu[s + 1]
        L = b - a
        tq = torch.tensor(q[a:b]).transpose(0, 1)
        tk = torch.tensor(np.concatenate([pk, k[a:b]])).transpose(0, 1)
        tv = torch.tensor(np.concatenate([pv, v[a:b]])).transpose(0, 1)
        mask = torch.cat([torch.ones(L, Lp, dtype=torch.bool), torch.ones(L, L, dtype=torch.bool).tril()], 1)
        ref = torch.nn.functional.scaled_dot_product_attention(tq, tk, tv, attn_mask=mask).transpose(0, 1).numpy()
        np.testing.assert_allclose(o[a:b], ref, rtol=0, atol=1e-12)


def test_zero_value_prefix_closed_form():
    """With zero prefix values the prefix only adds mass to the softmax denominator:
    O' = O exp(LSE - LSE') and LSE' = log(exp(LSE) + sum_p exp(q.k_p / sqrt(d_h)))."""
    rng = np.random.default_rng(61)
    seq = [6, 4]
    cu = np.cumsum([0] + seq).astype(np.int32)
    T, nh, hd, Lp = cu[-1], 2, 8, 5
    q, k, v = (rng.standard_normal((T, nh, hd)) for _ in range(3))
    pk = rng.standard_normal((Lp, nh, hd))
    o0, lse0 = O.attention_fwd(q, k, v, cu)
    o1, lse1 = O.attention_fwd(q, k, v, cu, pk, np.zeros((Lp, nh, hd)))
    lp = np.log(np.exp(np.einsum("thd,phd->htp", q, pk) / math.sqrt(hd)).sum(-1))
    np.testing.assert_allclose(lse1, np.logaddexp(lse0, lp), rtol=0, atol=1e-12)
    np.testing.assert_allclose(o1, o0 * np.exp(lse0 - lse1).T[:, :, None], rtol=0, atol=1e-12)


@pytest.mark.parametrize("rfl", [1, 0])
def test_finite_difference_prefix_gradients(rfl):
    cfg = tiny_cfg(residual_from_ln=rfl, n_blocks=2, seq_lens=(3, 5), b=1).with_(prefix_len=2)
    rng = np.random.default_rng(62 + rfl)
    params = random_params(cfg, rng)
    prefixes = [[0.5 * rng.standard_normal((2, cfg.hidden)) for _ in range(2)] for _ in range(cfg.n_blocks)]
    pk = O.make_packing(cfg.seq_lens, 1)
    X = rng.standard_normal((pk.T, cfg.hidden))
    dY = rng.standard_normal((pk.T, cfg.hidden))
    sh = O.BlockShape.of(cfg)

    def f(pre, X_):
        Y, _ = O.stack_fwd(params, X_, pk, sh, pre)
        return float((Y * dY).sum())
    _, saved = O.stack_fwd(params, X, pk, sh, prefixes)
    dX, grads = O.stack_bwd(params, saved, dY, pk, sh)
    h = 1e-5
    for b in range(cfg.n_blocks):
        for j in range(2):
            an = grads[b][12 + j].reshape(-1)
            scale = np.abs(an).max()
            for i in range(an.size):
                pp = [[p.copy() for p in blk] for blk in prefixes]
                pp[b][j].reshape(-1)[i] += h
                fp = f(pp, X)
                pp[b][j].reshape(-1)[i] -= 2 * h
                fm = f(pp, X)
                assert abs((fp - fm) / (2 * h) - an[i]) <= 1e-6 * scale, (b, j, i)
    # the input gradient with a prefix, spot-checked
    for i in (0, 17, 60, 127):
        Xp = X.copy()
        Xp.reshape(-1)[i] += h
        fp = f(prefixes, Xp)
        Xp.reshape(-1)[i] -= 2 * h
        fm = f(prefixes, Xp)
        assert abs((fp - fm) / (2 * h) - dX.reshape(-1)[i]) <= 1e-6 * np.abs(dX).max()


def test_prefix_batching_invariant_and_frozen_step():
    """The shared prefix keeps clients unmixed: packed results equal per-client runs and
    prefix gradients are the sum of the per-client ones; with a frozen base only the
    prefixes move."""
    cfg = tiny_cfg(n_blocks=2, seq_lens=(3, 6), b=1).with_(prefix_len=3, freeze_base=1)
    rng = np.random.default_rng(63)
    params = random_params(cfg, rng, std=0.2)
    prefixes = [[0.3 * rng.standard_normal((3, cfg.hidden)) for _ in range(2)] for _ in range(cfg.n_blocks)]
    states = [rng.standard_normal((1, L, cfg.hidden)) for L in cfg.seq_lens]
    gouts = [rng.standard_normal((1, L, cfg.hidden)) for L in cfg.seq_lens]
    srv = O.OracleServer(cfg, params, prefixes)
    outs = srv.forward(states)
    gins = srv.backward(gouts)
    gsum = [[np.zeros_like(p) for p in blk[12:]] for blk in srv.params]
    for k in range(cfg.K):
        s1 = O.OracleServer(cfg.with_(seq_lens=(cfg.seq_lens[k],)), params, prefixes)
        o1 = s1.forward([states[k]])
        g1 = s1.backward([gouts[k]])
        np.testing.assert_allclose(o1[0], outs[k], rtol=0, atol=1e-12)
        np.testing.assert_allclose(g1[0], gins[k], rtol=0, atol=1e-12)
        for b in range(cfg.n_blocks):
            for j in range(2):
                gsum[b][j] += s1.grads[b][12 + j]
    for b in range(cfg.n_blocks):
        for j in range(2):
            np.testing.assert_allclose(srv.grads[b][12 + j], gsum[b][j], rtol=1e-10, atol=1e-12)
    w_before = [[p.copy() for p in blk] for blk in srv.params]
    srv.step(1e-2)
    for b in range(cfg.n_blocks):
        for t in range(12):
            np.testing.assert_array_equal(srv.params[b][t], w_before[b][t])
        for t in (12, 13):
            assert np.abs(srv.params[b][t] - w_before[b][t]).max() > 1e-3


# ----------------------------------------------------------------------------- GLM blank infilling

def glm_mask_parts(L, c):
    """GLM's attention rule stated by parts: tokens of Part A (the context, t < c) see all
    of Part A; tokens of Part B (the span) see Part A and the span tokens up to themselves.
    c = 0: no Part A, the segment is plainly causal."""
    m = np.zeros((L, L), bool)
    for t in range(L):
        for u in range(L):
            if t < c:
                m[t, u] = u < c
            else:
                m[t, u] = u < c or (c <= u <= t)
    return m


def test_glm_positions_worked_example():
    p1, p2 = O.glm_positions(7, 4, 2)
    assert p1.tolist() == [0, 1, 2, 3, 2, 2, 2]
    assert p2.tolist() == [0, 0, 0, 0, 1, 2, 3]
    p1, p2 = O.glm_positions(5, 0, 0)
    assert p1.tolist() == [0, 1, 2, 3, 4] and p2.tolist() == [0] * 5
    p1, p2 = O.glm_positions(3, 3, 2)      # all context: no span
    assert p1.tolist() == [0, 1, 2] and p2.tolist() == [0, 0, 0]
    for bad in [(4, 5, 0), (4, 2, 2), (4, -1, 0)]:
        with pytest.raises(ValueError):
            O.glm_positions(*bad)
    pk = O.make_packing([4, 3], 1, context_lens=[2, 0], mask_pos=[0, 0])
    assert pk.pos.tolist() == [0, 1, 0, 0, 0, 1, 2]
    assert pk.pos2.tolist() == [0, 0, 1, 2, 0, 0, 0]
    # default [M] position: the last context token (summarisation layout)
    assert O.make_packing([4], 1, context_lens=[3]).pos.tolist() == [0, 1, 2, 2]


@pytest.mark.parametrize("Lp", [0, 3])
def test_glm_attention_matches_torch_sdpa(Lp):
    """Bidirectional context + causal span, per segment, against SDPA with the mask of
    glm_mask_parts (and every prefix key visible)."""
    rng = np.random.default_rng(70 + Lp)
    seq, ctx = [5, 1, 9, 6, 4], [3, 1, 0, 6, 1]
    cu = np.cumsum([0] + seq).astype(np.int32)
    T, nh, hd = cu[-1], 2, 8
    q, k, v = (rng.standard_normal((T, nh, hd)) for _ in range(3))
    pk = pv = None
    if Lp:
        pk, pv = (rng.standard_normal((Lp, nh, hd)) for _ in range(2))
    o, lse = O.attention_fwd(q, k, v, cu, pk, pv, ctx=np.array(ctx))
    for s in range(len(seq)):
        a, b = cu[s], cu[s + 1]
        L = b - a
        keys = k[a:b] if not Lp else np.concatenate([pk, k[a:b]])
        vals = v[a:b] if not Lp else np.concatenate([pv, v[a:b]])
        tq = torch.tensor(q[a:b]).transpose(0, 1)
        tk = torch.tensor(keys).transpose(0, 1)
        tv = torch.tensor(vals).transpose(0, 1)
        mask = torch.cat([torch.ones(L, Lp, dtype=torch.bool), torch.tensor(glm_mask_parts(L, ctx[s]))], 1)
        ref = torch.nn.functional.scaled_dot_product_attention(tq, tk, tv, attn_mask=mask).transpose(0, 1).numpy()
        np.testing.assert_allclose(o[a:b], ref, rtol=0, atol=1e-12)
        S = (torch.einsum("hid,hjd->hij", tq, tk) / math.sqrt(hd)).masked_fill(~mask, float("-inf"))
        np.testing.assert_allclose(lse[:, a:b], torch.logsumexp(S, -1).numpy(), rtol=0, atol=1e-12)


def test_glm_attention_special_cases():
    """c = L is plain (non-causal) attention over the segment; c = 0 and c = 1 are the
    causal case exactly."""
    rng = np.random.default_rng(72)
    seq = [7, 4]
    cu = np.cumsum([0] + seq).astype(np.int32)
    T, nh, hd = cu[-1], 2, 8
    q, k, v = (rng.standard_normal((T, nh, hd)) for _ in range(3))
    o_full, _ = O.attention_fwd(q, k, v, cu, ctx=np.array(seq))
    for s in range(2):
        a, b = cu[s], cu[s + 1]
        t = [torch.tensor(z[a:b]).transpose(0, 1) for z in (q, k, v)]
        ref = torch.nn.functional.scaled_dot_product_attention(*t, is_causal=False).transpose(0, 1).numpy()
        np.testing.assert_allclose(o_full[a:b], ref, rtol=0, atol=1e-12)
    o_c, l_c = O.attention_fwd(q, k, v, cu)
    for c in (0, 1):
        o_g, l_g = O.attention_fwd(q, k, v, cu, ctx=np.array([c, c]))
        np.testing.assert_array_equal(o_g, o_c)
        np.testing.assert_array_equal(l_g, l_c)


def test_rope_2d_properties():
    """ChatGLM's 2D rotary: the second half of each head turns by the block position with
    the first half's frequencies; block position 0 is the identity."""
    rng = np.random.default_rng(73)
    hd, rd, base = 16, 8, 10000.0
    pk = O.make_packing([9], 1, context_lens=[4], mask_pos=[1])
    x = rng.standard_normal((9, 2, hd))
    xr = O.rope_2d(x, pk, rd, base)
    theta = base ** (-2.0 * np.arange(rd // 2) / rd)
    for lo, p in ((0, pk.pos), (rd, pk.pos2)):
        z = (x[..., lo:lo + rd // 2] + 1j * x[..., lo + rd // 2:lo + rd]) * np.exp(1j * p[:, None, None] * theta)
        np.testing.assert_allclose(xr[..., lo:lo + rd // 2], z.real, atol=1e-13)
        np.testing.assert_allclose(xr[..., lo + rd // 2:lo + rd], z.imag, atol=1e-13)
    np.testing.assert_allclose(O.rope_2d(xr, pk, rd, base, inverse=True), x, atol=1e-13)
    # no GLM structure: the 1D rotation, second half untouched
    plain = O.make_packing([9], 1)
    np.testing.assert_array_equal(O.rope_2d(x, plain, rd, base)[..., rd:], x[..., rd:])
    # all block positions 0: bit-identical to the 1D rotation
    zero2 = O.make_packing([9], 1, context_lens=[9], mask_pos=[8])
    np.testing.assert_array_equal(O.rope_2d(x, zero2, rd, base), O.rope_2d(x, plain, rd, base))
    # q . k depends only on the differences of both positions
    q = rng.standard_normal((1, 1, hd))
    kk = rng.standard_normal((1, 1, hd))

    def dot(p1, p2, pp1, pp2):
        def one(v, a, b):
            fake = O.Packing(np.array([0, 1], np.int32), np.array([a], np.int32), np.zeros(1, np.int32),
                             np.zeros(1, np.int32), np.array([1], np.int32), np.array([b], np.int32))
            return O.rope_2d(v, fake, rd, base)
        return float((one(q, p1, p2) * one(kk, pp1, pp2)).sum())
    assert abs(dot(7, 3, 2, 1) - dot(12, 5, 7, 3)) < 1e-12
    assert abs(dot(7, 3, 2, 1) - dot(7, 4, 2, 1)) > 1e-6   # the block position matters


@pytest.mark.parametrize("rfl,Lp", [(1, 0), (0, 0), (1, 2)])
def test_finite_difference_glm_gradients(rfl, Lp):
    """Chain rule through the GLM mask and the 2D rotary (and a prefix): central
    differences on inputs and every parameter."""
    cfg = tiny_cfg(residual_from_ln=rfl, n_blocks=2, seq_lens=(4, 6), b=1).with_(prefix_len=Lp)
    rng = np.random.default_rng(74 + rfl + Lp)
    params = random_params(cfg, rng)
    if Lp:
        for blk in params:
            blk.extend(0.5 * rng.standard_normal(s) for s in syn.prefix_shapes(cfg))
    pk = O.make_packing(cfg.seq_lens, 1, context_lens=[2, 4], mask_pos=[0, 1])
    sh = O.BlockShape.of(cfg)
    X = rng.standard_normal((pk.T, cfg.hidden))
    dY = rng.standard_normal((pk.T, cfg.hidden))
    base = [blk[:12] for blk in params]
    pre = [blk[12:] for blk in params] if Lp else None
    Y, saved = O.stack_fwd(base, X, pk, sh, pre)
    dX, grads = O.stack_bwd(base, saved, dY, pk, sh)

    def f(pp, X_):
        Y_, _ = O.stack_fwd([b[:12] for b in pp], X_, pk, sh, [b[12:] for b in pp] if Lp else None)
        return float((Y_ * dY).sum())

    h = 1e-5
    irng = np.random.default_rng(98)

    def check(an, perturb, n):
        flat = an.reshape(-1)
        scale = max(np.abs(flat).max(), 1e-8)
        for i in irng.choice(flat.size, size=min(n, flat.size), replace=False):
            fd = (perturb(i, +h) - perturb(i, -h)) / (2 * h)
            assert abs(fd - flat[i]) <= 1e-6 * scale, (i, fd, flat[i], scale)

    def pert_x(i, d):
        Xp = X.copy()
        Xp.reshape(-1)[i] += d
        return f(params, Xp)
    check(dX, pert_x, 60)
    for b in range(cfg.n_blocks):
        for t in range(len(params[b])):
            def pert_p(i, d, b=b, t=t):
                pp = [[p.copy() if (bb == b and tt == t) else p for tt, p in enumerate(blk)]
                      for bb, blk in enumerate(params)]
                pp[b][t].reshape(-1)[i] += d
                return f(pp, X)
            check(grads[b][t], pert_p, 20)


def test_glm_context_is_bidirectional_and_span_causal():
    """A later context token changes an earlier context token's output (bidirectional); a
    span token changes neither the context nor earlier span tokens, nor another segment."""
    cfg = tiny_cfg(n_blocks=2, seq_lens=(7, 5), b=1)
    rng = np.random.default_rng(75)
    params = random_params(cfg, rng)
    pk = O.make_packing(cfg.seq_lens, 1, context_lens=[4, 2], mask_pos=[3, 0])
    X = rng.standard_normal((pk.T, cfg.hidden))
    Y, _ = run_stack(cfg, params, X, pk)
    Xa = X.copy()
    Xa[3] += 3.0 * rng.standard_normal(cfg.hidden)        # last context token of segment 0
    Ya, _ = run_stack(cfg, params, Xa, pk)
    assert np.abs(Ya[0] - Y[0]).max() > 1e-3
    np.testing.assert_array_equal(Ya[7:], Y[7:])
    Xb = X.copy()
    Xb[5] += 3.0 * rng.standard_normal(cfg.hidden)        # second span token of segment 0
    Yb, _ = run_stack(cfg, params, Xb, pk)
    np.testing.assert_array_equal(Yb[:5], Y[:5])
    assert np.abs(Yb[5:7] - Y[5:7]).max() > 1e-3
    np.testing.assert_array_equal(Yb[7:], Y[7:])


def test_glm_batching_invariant():
    """§3.3 stacking with GLM segments: packed outputs and input grads equal each segment
    alone; weight grads are the per-segment sum."""
    cfg = tiny_cfg(n_blocks=2, seq_lens=(5, 3), b=2)
    rng = np.random.default_rng(76)
    params = random_params(cfg, rng, std=0.2)
    ctx, mp = [3, 5, 1, 2], [2, 0, 0, 1]
    states = [rng.standard_normal((2, L, cfg.hidden)) for L in cfg.seq_lens]
    gouts = [rng.standard_normal((2, L, cfg.hidden)) for L in cfg.seq_lens]
    srv = O.OracleServer(cfg, params)
    outs = srv.forward(states, ctx, mp)
    gins = srv.backward(gouts)
    gsum = [[np.zeros_like(p) for p in blk] for blk in srv.params]
    s = 0
    for k in range(cfg.K):
        for r in range(2):
            one = O.OracleServer(cfg.with_(seq_lens=(cfg.seq_lens[k],), client_batch=1), params)
            o1 = one.forward([states[k][r:r + 1]], [ctx[s]], [mp[s]])
            g1 = one.backward([gouts[k][r:r + 1]])
            np.testing.assert_array_equal(o1[0][0], outs[k][r])
            np.testing.assert_array_equal(g1[0][0], gins[k][r])
            for b in range(cfg.n_blocks):
                for t in range(12):
                    gsum[b][t] += one.grads[b][t]
            s += 1
    for b in range(cfg.n_blocks):
        for t in range(12):
            np.testing.assert_allclose(srv.grads[b][t], gsum[b][t], rtol=1e-12, atol=1e-12)


def test_glm_structure_recipe():
    """The synthetic GLM structure: span of 1..L/4 tokens after the context, [M] inside it."""
    cfg = syn.CONFIGS["ragged26"]
    ctx, mp = syn.glm_structure(cfg)
    for L, c, m in zip(cfg.segment_lengths, ctx, mp):
        assert 1 <= L - c <= max(1, L // 4) and 0 <= m < c
    assert any(m == c - 1 for c, m in zip(ctx, mp)) and any(m < c - 1 for c, m in zip(ctx, mp))


# ----------------------------------------------------------------------------- client parts (§3.1)

def test_cross_entropy_matches_torch():
    rng = np.random.default_rng(80)
    T, V = 23, 37
    logits = 3.0 * rng.standard_normal((T, V))
    labels = rng.integers(0, V, size=T).astype(np.int32)
    labels[[2, 5, 11]] = -1
    loss, d = O.cross_entropy(logits, labels)
    tl = torch.tensor(logits, requires_grad=True)
    ref = torch.nn.functional.cross_entropy(tl, torch.tensor(labels, dtype=torch.long), ignore_index=-1)
    ref.backward()
    assert abs(loss - ref.item()) < 1e-12
    np.testing.assert_allclose(d, tl.grad.numpy(), rtol=0, atol=1e-14)
    # no target at all: zero loss and gradient
    l0, d0 = O.cross_entropy(logits, np.full(T, -1, np.int32))
    assert l0 == 0.0 and not d0.any()


def test_cross_entropy_uniform_closed_form():
    """Equal logits: loss = log V; gradient (1/V - onehot) / n on the rows with a target."""
    T, V = 6, 50
    labels = np.array([3, -1, 0, 49, -1, 7], np.int32)
    loss, d = O.cross_entropy(np.full((T, V), 0.7), labels)
    assert abs(loss - math.log(V)) < 1e-14
    want = np.zeros((T, V))
    for t, y in enumerate(labels):
        if y >= 0:
            want[t] = 1.0 / V
            want[t, y] -= 1.0
    np.testing.assert_allclose(d, want / 4, rtol=0, atol=1e-15)


def test_embedding_matches_torch():
    rng = np.random.default_rng(81)
    V, H = 20, 6
    E = rng.standard_normal((V, H))
    tokens = np.array([3, 7, 3, 19, 0, 3, 7], np.int64)
    dX = rng.standard_normal((len(tokens), H))
    tE = torch.tensor(E, requires_grad=True)
    out = torch.nn.functional.embedding(torch.tensor(tokens), tE)
    np.testing.assert_array_equal(O.embedding_fwd(E, tokens), out.detach().numpy())
    out.backward(torch.tensor(dX))
    np.testing.assert_allclose(O.embedding_bwd(dX, tokens, V), tE.grad.numpy(), rtol=0, atol=1e-14)


def client_cfg(**kw):
    return tiny_cfg(n_blocks=1, seq_lens=(5,), b=2).with_(vocab=29, **kw)


def random_client_params(cfg, rng):
    p = {"bottom": random_params(cfg, rng)[0], "top": random_params(cfg, rng)[0]}
    if cfg.prefix_len:
        for k in ("bottom", "top"):
            p[k] += [0.5 * rng.standard_normal(s) for s in syn.prefix_shapes(cfg)]
    p["embed"] = [rng.standard_normal((cfg.vocab, cfg.hidden))]
    p["head"] = [0.3 * rng.standard_normal((cfg.vocab, cfg.hidden))]
    p["final_ln"] = [1.0 + 0.3 * rng.standard_normal(cfg.hidden), 0.3 * rng.standard_normal(cfg.hidden)]
    return p


@pytest.mark.parametrize("Lp,glm", [(0, False), (2, True)])
def test_client_finite_differences(Lp, glm):
    """Loss of the client alone (bottom output handed straight to the top): central
    differences on every client parameter, with and without GLM segments and prefixes."""
    cfg = client_cfg(prefix_len=Lp)
    rng = np.random.default_rng(82 + Lp)
    params = random_client_params(cfg, rng)
    tokens = rng.integers(0, cfg.vocab, size=(2, 5)).astype(np.int32)
    ctx = [3, 1] if glm else None
    labels = syn.client_labels(tokens, ctx)

    def run(p, with_grads=False):
        cl = O.OracleClient(cfg, p)
        h0 = cl.bottom_forward(tokens, ctx)
        loss, gh = cl.top_forward_backward(h0, labels)
        if with_grads:
            cl.bottom_backward(gh)
        return loss, cl

    _, cl = run(params, True)
    h = 1e-5
    irng = np.random.default_rng(83)
    for part in O.CLIENT_PARTS:
        for i, an in enumerate(cl.grads[part]):
            flat = an.reshape(-1)
            scale = max(np.abs(flat).max(), 1e-8)
            if part == "embed":   # rows of tokens that occur, plus one that does not
                rows = sorted(set(tokens.reshape(-1).tolist()))[:3] + [int(np.setdiff1d(np.arange(cfg.vocab), tokens)[0])]
                idx = [r * cfg.hidden + c for r in rows for c in (0, 5)]
            else:
                idx = irng.choice(flat.size, size=min(12, flat.size), replace=False)
            for j in idx:
                vals = []
                for dlt in (h, -h):
                    pp = {k: [x.copy() for x in v] for k, v in params.items()}
                    pp[part][i].reshape(-1)[j] += dlt
                    vals.append(run(pp)[0])
                fd = (vals[0] - vals[1]) / (2 * h)
                assert abs(fd - flat[j]) <= 1e-6 * scale, (part, i, j, fd, flat[j])


def test_split_equals_unsplit_model():
    """§3.1 splits one model: client bottom -> server blocks -> client top gives the loss and
    the embedding gradient of the same model run in one piece (embedding, all blocks in
    order, final LayerNorm, head, cross-entropy)."""
    cfg = tiny_cfg(n_blocks=2, seq_lens=(6, 4), b=1).with_(vocab=31)
    rng = np.random.default_rng(84)
    cp = random_client_params(cfg.with_(n_blocks=1), rng)
    sp = random_params(cfg, rng)
    toks = [rng.integers(0, cfg.vocab, size=(1, L)).astype(np.int32) for L in cfg.seq_lens]
    ctx = [[4], [0]]
    clients = [O.OracleClient(cfg, cp) for _ in toks]
    srv = O.OracleServer(cfg, sp)
    h0 = [c.bottom_forward(t, cx) for c, t, cx in zip(clients, toks, ctx)]
    hs = srv.forward(h0, [cx[0] for cx in ctx])
    out = [c.top_forward_backward(h, syn.client_labels(t, cx)) for c, h, t, cx in zip(clients, hs, toks, ctx)]
    gi = srv.backward([g for _, g in out])
    for c, g in zip(clients, gi):
        c.bottom_backward(g)
    sh = O.BlockShape.of(cfg)
    E, W = cp["embed"][0], cp["head"][0]
    stack = [cp["bottom"]] + sp + [cp["top"]]
    for k, (t, cx) in enumerate(zip(toks, ctx)):
        pk = O.make_packing([t.shape[1]], 1, cx)
        x = E[t.reshape(-1)]
        y, saved = O.stack_fwd(stack, x, pk, sh)
        z, mu, rs = O.layer_norm_fwd(y, cp["final_ln"][0], cp["final_ln"][1], cfg.ln_eps)
        loss, dlog = O.cross_entropy(z @ W.T, syn.client_labels(t, cx).reshape(-1))
        assert abs(loss - out[k][0]) < 1e-12
        dz = dlog @ W
        dy, _, _ = O.layer_norm_bwd(dz, y, mu, rs, cp["final_ln"][0])
        dx, _ = O.stack_bwd(stack, saved, dy, pk, sh)
        np.testing.assert_allclose(clients[k].grads["embed"][0], O.embedding_bwd(dx, t.reshape(-1), cfg.vocab),
                                   rtol=1e-10, atol=1e-12)


def test_client_averaging_and_frozen_step():
    cfg = client_cfg(prefix_len=2, freeze_base=1)
    rng = np.random.default_rng(85)
    cls = [O.OracleClient(cfg, random_client_params(cfg, rng)) for _ in range(3)]
    want = {k: [sum(c.params[k][i] for c in cls) / 3 for i in range(len(cls[0].params[k]))] for k in O.CLIENT_PARTS}
    O.average_clients(cls)
    for c in cls:
        for k in O.CLIENT_PARTS:
            for i, w in enumerate(want[k]):
                np.testing.assert_array_equal(c.params[k][i], w)
    # P-tuning v2: a step moves only the client blocks' prefixes
    c = cls[0]
    tokens = rng.integers(0, cfg.vocab, size=(2, 5)).astype(np.int32)
    before = {k: [x.copy() for x in v] for k, v in c.params.items()}
    _, g = c.top_forward_backward(c.bottom_forward(tokens), syn.client_labels(tokens))
    c.bottom_backward(g)
    c.step(1e-2)
    for k in O.CLIENT_PARTS:
        for i, w in enumerate(c.params[k]):
            moved = not np.array_equal(w, before[k][i])
            assert moved == (k in ("bottom", "top") and i >= 12), (k, i)
