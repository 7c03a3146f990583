"""Client parts of the split (§3.1) on the GPU: embedding + block 0 at the bottom, block
N-1 + final LayerNorm + LM head + cross-entropy at the top, the full split round with the
server, and client averaging (§3.3).  Parity against the fp64 oracle (GPU only)."""
import numpy as np
import pytest
import torch

import synthetic as syn
from oracle import flglm_oracle as O
from tests._gpu import bits, dev_bf16_from_bits, dev_i32, f64, flglm, need_gpu, rel_inf
from tests.test_gpu_server import GRAD_TOL, OUT_TOL, check_updated_weights

pytestmark = pytest.mark.gpu

LOSS_TOL = 1e-2


@pytest.fixture(scope="module")
def F():
    need_gpu()
    return flglm()


def tiny_client(**kw):
    return syn.CONFIGS["tiny"].with_(client_batch=2, seq_lens=(64,), vocab=1000, lr=1e-3, **kw)


def bf16_dev(x64):
    return dev_bf16_from_bits(syn.f32_to_bf16_bits(np.asarray(x64, np.float32)))


def part_tensors(cfg):
    n_blk = 14 if cfg.prefix_len else 12
    out = [(F_part, t) for F_part in ("bottom", "top") for t in range(n_blk)]
    return out + [("embed", 0), ("head", 0), ("final_ln", 0), ("final_ln", 1)]


PART_IDS = {"bottom": 0, "top": 1, "embed": 2, "head": 3, "final_ln": 4}


def test_client_init_matches_generator(F):
    cfg = tiny_client(prefix_len=8)
    cl = F.Client(F.make_client_cfg(cfg, cfg.tokens), cfg.seed)
    want = syn.init_client(cfg)
    for part, t in part_tensors(cfg):
        got = cl.get_param(PART_IDS[part], t)
        w = want[part][t].reshape(-1)
        ulps = np.abs(got.view(np.int32).astype(np.int64) - w.astype(np.float32).view(np.int32).astype(np.int64))
        assert ulps.max() <= 1, (part, t, ulps.max())
    cl.close()


def client_round(F, cfg, ctx=None, mp=None, check_step=True, params=None):
    """One client alone (its bottom output handed straight to its top), GPU against the
    oracle on the same bf16 hand-offs."""
    cl = F.Client(F.make_client_cfg(cfg, cfg.tokens), cfg.seed)
    if params is None:
        params = syn.init_client(cfg)
    else:   # explicit values: loaded into the client, the oracle takes the same ones
        for part, t in part_tensors(cfg):
            cl.set_param(PART_IDS[part], t, params[part][t])
    tokens = syn.client_tokens(cfg, 0)
    labels = syn.client_labels(tokens, ctx)
    b, L = tokens.shape
    h0 = torch.empty((b, L, cfg.hidden), dtype=torch.bfloat16, device="cuda")
    cl.bottom_forward(dev_i32(tokens), L, h0, context_lens=ctx, mask_pos=mp)
    loss = torch.zeros(1, dtype=torch.float32, device="cuda")
    gh = torch.empty_like(h0)
    cl.top_forward_backward(h0, dev_i32(labels), loss, gh)
    gh_bits = bits(gh)
    cl.bottom_backward(gh)
    cl.sync()
    ref = O.OracleClient(cfg, params)
    h0_ref = ref.bottom_forward(tokens, ctx, mp)
    assert rel_inf(f64(h0), h0_ref) < OUT_TOL
    # the top and the bottom backward see the GPU's bf16 hand-offs, as the protocol sends them
    loss_ref, gh_ref = ref.top_forward_backward(syn.bf16_bits_to_f64(bits(h0)).reshape(b, L, -1), labels)
    assert abs(float(loss.item()) - loss_ref) / abs(loss_ref) < LOSS_TOL, (loss.item(), loss_ref)
    assert rel_inf(f64(gh), gh_ref) < GRAD_TOL
    ref.bottom_backward(syn.bf16_bits_to_f64(gh_bits).reshape(b, L, -1))
    trained = set(ref.trained())
    gref = {}
    for part, t in part_tensors(cfg):
        g = cl.get_grad(PART_IDS[part], t)
        gr = ref.grads[part][t].reshape(-1)
        gref[(part, t)] = gr.copy()
        if (part, t) in trained:
            e = rel_inf(g, gr)
            assert e < GRAD_TOL, ("grad", part, t, e)
        elif part not in ("bottom", "top"):
            assert not g.any()   # frozen: no gradient kept
    if check_step:
        cl.step(cfg.lr)
        ref.step(cfg.lr)
        cl.sync()
        for part, t in part_tensors(cfg):
            w0 = np.asarray(params[part][t], np.float32).reshape(-1)
            w = cl.get_param(PART_IDS[part], t)
            if (part, t) in trained:
                check_updated_weights(w, ref.params[part][t].reshape(-1), w0, gref[(part, t)], cfg.lr, (part, t))
            else:
                np.testing.assert_array_equal(w, w0)
    cl.close()


def test_client_parity(F):
    client_round(F, tiny_client())


def test_client_parity_glm_ptuning(F):
    """The paper's client: GLM blank-infilling rows, P-tuning v2 prefixes in both client
    blocks, everything else frozen."""
    cfg = tiny_client(prefix_len=16, freeze_base=1)
    ctx = [40, 63]
    client_round(F, cfg, ctx=ctx, mp=[39, 10])


def test_split_round_matches_oracle(F):
    """The whole protocol of §3.1 on one GPU: two clients' bottoms, one client-batched
    server call (§3.3), the clients' tops, the server backward, the clients' bottom
    backwards and every step, against the oracle client/server composition."""
    cfg = syn.CONFIGS["tiny"].with_(n_blocks=2, client_batch=2, seq_lens=(64, 48), vocab=1000, lr=1e-3)
    K, b = cfg.K, cfg.client_batch
    ctx_all, mp_all = syn.glm_structure(cfg)
    ccfgs = [cfg.with_(seq_lens=(L,)) for L in cfg.seq_lens]
    srv = F.Server(F.make_cfg(cfg, cfg.tokens), cfg.seed)
    clients = [F.Client(F.make_client_cfg(c, c.tokens), cfg.seed) for c in ccfgs]
    toks = [syn.client_tokens(cfg, k) for k in range(K)]
    ctxs = [ctx_all[k * b:(k + 1) * b] for k in range(K)]
    mps = [mp_all[k * b:(k + 1) * b] for k in range(K)]
    labs = [syn.client_labels(toks[k], ctxs[k]) for k in range(K)]
    h0 = [torch.empty((b, L, cfg.hidden), dtype=torch.bfloat16, device="cuda") for L in cfg.seq_lens]
    for k in range(K):
        clients[k].bottom_forward(dev_i32(toks[k]), cfg.seq_lens[k], h0[k], ctxs[k], mps[k])
    hs = [torch.empty_like(x) for x in h0]
    srv.forward(h0, cfg.seq_lens, hs, context_lens=ctx_all, mask_pos=mp_all)
    losses = [torch.zeros(1, dtype=torch.float32, device="cuda") for _ in range(K)]
    gh = [torch.empty_like(x) for x in h0]
    for k in range(K):
        clients[k].top_forward_backward(hs[k], dev_i32(labs[k]), losses[k], gh[k])
    g0 = [torch.empty_like(x) for x in h0]
    srv.backward(gh, g0)
    for k in range(K):
        clients[k].bottom_backward(g0[k])
        clients[k].sync()
    srv.sync()
    # oracle: the same composition in fp64
    cp = syn.init_client(cfg)
    rcl = [O.OracleClient(c, cp) for c in ccfgs]
    rsrv = O.OracleServer(cfg)
    rh0 = [rcl[k].bottom_forward(toks[k], ctxs[k], mps[k]) for k in range(K)]
    rhs = rsrv.forward(rh0, ctx_all, mp_all)
    rtop = [rcl[k].top_forward_backward(rhs[k], labs[k]) for k in range(K)]
    rg0 = rsrv.backward([g for _, g in rtop])
    for k in range(K):
        rcl[k].bottom_backward(rg0[k])
        assert rel_inf(f64(h0[k]), rh0[k]) < OUT_TOL
        assert rel_inf(f64(hs[k]), rhs[k]) < OUT_TOL
        assert abs(losses[k].item() - rtop[k][0]) / rtop[k][0] < LOSS_TOL
        assert rel_inf(f64(gh[k]), rtop[k][1]) < GRAD_TOL
        assert rel_inf(f64(g0[k]), rg0[k]) < GRAD_TOL
        for part, t in part_tensors(cfg):
            e = rel_inf(clients[k].get_grad(PART_IDS[part], t), rcl[k].grads[part][t].reshape(-1))
            assert e < GRAD_TOL, ("client", k, part, t, e)
    for bb in range(cfg.n_blocks):
        for t in range(12):
            assert rel_inf(srv.get_grad(bb, t), rsrv.grads[bb][t].reshape(-1)) < GRAD_TOL, ("server", bb, t)
    # steps (each client against its oracle), then the end-of-period client averaging (§3.3)
    gref = [{(p, t): rcl[k].grads[p][t].reshape(-1).copy() for p, t in part_tensors(cfg)} for k in range(K)]
    for c in clients:
        c.step(cfg.lr)
    srv.step(cfg.lr)
    for k in range(K):
        rcl[k].step(cfg.lr)
        for part, t in part_tensors(cfg):
            w0 = np.asarray(cp[part][t], np.float32).reshape(-1)
            check_updated_weights(clients[k].get_param(PART_IDS[part], t), rcl[k].params[part][t].reshape(-1), w0,
                                  gref[k][(part, t)], cfg.lr, (k, part, t))
    before = {(p, t): [c.get_param(PART_IDS[p], t) for c in clients] for p, t in part_tensors(cfg)}
    F.fl_client_average(clients)
    inv = np.float32(1.0) / np.float32(K)
    for (p, t), ws in before.items():
        want = (ws[0] + ws[1]) * inv
        for c in clients:
            np.testing.assert_array_equal(c.get_param(PART_IDS[p], t), want)
    for c in clients:
        c.close()
    srv.close()


def test_client_average_is_the_mean(F):
    """fl_client_average writes the fp32 mean (summed in client order) into every client."""
    cfg = tiny_client()
    cls = [F.Client(F.make_client_cfg(cfg, cfg.tokens), s) for s in (1, 2, 3)]
    before = {(p, t): [c.get_param(PART_IDS[p], t) for c in cls] for p, t in part_tensors(cfg)}
    F.fl_client_average(cls)
    inv = np.float32(1.0) / np.float32(3.0)
    for (p, t), ws in before.items():
        want = ((ws[0] + ws[1]) + ws[2]) * inv
        for c in cls:
            np.testing.assert_array_equal(c.get_param(PART_IDS[p], t), want)
    with pytest.raises(F.FlError):
        F.fl_client_average([cls[0], cls[0]])
    for c in cls:
        c.close()


def test_client_errors(F):
    cfg = tiny_client()
    cl = F.Client(F.make_client_cfg(cfg, cfg.tokens), 0)
    b, L, H = 2, 64, cfg.hidden
    h = torch.zeros((b, L, H), dtype=torch.bfloat16, device="cuda")
    loss = torch.zeros(1, dtype=torch.float32, device="cuda")
    labels = dev_i32(np.full((b, L), -1, np.int32))
    with pytest.raises(F.FlError) as ei:        # top before bottom
        cl.top_forward_backward(h, labels, loss, h)
    assert ei.value.code == -3
    with pytest.raises(F.FlError) as ei:        # too many tokens
        cl.bottom_forward(dev_i32(np.zeros((b, 65), np.int32)), 65, h)
    assert ei.value.code == -1
    bad = np.zeros((b, L), np.int32)
    bad[1, 5] = cfg.vocab                       # out-of-range token: embeds as zeros, reported at sync
    cl.bottom_forward(dev_i32(bad), L, h)
    with pytest.raises(F.FlError) as ei:
        cl.bottom_forward(dev_i32(bad), L, h)   # round already open
    assert ei.value.code == -3
    with pytest.raises(F.FlError) as ei:
        cl.sync()
    assert ei.value.code == -1
    lab = np.full((b, L), -1, np.int32)
    lab[0, 3] = cfg.vocab + 7                   # label >= vocab: ignored, reported
    cl.top_forward_backward(h, dev_i32(lab), loss, h)
    with pytest.raises(F.FlError) as ei:
        cl.sync()
    assert ei.value.code == -1
    assert float(loss.item()) == 0.0            # no valid target: zero loss
    cl.bottom_backward(h)
    cl.step(1e-3)
    cl.sync()
    cl.close()


@pytest.mark.slow
def test_client_chatglm6b_shapes(F):
    """The ChatGLM-6B client: H 4096, 32 x 128 heads, FFN 16384, vocabulary 130528 (head
    padded to 130560), one GLM row of 96 tokens, all client parameters trained."""
    cfg = syn._glm("client6b", 1, 1, 1, (96,)).with_(vocab=syn.CHATGLM6B_VOCAB, lr=1e-4)
    rng = np.random.default_rng(6)

    def draw(shape):
        return (0.02 * rng.standard_normal(shape, dtype=np.float32))

    params = {}
    for part in ("bottom", "top"):
        ts = [draw(s) for s in syn.param_shapes(cfg)]
        for t in (syn.T_G1, syn.T_G2):
            ts[t] = 1.0 + ts[t]
        params[part] = ts
    params["embed"] = [draw((cfg.vocab, cfg.hidden))]
    params["head"] = [draw((cfg.vocab, cfg.hidden))]
    params["final_ln"] = [1.0 + draw(cfg.hidden), draw(cfg.hidden)]
    client_round(F, cfg, ctx=[70], mp=[69], check_step=False, params=params)


@pytest.mark.parametrize("V,ld", [(1000, 1024), (130528, 130560), (5, 8)])
def test_cross_entropy_kernel(F, V, ld):
    """The row kernel against the oracle: loss, per-row losses and the logit gradient,
    ragged vocabulary tails, padded columns zero, rows without a target."""
    rng = np.random.default_rng(V)
    T = 37
    logits = np.zeros((T, ld), np.float32)
    logits[:, :V] = (2.0 * rng.standard_normal((T, V))).astype(np.float32)
    labels = rng.integers(0, V, size=T).astype(np.int32)
    labels[[0, 9, 30]] = -1
    dl = torch.from_numpy(logits).cuda()
    row = torch.empty(T, dtype=torch.float32, device="cuda")
    dlog = torch.full((T, ld), 7.0, dtype=torch.bfloat16, device="cuda")
    loss = torch.empty(1, dtype=torch.float32, device="cuda")
    cnt = torch.empty(1, dtype=torch.int32, device="cuda")
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    F.fl_k_cross_entropy(T, V, ld, dl, dev_i32(labels), row, dlog, loss, cnt, st)
    torch.cuda.synchronize()
    ref_loss, ref_d = O.cross_entropy(logits[:, :V].astype(np.float64), labels)
    assert int(cnt.item()) == T - 3 and int(st.item()) == 0
    assert abs(loss.item() - ref_loss) / ref_loss < 1e-5
    got = f64(dlog)
    assert not got[:, V:].any()
    assert rel_inf(got[:, :V], ref_d) < 1e-2        # bf16 gradient
    assert not got[[0, 9, 30]].any()


def test_embedding_kernels(F):
    rng = np.random.default_rng(5)
    V, H, T = 300, 256, 77
    table = rng.standard_normal((V, H)).astype(np.float32)
    tb = syn.bf16_bits_to_f32(syn.f32_to_bf16_bits(table))
    tokens = rng.integers(0, V, size=T).astype(np.int32)
    tokens[[3, 4]] = tokens[2]                      # repeated ids: their gradients add up
    tokens[10] = V                                  # out of range: zero row, flagged
    out = torch.empty((T, H), dtype=torch.bfloat16, device="cuda")
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    F.fl_k_embedding_gather(T, H, dev_i32(tokens), bf16_dev(tb), V, out, st)
    dx = rng.standard_normal((T, H))
    dxb = syn.bf16_bits_to_f64(syn.f32_to_bf16_bits(dx.astype(np.float32)))
    dE = torch.zeros((V, H), dtype=torch.float32, device="cuda")
    F.fl_k_embedding_scatter_add(T, H, dev_i32(tokens), V, bf16_dev(dxb), dE)
    torch.cuda.synchronize()
    ok = tokens < V
    want = np.zeros((T, H))
    want[ok] = tb[tokens[ok]]
    np.testing.assert_array_equal(f64(out), want)
    assert int(st.item()) == 1
    np.testing.assert_allclose(f64(dE), O.embedding_bwd(dxb[ok], tokens[ok], V), rtol=1e-6, atol=1e-5)
