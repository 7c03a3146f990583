"""GLM blank-infilling segments on the GPU (§4.1.1 casts every task as GLM blank infilling):
a bidirectional context holding the mask token, a causal answer span after it, and GLM's
two position streams (the second rotating the second half of each head).  Kernel-level
and server-level parity against the fp64 oracle (GPU only)."""
import numpy as np
import pytest
import torch

import synthetic as syn
from oracle import flglm_oracle as O
from tests._gpu import (bits, dev_bf16, dev_bf16_from_bits, dev_f32, dev_i32, f64, flglm, need_gpu,
                        rel_inf, rnd_bf16_f64, rope_table)
from tests.test_gpu_server import GRAD_TOL, OUT_TOL, check_updated_weights

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def F():
    need_gpu()
    return flglm()


# segments that put the end of the context everywhere that matters: one token, a whole
# tile, inside a tile, across a tile edge, 0 (plain causal), exactly on a tile edge, the
# whole multi-tile segment
SEQS = [1, 64, 100, 130, 7, 64, 200, 129]
CTX = [1, 64, 37, 70, 0, 1, 200, 128]
MPOS = [0, 10, 36, 5, 0, 0, 199, 64]


@pytest.mark.parametrize("hd", [64, 128])
@pytest.mark.parametrize("Lp", [0, 40])
def test_attention_glm(F, hd, Lp):
    nh = 2
    H = nh * hd
    cu = np.cumsum([0] + SEQS).astype(np.int32)
    T = int(cu[-1])
    rng = np.random.default_rng(hd + Lp)
    qkv = rnd_bf16_f64(rng, (T, 3 * H))
    do = rnd_bf16_f64(rng, (T, H))
    pk = pv = None
    kw = {}
    if Lp:
        pk = rnd_bf16_f64(rng, (Lp, H))
        pv = rnd_bf16_f64(rng, (Lp, H))
        kw = dict(prefix_k=dev_bf16(pk), prefix_v=dev_bf16(pv), prefix_len=Lp)
    dqkv_ = dev_bf16(qkv)
    dcu = dev_i32(cu)
    dctx = dev_i32(CTX)
    tiles = torch.empty(F.fl_k_attention_tiles(cu) * 2, dtype=torch.int32, device="cuda")
    o = torch.full((T, H), float("nan"), dtype=torch.bfloat16, device="cuda")
    lse = torch.empty((nh, T), dtype=torch.float32, device="cuda")
    F.fl_k_attention_fwd(T, nh, hd, dqkv_, cu, dcu, tiles, o, lse, context_lens=dctx, **kw)
    torch.cuda.synchronize()
    q = qkv[:, :H].reshape(T, nh, hd)
    k = qkv[:, H:2 * H].reshape(T, nh, hd)
    v = qkv[:, 2 * H:].reshape(T, nh, hd)
    ppk = None if pk is None else pk.reshape(Lp, nh, hd)
    ppv = None if pv is None else pv.reshape(Lp, nh, hd)
    o_ref, lse_ref = O.attention_fwd(q, k, v, cu, ppk, ppv, ctx=np.array(CTX))
    assert rel_inf(f64(o), o_ref.reshape(T, H)) < 2e-2
    np.testing.assert_allclose(f64(lse), lse_ref, rtol=0, atol=2e-2)
    # backward with GLM's two position streams folded into the inverse rotation
    rd = hd // 2
    pkg = O.make_packing(SEQS, 1, CTX, MPOS)
    tab = rope_table(256, rd, 10000.0)
    delta = torch.empty((nh, T), dtype=torch.float32, device="cuda")
    dq = torch.full((T, 3 * H), float("nan"), dtype=torch.bfloat16, device="cuda")
    dpk = dpv = None
    if Lp:
        dpk = torch.zeros((Lp, H), dtype=torch.float32, device="cuda")
        dpv = torch.zeros((Lp, H), dtype=torch.float32, device="cuda")
        kw.update(dprefix_k=dpk, dprefix_v=dpv)
    F.fl_k_attention_bwd(T, nh, hd, dqkv_, o, lse, dev_bf16(do), cu, dcu, tiles, delta, dev_f32(tab), rd, dq,
                         context_lens=dctx, positions=dev_i32(pkg.pos), block_positions=dev_i32(pkg.pos2), **kw)
    torch.cuda.synchronize()
    res = O.attention_bwd(do.reshape(T, nh, hd), q, k, v, cu, ppk, ppv, ctx=np.array(CTX))
    dq_ref = O.rope_2d(res[0], pkg, rd, 10000.0, inverse=True).reshape(T, H)
    dk_ref = O.rope_2d(res[1], pkg, rd, 10000.0, inverse=True).reshape(T, H)
    got = f64(dq)
    assert rel_inf(got[:, :H], dq_ref) < 5e-2
    assert rel_inf(got[:, H:2 * H], dk_ref) < 5e-2
    assert rel_inf(got[:, 2 * H:], res[2].reshape(T, H)) < 5e-2
    if Lp:
        assert rel_inf(f64(dpk), res[3].reshape(Lp, H)) < 5e-2
        assert rel_inf(f64(dpv), res[4].reshape(Lp, H)) < 5e-2


@pytest.mark.parametrize("hd", [64, 128])
def test_gemm_rope_2d_epilogue(F, hd):
    """The QKV GEMM epilogue turns dims [0, hd/2) by the position and [hd/2, hd) by the
    block position (ChatGLM's 2D rotary)."""
    nh = 2
    H = nh * hd
    M, N, K = 130, 3 * H, 256
    rng = np.random.default_rng(hd + 1)
    A = rnd_bf16_f64(rng, (M, K))
    B = rnd_bf16_f64(rng, (N, K), 0.1)
    bias = rng.standard_normal(N).astype(np.float32)
    pos = rng.integers(0, 300, size=M).astype(np.int32)
    pos2 = rng.integers(0, 300, size=M).astype(np.int32)
    rd = hd // 2
    tab = rope_table(300, rd, 10000.0)
    D = torch.empty((M, N), dtype=torch.bfloat16, device="cuda")
    F.gemm(M, N, K, dev_bf16(A), K, 0, dev_bf16(B), K, 0, D, N, epilogue=F.FL_EPI_BIAS_ROPE, bias=dev_f32(bias),
           pos=dev_i32(pos), pos2=dev_i32(pos2), rope_tab=dev_f32(tab), n_heads=nh, head_dim=hd, rotary_dim=rd)
    torch.cuda.synchronize()
    qkv = A @ B.T + bias[None, :]
    pkg = O.Packing(np.array([0, M], np.int32), pos, np.zeros(1, np.int32), np.zeros(1, np.int32),
                    np.array([1], np.int32), pos2)
    q = O.rope_2d(qkv[:, :H].reshape(M, nh, hd), pkg, rd, 10000.0).reshape(M, H)
    k = O.rope_2d(qkv[:, H:2 * H].reshape(M, nh, hd), pkg, rd, 10000.0).reshape(M, H)
    ref = np.concatenate([q, k, qkv[:, 2 * H:]], axis=1)
    assert rel_inf(f64(D), ref) < 1e-2
    # block position 0 everywhere: bit-identical to the 1D epilogue
    D0 = torch.empty_like(D)
    D1 = torch.empty_like(D)
    common = dict(epilogue=F.FL_EPI_BIAS_ROPE, bias=dev_f32(bias), pos=dev_i32(pos), rope_tab=dev_f32(tab),
                  n_heads=nh, head_dim=hd, rotary_dim=rd)
    F.gemm(M, N, K, dev_bf16(A), K, 0, dev_bf16(B), K, 0, D0, N, pos2=dev_i32(np.zeros(M, np.int32)), **common)
    F.gemm(M, N, K, dev_bf16(A), K, 0, dev_bf16(B), K, 0, D1, N, **common)
    torch.cuda.synchronize()
    np.testing.assert_array_equal(bits(D0), bits(D1))


def glm_case(F, cfg, ctx, mp, fused=False, check_grads=True):
    """Server forward/backward(/step) with GLM segments against the oracle server."""
    params = syn.init_params(cfg)
    prefixes = [syn.init_prefix(cfg, b) for b in range(cfg.n_blocks)] if cfg.prefix_len else None
    srv = F.Server(F.make_cfg(cfg, cfg.tokens, fused_step_min_tokens=1), cfg.seed)
    for b in range(cfg.n_blocks):
        for t in range(12):
            srv.set_param(b, t, params[b][t])
        if prefixes:
            srv.set_param(b, F.FL_T_PREFIX_K, prefixes[b][0])
            srv.set_param(b, F.FL_T_PREFIX_V, prefixes[b][1])
    states, grads = syn.client_states(cfg), syn.client_grads(cfg)
    st = [dev_bf16_from_bits(s) for s in states]
    outs = [torch.empty_like(s) for s in st]
    gi = [torch.empty_like(s) for s in st]
    srv.forward(st, cfg.seq_lens, outs, context_lens=ctx, mask_pos=mp)
    go = [dev_bf16_from_bits(g) for g in grads]
    ref = O.OracleServer(cfg, params, prefixes)
    ro = ref.forward([syn.bf16_bits_to_f64(s) for s in states], ctx, mp)
    rg = ref.backward([syn.bf16_bits_to_f64(g) for g in grads])
    gref = [[g.reshape(-1).copy() for g in blk] for blk in ref.grads]
    n_t = 14 if cfg.prefix_len else 12
    trained = [t for t in range(n_t) if not (cfg.freeze_base and t < 12)]
    if fused:
        srv.backward_step(go, gi, cfg.lr)
    else:
        srv.backward(go, gi)
        srv.sync()
        if check_grads:
            for b in range(cfg.n_blocks):
                for t in trained:
                    e = rel_inf(srv.get_grad(b, t), gref[b][t])
                    assert e < GRAD_TOL, ("wgrad", b, t, e)
        srv.step(cfg.lr)
    srv.sync()
    for k in range(cfg.K):
        assert rel_inf(f64(outs[k]), ro[k]) < OUT_TOL, ("out", k, rel_inf(f64(outs[k]), ro[k]))
        assert rel_inf(f64(gi[k]), rg[k]) < GRAD_TOL, ("grad_in", k, rel_inf(f64(gi[k]), rg[k]))
    ref.step(cfg.lr)
    for b in range(cfg.n_blocks):
        for t in range(n_t):
            w0 = (params[b][t] if t < 12 else prefixes[b][t - 12]).reshape(-1)
            w = srv.get_param(b, t)
            if t not in trained:
                np.testing.assert_array_equal(w, w0)
            else:
                check_updated_weights(w, ref.params[b][t].reshape(-1), w0, gref[b][t], cfg.lr, (b, t))
    srv.close()


@pytest.mark.parametrize("rfl", [1, 0], ids=["glm_block", "pre_ln"])
@pytest.mark.parametrize("fused", [False, True], ids=["step", "backward_step"])
def test_tiny_glm_parity(F, rfl, fused):
    cfg = syn.CONFIGS["tiny"].with_(residual_from_ln=rfl)
    ctx, mp = syn.glm_structure(cfg)
    glm_case(F, cfg, ctx, mp, fused=fused)


def test_ragged_glm_edge_segments(F):
    """Two blocks, ragged segments whose contexts end inside, on and across tile edges,
    plain causal (0) and whole-segment (L) contexts, default [M] position."""
    cfg = syn.CONFIGS["tiny"].with_(n_blocks=2, client_batch=1, seq_lens=(1, 64, 100, 130, 7, 129), lr=1e-3)
    glm_case(F, cfg, [1, 64, 37, 70, 0, 128], None)


@pytest.mark.parametrize("fused", [False, True], ids=["step", "backward_step"])
def test_ptuning_glm_parity(F, fused):
    """The paper's training setting end to end: GLM blank-infilling segments, P-tuning v2
    prefixes, frozen block weights."""
    cfg = syn.CONFIGS["tiny"].with_(n_blocks=2, client_batch=2, seq_lens=(64, 90), prefix_len=20, freeze_base=1,
                                    lr=1e-3)
    ctx, mp = syn.glm_structure(cfg)
    glm_case(F, cfg, ctx, mp, fused=fused)


def test_block6b_glm_parity(F):
    """One ChatGLM-6B-shaped block (H 4096, 32 x 128), K = 4 x 512 tokens, GLM segments."""
    cfg = syn.CONFIGS["block6b"]
    ctx, mp = syn.glm_structure(cfg)
    glm_case(F, cfg, ctx, mp)


def test_glm_batching_invariant_bitexact(F):
    """Stacking GLM segments does not mix them: each client's outputs and input gradients
    from the packed call equal, bit for bit, those of that client alone."""
    cfg = syn.CONFIGS["tiny"].with_(n_blocks=2, client_batch=2, seq_lens=(64, 20, 130))
    ctx, mp = syn.glm_structure(cfg)
    states, grads = syn.client_states(cfg), syn.client_grads(cfg)

    def run(c, st_bits, g_bits, cl, mpl, max_tokens):
        srv = F.Server(F.make_cfg(c, max_tokens, fused_step_min_tokens=1), cfg.seed)
        st = [dev_bf16_from_bits(s) for s in st_bits]
        outs = [torch.empty_like(s) for s in st]
        srv.forward(st, c.seq_lens, outs, context_lens=cl, mask_pos=mpl)
        gi = [torch.empty_like(s) for s in st]
        srv.backward([dev_bf16_from_bits(g) for g in g_bits], gi)
        srv.sync()
        srv.close()
        return [bits(o) for o in outs], [bits(g) for g in gi]

    outs, gins = run(cfg, states, grads, ctx, mp, cfg.tokens)
    b = cfg.client_batch
    for k in range(cfg.K):
        c1 = cfg.with_(seq_lens=(cfg.seq_lens[k],))
        o1, g1 = run(c1, [states[k]], [grads[k]], ctx[k * b:(k + 1) * b], mp[k * b:(k + 1) * b], cfg.tokens)
        np.testing.assert_array_equal(o1[0], outs[k])
        np.testing.assert_array_equal(g1[0], gins[k])


def test_glm_argument_errors(F):
    cfg = syn.CONFIGS["tiny"]
    srv = F.Server(F.make_cfg(cfg, cfg.tokens, fused_step_min_tokens=1), cfg.seed)
    st = [torch.zeros((2, 64, 256), dtype=torch.bfloat16, device="cuda")]
    for ctx, mp in [([65, 1], None), ([-1, 1], None), ([10, 4], [10, 0]), ([10, 4], [-1, 0])]:
        with pytest.raises(F.FlError) as ei:
            srv.forward(st, [64], st, context_lens=ctx, mask_pos=mp)
        assert ei.value.code == -1, (ctx, mp)
    srv.forward(st, [64], st, context_lens=[64, 0])    # whole-context and plain segments are valid
    srv.backward(st, st)
    srv.sync()
    srv.close()


def test_glm_prefix_parity_vs_fp32_oracle(F):
    """GLM segments with P-tuning v2 prefixes, two blocks, against the fp32 C++ oracle:
    outputs, input gradients, the 12 weight gradients and the prefix key / value gradients
    of every block."""
    from oracle import oracle32 as O32
    cfg = syn.CONFIGS["tiny"].with_(n_blocks=2, client_batch=2, seq_lens=(64, 90), prefix_len=20)
    ctx, mp = syn.glm_structure(cfg)
    params = syn.init_params(cfg)
    prefixes = [syn.init_prefix(cfg, b) for b in range(cfg.n_blocks)]
    srv = F.Server(F.make_cfg(cfg, cfg.tokens), cfg.seed)
    for b in range(cfg.n_blocks):
        for t in range(12):
            srv.set_param(b, t, params[b][t])
        srv.set_param(b, F.FL_T_PREFIX_K, prefixes[b][0])
        srv.set_param(b, F.FL_T_PREFIX_V, prefixes[b][1])
    states, grads = syn.client_states(cfg), syn.client_grads(cfg)
    st = [dev_bf16_from_bits(s) for s in states]
    outs = [torch.empty_like(s) for s in st]
    gi = [torch.empty_like(s) for s in st]
    srv.forward(st, cfg.seq_lens, outs, context_lens=ctx, mask_pos=mp)
    srv.backward([dev_bf16_from_bits(g) for g in grads], gi)
    srv.sync()
    H = cfg.hidden
    x = np.concatenate([syn.bf16_bits_to_f64(s).reshape(-1, H) for s in states])
    dy = np.concatenate([syn.bf16_bits_to_f64(g).reshape(-1, H) for g in grads])
    cu = np.concatenate([[0], np.cumsum([L for L in cfg.seq_lens for _ in range(cfg.client_batch)])])
    g32 = [[np.zeros(p.shape, np.float32) for p in blk] for blk in params]
    pg32 = [[np.zeros(np.shape(p), np.float32) for p in pre] for pre in prefixes]
    y, dx = O32.server_fwd_bwd(cfg, params, g32, cu, x, dy, ctx, mp, prefixes, pg32)
    y_gpu = np.concatenate([f64(o).reshape(-1, H) for o in outs])
    dx_gpu = np.concatenate([f64(g).reshape(-1, H) for g in gi])
    assert rel_inf(y_gpu, y) < OUT_TOL, rel_inf(y_gpu, y)
    assert rel_inf(dx_gpu, dx) < GRAD_TOL, rel_inf(dx_gpu, dx)
    for b in range(cfg.n_blocks):
        for t in range(12):
            e = rel_inf(srv.get_grad(b, t), g32[b][t].reshape(-1))
            assert e < GRAD_TOL, ("wgrad", b, syn.TENSOR_NAMES[t], e)
        for j, tid in enumerate((F.FL_T_PREFIX_K, F.FL_T_PREFIX_V)):
            e = rel_inf(srv.get_grad(b, tid), pg32[b][j].reshape(-1))
            assert e < GRAD_TOL, ("prefix grad", b, j, e)
    srv.close()
