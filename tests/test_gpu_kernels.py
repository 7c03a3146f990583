"""Kernel-level parity of the CUDA library against the fp64 oracle (GPU only).

Each test calls one kernel through the C ABI of include/flglm_kernels.h on seeded
inputs that are exactly representable in bf16, and compares with the oracle's
function of the same step (or, for the plain contractions, with the fp64 product
that defines them).  Shapes span several tiles and a ragged tail.
"""

import numpy as np
import pytest
import torch

from oracle import flglm_oracle as O
from tests._gpu import (bits, dev_bf16, dev_f32, dev_i32, f64, flglm, need_gpu, rel_inf, rnd_bf16_f64,
                        rope_table)

pytestmark = pytest.mark.gpu

# bf16 output rounding is 2^-9 relative; fp32 accumulation over K adds far less.
GEMM_TOL = 1e-2


@pytest.fixture(scope="module")
def F():
    need_gpu()
    return flglm()


def _store(mat: np.ndarray, mn_major: bool):
    """Device copy of a logical [rows, K] operand: row-major as is (K-major), or its
    transpose [K, rows] (MN-major).  Returns (tensor, leading dim)."""
    if mn_major:
        t = dev_bf16(np.ascontiguousarray(mat.T))
        return t, mat.shape[0]
    return dev_bf16(mat), mat.shape[1]


TILES = ["auto", "128x128", "128x256", "pair"]


def tile_id(F, name):
    return {"auto": F.FL_TILE_AUTO, "128x128": F.FL_TILE_128x128, "128x256": F.FL_TILE_128x256,
            "pair": F.FL_TILE_256x256_PAIR}[name]


@pytest.mark.parametrize("tile", TILES)
@pytest.mark.parametrize("layout", [(0, 0), (0, 1), (1, 1)], ids=["fwd", "dgrad", "wgrad"])
@pytest.mark.parametrize("shape", [(200, 256, 320), (136, 384, 200), (1000, 1024, 512), (64, 128, 64),
                                   (8, 256, 4096), (520, 768, 72), (104, 512, 256), (4000, 4096, 520)])
def test_gemm_layouts(F, layout, shape, tile):
    """Every operand layout and tile shape.  (104, 512, 256): the odd CTA of a pair loads
    rows wholly past M; (4000, 4096, 520): several 256 x 256 tiles per CTA pair, so both
    accumulator buffers and the 6-stage ring wrap, with a ragged last k-block."""
    M, N, K = shape
    a_mn, b_mn = layout
    if tile in ("128x256", "pair") and N % 256:
        pytest.skip("256-column tiles need N % 256 == 0")
    rng = np.random.default_rng(M * 7 + N + K + 31 * a_mn + 17 * b_mn)
    A = rnd_bf16_f64(rng, (M, K))
    B = rnd_bf16_f64(rng, (N, K))
    dA, lda = _store(A, bool(a_mn))
    dB, ldb = _store(B, bool(b_mn))
    D = torch.full((M, N), float("nan"), dtype=torch.bfloat16, device="cuda")
    F.gemm(M, N, K, dA, lda, a_mn, dB, ldb, b_mn, D, N, tile=tile_id(F, tile))
    torch.cuda.synchronize()
    ref = A @ B.T
    assert rel_inf(f64(D), ref) < GEMM_TOL


def test_gemm_accumulate_f32_repeated(F):
    """fp32 read-modify-write epilogue (weight gradients accumulate across calls)."""
    M, N, K = 384, 512, 300
    rng = np.random.default_rng(5)
    A = rnd_bf16_f64(rng, (M, K))
    B = rnd_bf16_f64(rng, (N, K))
    C0 = rng.standard_normal((M, N)).astype(np.float32)
    dA, lda = _store(A, True)
    dB, ldb = _store(B, True)
    D = dev_f32(C0)
    for _ in range(2):
        F.gemm(M, N, K, dA, lda, 1, dB, ldb, 1, D, N, epilogue=F.FL_EPI_ACCUM_F32)
    torch.cuda.synchronize()
    ref = C0.astype(np.float64) + 2 * (A @ B.T)
    assert rel_inf(f64(D), ref) < 1e-5


@pytest.mark.parametrize("tile", ["auto", "pair"])
def test_gemm_epilogues(F, tile):
    M, N, K = 192, 512, 256
    t = tile_id(F, tile)
    rng = np.random.default_rng(11)
    A = rnd_bf16_f64(rng, (M, K))
    B = rnd_bf16_f64(rng, (N, K), 0.1)
    bias = rng.standard_normal(N).astype(np.float32)
    R = rnd_bf16_f64(rng, (M, N))
    dA, lda = _store(A, False)
    dB, ldb = _store(B, False)
    db = dev_f32(bias)
    dR = dev_bf16(R)
    acc = A @ B.T
    alpha = 1.7
    # bias + gelu, pre-activation kept
    D = torch.empty((M, N), dtype=torch.bfloat16, device="cuda")
    U = torch.empty((M, N), dtype=torch.bfloat16, device="cuda")
    F.gemm(M, N, K, dA, lda, 0, dB, ldb, 0, D, N, tile=t, epilogue=F.FL_EPI_BIAS_GELU, bias=db, aux_out=U, ld_aux_out=N)
    torch.cuda.synchronize()
    u = acc + bias[None, :]
    assert rel_inf(f64(U), u) < GEMM_TOL
    assert rel_inf(f64(D), O.gelu(u)) < GEMM_TOL
    # bias + alpha * residual
    F.gemm(M, N, K, dA, lda, 0, dB, ldb, 0, D, N, tile=t, epilogue=F.FL_EPI_BIAS_RESID, bias=db, aux=dR, ld_aux=N,
           alpha=alpha)
    torch.cuda.synchronize()
    assert rel_inf(f64(D), u + alpha * R) < GEMM_TOL
    # alpha * residual, no bias
    F.gemm(M, N, K, dA, lda, 0, dB, ldb, 0, D, N, tile=t, epilogue=F.FL_EPI_RESID, aux=dR, ld_aux=N, alpha=alpha)
    torch.cuda.synchronize()
    assert rel_inf(f64(D), acc + alpha * R) < GEMM_TOL
    # gelu' of a stored pre-activation; its column sums added to a vector (the up-projection
    # bias gradient of the backward)
    c0 = rng.standard_normal(N).astype(np.float32)
    cs = dev_f32(c0)
    F.gemm(M, N, K, dA, lda, 0, dB, ldb, 0, D, N, tile=t, epilogue=F.FL_EPI_GELU_BWD, aux=dR, ld_aux=N, colsum=cs)
    torch.cuda.synchronize()
    du = acc * O.gelu_grad(R)
    assert rel_inf(f64(D), du) < GEMM_TOL
    assert rel_inf(f64(cs) - c0, du.sum(axis=0)) < 1e-4
    # plain store with bias
    F.gemm(M, N, K, dA, lda, 0, dB, ldb, 0, D, N, tile=t, epilogue=F.FL_EPI_STORE, bias=db)
    torch.cuda.synchronize()
    assert rel_inf(f64(D), u) < GEMM_TOL


@pytest.mark.parametrize("tile", ["auto", "pair"])
@pytest.mark.parametrize("hd", [64, 128])
def test_gemm_rope_epilogue(F, hd, tile):
    nh = 2
    H = nh * hd
    M, N, K = 130, 3 * H, 256
    if tile == "pair" and N % 256:
        pytest.skip("256-column tiles need N % 256 == 0")
    rng = np.random.default_rng(hd)
    A = rnd_bf16_f64(rng, (M, K))
    B = rnd_bf16_f64(rng, (N, K), 0.1)
    bias = rng.standard_normal(N).astype(np.float32)
    pos = rng.integers(0, 300, size=M).astype(np.int32)
    rd = hd // 2
    tab = rope_table(300, rd, 10000.0)
    dA, lda = _store(A, False)
    dB, ldb = _store(B, False)
    D = torch.empty((M, N), dtype=torch.bfloat16, device="cuda")
    F.gemm(M, N, K, dA, lda, 0, dB, ldb, 0, D, N, epilogue=F.FL_EPI_BIAS_ROPE, bias=dev_f32(bias),
           pos=dev_i32(pos), rope_tab=dev_f32(tab), n_heads=nh, head_dim=hd, rotary_dim=rd, tile=tile_id(F, tile))
    torch.cuda.synchronize()
    qkv = A @ B.T + bias[None, :]
    cos, sin = O.rope_cos_sin(pos, rd, 10000.0)
    q = O.rope_rotate(qkv[:, :H].reshape(M, nh, hd), cos, sin, rd).reshape(M, H)
    k = O.rope_rotate(qkv[:, H:2 * H].reshape(M, nh, hd), cos, sin, rd).reshape(M, H)
    ref = np.concatenate([q, k, qkv[:, 2 * H:]], axis=1)
    assert rel_inf(f64(D), ref) < GEMM_TOL


@pytest.mark.parametrize("H", [256, 768, 3072, 4096])  # 768: one chunk per thread; 3072: six warps
@pytest.mark.parametrize("dtype", ["bf16", "f32"])
def test_layernorm_fwd_bwd(F, H, dtype):
    T = 77
    rng = np.random.default_rng(H + (dtype == "f32"))
    if dtype == "f32":
        x = (2.0 * rng.standard_normal((T, H))).astype(np.float32).astype(np.float64)
        dev_io = dev_f32
        dt = F.FL_DT_F32
    else:
        x = rnd_bf16_f64(rng, (T, H), 2.0)
        dev_io = dev_bf16
        dt = F.FL_DT_BF16
    g = (1 + 0.2 * rng.standard_normal(H)).astype(np.float32)
    be = (0.2 * rng.standard_normal(H)).astype(np.float32)
    dx_, dg_, db_ = dev_io(x), dev_f32(g), dev_f32(be)
    y = torch.empty((T, H), dtype=torch.bfloat16, device="cuda")
    mean = torch.empty(T, dtype=torch.float32, device="cuda")
    rstd = torch.empty(T, dtype=torch.float32, device="cuda")
    F.fl_k_layernorm_fwd(T, H, dx_, dg_, db_, 1e-5, y, mean, rstd, x_dtype=dt)
    torch.cuda.synchronize()
    yr, mur, rsr = O.layer_norm_fwd(x, g.astype(np.float64), be.astype(np.float64), 1e-5)
    assert rel_inf(f64(y), yr) < 1e-2
    np.testing.assert_allclose(f64(mean), mur, rtol=0, atol=1e-5)
    np.testing.assert_allclose(f64(rstd), rsr, rtol=1e-4)
    # backward, with and without the alpha-scaled residual gradient; bf16 and fp32 dx
    if dtype == "f32":
        dy = rng.standard_normal((T, H)).astype(np.float32).astype(np.float64)
        res = rng.standard_normal((T, H)).astype(np.float32).astype(np.float64)
    else:
        dy = rnd_bf16_f64(rng, (T, H))
        res = rnd_bf16_f64(rng, (T, H))
    ws = torch.empty(F.fl_k_layernorm_bwd_workspace(T, H) // 4 + 64, dtype=torch.float32, device="cuda")
    for use_res in (False, True):
        dxo = torch.empty((T, H), dtype=torch.bfloat16, device="cuda")
        dxf = torch.empty((T, H), dtype=torch.float32, device="cuda")
        dgam = dev_f32(np.full(H, 0.5, np.float32))
        dbet = dev_f32(np.full(H, -0.25, np.float32))
        F.fl_k_layernorm_bwd(T, H, dev_io(dy), dx_, mean, rstd, dg_, dev_io(res) if use_res else None, 3.0,
                             dxo, dgam, dbet, ws, io_dtype=dt, dx_f32=dxf)
        torch.cuda.synchronize()
        dxr, dgr, dbr = O.layer_norm_bwd(dy, x, mur, rsr, g.astype(np.float64))
        if use_res:
            dxr = dxr + 3.0 * res
        assert rel_inf(f64(dxo), dxr) < 1e-2
        assert rel_inf(f64(dxf), dxr) < 1e-4
        assert rel_inf(f64(dgam) - 0.5, dgr) < 1e-4
        assert rel_inf(f64(dbet) + 0.25, dbr) < 1e-4


def test_layernorm_unsupported_widths(F):
    """Hidden sizes the forward has no launch shape for (an odd multiple of 256 above 2048, a
    width not a multiple of 256) and a negative row count are refused before any launch."""
    H = 2304
    x = torch.zeros((4, 4096), dtype=torch.bfloat16, device="cuda")
    v = torch.zeros(4096, device="cuda")
    y = torch.full((4, 4096), 1.0, dtype=torch.bfloat16, device="cuda")
    st = torch.zeros(4, device="cuda")
    for h, code in ((H, -7), (200, -7)):
        with pytest.raises(F.FlError) as ei:
            F.fl_k_layernorm_fwd(4, h, x, v, v, 1e-5, y, st, st)
        assert ei.value.code == code
    with pytest.raises(F.FlError) as ei:
        F.fl_k_layernorm_fwd(-1, 256, x, v, v, 1e-5, y, st, st)
    assert ei.value.code == -1
    torch.cuda.synchronize()
    assert (y == 1.0).all() and not st.any()


@pytest.mark.parametrize("tile", ["auto", "pair"])
def test_gemm_fp32_residual_epilogues(F, tile):
    """fp32 residual stream: D fp32 = acc + bias + alpha * R, with R an fp32 tensor or its
    LayerNorm recomputed in fp32 from the row statistics."""
    M, N, K = 200, 512, 256
    t = tile_id(F, tile)
    rng = np.random.default_rng(12)
    A = rnd_bf16_f64(rng, (M, K))
    B = rnd_bf16_f64(rng, (N, K), 0.1)
    bias = rng.standard_normal(N).astype(np.float32)
    X = (3.0 * rng.standard_normal((M, N)) + 0.5).astype(np.float32)
    g = (1 + 0.2 * rng.standard_normal(N)).astype(np.float32)
    be = (0.2 * rng.standard_normal(N)).astype(np.float32)
    _, mu, rs = O.layer_norm_fwd(X.astype(np.float64), g.astype(np.float64), be.astype(np.float64), 1e-5)
    dA, lda = _store(A, False)
    dB, ldb = _store(B, False)
    acc = A @ B.T
    D = torch.empty((M, N), dtype=torch.float32, device="cuda")
    dX = dev_f32(X)
    F.gemm(M, N, K, dA, lda, 0, dB, ldb, 0, D, N, tile=t, epilogue=F.FL_EPI_BIAS_RESID, bias=dev_f32(bias), aux=dX, ld_aux=N,
           alpha=7.5, aux_dtype=F.FL_DT_F32, d_dtype=F.FL_DT_F32)
    torch.cuda.synchronize()
    assert rel_inf(f64(D), acc + bias[None, :] + 7.5 * X) < 1e-5
    F.gemm(M, N, K, dA, lda, 0, dB, ldb, 0, D, N, tile=t, epilogue=F.FL_EPI_BIAS_RESID, bias=dev_f32(bias), aux=dX, ld_aux=N,
           alpha=7.5, aux_dtype=F.FL_DT_F32, d_dtype=F.FL_DT_F32, ln_mean=dev_f32(mu), ln_rstd=dev_f32(rs),
           ln_gamma=dev_f32(g), ln_beta=dev_f32(be))
    torch.cuda.synchronize()
    lnx = (X - mu[:, None]) * rs[:, None] * g[None, :] + be[None, :]
    assert rel_inf(f64(D), acc + bias[None, :] + 7.5 * lnx) < 1e-5
    F.gemm(M, N, K, dA, lda, 0, dB, ldb, 0, D, N, tile=t, epilogue=F.FL_EPI_RESID, aux=dX, ld_aux=N, alpha=-2.0,
           aux_dtype=F.FL_DT_F32, d_dtype=F.FL_DT_F32)
    torch.cuda.synchronize()
    assert rel_inf(f64(D), acc - 2.0 * X) < 1e-5


@pytest.mark.parametrize("hd", [64, 128])
def test_attention_fwd_bwd(F, hd):
    seqs = [1, 64, 100, 130, 7, 64, 200] + ([520, 1030] if hd == 128 else [])
    nh = 2
    H = nh * hd
    cu = np.cumsum([0] + seqs).astype(np.int32)
    T = int(cu[-1])
    rng = np.random.default_rng(hd + 3)
    qkv = rnd_bf16_f64(rng, (T, 3 * H))
    do = rnd_bf16_f64(rng, (T, H))
    dqkv_ = dev_bf16(qkv)
    dcu = dev_i32(cu)
    ntiles = F.fl_k_attention_tiles(cu)
    assert ntiles == sum((L + 63) // 64 for L in seqs)
    tiles = torch.empty(ntiles * 2, dtype=torch.int32, device="cuda")
    o = torch.full((T, H), float("nan"), dtype=torch.bfloat16, device="cuda")
    lse = torch.empty((nh, T), dtype=torch.float32, device="cuda")
    F.fl_k_attention_fwd(T, nh, hd, dqkv_, cu, dcu, tiles, o, lse)
    torch.cuda.synchronize()
    q = qkv[:, :H].reshape(T, nh, hd)
    k = qkv[:, H:2 * H].reshape(T, nh, hd)
    v = qkv[:, 2 * H:].reshape(T, nh, hd)
    o_ref, lse_ref = O.attention_fwd(q, k, v, cu)
    assert rel_inf(f64(o), o_ref.reshape(T, H)) < 2e-2
    np.testing.assert_allclose(f64(lse), lse_ref, rtol=0, atol=2e-2)
    # backward (inverse rotary rotation folded in, as the server uses it)
    rd = hd // 2
    pos = np.concatenate([np.arange(L) for L in seqs]).astype(np.int32)
    tab = rope_table(max(seqs), rd, 10000.0)
    delta = torch.empty((nh, T), dtype=torch.float32, device="cuda")
    dq = torch.full((T, 3 * H), float("nan"), dtype=torch.bfloat16, device="cuda")
    # the kernel differentiates through its own saved O (bf16), as the server does
    F.fl_k_attention_bwd(T, nh, hd, dqkv_, o, lse, dev_bf16(do), cu, dcu, tiles, delta, dev_f32(tab), rd, dq)
    torch.cuda.synchronize()
    dqr, dkr, dvr = O.attention_bwd(do.reshape(T, nh, hd), q, k, v, cu)
    cos, sin = O.rope_cos_sin(pos, rd, 10000.0)
    dq_ref = O.rope_rotate(dqr, cos, sin, rd, inverse=True).reshape(T, H)
    dk_ref = O.rope_rotate(dkr, cos, sin, rd, inverse=True).reshape(T, H)
    got = f64(dq)
    assert rel_inf(got[:, :H], dq_ref) < 5e-2
    assert rel_inf(got[:, H:2 * H], dk_ref) < 5e-2
    assert rel_inf(got[:, 2 * H:], dvr.reshape(T, H)) < 5e-2


def test_adamw(F):
    n = 4096 + 64
    rng = np.random.default_rng(9)
    w = rng.standard_normal(n).astype(np.float32) * 0.02
    m = np.zeros(n, np.float32)
    v = np.zeros(n, np.float32)
    dw, dm, dv = dev_f32(w), dev_f32(m), dev_f32(v)
    wb = torch.empty(n, dtype=torch.bfloat16, device="cuda")
    ref_w, ref_m, ref_v = w.astype(np.float64), m.astype(np.float64), v.astype(np.float64)
    for t in range(1, 4):
        g = (rng.standard_normal(n) * 1e-3).astype(np.float32)
        dg = dev_f32(g)
        F.fl_k_adamw(n, dw, dg, dm, dv, wb, 1e-3, 0.9, 0.999, 1e-8, 0.01, 1 - 0.9 ** t, 1 - 0.999 ** t)
        torch.cuda.synchronize()
        # the C ABI carries the hyperparameters as fp32: the oracle gets the same values
        f = lambda x: float(np.float32(x))
        ref_w, ref_m, ref_v = O.adamw_update(ref_w, g.astype(np.float64), ref_m, ref_v, t, f(1e-3), f(0.9),
                                             f(0.999), f(1e-8), f(0.01))
        assert not f64(dg).any()
    assert rel_inf(f64(dw), ref_w) < 1e-5
    assert rel_inf(f64(dm), ref_m) < 1e-5
    assert rel_inf(f64(dv), ref_v) < 1e-5
    np.testing.assert_array_equal(bits(wb), bits(dw.to(torch.bfloat16)))


def test_colsum(F):
    T, N = 1000, 768
    rng = np.random.default_rng(2)
    x = rnd_bf16_f64(rng, (T, N))
    out = dev_f32(np.ones(N, np.float32))
    F.fl_k_colsum(T, N, dev_bf16(x), out)
    torch.cuda.synchronize()
    np.testing.assert_allclose(f64(out), 1.0 + x.sum(0), rtol=1e-5, atol=1e-4)


def test_pack_clients_bitexact(F):
    rng = np.random.default_rng(4)
    H = 256
    lens = [3, 1, 64, 17, 200]
    clients = [dev_bf16(rnd_bf16_f64(rng, (2, L, H))) for L in lens]
    nbytes = [c.numel() * 2 for c in clients]
    packed = torch.empty(sum(c.numel() for c in clients), dtype=torch.bfloat16, device="cuda")
    F.fl_k_pack_clients(clients, nbytes, packed, scatter=False)
    back = [torch.empty_like(c) for c in clients]
    F.fl_k_pack_clients(back, nbytes, packed, scatter=True)
    torch.cuda.synchronize()
    want = np.concatenate([bits(c).reshape(-1) for c in clients])
    np.testing.assert_array_equal(bits(packed), want)
    for a, b in zip(back, clients):
        np.testing.assert_array_equal(bits(a), bits(b))


@pytest.mark.parametrize("hd", [64, 128])
def test_attention_bwd_many_units(F, hd):
    """Many more (tile, head) units than SMs, so that every persistent backward CTA walks
    several units (the next unit's tiles loading while a unit's output leaves): every
    element of dqkv written (NaN-filled before), sampled heads against the oracle, and the
    rope table's alignment checked before any launch."""
    nh = 32 if hd == 128 else 40
    H = nh * hd
    seqs = [256] * 24 + [1, 130, 300, 77, 512, 64]
    cu = np.cumsum([0] + seqs).astype(np.int32)
    T = int(cu[-1])
    rng = np.random.default_rng(hd + 11)
    qkv = rnd_bf16_f64(rng, (T, 3 * H))
    do = rnd_bf16_f64(rng, (T, H))
    dqkv_, dcu = dev_bf16(qkv), dev_i32(cu)
    tiles = torch.empty(F.fl_k_attention_tiles(cu) * 2, dtype=torch.int32, device="cuda")
    o = torch.empty((T, H), dtype=torch.bfloat16, device="cuda")
    lse = torch.empty((nh, T), dtype=torch.float32, device="cuda")
    F.fl_k_attention_fwd(T, nh, hd, dqkv_, cu, dcu, tiles, o, lse)
    rd = hd // 2
    pos = np.concatenate([np.arange(L) for L in seqs]).astype(np.int32)
    tab = dev_f32(rope_table(max(seqs), rd, 10000.0))
    delta = torch.empty((nh, T), dtype=torch.float32, device="cuda")
    dq = torch.full((T, 3 * H), float("nan"), dtype=torch.bfloat16, device="cuda")
    with pytest.raises(F.FlError, match="aligned"):
        F.fl_k_attention_bwd(T, nh, hd, dqkv_, o, lse, dev_bf16(do), cu, dcu, tiles, delta, tab.view(-1)[2:], rd, dq)
    F.fl_k_attention_bwd(T, nh, hd, dqkv_, o, lse, dev_bf16(do), cu, dcu, tiles, delta, tab, rd, dq)
    torch.cuda.synchronize()
    got = f64(dq)
    assert np.isfinite(got).all()
    cos, sin = O.rope_cos_sin(pos, rd, 10000.0)
    heads = [0, nh // 2 + 1, nh - 1]
    sel = lambda base: np.concatenate([np.arange(base + h * hd, base + (h + 1) * hd) for h in heads])
    q = qkv[:, sel(0)].reshape(T, len(heads), hd)
    k = qkv[:, sel(H)].reshape(T, len(heads), hd)
    v = qkv[:, sel(2 * H)].reshape(T, len(heads), hd)
    dos = do[:, sel(0)].reshape(T, len(heads), hd)
    dqr, dkr, dvr = O.attention_bwd(dos, q, k, v, cu)
    n = len(heads) * hd
    assert rel_inf(got[:, sel(0)], O.rope_rotate(dqr, cos, sin, rd, inverse=True).reshape(T, n)) < 5e-2
    assert rel_inf(got[:, sel(H)], O.rope_rotate(dkr, cos, sin, rd, inverse=True).reshape(T, n)) < 5e-2
    assert rel_inf(got[:, sel(2 * H)], dvr.reshape(T, n)) < 5e-2


@pytest.mark.parametrize("hd,Lp", [(64, 16), (128, 100)])
def test_attention_with_prefix(F, hd, Lp):
    """P-tuning v2 prefix (App. A): every query also sees Lp prefix keys/values (one or two
    64-key tiles, the second partial); prefix gradients are summed over all segments."""
    seqs = [1, 64, 100, 7, 130]
    nh = 2
    H = nh * hd
    cu = np.cumsum([0] + seqs).astype(np.int32)
    T = int(cu[-1])
    rng = np.random.default_rng(hd + Lp)
    qkv = rnd_bf16_f64(rng, (T, 3 * H))
    pk = rnd_bf16_f64(rng, (Lp, H))
    pv = rnd_bf16_f64(rng, (Lp, H))
    do = rnd_bf16_f64(rng, (T, H))
    dqkv_, dcu = dev_bf16(qkv), dev_i32(cu)
    dpk_, dpv_ = dev_bf16(pk), dev_bf16(pv)
    tiles = torch.empty(F.fl_k_attention_tiles(cu) * 2, dtype=torch.int32, device="cuda")
    o = torch.full((T, H), float("nan"), dtype=torch.bfloat16, device="cuda")
    lse = torch.empty((nh, T), dtype=torch.float32, device="cuda")
    F.fl_k_attention_fwd(T, nh, hd, dqkv_, cu, dcu, tiles, o, lse, dpk_, dpv_, Lp)
    torch.cuda.synchronize()
    q = qkv[:, :H].reshape(T, nh, hd)
    k = qkv[:, H:2 * H].reshape(T, nh, hd)
    v = qkv[:, 2 * H:].reshape(T, nh, hd)
    ppk, ppv = pk.reshape(Lp, nh, hd), pv.reshape(Lp, nh, hd)
    o_ref, lse_ref = O.attention_fwd(q, k, v, cu, ppk, ppv)
    assert rel_inf(f64(o), o_ref.reshape(T, H)) < 2e-2
    np.testing.assert_allclose(f64(lse), lse_ref, rtol=0, atol=2e-2)
    delta = torch.empty((nh, T), dtype=torch.float32, device="cuda")
    dq = torch.full((T, 3 * H), float("nan"), dtype=torch.bfloat16, device="cuda")
    gpk = dev_f32(np.full((Lp, H), 0.25, np.float32))
    gpv = torch.zeros((Lp, H), dtype=torch.float32, device="cuda")
    F.fl_k_attention_bwd(T, nh, hd, dqkv_, o, lse, dev_bf16(do), cu, dcu, tiles, delta, None, 0, dq,
                         dpk_, dpv_, Lp, gpk, gpv)
    torch.cuda.synchronize()
    dqr, dkr, dvr, dpkr, dpvr = O.attention_bwd(do.reshape(T, nh, hd), q, k, v, cu, ppk, ppv)
    got = f64(dq)
    assert rel_inf(got[:, :H], dqr.reshape(T, H)) < 5e-2
    assert rel_inf(got[:, H:2 * H], dkr.reshape(T, H)) < 5e-2
    assert rel_inf(got[:, 2 * H:], dvr.reshape(T, H)) < 5e-2
    assert rel_inf(f64(gpk) - 0.25, dpkr.reshape(Lp, H)) < 5e-2   # accumulated onto the 0.25
    assert rel_inf(f64(gpv), dpvr.reshape(Lp, H)) < 5e-2


@pytest.mark.parametrize("tile", ["auto", "pair"])
@pytest.mark.parametrize("M,N,K,mn", [(200, 384, 136, 1), (256, 512, 64, 1), (130, 256, 96, 0), (600, 1024, 520, 1)])
def test_gemm_adamw_epilogue(F, M, N, K, mn, tile):
    """The weight-gradient GEMM with the AdamW update in its epilogue equals the plain fp32
    gradient GEMM followed by the separate AdamW kernel: weights, moments and the bf16
    copy; ragged rows, every tile shape (N = 384 takes 128-column tiles)."""
    if tile == "pair" and N % 256:
        pytest.skip("256-column tiles need N % 256 == 0")
    rng = np.random.default_rng(M + N)
    A = rnd_bf16_f64(rng, (M, K))
    B = rnd_bf16_f64(rng, (N, K))
    dA, lda = _store(A, bool(mn))
    dB, ldb = _store(B, bool(mn))
    w0 = (0.05 * rng.standard_normal((M, N))).astype(np.float32)
    m0 = (0.01 * rng.standard_normal((M, N))).astype(np.float32)
    v0 = (1e-3 * rng.random((M, N))).astype(np.float32)
    lr, b1, b2, eps, wd, t = 1e-3, 0.9, 0.999, 1e-8, 0.01, 3
    bc1, bc2 = 1.0 - b1 ** t, 1.0 - b2 ** t
    # reference: g = A B^T stored in fp32, then fl_k_adamw
    g = torch.empty((M, N), dtype=torch.float32, device="cuda")
    F.gemm(M, N, K, dA, lda, mn, dB, ldb, mn, g, N, epilogue=F.FL_EPI_STORE_F32)
    wr, mr, vr = dev_f32(w0), dev_f32(m0), dev_f32(v0)
    wbr = torch.empty((M, N), dtype=torch.bfloat16, device="cuda")
    F.fl_k_adamw(M * N, wr, g, mr, vr, wbr, lr, b1, b2, eps, wd, bc1, bc2)
    # fused
    wf, mf, vf = dev_f32(w0), dev_f32(m0), dev_f32(v0)
    wbf = torch.empty((M, N), dtype=torch.bfloat16, device="cuda")
    ga = F.fl_gemm_args(M, N, K, F.ptr(dA), lda, mn, F.ptr(dB), ldb, mn, F.ptr(wf), N, F.FL_EPI_ADAMW)
    ga.aux_out, ga.ld_aux_out = F.ptr(wbf), N
    ga.adam_m, ga.adam_v = F.ptr(mf), F.ptr(vf)
    ga.lr, ga.beta1, ga.beta2, ga.eps, ga.weight_decay = lr, b1, b2, eps, wd
    ga.inv_bc1, ga.inv_bc2 = 1.0 / np.float32(bc1), 1.0 / np.float32(bc2)
    ga.tile = tile_id(F, tile)
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    F.fl_k_gemm(ga, status=status)
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    for got, want in ((wf, wr), (mf, mr), (vf, vr)):
        assert rel_inf(f64(got), f64(want)) < 1e-5
    np.testing.assert_array_equal(bits(wbf), bits(wf.to(torch.bfloat16)))


def test_zero_size_calls(F):
    """Degenerate sizes: a GEMM of M = 0 rows, LayerNorm forward and backward over T = 0
    rows, AdamW over 0 parameters, column sums over 0 rows, and attention over one empty
    segment are no-ops that succeed and leave every output untouched."""
    H, N, K = 256, 256, 64
    A = torch.zeros((8, K), dtype=torch.bfloat16, device="cuda")
    B = torch.zeros((N, K), dtype=torch.bfloat16, device="cuda")
    D = torch.full((8, N), 7.0, dtype=torch.bfloat16, device="cuda")
    F.gemm(0, N, K, A, K, 0, B, K, 0, D, N)
    x = torch.zeros((8, H), dtype=torch.bfloat16, device="cuda")
    gam = torch.ones(H, device="cuda")
    bet = torch.zeros(H, device="cuda")
    y = torch.full((8, H), 3.0, dtype=torch.bfloat16, device="cuda")
    mean = torch.full((8,), 5.0, device="cuda")
    rstd = torch.full((8,), 5.0, device="cuda")
    F.fl_k_layernorm_fwd(0, H, x, gam, bet, 1e-5, y, mean, rstd)
    dgam = torch.full((H,), 2.0, device="cuda")
    dbet = torch.full((H,), 2.0, device="cuda")
    ws = torch.empty(max(F.fl_k_layernorm_bwd_workspace(1, H), 16), dtype=torch.uint8, device="cuda")
    F.fl_k_layernorm_bwd(0, H, x, x, mean, rstd, gam, None, 0.0, y, dgam, dbet, ws)
    w = torch.full((8,), 4.0, device="cuda")
    F.fl_k_adamw(0, w, w, w, w, None, 1e-3, 0.9, 0.999, 1e-8, 0.0, 0.1, 0.001)
    cs = torch.full((N,), 6.0, device="cuda")
    F.fl_k_colsum(0, N, D, cs)
    nh, hd = 2, 128
    qkv = torch.zeros((8, 3 * nh * hd), dtype=torch.bfloat16, device="cuda")
    cu = np.array([0, 0], np.int32)
    tiles = torch.zeros(16, dtype=torch.int32, device="cuda")
    o = torch.full((8, nh * hd), 9.0, dtype=torch.bfloat16, device="cuda")
    lse = torch.full((nh, 8), 9.0, device="cuda")
    assert F.fl_k_attention_tiles(cu) == 0
    F.fl_k_attention_fwd(0, nh, hd, qkv, cu, dev_i32(cu), tiles, o, lse)
    torch.cuda.synchronize()
    assert (D == 7.0).all() and (y == 3.0).all() and (mean == 5.0).all() and (rstd == 5.0).all()
    assert (dgam == 2.0).all() and (dbet == 2.0).all() and (w == 4.0).all() and (cs == 6.0).all()
    assert (o == 9.0).all() and (lse == 9.0).all() and not tiles.any()
