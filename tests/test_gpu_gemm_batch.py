"""Batched GEMM launches (several problems of one shape in one launch, the replicas of the
server-hierarchical strategy of §3.3) against the same problems launched one by one:
every output bit-identical (the per-tile arithmetic does not depend on the batch), the
fused column sums equal within their atomic summation order.  GPU only."""
import numpy as np
import pytest
import torch

from tests._gpu import dev_bf16, dev_f32, dev_i32, flglm, need_gpu, rnd_bf16_f64, rope_table

pytestmark = pytest.mark.gpu

R = 3


@pytest.fixture(scope="module")
def F():
    need_gpu()
    return flglm()


def tile_id(F, name):
    return {"128x128": F.FL_TILE_128x128, "128x256": F.FL_TILE_128x256, "pair": F.FL_TILE_256x256_PAIR}[name]


def stacked(rng, shape, scale=1.0):
    """R problems' bf16 operands [R, *shape] in one buffer."""
    return dev_bf16(rnd_bf16_f64(rng, (R,) + shape, scale).reshape(R, *shape))


def test_batch_argument_errors(F):
    A = torch.zeros((2, 128, 64), dtype=torch.bfloat16, device="cuda")
    B = torch.zeros((2, 128, 64), dtype=torch.bfloat16, device="cuda")
    D = torch.zeros((2, 128, 128), dtype=torch.bfloat16, device="cuda")
    with pytest.raises(F.FlError):
        F.gemm(128, 128, 64, A, 64, 0, B, 64, 0, D, 128, batch=F.FL_GEMM_MAX_BATCH + 1)
    with pytest.raises(F.FlError):  # a stride that breaks the 16-byte alignment of problem 1
        F.gemm(128, 128, 64, A, 64, 0, B, 64, 0, D, 128, batch=2,
               bstrides={"a": 128 * 64 + 1, "b": 128 * 64, "d": 128 * 128})


def _cmp(a, b):
    np.testing.assert_array_equal(a.view(torch.int32 if a.element_size() == 4 else torch.int16).cpu().numpy(),
                                  b.view(torch.int32 if b.element_size() == 4 else torch.int16).cpu().numpy())


LAYOUTS = {"fwd": (0, 0), "dgrad": (0, 1), "wgrad": (1, 1)}


def operands(rng, M, N, K, layout):
    """Stacked A, B for the layout: K-major A [R, M, K] or MN-major [R, K, M]; B likewise."""
    a_mn, b_mn = LAYOUTS[layout]
    A = stacked(rng, (K, M) if a_mn else (M, K))
    B = stacked(rng, (K, N) if b_mn else (N, K), 0.1)
    lda = M if a_mn else K
    ldb = N if b_mn else K
    return A, lda, B, ldb, a_mn, b_mn


def batched_and_separate(F, M, N, K, layout, tile, epilogue, per_problem, outputs, **scalars):
    """per_problem: name -> stacked tensor [R, ...] (inputs, problem r at index r);
    outputs: name -> (shape, dtype, init) of the stacked outputs.  Returns the batched and
    the separate outputs, name -> [R, ...] tensors."""
    A, lda, B, ldb, a_mn, b_mn = per_problem.pop("_ops")
    stride_names = {"aux": "aux", "bias": "bias", "colsum": "bias", "pos": "row", "pos2": "row", "ln_mean": "row",
                    "ln_rstd": "row", "ln_gamma": "lnp", "ln_beta": "lnp", "adam_m": "adam", "adam_v": "adam",
                    "aux_out": "aux_out"}

    def fresh():
        return {k: init(shape, dtype) for k, (shape, dtype, init) in outputs.items()}

    def call(bufs, r, batch):
        kw = dict(scalars)
        bs = {}
        for k, t in list(per_problem.items()) + [(k, v) for k, v in bufs.items() if k != "D"]:
            kw[k] = t[r]
            if batch > 1:
                bs[stride_names[k]] = t.stride(0)
        D = bufs["D"]
        if batch > 1:
            bs.update(a=A.stride(0), b=B.stride(0), d=D.stride(0))
        F.gemm(M, N, K, A[r], lda, a_mn, B[r], ldb, b_mn, D[r], N, epilogue=epilogue, tile=tile_id(F, tile),
               batch=batch, bstrides=bs, **kw)

    bat = fresh()
    call(bat, 0, R)
    sep = fresh()
    for r in range(R):
        call(sep, r, 1)
    torch.cuda.synchronize()
    return bat, sep


def zeros(shape, dtype):
    return torch.zeros((R,) + shape, dtype=dtype, device="cuda")


def nans(shape, dtype):
    return torch.full((R,) + shape, float("nan"), dtype=dtype, device="cuda")


TILES = ["128x128", "128x256", "pair"]


@pytest.mark.parametrize("tile", TILES)
@pytest.mark.parametrize("layout", ["fwd", "dgrad", "wgrad"])
def test_batched_store(F, tile, layout):
    M, N, K = 200, 512, 136
    rng = np.random.default_rng(1)
    ops = operands(rng, M, N, K, layout)
    bias = dev_f32(rng.standard_normal((R, N)).astype(np.float32))
    bat, sep = batched_and_separate(F, M, N, K, layout, tile, F.FL_EPI_STORE, {"_ops": ops, "bias": bias},
                                    {"D": ((M, N), torch.bfloat16, nans)})
    _cmp(bat["D"], sep["D"])


@pytest.mark.parametrize("tile", TILES)
def test_batched_f32_store_and_accumulate(F, tile):
    M, N, K = 256, 512, 200
    rng = np.random.default_rng(2)
    ops = operands(rng, M, N, K, "wgrad")
    for epi in (F.FL_EPI_STORE_F32, F.FL_EPI_ACCUM_F32):
        init = (lambda s, d: torch.ones((R,) + s, dtype=d, device="cuda")) if epi == F.FL_EPI_ACCUM_F32 else nans
        bat, sep = batched_and_separate(F, M, N, K, "wgrad", tile, epi, {"_ops": ops},
                                        {"D": ((M, N), torch.float32, init)})
        _cmp(bat["D"], sep["D"])


@pytest.mark.parametrize("tile", TILES)
def test_batched_gelu_and_gelu_backward(F, tile):
    M, N, K = 192, 512, 256
    rng = np.random.default_rng(3)
    ops = operands(rng, M, N, K, "fwd")
    bias = dev_f32(rng.standard_normal((R, N)).astype(np.float32))
    bat, sep = batched_and_separate(F, M, N, K, "fwd", tile, F.FL_EPI_BIAS_GELU, {"_ops": ops, "bias": bias},
                                    {"D": ((M, N), torch.bfloat16, nans), "aux_out": ((M, N), torch.bfloat16, nans)},
                                    ld_aux_out=N)
    _cmp(bat["D"], sep["D"])
    _cmp(bat["aux_out"], sep["aux_out"])
    ops = operands(rng, M, N, K, "dgrad")
    U = stacked(rng, (M, N))
    bat, sep = batched_and_separate(F, M, N, K, "dgrad", tile, F.FL_EPI_GELU_BWD, {"_ops": ops, "aux": U},
                                    {"D": ((M, N), torch.bfloat16, nans), "colsum": ((N,), torch.float32, zeros)},
                                    ld_aux=N)
    _cmp(bat["D"], sep["D"])
    torch.testing.assert_close(bat["colsum"], sep["colsum"], rtol=1e-5, atol=1e-5)


@pytest.mark.parametrize("tile", TILES)
def test_batched_residual_with_layernorm(F, tile):
    M, N, K = 130, 256, 256
    rng = np.random.default_rng(4)
    ops = operands(rng, M, N, K, "fwd")
    X = dev_f32(rng.standard_normal((R, M, N)).astype(np.float32))
    mean = dev_f32(rng.standard_normal((R, M)).astype(np.float32))
    rstd = dev_f32((1 + 0.1 * rng.random((R, M))).astype(np.float32))
    g = dev_f32(rng.standard_normal((R, N)).astype(np.float32))
    b = dev_f32(rng.standard_normal((R, N)).astype(np.float32))
    bias = dev_f32(rng.standard_normal((R, N)).astype(np.float32))
    bat, sep = batched_and_separate(F, M, N, K, "fwd", tile, F.FL_EPI_BIAS_RESID,
                                    {"_ops": ops, "aux": X, "ln_mean": mean, "ln_rstd": rstd, "ln_gamma": g,
                                     "ln_beta": b, "bias": bias},
                                    {"D": ((M, N), torch.float32, nans)}, ld_aux=N, alpha=1.5,
                                    aux_dtype=F.FL_DT_F32, d_dtype=F.FL_DT_F32)
    _cmp(bat["D"], sep["D"])


@pytest.mark.parametrize("tile", TILES)
def test_batched_rope(F, tile):
    nh, hd = 2, 128
    H = nh * hd
    M, N, K = 130, 3 * H, 256
    rng = np.random.default_rng(5)
    ops = operands(rng, M, N, K, "fwd")
    bias = dev_f32(rng.standard_normal((R, N)).astype(np.float32))
    pos = dev_i32(rng.integers(0, 300, (R, M)))
    pos2 = dev_i32(rng.integers(0, 300, (R, M)))
    tab = dev_f32(rope_table(300, hd // 2, 10000.0))
    bat, sep = batched_and_separate(F, M, N, K, "fwd", tile, F.FL_EPI_BIAS_ROPE,
                                    {"_ops": ops, "bias": bias, "pos": pos, "pos2": pos2},
                                    {"D": ((M, N), torch.bfloat16, nans)}, rope_tab=tab, n_heads=nh, head_dim=hd,
                                    rotary_dim=hd // 2)
    _cmp(bat["D"], sep["D"])


@pytest.mark.parametrize("tile", TILES)
def test_batched_adamw(F, tile):
    M, N, K = 256, 512, 200
    rng = np.random.default_rng(6)
    ops = operands(rng, M, N, K, "wgrad")
    w0 = (0.02 * rng.standard_normal((R, M, N))).astype(np.float32)
    m0 = (1e-3 * rng.standard_normal((R, M, N))).astype(np.float32)
    v0 = (1e-6 * rng.random((R, M, N))).astype(np.float32)
    outs = {"D": ((M, N), torch.float32, lambda s, d: dev_f32(w0)),
            "adam_m": ((M, N), torch.float32, lambda s, d: dev_f32(m0)),
            "adam_v": ((M, N), torch.float32, lambda s, d: dev_f32(v0)),
            "aux_out": ((M, N), torch.bfloat16, nans)}
    bat, sep = batched_and_separate(F, M, N, K, "wgrad", tile, F.FL_EPI_ADAMW, {"_ops": ops}, outs, ld_aux_out=N,
                                    lr=1e-3, beta1=0.9, beta2=0.999, eps=1e-8, weight_decay=0.01, inv_bc1=1 / 0.19,
                                    inv_bc2=1 / 0.002997)
    for k in ("D", "adam_m", "adam_v", "aux_out"):
        _cmp(bat[k], sep[k])


# ---------------------------------------------------------------- fl_k_gemm_multi
def test_multi_argument_errors(F):
    A = torch.zeros((128, 64), dtype=torch.bfloat16, device="cuda")
    D = torch.zeros((128, 128), dtype=torch.bfloat16, device="cuda")
    a0 = F.gemm_args(128, 128, 64, A, 64, 0, A, 64, 0, D, 128)
    with pytest.raises(F.FlError):
        F.fl_k_gemm_multi([a0] * (F.FL_GEMM_MAX_BATCH + 1))
    with pytest.raises(F.FlError, match="differs"):  # another M
        F.fl_k_gemm_multi([a0, F.gemm_args(64, 128, 64, A, 64, 0, A, 64, 0, D, 128)])
    with pytest.raises(F.FlError, match="differs"):  # another epilogue
        F.fl_k_gemm_multi([a0, F.gemm_args(128, 128, 64, A, 64, 0, A, 64, 0, D, 128, epilogue=F.FL_EPI_STORE_F32)])
    bias = torch.zeros(128, dtype=torch.float32, device="cuda")
    with pytest.raises(F.FlError, match="lacks"):  # a bias in one problem only
        F.fl_k_gemm_multi([a0, F.gemm_args(128, 128, 64, A, 64, 0, A, 64, 0, D, 128, bias=bias)])
    with pytest.raises(F.FlError):  # a batched entry
        F.fl_k_gemm_multi([a0, F.gemm_args(128, 128, 64, A, 64, 0, A, 64, 0, D, 128, batch=2)])


@pytest.mark.parametrize("tile", TILES)
def test_multi_weight_gradients_adamw(F, tile):
    """The backward's grouped weight gradients: problems 0-2 read column slices of one
    [K, 3M] gradient (lda = 3M, as the q, k, v rows of a QKV weight), problem 3 its own
    [K, M] tensor; the four updated weights, moments and bf16 copies sit at irregular
    offsets of shared arenas.  Bit-identical to four separate launches."""
    M, N, K = 256, 512, 200
    n = 4
    rng = np.random.default_rng(7)
    dqkv = dev_bf16(rnd_bf16_f64(rng, (K, 3 * M)))
    dh = dev_bf16(rnd_bf16_f64(rng, (K, M)))
    X = [dev_bf16(rnd_bf16_f64(rng, (K, N), 0.1)) for _ in range(2)]
    offs = [0, M * N + 64, 2 * M * N + 128, 3 * M * N + 1024]  # element offsets in the arenas
    size = offs[-1] + M * N
    w0 = (0.02 * rng.standard_normal(size)).astype(np.float32)
    m0 = (1e-3 * rng.standard_normal(size)).astype(np.float32)
    v0 = (1e-6 * rng.random(size)).astype(np.float32)
    hyper = dict(lr=1e-3, beta1=0.9, beta2=0.999, eps=1e-8, weight_decay=0.01, inv_bc1=1 / 0.19, inv_bc2=1 / 0.002997)

    def run(multi):
        w, m, v = dev_f32(w0), dev_f32(m0), dev_f32(v0)
        wb = torch.full((size,), float("nan"), dtype=torch.bfloat16, device="cuda")
        args = []
        for r in range(n):
            A, lda = (dqkv[:, r * M:], 3 * M) if r < 3 else (dh, M)
            o = offs[r]
            args.append(F.gemm_args(M, N, K, A, lda, 1, X[r % 2], N, 1, w[o:], N, epilogue=F.FL_EPI_ADAMW,
                                    aux_out=wb[o:], ld_aux_out=N, adam_m=m[o:], adam_v=v[o:], tile=tile_id(F, tile),
                                    **hyper))
        if multi:
            F.fl_k_gemm_multi(args)
        else:
            for a in args:
                F.fl_k_gemm(a)
        torch.cuda.synchronize()
        return w, m, v, wb

    got, want = run(True), run(False)
    for g, x in zip(got, want):
        _cmp(g, x)


@pytest.mark.parametrize("tile", TILES)
def test_multi_forward_bias_residual_layernorm(F, tile):
    """Three forward problems in separate buffers (K-major A with different row strides),
    bias + fp32 residual with the LayerNorm recomputed, each problem's per-row statistics
    and gain / shift at their own offsets; bit-identical to separate launches."""
    M, N, K = 130, 256, 192
    rng = np.random.default_rng(8)
    n = 3
    As = [dev_bf16(rnd_bf16_f64(rng, (M, K + 64 * r))) for r in range(n)]
    Bs = [dev_bf16(rnd_bf16_f64(rng, (N, K), 0.1)) for _ in range(n)]
    X = dev_f32(rng.standard_normal((n, M, N)).astype(np.float32))
    stats = dev_f32(rng.standard_normal((2, n * M + 32)).astype(np.float32))
    lnp = dev_f32(rng.standard_normal((2, n * N + 64)).astype(np.float32))
    bias = dev_f32(rng.standard_normal(n * N + 16).astype(np.float32))

    def run(multi):
        D = torch.full((n, M, N), float("nan"), dtype=torch.float32, device="cuda")
        args = []
        for r in range(n):
            ro, co = r * M + 8 * r, r * N + 16 * r
            args.append(F.gemm_args(M, N, K, As[r], K + 64 * r, 0, Bs[r], K, 0, D[r], N, epilogue=F.FL_EPI_BIAS_RESID,
                                    bias=bias[r * N + 4 * r:], aux=X[r], ld_aux=N, alpha=1.5, aux_dtype=F.FL_DT_F32,
                                    d_dtype=F.FL_DT_F32, ln_mean=stats[0, ro:], ln_rstd=stats[1, ro:],
                                    ln_gamma=lnp[0, co:], ln_beta=lnp[1, co:], tile=tile_id(F, tile)))
        if multi:
            F.fl_k_gemm_multi(args)
        else:
            for a in args:
                F.fl_k_gemm(a)
        torch.cuda.synchronize()
        return D

    _cmp(run(True), run(False))
