"""Per-kernel timing of the server's hot-path kernels at a workload's shapes.

    python -m paper_2406_14898_gb300.kernel_bench [--workload stack26] [--kernel all|<name>] [--reps 5]

<name>: gemm or one GEMM case (qkv_fwd, ..., qkv_wgrad), attention, layernorm, adamw, colsum,
client (cross-entropy over the ChatGLM-6B vocabulary and the embedding gather).

Each kernel runs on random device buffers (uninitialised values are never read: every
input is filled first) with CUDA events around `reps` launches on one stream, after one
warm-up launch.  Prints one JSON line per kernel with its algorithmic work (FLOPs for
the contractions, bytes for the row kernels), mean time and achieved rate.  The inputs
of every GEMM here are larger than L2 at the ChatGLM-6B shapes.
"""
from __future__ import annotations

import argparse
import json
import os
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def gemm_cases(cfg):
    """(name, M, N, K, a_mn, b_mn, epilogue, fp32 residual stream) of the 12 GEMMs of one
    block at T tokens, with the operand layouts and epilogues the server uses (the FFN
    up-projection weight stored transposed, [H, F]; weight gradients as the first backward
    after a step stores them)."""
    from paper_2406_14898_gb300 import flglm as F
    T, H, Fh = cfg.tokens, cfg.hidden, cfg.ffn_hidden
    return [
        ("qkv_fwd", T, 3 * H, H, 0, 0, F.FL_EPI_BIAS_ROPE, False),
        ("dense_fwd", T, H, H, 0, 0, F.FL_EPI_BIAS_RESID, True),
        ("up_fwd", T, Fh, H, 0, 1, F.FL_EPI_BIAS_GELU, False),
        ("down_fwd", T, H, Fh, 0, 0, F.FL_EPI_BIAS_RESID, True),
        ("down_dgrad", T, Fh, H, 0, 1, F.FL_EPI_GELU_BWD, False),
        ("down_wgrad", H, Fh, T, 1, 1, F.FL_EPI_STORE_F32, False),
        ("up_dgrad", T, H, Fh, 0, 0, F.FL_EPI_RESID, True),
        ("up_wgrad", H, Fh, T, 1, 1, F.FL_EPI_STORE_F32, False),
        ("dense_dgrad", T, H, H, 0, 1, F.FL_EPI_STORE, False),
        ("dense_wgrad", H, H, T, 1, 1, F.FL_EPI_STORE_F32, False),
        ("qkv_dgrad", T, H, 3 * H, 0, 1, F.FL_EPI_RESID, True),
        ("qkv_wgrad", 3 * H, H, T, 1, 1, F.FL_EPI_STORE_F32, False),
    ]


def main():
    import numpy as np
    import torch

    import synthetic as syn
    from paper_2406_14898_gb300 import flglm as F

    ap = argparse.ArgumentParser()
    ap.add_argument("--workload", default="stack26")
    ap.add_argument("--kernel", default="all")
    ap.add_argument("--reps", type=int, default=5)
    ap.add_argument("--wgrad-epilogue", default="store", choices=["store", "adamw"],
                    help="epilogue of the weight-gradient GEMMs: fp32 store (the separate-step path) or the "
                         "fused AdamW update of the backward + step call")
    ap.add_argument("--tiles", default="auto",
                    help="comma-separated GEMM tile shapes to time: auto, 128x128, 128x256, pair (256 x 256 on a "
                         "CTA pair)")
    args = ap.parse_args()
    tile_ids = {"auto": F.FL_TILE_AUTO, "128x128": F.FL_TILE_128x128, "128x256": F.FL_TILE_128x256,
                "pair": F.FL_TILE_256x256_PAIR}
    tiles_wanted = [t.strip() for t in args.tiles.split(",") if t.strip()]
    cfg = syn.CONFIGS[args.workload]
    F.lib()
    dev = torch.device("cuda", 0)
    st = torch.cuda.Stream(device=dev)
    ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    g = torch.Generator(device=dev)
    g.manual_seed(0)

    def rnd(*shape, scale=1.0, dtype=torch.bfloat16):
        return (torch.randn(*shape, device=dev, generator=g) * scale).to(dtype)

    def timed(fn):
        with torch.cuda.stream(st):
            fn()
            torch.cuda.synchronize()
            ev0.record(st)
            for _ in range(args.reps):
                fn()
            ev1.record(st)
        torch.cuda.synchronize()
        return ev0.elapsed_time(ev1) / args.reps

    T, H, Fh, nh, hd = cfg.tokens, cfg.hidden, cfg.ffn_hidden, cfg.n_heads, cfg.head_dim
    out = []
    for (name, M, N, K, amn, bmn, epi, f32res) in gemm_cases(cfg):
        if args.kernel not in ("all", "gemm", name):
            continue
        A = rnd(K, M, scale=0.1) if amn else rnd(M, K, scale=0.1)
        B = rnd(K, N, scale=0.1) if bmn else rnd(N, K, scale=0.1)
        f32_out = epi in (F.FL_EPI_ACCUM_F32, F.FL_EPI_STORE_F32) or f32res
        D = torch.zeros(M, N, device=dev, dtype=torch.float32 if f32_out else torch.bfloat16)
        kw = {}
        if epi in (F.FL_EPI_BIAS_ROPE, F.FL_EPI_BIAS_RESID, F.FL_EPI_BIAS_GELU):
            kw["bias"] = rnd(N, dtype=torch.float32)
        if epi in (F.FL_EPI_BIAS_RESID, F.FL_EPI_RESID, F.FL_EPI_GELU_BWD):
            kw["aux"] = rnd(M, N, dtype=torch.float32 if f32res else torch.bfloat16)
            kw["ld_aux"] = N
            kw["alpha"] = 1.5
        if f32res:
            kw.update(aux_dtype=F.FL_DT_F32, d_dtype=F.FL_DT_F32)
            if epi == F.FL_EPI_BIAS_RESID:   # residual = alpha * LN(x) recomputed in the epilogue
                kw.update(ln_mean=rnd(M, dtype=torch.float32), ln_rstd=rnd(M, dtype=torch.float32),
                          ln_gamma=rnd(N, dtype=torch.float32), ln_beta=rnd(N, dtype=torch.float32))
        if epi == F.FL_EPI_BIAS_GELU:
            kw["aux_out"] = torch.empty(M, N, device=dev, dtype=torch.bfloat16)
            kw["ld_aux_out"] = N
        if epi == F.FL_EPI_BIAS_ROPE:
            L = max(cfg.seq_lens)
            kw["pos"] = (torch.arange(M, device=dev, dtype=torch.int32) % L)
            kw["rope_tab"] = rnd(L, hd // 4, 2, dtype=torch.float32)
            kw.update(n_heads=nh, head_dim=hd, rotary_dim=hd // 2)
        lda = M if amn else K
        ldb = N if bmn else K
        adamw = epi == F.FL_EPI_STORE_F32 and args.wgrad_epilogue == "adamw"
        if adamw:
            # g = A . B^T updates fp32 weights D with their moments, writes the bf16 copy
            mom = torch.zeros(2, M, N, device=dev, dtype=torch.float32)
            wb16 = torch.empty(M, N, device=dev, dtype=torch.bfloat16)
            ga = F.fl_gemm_args(M, N, K, F.ptr(A), lda, amn, F.ptr(B), ldb, bmn, F.ptr(D), N, F.FL_EPI_ADAMW)
            ga.aux_out, ga.ld_aux_out = F.ptr(wb16), N
            ga.adam_m, ga.adam_v = F.ptr(mom[0]), F.ptr(mom[1])
            ga.lr, ga.beta1, ga.beta2, ga.eps, ga.weight_decay = 1e-4, 0.9, 0.999, 1e-8, 0.0
            ga.inv_bc1, ga.inv_bc2 = 10.0, 1000.0
        for tname in tiles_wanted:
            tile = tile_ids[tname]
            if tile >= F.FL_TILE_128x256 and N % 256:
                continue
            if adamw:
                ga.tile = tile
                ms = timed(lambda: F.fl_k_gemm(ga, stream=st))
            else:
                ms = timed(lambda: F.gemm(M, N, K, A, lda, amn, B, ldb, bmn, D, N, epilogue=epi, tile=tile, stream=st,
                                          **kw))
            flops = 2.0 * M * N * K
            rec = {"kernel": f"gemm_{name}" + ("_adamw" if adamw else ""), "M": M, "N": N, "K": K, "ms": ms,
                   "tflops": flops / ms / 1e9}
            if tname != "auto":
                rec["tile"] = tname
            out.append(rec)
        del A, B, D, kw
    if args.kernel in ("all", "attention"):
        seqs = cfg.segment_lengths
        cu = np.cumsum([0] + list(seqs)).astype(np.int32)
        qkv = rnd(T, 3 * H)
        o = torch.empty(T, H, device=dev, dtype=torch.bfloat16)
        lse = torch.empty(nh, T, device=dev, dtype=torch.float32)
        tiles = torch.empty(2 * F.fl_k_attention_tiles(cu), device=dev, dtype=torch.int32)
        dcu = torch.from_numpy(cu).to(dev)
        fl = float(sum(2 * H * L * (L + 1) for L in seqs))
        ms = timed(lambda: F.fl_k_attention_fwd(T, nh, hd, qkv, cu, dcu, tiles, o, lse, stream=st))
        out.append({"kernel": "attention_fwd", "T": T, "ms": ms, "tflops": fl / ms / 1e9})
        do = rnd(T, H)
        delta = torch.empty(nh, T, device=dev, dtype=torch.float32)
        dqkv = torch.empty(T, 3 * H, device=dev, dtype=torch.bfloat16)
        tab = rnd(max(seqs), hd // 4, 2, dtype=torch.float32)
        ms = timed(lambda: F.fl_k_attention_bwd(T, nh, hd, qkv, o, lse, do, cu, dcu, tiles, delta, tab, hd // 2, dqkv,
                                                stream=st))
        out.append({"kernel": "attention_bwd", "T": T, "ms": ms, "tflops": 2.5 * fl / ms / 1e9})
    if args.kernel in ("all", "layernorm"):
        # as the server runs them: fp32 residual-stream input, bf16 LN output; backward with
        # fp32 dy and x, dx written as bf16 and fp32
        x = rnd(T, H, dtype=torch.float32)
        gm = rnd(H, dtype=torch.float32)
        bt = rnd(H, dtype=torch.float32)
        y = torch.empty(T, H, device=dev, dtype=torch.bfloat16)
        mean = torch.empty(T, device=dev, dtype=torch.float32)
        rstd = torch.empty(T, device=dev, dtype=torch.float32)
        ms = timed(lambda: F.fl_k_layernorm_fwd(T, H, x, gm, bt, 1e-5, y, mean, rstd, x_dtype=F.FL_DT_F32, stream=st))
        nbytes = T * H * (4 + 2) + 8 * T
        out.append({"kernel": "layernorm_fwd", "ms": ms, "gbs": nbytes / ms / 1e6, "bytes": nbytes})
        dy = rnd(T, H, dtype=torch.float32)
        dxb = torch.empty(T, H, device=dev, dtype=torch.bfloat16)
        dxf = torch.empty(T, H, device=dev, dtype=torch.float32)
        ws = torch.empty(F.fl_k_layernorm_bwd_workspace(T, H) // 4 + 64, device=dev, dtype=torch.float32)
        dg = torch.zeros(H, device=dev, dtype=torch.float32)
        db = torch.zeros(H, device=dev, dtype=torch.float32)
        ms = timed(lambda: F.fl_k_layernorm_bwd(T, H, dy, x, mean, rstd, gm, None, 0.0, dxb, dg, db, ws,
                                                io_dtype=F.FL_DT_F32, dx_f32=dxf, stream=st))
        nbytes = T * H * (4 + 4 + 2 + 4) + 8 * T
        out.append({"kernel": "layernorm_bwd", "ms": ms, "gbs": nbytes / ms / 1e6, "bytes": nbytes})
    if args.kernel in ("all", "adamw"):
        n = syn.params_per_block(cfg) // 4 * 4
        w = rnd(n, dtype=torch.float32)
        gr = rnd(n, dtype=torch.float32)
        m = torch.zeros(n, device=dev, dtype=torch.float32)
        v = torch.zeros(n, device=dev, dtype=torch.float32)
        wb = torch.empty(n, device=dev, dtype=torch.bfloat16)
        ms = timed(lambda: F.fl_k_adamw(n, w, gr, m, v, wb, 1e-4, 0.9, 0.999, 1e-8, 0.0, 0.1, 0.001, stream=st))
        nbytes = n * (16 + 16 + 2)  # read w g m v, write w g m v, write bf16 copy
        out.append({"kernel": "adamw_one_block", "n": n, "ms": ms, "gbs": nbytes / ms / 1e6})
    if args.kernel in ("all", "colsum"):
        # bias gradient of the FFN up-projection: column sums of dU [T, F]
        du = rnd(T, Fh)
        db = torch.zeros(Fh, device=dev, dtype=torch.float32)
        ms = timed(lambda: F.fl_k_colsum(T, Fh, du, db, stream=st))
        nbytes = T * Fh * 2 + Fh * 8
        out.append({"kernel": "colsum_dU", "ms": ms, "gbs": nbytes / ms / 1e6, "bytes": nbytes})
        del du
    if args.kernel in ("all", "client"):
        # the client's cross-entropy over the ChatGLM-6B vocabulary (1024 tokens: 4 rows x 256)
        # and the embedding gather of a full packed batch
        V = syn.CHATGLM6B_VOCAB
        ld = (V + 255) // 256 * 256
        Tc = 1024
        logits = rnd(Tc, ld, scale=2.0, dtype=torch.float32)
        labels = torch.randint(0, V, (Tc,), device=dev, dtype=torch.int32, generator=g)
        row = torch.empty(Tc, device=dev, dtype=torch.float32)
        dlog = torch.empty(Tc, ld, device=dev, dtype=torch.bfloat16)
        loss = torch.empty(1, device=dev, dtype=torch.float32)
        cnt = torch.empty(1, device=dev, dtype=torch.int32)
        status = torch.zeros(1, device=dev, dtype=torch.int32)
        ms = timed(lambda: F.fl_k_cross_entropy(Tc, V, ld, logits, labels, row, dlog, loss, cnt, status, stream=st))
        nbytes = Tc * V * 4 + Tc * ld * 2   # read the logits once, write the gradient
        out.append({"kernel": "cross_entropy_vocab130528", "T": Tc, "ms": ms, "gbs": nbytes / ms / 1e6,
                    "bytes": nbytes})
        del logits, dlog
        table = rnd(V, H)
        toks = torch.randint(0, V, (T,), device=dev, dtype=torch.int32, generator=g)
        emb = torch.empty(T, H, device=dev, dtype=torch.bfloat16)
        ms = timed(lambda: F.fl_k_embedding_gather(T, H, toks, table, V, emb, status, stream=st))
        nbytes = 2 * T * H * 2
        out.append({"kernel": "embedding_gather", "T": T, "ms": ms, "gbs": nbytes / ms / 1e6, "bytes": nbytes})
    for r in out:
        print(json.dumps(r), flush=True)


if __name__ == "__main__":
    main()
