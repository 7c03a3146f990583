"""Full-size parity of the 26-block ChatGLM-6B-shaped workloads (GPU only, slow).

At these sizes the oracle cannot run the whole packed batch, so the checks use what
§3.3 fixes at any size (stacking clients does not mix them):

* the GPU runs the full packed call exactly as bench.py times it; for sampled segments
  (first and last, shortest and longest for the ragged workload) the fp64 oracle runs
  that segment alone through all 26 blocks, and the GPU's output states and input
  gradients of that segment must match (2e-2 / 5e-2);
* the same segment run alone on the GPU gives weight gradients (first and last block,
  all 12 tensors) that must match the oracle's single-segment gradients (5e-2);
* the packed call's weight gradients equal the serial strategy's (one client per call,
  accumulated), and each client's outputs are bit-identical in both;
* on the bench workload, one segment through fl_server_backward_step with the AdamW update
  fused into the weight-gradient GEMM epilogues (the path bench.py times): the updated
  weights and first Adam moments of the first and last block against the oracle's AdamW
  step from its own gradients.

The oracle uses the seeded weights of the synthetic generator; the library draws the
same streams on the device (equal to within one fp32 ulp, tested elsewhere).
"""
import os

import numpy as np
import pytest
import torch

import synthetic as syn
from oracle import flglm_oracle as O
from tests._gpu import bits, dev_bf16_from_bits, f64, flglm, need_gpu, rel_inf
from tests.test_gpu_server import check_updated_weights

pytestmark = [pytest.mark.gpu, pytest.mark.slow]

OUT_TOL, GRAD_TOL = 2e-2, 5e-2
CHECK_BLOCKS = (0, 25)


def _mem_available_gb() -> float:
    try:
        for line in open("/proc/meminfo"):
            if line.startswith("MemAvailable:"):
                return int(line.split()[1]) / 2 ** 20
    except OSError:
        pass
    return 0.0


@pytest.fixture(scope="module")
def F():
    need_gpu()
    return flglm()


@pytest.fixture(scope="module")
def weights():
    """fp32 master weights of all 26 blocks (seed 0), shared by every workload here."""
    need_gpu()
    if _mem_available_gb() < 48:
        pytest.skip(f"needs ~48 GB of host memory for the 26-block oracle, {_mem_available_gb():.0f} GB free")
    return syn.init_params(syn.CONFIGS["stack26"])


def oracle_segment(params, cfg, x_bits, g_bits):
    """One segment alone through the stack: output, input gradient and the weight
    gradients of CHECK_BLOCKS (fp64, one block's weights converted at a time)."""
    L = x_bits.shape[0]
    sh = O.BlockShape.of(cfg)
    pk = O.make_packing([L], 1)
    x = syn.bf16_bits_to_f64(x_bits)
    saved = []
    for b in range(cfg.n_blocks):
        P = [p.astype(np.float64) for p in params[b]]
        x, sv = O.block_fwd(P, x, pk, sh)
        saved.append(sv)
    y = x
    dy = syn.bf16_bits_to_f64(g_bits)
    wgrads = {}
    for b in range(cfg.n_blocks - 1, -1, -1):
        P = [p.astype(np.float64) for p in params[b]]
        dy, gb = O.block_bwd(P, saved[b], dy, pk, sh)
        saved[b] = None
        if b in CHECK_BLOCKS:
            wgrads[b] = gb
    return y, dy, wgrads


def gpu_call(F, cfg, states, grads, max_tokens, keep_clients):
    """Packed (or single-client) call on a fresh seeded server, as bench.py launches it.
    Returns host bits of the kept clients' outputs / input grads and CHECK_BLOCKS grads."""
    srv = F.Server(F.make_cfg(cfg, max_tokens, max(cfg.seq_lens)), cfg.seed)
    st = [dev_bf16_from_bits(s) for s in states]
    outs = [torch.empty_like(s) for s in st]
    srv.forward(st, cfg.seq_lens, outs)
    go = [dev_bf16_from_bits(g) for g in grads]
    gi = [torch.empty_like(s) for s in st]
    srv.backward(go, gi)
    srv.sync()
    res = {k: (bits(outs[k]), bits(gi[k])) for k in keep_clients}
    wg = {b: [srv.get_grad(b, t) for t in range(12)] for b in CHECK_BLOCKS}
    srv.close()
    del st, outs, go, gi
    torch.cuda.empty_cache()
    return res, wg


def serial_calls(F, cfg, states, grads, keep_clients):
    """The serial strategy: one client per call, gradients accumulated, no step."""
    srv = F.Server(F.make_cfg(cfg, cfg.tokens, max(cfg.seq_lens)), cfg.seed)
    res = {}
    for k in range(cfg.K):
        s = dev_bf16_from_bits(states[k])
        o = torch.empty_like(s)
        srv.forward([s], [cfg.seq_lens[k]], [o])
        g = dev_bf16_from_bits(grads[k])
        gi = torch.empty_like(s)
        srv.backward([g], [gi])
        if k in keep_clients:
            srv.sync()
            res[k] = (bits(o), bits(gi))
    srv.sync()
    wg = {b: [srv.get_grad(b, t) for t in range(12)] for b in CHECK_BLOCKS}
    srv.close()
    torch.cuda.empty_cache()
    return res, wg


def gpu_step_call(F, cfg, x_bits, g_bits):
    """One segment alone through forward + fl_server_backward_step with the update fused into
    the weight-gradient GEMMs (fused_step_min_tokens = 1: fused whatever the call's size).
    Returns the updated fp32 weights and Adam moments (m) of CHECK_BLOCKS."""
    L = x_bits.shape[0]
    srv = F.Server(F.make_cfg(cfg, L, L, fused_step_min_tokens=1), cfg.seed)
    st = [dev_bf16_from_bits(x_bits[None])]
    outs = [torch.empty_like(st[0])]
    srv.forward(st, [L], outs)
    gi = [torch.empty_like(st[0])]
    srv.backward_step([dev_bf16_from_bits(g_bits[None])], gi, cfg.lr)
    srv.sync()
    res = {b: [(srv.get_param(b, t), srv.get_adam_moments(b, t)[0]) for t in range(12)] for b in CHECK_BLOCKS}
    assert not any(srv.get_grad(b, t).any() for b in CHECK_BLOCKS for t in range(12))
    srv.close()
    torch.cuda.empty_cache()
    return res


def check_fused_step(cfg, weights, stepped, wg_ref):
    """Updated weights and m of CHECK_BLOCKS against the oracle's first AdamW step (t = 1,
    zero moments) taken from the oracle's gradients of the same segment."""
    for b in CHECK_BLOCKS:
        for t in range(12):
            w0 = weights[b][t].reshape(-1)
            g = wg_ref[b][t].reshape(-1)
            w_ref, m_ref, _ = O.adamw_update(w0.astype(np.float64), g, np.zeros_like(g), np.zeros_like(g), 1,
                                             cfg.lr, cfg.adam_beta1, cfg.adam_beta2, cfg.adam_eps, cfg.weight_decay)
            w, m = stepped[b][t]
            check_updated_weights(w, w_ref, w0, g, cfg.lr, (cfg.name, "step", b, syn.TENSOR_NAMES[t]))
            assert rel_inf(m, m_ref) < GRAD_TOL, (cfg.name, "adam m", b, syn.TENSOR_NAMES[t], rel_inf(m, m_ref))


def sampled_segments(cfg):
    """(client, row) pairs to check: the shortest and the longest segment when the lengths
    are ragged (one and eight query tiles at ragged26), else the first and the last."""
    if len(set(cfg.seq_lens)) > 1:
        return sorted({(int(np.argmin(cfg.seq_lens)), 0), (int(np.argmax(cfg.seq_lens)), 0)})
    return sorted({(0, 0), (cfg.K - 1, cfg.client_batch - 1)})


def run_workload(F, weights, cfg, n_oracle_segments=None, serial=True, step=False):
    states = syn.client_states(cfg)
    grads = syn.client_grads(cfg)
    picks = sampled_segments(cfg)[:n_oracle_segments]
    keep = sorted({k for k, _ in picks})
    packed, packed_wg = gpu_call(F, cfg, states, grads, cfg.tokens, keep)
    if serial:
        ser, ser_wg = serial_calls(F, cfg, states, grads, keep)
        for k in keep:   # batching invariant at full size: bit-identical per client
            np.testing.assert_array_equal(ser[k][0], packed[k][0])
            np.testing.assert_array_equal(ser[k][1], packed[k][1])
        for b in CHECK_BLOCKS:
            for t in range(12):
                assert rel_inf(packed_wg[b][t], ser_wg[b][t]) < 1e-3, (cfg.name, b, t)
    for (k, r) in picks:
        L = cfg.seq_lens[k]
        H = cfg.hidden
        x = states[k][r]
        g = grads[k][r]
        y_ref, dx_ref, wg_ref = oracle_segment(weights, cfg, x, g)
        out_bits, gin_bits = packed[k]
        y = syn.bf16_bits_to_f64(out_bits.reshape(cfg.client_batch, L, H)[r])
        dx = syn.bf16_bits_to_f64(gin_bits.reshape(cfg.client_batch, L, H)[r])
        assert rel_inf(y, y_ref) < OUT_TOL, (cfg.name, k, r, "out", rel_inf(y, y_ref))
        assert rel_inf(dx, dx_ref) < GRAD_TOL, (cfg.name, k, r, "grad_in", rel_inf(dx, dx_ref))
        # the same segment alone on the GPU: weight gradients vs the oracle's
        one = cfg.with_(client_batch=1, seq_lens=(L,))
        _, wg1 = gpu_call(F, one, [x[None]], [g[None]], L, [])
        for b in CHECK_BLOCKS:
            for t in range(12):
                e = rel_inf(wg1[b][t], wg_ref[b][t].reshape(-1))
                assert e < GRAD_TOL, (cfg.name, k, r, "wgrad", b, syn.TENSOR_NAMES[t], e)
        if step:
            check_fused_step(cfg, weights, gpu_step_call(F, one, x, g), wg_ref)
            step = False   # one segment is enough: the update is per element


def test_stack26_fullsize(F, weights):
    """26 blocks, K=8 clients x 4 rows x 256 tokens (T=8192), the bench workload, with the
    fused backward + AdamW step of one segment."""
    run_workload(F, weights, syn.CONFIGS["stack26"], step=True)


def test_ragged26_fullsize(F, weights):
    """26 blocks, K=16 clients x 1 row, lengths U[64,1024] (seed 7), no padding."""
    run_workload(F, weights, syn.CONFIGS["ragged26"])


@pytest.mark.parametrize("K", [1, 8])
def test_sweep26_fullsize_vs_serial(F, weights, K):
    """Sweep points K=1 and K=8 (2 rows x 512 tokens per client): the packed call against
    the serial strategy (bit-identical per client, equal weight gradients) and one segment
    against the oracle."""
    run_workload(F, weights, syn.sweep_config(K), n_oracle_segments=1, serial=True)


def test_sweep26_K32_fullsize(F, weights):
    """The largest sweep point: K=32 clients x 2 rows x 512 tokens (T=32768)."""
    run_workload(F, weights, syn.sweep_config(32), n_oracle_segments=1, serial=False)
