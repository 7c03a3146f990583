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
  accumulated), and each client's outputs are bit-identical in both.

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


def sampled_segments(cfg):
    """(client, row) pairs to check: first and last; shortest and longest if ragged."""
    picks = {(0, 0), (cfg.K - 1, cfg.client_batch - 1)}
    if len(set(cfg.seq_lens)) > 1:
        picks.add((int(np.argmin(cfg.seq_lens)), 0))
        picks.add((int(np.argmax(cfg.seq_lens)), 0))
    return sorted(picks)


def run_workload(F, weights, cfg, n_oracle_segments=None, serial=True):
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


def test_stack26_fullsize(F, weights):
    """26 blocks, K=8 clients x 4 rows x 256 tokens (T=8192), the bench workload."""
    run_workload(F, weights, syn.CONFIGS["stack26"])


def test_ragged26_fullsize(F, weights):
    """26 blocks, K=16 clients x 1 row, lengths U[64,1024] (seed 7), no padding."""
    run_workload(F, weights, syn.CONFIGS["ragged26"])


def test_sweep26_K32_fullsize(F, weights):
    """The largest sweep point: K=32 clients x 2 rows x 512 tokens (T=32768)."""
    run_workload(F, weights, syn.sweep_config(32), n_oracle_segments=1, serial=False)
