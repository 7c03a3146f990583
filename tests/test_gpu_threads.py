"""Launch set-up under concurrent first calls.

The launchers keep per-device state that their first call sets up (a kernel's dynamic
shared-memory limit, the SM count, the CTA-pair GEMM's resident-cluster count).  A fresh
process here makes its first call of every kernel from four host threads at once, each
on its own stream (ctypes releases the GIL, so the calls overlap inside the library);
every thread's results must equal, bit for bit, the same calls made afterwards by one
thread.  The kernels involved are deterministic (no atomics on these paths).
"""
import os
import subprocess
import sys

import pytest

from _gpu import need_gpu

pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

CHILD = r"""
import sys, threading
import numpy as np
import torch
sys.path.insert(0, sys.argv[1])
from paper_2406_14898_gb300 import flglm as F

F.lib()
rng = np.random.default_rng(11)
dev = "cuda"
def bf(shape, s=1.0):
    return torch.from_numpy((s * rng.standard_normal(shape)).astype(np.float32)).to(dev).bfloat16()

# GEMM inputs (A [M, K], B [N, K], both K-major), LayerNorm rows, attention over two segments
M, N, K = 512, 512, 256
A, B = bf((M, K)), bf((N, K), 0.1)
T, H = 64, 1024
x = bf((T, H))
gamma = torch.ones(H, device=dev)
beta = torch.zeros(H, device=dev)
TA, NH, HD = 256, 2, 128
HA = NH * HD
qkv = bf((TA, 3 * HA))
cu_host = np.array([0, 100, TA], np.int32)
cu_dev = torch.from_numpy(cu_host).to(dev)
n_tiles = F.fl_k_attention_tiles(cu_host)
torch.cuda.synchronize()

def run(stream):
    out = {}
    with torch.cuda.stream(stream):
        for tile in (F.FL_TILE_256x256_PAIR, F.FL_TILE_128x256, F.FL_TILE_128x128):
            D = torch.empty((M, N), device=dev, dtype=torch.bfloat16)
            F.gemm(M, N, K, A, K, 0, B, K, 0, D, N, tile=tile, stream=stream)
            out[f"gemm{tile}"] = D
        y = torch.empty((T, H), device=dev, dtype=torch.bfloat16)
        mean = torch.empty(T, device=dev)
        rstd = torch.empty(T, device=dev)
        F.fl_k_layernorm_fwd(T, H, x, gamma, beta, 1e-5, y, mean, rstd, stream=stream)
        out["ln"] = y
        tile_ws = torch.empty(2 * n_tiles, device=dev, dtype=torch.int32)
        o = torch.empty((TA, HA), device=dev, dtype=torch.bfloat16)
        lse = torch.empty((NH, TA), device=dev)
        F.fl_k_attention_fwd(TA, NH, HD, qkv, cu_host, cu_dev, tile_ws, o, lse, stream=stream)
        out["attn_o"] = o
        out["attn_lse"] = lse
    stream.synchronize()
    return out

n = 4
streams = [torch.cuda.Stream() for _ in range(n)]
results = [None] * n
errors = []
start = threading.Barrier(n)
def worker(i):
    try:
        start.wait()
        results[i] = run(streams[i])
    except Exception as e:  # reported below; the test fails on any
        errors.append(repr(e))
threads = [threading.Thread(target=worker, args=(i,)) for i in range(n)]
for t in threads:
    t.start()
for t in threads:
    t.join()
assert not errors, errors
ref = run(torch.cuda.Stream())
for i, r in enumerate(results):
    for k, v in ref.items():
        assert torch.equal(r[k], v), (i, k)
print("ok", sorted(ref))
"""


def test_concurrent_first_calls_from_threads():
    need_gpu()
    from _gpu import flglm
    flglm()  # builds the library if needed, before the child loads it
    p = subprocess.run([sys.executable, "-c", CHILD, ROOT], capture_output=True, text=True, timeout=600)
    assert p.returncode == 0, p.stdout[-2000:] + p.stderr[-4000:]
    assert p.stdout.strip().startswith("ok")
