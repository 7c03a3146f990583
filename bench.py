"""Throughput of the client-batched FL-GLM server step on GB300.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--workload stack26] [--impl reference]

A step is one pass of the whole server hot path for one call: pack the K clients'
hidden states, forward through the block stack, unpack; pack the output-state
gradients, backward through the stack (input-state and weight gradients), unpack;
one AdamW update.  `value` is tokens/s of the whole job with the inputs resident in
HBM; `e2e` repeats the measurement through host (pinned) buffers with the
host<->device copies of every step inside the timed region.  The default workload is
the 26-block ChatGLM-6B-shaped server stack with K=8 clients x 4 rows x 256 tokens.

Under torchrun (N > 1) each rank runs an independent replica of the server (the path
is one GPU; there is no collective on the data path) and `value` counts every rank's
tokens over the slowest rank's time.

--impl reference times the fp32 C++ CPU oracle on a bounded sample of the same workload
(the repository's reference arm; rank 0 only).
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import numpy as np  # noqa: E402

import synthetic as syn  # noqa: E402

METRIC = "server fwd+bwd tokens/s, client-batched GLM stack bf16; % of BF16 peak"


def workload(name: str) -> syn.ServerConfig:
    if name.startswith("sweep26_K"):
        return syn.sweep_config(int(name[len("sweep26_K"):]))
    return syn.CONFIGS[name]


def describe(cfg: syn.ServerConfig) -> str:
    lens = sorted(set(cfg.seq_lens))
    L = f"{lens[0]}" if len(lens) == 1 else f"{min(lens)}..{max(lens)} (ragged)"
    d = (f"{cfg.name}: {cfg.n_blocks} GLM blocks, hidden {cfg.hidden}, {cfg.n_heads} heads x {cfg.head_dim}, "
         f"FFN {cfg.ffn_hidden}, K={cfg.K} clients x {cfg.client_batch} rows x {L} tokens, T={cfg.tokens}")
    if cfg.prefix_len:
        d += f", P-tuning v2 prefix of {cfg.prefix_len} per block" + (", block weights frozen" if cfg.freeze_base else "")
    if cfg.glm:
        d += (", GLM blank-infilling segments (bidirectional context, causal answer span of 1..L/4 tokens, "
              "2D rotary positions)")
    return d


def config_dict(cfg: syn.ServerConfig, world: int = 1, recompute: bool = False) -> dict:
    """The `config` object of the JSON line; the GPU arm and the reference arm print the same one."""
    return {"workload": describe(cfg), "global_batch": world * cfg.tokens, "seq_len": max(cfg.seq_lens),
            "parallelism": "replicas" if world > 1 else "single GPU",
            "l2": "working set (~125 GB of weights, optimizer state and activations) is far larger "
                  "than L2; no flush needed",
            "step": "pack + forward + unpack + backward with the AdamW update of every parameter "
                    "(fl_server_forward + fl_server_backward_step: the weight-matrix update runs in "
                    "the weight-gradient GEMM epilogues)",
            "recompute": (f"on: each block's activations recomputed in the backward "
                          f"({recompute_flops(cfg) / 1e12:.1f} TFLOP per step beyond the algorithmic "
                          f"FLOPs; counted in roofline.achieved, not in pct_bf16_peak)")
            if recompute else "off: every activation kept"}


def glm_args(cfg: syn.ServerConfig) -> dict:
    """forward() keyword arguments of a workload: the GLM structure when it has one."""
    if not cfg.glm:
        return {}
    ctx, mp = syn.glm_structure(cfg)
    return {"context_lens": ctx, "mask_pos": mp}


def gemm_flops(cfg: syn.ServerConfig) -> float:
    """Dense contractions of one fwd+bwd: forward 2T(3H^2 + H^2 + 2HF) per block, data
    and weight gradients the same again each (no weight gradients with a frozen base)."""
    H, F, T = cfg.hidden, cfg.ffn_hidden, cfg.tokens
    passes = 2 if cfg.freeze_base else 3
    return float(cfg.n_blocks * passes * 2 * T * (4 * H * H + 2 * H * F))


def recompute_flops(cfg: syn.ServerConfig) -> float:
    """GEMM work the backward repeats with activation recompute: the QKV, dense and FFN-up
    forward contractions of every block, 2T(3H^2 + H^2 + HF) each (not algorithmic work)."""
    H, F, T = cfg.hidden, cfg.ffn_hidden, cfg.tokens
    return float(cfg.n_blocks * 2 * T * (4 * H * H + H * F))


def attn_flops(cfg: syn.ServerConfig) -> float:
    """Attention: 4 H FLOPs per visible (query, key) pair forward and 2.5x that backward,
    per block.  Causal: L (L+1) / 2 pairs per segment; a GLM segment with context c sees
    c^2 + (L (L+1) - c (c+1)) / 2; a prefix of Lp keys adds L Lp."""
    Lp = cfg.prefix_len
    ctx = syn.glm_structure(cfg)[0] if cfg.glm else [0] * len(cfg.segment_lengths)
    pairs = sum(c * c + (L * (L + 1) - c * (c + 1)) / 2 + L * Lp for L, c in zip(cfg.segment_lengths, ctx))
    return float(cfg.n_blocks * 3.5 * 4 * cfg.hidden * pairs)


def peaks() -> dict:
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        d = json.load(open(p))
        return {"hbm_gbs": d["hbm_gbs"], "bf16": d["bf16_tflops"], "bf16_sustained": d["bf16_tflops_sustained"],
                "source": "measured"}
    return {"hbm_gbs": 6800.0, "bf16": 1900.0, "bf16_sustained": 1700.0, "source": "fallback"}


# ----------------------------------------------------------------------------- clocks

class ClockSampler:
    """nvidia-smi samples every 200 ms while the timed region runs."""
    Q = ("index,pci.bus_id,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
         "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, bus_id: str | None):
        self.bus_id = bus_id
        self.proc = None
        self.path = None

    def start(self):
        try:
            fd, self.path = tempfile.mkstemp(suffix=".csv")
            os.close(fd)
            cmd = ["nvidia-smi", f"--query-gpu={self.Q}", "--format=csv,noheader,nounits", "-lms", "200"]
            if self.bus_id:
                cmd += ["-i", self.bus_id]
            self.proc = subprocess.Popen(cmd, stdout=open(self.path, "w"), stderr=subprocess.DEVNULL)
        except Exception:
            self.proc = None

    def stop(self) -> dict:
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        with open(self.path) as fh:
            text = fh.read()
        rows = [l.split(", ") for l in text.strip().splitlines() if l.strip()]
        os.unlink(self.path)
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for r in rows:
            if len(r) < 10:
                continue
            try:
                sm.append(float(r[2]))
                mx.append(float(r[3]))
            except ValueError:
                continue
            for i, n in enumerate(names):
                if r[6 + i].strip().lower() == "active":
                    reasons.add(n)
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": max(mx) if mx else None,
                "reasons": sorted(reasons), "samples": len(sm)}


# ----------------------------------------------------------------------------- oracle CPU sample

class OracleSample:
    """Times the fp32 C++ oracle (oracle/flglm_oracle32.cpp, OpenMP over the host cores) on a
    bounded sample of `cfg`'s step: forward + backward of one block at the workload's shapes
    over `tokens` tokens (segments of the workload's first length), and one AdamW update over
    1/ADAM_FRACTION of that block's parameters.  The full step is estimated as
    n_blocks x (t_fwd_bwd x T / tokens + t_adamw x ADAM_FRACTION).  GLM and prefix workloads
    are timed on their plain-causal block (the fp32 oracle covers the base path)."""
    ADAM_FRACTION = 16

    def __init__(self, cfg: syn.ServerConfig, tokens: int, seed: int = 0):
        from oracle import oracle32 as O32
        self.O32 = O32
        self.cfg = cfg
        rng = np.random.default_rng(seed)
        L = min(cfg.segment_lengths[0], tokens)
        self.nseg = max(1, tokens // L)
        self.L = L
        self.one = cfg.with_(n_blocks=1, client_batch=1, seq_lens=(L,) * self.nseg, prefix_len=0, glm=0)
        shapes = syn.param_shapes(self.one)
        params = [[(cfg.init_std * rng.standard_normal(s)).astype(np.float32) for s in shapes]]
        for t, v in ((syn.T_G1, 1.0), (syn.T_G2, 1.0), (syn.T_BE1, 0.0), (syn.T_BE2, 0.0)):
            params[0][t][:] = v
        self.params = params
        self.grads = [[np.zeros(s, np.float32) for s in shapes]]
        T = self.nseg * L
        self.cu = np.arange(self.nseg + 1, dtype=np.int32) * L
        self.x = rng.standard_normal((T, cfg.hidden)).astype(np.float32)
        self.dy = (1e-3 * rng.standard_normal((T, cfg.hidden))).astype(np.float32)
        n = sum(p.size for p in params[0]) // self.ADAM_FRACTION
        self.adam = [(rng.standard_normal(n) * 0.02).astype(np.float32),
                     (rng.standard_normal(n) * 1e-3).astype(np.float32), np.zeros(n, np.float32),
                     np.zeros(n, np.float32)]

    def run(self) -> dict:
        cfg, O32 = self.cfg, self.O32
        t0 = time.perf_counter()
        O32.server_fwd_bwd(self.one, self.params, self.grads, self.cu, self.x, self.dy)
        t1 = time.perf_counter()
        w, g, m, v = self.adam
        O32.adamw(w, g, m, v, 1, cfg.lr, cfg.adam_beta1, cfg.adam_beta2, cfg.adam_eps, cfg.weight_decay)
        t2 = time.perf_counter()
        sample_tokens = self.nseg * self.L
        t_step = cfg.n_blocks * ((t1 - t0) * cfg.tokens / sample_tokens + (t2 - t1) * self.ADAM_FRACTION)
        return {"t_fwd_bwd_s": t1 - t0, "t_adamw_s": t2 - t1, "sample_tokens": sample_tokens,
                "t_sample_s": t2 - t0, "t_step_s": t_step, "tokens_per_s": cfg.tokens / t_step,
                "dtype": "f32", "cores": O32.threads(),
                "rule": (f"full step = n_blocks x (t_fwd_bwd x {cfg.tokens}/{sample_tokens} + t_adamw x "
                         f"{self.ADAM_FRACTION})"),
                "sample": (f"1 of {cfg.n_blocks} blocks at the workload's shapes, {self.nseg} segment(s) x {self.L} "
                           f"tokens fwd+bwd, plus AdamW over 1/{self.ADAM_FRACTION} of that block's parameters; "
                           f"fp32 C++ oracle (plain loops, OpenMP on {O32.threads()} threads, no BLAS); full step "
                           f"estimated as n_blocks x (t_fwd_bwd x {cfg.tokens}/{sample_tokens} + t_adamw x "
                           f"{self.ADAM_FRACTION})")}


def cpu_cores() -> int:
    try:
        return len(os.sched_getaffinity(0))
    except Exception:
        return os.cpu_count() or 1


def run_reference(args, cfg: syn.ServerConfig):
    """The reference arm: the oracle as it stands, on the host cores.  Each of the K timed
    steps is one bounded sample of the workload (see OracleSample); `ms_per_step` is the
    sample's own measured time, and `value` the workload's tokens/s extrapolated from it
    (flagged, with the factor)."""
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return
    sample = OracleSample(cfg, min(cfg.tokens, args.ref_tokens))
    for _ in range(args.warmup):
        sample.run()
    runs = []
    t0 = time.perf_counter()
    for _ in range(args.steps):
        runs.append(sample.run())
    wall = time.perf_counter() - t0
    t_sample = statistics.mean(r["t_sample_s"] for r in runs)
    t_step = statistics.mean(r["t_step_s"] for r in runs)
    value = cfg.tokens / t_step
    last = runs[-1]
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": "tokens/s", "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * t_sample,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": last["dtype"],
            "data": "synthetic", "config": config_dict(cfg, int(os.environ.get("WORLD_SIZE", "1"))),
            "extrapolated": True,
            "extrapolation": {"factor": t_step / t_sample,
                              "basis": "each timed step is one sample (ms_per_step is its measured time); value = "
                                       "the workload's tokens / (sample time x factor), " + last["rule"],
                              "sample_tokens": last["sample_tokens"], "timed_wall_s": wall},
            "cpu_baseline": {"value": value, "unit": "tokens/s", "cores": last["cores"], "kind": "oracle",
                             "sample": last["sample"]},
            "e2e": {"value": value, "unit": "tokens/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


# ----------------------------------------------------------------------------- GPU arm

def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=10)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--workload", default="stack26")
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-other-configs", action="store_true",
                    help="skip the ragged workload and the packed-vs-sequential points after the main line")
    ap.add_argument("--cpu-tokens", type=int, default=256, help="tokens of the oracle sample")
    ap.add_argument("--ref-tokens", type=int, default=256, help="tokens of the reference-arm sample")
    ap.add_argument("--sweep", action="store_true",
                    help="client-batching sweep: 26 blocks, 2 x 512 tokens per client, K in 1..32, "
                         "one packed call vs K sequential single-client calls (one JSON line per K)")
    ap.add_argument("--hierarchical", type=int, default=0, metavar="K",
                    help="the paper's three server strategies for K clients of 2 x 512 tokens on the 26-block "
                         "stack: K server replicas (one per client, averaged every --period steps), one "
                         "client-batched server, and one server taking the clients one after another")
    ap.add_argument("--period", type=int, default=50, help="averaging period of --hierarchical (steps)")
    ap.add_argument("--ptuning", type=int, default=0, metavar="LP",
                    help="P-tuning v2, the paper's training setting: LP prefix keys/values per block, block "
                         "weights frozen, only the prefixes trained")
    ap.add_argument("--split", action="store_true",
                    help="the whole split-learning round: K client models (embedding + block 0, block N-1 + head "
                         "+ cross-entropy) around the client-batched server, one GPU")
    ap.add_argument("--glm", action="store_true",
                    help="GLM blank-infilling segments (the paper's task format): each segment a bidirectional "
                         "context with a mask token and a causal answer span, GLM 2D positions")
    ap.add_argument("--recompute", action="store_true",
                    help="keep only the block inputs and recompute each block's activations in the backward "
                         "(for workloads whose activations do not fit, e.g. --workload sweep26_K64)")
    ap.add_argument("--ncu-traffic", default=os.path.join(ROOT, "profiles", "gemm_pair_up_fwd_stack26.md"))
    args = ap.parse_args()
    cfg = workload(args.workload)
    if args.ptuning:
        cfg = cfg.with_(prefix_len=args.ptuning, freeze_base=1)
    if args.glm:
        cfg = cfg.with_(glm=1)
    if args.impl == "reference":
        run_reference(args, cfg)
        return
    if args.sweep:
        run_sweep(args)
        return
    if args.hierarchical:
        run_strategies(args, args.hierarchical)
        return
    if args.split:
        run_split(args, cfg)
        return

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local_rank = int(os.environ.get("LOCAL_RANK", "0"))
    if args.warmup < 3:
        raise SystemExit("--warmup must be >= 3")

    # oracle CPU sample first (rank 0, one GPU): no CUDA context exists yet
    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        sample = OracleSample(cfg, min(cfg.tokens, args.cpu_tokens))
        cpu = sample.run()
        del sample

    import torch
    import torch.distributed as dist
    from paper_2406_14898_gb300 import flglm as F

    torch.cuda.set_device(local_rank)
    if world > 1:
        dist.init_process_group("nccl" if torch.cuda.is_available() else "gloo")
    dev = torch.device("cuda", local_rank)
    F.lib()
    stream = torch.cuda.Stream(device=dev)
    srv = F.Server(F.make_cfg(cfg, cfg.tokens, max(cfg.seq_lens), recompute=int(args.recompute)), cfg.seed,
                   stream=stream)

    states_bits = syn.client_states(cfg)
    grads_bits = syn.client_grads(cfg)

    def to_dev(b):
        return torch.from_numpy(b.view(np.int16)).view(torch.bfloat16).to(dev)

    states = [to_dev(s) for s in states_bits]
    gouts = [to_dev(g) for g in grads_bits]
    outs = [torch.empty_like(s) for s in states]
    gins = [torch.empty_like(s) for s in states]
    torch.cuda.synchronize()
    free_b, total_b = torch.cuda.mem_get_info(dev)

    gk = glm_args(cfg)

    def step():
        srv.forward(states, cfg.seq_lens, outs, **gk)
        srv.backward_step(gouts, gins, cfg.lr)

    def barrier():
        if world > 1:
            dist.barrier()

    def max_over_ranks(x: float) -> float:
        return slowest_rank_ms(x, world, dev)

    for _ in range(args.warmup):
        step()
    srv.sync()

    # ---- device-resident timed region (no per-launch events: consecutive kernels overlap
    # their launch with the previous kernel's tail)
    clocks = ClockSampler(pci_bus_id(torch, dev))
    clocks.start()
    l0 = srv.launch_count()
    barrier()
    torch.cuda.synchronize()
    e0 = torch.cuda.Event(enable_timing=True)
    e1 = torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for _ in range(args.steps):
        step()
    e1.record(stream)
    srv.sync()
    torch.cuda.synchronize()
    barrier()
    ms = e0.elapsed_time(e1)
    launches = srv.launch_count() - l0
    clk = clocks.stop()
    ms = max_over_ranks(ms)
    ms_step = ms / args.steps
    value = job_tokens_per_s(world, cfg.tokens, args.steps, ms)

    # ---- the same steps again with CUDA events around every launch on the library's
    # stream: per-class kernel time and the GEMM's live throughput (the roofline line)
    srv.profile(True)
    barrier()
    torch.cuda.synchronize()
    e0.record(stream)
    for _ in range(args.steps):
        step()
    e1.record(stream)
    srv.sync()
    prof_ms_step = max_over_ranks(e0.elapsed_time(e1)) / args.steps
    prof = srv.profile_read()
    srv.profile(False)
    adam_ms = prof["adamw"][0] / args.steps

    # forward + backward alone (no optimizer), the metric's "fwd+bwd" in the narrow sense
    barrier()
    torch.cuda.synchronize()
    e0.record(stream)
    for _ in range(args.steps):
        srv.forward(states, cfg.seq_lens, outs, **gk)
        srv.backward(gouts, gins)
    e1.record(stream)
    srv.sync()
    barrier()
    fb_ms = max_over_ranks(e0.elapsed_time(e1)) / args.steps
    srv.step(cfg.lr)
    pk = peaks()
    flops = gemm_flops(cfg) + attn_flops(cfg)
    gemm_ms, gemm_n = prof["gemm"]
    # executed contractions per GEMM launch: the recomputed forward GEMMs are work the kernel does
    gemm_exec = gemm_flops(cfg) + (recompute_flops(cfg) if args.recompute else 0.0)
    gemm_per_launch_flops = gemm_exec * args.steps / max(gemm_n, 1)
    achieved = gemm_per_launch_flops / (gemm_ms / max(gemm_n, 1) / 1e3) / 1e12
    traffic = ncu_traffic(args.ncu_traffic, cfg.name)

    # ---- end to end through host buffers (pinned), copies inside the timed region
    e2e = None
    if not args.no_e2e:
        h_states = [torch.from_numpy(s.view(np.int16)).view(torch.bfloat16).pin_memory() for s in states_bits]
        h_gouts = [torch.from_numpy(g.view(np.int16)).view(torch.bfloat16).pin_memory() for g in grads_bits]
        h_outs = [torch.empty(s.shape, dtype=torch.bfloat16).pin_memory() for s in states_bits]
        h_gins = [torch.empty(s.shape, dtype=torch.bfloat16).pin_memory() for s in states_bits]

        def e2e_step():
            with torch.cuda.stream(stream):
                for d, h in zip(states, h_states):
                    d.copy_(h, non_blocking=True)
                srv.forward(states, cfg.seq_lens, outs, **gk)
                for h, d in zip(h_outs, outs):
                    h.copy_(d, non_blocking=True)
                for d, h in zip(gouts, h_gouts):
                    d.copy_(h, non_blocking=True)
                srv.backward_step(gouts, gins, cfg.lr)
                for h, d in zip(h_gins, gins):
                    h.copy_(d, non_blocking=True)

        for _ in range(2):
            e2e_step()
        srv.sync()
        barrier()
        torch.cuda.synchronize()
        t0 = time.perf_counter()
        e0.record(stream)
        for _ in range(args.steps):
            e2e_step()
        e1.record(stream)
        srv.sync()
        torch.cuda.synchronize()
        wall = time.perf_counter() - t0
        barrier()
        ems = max_over_ranks(max(e0.elapsed_time(e1), 1e3 * wall))
        nbytes = sum(s.nbytes for s in states_bits)
        e2e = {"value": job_tokens_per_s(world, cfg.tokens, args.steps, ems), "unit": "tokens/s",
               "h2d_bytes_per_step": 2 * nbytes, "d2h_bytes_per_step": 2 * nbytes,
               "ms_per_step": ems / args.steps}

    srv.close()
    del states, gouts, outs, gins
    torch.cuda.empty_cache()
    others = None
    if world == 1 and args.workload == "stack26" and not (args.ptuning or args.glm or args.recompute) \
            and not args.no_other_configs:
        others = run_other_configs(max(3, min(args.steps, 5)), 3, dev, stream)
    if rank == 0:
        line = {
            "metric": METRIC, "value": value, "unit": "tokens/s", "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": ms_step, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "bf16", "data": "synthetic (seeded N(0,0.02) weights, N(0,1) states, "
                                                       "N(0,1e-3) output-state grads)",
            "config": config_dict(cfg, world, args.recompute),
            "pct_bf16_peak": 100.0 * flops / (ms_step / 1e3) / (pk["bf16_sustained"] * 1e12),
            "pct_bf16_peak_basis": f"algorithmic FLOPs (GEMM + causal attention) of the whole step over the "
                                   f"{pk['source']} sustained bf16 peak {pk['bf16_sustained']} TFLOP/s",
            "fwd_bwd_tokens_per_s": world * cfg.tokens / (fb_ms / 1e3),
            "fwd_bwd_ms": fb_ms,
            "fwd_bwd_basis": "separate timed loop of fl_server_forward + fl_server_backward, no optimizer step",
            "vector_adamw_ms": adam_ms,
            "kernel_ms_per_step": {k: v[0] / args.steps for k, v in prof.items()},
            "kernel_ms_basis": (f"a second timed region of the same {args.steps} steps with CUDA events around every "
                                f"launch ({prof_ms_step:.2f} ms per step there)"),
            "roofline": {"kernel": "gemm_pair_kernel (tcgen05.mma.cta_group::2, 256 x 256 tiles on SM pairs)", "bound": "tensor", "achieved": achieved,
                         "peak": pk["bf16_sustained"], "unit": "TFLOP/s", "frac": achieved / pk["bf16_sustained"],
                         "peak_basis": f"{pk['source']} sustained bf16 (kernel timed inside a long step)",
                         "traffic": traffic["bytes_per_launch"] if traffic else None,
                         "traffic_basis": (f"{traffic['launch']}, one ncu capture ({traffic['source']}); achieved is "
                                           f"the mean over all GEMM launches of the step") if traffic else None,
                         "launches_per_step": gemm_n / args.steps,
                         "share_of_step": gemm_ms / (prof_ms_step * args.steps),
                         "timed_region": "the profiled repeat of the timed steps (kernel_ms_basis)"},
            "gpu_launches": launches,
            "clocks": clk,
            "hbm_used_gb": (total_b - free_b) / 1e9,
        }
        if cpu is not None:
            line["cpu_baseline"] = {"value": cpu["tokens_per_s"], "unit": "tokens/s", "cores": cpu_cores(),
                                    "kind": "oracle", "sample": cpu["sample"]}
        if e2e is not None:
            line["e2e"] = e2e
        if others is not None:
            line["other_configs"] = others
        print(json.dumps(line), flush=True)
    if world > 1:
        dist.destroy_process_group()


def slowest_rank_ms(ms: float, world: int, device=None) -> float:
    """The timed region's duration of the slowest rank (all-reduce MAX); the job's time."""
    if world == 1:
        return ms
    import torch
    import torch.distributed as dist
    t = torch.tensor([ms], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_tokens_per_s(world: int, tokens_per_rank: int, steps: int, ms: float) -> float:
    """Whole-job throughput: every rank's tokens over the slowest rank's time (replicas,
    weak scaling: each rank serves its own clients)."""
    return world * tokens_per_rank * steps / (ms / 1e3)


def run_sweep(args):
    """Client-batching sweep (§3.3): for each K, the K clients' step as one packed call
    (client-batch) and as K single-client calls followed by one AdamW update (serial),
    on one server sized for the largest K."""
    import torch
    from paper_2406_14898_gb300 import flglm as F

    ks = syn.SWEEP_KS
    big = syn.sweep_config(max(ks))
    F.lib()
    dev = torch.device("cuda", 0)
    stream = torch.cuda.Stream(device=dev)
    srv = F.Server(F.make_cfg(big, big.tokens, max(big.seq_lens)), big.seed, stream=stream)
    sb = syn.client_states(big)
    gb = syn.client_grads(big)
    st = [torch.from_numpy(b.view(np.int16)).view(torch.bfloat16).to(dev) for b in sb]
    go = [torch.from_numpy(b.view(np.int16)).view(torch.bfloat16).to(dev) for b in gb]
    outs = [torch.empty_like(s) for s in st]
    gin = [torch.empty_like(s) for s in st]
    for K in ks:
        cfg = syn.sweep_config(K)
        res = sweep_point(srv, K, st, go, outs, gin, args.steps, args.warmup, stream)
        line = {"metric": METRIC, "mode": "client-batching sweep", "K": K, "value": res["batched"]["tokens_per_s"],
                "unit": "tokens/s", "n_gpus": 1, "steps": args.steps, "warmup": args.warmup,
                "higher_is_better": True, "dtype": "bf16", "data": "synthetic",
                "config": {"workload": describe(cfg), "global_batch": cfg.tokens, "seq_len": 512},
                "batched": res["batched"], "sequential": res["sequential"],
                "batched_over_sequential": res["batched"]["tokens_per_s"] / res["sequential"]["tokens_per_s"]}
        print(json.dumps(line), flush=True)
    srv.close()


def sweep_point(srv, K: int, st, go, outs, gin, steps: int, warmup: int, stream) -> dict:
    """One client-batching point (§3.3) on a server sized for at least K clients of the
    sweep workload: the K clients' step as one packed call (client-batch) and as K
    single-client calls followed by one AdamW update (serial), CUDA events on `stream`."""
    import torch
    cfg = syn.sweep_config(K)
    pk = peaks()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)

    def batched():
        srv.forward(st[:K], cfg.seq_lens, outs[:K])
        srv.backward_step(go[:K], gin[:K], cfg.lr)

    def sequential():
        for k in range(K):
            srv.forward(st[k:k + 1], cfg.seq_lens[k:k + 1], outs[k:k + 1])
            srv.backward(go[k:k + 1], gin[k:k + 1])
        srv.step(cfg.lr)

    res = {}
    for name, fn in (("batched", batched), ("sequential", sequential)):
        for _ in range(warmup):
            fn()
        srv.sync()
        e0.record(stream)
        for _ in range(steps):
            fn()
        e1.record(stream)
        srv.sync()
        ms = e0.elapsed_time(e1) / steps
        res[name] = {"tokens_per_s": cfg.tokens / (ms / 1e3), "ms_per_step": ms, "steps": steps, "warmup": warmup,
                     "pct_bf16_peak": 100.0 * (gemm_flops(cfg) + attn_flops(cfg)) / (ms / 1e3)
                     / (pk["bf16_sustained"] * 1e12)}
    return res


def dev_bf16(torch, bits_list, dev):
    return [torch.from_numpy(b.view(np.int16)).view(torch.bfloat16).to(dev) for b in bits_list]


def run_other_configs(steps: int, warmup: int, dev, stream) -> dict:
    """The workload's sibling configurations, a few steps each, on fresh servers after the
    main measurement: the ragged client-batching workload (26 blocks, K=16 clients x 1 row,
    lengths U[64,1024] drawn with seed 7) and the client-batching sweep (26 blocks, K in
    1..32 clients x 2 x 512 tokens, one server sized for K=32): one packed call against K
    single-client calls."""
    import torch
    from paper_2406_14898_gb300 import flglm as F
    pk = peaks()
    out = {}
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    cfg = syn.CONFIGS["ragged26"]
    srv = F.Server(F.make_cfg(cfg, cfg.tokens, max(cfg.seq_lens)), cfg.seed, stream=stream)
    st, go = dev_bf16(torch, syn.client_states(cfg), dev), dev_bf16(torch, syn.client_grads(cfg), dev)
    outs, gin = [torch.empty_like(x) for x in st], [torch.empty_like(x) for x in st]
    for _ in range(warmup):
        srv.forward(st, cfg.seq_lens, outs)
        srv.backward_step(go, gin, cfg.lr)
    srv.sync()
    e0.record(stream)
    for _ in range(steps):
        srv.forward(st, cfg.seq_lens, outs)
        srv.backward_step(go, gin, cfg.lr)
    e1.record(stream)
    srv.sync()
    ms = e0.elapsed_time(e1) / steps
    out[cfg.name] = {"workload": describe(cfg), "tokens": cfg.tokens, "steps": steps, "warmup": warmup,
                     "ms_per_step": ms, "tokens_per_s": cfg.tokens / (ms / 1e3),
                     "pct_bf16_peak": 100.0 * (gemm_flops(cfg) + attn_flops(cfg)) / (ms / 1e3)
                     / (pk["bf16_sustained"] * 1e12)}
    srv.close()
    del st, go, outs, gin
    torch.cuda.empty_cache()
    big = syn.sweep_config(max(OTHER_SWEEP_KS))
    srv = F.Server(F.make_cfg(big, big.tokens, max(big.seq_lens)), big.seed, stream=stream)
    st, go = dev_bf16(torch, syn.client_states(big), dev), dev_bf16(torch, syn.client_grads(big), dev)
    outs, gin = [torch.empty_like(x) for x in st], [torch.empty_like(x) for x in st]
    for K in OTHER_SWEEP_KS:
        cfg = syn.sweep_config(K)
        r = sweep_point(srv, K, st, go, outs, gin, steps, warmup, stream)
        out[cfg.name] = {"workload": describe(cfg), "tokens": cfg.tokens, **r,
                         "batched_over_sequential": r["batched"]["tokens_per_s"] / r["sequential"]["tokens_per_s"]}
    srv.close()
    del st, go, outs, gin
    torch.cuda.empty_cache()
    return out


OTHER_SWEEP_KS = syn.SWEEP_KS


def run_strategies(args, K: int):
    """§3.3 strategies on one GPU for K clients of 2 x 512 tokens (the 26-block stack):
    server-hierarchical (K replicas, one client each, parameters averaged every period),
    client-batch (one server, the K clients packed in one call) and serial (one server, the
    clients one call after another, one update)."""
    import torch
    from paper_2406_14898_gb300 import flglm as F
    from paper_2406_14898_gb300.hierarchical import BatchedReplicas, HierarchicalServers

    cfg = syn.sweep_config(K)
    one = cfg.with_(seq_lens=cfg.seq_lens[:1])
    dev = torch.device("cuda", 0)
    sb, gb = syn.client_states(cfg), syn.client_grads(cfg)
    st = [torch.from_numpy(b.view(np.int16)).view(torch.bfloat16).to(dev) for b in sb]
    go = [torch.from_numpy(b.view(np.int16)).view(torch.bfloat16).to(dev) for b in gb]
    outs = [torch.empty_like(s) for s in st]
    gin = [torch.empty_like(s) for s in st]
    pk = peaks()
    flops = gemm_flops(cfg) + attn_flops(cfg)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    res = {}

    def timed(fn, sync):
        for _ in range(args.warmup):
            fn()
        sync()
        torch.cuda.synchronize()
        t0 = time.perf_counter()
        for _ in range(args.steps):
            fn()
        sync()
        torch.cuda.synchronize()
        return 1e3 * (time.perf_counter() - t0) / args.steps

    # server-hierarchical: K replicas on their own streams
    hs = HierarchicalServers(F.make_cfg(one, one.tokens, 512), cfg.seed, K)
    ms = timed(lambda: hs.step(st, cfg.seq_lens, outs, go, gin, cfg.lr), hs.sync)
    t0 = time.perf_counter()
    hs.average()
    avg_ms = 1e3 * (time.perf_counter() - t0)
    hs.close()
    torch.cuda.empty_cache()
    amort = ms + avg_ms / args.period
    res["server_hierarchical"] = {"replicas": K, "ms_per_step": ms, "average_ms": avg_ms, "period": args.period,
                                  "tokens_per_s": cfg.tokens / (amort / 1e3),
                                  "pct_bf16_peak": 100.0 * flops / (amort / 1e3) / (pk["bf16_sustained"] * 1e12)}
    # the same K replicas held in one handle, every block GEMM one batched launch
    if 2 <= K <= F.FL_GEMM_MAX_BATCH:
        br = BatchedReplicas(F.make_cfg(cfg, cfg.tokens, 512), cfg.seed, K)
        ms = timed(lambda: br.step(st, cfg.seq_lens, outs, go, gin, cfg.lr), br.sync)
        t0 = time.perf_counter()
        br.average()
        br.sync()
        avg_ms = 1e3 * (time.perf_counter() - t0)
        br.close()
        torch.cuda.empty_cache()
        amort = ms + avg_ms / args.period
        res["server_hierarchical_batched"] = {
            "replicas": K, "ms_per_step": ms, "average_ms": avg_ms, "period": args.period,
            "tokens_per_s": cfg.tokens / (amort / 1e3),
            "pct_bf16_peak": 100.0 * flops / (amort / 1e3) / (pk["bf16_sustained"] * 1e12)}
    # client-batch and serial on one server
    srv = F.Server(F.make_cfg(cfg, cfg.tokens, 512), cfg.seed)

    def batched():
        srv.forward(st, cfg.seq_lens, outs)
        srv.backward_step(go, gin, cfg.lr)

    def serial():
        for k in range(K):
            srv.forward(st[k:k + 1], cfg.seq_lens[k:k + 1], outs[k:k + 1])
            srv.backward(go[k:k + 1], gin[k:k + 1])
        srv.step(cfg.lr)

    for name, fn in (("client_batch", batched), ("serial", serial)):
        ms = timed(fn, srv.sync)
        res[name] = {"ms_per_step": ms, "tokens_per_s": cfg.tokens / (ms / 1e3),
                     "pct_bf16_peak": 100.0 * flops / (ms / 1e3) / (pk["bf16_sustained"] * 1e12)}
    srv.close()
    line = {"metric": METRIC, "mode": "server strategies (Sec. 3.3)", "K": K,
            "value": res["client_batch"]["tokens_per_s"], "unit": "tokens/s", "n_gpus": 1, "steps": args.steps,
            "warmup": args.warmup, "higher_is_better": True, "dtype": "bf16", "data": "synthetic",
            "config": {"workload": describe(cfg), "global_batch": cfg.tokens, "seq_len": 512},
            "timing": "host wall clock around the timed steps, after a device synchronisation on both sides",
            **res}
    print(json.dumps(line), flush=True)


def client_flops(cfg: syn.ServerConfig) -> float:
    """Dense work of the K clients in one round: two blocks each (the server's block FLOPs,
    GEMM + attention, per block) and the LM head (forward and data gradient, plus the weight
    gradient when the head is trained); the embedding is a gather."""
    per_block = (gemm_flops(cfg) + attn_flops(cfg)) / cfg.n_blocks
    head_passes = 2 if cfg.freeze_base else 3
    vp = (cfg.vocab + 255) // 256 * 256
    return 2 * per_block + head_passes * 2.0 * cfg.tokens * cfg.hidden * vp


def run_split(args, cfg: syn.ServerConfig):
    """The whole split-learning round of §3.1 on one GPU: K clients (each its own client
    model: embedding + block 0, block N-1 + final LayerNorm + LM head + cross-entropy) and
    the client-batched server, all on one stream:
      K bottom forwards -> server forward (one packed call) -> K top forward/backward ->
      server backward with the fused update -> K bottom backwards -> K client steps."""
    import torch
    from paper_2406_14898_gb300 import flglm as F

    dev = torch.device("cuda", 0)
    stream = torch.cuda.Stream(device=dev)
    K, b = cfg.K, cfg.client_batch
    srv = F.Server(F.make_cfg(cfg, cfg.tokens, max(cfg.seq_lens)), cfg.seed, stream=stream)
    ccfgs = [cfg.with_(seq_lens=(L,)) for L in cfg.seq_lens]
    clients = [F.Client(F.make_client_cfg(c, c.tokens), cfg.seed, stream=stream) for c in ccfgs]
    gk = glm_args(cfg)
    ctx_all = gk.get("context_lens")
    toks, labs = [], []
    for k in range(K):
        t = syn.client_tokens(cfg, k)
        ctx = None if ctx_all is None else ctx_all[k * b:(k + 1) * b]
        toks.append(torch.from_numpy(t).to(dev))
        labs.append(torch.from_numpy(syn.client_labels(t, ctx)).to(dev))
    h0 = [torch.empty((b, L, cfg.hidden), dtype=torch.bfloat16, device=dev) for L in cfg.seq_lens]
    hs = [torch.empty_like(x) for x in h0]
    gh = [torch.empty_like(x) for x in h0]
    g0 = [torch.empty_like(x) for x in h0]
    loss = torch.zeros(K, dtype=torch.float32, device=dev)
    torch.cuda.synchronize()

    def round_():
        for k in range(K):
            ctx = None if ctx_all is None else ctx_all[k * b:(k + 1) * b]
            mp = None if ctx_all is None else gk["mask_pos"][k * b:(k + 1) * b]
            clients[k].bottom_forward(toks[k], cfg.seq_lens[k], h0[k], ctx, mp)
        srv.forward(h0, cfg.seq_lens, hs, **gk)
        for k in range(K):
            clients[k].top_forward_backward(hs[k], labs[k], loss[k:k + 1], gh[k])
        srv.backward_step(gh, g0, cfg.lr)
        for k in range(K):
            clients[k].bottom_backward(g0[k])
            clients[k].step(cfg.lr)

    for _ in range(args.warmup):
        round_()
    for c in clients:
        c.sync()
    srv.sync()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    l0 = srv.launch_count() + sum(c.launch_count() for c in clients)
    clocks = ClockSampler(pci_bus_id(torch, dev))
    clocks.start()
    torch.cuda.synchronize()
    e0.record(stream)
    for _ in range(args.steps):
        round_()
    e1.record(stream)
    torch.cuda.synchronize()
    clk = clocks.stop()
    ms = e0.elapsed_time(e1) / args.steps
    launches = srv.launch_count() + sum(c.launch_count() for c in clients) - l0
    # the server's share of the round, timed alone the same way
    srv.forward(h0, cfg.seq_lens, hs, **gk)
    srv.backward_step(gh, g0, cfg.lr)
    torch.cuda.synchronize()
    e0.record(stream)
    for _ in range(args.steps):
        srv.forward(h0, cfg.seq_lens, hs, **gk)
        srv.backward_step(gh, g0, cfg.lr)
    e1.record(stream)
    torch.cuda.synchronize()
    srv_ms = e0.elapsed_time(e1) / args.steps
    for c in clients:
        c.sync()
    pk = peaks()
    flops = gemm_flops(cfg) + attn_flops(cfg) + client_flops(cfg)
    line = {"metric": "split-learning round tokens/s (K clients + client-batched server, one GB300)",
            "mode": "split round (Sec. 3.1 protocol)", "value": cfg.tokens / (ms / 1e3), "unit": "tokens/s",
            "n_gpus": 1, "steps": args.steps, "warmup": args.warmup, "ms_per_round": ms, "higher_is_better": True,
            "dtype": "bf16", "data": "synthetic (seeded weights, uniform token ids, next-token labels on the answer "
                                     "span)",
            "config": {"workload": describe(cfg) + f"; clients: vocabulary {cfg.vocab}, embedding + block 0 and "
                                                   "block N-1 + final LayerNorm + LM head + cross-entropy",
                       "global_batch": cfg.tokens, "seq_len": max(cfg.seq_lens)},
            "server_ms_per_round": srv_ms, "clients_ms_per_round": ms - srv_ms,
            "pct_bf16_peak": 100.0 * flops / (ms / 1e3) / (pk["bf16_sustained"] * 1e12),
            "pct_bf16_peak_basis": "algorithmic FLOPs of server and clients over the measured sustained bf16 peak",
            "loss_mean": float(loss.mean().item()), "gpu_launches": launches, "clocks": clk}
    print(json.dumps(line), flush=True)
    for c in clients:
        c.close()
    srv.close()


def pci_bus_id(torch, dev):
    """nvidia-smi id (domain:bus:device.function) of the CUDA device, or None."""
    try:
        p = torch.cuda.get_device_properties(dev)
        return f"{p.pci_domain_id:08X}:{p.pci_bus_id:02X}:{p.pci_device_id:02X}.0"
    except Exception:
        return None


def ncu_traffic(path: str, workload_name: str):
    """DRAM bytes per launch of the GEMM from the committed ncu summary, if it was taken on
    this workload and on the current GEMM source; else None."""
    if not os.path.exists(path) or workload_name not in os.path.basename(path):
        return None
    with open(path) as fh:
        txt = fh.read()
    if kernel_version() not in txt:
        return None
    for line in txt.splitlines():
        if line.startswith("traffic_bytes_per_launch:"):
            return {"bytes_per_launch": int(line.split(":")[1]), "source": os.path.relpath(path, ROOT),
                    "launch": "FFN up-projection forward GEMM (M=8192, N=16384, K=4096)"}
    return None


def kernel_version() -> str:
    """Fingerprint of the GEMM sources (the kernel, its instantiations and the device
    helpers its epilogues call), so that stored ncu traffic is used only for the kernel it
    was measured on."""
    import glob
    import hashlib
    h = hashlib.sha256()
    csrc = os.path.join(ROOT, "paper_2406_14898_gb300", "csrc")
    files = sorted(glob.glob(os.path.join(csrc, "gemm_*"))) + [os.path.join(csrc, "common.cuh"),
                                                                 os.path.join(csrc, "ptx.cuh")]
    for f in files:
        with open(f, "rb") as fh:
            h.update(fh.read())
    return h.hexdigest()[:16]


if __name__ == "__main__":
    main()
