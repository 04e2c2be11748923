#!/usr/bin/env python
"""Benchmark of the DFlow round on GB300.

One step = one dflow_round (draft -> verify -> accept/commit -> carry) over the
whole batch of the Qwen3-8B-shaped workload (bf16 random-init weights, 2048
uniform-random prompt tokens, block 16, seeded uniform{0..16} forced
acceptance), inputs resident in HBM.  Weights (18.7 GB per round) exceed L2, so
no flush is needed between steps.

Prints one JSON line (rank 0).  `--impl reference` times the CPU oracle on a
bounded sample of the same workload instead.
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import threading
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import synth  # noqa: E402

METRIC = "draft+verify round latency & committed tokens/s, Qwen3-8B shape; % HBM roofline"
DEFAULT_CONFIG = "qwen3_8b_b1"
T1_SEED = 4  # seed of the T = 1 leg's draws


def parse():
    p = argparse.ArgumentParser()
    p.add_argument("--gpus", type=int, default=1)
    p.add_argument("--steps", type=int, default=56)
    p.add_argument("--warmup", type=int, default=8)
    p.add_argument("--impl", choices=["ours", "reference"], default="ours")
    # workloads with a forced acceptance schedule (the tiny fp32 model decodes with natural
    # acceptance and serves the parity tests only)
    p.add_argument("--config", default=DEFAULT_CONFIG,
                   choices=sorted(n for n, c in synth.CONFIGS.items() if c.schedule != "natural"))
    p.add_argument("--relay", type=int, default=1, help="0 runs the DFlash baseline (no carry)")
    p.add_argument("--no-cpu-baseline", action="store_true")
    p.add_argument("--no-e2e", action="store_true")
    p.add_argument("--no-other-workloads", action="store_true",
                   help="skip the device legs of the other three bf16 workloads")
    p.add_argument("--profile-only", action="store_true", help="warmup + a few steps, no timing legs (for ncu)")
    p.add_argument("--depth", type=int, default=0,
                   help="with --profile-only: target layers of a reduced-depth copy (same widths), for small ncu captures")
    # one projection through the tcgen05 GEMM alone (timing and ncu captures of that kernel)
    p.add_argument("--kernel", choices=["gemm"], default=None,
                   help="time one kernel instead of the round: gemm = out = X W^T with epilogue --mode")
    p.add_argument("--N", type=int, default=151936)
    p.add_argument("--K", type=int, default=4096)
    p.add_argument("--M", type=int, default=17)
    p.add_argument("--mode", type=int, default=4, help="0 fp32 store, 1 residual add, 2 SwiGLU, 3 SiLU, 4 argmax")
    p.add_argument("--reps", type=int, default=3)
    p.add_argument("--path", type=int, default=1, choices=[1, 2, 3],
                   help="with --kernel gemm: 1 row-tiled tcgen05 launch, 2 persistent launch (16-128 rows), "
                        "3 one-pass launch (above 128 rows)")
    p.add_argument("--cublas", action="store_true",
                   help="with --kernel gemm: also time torch.matmul of the same bf16 tensors (for scale)")
    return p.parse_args()


def peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            pk = json.load(f)
        return float(pk["hbm_gbs"]), float(pk["bf16_tflops"]), "measured"
    except Exception:
        return 6800.0, 1900.0, "fallback"


# --------------------------------------------------------------------------
# algorithmic bytes of one round
# --------------------------------------------------------------------------


def round_bytes(cfg, mean_ctx: float) -> dict:
    """DRAM bytes a round must move at minimum: every weight it reads once, the
    K/V context it attends over, plus the (small) activations.  bf16."""
    es = 2 if cfg.dtype == "bf16" else 4
    d, hd, I, V = cfg.d, cfg.head_dim, cfg.inter, cfg.vocab
    qkv = (cfg.n_q_heads + 2 * cfg.n_kv_heads) * hd * d
    layer = qkv + d * cfg.n_q_heads * hd + 2 * I * d + d * I
    kv_tok = 2 * cfg.n_kv_heads * hd * es
    target_w = (cfg.n_layers * layer + V * d) * es
    draft_w = (cfg.draft_layers * layer + V * d + cfg.n_feat * d * d + 3 * d * d + 2 * d * d
               + cfg.draft_layers * 2 * cfg.n_kv_heads * hd * d) * es
    R = cfg.rows
    kv = cfg.batch * ((mean_ctx + R) * cfg.n_layers + mean_ctx * cfg.draft_layers) * kv_tok
    return dict(weights=target_w + draft_w, kv=kv, total=target_w + draft_w + kv)


# --------------------------------------------------------------------------
# clocks during the timed region
# --------------------------------------------------------------------------


class ClockSampler:
    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.hw_slowdown,"
              "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
              "clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu: int):
        self.gpu, self.proc, self.lines = gpu, None, []

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.gpu), f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                 "-lms", "100"], stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.t = threading.Thread(target=self._read, daemon=True)
            self.t.start()
            time.sleep(0.3)
        except Exception:
            self.proc = None
        return self

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append(line.strip())

    def __exit__(self, *a):
        if self.proc:
            self.proc.terminate()
            self.proc.wait(timeout=5)

    def summary(self):
        sm, mx, reasons = [], 0.0, set()
        names = ("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap")
        for ln in self.lines:
            parts = [x.strip() for x in ln.split(",")]
            if len(parts) < 7:
                continue
            try:
                sm.append(float(parts[0]))
                mx = max(mx, float(parts[1]))
            except ValueError:
                continue
            for n, v in zip(names, parts[3:7]):
                if v.lower().startswith("active"):
                    reasons.add(n)
        if not sm:
            return None
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": mx, "reasons": sorted(reasons), "samples": len(sm)}


# --------------------------------------------------------------------------
# CPU oracle on a bounded sample of the workload
# --------------------------------------------------------------------------


class OracleSample:
    """The oracle's round on a 1-target-layer, 1-draft-layer copy of the workload
    (full width, batch and context) whose LM head and embedding keep one in
    `vocab_div` vocabulary rows.  Timers on the oracle's own calls give the
    per-layer and LM-head costs, from which the full round's time is
    extrapolated: + (L-1) target layers, + (Ld-1) draft layers and context
    appends, and the LM heads scaled back to the full vocabulary."""

    def __init__(self, cfg, vocab_div: int = 32):
        from oracle import Oracle
        self.cfg = cfg
        self.vocab_div = vocab_div
        self.c1 = cfg.replace(n_layers=1, draft_layers=1, feat_layers=(1,), vocab=cfg.vocab // vocab_div)
        self.o = Oracle(self.c1, timing_weights(self.c1))
        lens = synth.prompt_lengths(cfg) + 1
        self.st0 = self.o.state_from_synthetic(synth.synthetic_state(self.c1, ctx_lens=lens,
                                                                     n_carry=np.full(cfg.batch, cfg.block // 2)))
        self.acc = {}
        for name in ("target_forward", "draft_block", "lm_logits", "feature_projection", "draft_inputs", "ctx_append"):
            self._wrap(name)
        self.threads = os.cpu_count()

    def _wrap(self, name):
        f = getattr(self.o, name)

        def w(*a, **k):
            t = time.perf_counter()
            r = f(*a, **k)
            self.acc[name] = self.acc.get(name, 0.0) + time.perf_counter() - t
            return r
        setattr(self.o, name, w)

    def step(self, forced):
        """One sampled round: (measured seconds, extrapolated full-round seconds, committed tokens)."""
        st = self.st0.copy()
        self.acc = {}
        t0 = time.perf_counter()
        ro = self.o.round(st, forced=list(forced))
        t = time.perf_counter() - t0
        a = self.acc
        lm = a.get("lm_logits", 0.0)
        t_tlayer = a["target_forward"] - a.get("feature_projection", 0.0) - lm / 2
        t_dlayer = a["draft_block"] - a.get("draft_inputs", 0.0) - lm / 2
        c = self.cfg
        full = (t + (c.n_layers - 1) * t_tlayer + (c.draft_layers - 1) * (t_dlayer + a.get("ctx_append", 0.0))
                + (self.vocab_div - 1) * lm)
        return t, full, int((ro.accept + 1).sum())

    def describe(self):
        c = self.cfg
        return (f"oracle round (numpy fp64) on a copy of {c.name} with 1 target + 1 draft layer and 1/"
                f"{self.vocab_div} of the vocabulary (full width {c.d}, batch {c.batch}, context as the workload); "
                f"its measured time extrapolated to {c.n_layers}+{c.draft_layers} layers and the full LM head with "
                f"timers on the oracle's own calls")


def timing_weights(cfg):
    """Weights of the workload's shapes for timing the oracle: one random block
    of N(0, 0.02) values reused for every matrix of the same name and shape
    across layers and stacks (the oracle does the full arithmetic of every
    layer; only the values repeat, which keeps host memory at one layer)."""
    block = np.random.default_rng(0).standard_normal(1 << 22, dtype=np.float32) * np.float32(0.02)
    shared, W = {}, {}
    for name, shape in synth.tensor_shapes(cfg).items():
        if len(shape) == 1:
            W[name] = np.zeros(shape, np.float32) if name == "ln_b" else np.ones(shape, np.float32)
            continue
        base = name.split(".", 1)[1] if name[0] in "td" and name[1].isdigit() else name
        key = (base, shape)
        if key not in shared:
            shared[key] = np.resize(block, int(np.prod(shape))).reshape(shape)
        W[name] = shared[key]
    return W


def host_mem_available_gb() -> float:
    try:
        with open("/proc/meminfo") as f:
            for ln in f:
                if ln.startswith("MemAvailable:"):
                    return int(ln.split()[1]) / 2 ** 20
    except OSError:
        pass
    return 0.0


def cpu_baseline_full_round(cfg, timed_sched):
    """The oracle as it stands timed on one full-depth round of the workload
    (every target and draft layer, full vocabulary, width, batch and context;
    synthetic caches, layer-shared weight values), on this host's cores.
    tokens/s = the schedule's mean committed tokens per round over the timed
    rounds / the measured round time."""
    from oracle import Oracle
    mean_commit = float((np.asarray(timed_sched) + 1).sum(axis=1).mean())
    if cfg.batch > 1 or host_mem_available_gb() < 48:
        s = OracleSample(cfg)
        tm, tf, _ = s.step(timed_sched[0])
        return {"value": round(mean_commit / tf, 4), "unit": "tokens/s", "cores": s.threads, "kind": "oracle",
                "sample": s.describe(), "sec_measured": round(tm, 2), "sec_per_round_est": round(tf, 2),
                "mean_committed_per_round": mean_commit}
    o = Oracle(cfg, timing_weights(cfg))
    lens = synth.prompt_lengths(cfg) + 1
    st = o.state_from_synthetic(synth.synthetic_state(cfg, ctx_lens=lens, n_carry=np.full(cfg.batch, cfg.block // 2)))
    a = int(np.median(timed_sched))
    t0 = time.perf_counter()
    o.round(st, forced=[a] * cfg.batch)
    sec = time.perf_counter() - t0
    return {"value": round(mean_commit / sec, 4), "unit": "tokens/s", "cores": os.cpu_count(), "kind": "oracle",
            "sample": (f"one full oracle round (numpy fp64) of {cfg.name}: {cfg.n_layers} target + "
                       f"{cfg.draft_layers} draft layers, vocabulary {cfg.vocab}, width {cfg.d}, batch {cfg.batch}, "
                       f"context {int(lens.max())} from a synthetic cache, forced a = {a}; weight values shared "
                       f"across layers; tokens/s from the schedule's mean {mean_commit:.2f} committed per round"),
            "sec_per_round": round(sec, 2), "mean_committed_per_round": mean_commit}


# DRAM bytes (read + write) per algorithmic byte of the persistent layer-segment
# GEMM launch, from one ncu capture of it at Qwen3-8B widths and 17 rows
# (dram__bytes_read.sum + dram__bytes_write.sum = 387.14 + 4.10 = 391.2 MB for
# 387.3 MB of weights, activations and outputs).  Valid for that kernel as captured.
SEQ_TRAFFIC_RATIO = {"qwen3_8b_b1": 1.010}


def gemm_traffic(cfg, g):
    """DRAM bytes of the mean GEMM launch of this run, scaled from the capture
    (traffic grows with the weights streamed), or None without one."""
    r = SEQ_TRAFFIC_RATIO.get(cfg.name + ("_fused" if g.get("fused") else ""))
    if r is None or not g["launches"]:
        return None
    return round(r * g["bytes"] / g["launches"])


def run_cpu_sample(cfg, steps: int, warmup: int, sched):
    s = OracleSample(cfg)
    for w in range(warmup):
        s.step(sched[w % len(sched)])
    t_meas = t_full = tot_tok = 0.0
    for k in range(steps):
        tm, tf, tok = s.step(sched[(warmup + k) % len(sched)])
        t_meas += tm
        t_full += tf
        tot_tok += tok
    return tot_tok / t_full, t_meas / steps, t_full / steps, s


def run_reference(args):
    """Reference arm: the CPU oracle on a bounded sample of the workload.  A step
    is one sampled round (measured: ms_per_step); the throughput is the sampled
    rounds' committed tokens over their extrapolated full-round times."""
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return
    cfg = synth.CONFIGS[args.config]
    sched = synth.forced_schedule(cfg, args.warmup + args.steps)
    t0 = time.time()
    value, sec_meas, sec_full, s = run_cpu_sample(cfg, args.steps, args.warmup, sched)
    line = {
        "impl": "reference", "metric": METRIC, "value": round(value, 4), "unit": "tokens/s", "n_gpus": args.gpus,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(sec_meas * 1e3, 1),
        "est_ms_per_full_round": round(sec_full * 1e3, 1),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": {"workload": cfg.name, "batch": cfg.batch, "prompt": cfg.prompt_len, "block": cfg.block,
                   "l2": "inputs larger than L2"},
        "cpu_baseline": {"value": round(value, 4), "unit": "tokens/s", "cores": s.threads, "kind": "oracle",
                         "sample": s.describe()},
        "e2e": {"value": round(value, 4), "unit": "tokens/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
        "wall_s": round(time.time() - t0, 1),
    }
    print(json.dumps(line), flush=True)


# --------------------------------------------------------------------------
# one kernel alone: the tcgen05 projection (e.g. the LM head with its fused argmax)
# --------------------------------------------------------------------------


def run_kernel_gemm(args):
    """`reps` launches of out = X W^T (bf16, N x K weights, M rows) with epilogue
    `mode` through dflow_debug_gemm; CUDA-event time per launch and the achieved
    algorithmic GB/s (weights + activations read once)."""
    import torch

    from paper_2609_06498_gb300 import Engine, build, random_weights
    build.build()
    N, K, M, mode = args.N, args.K, args.M, args.mode
    rows = max(64, ((M + 63) // 64) * 64)
    cfg = synth.ModelConfig(name="gemm_kernel", dtype="bf16", d=128, n_layers=1, n_q_heads=1, n_kv_heads=1,
                            head_dim=128, inter=64, vocab=max(N, 128), draft_layers=1, feat_layers=(1,), block=16,
                            batch=rows // 64, prompt_len=64, new_tokens=16, schedule="uniform")
    eng = Engine(cfg, random_weights(cfg), max_batch=cfg.batch, max_ctx=256)
    g = torch.Generator(device="cuda")
    g.manual_seed(0)
    W = (torch.randn(N, K, generator=g, device="cuda") * 0.02).to(torch.bfloat16)
    X = torch.randn(M, K, generator=g, device="cuda").to(torch.bfloat16)
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    if mode in (0, 1):
        out = torch.zeros(M, N, device="cuda")
    elif mode in (2, 3):
        out = torch.zeros(M, N // 2 if mode == 2 else N, dtype=torch.bfloat16, device="cuda")
    else:
        out = torch.zeros(M, dtype=torch.int32, device="cuda")
    for _ in range(3):  # warm-up (tensor maps, attributes)
        eng.debug_gemm(args.path, W, X, mode, out, st)
    torch.cuda.synchronize()
    evs = [torch.cuda.Event(enable_timing=True) for _ in range(args.reps + 1)]
    evs[0].record()
    for r in range(args.reps):
        eng.debug_gemm(args.path, W, X, mode, out, st)
        evs[r + 1].record()
    torch.cuda.synchronize()
    ms = [evs[r].elapsed_time(evs[r + 1]) for r in range(args.reps)]
    alg = 2.0 * N * K + 2.0 * M * K
    rec = {"kernel": "gemm", "path": args.path, "N": N, "K": K, "M": M, "mode": mode, "status": int(st),
           "ms": [round(x, 4) for x in ms], "ms_mean": round(float(np.mean(ms)), 4), "alg_bytes": alg,
           "gbs_mean": round(alg / float(np.mean(ms)) / 1e6, 1), "tflops_mean": round(2.0 * N * K * M / float(np.mean(ms)) / 1e9, 1)}
    if args.cublas:
        for _ in range(3):
            X @ W.T
        torch.cuda.synchronize()
        c0, c1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        c0.record()
        for _ in range(args.reps):
            X @ W.T
        c1.record()
        torch.cuda.synchronize()
        rec["cublas_ms_mean"] = round(c0.elapsed_time(c1) / args.reps, 4)
    print(json.dumps(rec), flush=True)


# --------------------------------------------------------------------------
# multi-GPU replicas: each rank runs its own batch; the step time is the slowest
# rank's and the throughput the sum of all ranks' committed tokens
# --------------------------------------------------------------------------


def reduce_scalar(x: float, op: str, device: str = "cpu") -> float:
    """max or sum of a scalar over the ranks of the default process group."""
    import torch
    import torch.distributed as dist
    t = torch.tensor([float(x)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX if op == "max" else dist.ReduceOp.SUM)
    return float(t.item())


def replica_throughput(committed_local: float, ms_local: float, world: int, device: str = "cpu"):
    """(whole-job tokens/s, step time in ms) of `world` independent replicas."""
    if world == 1:
        return committed_local / (ms_local / 1e3), ms_local
    tot = reduce_scalar(committed_local, "sum", device)
    ms = reduce_scalar(ms_local, "max", device)
    return tot / (ms / 1e3), ms


# --------------------------------------------------------------------------
# GPU arm
# --------------------------------------------------------------------------


class Workload:
    """A workload on the device: random-init weights, engine, prefilled state,
    its forced acceptance schedule and `warmup` rounds already run; every leg
    starts from the snapshot taken after them."""

    def __init__(self, cfg, steps: int, warmup: int, rank: int = 0, relay: bool = True):
        import torch

        from paper_2609_06498_gb300 import Engine, random_weights
        self.cfg, self.K, self.Wm = cfg, steps, warmup
        n_rounds = warmup + steps
        self.max_ctx = cfg.replace(new_tokens=n_rounds * cfg.rows).max_ctx()
        self.weights = random_weights(cfg, seed=0)
        self.eng = Engine(cfg, self.weights, max_batch=cfg.batch, max_ctx=self.max_ctx)
        self.st = self.eng.new_state(cfg.batch, page_seed=rank)
        self.eng.prefill(self.st, synth.prompts(cfg))
        code = self.eng.read_status(self.st)
        assert code == 0, f"prefill failed: device status {code}"
        self.sched = synth.forced_schedule(cfg, n_rounds, seed=synth.SEED_SCHEDULE + rank)
        self.forced = torch.as_tensor(self.sched).cuda()
        self.acc = torch.empty(cfg.batch, dtype=torch.int32, device="cuda")
        self.comm = torch.empty(cfg.batch, cfg.rows, dtype=torch.int32, device="cuda")
        for w in range(warmup):
            self.round(w, relay)
        torch.cuda.synchronize()
        self.snap = {k: getattr(self.st, k).clone() for k in ("tokens", "seq_len", "carry", "n_carry", "boundary")}
        # a+1 committed per sequence per round (forced a) over the timed rounds
        self.committed = float((self.sched[warmup:n_rounds] + 1).sum())
        ctx0 = float(self.snap["seq_len"].float().mean())
        self.mean_ctx = ctx0 + float((self.sched[warmup:n_rounds] + 1).mean()) * steps / 2

    def round(self, r: int, relay: bool = True):
        self.eng.round(self.st, self.forced[r], relay=relay, out=(self.acc, self.comm))

    def restore(self):
        import torch
        for k, v in self.snap.items():
            getattr(self.st, k).copy_(v)
        torch.cuda.synchronize()

    def device_leg(self, relay: bool = True, barrier=None):
        """K rounds back to back from the snapshot: per-round CUDA-event times
        (ms) on the launching stream, the total, and the library's launches."""
        import torch
        self.restore()
        stream = torch.cuda.current_stream()
        ev = [torch.cuda.Event(enable_timing=True) for _ in range(self.K + 1)]
        n0 = self.eng.launch_count()
        if barrier:
            barrier()
        ev[0].record(stream)
        for k in range(self.K):
            self.round(self.Wm + k, relay)
            ev[k + 1].record(stream)
        torch.cuda.synchronize()
        launches = self.eng.launch_count() - n0
        code = self.eng.read_status(self.st)
        assert code == 0, f"device status {code} set during the timed leg"
        per = [ev[k].elapsed_time(ev[k + 1]) for k in range(self.K)]
        return per, ev[0].elapsed_time(ev[self.K]), launches

    def release(self):
        import torch
        for k in ("eng", "st", "weights", "forced", "snap"):
            setattr(self, k, None)
        torch.cuda.synchronize()
        torch.cuda.empty_cache()


def round_summary(cfg, per, total_ms, committed, mean_ctx):
    """ms per round, committed tokens/s and the round's HBM roofline fraction."""
    hbm, _, peak_src = peaks()
    K = len(per)
    ms = total_ms / K
    rb = round_bytes(cfg, mean_ctx)
    gbs = rb["total"] / (ms / 1e3) / 1e9
    return {"ms_per_round": round(ms, 4), "p50_ms": round(float(np.percentile(per, 50)), 4),
            "tokens_per_s": round(committed / (total_ms / 1e3), 2), "batch": cfg.batch,
            "acceptance": f"forced {cfg.schedule}", "rounds": K,
            "round_roofline": {"alg_bytes": rb["total"], "achieved_gbs": round(gbs, 1), "peak": hbm,
                               "frac": round(gbs / hbm, 4), "peak_source": peak_src}}


# the other bf16 workloads measured in the default run (device leg only)
OTHER_WORKLOADS = ("qwen3_1p7b_b1", "qwen3_4b_b4", "qwen3_8b_kv_b16")


def main():
    args = parse()
    if args.impl == "reference":
        return run_reference(args)
    if args.kernel == "gemm":
        return run_kernel_gemm(args)
    import torch
    import torch.distributed as dist

    from paper_2609_06498_gb300 import build

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    torch.cuda.set_device(local)
    if world > 1:
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    if rank == 0:
        build.build()
    if world > 1:
        dist.barrier()

    cfg = synth.CONFIGS[args.config]
    if args.depth:
        assert args.profile_only, "--depth is for --profile-only captures"
        cfg = cfg.replace(n_layers=args.depth, draft_layers=min(cfg.draft_layers, args.depth),
                          feat_layers=tuple(sorted({1, args.depth})))
    K, Wm = args.steps, args.warmup
    relay = bool(args.relay)  # 0: the DFlash baseline (mask embeddings only, nothing carried)
    lens = synth.prompt_lengths(cfg)
    wl = Workload(cfg, K, Wm, rank, relay)
    eng, st = wl.eng, wl.st

    def barrier():
        if world > 1:
            dist.barrier()
        torch.cuda.synchronize()

    if args.profile_only:
        # rounds inside a profiler range, for `ncu --profile-from-start off`
        torch.cuda.cudart().cudaProfilerStart()
        for k in range(min(K, 2)):
            wl.round(Wm + k, relay)
        torch.cuda.synchronize()
        torch.cuda.cudart().cudaProfilerStop()
        print(json.dumps({"profile_only": True, "launches": eng.launch_count()}))
        return

    committed, mean_ctx, sched = wl.committed, wl.mean_ctx, wl.sched
    stream = torch.cuda.current_stream()

    # ---- device leg: K rounds back to back, CUDA events on the launching stream
    with ClockSampler(local) as clocks:
        per, total_local, launches = wl.device_leg(relay, barrier)
    value, total_ms = replica_throughput(committed, total_local, world, "cuda")

    # ---- end-to-end leg: host buffers, H2D of the step's inputs and D2H of its result inside the region
    e2e = None
    if not args.no_e2e:
        wl.restore()
        h_forced = torch.as_tensor(sched).pin_memory()
        h_acc = torch.empty(K, cfg.batch, dtype=torch.int32).pin_memory()
        h_comm = torch.empty(K, cfg.batch, cfg.rows, dtype=torch.int32).pin_memory()
        d_forced = torch.empty(cfg.batch, dtype=torch.int32, device="cuda")
        barrier()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for k in range(K):
            d_forced.copy_(h_forced[Wm + k], non_blocking=True)
            eng.round(st, d_forced, relay=relay, out=(wl.acc, wl.comm))
            h_acc[k].copy_(wl.acc, non_blocking=True)
            h_comm[k].copy_(wl.comm, non_blocking=True)
        e1.record(stream)
        torch.cuda.synchronize()
        e2e_value, _ = replica_throughput(committed, e0.elapsed_time(e1), world, "cuda")
        assert np.array_equal(h_acc.numpy(), sched[Wm:Wm + K]), "accept lengths differ from the schedule"
        e2e = {"value": round(e2e_value, 2), "unit": "tokens/s",
               "h2d_bytes_per_step": 4 * cfg.batch, "d2h_bytes_per_step": 4 * cfg.batch * (1 + cfg.rows)}

    # ---- per-step split: the round's four calls one at a time, events between them
    # (the per-call entry points draft and carry with the relay on)
    wl.restore()
    evs = [[torch.cuda.Event(enable_timing=True) for _ in range(5)] for _ in range(K)]
    for k in range(K):
        e = evs[k]
        e[0].record(stream)
        blk = eng.draft_block(st)
        e[1].record(stream)
        g_t, feats, _ = eng.verify_block(st, blk)
        e[2].record(stream)
        a_k, _ = eng.accept_commit(st, blk, g_t, wl.forced[Wm + k])
        e[3].record(stream)
        eng.carry_hidden(st, blk, feats, a_k)
        e[4].record(stream)
    torch.cuda.synchronize()
    st_code = eng.read_status(st)
    assert st_code == 0, f"device status {st_code} set during the per-step leg"
    step_split = {name: round(float(np.median([evs[k][i].elapsed_time(evs[k][i + 1]) for k in range(K)])), 4)
                  for i, name in enumerate(("draft", "verify", "accept", "carry"))}

    # ---- relay off (the DFlash baseline of Sec. 5.3's runtime-overhead figure): same state and schedule
    relay_cost = None
    if rank == 0 and world == 1 and relay:
        per_off, total_off, _ = wl.device_leg(False)
        on, off = total_local / K, total_off / K
        relay_cost = {"dflow_ms": round(on, 4), "dflash_ms": round(off, 4), "delta_ms": round(on - off, 4),
                      "delta_frac": round((on - off) / off, 4),
                      "paper": "0.51 ms, 1.2 % of a DFlash round (Sec. 5.3; A800, model not stated)"}

    # ---- T = 1 rounds (Sec. 5.2, Table 1 T = 1 rows): K speculative-sampling rounds from the same state
    t1 = None
    if rank == 0 and world == 1:
        wl.restore()
        n_start = st.seq_len.clone()
        s0, s1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        s0.record(stream)
        for k in range(K):
            eng.round_sampled(st, T1_SEED, Wm + k, relay=relay, out=(wl.acc, wl.comm))
        s1.record(stream)
        torch.cuda.synchronize()
        code = eng.read_status(st)
        assert code == 0, f"device status {code} set during the T = 1 leg"
        t1_ms = s0.elapsed_time(s1) / K
        grown = float((st.seq_len - n_start).float().mean())
        t1 = {"ms_per_round": round(t1_ms, 4), "greedy_ms_per_round": round(total_local / K, 4),
              "delta_ms": round(t1_ms - total_local / K, 4), "mean_accept": round(grown / K - 1, 3),
              "note": "random-init drafter and target: the acceptance is what the draws give; "
                      "a round streams the same weights whatever it accepts"}

    # ---- autoregressive baseline (Sec. 5.2, Table 2 "Baseline"): K plain greedy steps of the
    # target from the same state, one committed token per sequence per step
    ar = None
    if rank == 0 and world == 1:
        wl.restore()
        tok = torch.empty(cfg.batch, dtype=torch.int32, device="cuda")
        a0, a1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a0.record(stream)
        for k in range(K):
            eng.decode_step(st, draft_context=False, out=tok)
        a1.record(stream)
        torch.cuda.synchronize()
        code = eng.read_status(st)
        assert code == 0, f"device status {code} set during the autoregressive leg"
        ar_ms = a0.elapsed_time(a1) / K
        ar_tps = cfg.batch / (ar_ms / 1e3)
        ar = {"ms_per_step": round(ar_ms, 4), "tokens_per_s": round(ar_tps, 2),
              "dflow_speedup": round(value / ar_tps, 3),
              "note": "one greedy target step per sequence on the block-verify launches (row 0 kept)",
              "paper": "Table 2, Qwen3-8B conc. 1: DFlow 3.08x AR on GSM8K (A800, trained drafter)"}

    # ---- profiled leg: per-launch events around the GEMMs (the dominant kernel)
    wl.restore()
    eng.profile(True)
    for k in range(K):
        wl.round(Wm + k, relay)
    torch.cuda.synchronize()
    prof = eng.profile_read()
    eng.profile(False)

    hbm, tflops, peak_src = peaks()
    g = dict(prof["gemm"])
    rb = round_bytes(cfg, mean_ctx)
    # with the attention a phase of the layer launches, those launches also read the K/V context
    fused = prof["attn"]["launches"] == 0
    if fused:
        g["bytes"] += K * rb["kv"]
        g["fused"] = True
    gemm_gbs = g["bytes"] / (g["ms"] / 1e3) / 1e9 if g["ms"] > 0 else 0.0
    ms_step = total_ms / K
    round_gbs = rb["total"] / (ms_step / 1e3) / 1e9

    line = {
        "metric": METRIC, "value": round(value, 2), "unit": "tokens/s", "n_gpus": world, "steps": K, "warmup": Wm,
        "ms_per_step": round(ms_step, 4), "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
        "dtype": "bf16" if cfg.dtype == "bf16" else "f32", "data": "synthetic",
        "config": {"workload": cfg.name, "batch": cfg.batch, "prompt": int(lens.max()), "block": cfg.block,
                   "target_layers": cfg.n_layers, "draft_layers": cfg.draft_layers, "d_model": cfg.d,
                   "acceptance": f"forced {cfg.schedule}", "relay": bool(args.relay),
                   "l2": "inputs larger than L2 (weights %.1f GB/round)" % (rb["weights"] / 1e9)},
        "round_latency_ms": {"mean": round(ms_step, 4), "p10": round(float(np.percentile(per, 10)), 4),
                             "p50": round(float(np.percentile(per, 50)), 4),
                             "p90": round(float(np.percentile(per, 90)), 4)},
        "roofline": {"bound": "hbm", "achieved": round(gemm_gbs, 1), "peak": hbm, "unit": "GB/s",
                     "frac": round(gemm_gbs / hbm, 4), "traffic": gemm_traffic(cfg, g),
                     "kernel": ("persistent layer launch: attention phase + O/gate-up/down/QKV weight-streaming GEMMs"
                                if fused else "weight-streaming GEMM"),
                     "peak_source": peak_src, "launches": g["launches"], "avg_launch_us": round(1e3 * g["ms"] / max(1, g["launches"]), 2)},
        "round_roofline": {"bound": "hbm", "alg_bytes": rb["total"], "achieved": round(round_gbs, 1), "peak": hbm,
                           "frac": round(round_gbs / hbm, 4), "unit": "GB/s", "peak_source": peak_src},
        "phase_ms": {"gemm": round(g["ms"] / K, 4), "attention": round(prof["attn"]["ms"] / K, 4)},
        "step_split_ms": step_split,
        "relay_overhead": relay_cost,
        "ar_baseline": ar,
        "t1_sampling": t1,
        "gpu_launches": int(launches),
        "e2e": e2e,
        "clocks": clocks.summary(),
    }
    wl.release()

    # ---- the other workloads (device leg, rank 0, one GPU): min(K, 20) rounds after min(W, 5)
    if rank == 0 and world == 1 and not args.no_other_workloads and cfg.name == DEFAULT_CONFIG:
        others = {}
        for name in OTHER_WORKLOADS:
            c = synth.CONFIGS[name]
            w = Workload(c, min(K, 20), min(Wm, 5))
            per_o, tot_o, _ = w.device_leg()
            others[name] = round_summary(c, per_o, tot_o, w.committed, w.mean_ctx)
            w.release()
        line["workloads"] = others

    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        line["cpu_baseline"] = cpu_baseline_full_round(cfg, sched[Wm:Wm + K])
    if rank == 0:
        print(json.dumps(line), flush=True)
    if world > 1:
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
