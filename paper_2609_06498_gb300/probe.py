"""Kernel probes: run one library kernel on synthetic data, for timing and ncu.

  python -m paper_2609_06498_gb300.probe gemm --N 151936 --K 4096 --M 17 [--mode 4] [--reps 3]

runs `reps` launches of the tcgen05 projection kernel (out = X W^T with the
given fused epilogue) through dflow_debug_gemm and prints the CUDA-event time
per launch and the achieved algorithmic GB/s.
"""
from __future__ import annotations

import argparse
import json

import torch


def _engine(max_rows: int = 64):
    import synth
    from . import Engine, build, random_weights
    build.build()
    cfg = synth.ModelConfig(name="probe", dtype="bf16", d=128, n_layers=1, n_q_heads=1, n_kv_heads=1, head_dim=128,
                            inter=64, vocab=152064, draft_layers=1, feat_layers=(1,), block=16, batch=max_rows // 64 or 1,
                            prompt_len=64, new_tokens=16, schedule="uniform")
    return Engine(cfg, random_weights(cfg), max_batch=cfg.batch, max_ctx=256)


def gemm(N: int, K: int, M: int, mode: int, reps: int, path: int = 1):
    eng = _engine(max(64, ((M + 63) // 64) * 64))
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
    eng.debug_gemm(path, W, X, mode, out, st)  # warm-up (tensor maps, attributes)
    torch.cuda.synchronize()
    evs = [torch.cuda.Event(enable_timing=True) for _ in range(reps + 1)]
    evs[0].record()
    for r in range(reps):
        eng.debug_gemm(path, W, X, mode, out, st)
        evs[r + 1].record()
    torch.cuda.synchronize()
    ms = [evs[r].elapsed_time(evs[r + 1]) for r in range(reps)]
    bytes_ = 2.0 * N * K + 2.0 * M * K
    best = min(ms)
    print(json.dumps({"probe": "gemm", "N": N, "K": K, "M": M, "mode": mode, "path": path, "status": int(st),
                      "ms": [round(x, 4) for x in ms], "gbs_best": round(bytes_ / best / 1e6, 1)}))


def main():
    p = argparse.ArgumentParser()
    sub = p.add_subparsers(dest="what", required=True)
    q = sub.add_parser("gemm")
    q.add_argument("--N", type=int, default=151936)
    q.add_argument("--K", type=int, default=4096)
    q.add_argument("--M", type=int, default=17)
    q.add_argument("--mode", type=int, default=0)
    q.add_argument("--reps", type=int, default=3)
    q.add_argument("--path", type=int, default=1)
    a = p.parse_args()
    if a.what == "gemm":
        gemm(a.N, a.K, a.M, a.mode, a.reps, a.path)


if __name__ == "__main__":
    main()
