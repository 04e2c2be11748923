"""Helpers for GPU-vs-oracle parity tests: move an oracle State into the
library's paged device state, read device results back, compare with the
tolerances of the method's precision."""
import numpy as np
import torch

TOL = {"f32": 1e-4, "bf16": 2e-2}  # max |gpu - ref| / max |ref| per tensor
GAP = 0.05  # token identity is required where the oracle's top-1/top-2 gap exceeds this


def rel_err(got, ref) -> float:
    got = np.asarray(got, np.float64)
    ref = np.asarray(ref, np.float64)
    den = np.abs(ref).max()
    return float(np.abs(got - ref).max() / (den if den > 0 else 1.0))


def assert_close(got, ref, cfg, what=""):
    e = rel_err(got, ref)
    assert e <= TOL[cfg.dtype], f"{what}: max rel err {e:.3g} > {TOL[cfg.dtype]}"


def to_np(t: torch.Tensor) -> np.ndarray:
    return t.detach().float().cpu().numpy() if t.dtype == torch.bfloat16 else t.detach().cpu().numpy()


def upload_state(eng, dst, ost):
    """Copy an oracle State (logical arrays) into a DeviceState."""
    cfg = eng.cfg
    cap = min(ost.tokens.shape[1], dst.max_ctx)
    dst.tokens.zero_()
    dst.tokens[:, :cap] = torch.as_tensor(ost.tokens[:, :cap])
    dst.seq_len.copy_(torch.as_tensor(ost.seq_len))
    dt = dst.kv.dtype
    for b in range(dst.batch):
        n = int(ost.seq_len[b])
        if n > 1:
            m = n - 1
            dst.write_cache(dst.kv, b, torch.as_tensor(ost.k[:, b, :m]).to("cuda"), torch.as_tensor(ost.v[:, b, :m]).to("cuda"))
            dst.write_cache(dst.draft_kv, b, torch.as_tensor(ost.dk[:, b, :m]).to("cuda"),
                            torch.as_tensor(ost.dv[:, b, :m]).to("cuda"))
    dst.carry.copy_(torch.as_tensor(ost.carry).to(dt))
    dst.n_carry.copy_(torch.as_tensor(ost.n_carry))
    dst.boundary.copy_(torch.as_tensor(ost.boundary))
    dst.active.copy_(torch.as_tensor(ost.active.astype(np.int32)))
    dst.status.zero_()
    torch.cuda.synchronize()


def token_check(got, ref_tokens, ref_logits, rows=None):
    """Tokens must match wherever the oracle's decision is safe (gap > GAP).
    Returns (n_checked, n_allowed_flips)."""
    from oracle import top2_gap
    got = np.asarray(got)
    gap = top2_gap(ref_logits)
    rows = range(len(ref_tokens)) if rows is None else rows
    checked = flips = 0
    for i in rows:
        if gap[i] > GAP:
            assert got[i] == ref_tokens[i], f"row {i}: got {got[i]} want {ref_tokens[i]} (gap {gap[i]:.3f})"
            checked += 1
        elif got[i] != ref_tokens[i]:
            flips += 1
    return checked, flips


def lmhead_engine(max_rows: int = 64):
    """A bf16 handle whose workspace holds LM-head argmax partials for up to
    max_rows rows over a 152064-token vocabulary (for GEMM-level tests)."""
    import synth
    from paper_2609_06498_gb300 import Engine, build, random_weights
    build.build()
    cfg = synth.ModelConfig(name="lmhead", dtype="bf16", d=128, n_layers=1, n_q_heads=1, n_kv_heads=1, head_dim=128,
                            inter=64, vocab=152064, draft_layers=1, feat_layers=(1,), block=16,
                            batch=max_rows // 64 or 1, prompt_len=64, new_tokens=16, schedule="uniform")
    return Engine(cfg, random_weights(cfg), max_batch=cfg.batch, max_ctx=256)
