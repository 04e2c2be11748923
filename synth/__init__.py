"""Seeded synthetic inputs for the DFlow round: shapes, random weights, prompts,
acceptance schedules and synthetic decoding states.

This module is shared by the CUDA path's tests and bench and by the CPU oracle.
It holds no arithmetic of the method itself (no norms, projections, attention,
acceptance or relay); it only draws numbers and names shapes.

Workload shapes follow the paper's evaluation setup: Qwen3 targets of 1.7B / 4B
/ 8B parameters (Sec. 5.1) with a 5-layer drafter and a draft block of 16
(Sec. 5.1, "Training and Implementation Details").  Weights are random-init
N(0, 0.02) because no trained checkpoint exists here; prompts are uniform random
token ids standing in for the paper's benchmark prompts (GSM8K, MATH-500,
HumanEval, MBPP, MT-Bench, Alpaca), which are not used.
"""
from __future__ import annotations

import dataclasses
import hashlib
from typing import Dict, Iterable, List, Optional, Tuple

import numpy as np

# --------------------------------------------------------------------------
# configurations
# --------------------------------------------------------------------------


@dataclasses.dataclass(frozen=True)
class ModelConfig:
    """Shape of one target + drafter pair and the decoding workload around it."""

    name: str
    dtype: str  # "f32" or "bf16": storage/compute type of the GPU path
    d: int  # hidden size
    n_layers: int  # target decoder layers L
    n_q_heads: int
    n_kv_heads: int
    head_dim: int
    inter: int  # SwiGLU intermediate size
    vocab: int
    draft_layers: int  # drafter decoder layers
    feat_layers: Tuple[int, ...]  # target layers whose outputs feed Eq. 1 (1-indexed)
    block: int  # B: draft tokens per round (the block holds B+1 rows incl. the anchor)
    batch: int
    prompt_len: int  # prompt length (or the lower bound when ctx_range is set)
    new_tokens: int
    schedule: str  # "natural", "uniform" or "geometric"
    ctx_range: Optional[Tuple[int, int]] = None  # per-sequence context length range
    page_size: int = 64
    rope_theta: float = 1.0e6
    rms_eps: float = 1.0e-6
    ln_eps: float = 1.0e-6
    geo_p: float = 0.25

    @property
    def rows(self) -> int:
        return self.block + 1

    @property
    def n_feat(self) -> int:
        return len(self.feat_layers)

    @property
    def qkv_dim(self) -> int:
        return (self.n_q_heads + 2 * self.n_kv_heads) * self.head_dim

    def replace(self, **kw) -> "ModelConfig":
        return dataclasses.replace(self, **kw)

    def max_prompt(self) -> int:
        return self.ctx_range[1] if self.ctx_range else self.prompt_len

    def max_ctx(self, extra: int = 0) -> int:
        """Token capacity per sequence: prompt + new tokens + one block of slack."""
        need = self.max_prompt() + self.new_tokens + 2 * self.rows + extra
        return ((need + self.page_size - 1) // self.page_size) * self.page_size


def feature_layers(n_layers: int, m: int = 5) -> Tuple[int, ...]:
    """m target layers spread from shallow to deep (1-indexed, first and last included)."""
    if m == 1:
        return (n_layers,)
    return tuple(1 + (i * (n_layers - 1)) // (m - 1) for i in range(m))


TINY = ModelConfig(
    name="tiny_fp32", dtype="f32", d=256, n_layers=2, n_q_heads=4, n_kv_heads=2,
    head_dim=64, inter=768, vocab=1024, draft_layers=1, feat_layers=(1, 2), block=8,
    batch=1, prompt_len=64, new_tokens=64, schedule="natural")

QWEN3_1P7B = ModelConfig(
    name="qwen3_1p7b_b1", dtype="bf16", d=2048, n_layers=28, n_q_heads=16, n_kv_heads=8,
    head_dim=128, inter=6144, vocab=151936, draft_layers=3, feat_layers=feature_layers(28),
    block=16, batch=1, prompt_len=512, new_tokens=256, schedule="uniform")

QWEN3_4B = ModelConfig(
    name="qwen3_4b_b4", dtype="bf16", d=2560, n_layers=36, n_q_heads=32, n_kv_heads=8,
    head_dim=128, inter=9728, vocab=151936, draft_layers=5, feat_layers=feature_layers(36),
    block=16, batch=4, prompt_len=2048, new_tokens=512, schedule="geometric")

QWEN3_8B = ModelConfig(
    name="qwen3_8b_b1", dtype="bf16", d=4096, n_layers=36, n_q_heads=32, n_kv_heads=8,
    head_dim=128, inter=12288, vocab=151936, draft_layers=5, feat_layers=feature_layers(36),
    block=16, batch=1, prompt_len=2048, new_tokens=512, schedule="uniform")

QWEN3_8B_KV = QWEN3_8B.replace(
    name="qwen3_8b_kv_b16", batch=16, prompt_len=4096, ctx_range=(4096, 8192),
    new_tokens=256, schedule="geometric")

CONFIGS: Dict[str, ModelConfig] = {c.name: c for c in
                                   (TINY, QWEN3_1P7B, QWEN3_4B, QWEN3_8B, QWEN3_8B_KV)}

SEED_WEIGHTS = 0
SEED_PROMPTS = 1
SEED_SCHEDULE = 2
SEED_STATE = 3

# --------------------------------------------------------------------------
# bf16 storage helpers (round to nearest even; the data never holds NaN)
# --------------------------------------------------------------------------


def bf16_bits(x: np.ndarray) -> np.ndarray:
    """fp32 array -> uint16 bf16 bit patterns, round to nearest even."""
    u = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32)
    return ((u + (((u >> 16) & 1) + 0x7FFF)) >> 16).astype(np.uint16)


def bf16_to_f32(bits: np.ndarray) -> np.ndarray:
    return (bits.astype(np.uint32) << 16).view(np.float32)


def bf16_round(x: np.ndarray) -> np.ndarray:
    """fp32 values rounded to the nearest bf16 value (still stored as fp32)."""
    return bf16_to_f32(bf16_bits(x))


# --------------------------------------------------------------------------
# counter-based generators
# --------------------------------------------------------------------------

_M64 = (1 << 64) - 1


def splitmix64(x: int) -> int:
    """SplitMix64 finaliser (Steele, Lea, Flood 2014) on a Python int."""
    x = (x + 0x9E3779B97F4A7C15) & _M64
    z = x
    z = ((z ^ (z >> 30)) * 0xBF58476D1CE4E5B9) & _M64
    z = ((z ^ (z >> 27)) * 0x94D049BB133111EB) & _M64
    return z ^ (z >> 31)


def _stream(seed: int, name: str) -> np.random.Generator:
    h = hashlib.sha256(f"{seed}:{name}".encode()).digest()
    key = [int.from_bytes(h[0:8], "little"), int.from_bytes(h[8:16], "little")]
    return np.random.Generator(np.random.Philox(key=key))


_CHUNK = 1 << 24
_POOL = None


def _pool():
    global _POOL
    if _POOL is None:
        import concurrent.futures
        import os
        _POOL = concurrent.futures.ThreadPoolExecutor(max_workers=min(16, os.cpu_count() or 1))
    return _POOL


def normal(seed: int, name: str, shape, std: float = 0.02, bf16: bool = False) -> np.ndarray:
    """N(0, std^2) fp32 tensor, a pure function of (seed, name, shape).

    Drawn in chunks of 2^24 values, chunk i from its own stream (seed, name#i),
    so large tensors fill in parallel.  bf16=True rounds every value to the
    nearest bf16 (kept in fp32 storage).
    """
    n = int(np.prod(shape))
    out = np.empty(n, np.float32)

    def fill(i):
        lo, hi = i * _CHUNK, min(n, (i + 1) * _CHUNK)
        seg = out[lo:hi]
        _stream(seed, f"{name}#{i}").standard_normal(hi - lo, dtype=np.float32, out=seg)
        seg *= np.float32(std)
        if bf16:
            seg[:] = bf16_round(seg)

    nchunks = (n + _CHUNK - 1) // _CHUNK
    if nchunks <= 1:
        fill(0) if n else None
    else:
        list(_pool().map(fill, range(nchunks)))
    return out.reshape(shape)


def uniform_ints(seed: int, name: str, n: int, low: int, high: int) -> np.ndarray:
    """n int32 values uniform on [low, high)."""
    return _stream(seed, name).integers(low, high, size=n, dtype=np.int64).astype(np.int32)


# --------------------------------------------------------------------------
# weights
# --------------------------------------------------------------------------

LAYER_MATS = ("wq", "wk", "wv", "wo", "wg", "wu", "wd")
LAYER_VECS = ("attn_norm", "mlp_norm", "q_norm", "k_norm")


def layer_shapes(cfg: ModelConfig) -> Dict[str, Tuple[int, ...]]:
    d, hd = cfg.d, cfg.head_dim
    return {
        "wq": (cfg.n_q_heads * hd, d), "wk": (cfg.n_kv_heads * hd, d),
        "wv": (cfg.n_kv_heads * hd, d), "wo": (d, cfg.n_q_heads * hd),
        "wg": (cfg.inter, d), "wu": (cfg.inter, d), "wd": (d, cfg.inter),
        "attn_norm": (d,), "mlp_norm": (d,), "q_norm": (hd,), "k_norm": (hd,),
    }


def tensor_shapes(cfg: ModelConfig) -> Dict[str, Tuple[int, ...]]:
    """Every named weight tensor of the target + drafter pair."""
    d, V, m = cfg.d, cfg.vocab, cfg.n_feat
    shapes: Dict[str, Tuple[int, ...]] = {
        "embed": (V, d), "lm_head": (V, d), "final_norm": (d,),
        "d.final_norm": (d,), "w_c": (d, m * d), "c_norm": (d,), "e_mask": (d,),
        "relay_w1": (d, 3 * d), "relay_w2": (2 * d, d), "ln_w": (d,), "ln_b": (d,),
    }
    for prefix, n in (("t", cfg.n_layers), ("d", cfg.draft_layers)):
        for l in range(n):
            for k, s in layer_shapes(cfg).items():
                shapes[f"{prefix}{l}.{k}"] = s
    return shapes


def _is_vector(name: str) -> bool:
    base = name.split(".")[-1]
    return base in LAYER_VECS or name in ("final_norm", "d.final_norm", "c_norm", "ln_w", "ln_b")


def weight(cfg: ModelConfig, name: str, seed: int = SEED_WEIGHTS,
           perturb_norms: bool = False) -> np.ndarray:
    """One weight tensor as fp32 (bf16-representable values for bf16 configs).

    Matrices and E_mask are N(0, 0.02).  Norm gains are 1 and the LayerNorm bias
    is 0, unless perturb_norms is set (then gains are 1 + N(0, 0.1) and the bias
    N(0, 0.1)), which tests use so that a dropped gain or bias shows up.
    """
    shape = tensor_shapes(cfg)[name]
    if _is_vector(name):
        if perturb_norms:
            w = normal(seed, name, shape, 0.1)
            if name != "ln_b":
                w += 1.0
        else:
            w = np.zeros(shape, np.float32) if name == "ln_b" else np.ones(shape, np.float32)
        if cfg.dtype == "bf16":
            w = bf16_round(w)
    else:
        w = normal(seed, name, shape, 0.02, bf16=cfg.dtype == "bf16")
    return w.astype(np.float32, copy=False)


def weights(cfg: ModelConfig, seed: int = SEED_WEIGHTS, perturb_norms: bool = False,
            names: Optional[Iterable[str]] = None) -> Dict[str, np.ndarray]:
    names = list(tensor_shapes(cfg)) if names is None else list(names)
    big = [n for n in names if int(np.prod(tensor_shapes(cfg)[n])) > _CHUNK]
    small = [n for n in names if n not in big]
    out = {n: weight(cfg, n, seed, perturb_norms) for n in big}  # chunk-parallel inside
    out.update(zip(small, _pool().map(lambda n: weight(cfg, n, seed, perturb_norms), small)))
    return {n: out[n] for n in names}


# --------------------------------------------------------------------------
# prompts, context lengths, acceptance schedules
# --------------------------------------------------------------------------


def prompt_lengths(cfg: ModelConfig, seed: int = SEED_PROMPTS) -> np.ndarray:
    if cfg.ctx_range is None:
        return np.full(cfg.batch, cfg.prompt_len, np.int32)
    lo, hi = cfg.ctx_range
    return uniform_ints(seed, "ctx_len", cfg.batch, lo, hi + 1)


def prompts(cfg: ModelConfig, seed: int = SEED_PROMPTS) -> List[np.ndarray]:
    """Uniform random token ids in [0, vocab), one array per sequence."""
    lens = prompt_lengths(cfg, seed)
    return [uniform_ints(seed, f"prompt{b}", int(lens[b]), 0, cfg.vocab) for b in range(cfg.batch)]


def schedule_draw(seed: int, seq: int, rnd: int) -> int:
    """One 64-bit draw of the acceptance-schedule stream for (sequence, round)."""
    return splitmix64(seed ^ ((seq << 32) ^ rnd))


def forced_accept(cfg: ModelConfig, seq: int, rnd: int, seed: int = SEED_SCHEDULE) -> int:
    """Acceptance length imposed in benchmark mode for (sequence, round).

    "uniform": integer uniform on {0..B}.  "geometric": number of failures before
    the first success with success probability p, capped at B.
    """
    u = schedule_draw(seed, seq, rnd)
    B = cfg.block
    if cfg.schedule == "uniform":
        return int(u % (B + 1))
    if cfg.schedule == "geometric":
        x = ((u >> 11) + 0.5) / float(1 << 53)  # in (0, 1)
        k = int(np.floor(np.log(x) / np.log1p(-cfg.geo_p)))
        return min(k, B)
    raise ValueError(f"schedule {cfg.schedule!r} has no forced acceptance")


def forced_schedule(cfg: ModelConfig, rounds: int, seed: int = SEED_SCHEDULE) -> np.ndarray:
    """[rounds][batch] int32 forced acceptance lengths."""
    return np.array([[forced_accept(cfg, b, r, seed) for b in range(cfg.batch)]
                     for r in range(rounds)], dtype=np.int32)


# --------------------------------------------------------------------------
# synthetic decoding state (for per-call tests at sizes where a prefill through
# the oracle would take too long): random caches, carry and boundary tokens
# --------------------------------------------------------------------------


def synthetic_state(cfg: ModelConfig, ctx_lens: Optional[np.ndarray] = None,
                    n_carry: Optional[np.ndarray] = None, seed: int = SEED_STATE,
                    kv_std: float = 1.0) -> Dict[str, np.ndarray]:
    """A decoding state with n committed tokens per sequence.

    Returns logical (position-indexed) arrays: tokens [b][n], target K/V
    [L][b][max_ctx][Hkv][hd], drafter context K/V [Ld][b][max_ctx][Hkv][hd],
    carry [b][B][d], n_carry [b], boundary [b][2].  Cache rows at positions
    >= n-1 are zero.
    """
    bs, hkv, hd, d, B = cfg.batch, cfg.n_kv_heads, cfg.head_dim, cfg.d, cfg.block
    lens = prompt_lengths(cfg) + 1 if ctx_lens is None else np.asarray(ctx_lens, np.int32)
    cap = cfg.max_ctx()
    st: Dict[str, np.ndarray] = {"seq_len": lens.astype(np.int32)}
    st["tokens"] = np.zeros((bs, cap), np.int32)
    for b in range(bs):
        st["tokens"][b, : lens[b]] = uniform_ints(seed, f"st.tok{b}", int(lens[b]), 0, cfg.vocab)

    def cache(tag: str, nl: int) -> np.ndarray:
        arr = np.zeros((nl, bs, cap, hkv, hd), np.float32)
        for l in range(nl):
            for b in range(bs):
                valid = int(lens[b]) - 1
                arr[l, b, :valid] = normal(seed, f"st.{tag}{l}.{b}", (valid, hkv, hd), kv_std,
                                           bf16=cfg.dtype == "bf16")
        return arr

    st["k"] = cache("k", cfg.n_layers)
    st["v"] = cache("v", cfg.n_layers)
    st["dk"] = cache("dk", cfg.draft_layers)
    st["dv"] = cache("dv", cfg.draft_layers)
    if n_carry is None:
        n_carry = uniform_ints(seed, "st.ncarry", bs, 0, B)
    st["n_carry"] = np.asarray(n_carry, np.int32)
    carry = normal(seed, "st.carry", (bs, B, d), 1.0)
    st["carry"] = bf16_round(carry) if cfg.dtype == "bf16" else carry
    st["boundary"] = uniform_ints(seed, "st.boundary", 2 * bs, 0, cfg.vocab).reshape(bs, 2)
    return st


def block_tokens(cfg: ModelConfig, anchors: np.ndarray, seed: int = SEED_STATE) -> np.ndarray:
    """[b][B+1] draft blocks with the given anchors in row 0 and random drafts."""
    out = uniform_ints(seed, "st.block", cfg.batch * cfg.rows, 0, cfg.vocab).reshape(cfg.batch, cfg.rows)
    out[:, 0] = anchors
    return out


# --------------------------------------------------------------------------
# random draws of T = 1 sampling verification: a counter-based SplitMix64
# stream per (seed, sequence, round, row, purpose), indexed by token id.  The
# draws are odd multiples of 2^-24 in (0, 1), (2k + 1) / 2^24 with k the top 23
# bits of the hash: exactly representable in fp32 (24 significant bits), so a
# float32 and a float64 consumer see the same number, and never 0 or 1.
# --------------------------------------------------------------------------

NOISE_DRAFT, NOISE_ACCEPT, NOISE_RESAMPLE = 0, 1, 2
SEED_SAMPLING = 4


def noise_key(seed: int, seq: int, rnd: int, row: int, purpose: int) -> int:
    """Key of one (sequence, round, row, purpose) stream."""
    return splitmix64(seed ^ splitmix64((seq << 48) ^ (rnd << 24) ^ (row << 8) ^ purpose))


def _splitmix64_np(x: np.ndarray) -> np.ndarray:
    """SplitMix64 finaliser on uint64 arrays (wrap-around arithmetic)."""
    with np.errstate(over="ignore"):
        z = x + np.uint64(0x9E3779B97F4A7C15)
        z = (z ^ (z >> np.uint64(30))) * np.uint64(0xBF58476D1CE4E5B9)
        z = (z ^ (z >> np.uint64(27))) * np.uint64(0x94D049BB133111EB)
        return z ^ (z >> np.uint64(31))


def noise_uniform(key: int, n: int) -> np.ndarray:
    """Uniforms u_v = (2 (splitmix64(key ^ v) >> 41) + 1) / 2^24, v = 0..n-1 (float64)."""
    v = np.arange(n, dtype=np.uint64) ^ np.uint64(key)
    z = _splitmix64_np(v)
    return ((z >> np.uint64(41)).astype(np.float64) * 2.0 + 1.0) / float(1 << 24)


def sampling_noise(cfg: ModelConfig, seq: int, rnd: int, seed: int = SEED_SAMPLING) -> Dict[str, np.ndarray]:
    """The draws one T = 1 round of sequence `seq` consumes.

    gd [R][V]: Gumbel noise -log(-log u) of the drafter's sample at rows 1..B (row 0 unused)
    ua [R]:    uniform of the acceptance test of the proposal in row i (i = 1..B; row 0 unused)
    gr [R][V]: Gumbel noise of the token sampled for offset i = 1..B+1 (index i - 1):
               the residual after a rejection at i, or the bonus after B acceptances
    """
    R, V = cfg.rows, cfg.vocab
    gd = np.zeros((R, V))
    gr = np.zeros((R, V))
    ua = np.zeros(R)
    for i in range(1, R):
        gd[i] = -np.log(-np.log(noise_uniform(noise_key(seed, seq, rnd, i, NOISE_DRAFT), V)))
        ua[i] = noise_uniform(noise_key(seed, seq, rnd, i, NOISE_ACCEPT), 1)[0]
    for i in range(1, R + 1):
        gr[i - 1] = -np.log(-np.log(noise_uniform(noise_key(seed, seq, rnd, i, NOISE_RESAMPLE), V)))
    return {"gd": gd, "ua": ua, "gr": gr}
