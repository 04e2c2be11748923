"""Python binding of libdflow: PyTorch owns device memory and streams; every step
of the round runs in the library's kernels through the C ABI.

This module only marshals arguments: it packs weights into the layout
include/dflow.h documents, allocates the decoding state and the workspace with
torch, and passes raw device pointers to the library.
"""
from __future__ import annotations

import ctypes
from typing import Dict, List, Optional, Sequence, Tuple

import numpy as np
import torch

from . import _abi
from ._abi import call

LAYER_FIELDS = ("w_qkv", "w_o", "w_gate_up", "w_down", "attn_norm", "mlp_norm", "q_norm", "k_norm")


def torch_dtype(cfg) -> torch.dtype:
    return torch.bfloat16 if cfg.dtype == "bf16" else torch.float32


def interleave_gate_up(wg: torch.Tensor, wu: torch.Tensor) -> torch.Tensor:
    """[I][d] gate and up -> [2I][d] in groups of 128 rows: 64 gate rows, then their 64 up rows."""
    inter, d = wg.shape
    return torch.stack([wg.reshape(inter // 64, 64, d), wu.reshape(inter // 64, 64, d)], 1).reshape(2 * inter, d)


class DeviceWeights:
    """Packed device weights plus the dflow_weights struct that points at them."""

    def __init__(self, cfg, tensors: Dict[str, torch.Tensor]):
        self.cfg = cfg
        self.t = tensors
        self._target = (_abi.LayerWeights * cfg.n_layers)()
        self._draft = (_abi.LayerWeights * cfg.draft_layers)()
        for arr, pfx, n in ((self._target, "t", cfg.n_layers), (self._draft, "d", cfg.draft_layers)):
            for l in range(n):
                for f in LAYER_FIELDS:
                    setattr(arr[l], f, tensors[f"{pfx}{l}.{f}"].data_ptr())
        p = lambda k: tensors[k].data_ptr()  # noqa: E731
        self.c = _abi.Weights(
            embed=p("embed"), lm_head=p("lm_head"), final_norm=p("final_norm"), target=self._target,
            draft=self._draft, draft_final_norm=p("d.final_norm"), w_c=p("w_c"), c_norm=p("c_norm"),
            e_mask=p("e_mask"), relay_w1=p("relay_w1"), relay_w2=p("relay_w2"), ln_w=p("ln_w"), ln_b=p("ln_b"))

    def nbytes(self) -> int:
        return sum(t.numel() * t.element_size() for t in self.t.values())


_VEC = ("final_norm", "d.final_norm", "c_norm", "e_mask", "ln_w", "ln_b")


def pack_weights(cfg, W: Dict[str, np.ndarray], device="cuda") -> DeviceWeights:
    """Weights named as in `synth` (wq, wk, wv, wo, wg, wu, wd, norms) -> packed device tensors."""
    dt = torch_dtype(cfg)

    def mat(x):
        return torch.as_tensor(np.ascontiguousarray(x), dtype=torch.float32).to(device=device, dtype=dt)

    def vec(x):
        return torch.as_tensor(np.ascontiguousarray(x), dtype=torch.float32).to(device)

    t: Dict[str, torch.Tensor] = {}
    for k in ("embed", "lm_head", "w_c", "relay_w1", "relay_w2"):
        t[k] = mat(W[k])
    for k in _VEC:
        t[k] = vec(W[k])
    for pfx, n in (("t", cfg.n_layers), ("d", cfg.draft_layers)):
        for l in range(n):
            g = lambda k: W[f"{pfx}{l}.{k}"]  # noqa: E731
            t[f"{pfx}{l}.w_qkv"] = mat(np.concatenate([g("wq"), g("wk"), g("wv")], 0))
            t[f"{pfx}{l}.w_o"] = mat(g("wo"))
            t[f"{pfx}{l}.w_gate_up"] = interleave_gate_up(mat(g("wg")), mat(g("wu"))).contiguous()
            t[f"{pfx}{l}.w_down"] = mat(g("wd"))
            for k in ("attn_norm", "mlp_norm", "q_norm", "k_norm"):
                t[f"{pfx}{l}.{k}"] = vec(g(k))
    return DeviceWeights(cfg, t)


def random_weights(cfg, seed: int = 0, device="cuda", std: float = 0.02) -> DeviceWeights:
    """Random-init N(0, std) weights drawn directly on the device (benchmark workloads)."""
    dt = torch_dtype(cfg)
    gen = torch.Generator(device=device)
    gen.manual_seed(seed)
    d, hd, I, V = cfg.d, cfg.head_dim, cfg.inter, cfg.vocab
    qkv = (cfg.n_q_heads + 2 * cfg.n_kv_heads) * hd

    def mat(*shape):
        out = torch.empty(shape, dtype=dt, device=device)
        rows_per = max(1, (1 << 26) // shape[1])
        for r0 in range(0, shape[0], rows_per):
            blk = torch.randn((min(rows_per, shape[0] - r0), shape[1]), generator=gen, device=device)
            out[r0:r0 + blk.shape[0]] = (blk * std).to(dt)
        return out

    ones = lambda: torch.ones(d, device=device)  # noqa: E731
    t: Dict[str, torch.Tensor] = {
        "embed": mat(V, d), "lm_head": mat(V, d), "w_c": mat(d, cfg.n_feat * d), "relay_w1": mat(d, 3 * d),
        "relay_w2": mat(2 * d, d), "final_norm": ones(), "d.final_norm": ones(), "c_norm": ones(),
        "e_mask": (torch.randn(d, generator=gen, device=device) * std).to(dt).float(), "ln_w": ones(),
        "ln_b": torch.zeros(d, device=device)}
    for pfx, n in (("t", cfg.n_layers), ("d", cfg.draft_layers)):
        for l in range(n):
            t[f"{pfx}{l}.w_qkv"] = mat(qkv, d)
            t[f"{pfx}{l}.w_o"] = mat(d, cfg.n_q_heads * hd)
            t[f"{pfx}{l}.w_gate_up"] = mat(2 * I, d)
            t[f"{pfx}{l}.w_down"] = mat(d, I)
            for k in ("attn_norm", "mlp_norm"):
                t[f"{pfx}{l}.{k}"] = ones()
            for k in ("q_norm", "k_norm"):
                t[f"{pfx}{l}.{k}"] = torch.ones(hd, device=device)
    return DeviceWeights(cfg, t)


class DeviceState:
    """Decoding state of a batch in device memory (see dflow_state in include/dflow.h)."""

    def __init__(self, cfg, batch: int, max_ctx: int, page_seed: int = 0, device="cuda"):
        dt = torch_dtype(cfg)
        ps = cfg.page_size
        self.batch, self.max_ctx, self.page_size = batch, max_ctx, ps
        self.pages_per_seq = max_ctx // ps
        self.num_pages = batch * self.pages_per_seq
        perm = np.random.default_rng(page_seed).permutation(self.num_pages).astype(np.int32)
        i32 = dict(dtype=torch.int32, device=device)
        self.tokens = torch.zeros(batch, max_ctx, **i32)
        self.seq_len = torch.zeros(batch, **i32)
        self.page_table = torch.as_tensor(perm.reshape(batch, self.pages_per_seq)).to(device)
        self.kv = torch.zeros(cfg.n_layers, self.num_pages, 2, cfg.n_kv_heads, ps, cfg.head_dim, dtype=dt, device=device)
        self.draft_kv = torch.zeros(cfg.draft_layers, self.num_pages, 2, cfg.n_kv_heads, ps, cfg.head_dim, dtype=dt,
                                    device=device)
        self.carry = torch.zeros(batch, cfg.block, cfg.d, dtype=dt, device=device)
        self.n_carry = torch.zeros(batch, **i32)
        self.boundary = torch.full((batch, 2), -1, **i32)
        self.active = torch.ones(batch, **i32)
        self.status = torch.zeros(1, **i32)
        self.c = _abi.State(batch=batch, tokens=self.tokens.data_ptr(), seq_len=self.seq_len.data_ptr(),
                            page_table=self.page_table.data_ptr(), kv=self.kv.data_ptr(),
                            draft_kv=self.draft_kv.data_ptr(), carry=self.carry.data_ptr(),
                            n_carry=self.n_carry.data_ptr(), boundary=self.boundary.data_ptr(),
                            active=self.active.data_ptr(), status=self.status.data_ptr())

    # -- logical (position-indexed) views of the paged pools, for setup and inspection

    def _pool_view(self, pool):
        # [layers][pages][2][hkv][ps][hd] -> [layers][2][pages][ps][hkv][hd]
        return pool.permute(0, 2, 1, 4, 3, 5)

    def _slots(self, b: int, n: int):
        p = torch.arange(n, device=self.page_table.device)
        return self.page_table[b].long()[p // self.page_size], p % self.page_size

    def write_cache(self, pool, b: int, k: torch.Tensor, v: torch.Tensor):
        """k, v: [layers][n][hkv][hd] for positions 0..n-1 of sequence b."""
        n = k.shape[1]
        pages, slots = self._slots(b, n)
        P = self._pool_view(pool)
        P[:, 0, pages, slots] = k.to(pool.dtype)
        P[:, 1, pages, slots] = v.to(pool.dtype)

    def read_cache(self, pool, b: int, n: int):
        pages, slots = self._slots(b, n)
        P = self._pool_view(pool)
        return P[:, 0, pages, slots], P[:, 1, pages, slots]


class Engine:
    """One dflow handle + its workspace, for one config and batch capacity."""

    def __init__(self, cfg, weights: DeviceWeights, max_batch: int, max_ctx: int, device="cuda"):
        self.cfg, self.weights, self.max_batch, self.max_ctx = cfg, weights, max_batch, max_ctx
        fl = list(cfg.feat_layers) + [0] * (_abi.MAX_FEAT - len(cfg.feat_layers))
        self.ccfg = _abi.Config(
            dtype=_abi.DFLOW_BF16 if cfg.dtype == "bf16" else _abi.DFLOW_F32, d_model=cfg.d,
            n_layers=cfg.n_layers, n_q_heads=cfg.n_q_heads, n_kv_heads=cfg.n_kv_heads, head_dim=cfg.head_dim,
            d_inter=cfg.inter, vocab=cfg.vocab, draft_layers=cfg.draft_layers, n_feat=len(cfg.feat_layers),
            feat_layers=(ctypes.c_int32 * _abi.MAX_FEAT)(*fl), block=cfg.block, page_size=cfg.page_size,
            max_batch=max_batch, max_ctx=max_ctx, num_pages=max_batch * (max_ctx // cfg.page_size),
            rope_theta=cfg.rope_theta, rms_eps=cfg.rms_eps, ln_eps=cfg.ln_eps)
        h = ctypes.c_void_p()
        call("dflow_create", ctypes.byref(self.ccfg), ctypes.byref(weights.c), ctypes.byref(h))
        self.h = h
        nbytes = ctypes.c_size_t()
        call("dflow_workspace_size", self.h, ctypes.byref(nbytes))
        self.workspace = torch.empty(nbytes.value + 256, dtype=torch.uint8, device=device)
        base = self.workspace.data_ptr()
        aligned = (base + 255) & ~255
        call("dflow_set_workspace", self.h, ctypes.c_void_p(aligned), nbytes.value)
        self.device = device

    def __del__(self):
        h = getattr(self, "h", None)
        if h is not None and h.value:
            try:
                _abi.lib().dflow_destroy(h)
            except Exception:
                pass

    @staticmethod
    def _stream():
        return ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)

    def new_state(self, batch: int, page_seed: int = 0) -> DeviceState:
        return DeviceState(self.cfg, batch, self.max_ctx, page_seed, self.device)

    def _i32(self, *shape):
        return torch.empty(*shape, dtype=torch.int32, device=self.device)

    def prefill(self, st: DeviceState, prompts: Sequence[Sequence[int]]):
        lens = np.array([len(p) for p in prompts], np.int32)
        stride = int(lens.max())
        buf = np.zeros((st.batch, stride), np.int32)
        for b, p in enumerate(prompts):
            buf[b, :len(p)] = p
        dev = torch.as_tensor(buf).to(self.device)
        call("dflow_prefill", self.h, ctypes.byref(st.c), ctypes.c_void_p(dev.data_ptr()), stride,
             lens.ctypes.data_as(_abi.c_i32p), self._stream())
        torch.cuda.current_stream().synchronize()

    def draft_block(self, st: DeviceState, logits: bool = False):
        """Block tokens [batch][B+1]; with logits=True also the drafter's fp32 logits."""
        blk = self._i32(st.batch, self.cfg.rows)
        lg = (torch.empty(st.batch, self.cfg.rows, self.cfg.vocab, dtype=torch.float32, device=self.device)
              if logits else None)
        call("dflow_draft_block", self.h, ctypes.byref(st.c), ctypes.c_void_p(blk.data_ptr()),
             ctypes.c_void_p(lg.data_ptr() if lg is not None else 0), self._stream())
        return (blk, lg) if logits else blk

    def verify_block(self, st: DeviceState, blk: torch.Tensor, logits: bool = False):
        g = self._i32(st.batch, self.cfg.rows)
        feats = torch.empty(st.batch, self.cfg.rows, self.cfg.d, dtype=torch_dtype(self.cfg), device=self.device)
        lg = (torch.empty(st.batch, self.cfg.rows, self.cfg.vocab, dtype=torch.float32, device=self.device)
              if logits else None)
        call("dflow_verify_block", self.h, ctypes.byref(st.c), ctypes.c_void_p(blk.data_ptr()),
             ctypes.c_void_p(g.data_ptr()), ctypes.c_void_p(feats.data_ptr()),
             ctypes.c_void_p(lg.data_ptr() if lg is not None else 0), self._stream())
        return g, feats, lg

    def accept_commit(self, st: DeviceState, blk, g, forced: Optional[torch.Tensor] = None):
        acc = self._i32(st.batch)
        comm = self._i32(st.batch, self.cfg.rows)
        call("dflow_accept_commit", self.h, ctypes.byref(st.c), ctypes.c_void_p(blk.data_ptr()),
             ctypes.c_void_p(g.data_ptr()), ctypes.c_void_p(forced.data_ptr() if forced is not None else 0),
             ctypes.c_void_p(acc.data_ptr()), ctypes.c_void_p(comm.data_ptr()), self._stream())
        return acc, comm

    def carry_hidden(self, st: DeviceState, blk, feats, acc):
        call("dflow_carry_hidden", self.h, ctypes.byref(st.c), ctypes.c_void_p(blk.data_ptr()),
             ctypes.c_void_p(feats.data_ptr()), ctypes.c_void_p(acc.data_ptr()), self._stream())

    def round(self, st: DeviceState, forced: Optional[torch.Tensor] = None, relay: bool = True, out=None):
        acc, comm = out if out is not None else (self._i32(st.batch), self._i32(st.batch, self.cfg.rows))
        call("dflow_round", self.h, ctypes.byref(st.c),
             ctypes.c_void_p(forced.data_ptr() if forced is not None else 0), ctypes.c_void_p(acc.data_ptr()),
             ctypes.c_void_p(comm.data_ptr()), int(relay), self._stream())
        return acc, comm

    def round_sampled(self, st: DeviceState, seed: int, round_index: int, relay: bool = True, out=None,
                      logits: Optional[Tuple[torch.Tensor, torch.Tensor]] = None):
        """One T = 1 round (speculative sampling, see dflow_round_sampled); (accept_len, committed).
        logits: optional fp32 (drafter, target) buffers [batch][B+1][vocab] that receive the round's logits."""
        acc, comm = out if out is not None else (self._i32(st.batch), self._i32(st.batch, self.cfg.rows))
        ql, pl = (0, 0) if logits is None else (logits[0].data_ptr(), logits[1].data_ptr())
        call("dflow_round_sampled", self.h, ctypes.byref(st.c), ctypes.c_uint64(seed), int(round_index),
             ctypes.c_void_p(acc.data_ptr()), ctypes.c_void_p(comm.data_ptr()), int(relay), ctypes.c_void_p(ql),
             ctypes.c_void_p(pl), self._stream())
        return acc, comm

    def decode_step(self, st: DeviceState, draft_context: bool = False, out: Optional[torch.Tensor] = None):
        """Plain greedy decoding step of the target (the Sec. 5.2 baseline); the committed tokens [batch]."""
        tok = out if out is not None else self._i32(st.batch)
        call("dflow_decode_step", self.h, ctypes.byref(st.c), ctypes.c_void_p(tok.data_ptr()), int(draft_context),
             self._stream())
        return tok

    def profile(self, enable: bool) -> None:
        call("dflow_profile_enable", self.h, int(enable))

    def profile_read(self):
        out = (_abi.KernelProfile * _abi.PROF_N)()
        call("dflow_profile_read", self.h, out)
        return {k: dict(launches=out[i].launches, ms=out[i].total_ms, bytes=out[i].alg_bytes, flops=out[i].alg_flops)
                for i, k in enumerate(("gemm", "attn", "other"))}

    def debug_gemm(self, path: int, W: torch.Tensor, X: torch.Tensor, mode: int, out: torch.Tensor,
                   status: torch.Tensor, ldx: Optional[int] = None, M: Optional[int] = None):
        """Test hook: one GEMM with a fused epilogue through the library (see dflow_debug_gemm)."""
        N, K = W.shape
        M = X.shape[0] if M is None else M
        ldx = X.stride(0) if ldx is None else ldx
        ldo = out.stride(0) if out.dim() > 1 else 1
        call("dflow_debug_gemm", self.h, int(path), ctypes.c_void_p(W.data_ptr()), N, K, ctypes.c_void_p(X.data_ptr()),
             M, ldx, int(mode), ctypes.c_void_p(out.data_ptr()), ldo, ctypes.c_void_p(status.data_ptr()), self._stream())

    def launch_count(self) -> int:
        v = ctypes.c_uint64()
        call("dflow_launch_count", self.h, ctypes.byref(v))
        return v.value

    def read_status(self, st: DeviceState) -> int:
        v = ctypes.c_int32()
        call("dflow_read_status", self.h, ctypes.byref(st.c), ctypes.byref(v), self._stream())
        return v.value

    def generate(self, st: DeviceState, prompts: List[Sequence[int]], n_new: int, forced_fn=None,
                 relay: bool = True) -> List[np.ndarray]:
        """Prefill + rounds until every sequence has n_new new tokens (host loop)."""
        self.prefill(st, prompts)
        plen = np.array([len(p) for p in prompts])
        r = 0
        while True:
            n = st.seq_len.cpu().numpy()
            act = (n - plen) < n_new
            if not act.any():
                break
            st.active.copy_(torch.as_tensor(act.astype(np.int32)))
            forced = None
            if forced_fn is not None:
                forced = torch.as_tensor(np.array([forced_fn(b, r) for b in range(st.batch)], np.int32)).to(self.device)
            self.round(st, forced, relay)
            r += 1
        toks = st.tokens.cpu().numpy()
        return [toks[b, plen[b]:plen[b] + n_new].copy() for b in range(st.batch)]
