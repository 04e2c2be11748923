"""Plain, slow CPU oracle of one DFlow speculative round (TEST INFRASTRUCTURE).

This module is test infrastructure: only tests/, __graft_entry__.smoke() and
bench.py's CPU-baseline leg may import it.  It shares no code with the CUDA
path.  Everything is computed in float64 with numpy, one sequence at a time,
in the order the paper states the method:

  * Sec. 3, Eq. 1  -- fused target context  H_T = RMSNorm(W_c [H^l1; ...; H^lm])
  * Sec. 3, Eq. 2  -- block-diffusion drafting  y^ = D(E_mask; H_T), with H_T
                      injected into the Key and Value projections of every
                      draft layer
  * Sec. 3, Eq. 3  -- exact-match verification: accepted prefix, first
                      rejection, rejected suffix; bonus token; commit
  * Sec. 4.2       -- verifier representation alignment (shared W_c + RMSNorm,
                      shift by one position)
  * Sec. 4.2, Eq. 4 -- reject-conditioned MLP  [beta; gamma] = MLP([E(b); E(y_{a+1}); h])
  * Sec. 4.2, Eq. 5 -- x = E_mask + beta * LN(h) + gamma at valid carried slots,
                      E_mask elsewhere, masks only when nothing is carried
  * Sec. 5.2        -- the autoregressive baseline (one greedy target step), and
                      T = 1 verification by speculative sampling (a reading:
                      the paper reports T = 1 results without printing the rule)

Readings of points the paper leaves open (all shared with the CUDA path by
specification, not by code):

  * The draft block has B+1 rows: the anchor (last committed token) in row 0
    and B drafted tokens.  Row i sits at position n-1+i for a sequence with n
    committed tokens.  a ranges over 0..B; a+1 tokens are committed per round.
  * Target: Qwen3 decoder layers (pre-RMSNorm, per-head q/k RMSNorm, rotary
    embedding with rotate-half pairing, grouped-query attention, SwiGLU MLP,
    untied LM head).  "Hidden state of layer l" is the residual stream after
    decoder layer l (1-indexed).
  * Drafter: Qwen3 layers of the target's width; context K/V of a committed
    position p are k = RoPE(k_norm(W_k f_p), p), v = W_v f_p (no input norm:
    f is already RMSNormed by Eq. 1); block rows attend to every context
    position 0..n-2 and to every block row (no mask); own final RMSNorm; LM
    head shared with the target.
  * Carry: next-round slot j (position n'+j-1, n' the new length) takes the
    feature of the previous verify row a+j, for j = 1..B-a-1: the verifier
    states whose next-token predictions land on the rejected-suffix positions.
  * MLP_phi = Linear(3d->d) -> SiLU -> Linear(d->2d), output split [beta; gamma].
    LN = LayerNorm over d with gain ln_w and bias ln_b.  (parity unpinned: the
    paper fixes neither layer sizes nor activation; only the wiring is pinned)
  * argmax ties resolve to the lowest token id.
  * Benchmark mode: a forced acceptance length replaces a; the bonus is still
    the target's prediction at row a.
"""
from __future__ import annotations

import dataclasses
from typing import Callable, Dict, List, Optional, Sequence

import numpy as np

F = np.float64

# ---------------------------------------------------------------------------
# elementary operations
# ---------------------------------------------------------------------------


def rmsnorm(x, w, eps):
    """RMSNorm over the last axis: x / sqrt(mean(x^2) + eps) * w (Eq. 1; Qwen3 norms)."""
    x = np.asarray(x, F)
    return x / np.sqrt(np.mean(x * x, axis=-1, keepdims=True) + eps) * np.asarray(w, F)


def layernorm(x, w, b, eps):
    """LayerNorm over the last axis with gain w and bias b (the LN of Eq. 5)."""
    x = np.asarray(x, F)
    mu = np.mean(x, axis=-1, keepdims=True)
    var = np.mean((x - mu) ** 2, axis=-1, keepdims=True)
    return (x - mu) / np.sqrt(var + eps) * np.asarray(w, F) + np.asarray(b, F)


def silu(x):
    x = np.asarray(x, F)
    return x / (1.0 + np.exp(-x))


def rope(x, pos, theta):
    """Rotary embedding, rotate-half pairing (i, i + hd/2), frequency theta^(-2i/hd).

    x: [..., hd]; pos: scalar or array broadcasting against x[..., 0].
    """
    x = np.asarray(x, F)
    hd = x.shape[-1]
    half = hd // 2
    inv = float(theta) ** (-2.0 * np.arange(half, dtype=F) / hd)
    ang = np.asarray(pos, F)[..., None] * inv
    c, s = np.cos(ang), np.sin(ang)
    while c.ndim < x.ndim:  # broadcast over head axes
        c, s = c[..., None, :], s[..., None, :]
    x1, x2 = x[..., :half], x[..., half:]
    return np.concatenate([x1 * c - x2 * s, x2 * c + x1 * s], axis=-1)


def attend(q, K, V, n_kv_heads):
    """Grouped-query softmax attention of one query row over the given keys.

    q: [Hq][hd]; K, V: [n][Hkv][hd].  Query head h reads kv head h // (Hq/Hkv).
    Scores are scaled by 1/sqrt(hd).  Returns [Hq][hd].
    """
    hq, hd = q.shape
    g = hq // n_kv_heads
    qg = q.reshape(n_kv_heads, g, hd)
    s = np.einsum("kgd,nkd->kgn", qg, K) / np.sqrt(hd)
    s = s - s.max(axis=-1, keepdims=True)
    p = np.exp(s)
    p = p / p.sum(axis=-1, keepdims=True)
    return np.einsum("kgn,nkd->kgd", p, V).reshape(hq, hd)


def argmax_rows(logits):
    """Greedy token per row; ties go to the lowest id (numpy argmax rule)."""
    return np.argmax(logits, axis=-1).astype(np.int32)


def top2_gap(logits):
    """top-1 minus top-2 logit per row (how safely the argmax is decided)."""
    part = np.sort(np.asarray(logits, F), axis=-1)
    return part[..., -1] - part[..., -2]


def log_softmax(z):
    """log of the softmax of the last axis (temperature 1), in float64."""
    z = np.asarray(z, F)
    m = z.max(axis=-1, keepdims=True)
    return z - m - np.log(np.exp(z - m).sum(axis=-1, keepdims=True))


def gumbel_argmax(logw, g):
    """A sample of the distribution proportional to exp(logw) by the Gumbel-max
    rule: argmax_v (logw_v + g_v) with g_v standard Gumbel; -inf never wins."""
    return int(np.argmax(np.asarray(logw, F) + np.asarray(g, F)))


def speculative_sample(block, p_logits, q_logits, ua, gr):
    """T = 1 verification of one draft block by speculative sampling (the reading
    of Sec. 5.2's T = 1 rows: the paper does not print its rule; this is the
    standard rule for proposals drawn from a known distribution).

    p_i = softmax(p_logits[i - 1]) is the target's distribution for offset i
    (verify row i - 1), q_i = softmax(q_logits[i]) the drafter's for the
    proposal block[i], i = 1..B.  Proposal i is accepted when ua[i] <
    p_i(y_i) / q_i(y_i); at the first rejection the token of offset i is drawn
    from max(0, p_i - q_i) normalised; after B acceptances the bonus is drawn
    from p_{B+1}.  gr[i - 1] is the Gumbel noise of offset i's draw.
    Returns (a, token committed after the a accepted proposals)."""
    B = len(block) - 1
    for i in range(1, B + 1):
        lp, lq = log_softmax(p_logits[i - 1]), log_softmax(q_logits[i])
        y = int(block[i])
        if np.log(ua[i]) < lp[y] - lq[y]:
            continue
        r = np.exp(lp) - np.exp(lq)
        if not (r > 0).any():  # only through rounding (a rejection implies p_i(v) > q_i(v) somewhere): draw from p_i
            return i - 1, gumbel_argmax(lp, gr[i - 1])
        with np.errstate(divide="ignore"):
            logr = np.where(r > 0, np.log(np.where(r > 0, r, 1.0)), -np.inf)
        return i - 1, gumbel_argmax(logr, gr[i - 1])
    return B, gumbel_argmax(log_softmax(p_logits[B]), gr[B])


# ---------------------------------------------------------------------------
# state
# ---------------------------------------------------------------------------


@dataclasses.dataclass
class State:
    """Logical (position-indexed) decoding state of a batch.

    tokens[b][0..n-1] committed; target K/V valid at positions 0..n-2; drafter
    context K/V valid at 0..n-2; tokens[b][n-1] is the anchor whose KV is not
    yet computed.  carry[b][j-1] holds slot j's relayed feature for j <= n_carry.
    """

    tokens: np.ndarray  # [bs][cap] int32
    seq_len: np.ndarray  # [bs] int32 (n)
    k: np.ndarray  # [L][bs][cap][Hkv][hd]
    v: np.ndarray
    dk: np.ndarray  # [Ld][bs][cap][Hkv][hd]
    dv: np.ndarray
    carry: np.ndarray  # [bs][B][d]
    n_carry: np.ndarray  # [bs]
    boundary: np.ndarray  # [bs][2]: (bonus b, first rejected proposal y_{a+1}); -1 if none
    active: np.ndarray  # [bs] bool

    def copy(self) -> "State":
        return State(**{f.name: np.array(getattr(self, f.name), copy=True)
                        for f in dataclasses.fields(self)})


@dataclasses.dataclass
class RoundOut:
    block: np.ndarray  # [bs][B+1] draft block (row 0 = anchor)
    draft_logits: np.ndarray  # [bs][B+1][V] (row 0 unused)
    draft_x: np.ndarray  # [bs][B+1][d] drafter inputs (Eq. 5)
    g: np.ndarray  # [bs][B+1] target argmax per row
    verify_logits: np.ndarray  # [bs][B+1][V]
    feats: np.ndarray  # [bs][B+1][d] Eq. 1 features of the verify rows
    accept: np.ndarray  # [bs] a
    committed: np.ndarray  # [bs][B+1] committed tokens, -1 padded
    n_before: np.ndarray  # [bs] n at the start of the round


# ---------------------------------------------------------------------------
# the oracle
# ---------------------------------------------------------------------------


class Oracle:
    """The DFlow round on the CPU.  `W` maps synth tensor names to fp32 arrays."""

    def __init__(self, cfg, W: Dict[str, np.ndarray]):
        self.cfg = cfg
        self.W = W

    # -- helpers -----------------------------------------------------------

    def w(self, name):
        return self.W[name]

    def new_state(self, cap: Optional[int] = None) -> State:
        c = self.cfg
        cap = c.max_ctx() if cap is None else cap
        bs, hkv, hd = c.batch, c.n_kv_heads, c.head_dim
        return State(
            tokens=np.zeros((bs, cap), np.int32), seq_len=np.zeros(bs, np.int32),
            k=np.zeros((c.n_layers, bs, cap, hkv, hd), F), v=np.zeros((c.n_layers, bs, cap, hkv, hd), F),
            dk=np.zeros((c.draft_layers, bs, cap, hkv, hd), F),
            dv=np.zeros((c.draft_layers, bs, cap, hkv, hd), F),
            carry=np.zeros((bs, c.block, c.d), F), n_carry=np.zeros(bs, np.int32),
            boundary=np.full((bs, 2), -1, np.int32), active=np.ones(bs, bool))

    def state_from_synthetic(self, s: Dict[str, np.ndarray]) -> State:
        """Wrap a synth.synthetic_state() dict (logical arrays) as an oracle State."""
        bs = self.cfg.batch
        return State(tokens=s["tokens"].copy(), seq_len=s["seq_len"].copy(),
                     k=s["k"].astype(F), v=s["v"].astype(F), dk=s["dk"].astype(F),
                     dv=s["dv"].astype(F), carry=s["carry"].astype(F),
                     n_carry=s["n_carry"].copy(), boundary=s["boundary"].copy(),
                     active=np.ones(bs, bool))

    def _mlp(self, pfx, x):
        """Qwen3 SwiGLU MLP: W_d (silu(W_g h) * W_u h) with h = RMSNorm(x)."""
        h = rmsnorm(x, self.w(pfx + "mlp_norm"), self.cfg.rms_eps)
        return (silu(h @ self.w(pfx + "wg").T) * (h @ self.w(pfx + "wu").T)) @ self.w(pfx + "wd").T

    def _qkv(self, pfx, x, pos):
        """Pre-norm Q/K/V projections with per-head q/k RMSNorm and RoPE at `pos`."""
        c = self.cfg
        h = rmsnorm(x, self.w(pfx + "attn_norm"), c.rms_eps)
        r = x.shape[0]
        q = (h @ self.w(pfx + "wq").T).reshape(r, c.n_q_heads, c.head_dim)
        k = (h @ self.w(pfx + "wk").T).reshape(r, c.n_kv_heads, c.head_dim)
        v = (h @ self.w(pfx + "wv").T).reshape(r, c.n_kv_heads, c.head_dim)
        q = rope(rmsnorm(q, self.w(pfx + "q_norm"), c.rms_eps), pos, c.rope_theta)
        k = rope(rmsnorm(k, self.w(pfx + "k_norm"), c.rms_eps), pos, c.rope_theta)
        return q, k, v

    def lm_logits(self, x, norm_name):
        return rmsnorm(x, self.w(norm_name), self.cfg.rms_eps) @ self.w("lm_head").T

    # -- Eq. 1 -------------------------------------------------------------

    def feature_projection(self, stash: List[np.ndarray]) -> np.ndarray:
        """Eq. 1: H_T = RMSNorm(W_c [H^l1; ...; H^lm]) per row."""
        cat = np.concatenate(stash, axis=-1)
        return rmsnorm(cat @ self.w("w_c").T, self.w("c_norm"), self.cfg.rms_eps)

    # -- target forward over a block of rows (Sec. 3, exact-match verification)

    def target_forward(self, st: State, b: int, toks: Sequence[int], pos0: int):
        """Target forward of rows toks at positions pos0.. against the cached K/V.

        Writes K/V of every row into the cache, attends causally (row at
        position p sees keys 0..p) and returns (logits, features Eq. 1).
        """
        c = self.cfg
        toks = np.asarray(toks, np.int64)
        r = len(toks)
        pos = pos0 + np.arange(r)
        x = self.w("embed")[toks].astype(F)
        stash = []
        for l in range(c.n_layers):
            pfx = f"t{l}."
            q, k, v = self._qkv(pfx, x, pos)
            st.k[l, b, pos0:pos0 + r] = k
            st.v[l, b, pos0:pos0 + r] = v
            o = np.stack([attend(q[i], st.k[l, b, :pos[i] + 1], st.v[l, b, :pos[i] + 1], c.n_kv_heads)
                          for i in range(r)])
            x = x + o.reshape(r, -1) @ self.w(pfx + "wo").T
            x = x + self._mlp(pfx, x)
            if (l + 1) in c.feat_layers:
                stash.append(x.copy())
        logits = self.lm_logits(x, "final_norm")
        return logits, self.feature_projection(stash)

    # -- drafter context injection (Sec. 3: H_T into draft K/V) -------------

    def ctx_append(self, st: State, b: int, feats: np.ndarray, pos0: int):
        """K/V of fused target features for positions pos0.. in every draft layer."""
        c = self.cfg
        r = feats.shape[0]
        pos = pos0 + np.arange(r)
        for l in range(c.draft_layers):
            pfx = f"d{l}."
            k = (feats @ self.w(pfx + "wk").T).reshape(r, c.n_kv_heads, c.head_dim)
            v = (feats @ self.w(pfx + "wv").T).reshape(r, c.n_kv_heads, c.head_dim)
            st.dk[l, b, pos0:pos0 + r] = rope(rmsnorm(k, self.w(pfx + "k_norm"), c.rms_eps), pos, c.rope_theta)
            st.dv[l, b, pos0:pos0 + r] = v

    # -- prefill -------------------------------------------------------------

    def prefill(self, st: State, b: int, prompt: Sequence[int]):
        """Prompt rows 0..P-1 through the target; first new token = argmax at P-1."""
        p = len(prompt)
        st.tokens[b, :p] = prompt
        logits, feats = self.target_forward(st, b, prompt, 0)
        st.tokens[b, p] = argmax_rows(logits[-1:])[0]
        st.seq_len[b] = p + 1
        self.ctx_append(st, b, feats, 0)
        st.n_carry[b] = 0
        st.boundary[b] = -1
        st.active[b] = True
        return logits

    # -- Eq. 4 and Eq. 5 -----------------------------------------------------

    def relay_mlp(self, e_b, e_rej, h):
        """Eq. 4: [beta; gamma] = MLP_phi([E(b); E(y_{a+1}); h])."""
        d = self.cfg.d
        u = np.concatenate([e_b, e_rej, h])
        bg = self.w("relay_w2") @ silu(self.w("relay_w1") @ u)
        return bg[:d], bg[d:]

    def draft_inputs(self, st: State, b: int) -> np.ndarray:
        """Eq. 5 drafter inputs: E(anchor) in row 0, relay at valid carried slots, E_mask elsewhere."""
        c = self.cfg
        n = int(st.seq_len[b])
        e_mask = self.w("e_mask").astype(F)
        x = np.tile(e_mask, (c.rows, 1))
        x[0] = self.w("embed")[st.tokens[b, n - 1]]
        nc = int(st.n_carry[b])
        if nc > 0:
            e_b = self.w("embed")[st.boundary[b, 0]].astype(F)
            e_r = self.w("embed")[st.boundary[b, 1]].astype(F)
            for j in range(1, nc + 1):
                h = st.carry[b, j - 1]
                beta, gamma = self.relay_mlp(e_b, e_r, h)
                x[j] = e_mask + beta * layernorm(h, self.w("ln_w"), self.w("ln_b"), c.ln_eps) + gamma
        return x

    # -- Eq. 2: one-shot block drafting -------------------------------------

    def draft_block(self, st: State, b: int, x: Optional[np.ndarray] = None, gd: Optional[np.ndarray] = None):
        """Drafter forward over the B+1 block rows; argmax of rows 1..B, or with
        gd (Gumbel noise [B+1][V]) a T = 1 sample of each row's distribution.

        Keys/values of draft layer l are [context K/V at 0..n-2 ; block rows],
        all visible to every block row.  Returns (block tokens, logits, inputs).
        """
        c = self.cfg
        n = int(st.seq_len[b])
        pos = n - 1 + np.arange(c.rows)
        x = self.draft_inputs(st, b) if x is None else np.asarray(x, F)
        x0 = x.copy()
        for l in range(c.draft_layers):
            pfx = f"d{l}."
            q, k, v = self._qkv(pfx, x, pos)
            K = np.concatenate([st.dk[l, b, :n - 1], k])
            V = np.concatenate([st.dv[l, b, :n - 1], v])
            o = np.stack([attend(q[i], K, V, c.n_kv_heads) for i in range(c.rows)])
            x = x + o.reshape(c.rows, -1) @ self.w(pfx + "wo").T
            x = x + self._mlp(pfx, x)
        logits = self.lm_logits(x, "d.final_norm")
        block = np.empty(c.rows, np.int32)
        block[0] = st.tokens[b, n - 1]
        block[1:] = argmax_rows(logits[1:]) if gd is None else [gumbel_argmax(logits[i], gd[i])
                                                                 for i in range(1, c.rows)]
        return block, logits, x0

    # -- Eq. 3: verification ---------------------------------------------------

    def verify_block(self, st: State, b: int, block: Sequence[int]):
        """Target forward over [anchor, y^_1..y^_B] at positions n-1..n-1+B."""
        n = int(st.seq_len[b])
        logits, feats = self.target_forward(st, b, block, n - 1)
        return argmax_rows(logits), logits, feats

    def accept_commit(self, st: State, b: int, block, g, forced: Optional[int] = None):
        """Eq. 3: a = number of leading proposals equal to the target's predictions.

        y^_i is checked against g[i-1] (the target's prediction for its position).
        Commit y^_1..y^_a and the bonus g[a]; n grows by a+1.  A forced a
        (benchmark mode) replaces the matched length.
        """
        B = self.cfg.block
        a = 0
        while a < B and int(block[a + 1]) == int(g[a]):
            a += 1
        if forced is not None:
            a = int(forced)
        bonus = int(g[a])
        committed = np.full(B + 1, -1, np.int32)
        committed[:a] = block[1:a + 1]
        committed[a] = bonus
        n = int(st.seq_len[b])
        st.tokens[b, n:n + a + 1] = committed[:a + 1]
        st.seq_len[b] = n + a + 1
        return a, committed

    def carry_hidden(self, st: State, b: int, block, feats: np.ndarray, a: int, relay: bool = True):
        """Sec. 4.2 alignment + Sec. 3 context injection after a commit.

        Rows 0..a (anchor and accepted tokens, positions n-1..n-1+a) join the
        drafter context.  Rows a+1..B-1 are carried, shifted by one: next-round
        slot j takes row a+j.  Boundary tokens are (bonus, y^_{a+1}).  With the
        relay off (the DFlash baseline of Sec. 5.3) nothing is carried.
        """
        B = self.cfg.block
        n_new = int(st.seq_len[b])
        n_old = n_new - a - 1
        self.ctx_append(st, b, feats[:a + 1], n_old - 1)
        nc = max(0, B - a - 1) if relay else 0
        st.n_carry[b] = nc
        st.carry[b] = 0.0
        for j in range(1, nc + 1):
            st.carry[b, j - 1] = feats[a + j]
        st.boundary[b, 0] = st.tokens[b, n_new - 1]
        st.boundary[b, 1] = int(block[a + 1]) if a < B else -1

    # -- one round ---------------------------------------------------------

    def round(self, st: State, forced: Optional[Sequence[Optional[int]]] = None,
              draft_override: Optional[Callable[[int, State], np.ndarray]] = None,
              relay: bool = True) -> RoundOut:
        """draft -> verify -> accept/commit -> carry for every active sequence."""
        c = self.cfg
        bs, R, V = c.batch, c.rows, c.vocab
        out = RoundOut(block=np.zeros((bs, R), np.int32), draft_logits=np.zeros((bs, R, V)),
                       draft_x=np.zeros((bs, R, c.d)), g=np.zeros((bs, R), np.int32),
                       verify_logits=np.zeros((bs, R, V)), feats=np.zeros((bs, R, c.d)),
                       accept=np.zeros(bs, np.int32), committed=np.full((bs, R), -1, np.int32),
                       n_before=st.seq_len.copy())
        for b in range(bs):
            if not st.active[b]:
                continue
            if not relay:
                st.n_carry[b] = 0
            if draft_override is not None:
                blk = np.asarray(draft_override(b, st), np.int32)
                out.draft_x[b] = self.draft_inputs(st, b)
            else:
                blk, out.draft_logits[b], out.draft_x[b] = self.draft_block(st, b)
            g, out.verify_logits[b], feats = self.verify_block(st, b, blk)
            a, comm = self.accept_commit(st, b, blk, g, None if forced is None else forced[b])
            self.carry_hidden(st, b, blk, feats, a, relay)
            out.block[b], out.g[b], out.feats[b] = blk, g, feats
            out.accept[b], out.committed[b] = a, comm
        return out

    # -- one round with T = 1 sampling verification (Sec. 5.2, Table 1 T = 1) --

    def round_sampled(self, st: State, noise: Callable[[int], Dict[str, np.ndarray]],
                      relay: bool = True) -> RoundOut:
        """draft (T = 1 samples) -> verify -> speculative sampling -> commit -> carry.

        noise(b) gives sequence b's draws for this round (synth.sampling_noise:
        gd, ua, gr).  The relay and the carry are those of the greedy round: the
        boundary tokens are the committed last token and the first rejected
        proposal."""
        c = self.cfg
        bs, R, V = c.batch, c.rows, c.vocab
        out = RoundOut(block=np.zeros((bs, R), np.int32), draft_logits=np.zeros((bs, R, V)),
                       draft_x=np.zeros((bs, R, c.d)), g=np.zeros((bs, R), np.int32),
                       verify_logits=np.zeros((bs, R, V)), feats=np.zeros((bs, R, c.d)),
                       accept=np.zeros(bs, np.int32), committed=np.full((bs, R), -1, np.int32),
                       n_before=st.seq_len.copy())
        for b in range(bs):
            if not st.active[b]:
                continue
            if not relay:
                st.n_carry[b] = 0
            nz = noise(b)
            blk, out.draft_logits[b], out.draft_x[b] = self.draft_block(st, b, gd=nz["gd"])
            g, out.verify_logits[b], feats = self.verify_block(st, b, blk)
            a, tok = speculative_sample(blk, out.verify_logits[b], out.draft_logits[b], nz["ua"], nz["gr"])
            gs = np.array(g, copy=True)
            gs[a] = tok
            a, comm = self.accept_commit(st, b, blk, gs, a)
            self.carry_hidden(st, b, blk, feats, a, relay)
            out.block[b], out.g[b], out.feats[b] = blk, gs, feats
            out.accept[b], out.committed[b] = a, comm
        return out

    # -- whole generation ----------------------------------------------------

    def generate(self, prompts: List[Sequence[int]], n_new: int,
                 forced: Optional[Callable[[int, int], int]] = None,
                 draft_override: Optional[Callable[[int, State], np.ndarray]] = None,
                 relay: bool = True, rounds_out: Optional[list] = None):
        """Prefill, then rounds until every sequence has >= n_new new tokens.

        Returns the first n_new generated tokens of each sequence.
        """
        st = self.new_state()
        plen = [len(p) for p in prompts]
        for b, p in enumerate(prompts):
            self.prefill(st, b, p)
        r = 0
        while True:
            for b in range(self.cfg.batch):
                st.active[b] = (st.seq_len[b] - plen[b]) < n_new
            if not st.active.any():
                break
            fa = None if forced is None else [forced(b, r) for b in range(self.cfg.batch)]
            ro = self.round(st, fa, draft_override, relay)
            if rounds_out is not None:
                rounds_out.append(ro)
            r += 1
        return [st.tokens[b, plen[b]:plen[b] + n_new].copy() for b in range(self.cfg.batch)], st

    # -- plain autoregressive decoding (Sec. 5.2, Table 2 "Baseline") ----------

    def decode_step(self, st: State, b: int, draft_context: bool = False):
        """One step of ordinary greedy decoding of the target with its KV cache:
        the last committed token (position n-1) runs through the target, its
        K/V join the cache, and its greedy prediction is committed (n grows by
        one).  draft_context: the row's Eq. 1 feature also joins the drafter
        context, so that speculative rounds can follow.  Returns the token."""
        n = int(st.seq_len[b])
        logits, feats = self.target_forward(st, b, [int(st.tokens[b, n - 1])], n - 1)
        tok = int(argmax_rows(logits)[0])
        st.tokens[b, n] = tok
        st.seq_len[b] = n + 1
        if draft_context:
            self.ctx_append(st, b, feats, n - 1)
        st.n_carry[b] = 0
        st.boundary[b] = -1
        return tok, logits[0]

    # -- brute-force greedy reference (no cache, full causal recompute) -------

    def full_logits(self, seq: Sequence[int]) -> np.ndarray:
        """Target logits at every position of seq, recomputed from scratch.

        Causal attention is evaluated as full score matrices with the upper
        triangle masked, with no KV cache and no blocks.
        """
        c = self.cfg
        seq = np.asarray(seq, np.int64)
        T = len(seq)
        pos = np.arange(T)
        x = self.w("embed")[seq].astype(F)
        g = c.n_q_heads // c.n_kv_heads
        mask = np.triu(np.full((T, T), -np.inf), 1)
        for l in range(c.n_layers):
            pfx = f"t{l}."
            q, k, v = self._qkv(pfx, x, pos)
            o = np.empty_like(q)
            for h in range(c.n_q_heads):
                s = q[:, h] @ k[:, h // g].T / np.sqrt(c.head_dim) + mask
                p = np.exp(s - s.max(axis=1, keepdims=True))
                o[:, h] = (p / p.sum(axis=1, keepdims=True)) @ v[:, h // g]
            x = x + o.reshape(T, -1) @ self.w(pfx + "wo").T
            x = x + self._mlp(pfx, x)
        return self.lm_logits(x, "final_norm")

    def greedy_decode(self, prompt: Sequence[int], n_new: int) -> np.ndarray:
        """Plain token-by-token greedy decoding of the target (brute force)."""
        seq = list(int(t) for t in prompt)
        for _ in range(n_new):
            seq.append(int(argmax_rows(self.full_logits(seq)[-1:])[0]))
        return np.asarray(seq[len(prompt):], np.int32)
