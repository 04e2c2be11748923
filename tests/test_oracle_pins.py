"""Pins of the CPU oracle against what the paper and the mathematics fix.

No test here retypes an oracle formula: each one checks a closed form worked by
hand, a library routine, an invariant, or a brute-force recomputation.
"""
import math
from pathlib import Path

import numpy as np
import pytest
import torch

import synth
from oracle import Oracle, argmax_rows, attend, layernorm, rmsnorm, rope, silu, top2_gap

TINY = synth.TINY


@pytest.fixture(scope="module")
def tiny_w():
    return synth.weights(TINY, perturb_norms=True)


@pytest.fixture(scope="module")
def tiny_oracle(tiny_w):
    return Oracle(TINY, tiny_w)


# ---------------------------------------------------------------------------
# elementary operations
# ---------------------------------------------------------------------------


def test_rmsnorm_hand_value():
    # x = (3, 4): mean square 12.5; gains (1, 2)
    y = rmsnorm(np.array([3.0, 4.0]), np.array([1.0, 2.0]), 0.0)
    r = math.sqrt(12.5)
    assert np.allclose(y, [3 / r, 8 / r], rtol=0, atol=1e-15)


def test_layernorm_matches_torch():
    rng = np.random.default_rng(0)
    x, w, b = rng.normal(size=(5, 32)), rng.normal(size=32), rng.normal(size=32)
    ref = torch.nn.functional.layer_norm(torch.tensor(x), (32,), torch.tensor(w), torch.tensor(b), 1e-6)
    assert np.allclose(layernorm(x, w, b, 1e-6), ref.numpy(), atol=1e-12)


def test_silu_matches_torch():
    x = np.linspace(-12, 12, 97)
    assert np.allclose(silu(x), torch.nn.functional.silu(torch.tensor(x)).numpy(), atol=1e-14)


def test_rope_complex_form_and_relative_offsets():
    hd, theta = 16, 1.0e6
    rng = np.random.default_rng(1)
    x = rng.normal(size=hd)
    for p in (0, 1, 7, 4097):
        # rotate-half pairing as a complex number z_i = x_i + i x_{i+hd/2} times e^{i p w_i}
        w = theta ** (-np.arange(hd // 2) * 2.0 / hd)
        z = (x[: hd // 2] + 1j * x[hd // 2:]) * np.exp(1j * p * w)
        assert np.allclose(rope(x, p, theta), np.concatenate([z.real, z.imag]), atol=1e-12)
    assert np.allclose(rope(x, 0, theta), x)
    q, k = rng.normal(size=hd), rng.normal(size=hd)
    d1 = rope(q, 40, theta) @ rope(k, 33, theta)
    d2 = rope(q, 1007, theta) @ rope(k, 1000, theta)
    assert abs(d1 - d2) < 1e-10
    assert abs(np.linalg.norm(rope(q, 123, theta)) - np.linalg.norm(q)) < 1e-12


def test_attend_matches_torch_sdpa_gqa():
    rng = np.random.default_rng(2)
    hq, hkv, hd, n = 8, 2, 16, 11
    q = rng.normal(size=(hq, hd))
    K, V = rng.normal(size=(n, hkv, hd)), rng.normal(size=(n, hkv, hd))
    # library routine in plain multi-head form: each kv head repeated for its query group
    Kr = torch.tensor(K).permute(1, 0, 2).repeat_interleave(hq // hkv, dim=0)
    Vr = torch.tensor(V).permute(1, 0, 2).repeat_interleave(hq // hkv, dim=0)
    ref = torch.nn.functional.scaled_dot_product_attention(torch.tensor(q)[:, None, :], Kr, Vr)[:, 0]
    assert np.allclose(attend(q, K, V, hkv), ref.numpy(), atol=1e-12)


def test_argmax_ties_lowest_id_and_gap():
    lg = np.array([[0.0, 2.0, 2.0, 1.0], [5.0, 5.0, 5.0, 5.0]])
    assert list(argmax_rows(lg)) == [1, 0]
    assert np.allclose(top2_gap(np.array([[1.0, 3.0, 2.5]])), [0.5])


# ---------------------------------------------------------------------------
# a hand-sized model: the SwiGLU gate/up order and the pre-norm placement
# ---------------------------------------------------------------------------


def _micro_oracle(**over):
    cfg = synth.TINY.replace(d=4, n_layers=1, n_q_heads=2, n_kv_heads=1, head_dim=2, inter=2,
                             vocab=5, draft_layers=1, feat_layers=(1,), block=2)
    W = {k: np.zeros(s, np.float32) for k, s in synth.tensor_shapes(cfg).items()}
    for k in W:
        if k.endswith("norm") or k == "ln_w":
            W[k][:] = 1.0
    W.update(over)
    return cfg, Oracle(cfg, W)


def test_mlp_gate_up_order_hand_value():
    # x = (c, c, c, c) has RMSNorm h = (1, 1, 1, 1) (eps 1e-6 negligible at c = 10)
    wg = np.full((2, 4), 0.25, np.float32)  # gate pre-activation 1
    wu = np.full((2, 4), 0.50, np.float32)  # up pre-activation 2
    wd = np.zeros((4, 2), np.float32)
    wd[0, 0] = 1.0
    cfg, o = _micro_oracle(**{"t0.wg": wg, "t0.wu": wu, "t0.wd": wd})
    out = o._mlp("t0.", np.full((1, 4), 10.0))
    # silu(1) * 2 = 2 / (1 + e^-1) = 1.4621171572600098; swapping gate and up would give silu(2) * 1
    assert abs(out[0, 0] - 1.4621171572600098) < 1e-6
    assert np.allclose(out[0, 1:], 0.0)


def test_zero_blocks_leave_embedding_in_residual():
    # W_o = W_d = 0: every layer is the identity on the residual stream, so the
    # logits are RMSNorm(E[tok]) . lm_head^T exactly
    rng = np.random.default_rng(3)
    emb = rng.normal(size=(5, 4)).astype(np.float32)
    lm = rng.normal(size=(5, 4)).astype(np.float32)
    cfg, o = _micro_oracle(embed=emb, lm_head=lm, **{"t0.wq": rng.normal(size=(4, 4)).astype(np.float32)})
    st = o.new_state(cap=16)
    logits, _ = o.target_forward(st, 0, [3, 1], 0)
    for i, t in enumerate([3, 1]):
        x = emb[t].astype(np.float64)
        ref = (x / np.sqrt(np.mean(x * x) + cfg.rms_eps)) @ lm.T.astype(np.float64)
        assert np.allclose(logits[i], ref, atol=1e-12)


# ---------------------------------------------------------------------------
# Qwen3 attention inputs: per-head q/k RMSNorm (with its gains) comes first,
# the rotary embedding last; the drafter's context keys/values (Sec. 3: target
# features injected into the K and V projections) follow the same order with no
# input norm.  Hand values use head_dim 2, where the rotary embedding at
# position p is multiplication of (x0 + i x1) by e^{ip} (theta^0 = 1).
# ---------------------------------------------------------------------------


def _rot(x0, x1, p):
    z = complex(x0, x1) * complex(math.cos(p), math.sin(p))
    return [z.real, z.imag]


def _attn_micro(**over):
    f32 = lambda rows: np.array(rows, np.float32)  # noqa: E731
    w = {
        "t0.wq": f32([[3, 0, 0, 0], [0, 4, 0, 0], [0, 0, 1, 0], [0, 0, 0, -2]]),
        "t0.wk": f32([[0, 0, 2, 0], [0, 0, 0, 1]]),
        "t0.wv": f32([[1, 1, 0, 0], [0, 0, 1, 1]]),
        "t0.q_norm": f32([1, 2]),
        "t0.k_norm": f32([0.5, 3]),
        "embed": f32([[0, 0, 0, 0], [10, 10, 10, 10], [-5, -5, -5, -5], [0, 0, 0, 0], [0, 0, 0, 0]]),
    }
    w.update(over)
    return _micro_oracle(**w)


def test_qk_rmsnorm_with_gains_then_rotary_hand_values():
    cfg, o = _attn_micro()
    # h = RMSNorm(10, 10, 10, 10) = (1, 1, 1, 1): q head 0 = (3, 4), head 1 = (1, -2), k = (2, 1)
    q, k, v = o._qkv("t0.", np.full((1, 4), 10.0), np.array([5]))
    r0, r1, rk = math.sqrt(12.5), math.sqrt(2.5), math.sqrt(2.5)
    want_q0 = _rot(3 / r0 * 1, 4 / r0 * 2, 5)  # normalised, gains (1, 2), then rotated by 5 rad
    want_q1 = _rot(1 / r1 * 1, -2 / r1 * 2, 5)
    want_k = _rot(2 / rk * 0.5, 1 / rk * 3, 5)  # gains (0.5, 3)
    assert np.allclose(q[0, 0], want_q0, atol=1e-6)
    assert np.allclose(q[0, 1], want_q1, atol=1e-6)
    assert np.allclose(k[0, 0], want_k, atol=1e-6)
    assert np.allclose(v[0, 0], [2, 2], atol=1e-6)  # values: no norm, no rotation


def test_target_cache_keys_hand_values_at_their_positions():
    # W_o = W_d = 0 keep the residual at the embedding; tokens 1 and 2 have
    # RMSNorm(E) = (1, 1, 1, 1) and (-1, -1, -1, -1); written at positions 3 and 4
    cfg, o = _attn_micro()
    st = o.new_state(cap=16)
    o.target_forward(st, 0, [1, 2], 3)
    rk = math.sqrt(2.5)
    assert np.allclose(st.k[0, 0, 3, 0], _rot(1 / rk, 3 / rk, 3), atol=1e-6)
    assert np.allclose(st.k[0, 0, 4, 0], _rot(-1 / rk, -3 / rk, 4), atol=1e-6)
    assert np.allclose(st.v[0, 0, 3, 0], [2, 2], atol=1e-6)
    assert np.allclose(st.v[0, 0, 4, 0], [-2, -2], atol=1e-6)
    assert not st.k[0, 0, :3].any() and not st.k[0, 0, 5:].any()


def test_qk_scores_depend_only_on_relative_offset(tiny_oracle):
    """RoPE's defining property holds for the projected q/k only if the rotation
    is applied after the per-head norm (the gains are not rotation invariant)."""
    o = tiny_oracle
    assert np.ptp(o.W["t0.q_norm"]) > 0.1 and np.ptp(o.W["t0.k_norm"]) > 0.1
    x = np.random.default_rng(11).normal(size=(2, TINY.d))
    qa, _, _ = o._qkv("t0.", x[:1], np.array([37]))
    _, ka, _ = o._qkv("t0.", x[1:], np.array([30]))
    qb, _, _ = o._qkv("t0.", x[:1], np.array([1037]))
    _, kb, _ = o._qkv("t0.", x[1:], np.array([1030]))
    sa = np.einsum("hd,kd->hk", qa[0], ka[0])
    sb = np.einsum("hd,kd->hk", qb[0], kb[0])
    assert np.allclose(sa, sb, atol=1e-9)


def test_target_keys_and_logits_invariant_to_qk_projection_scale(tiny_w):
    """Per-head RMSNorm on q and k removes the scale of W_q and W_k (up to eps)."""
    prompt = synth.prompts(TINY)[0][:12]
    o = Oracle(TINY, tiny_w)
    st = o.new_state()
    lg, _ = o.target_forward(st, 0, prompt, 0)
    W = dict(tiny_w)
    for l in range(TINY.n_layers):
        W[f"t{l}.wq"] = W[f"t{l}.wq"] * 4.0
        W[f"t{l}.wk"] = W[f"t{l}.wk"] * 4.0
    o2 = Oracle(TINY, W)
    st2 = o2.new_state()
    lg2, _ = o2.target_forward(st2, 0, prompt, 0)
    # eps 1e-6 against mean squares near 0.1 leaves about 1e-5 of the scale
    k1, k2 = st.k[:, 0, :12], st2.k[:, 0, :12]
    assert np.abs(k1 - k2).max() < 1e-4 * np.abs(k1).max()
    assert np.abs(lg - lg2).max() < 1e-4 * np.abs(lg).max()


def test_context_kv_injection_hand_values():
    """Sec. 3: feature f at position p enters draft layer l as
    k = RoPE(k_norm(W_k f), p), v = W_v f (f is RMSNormed by Eq. 1 already)."""
    f32 = lambda rows: np.array(rows, np.float32)  # noqa: E731
    cfg, o = _micro_oracle(**{"d0.wk": f32([[1, 0, 0, 0], [0, 1, 0, 0]]), "d0.wv": f32([[0, 0, 0, 1], [1, 1, 0, 0]]),
                              "d0.k_norm": f32([2, 0.5])})
    st = o.new_state(cap=16)
    feats = np.array([[1.0, 2.0, 0.0, -1.0], [-3.0, 1.0, 5.0, 2.0]])
    o.ctx_append(st, 0, feats, 7)
    r1, r2 = math.sqrt(2.5), math.sqrt(5.0)  # RMS of (1, 2) and of (-3, 1)
    assert np.allclose(st.dk[0, 0, 7, 0], _rot(1 / r1 * 2, 2 / r1 * 0.5, 7), atol=1e-6)
    assert np.allclose(st.dk[0, 0, 8, 0], _rot(-3 / r2 * 2, 1 / r2 * 0.5, 8), atol=1e-6)
    assert np.allclose(st.dv[0, 0, 7, 0], [-1, 3], atol=1e-12)
    assert np.allclose(st.dv[0, 0, 8, 0], [2, -2], atol=1e-12)
    assert not st.dk[0, 0, :7].any() and not st.dk[0, 0, 9:].any()


def test_context_keys_scale_free_values_linear(tiny_oracle):
    """The context key is k-normed (invariant to the feature's scale); the value
    is a plain projection (linear in it: no input norm)."""
    o = tiny_oracle
    f = np.random.default_rng(12).normal(size=(3, TINY.d))
    s1, s2 = o.new_state(), o.new_state()
    o.ctx_append(s1, 0, f, 20)
    o.ctx_append(s2, 0, 3.0 * f, 20)
    k1, k2 = s1.dk[:, 0, 20:23], s2.dk[:, 0, 20:23]
    assert np.abs(k1 - k2).max() < 1e-4 * np.abs(k1).max()  # eps 1e-6 leaves about 1e-5
    assert np.allclose(3.0 * s1.dv[:, 0, 20:23], s2.dv[:, 0, 20:23], atol=1e-12)


# ---------------------------------------------------------------------------
# target forward: cached block forward == brute-force full recompute
# ---------------------------------------------------------------------------


def test_cached_block_forward_equals_full_recompute(tiny_oracle):
    o = tiny_oracle
    prompt = synth.prompts(TINY)[0][:20]
    st = o.new_state()
    o.prefill(st, 0, prompt)
    blk = [int(st.tokens[0, 20])] + [5, 77, 900, 3, 3, 41, 2, 1000]
    g, logits, _ = o.verify_block(st, 0, blk)
    full = o.full_logits(list(prompt) + blk)
    assert np.allclose(logits, full[20:29], rtol=0, atol=1e-9)
    assert list(g) == list(argmax_rows(full[20:29]))


def test_verify_is_causal_inside_the_block(tiny_oracle):
    o = tiny_oracle
    prompt = synth.prompts(TINY)[0][:16]
    st = o.new_state()
    o.prefill(st, 0, prompt)
    anchor = int(st.tokens[0, 16])
    blk = [anchor, 1, 2, 3, 4, 5, 6, 7, 8]
    _, l1, _ = o.verify_block(st.copy(), 0, blk)
    _, l2, _ = o.verify_block(st.copy(), 0, blk[:-1] + [999])
    assert np.allclose(l1[:-1], l2[:-1], atol=0)
    assert not np.allclose(l1[-1], l2[-1])


# ---------------------------------------------------------------------------
# Eq. 1 feature projection: with W_c selecting the last layer's stream and
# c_norm == final_norm, feats . lm_head^T reproduces the target logits
# ---------------------------------------------------------------------------


def test_feature_projection_selects_layer_outputs(tiny_w):
    W = dict(tiny_w)
    d = TINY.d
    wc = np.zeros((d, 2 * d), np.float32)
    wc[:, d:] = np.eye(d)  # second feature layer (= layer 2, the last)
    W["w_c"] = wc
    W["c_norm"] = W["final_norm"]
    o = Oracle(TINY, W)
    st = o.new_state()
    logits, feats = o.target_forward(st, 0, synth.prompts(TINY)[0][:12], 0)
    assert np.allclose(feats @ W["lm_head"].T.astype(np.float64), logits, atol=1e-9)
    # selecting layer 1 instead gives something else
    wc2 = np.zeros_like(wc)
    wc2[:, :d] = np.eye(d)
    W["w_c"] = wc2
    _, f1 = Oracle(TINY, W).target_forward(o.new_state(), 0, synth.prompts(TINY)[0][:12], 0)
    assert not np.allclose(f1, feats, atol=1e-3)


# ---------------------------------------------------------------------------
# Eq. 3: acceptance, bonus, commit (hand cases)
# ---------------------------------------------------------------------------


GOLDEN = Path(__file__).parent / "golden"


def _golden_lines(name):
    return [ln for ln in (GOLDEN / name).read_text().splitlines() if ln.strip() and not ln.startswith("#")]


def _accept_cases():
    cases = []
    for ln in _golden_lines("accept_eq3_hand_cases.txt"):
        block, g, a, committed = (f.split() for f in ln.split("|"))
        cases.append(([int(x) for x in block], [int(x) for x in g], int(a[0]), [int(x) for x in committed]))
    return cases


@pytest.mark.parametrize("block,g,a,committed", _accept_cases())
def test_accept_partition_hand_cases(block, g, a, committed):
    cfg, o = _micro_oracle()
    cfg = cfg.replace(block=3)
    o = Oracle(cfg, o.W)
    st = o.new_state(cap=32)
    st.seq_len[0] = 10
    got_a, got_c = o.accept_commit(st, 0, np.array(block), np.array(g))
    assert got_a == a and list(got_c) == committed
    assert st.seq_len[0] == 10 + a + 1
    assert list(st.tokens[0, 10:10 + a + 1]) == committed[:a + 1]


def test_forced_accept_overrides_and_bonus_is_prediction():
    cfg, o = _micro_oracle()
    cfg = cfg.replace(block=3)
    o = Oracle(cfg, o.W)
    st = o.new_state(cap=32)
    st.seq_len[0] = 4
    a, c = o.accept_commit(st, 0, np.array([7, 1, 2, 3]), np.array([9, 8, 4, 0]), forced=2)
    assert a == 2 and list(c) == [1, 2, 4, -1]


# ---------------------------------------------------------------------------
# Sec. 4.2 carry: shift by one, rejected-suffix positions only
# ---------------------------------------------------------------------------


@pytest.mark.parametrize("forced", [0, 3, TINY.block - 2, TINY.block - 1, TINY.block])
def test_carry_slots_hold_states_predicting_their_positions(tiny_oracle, forced):
    o = tiny_oracle
    B = TINY.block
    st = o.new_state()
    o.prefill(st, 0, synth.prompts(TINY)[0][:24])
    n = int(st.seq_len[0])
    ro = o.round(st, forced=[forced])
    a = int(ro.accept[0])
    assert a == forced
    n_new = int(st.seq_len[0])
    assert n_new == n + a + 1
    # the positions the rejected suffix y^_{a+2..B} occupied: n+a+1 .. n+B-1
    suffix_pos = list(range(n + a + 1, n + B))
    assert int(st.n_carry[0]) == len(suffix_pos)
    for j in range(1, B + 1):
        slot_pos = n_new - 1 + j  # position of next-round slot j
        if slot_pos in suffix_pos:
            # the verifier state that predicts slot_pos sits one position earlier
            row = (slot_pos - 1) - (n - 1)
            assert np.array_equal(st.carry[0, j - 1], ro.feats[0, row])
        else:
            assert j > st.n_carry[0]
    assert st.boundary[0, 0] == ro.committed[0, a]
    assert st.boundary[0, 1] == (ro.block[0, a + 1] if a < B else -1)


def test_context_after_round_equals_fresh_prefill(tiny_oracle):
    """Target KV and drafter context at positions < n-1 equal a recompute of the committed prefix."""
    o = tiny_oracle
    st = o.new_state()
    o.prefill(st, 0, synth.prompts(TINY)[0][:24])
    for r in range(3):
        o.round(st, forced=[[2, 8, 0][r]])
    n = int(st.seq_len[0])
    fresh = o.new_state()
    logits, feats = o.target_forward(fresh, 0, st.tokens[0, :n - 1], 0)
    o.ctx_append(fresh, 0, feats, 0)
    assert np.allclose(st.k[:, 0, :n - 1], fresh.k[:, 0, :n - 1], atol=1e-9)
    assert np.allclose(st.v[:, 0, :n - 1], fresh.v[:, 0, :n - 1], atol=1e-9)
    assert np.allclose(st.dk[:, 0, :n - 1], fresh.dk[:, 0, :n - 1], atol=1e-9)
    assert np.allclose(st.dv[:, 0, :n - 1], fresh.dv[:, 0, :n - 1], atol=1e-9)


# ---------------------------------------------------------------------------
# losslessness and full-block acceptance
# ---------------------------------------------------------------------------


def test_lossless_against_plain_greedy(tiny_oracle):
    o = tiny_oracle
    prompt = synth.prompts(TINY)[0]
    toks, _ = o.generate([prompt], TINY.new_tokens)
    assert np.array_equal(toks[0], o.greedy_decode(prompt, TINY.new_tokens))


def test_decode_steps_equal_plain_greedy(tiny_oracle):
    """Sec. 5.2 baseline: cached one-token steps reproduce brute-force greedy
    decoding (full recompute of every prefix); with draft_context the drafter
    context equals a fresh recompute of the committed prefix."""
    o = tiny_oracle
    prompt = synth.prompts(TINY)[0][:30]
    st = o.new_state()
    o.prefill(st, 0, prompt)
    got = [int(st.tokens[0, 30])] + [o.decode_step(st, 0, draft_context=True)[0] for _ in range(11)]
    assert got == list(o.greedy_decode(prompt, 12))
    n = int(st.seq_len[0])
    assert n == 30 + 12
    fresh = o.new_state()
    _, feats = o.target_forward(fresh, 0, st.tokens[0, :n - 1], 0)
    o.ctx_append(fresh, 0, feats, 0)
    assert np.allclose(st.dk[:, 0, :n - 1], fresh.dk[:, 0, :n - 1], atol=1e-9)
    assert np.allclose(st.k[:, 0, :n - 1], fresh.k[:, 0, :n - 1], atol=1e-9)


def test_lossless_batch_of_ragged_prompts(tiny_w):
    cfg = TINY.replace(batch=2)
    o = Oracle(cfg, tiny_w)
    prompts = [synth.prompts(TINY)[0][:40], synth.prompts(TINY)[0][7:30]]
    toks, _ = o.generate(prompts, 20)
    for b in range(2):
        assert np.array_equal(toks[b], o.greedy_decode(prompts[b], 20))


def test_full_block_acceptance_when_drafts_are_target_greedy(tiny_oracle):
    o = tiny_oracle
    prompt = synth.prompts(TINY)[0][:32]
    B = TINY.block
    truth = o.greedy_decode(prompt, 4 * (B + 1) + 1)

    def draft(b, st):
        n = int(st.seq_len[b])
        k = n - 1 - len(prompt)  # index of the anchor inside the greedy continuation
        return np.concatenate([[st.tokens[b, n - 1]], truth[k + 1:k + 1 + B]])

    rounds = []
    toks, st = o.generate([prompt], 4 * (B + 1), draft_override=draft, rounds_out=rounds)
    assert len(rounds) == 4
    for ro in rounds:
        assert ro.accept[0] == B
    assert int(st.n_carry[0]) == 0
    assert np.array_equal(toks[0], truth[:4 * (B + 1)])


# ---------------------------------------------------------------------------
# Eq. 4 / Eq. 5 relay wiring
# ---------------------------------------------------------------------------


def _carry_state(o, n_carry):
    st = o.new_state()
    o.prefill(st, 0, synth.prompts(o.cfg)[0][:24])
    rng = np.random.default_rng(5)
    st.carry[0] = rng.normal(size=st.carry[0].shape)
    st.n_carry[0] = n_carry
    st.boundary[0] = (11, 222)
    return st


def test_relay_zero_output_layer_gives_mask_embedding(tiny_w):
    W = dict(tiny_w)
    W["relay_w2"] = np.zeros_like(W["relay_w2"])
    o = Oracle(TINY, W)
    x = o.draft_inputs(_carry_state(o, 5), 0)
    assert np.allclose(x[1:], W["e_mask"][None, :].astype(np.float64), atol=0)


@pytest.mark.parametrize("src", ["bonus", "rejected", "carried"])
def test_relay_input_wiring(tiny_w, src):
    """Select one of the three MLP inputs with identity blocks and read it back."""
    W = dict(tiny_w)
    d = TINY.d
    w1 = np.zeros((d, 3 * d), np.float32)
    col = {"bonus": 0, "rejected": d, "carried": 2 * d}[src]
    w1[:, col:col + d] = np.eye(d)
    w2 = np.zeros((2 * d, d), np.float32)
    w2[d:, :] = np.eye(d)  # gamma = silu(selected input); beta = 0
    W["relay_w1"], W["relay_w2"] = w1, w2
    o = Oracle(TINY, W)
    st = _carry_state(o, 3)
    x = o.draft_inputs(st, 0)
    for j in (1, 2, 3):
        sel = {"bonus": W["embed"][11], "rejected": W["embed"][222], "carried": st.carry[0, j - 1]}[src]
        assert np.allclose(x[j], W["e_mask"] + silu(sel), atol=1e-12)
    assert np.allclose(x[4:], W["e_mask"][None, :], atol=0)


def test_relay_beta_scales_layernormed_carry(tiny_w):
    W = dict(tiny_w)
    d = TINY.d
    w1 = np.zeros((d, 3 * d), np.float32)
    w1[:, 2 * d:] = np.eye(d)
    w2 = np.zeros((2 * d, d), np.float32)
    w2[:d, :] = np.eye(d)  # beta = silu(h); gamma = 0
    W["relay_w1"], W["relay_w2"] = w1, w2
    o = Oracle(TINY, W)
    st = _carry_state(o, 2)
    x = o.draft_inputs(st, 0)
    h = st.carry[0, 0]
    ln = torch.nn.functional.layer_norm(torch.tensor(h), (d,), torch.tensor(W["ln_w"], dtype=torch.float64),
                                        torch.tensor(W["ln_b"], dtype=torch.float64), TINY.ln_eps).numpy()
    assert np.allclose(x[1], W["e_mask"] + silu(h) * ln, atol=1e-12)


def test_draft_ignores_carry_when_nothing_is_carried(tiny_oracle):
    o = tiny_oracle
    st = _carry_state(o, 0)
    blk1, l1, _ = o.draft_block(st, 0)
    st.carry[0] = np.nan
    blk2, l2, _ = o.draft_block(st, 0)
    assert np.array_equal(blk1, blk2) and np.allclose(l1, l2, atol=0)


def test_draft_block_is_bidirectional(tiny_oracle):
    o = tiny_oracle
    st = _carry_state(o, 0)
    x = o.draft_inputs(st, 0)
    _, l1, _ = o.draft_block(st, 0, x)
    x2 = x.copy()
    x2[-1] += 1.0  # perturb the last slot only
    _, l2, _ = o.draft_block(st, 0, x2)
    assert not np.allclose(l1[1], l2[1], atol=1e-9)  # an earlier slot sees it


def test_draft_reads_context_features_up_to_n_minus_2(tiny_oracle):
    o = tiny_oracle
    st = _carry_state(o, 0)
    n = int(st.seq_len[0])
    _, l1, _ = o.draft_block(st, 0)
    s2 = st.copy()
    s2.dk[:, 0, n - 2] += 0.5  # last committed context position
    _, l2, _ = o.draft_block(s2, 0)
    assert not np.allclose(l1, l2, atol=1e-9)
    s3 = st.copy()
    s3.dk[:, 0, n - 1:] = 7.0  # beyond the context: never read
    _, l3, _ = o.draft_block(s3, 0)
    assert np.allclose(l1, l3, atol=0)


# ---------------------------------------------------------------------------
# seeded generators
# ---------------------------------------------------------------------------


def test_splitmix64_published_vector():
    # the generator's i-th output is the finaliser applied to state i * gamma
    gamma = 0x9E3779B97F4A7C15
    want = [int(h, 16) for h in _golden_lines("splitmix64_seed0.txt")]
    assert len(want) == 4
    assert [synth.splitmix64((i * gamma) % 2 ** 64) for i in range(4)] == want


def test_schedules():
    u = synth.forced_schedule(synth.QWEN3_8B, 4000)
    assert u.min() == 0 and u.max() == 16 and abs(u.mean() - 8.0) < 0.3
    g = synth.forced_schedule(synth.QWEN3_8B_KV, 400)
    assert g.min() == 0 and g.max() <= 16
    assert abs((g == 0).mean() - 0.25) < 0.03
    assert abs(g.mean() - 2.9) < 0.25  # (1-p)/p = 3, slightly less after the cap
    assert np.array_equal(g, synth.forced_schedule(synth.QWEN3_8B_KV, 400))


def test_bf16_rounding_nearest_even():
    x = np.array([1.0, 1.0 + 2 ** -8, 1.0 + 3 * 2 ** -8, -2.5], np.float32)
    assert list(synth.bf16_round(x)) == [1.0, 1.0, 1.0 + 2 ** -6, -2.5]
    t = torch.tensor(x).to(torch.bfloat16).to(torch.float32).numpy()
    assert np.array_equal(synth.bf16_round(x), t)


def test_lossless_with_partially_correct_drafts(tiny_oracle):
    """Drafts equal to the greedy continuation with some positions corrupted:
    acceptance lengths vary naturally and the output is still plain greedy."""
    o = tiny_oracle
    prompt = synth.prompts(TINY)[0][:30]
    B = TINY.block
    truth = o.greedy_decode(prompt, 80)
    rng = np.random.default_rng(9)

    def draft(b, st):
        n = int(st.seq_len[b])
        k = n - 1 - len(prompt)
        d = truth[k + 1:k + 1 + B].copy()
        if len(d) < B:
            d = np.concatenate([d, np.zeros(B - len(d), np.int32)])
        bad = rng.integers(0, B + 3)
        if bad < B:
            d[bad] = (d[bad] + 1) % TINY.vocab
        return np.concatenate([[st.tokens[b, n - 1]], d])

    rounds = []
    toks, _ = o.generate([prompt], 60, draft_override=draft, rounds_out=rounds)
    assert np.array_equal(toks[0], truth[:60])
    assert len({int(r.accept[0]) for r in rounds}) >= 3
