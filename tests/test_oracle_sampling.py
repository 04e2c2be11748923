"""Pins of the oracle's T = 1 verification (speculative sampling) against what
the mathematics fixes: the tokens it commits are distributed as the target's
own samples, whatever the drafter proposes.  Chi-square tests on seeded Monte
Carlo draws (numpy's generator, independent of the round's SplitMix64 noise),
plus the two limit cases of the acceptance rule."""
import numpy as np
import pytest

import synth
from oracle import Oracle, speculative_sample

scipy_stats = pytest.importorskip("scipy.stats")

P_VALUE = 1e-4  # fixed seeds: a correct rule passes deterministically, a wrong one fails by far


def _softmax(z):
    z = np.asarray(z, np.float64)
    e = np.exp(z - z.max())
    return e / e.sum()


def _gumbel(rng, shape):
    return -np.log(-np.log(rng.random(shape)))


def _chi2_ok(counts, probs):
    n = counts.sum()
    keep = probs * n >= 5  # pool the rare cells
    obs = np.append(counts[keep], counts[~keep].sum())
    exp = np.append(probs[keep] * n, probs[~keep].sum() * n)
    if exp[-1] == 0:
        obs, exp = obs[:-1], exp[:-1]
    return scipy_stats.chisquare(obs, exp).pvalue > P_VALUE


def _trials(p_logits, q_logits, n, seed):
    """n blocks: proposals drawn from q (Gumbel-max), verified; returns the tokens at offsets 1..B+1
    (-1 where the block ended before) and the acceptance lengths."""
    rng = np.random.default_rng(seed)
    R, V = q_logits.shape
    out = np.full((n, R), -1, np.int64)
    acc = np.zeros(n, np.int64)
    for t in range(n):
        gd = _gumbel(rng, (R, V))
        block = [0] + [int(np.argmax(q_logits[i] + gd[i])) for i in range(1, R)]
        a, tok = speculative_sample(block, p_logits, q_logits, rng.random(R), _gumbel(rng, (R, V)))
        out[t, :a] = block[1:a + 1]
        out[t, a] = tok
        acc[t] = a
    return out, acc


def test_committed_tokens_follow_the_target_distribution():
    rng = np.random.default_rng(0)
    V, B = 7, 2
    p_logits = rng.normal(size=(B + 1, V)) * 1.5  # p_1, p_2, p_3 (verify rows 0..2)
    q_logits = rng.normal(size=(B + 1, V)) * 1.5  # q_1, q_2 at rows 1..2 (row 0 unused)
    toks, acc = _trials(p_logits, q_logits, 30000, 1)
    assert 0 < (acc == 0).mean() < 1 and (acc == B).any()  # both outcomes occur
    for off in range(1, B + 2):
        got = toks[:, off - 1]
        got = got[got >= 0]
        counts = np.bincount(got, minlength=V)
        assert _chi2_ok(counts, _softmax(p_logits[off - 1])), f"offset {off}"


def test_identical_drafter_accepts_every_proposal():
    rng = np.random.default_rng(2)
    V, B = 9, 3
    p_logits = rng.normal(size=(B + 1, V))
    q_logits = np.vstack([np.zeros(V), p_logits[:B]])  # q_i = p_i
    _, acc = _trials(p_logits, q_logits, 500, 3)
    assert (acc == B).all()


def test_proposals_the_target_excludes_are_rejected_and_resampled():
    rng = np.random.default_rng(4)
    V, B = 6, 2
    p_logits = rng.normal(size=(B + 1, V))
    p_logits[:, 0] = -60.0  # the target gives token 0 no mass
    q_logits = np.full((B + 1, V), -60.0)
    q_logits[:, 0] = 0.0  # the drafter always proposes token 0
    toks, acc = _trials(p_logits, q_logits, 8000, 5)
    assert (acc == 0).all()
    assert _chi2_ok(np.bincount(toks[:, 0], minlength=V), _softmax(p_logits[0]))


def _micro():
    cfg = synth.TINY.replace(d=8, n_layers=1, n_q_heads=2, n_kv_heads=1, head_dim=4, inter=8, vocab=10,
                             draft_layers=1, feat_layers=(1,), block=3, prompt_len=6, new_tokens=8)
    W = synth.weights(cfg, perturb_norms=True)
    W = {k: (v * 40.0 if v.ndim == 2 else v) for k, v in W.items()}  # spread-out distributions
    return cfg, Oracle(cfg, W)


def test_sampled_round_first_token_follows_the_target():
    """A whole T = 1 round on a hand-sized model, many noise draws from one
    state: the first committed token is distributed as the target's softmax at
    the anchor (brute-force full recompute), the drafter notwithstanding."""
    cfg, o = _micro()
    prompt = [3, 1, 4, 1, 5, 9]
    st0 = o.new_state(cap=32)
    o.prefill(st0, 0, prompt)
    n = int(st0.seq_len[0])
    p1 = _softmax(o.full_logits(list(st0.tokens[0, :n]))[-1])
    rng = np.random.default_rng(6)
    R, V = cfg.rows, cfg.vocab
    first = []
    accs = []
    for _ in range(3000):
        st = st0.copy()
        nz = {"gd": _gumbel(rng, (R, V)), "ua": rng.random(R), "gr": _gumbel(rng, (R, V))}
        ro = o.round_sampled(st, lambda b: nz)
        first.append(int(ro.committed[0, 0]))
        accs.append(int(ro.accept[0]))
        assert int(st.seq_len[0]) == n + int(ro.accept[0]) + 1
    assert len(set(accs)) >= 2
    assert _chi2_ok(np.bincount(first, minlength=V), p1)


def test_sampling_noise_is_reproducible_and_uniform():
    cfg = synth.TINY.replace(vocab=4096, block=3)
    a = synth.sampling_noise(cfg, 2, 5)
    b = synth.sampling_noise(cfg, 2, 5)
    assert all(np.array_equal(a[k], b[k]) for k in a)
    assert not np.array_equal(a["gd"][1], synth.sampling_noise(cfg, 2, 6)["gd"][1])
    u = np.exp(-np.exp(-a["gd"][1:].ravel()))  # back to the uniforms
    assert abs(u.mean() - 0.5) < 0.01 and scipy_stats.kstest(u, "uniform").pvalue > 1e-4
    assert ((a["ua"][1:] > 0) & (a["ua"][1:] < 1)).all()
    raw = synth.noise_uniform(synth.noise_key(4, 0, 0, 1, synth.NOISE_DRAFT), 1 << 16)
    assert (raw.astype(np.float32).astype(np.float64) == raw).all()  # the same value in fp32
    assert raw.min() > 0 and raw.max() < 1 and np.isfinite(-np.log(-np.log(raw.astype(np.float32)))).all()


def test_draw_rows_follow_the_documented_convention():
    """The token of offset i is drawn with gr[i - 1] (the bonus with gr[B]), the
    proposal of row i with gd[i] and its test with ua[i]: hand cases where each
    other row of draws would pick another token (no distribution test can see
    which independent row is used; the GPU kernels key their draws the same way)."""
    V, B, big = 4, 2, 50.0
    p = np.zeros((B + 1, V))
    p[:, 0] = -60.0  # the target never takes token 0
    q = np.full((B + 1, V), -60.0)
    q[:, 0] = 0.0  # the drafter always proposes token 0: rejected at offset 1
    gr = np.zeros((B + 1, V))
    gr[0, 2] = big  # offset 1's draw
    gr[1, 3] = big
    gr[2, 1] = big
    a, tok = speculative_sample([7, 0, 0], p, q, np.full(B + 1, 0.5), gr)
    assert (a, tok) == (0, 2)
    # all accepted (q = p): the bonus comes from p_{B+1} with gr[B]
    q2 = np.vstack([np.zeros(V), p[:B]])
    a, tok = speculative_sample([7, 1, 1], p, q2, np.full(B + 1, 0.5), gr)
    assert (a, tok) == (B, 1)
    # the acceptance test of row i reads ua[i]: u = 1 - 1e-9 rejects wherever p/q < 1
    p3 = np.log(np.array([[0.5, 0.5, 1e-9, 1e-9]] * (B + 1)))
    q3 = np.log(np.array([[0.9, 0.1, 1e-9, 1e-9]] * (B + 1)))
    ua = np.array([0.0, 0.1, 1 - 1e-9])  # row 1 accepts (0.1 < 0.5/0.9), row 2 rejects
    a, _ = speculative_sample([7, 0, 0], p3, q3, ua, gr)
    assert a == 1
    ua = np.array([0.0, 1 - 1e-9, 0.1])  # the other way round: row 1 rejects
    a, _ = speculative_sample([7, 0, 0], p3, q3, ua, gr)
    assert a == 0
