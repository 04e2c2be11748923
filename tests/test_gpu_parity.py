"""GPU parity: every entry point of the C ABI against the oracle on the same
seeded inputs.  Integer outputs (acceptance, commits, carry counts, boundary
tokens) are compared bit for bit; floating-point outputs within 1e-4 (fp32) or
2e-2 (bf16) max relative error; tokens wherever the oracle's top-1/top-2 gap
exceeds 0.05."""
import numpy as np
import pytest
import torch

import synth
from oracle import Oracle
from parity_util import GAP, assert_close, to_np, token_check, upload_state

pytestmark = pytest.mark.gpu

# A bf16 model small enough for the oracle yet spanning several tiles of every
# kernel, with ragged tails: vocab 1000 (not a multiple of 128), 23 SwiGLU
# groups of 64, contexts over several 64-token pages, a batch of 3.
SMALL_BF16 = synth.ModelConfig(
    name="small_bf16", dtype="bf16", d=512, n_layers=3, n_q_heads=8, n_kv_heads=2, head_dim=128, inter=1472,
    vocab=1000, draft_layers=2, feat_layers=(1, 2, 3), block=16, batch=3, prompt_len=150, new_tokens=48,
    schedule="uniform")

CONFIGS = [synth.TINY, SMALL_BF16]


@pytest.fixture(scope="module", params=CONFIGS, ids=lambda c: c.name)
def setup(request):
    from paper_2609_06498_gb300 import Engine, build, pack_weights
    build.build()
    cfg = request.param
    W = synth.weights(cfg, perturb_norms=True)
    eng = Engine(cfg, pack_weights(cfg, W), max_batch=cfg.batch, max_ctx=cfg.max_ctx())
    return cfg, W, Oracle(cfg, W), eng


def oracle_after_prefill(cfg, o, lens, logits_out=None):
    ps = synth.prompts(cfg)
    st = o.new_state()
    for b in range(cfg.batch):
        lg = o.prefill(st, b, ps[b][:lens[b]])
        if logits_out is not None:
            logits_out.append(lg)
    return st, [ps[b][:lens[b]] for b in range(cfg.batch)]


def prompt_lens(cfg):
    return [cfg.prompt_len - 13 * b for b in range(cfg.batch)]


def test_prefill(setup):
    cfg, W, o, eng = setup
    lens = prompt_lens(cfg)
    logits = []
    ost, prompts = oracle_after_prefill(cfg, o, lens, logits)
    st = eng.new_state(cfg.batch, page_seed=7)
    eng.prefill(st, prompts)
    assert eng.read_status(st) == 0
    assert np.array_equal(to_np(st.seq_len), ost.seq_len)
    for b in range(cfg.batch):
        n = int(ost.seq_len[b])
        assert np.array_equal(to_np(st.tokens)[b, :n - 1], ost.tokens[b, :n - 1])
        token_check([to_np(st.tokens)[b, n - 1]], [ost.tokens[b, n - 1]], logits[b][-1:])
        k, v = st.read_cache(st.kv, b, n - 1)
        assert_close(to_np(k), ost.k[:, b, :n - 1], cfg, "prefill K")
        assert_close(to_np(v), ost.v[:, b, :n - 1], cfg, "prefill V")
        dk, dv = st.read_cache(st.draft_kv, b, n - 1)
        assert_close(to_np(dk), ost.dk[:, b, :n - 1], cfg, "prefill ctx K")
        assert_close(to_np(dv), ost.dv[:, b, :n - 1], cfg, "prefill ctx V")


def _oracle_round_state(cfg, o):
    """Oracle state after prefill and two forced rounds, so carry and context are populated."""
    ost, _ = oracle_after_prefill(cfg, o, prompt_lens(cfg))
    for r in range(2):
        o.round(ost, forced=[synth.forced_accept(cfg.replace(schedule="uniform"), b, r) % (cfg.block - 1)
                             for b in range(cfg.batch)])
    return ost


def test_per_call_parity(setup):
    """draft -> verify -> accept -> carry, each call fed the oracle's inputs."""
    cfg, W, o, eng = setup
    ost = _oracle_round_state(cfg, o)
    assert ost.n_carry.max() > 0
    st = eng.new_state(cfg.batch, page_seed=3)
    upload_state(eng, st, ost)
    ref = ost.copy()
    R, B = cfg.rows, cfg.block

    # dflow_draft_block (Eq. 2, Eq. 4-5): drafter logits elementwise, tokens where safe
    blk, dlogits = eng.draft_block(st, logits=True)
    gblk, gdl = to_np(blk), to_np(dlogits)
    oblk = np.zeros((cfg.batch, R), np.int32)
    checked = 0
    for b in range(cfg.batch):
        oblk[b], lg, _ = o.draft_block(ref, b)
        assert gblk[b, 0] == oblk[b, 0]
        assert_close(gdl[b, 1:], lg[1:], cfg, "draft logits")
        c, _ = token_check(gblk[b], oblk[b], lg, rows=range(1, R))
        checked += c
    assert checked >= cfg.batch * (R - 1) // 4

    # dflow_verify_block (Eq. 3 target side, Eq. 1) on the oracle's block
    blk_t = torch.as_tensor(oblk).cuda()
    g, feats, logits = eng.verify_block(st, blk_t, logits=True)
    gg, gf, gl = to_np(g), to_np(feats), to_np(logits)
    og = np.zeros((cfg.batch, R), np.int32)
    ofeats = np.zeros((cfg.batch, R, cfg.d))
    for b in range(cfg.batch):
        og[b], lg, ofeats[b] = o.verify_block(ref, b, oblk[b])
        assert_close(gl[b], lg, cfg, "verify logits")
        assert_close(gf[b], ofeats[b], cfg, "features")
        token_check(gg[b], og[b], lg)
        n = int(ref.seq_len[b])
        k, v = st.read_cache(st.kv, b, n - 1 + R)
        assert_close(to_np(k)[:, n - 1:], ref.k[:, b, n - 1:n - 1 + R], cfg, "block K")
        assert_close(to_np(v)[:, n - 1:], ref.v[:, b, n - 1:n - 1 + R], cfg, "block V")

    # dflow_accept_commit (Eq. 3) on the oracle's block and predictions: bit exact
    forced = np.array([[0, B, B - 1, 5][b % 4] for b in range(cfg.batch)], np.int32)
    acc, comm = eng.accept_commit(st, blk_t, torch.as_tensor(og).cuda(), torch.as_tensor(forced).cuda())
    oacc = np.zeros(cfg.batch, np.int32)
    ocomm = np.zeros((cfg.batch, R), np.int32)
    for b in range(cfg.batch):
        oacc[b], ocomm[b] = o.accept_commit(ref, b, oblk[b], og[b], int(forced[b]))
    assert np.array_equal(to_np(acc), oacc)
    assert np.array_equal(to_np(comm), ocomm)
    assert np.array_equal(to_np(st.seq_len), ref.seq_len)
    assert np.array_equal(to_np(st.tokens)[:, :ref.tokens.shape[1]], ref.tokens[:, :st.max_ctx])

    # natural acceptance on the same inputs (no forcing) against Eq. 3 directly
    st2 = eng.new_state(cfg.batch, page_seed=3)
    upload_state(eng, st2, ost)
    acc2, _ = eng.accept_commit(st2, blk_t, torch.as_tensor(og).cuda())
    for b in range(cfg.batch):
        a = 0
        while a < B and oblk[b, a + 1] == og[b, a]:
            a += 1
        assert int(acc2[b]) == a

    # dflow_carry_hidden on the oracle's features (in the model dtype)
    fin = torch.as_tensor(ofeats).to(feats.dtype).cuda()
    eng.carry_hidden(st, blk_t, fin, acc)
    fin_np = to_np(fin)
    for b in range(cfg.batch):
        o.carry_hidden(ref, b, oblk[b], fin_np[b].astype(np.float64), int(oacc[b]))
    assert np.array_equal(to_np(st.n_carry), ref.n_carry)
    assert np.array_equal(to_np(st.boundary), ref.boundary)
    gcarry = to_np(st.carry)
    for b in range(cfg.batch):
        nc = int(ref.n_carry[b])
        # the carry is a copy of the feature rows a+1..B-1: bit exact
        assert np.array_equal(gcarry[b, :nc], fin_np[b, oacc[b] + 1:oacc[b] + 1 + nc])
        n = int(ref.seq_len[b])
        dk, dv = st.read_cache(st.draft_kv, b, n - 1)
        lo = n - 2 - int(oacc[b])
        assert_close(to_np(dk)[:, lo:], ref.dk[:, b, lo:n - 1], cfg, "ctx K append")
        assert_close(to_np(dv)[:, lo:], ref.dv[:, b, lo:n - 1], cfg, "ctx V append")
    assert eng.read_status(st) == 0


@pytest.mark.parametrize("relay", [True, False], ids=["dflow", "relay_off"])
def test_round_parity(setup, relay):
    """dflow_round from the oracle's state, several rounds, resynchronised from
    the oracle whenever an allowed near-tie flip makes the two diverge.  relay
    off is the DFlash baseline of Sec. 5.3 (mask embeddings only, nothing
    carried: Eq. 5 with no valid slot)."""
    cfg, W, o, eng = setup
    ost = _oracle_round_state(cfg, o)
    st = eng.new_state(cfg.batch, page_seed=11)
    sched = synth.forced_schedule(cfg.replace(schedule="uniform"), 6)
    exact_rounds = 0
    for r in range(6):
        upload_state(eng, st, ost)
        forced = sched[r] if cfg.schedule != "natural" else None
        acc, comm = eng.round(st, torch.as_tensor(forced).cuda() if forced is not None else None, relay=relay)
        ro = o.round(ost, forced=None if forced is None else list(forced), relay=relay)
        assert eng.read_status(st) == 0
        ga, gc = to_np(acc), to_np(comm)
        for b in range(cfg.batch):
            if ga[b] == ro.accept[b] and np.array_equal(gc[b], ro.committed[b]):
                exact_rounds += 1
                assert int(st.seq_len[b]) == int(ost.seq_len[b])
                assert int(st.n_carry[b]) == int(ost.n_carry[b])
                if not relay:
                    assert int(st.n_carry[b]) == 0
                gb = to_np(st.boundary)[b]
                assert gb[0] == ost.boundary[b, 0]
                a = int(ro.accept[b])
                if a < cfg.block and gb[1] != ost.boundary[b, 1]:
                    # the first rejected proposal is a drafter token: identity only where its decision is safe
                    from oracle import top2_gap
                    gap = top2_gap(ro.draft_logits[b][a + 1:a + 2])[0]
                    assert gap <= GAP, f"round {r} seq {b}: draft token {a + 1} differs at gap {gap:.3f}"
                else:
                    assert gb[1] == ost.boundary[b, 1]
            else:
                # a divergence must come from a near tie in the oracle's own logits
                from oracle import top2_gap
                gaps = np.concatenate([top2_gap(ro.draft_logits[b][1:]), top2_gap(ro.verify_logits[b])])
                assert gaps.min() <= GAP, f"round {r} seq {b}: diverged without a near tie"
    assert exact_rounds >= cfg.batch * 4


def test_round_parity_separate_gemms(setup, monkeypatch):
    """The same rounds with one launch per projection instead of the persistent
    per-layer launch the bf16 path with 128-dim heads and few rows takes."""
    cfg = setup[0]
    if cfg.dtype != "bf16" or cfg.head_dim != 128:
        pytest.skip("the persistent GEMM sequence is the bf16 path with 128-dim heads")
    monkeypatch.setenv("DFLOW_SEPARATE_GEMMS", "1")
    test_round_parity(setup, True)


def test_round_parity_fused_attention(setup, monkeypatch):
    """The same rounds with the attention as the first phase of each layer's
    persistent launch instead of its own launch."""
    cfg = setup[0]
    if cfg.dtype != "bf16" or cfg.head_dim != 128:
        pytest.skip("the fused attention phase is the bf16 path with 128-dim heads")
    monkeypatch.setenv("DFLOW_FUSED_ATTENTION", "1")
    test_round_parity(setup, True)


def test_generate_matches_oracle_tiny():
    """fp32: the whole generation (prefill + natural-acceptance rounds) equals the
    oracle's, which the oracle tests pin to plain greedy decoding."""
    from paper_2609_06498_gb300 import Engine, build, pack_weights
    build.build()
    cfg = synth.TINY
    W = synth.weights(cfg)
    o = Oracle(cfg, W)
    prompt = synth.prompts(cfg)[0]
    want, _ = o.generate([prompt], cfg.new_tokens)
    eng = Engine(cfg, pack_weights(cfg, W), max_batch=1, max_ctx=cfg.max_ctx())
    st = eng.new_state(1)
    got = eng.generate(st, [prompt], cfg.new_tokens)
    assert eng.read_status(st) == 0
    assert np.array_equal(got[0], want[0])


def test_device_errors_are_reported(setup):
    cfg, W, o, eng = setup
    st = eng.new_state(cfg.batch)
    # capacity: a sequence at max_ctx cannot take another block
    st.seq_len.fill_(st.max_ctx - 2)
    eng.round(st, None)
    assert eng.read_status(st) == 3
    # bad carried count
    st2 = eng.new_state(cfg.batch)
    st2.seq_len.fill_(5)
    st2.n_carry.fill_(cfg.block)
    eng.draft_block(st2)
    assert eng.read_status(st2) == 6
    # the same checks open the T = 1 round and the verify call
    st3 = eng.new_state(cfg.batch)
    st3.seq_len.fill_(st3.max_ctx - 2)
    eng.round_sampled(st3, 1, 0)
    assert eng.read_status(st3) == 3
    st4 = eng.new_state(cfg.batch)
    st4.seq_len.fill_(5)
    st4.tokens[:, 4] = cfg.vocab  # the anchor is not a token
    blk = torch.zeros(cfg.batch, cfg.rows, dtype=torch.int32, device="cuda")
    eng.verify_block(st4, blk)
    assert eng.read_status(st4) == 6


@pytest.mark.parametrize("ctx", [[3905, 4100, 2001], [64 * 41 + 1, 64 * 60, 130]])
def test_long_context_per_call(ctx):
    """Draft and verify at contexts long enough that a key split holds several
    64-token pages (and, in the drafter, the block's own keys on top), from a
    synthetic random cache."""
    from paper_2609_06498_gb300 import Engine, build, pack_weights
    build.build()
    cfg = SMALL_BF16.replace(n_layers=2, draft_layers=1, feat_layers=(1, 2), prompt_len=4200)
    W = synth.weights(cfg, perturb_norms=True)
    o = Oracle(cfg, W)
    ost = o.state_from_synthetic(synth.synthetic_state(cfg, ctx_lens=np.array(ctx), n_carry=np.array([3, 0, 15])))
    eng = Engine(cfg, pack_weights(cfg, W), max_batch=cfg.batch, max_ctx=cfg.max_ctx())
    st = eng.new_state(cfg.batch, page_seed=5)
    upload_state(eng, st, ost)
    blk, dl = eng.draft_block(st, logits=True)
    blk, dl = to_np(blk), to_np(dl)
    for b in range(cfg.batch):
        oblk, lg, _ = o.draft_block(ost, b)
        assert_close(dl[b, 1:], lg[1:], cfg, "draft logits")
        token_check(blk[b], oblk, lg, rows=range(1, cfg.rows))
    oblk = synth.block_tokens(cfg, ost.tokens[np.arange(cfg.batch), ost.seq_len - 1])
    g, feats, logits = eng.verify_block(st, torch.as_tensor(oblk).cuda(), logits=True)
    for b in range(cfg.batch):
        og, lg, of = o.verify_block(ost, b, oblk[b])
        assert_close(to_np(logits)[b], lg, cfg, "verify logits")
        assert_close(to_np(feats)[b], of, cfg, "features")
        token_check(to_np(g)[b], og, lg)
    assert eng.read_status(st) == 0


def test_decode_steps_tiny_equal_plain_greedy():
    """Sec. 5.2 baseline on the fp32 model: prefill + 24 plain decoding steps
    through dflow_decode_step give the target's greedy continuation."""
    from paper_2609_06498_gb300 import Engine, build, pack_weights
    build.build()
    cfg = synth.TINY
    W = synth.weights(cfg)
    o = Oracle(cfg, W)
    prompt = synth.prompts(cfg)[0][:40]
    want = o.greedy_decode(prompt, 25)
    eng = Engine(cfg, pack_weights(cfg, W), max_batch=1, max_ctx=cfg.max_ctx())
    st = eng.new_state(1)
    eng.prefill(st, [prompt])
    got = [int(st.tokens[0, 40])] + [int(eng.decode_step(st)[0]) for _ in range(24)]
    assert eng.read_status(st) == 0
    assert got == list(want)
    assert int(st.seq_len[0]) == 40 + 25 and int(st.n_carry[0]) == 0


def test_decode_step_parity(setup):
    """dflow_decode_step against Oracle.decode_step from the oracle's state:
    committed tokens bit exact where the decision is safe, the new K/V rows and
    (draft_context = 1) the drafter context rows within tolerance."""
    cfg, W, o, eng = setup
    ost = _oracle_round_state(cfg, o)
    st = eng.new_state(cfg.batch, page_seed=9)
    for step in range(3):
        upload_state(eng, st, ost)
        n0 = ost.seq_len.copy()
        tok = to_np(eng.decode_step(st, draft_context=True))
        assert eng.read_status(st) == 0
        for b in range(cfg.batch):
            want, lg = o.decode_step(ost, b, draft_context=True)
            token_check([tok[b]], [want], lg[None])
            n = int(n0[b])
            assert int(st.seq_len[b]) == n + 1 and int(st.n_carry[b]) == 0
            k, v = st.read_cache(st.kv, b, n)
            assert_close(to_np(k)[:, n - 1], ost.k[:, b, n - 1], cfg, "decode K")
            assert_close(to_np(v)[:, n - 1], ost.v[:, b, n - 1], cfg, "decode V")
            dk, dv = st.read_cache(st.draft_kv, b, n)
            assert_close(to_np(dk)[:, n - 1], ost.dk[:, b, n - 1], cfg, "decode ctx K")
            assert_close(to_np(dv)[:, n - 1], ost.dv[:, b, n - 1], cfg, "decode ctx V")
            # continue from the oracle's token, whatever a near tie did on the GPU
            ost.tokens[b, n] = want
