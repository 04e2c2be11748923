"""Parity at the real model widths of the four bf16 workloads (Qwen3 1.7B / 4B /
8B shapes, batch 1-16, contexts 512-8192), one call at a time, and invariants
of full-depth 8B rounds.

The per-call tests run the kernels in exactly the launch configuration of the
benchmark (every projection, attention and LM-head shape is per layer), on a
copy of each model with 2 target layers and 1 draft layer so that the float64
oracle finishes in seconds.  Caches are synthetic (seeded random K/V at the
workload's context lengths)."""
import numpy as np
import pytest
import torch

import synth
from oracle import Oracle
from parity_util import assert_close, to_np, token_check, upload_state

pytestmark = pytest.mark.gpu

def reduced(cfg):
    return cfg.replace(n_layers=2, draft_layers=1, feat_layers=(1, 2))


# the four bf16 workloads at 2 + 1 layers, and the headline workload with its
# five feature layers (Eq. 1 over m = 5 layers: W_c is 4096 x 20480)
FULL = [reduced(synth.QWEN3_1P7B), reduced(synth.QWEN3_4B), reduced(synth.QWEN3_8B), reduced(synth.QWEN3_8B_KV),
        synth.QWEN3_8B.replace(name="qwen3_8b_b1_m5", n_layers=5, draft_layers=1, feat_layers=(1, 2, 3, 4, 5))]


@pytest.fixture(scope="module", params=FULL, ids=lambda c: c.name)
def full(request):
    from paper_2609_06498_gb300 import Engine, build, pack_weights
    build.build()
    cfg = request.param
    W = synth.weights(cfg, perturb_norms=True)
    eng = Engine(cfg, pack_weights(cfg, W), max_batch=cfg.batch, max_ctx=cfg.max_ctx())
    o = Oracle(cfg, {k: v.astype(np.float64) for k, v in W.items()})
    lens = synth.prompt_lengths(cfg) + 1
    nc = np.array([[5, 0, 15, 9][b % 4] for b in range(cfg.batch)], np.int32)
    ost = o.state_from_synthetic(synth.synthetic_state(cfg, ctx_lens=lens, n_carry=nc))
    yield cfg, o, ost, eng
    del eng
    torch.cuda.empty_cache()


def test_full_width_round_calls(full):
    cfg, o, ost, eng = full
    R, B, bs = cfg.rows, cfg.block, cfg.batch
    st = eng.new_state(bs, page_seed=13)
    upload_state(eng, st, ost)
    ref = ost.copy()

    # draft (Eq. 2, Eq. 4-5): logits elementwise, tokens where the decision is safe
    gblk, gdl = eng.draft_block(st, logits=True)
    gblk, gdl = to_np(gblk), to_np(gdl)
    oblk = np.zeros((bs, R), np.int32)
    checked = 0
    for b in range(bs):
        oblk[b], lg, _ = o.draft_block(ref, b)
        assert gblk[b, 0] == oblk[b, 0]
        assert_close(gdl[b, 1:], lg[1:], cfg, "draft logits")
        c, _ = token_check(gblk[b], oblk[b], lg, rows=range(1, R))
        checked += c
    assert checked >= bs * (B // 2)

    # verify (Eq. 3 target side, Eq. 1) on the oracle's block
    blk_t = torch.as_tensor(oblk).cuda()
    g, feats, logits = eng.verify_block(st, blk_t, logits=True)
    gg, gf, gl = to_np(g), to_np(feats), to_np(logits)
    og = np.zeros((bs, R), np.int32)
    of = np.zeros((bs, R, cfg.d))
    for b in range(bs):
        og[b], lg, of[b] = o.verify_block(ref, b, oblk[b])
        assert_close(gl[b], lg, cfg, "verify logits")
        assert_close(gf[b], of[b], cfg, "features")
        token_check(gg[b], og[b], lg)
        n = int(ref.seq_len[b])
        k, v = st.read_cache(st.kv, b, n - 1 + R)
        assert_close(to_np(k)[:, n - 1:], ref.k[:, b, n - 1:n - 1 + R], cfg, "block K")
        assert_close(to_np(v)[:, n - 1:], ref.v[:, b, n - 1:n - 1 + R], cfg, "block V")

    # accept/commit (Eq. 3) with the workload's forced schedule: bit exact
    forced = synth.forced_schedule(cfg, 1)[0]
    acc, comm = eng.accept_commit(st, blk_t, torch.as_tensor(og).cuda(), torch.as_tensor(forced).cuda())
    oacc = np.zeros(bs, np.int32)
    ocomm = np.zeros((bs, R), np.int32)
    for b in range(bs):
        oacc[b], ocomm[b] = o.accept_commit(ref, b, oblk[b], og[b], int(forced[b]))
    assert np.array_equal(to_np(acc), oacc) and np.array_equal(to_np(comm), ocomm)
    assert np.array_equal(to_np(st.seq_len), ref.seq_len)

    # carry (Sec. 4.2) and context injection on the oracle's features
    fin = torch.as_tensor(of).to(feats.dtype).cuda()
    eng.carry_hidden(st, blk_t, fin, acc)
    fin_np = to_np(fin)
    for b in range(bs):
        o.carry_hidden(ref, b, oblk[b], fin_np[b].astype(np.float64), int(oacc[b]))
    assert np.array_equal(to_np(st.n_carry), ref.n_carry)
    assert np.array_equal(to_np(st.boundary), ref.boundary)
    gc = to_np(st.carry)
    for b in range(bs):
        nc = int(ref.n_carry[b])
        assert np.array_equal(gc[b, :nc], fin_np[b, oacc[b] + 1:oacc[b] + 1 + nc])
        n = int(ref.seq_len[b])
        dk, dv = st.read_cache(st.draft_kv, b, n - 1)
        lo = n - 2 - int(oacc[b])
        assert_close(to_np(dk)[:, lo:], ref.dk[:, b, lo:n - 1], cfg, "ctx K append")
        assert_close(to_np(dv)[:, lo:], ref.dv[:, b, lo:n - 1], cfg, "ctx V append")
    assert eng.read_status(st) == 0


@pytest.mark.parametrize("bs", [6, 9])
def test_ragged_contexts_two_split_attention(bs):
    """Batch 6 or 9 x 8 kv heads is more (kv head, sequence) units than one wave of
    4-CTA clusters holds, so both attentions run 2-CTA clusters, with contexts of
    2 to 65 pages (partial last pages) in one launch.  At batch 9 the 153 rows also
    take the one-pass GEMM (above 128 rows): k-split projections reduced by every CTA
    of a tile, the Q/K/V epilogue included."""
    from paper_2609_06498_gb300 import Engine, build, pack_weights
    build.build()
    cfg = reduced(synth.QWEN3_8B_KV).replace(name=f"kv_b{bs}_ragged", batch=bs, prompt_len=70, ctx_range=(70, 4100))
    W = synth.weights(cfg, perturb_norms=True)
    eng = Engine(cfg, pack_weights(cfg, W), max_batch=cfg.batch, max_ctx=cfg.max_ctx())
    o = Oracle(cfg, {k: v.astype(np.float64) for k, v in W.items()})
    lens = np.array([70, 4100, 1500, 130, 2900, 700, 2049, 64 * 17 + 5, 3333], np.int32)[:bs]
    nc = np.array([5, 0, 15, 9, 1, 3, 7, 12, 2], np.int32)[:bs]
    ost = o.state_from_synthetic(synth.synthetic_state(cfg, ctx_lens=lens, n_carry=nc))
    R, bs = cfg.rows, cfg.batch
    st = eng.new_state(bs, page_seed=21)
    upload_state(eng, st, ost)
    ref = ost.copy()
    gblk, gdl = eng.draft_block(st, logits=True)
    gdl = to_np(gdl)
    oblk = np.zeros((bs, R), np.int32)
    for b in range(bs):
        oblk[b], lg, _ = o.draft_block(ref, b)
        assert_close(gdl[b, 1:], lg[1:], cfg, "draft logits")
    g, feats, logits = eng.verify_block(st, torch.as_tensor(oblk).cuda(), logits=True)
    gl = to_np(logits)
    for b in range(bs):
        _, lg, _ = o.verify_block(ref, b, oblk[b])
        assert_close(gl[b], lg, cfg, "verify logits")
    assert eng.read_status(st) == 0
    del eng
    torch.cuda.empty_cache()


@pytest.mark.parametrize("name", ["qwen3_8b_b1", "qwen3_4b_b4"])
def test_full_width_rounds(name):
    """Three dflow_round calls in a row at full widths (2 + 1 layers) from a
    synthetic state, against the oracle's rounds: acceptance, commits, lengths,
    carry counts and boundaries bit exact, carried states at tolerance.  Each
    round starts from the oracle's state (resynchronised after an allowed
    near-tie flip), as in the small-model round test."""
    from oracle import top2_gap
    from paper_2609_06498_gb300 import Engine, build, pack_weights
    build.build()
    cfg = reduced(synth.CONFIGS[name])
    W = synth.weights(cfg, perturb_norms=True)
    eng = Engine(cfg, pack_weights(cfg, W), max_batch=cfg.batch, max_ctx=cfg.max_ctx())
    o = Oracle(cfg, {k: v.astype(np.float64) for k, v in W.items()})
    lens = synth.prompt_lengths(cfg) + 1
    nc = np.array([[5, 0, 15, 9][b % 4] for b in range(cfg.batch)], np.int32)
    ost = o.state_from_synthetic(synth.synthetic_state(cfg, ctx_lens=lens, n_carry=nc))
    st = eng.new_state(cfg.batch, page_seed=17)
    sched = synth.forced_schedule(cfg, 3)
    exact = compared = 0
    for r in range(3):
        upload_state(eng, st, ost)
        acc, comm = eng.round(st, torch.as_tensor(sched[r]).cuda())
        ro = o.round(ost, forced=list(sched[r]))
        assert eng.read_status(st) == 0
        ga, gc = to_np(acc), to_np(comm)
        assert np.array_equal(ga, ro.accept)  # forced
        for b in range(cfg.batch):
            if np.array_equal(gc[b], ro.committed[b]):
                exact += 1
                assert int(st.seq_len[b]) == int(ost.seq_len[b])
                assert int(st.n_carry[b]) == int(ost.n_carry[b])
                # carry slot j is verify row a + j, which depends on the draft block's
                # rows 0..a+j: compare it where every draft decision up to it is safe
                gap = top2_gap(ro.draft_logits[b])
                unsafe = [i for i in range(1, cfg.rows) if gap[i] <= 0.05]
                first_unsafe = unsafe[0] if unsafe else cfg.rows
                a = int(ro.accept[b])
                nc_b = min(int(ost.n_carry[b]), max(0, first_unsafe - a - 1))
                if nc_b:
                    compared += 1
                    assert_close(to_np(st.carry)[b, :nc_b], ost.carry[b, :nc_b], cfg, "carried states")
                assert int(to_np(st.boundary)[b, 0]) == int(ost.boundary[b, 0])
            else:
                gaps = np.concatenate([top2_gap(ro.draft_logits[b][1:]), top2_gap(ro.verify_logits[b])])
                assert gaps.min() <= 0.05, f"round {r} seq {b}: diverged without a near tie"
    assert exact >= 2 * cfg.batch and (compared >= 1 or cfg.batch == 1)


def test_full_depth_8b_round_invariants():
    """The benchmark workload itself (36 + 5 layers, prefill of 2048 tokens):
    per-round properties that hold at any size, from the calls' own outputs."""
    from paper_2609_06498_gb300 import Engine, build, random_weights
    build.build()
    cfg = synth.QWEN3_8B
    R, B = cfg.rows, cfg.block
    eng = Engine(cfg, random_weights(cfg, seed=0), max_batch=1, max_ctx=cfg.max_ctx())
    st = eng.new_state(1, page_seed=1)
    eng.prefill(st, synth.prompts(cfg))
    assert eng.read_status(st) == 0 and int(st.seq_len[0]) == cfg.prompt_len + 1
    sched = synth.forced_schedule(cfg, 4)
    for r in range(4):
        n = int(st.seq_len[0])
        blk = eng.draft_block(st)
        g, feats, _ = eng.verify_block(st, blk)
        forced = torch.as_tensor(sched[r]).cuda()
        acc, comm = eng.accept_commit(st, blk, g, forced)
        eng.carry_hidden(st, blk, feats, acc)
        bk, gk, ck = to_np(blk)[0], to_np(g)[0], to_np(comm)[0]
        a = int(acc[0])
        assert a == int(sched[r][0])
        assert bk[0] == to_np(st.tokens)[0, n - 1]  # row 0 is the anchor
        assert list(ck[:a]) == list(bk[1:a + 1]) and ck[a] == gk[a] and (ck[a + 1:] == -1).all()
        assert int(st.seq_len[0]) == n + a + 1
        assert list(to_np(st.tokens)[0, n:n + a + 1]) == list(ck[:a + 1])
        nc = max(0, B - a - 1)
        assert int(st.n_carry[0]) == nc
        assert np.array_equal(to_np(st.carry)[0, :nc], to_np(feats)[0, a + 1:a + 1 + nc])
        bd = to_np(st.boundary)[0]
        assert bd[0] == gk[a] and bd[1] == (bk[a + 1] if a < B else -1)
        assert np.isfinite(to_np(feats)).all()
    assert eng.read_status(st) == 0


def test_full_depth_8b_many_rounds_stay_clean_and_deterministic():
    """120 rounds of the benchmark workload through the round call: every
    bounded wait holds and no completion count passes its target (either sets
    the device status); the sequence grows by the forced acceptance.  A second
    engine state replaying the same rounds gives bit-identical target tokens and
    features (the split-K sums, across clusters too, have a fixed order)."""
    from paper_2609_06498_gb300 import Engine, build, random_weights
    build.build()
    cfg = synth.QWEN3_8B
    rounds = 120
    eng = Engine(cfg, random_weights(cfg, seed=0), max_batch=1,
                 max_ctx=cfg.replace(new_tokens=rounds * cfg.rows).max_ctx())
    sched = synth.forced_schedule(cfg, rounds)
    runs = []
    for _ in range(2):
        st = eng.new_state(1, page_seed=3)
        eng.prefill(st, synth.prompts(cfg))
        n0 = int(st.seq_len[0])
        toks = []
        for r in range(rounds):
            acc, comm = eng.round(st, torch.as_tensor(sched[r]).cuda())
            toks.append(to_np(comm)[0].copy())
        assert eng.read_status(st) == 0
        assert int(st.seq_len[0]) == n0 + int((sched[:, 0] + 1).sum())
        blk = eng.draft_block(st)
        g, feats, _ = eng.verify_block(st, blk)
        runs.append((np.array(toks), to_np(blk), to_np(g), to_np(feats)))
        assert eng.read_status(st) == 0
        del st
    for x, y in zip(runs[0], runs[1]):
        assert np.array_equal(x, y)


def test_batch16_long_context_rounds_stay_clean():
    """Forty rounds of the batch-16, 8K-context shape (2 + 1 layers, full widths):
    no bounded device wait may expire, and every sequence grows by exactly its
    forced acceptance + 1 per round (Eq. 3).  Exercises every pipeline barrier of
    the attention and GEMM kernels over several hundred launches."""
    from paper_2609_06498_gb300 import Engine, build, random_weights
    build.build()
    cfg = reduced(synth.QWEN3_8B_KV)
    rounds = 40
    max_ctx = cfg.replace(new_tokens=rounds * cfg.rows).max_ctx()
    eng = Engine(cfg, random_weights(cfg, seed=0), max_batch=cfg.batch, max_ctx=max_ctx)
    st = eng.new_state(cfg.batch, page_seed=0)
    eng.prefill(st, synth.prompts(cfg))
    assert eng.read_status(st) == 0
    n0 = to_np(st.seq_len).astype(np.int64)
    sched = synth.forced_schedule(cfg, rounds)
    for r in range(rounds):
        eng.round(st, torch.as_tensor(sched[r]).cuda())
    assert eng.read_status(st) == 0
    assert np.array_equal(to_np(st.seq_len).astype(np.int64), n0 + (sched + 1).sum(axis=0))


def test_full_depth_8b_decode_steps():
    """The Sec. 5.2 baseline at the benchmark's shape: 2048-token prefill, then
    64 plain decoding steps (one row through 36 layers, the LM head and its
    argmax per step).  Every step commits exactly one token, leaves nothing
    carried and sets no device status; the committed tokens are the target's
    own predictions (a verify of the same positions reproduces them where the
    decision is not a near tie)."""
    from paper_2609_06498_gb300 import Engine, build, random_weights
    build.build()
    cfg = synth.QWEN3_8B
    steps = 64
    eng = Engine(cfg, random_weights(cfg, seed=0), max_batch=1, max_ctx=cfg.replace(new_tokens=steps + 64).max_ctx())
    st = eng.new_state(1, page_seed=4)
    eng.prefill(st, synth.prompts(cfg))
    assert eng.read_status(st) == 0
    n0 = int(st.seq_len[0])
    toks = [int(eng.decode_step(st)[0]) for _ in range(steps)]
    assert eng.read_status(st) == 0
    assert int(st.seq_len[0]) == n0 + steps and int(st.n_carry[0]) == 0
    assert list(to_np(st.tokens)[0, n0:n0 + steps]) == toks
    assert all(0 <= t < cfg.vocab for t in toks)
