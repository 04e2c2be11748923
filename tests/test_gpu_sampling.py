"""GPU parity of the T = 1 round (dflow_round_sampled: Gumbel-max proposals,
speculative acceptance, residual / bonus draw) against the oracle.

Three checks per round and sequence:
  A. the kernels' decisions on the round's own logits (returned by the call):
     the oracle's rule (speculative_sample, Gumbel-max rows) applied in
     float64 to those fp32 logits with the same draws must give the same
     proposals, acceptance length and committed token wherever every decision
     on the path clears MARGIN (both sides then differ only by fp32 rounding);
  B. the logits themselves against the oracle's drafter and target forward;
  C. (fp32 model) the whole round against Oracle.round_sampled where the
     oracle's own decisions clear GAP_F32.
A holds at any size, so it also runs at the real model widths (151936-token
vocabulary) and on the full-depth 8B workload."""
import numpy as np
import pytest
import torch

import synth
from oracle import Oracle, log_softmax, speculative_sample
from parity_util import assert_close, to_np, upload_state

pytestmark = pytest.mark.gpu

MARGIN = 1e-3   # decisions on identical fp32 logits: fp32 vs fp64 evaluation of the draws
GAP_F32 = 1e-3  # fp32 model vs float64 oracle logits (max rel err 1e-4 of logits of size ~1)
SEED = 1234

SMALL_BF16 = synth.ModelConfig(
    name="small_bf16", dtype="bf16", d=512, n_layers=3, n_q_heads=8, n_kv_heads=2, head_dim=128, inter=1472,
    vocab=1000, draft_layers=2, feat_layers=(1, 2, 3), block=16, batch=3, prompt_len=150, new_tokens=48,
    schedule="uniform")


def _gap(w):
    w = w[np.isfinite(w)]
    if len(w) < 2:
        return np.inf
    t = np.partition(w, -2)[-2:]
    return float(t[1] - t[0])


def oracle_path(ql, pl, nz, B):
    """The oracle's T = 1 decisions on logits ql (drafter) and pl (target), both
    [B+1][V] float64: (block with 0 in the anchor row, a, token, smallest decision
    margin on the path)."""
    blk = [0] + [int(np.argmax(ql[i] + nz["gd"][i])) for i in range(1, B + 1)]
    a, tok = speculative_sample(blk, pl, ql, nz["ua"], nz["gr"])
    m = np.inf
    for i in range(1, min(a + 1, B) + 1):
        m = min(m, _gap(ql[i] + nz["gd"][i]))
        lp, lq = log_softmax(pl[i - 1]), log_softmax(ql[i])
        m = min(m, abs(np.log(nz["ua"][i]) - (lp[blk[i]] - lq[blk[i]])))
    if a < B:
        lp, lq = log_softmax(pl[a]), log_softmax(ql[a + 1])
        r = np.exp(lp) - np.exp(lq)
        with np.errstate(divide="ignore"):
            w = np.where(r > 0, np.log(np.where(r > 0, r, 1.0)), -np.inf)
        m = min(m, _gap(w + nz["gr"][a]))
    else:
        m = min(m, _gap(log_softmax(pl[B]) + nz["gr"][B]))
    return blk, a, tok, m


def check_own_logits(cfg, b, ql, pl, acc, comm, boundary, nz):
    """Check A for sequence b; True when every decision was safe (and compared)."""
    B = cfg.block
    blk, a, tok, m = oracle_path(ql.astype(np.float64), pl.astype(np.float64), nz, B)
    ga = int(acc[b])
    # proposals visible in the outputs: accepted ones and the first rejected one
    for i in range(1, min(ga + 1, B) + 1):
        if _gap(ql[i].astype(np.float64) + nz["gd"][i]) > MARGIN:
            got = int(comm[b, i - 1]) if i <= ga else int(boundary[b, 1])
            assert got == blk[i], f"seq {b} row {i}: proposal {got}, oracle rule {blk[i]}"
    if m <= MARGIN:
        return False
    assert ga == a, f"seq {b}: accepted {ga}, oracle rule {a}"
    assert list(comm[b, :a]) == blk[1:a + 1] and int(comm[b, a]) == tok and (comm[b, a + 1:] == -1).all()
    assert int(boundary[b, 0]) == tok and int(boundary[b, 1]) == (blk[a + 1] if a < B else -1)
    return True


@pytest.fixture(scope="module", params=[synth.TINY, SMALL_BF16], ids=lambda c: c.name)
def setup(request):
    from paper_2609_06498_gb300 import Engine, build, pack_weights
    build.build()
    cfg = request.param
    W = synth.weights(cfg, perturb_norms=True)
    eng = Engine(cfg, pack_weights(cfg, W), max_batch=cfg.batch, max_ctx=cfg.max_ctx())
    return cfg, Oracle(cfg, W), eng


def _start_state(cfg, o):
    ps = synth.prompts(cfg)
    st = o.new_state()
    for b in range(cfg.batch):
        o.prefill(st, b, ps[b][:cfg.prompt_len - 13 * b])
    for r in range(2):  # forced greedy rounds: carry and context populated
        o.round(st, forced=[synth.forced_accept(cfg.replace(schedule="uniform"), b, r) % (cfg.block - 1)
                            for b in range(cfg.batch)])
    return st


@pytest.mark.parametrize("relay", [True, False], ids=["dflow", "relay_off"])
def test_sampled_round_parity(setup, relay):
    cfg, o, eng = setup
    R, B, V, bs = cfg.rows, cfg.block, cfg.vocab, cfg.batch
    ost = _start_state(cfg, o)
    st = eng.new_state(bs, page_seed=5)
    QL = torch.zeros(bs, R, V, device="cuda")
    PL = torch.zeros(bs, R, V, device="cuda")
    safe = e2e = 0
    for r in range(4):
        upload_state(eng, st, ost)
        ref = ost.copy()
        if not relay:
            ref.n_carry[:] = 0  # the DFlash drafter sees mask embeddings only
        n0 = to_np(st.seq_len).copy()
        acc, comm = eng.round_sampled(st, SEED, r, relay=relay, logits=(QL, PL))
        assert eng.read_status(st) == 0
        ga, gc, gb = to_np(acc), to_np(comm), to_np(st.boundary)
        ql, pl = to_np(QL), to_np(PL)
        noise = [synth.sampling_noise(cfg, b, r, SEED) for b in range(bs)]
        for b in range(bs):
            a = int(ga[b])
            # invariants of any commit
            assert 0 <= a <= B and int(st.seq_len[b]) == n0[b] + a + 1
            assert list(to_np(st.tokens)[b, n0[b]:n0[b] + a + 1]) == list(gc[b, :a + 1])
            assert int(st.n_carry[b]) == (max(0, B - a - 1) if relay else 0)
            safe += check_own_logits(cfg, b, ql[b], pl[b], ga, gc, gb, noise[b])
            # B: the round's logits against the oracle's forward passes
            _, dl, _ = o.draft_block(ref, b)
            assert_close(ql[b, 1:], dl[1:], cfg, "sampled-round drafter logits")
            blk, _, _, _ = oracle_path(ql[b].astype(np.float64), pl[b].astype(np.float64), noise[b], B)
            blk[0] = int(ref.tokens[b, int(ref.seq_len[b]) - 1])  # the anchor
            if min(_gap(ql[b, i].astype(np.float64) + noise[b]["gd"][i]) for i in range(1, R)) > MARGIN:
                _, vl, _ = o.verify_block(ref, b, np.asarray(blk, np.int32))
                assert_close(pl[b], vl, cfg, "sampled-round target logits")
        # C: the oracle's own sampled round
        ro = o.round_sampled(ost, lambda b: noise[b], relay=relay)
        if cfg.dtype == "f32":
            for b in range(bs):
                _, _, _, m = oracle_path(ro.draft_logits[b], ro.verify_logits[b], noise[b], B)
                if m > GAP_F32:
                    assert int(ga[b]) == int(ro.accept[b]) and np.array_equal(gc[b], ro.committed[b])
                    e2e += 1
    assert safe >= 4 * bs // 2, f"only {safe} sequence-rounds with every decision clear of {MARGIN}"
    if cfg.dtype == "f32":
        assert e2e >= 4 * bs // 2


def test_sampled_round_is_deterministic_and_seeded(setup):
    """Same seed and round index: identical commits; another round index: other draws."""
    cfg, o, eng = setup
    ost = _start_state(cfg, o)
    outs = []
    for rnd in (7, 7, 8):
        st = eng.new_state(cfg.batch, page_seed=2)
        upload_state(eng, st, ost)
        acc, comm = eng.round_sampled(st, SEED, rnd)
        assert eng.read_status(st) == 0
        outs.append((to_np(acc).copy(), to_np(comm).copy()))
    assert np.array_equal(outs[0][0], outs[1][0]) and np.array_equal(outs[0][1], outs[1][1])
    assert not np.array_equal(outs[0][1], outs[2][1])


def test_sampled_round_leaves_inactive_sequences_untouched(setup):
    """A frozen sequence (active = 0) keeps its tokens, length, carry and boundary
    and reports accept_len -1; the others still follow the oracle's rule."""
    cfg, o, eng = setup
    if cfg.batch < 2:
        pytest.skip("needs two sequences")
    R, V, bs = cfg.rows, cfg.vocab, cfg.batch
    ost = _start_state(cfg, o)
    ost.active[1] = False
    st = eng.new_state(bs, page_seed=4)
    upload_state(eng, st, ost)
    before = {k: to_np(getattr(st, k)).copy() for k in ("tokens", "seq_len", "n_carry", "boundary")}
    carry0 = to_np(st.carry)[1].copy()
    QL = torch.zeros(bs, R, V, device="cuda")
    PL = torch.zeros(bs, R, V, device="cuda")
    acc, comm = eng.round_sampled(st, SEED, 2, logits=(QL, PL))
    assert eng.read_status(st) == 0
    ga, gc, gb = to_np(acc), to_np(comm), to_np(st.boundary)
    assert ga[1] == -1 and (gc[1] == -1).all()
    for k, v in before.items():
        assert np.array_equal(to_np(getattr(st, k))[1], v[1]), k
    assert np.array_equal(to_np(st.carry)[1], carry0)
    ql, pl = to_np(QL), to_np(PL)
    for b in (0, 2):
        if b < bs:
            check_own_logits(cfg, b, ql[b], pl[b], ga, gc, gb, synth.sampling_noise(cfg, b, 2, SEED))


def test_sampled_round_rejects_bad_round_index(setup):
    from paper_2609_06498_gb300._abi import DFlowError
    cfg, o, eng = setup
    st = eng.new_state(cfg.batch, page_seed=2)
    with pytest.raises(DFlowError):
        eng.round_sampled(st, SEED, 1 << 24)


# ---------------------------------------------------------------------------
# real model widths (151936-token vocabulary) and the full-depth 8B workload
# ---------------------------------------------------------------------------

def _reduced(cfg):
    return cfg.replace(n_layers=2, draft_layers=1, feat_layers=(1, 2))


@pytest.mark.parametrize("cfg", [_reduced(synth.QWEN3_8B), _reduced(synth.QWEN3_8B_KV)], ids=lambda c: c.name)
def test_sampled_round_full_width(cfg):
    from paper_2609_06498_gb300 import Engine, build, pack_weights
    build.build()
    W = synth.weights(cfg, perturb_norms=True)
    eng = Engine(cfg, pack_weights(cfg, W), max_batch=cfg.batch, max_ctx=cfg.max_ctx())
    o = Oracle(cfg, {k: v.astype(np.float64) for k, v in W.items()})
    lens = synth.prompt_lengths(cfg) + 1
    nc = np.array([[5, 0, 15, 9][b % 4] for b in range(cfg.batch)], np.int32)
    ost = o.state_from_synthetic(synth.synthetic_state(cfg, ctx_lens=lens, n_carry=nc))
    R, V, bs = cfg.rows, cfg.vocab, cfg.batch
    st = eng.new_state(bs, page_seed=13)
    upload_state(eng, st, ost)
    QL = torch.zeros(bs, R, V, device="cuda")
    PL = torch.zeros(bs, R, V, device="cuda")
    acc, comm = eng.round_sampled(st, SEED, 3, logits=(QL, PL))
    assert eng.read_status(st) == 0
    ga, gc, gb = to_np(acc), to_np(comm), to_np(st.boundary)
    ql, pl = to_np(QL), to_np(PL)
    safe = 0
    for b in range(bs):
        nz = synth.sampling_noise(cfg, b, 3, SEED)
        safe += check_own_logits(cfg, b, ql[b], pl[b], ga, gc, gb, nz)
        if b < 2:  # the oracle's drafter forward at full width (a few seconds per sequence)
            _, dl, _ = o.draft_block(ost, b)
            assert_close(ql[b, 1:], dl[1:], cfg, "drafter logits")
    assert safe >= max(1, bs // 2)
    del eng
    torch.cuda.empty_cache()


def test_full_depth_8b_sampled_rounds():
    """The benchmark workload (36 + 5 layers, 2048-token prompt) at T = 1: the
    kernels' decisions on the rounds' own logits, and the commit invariants."""
    from paper_2609_06498_gb300 import Engine, build, random_weights
    build.build()
    cfg = synth.QWEN3_8B
    R, B, V = cfg.rows, cfg.block, cfg.vocab
    eng = Engine(cfg, random_weights(cfg, seed=0), max_batch=1, max_ctx=cfg.max_ctx())
    st = eng.new_state(1, page_seed=1)
    eng.prefill(st, synth.prompts(cfg))
    QL = torch.zeros(1, R, V, device="cuda")
    PL = torch.zeros(1, R, V, device="cuda")
    safe = 0
    for r in range(4):
        n = int(st.seq_len[0])
        acc, comm = eng.round_sampled(st, SEED, r, logits=(QL, PL))
        assert eng.read_status(st) == 0
        ga, gc, gb = to_np(acc), to_np(comm), to_np(st.boundary)
        a = int(ga[0])
        assert int(st.seq_len[0]) == n + a + 1 and int(st.n_carry[0]) == max(0, B - a - 1)
        assert list(to_np(st.tokens)[0, n:n + a + 1]) == list(gc[0, :a + 1])
        ql, pl = to_np(QL)[0], to_np(PL)[0]
        assert np.isfinite(ql).all() and np.isfinite(pl).all()
        safe += check_own_logits(cfg, 0, ql, pl, ga, gc, gb, synth.sampling_noise(cfg, 0, r, SEED))
    assert safe >= 2
