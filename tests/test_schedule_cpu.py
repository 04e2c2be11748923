"""The persistent tcgen05 launch's work split, checked on the host for every
projection shape of the workloads, every row count it takes (1..128) and a
range of cluster counts.

The schedule comes from the library itself (dflow_debug_seq_schedule, the
functions the kernel evaluates); the checks here re-derive, from the launch's
rules, what each CTA streams and receives:

  * every (tile, k-block) unit of the GEMM is streamed exactly once, and every
    CTA's k-range of a tile is non-empty (an empty range would leave its
    accumulator unwritten);
  * the four CTAs of a cluster take the same tiles in the same order (the
    split-K exchange pairs them tile by tile);
  * the bytes a CTA's receive barrier expects per tile equal what its three
    peers push to it (a float4 per row and 4-column group it owns, for columns
    below M);
  * a tile split over several clusters is counted exactly once per column
    owner, and its part slots stay inside the reserved area.
"""
import ctypes

import numpy as np
import pytest

import synth

SEQ_P, BM, BK = 4, 128, 64


@pytest.fixture(scope="module")
def lib():
    from paper_2609_06498_gb300 import _abi, build
    build.build()
    return _abi.lib()


def schedule(lib, N, K, M, Q):
    plan = (ctypes.c_int32 * 8)()
    ctas = (ctypes.c_int32 * (Q * SEQ_P * 10))()
    code = lib.dflow_debug_seq_schedule(N, K, M, Q, plan, ctas)
    if code != 0:
        return code, None, None
    return 0, list(plan), np.frombuffer(ctas, dtype=np.int32).reshape(Q * SEQ_P, 10).copy()


def model_shapes(cfg):
    d, hq, hkv, hd, I, m = cfg.d, cfg.n_q_heads, cfg.n_kv_heads, cfg.head_dim, cfg.inter, cfg.n_feat
    return {"qkv": ((hq + 2 * hkv) * hd, d), "o": (d, hq * hd), "gate_up": (2 * I, d), "down": (d, I),
            "w_c": (d, m * d), "relay1": (d, 3 * d), "relay2": (2 * d, d), "ctx_kv": (2 * hkv * hd, d)}


SHAPES = sorted({s for c in (synth.QWEN3_1P7B, synth.QWEN3_4B, synth.QWEN3_8B) for s in model_shapes(c).values()}
                | {(1000, 512), (2944, 512), (512, 512), (1536, 512), (512, 1472), (4096, 2 * 4096)})
ROWS = [1, 2, 3, 5, 16, 17, 31, 32, 33, 48, 51, 64, 65, 68, 80, 96, 100, 112, 128]
CLUSTERS = [36, 38, 37, 32, 28, 24, 16]


def check(N, K, M, Q, plan, ctas):
    npad, T, kb, Tf, Tl, ls, done_n, slots = plan
    assert npad % 16 == 0 and M <= npad <= 128 and npad - M < 16 + (16 if npad == 128 else 0)
    assert T == -(-N // BM) and kb == K // BK and Tf + Tl == T and done_n == SEQ_P * T
    if Tl:
        assert 32 <= npad <= 64, "leftover split: 32 to 64 columns (one epilogue chunk per owner)"
        assert Tl * ls == Q and Tl == T % Q
    w4 = npad // SEQ_P
    cover = np.zeros((T, kb), np.int32)
    counted = np.zeros((T, SEQ_P), np.int32)
    for q in range(Q):
        rows = ctas[q * SEQ_P:(q + 1) * SEQ_P]
        # the cluster's ranks agree on tiles and leftover assignment
        for col in (0, 1, 2, 5, 8):
            assert len(set(rows[:, col])) == 1, (q, col, rows)
        nt, t0, dt, lt, part = rows[0, 0], rows[0, 1], rows[0, 2], rows[0, 5], rows[0, 8]
        tiles = [t0 + i * dt for i in range(nt)]
        assert all(0 <= t < Tf for t in tiles)
        for rr in range(SEQ_P):
            k0, k1, lk0, lk1, recv = rows[rr, 3], rows[rr, 4], rows[rr, 6], rows[rr, 7], rows[rr, 9]
            # what the three peers push to this owner per tile
            owned = [c for c in range(0, M, 4) if c // w4 == rr]
            assert recv == (SEQ_P - 1) * BM * 16 * len(owned), (rr, recv, owned)
            has_cols = min(rr * w4, M) < min((rr + 1) * w4, M)
            if tiles:
                assert 0 <= k0 < k1 <= kb
            for t in tiles:
                cover[t, k0:k1] += 1
                counted[t, rr] += 1
            if lt >= 0:
                assert 0 <= lt < Tl and 0 <= part < ls
                assert 0 <= lk0 < lk1 <= kb, "every part of a leftover tile keeps a k-block"
                cover[Tf + lt, lk0:lk1] += 1
                assert lt * ls + part < slots and lt * SEQ_P + rr < slots * SEQ_P
                # an owner with columns counts the tile when its count completes (once);
                # one without columns counts it through the tile's first part
                if not has_cols and part == 0:
                    counted[Tf + lt, rr] += 1
            else:
                assert q >= Tl * ls
        if lt >= 0:
            for rr in range(SEQ_P):
                has_cols = min(rr * w4, M) < min((rr + 1) * w4, M)
                if has_cols and part == ls - 1:
                    counted[Tf + lt, rr] += 1  # exactly one part completes the count of ls arrivals
    assert (cover == 1).all(), "every (tile, k-block) unit streamed exactly once"
    assert (counted == 1).all(), "every tile counted once per column owner"
    assert counted.sum() == done_n


@pytest.mark.parametrize("N,K", SHAPES)
def test_persistent_schedule_covers_every_unit_once(lib, N, K):
    n = 0
    for M in ROWS:
        for Q in CLUSTERS:
            code, plan, ctas = schedule(lib, N, K, M, Q)
            if code == 5:
                assert K // BK < SEQ_P
                continue
            assert code == 0
            check(N, K, M, Q, plan, ctas)
            n += 1
    assert n > 0


def test_schedule_leftover_split_at_the_headline_shapes(lib):
    # Qwen3-8B gate/up (192 tiles) and QKV (48 tiles) on 36 clusters: 12 leftover
    # tiles each, split over 3 clusters (12 parts of the K range), from 32 columns
    for N in (24576, 6144):
        code, plan, ctas = schedule(lib, N, 4096, 17, 36)
        assert code == 0 and plan[4] == 12 and plan[5] == 3
        code, plan, ctas = schedule(lib, N, 4096, 1, 36)
        assert code == 0 and plan[4] == 0 and plan[3] == plan[1]
    code, _, _ = schedule(lib, 24576, 4096, 68, 36)
    assert code == 0


def test_schedule_rejects_what_the_launch_does_not_cover(lib):
    assert schedule(lib, 4096, 4096, 129, 36)[0] == 5
    assert schedule(lib, 4096, 192, 17, 36)[0] == 5
    assert schedule(lib, 4096, 4100, 17, 36)[0] == 1
