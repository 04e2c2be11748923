"""The tcgen05 GEMM kernel against a plain fp32 matmul of the same bf16
inputs, for every fused epilogue, on shapes with ragged tails (N not a
multiple of 128, M not a multiple of 16, M above one 256-row token tile) and
with k-blocks split across CTAs."""
import numpy as np
import pytest
import torch

import synth

pytestmark = pytest.mark.gpu

SHAPES = [  # (N, K, M)
    (256, 64, 1), (1000, 512, 17), (6144, 4096, 17), (4096, 4096, 32), (24576, 4096, 17), (4096, 12288, 17),
    (151936, 4096, 17), (2048, 4096, 272), (512, 1472, 48), (384, 3072, 300), (2944, 512, 5),
    # persistent kernel above 64 columns: two epilogue chunks per owner (68 -> 80, 100 -> 128 columns)
    (6144, 2560, 68), (2560, 9728, 100), (4096, 4096, 128),
    # Eq. 1 feature projection of the 5-feature-layer workloads (K = 5 d)
    (4096, 20480, 17), (2560, 12800, 68),
    # batch 16 x 17 rows: one pass with two MMAs per k-step (256 + 16 columns), split over k through L2
    (4096, 4096, 272), (6144, 4096, 272), (4096, 12288, 272), (4096, 20480, 272), (1000, 512, 511), (2048, 1024, 600),
]


@pytest.fixture(scope="module")
def eng():
    from paper_2609_06498_gb300 import Engine, build, random_weights
    build.build()
    cfg = synth.ModelConfig(name="gemm_probe", dtype="bf16", d=512, n_layers=1, n_q_heads=4, n_kv_heads=1,
                            head_dim=128, inter=1472, vocab=151936, draft_layers=1, feat_layers=(1,), block=16,
                            batch=16, prompt_len=64, new_tokens=16, schedule="uniform")
    return Engine(cfg, random_weights(cfg), max_batch=16, max_ctx=256)


def _inputs(N, K, M, seed):
    g = torch.Generator(device="cuda")
    g.manual_seed(seed)
    W = (torch.randn(N, K, generator=g, device="cuda") * 0.05).to(torch.bfloat16)
    X = torch.randn(M, K, generator=g, device="cuda").to(torch.bfloat16)
    ref = X.float() @ W.float().T  # plain fp32 matmul of the same bf16 values
    return W, X, ref


def _rel(a, b):
    return float((a - b).abs().max() / b.abs().max())


def _tol(K):
    # both sides accumulate K products in fp32: rounding walks like sqrt(K) u
    # (u = 2^-24) of the largest output on each side; 4 sqrt(K) u, 1e-5 at least
    return max(1e-5, 4 * K ** 0.5 * 2.0 ** -24)


def _seq_ok(K, M):
    # the persistent launch (path 2) takes 16 to 128 rows and at least 4 k-blocks
    return 16 <= M <= 128 and K % 64 == 0 and K // 64 >= 4


PATHS = pytest.mark.parametrize("path", [1, 2, 3], ids=["tc", "persistent", "wide"])


def _path_ok(path, K, M):
    if path == 2:
        return _seq_ok(K, M)
    if path == 1:
        return M <= 272 or M % 256 == 0  # the one-projection kernel: passes of 256 rows (kept to the old shapes)
    return K % 64 == 0


@PATHS
@pytest.mark.parametrize("N,K,M", SHAPES)
def test_store_and_resid(eng, path, N, K, M):
    if not _path_ok(path, K, M):
        pytest.skip("outside this launch")
    W, X, ref = _inputs(N, K, M, N + K + M)
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    out = torch.full((M, N), float("nan"), device="cuda")
    eng.debug_gemm(path, W, X, 0, out, st)
    torch.cuda.synchronize()
    assert int(st) == 0
    assert _rel(out, ref) < _tol(K)
    base = torch.randn(M, N, device="cuda")
    acc = base.clone()
    eng.debug_gemm(path, W, X, 1, acc, st)
    torch.cuda.synchronize()
    assert _rel(acc - base, ref) < 1e-4
    out2 = torch.empty_like(out)
    eng.debug_gemm(path, W, X, 0, out2, st)
    torch.cuda.synchronize()
    assert torch.equal(out, out2), "not deterministic"


@PATHS
@pytest.mark.parametrize("N,K,M", [(2944, 512, 17), (24576, 4096, 17), (19456, 2560, 68), (3072, 1024, 300),
                                   (24576, 4096, 272)])
def test_swiglu_and_silu(eng, path, N, K, M):
    if not _path_ok(path, K, M):
        pytest.skip("outside this launch")
    W, X, ref = _inputs(N, K, M, 7 * N + M)
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    h = torch.empty(M, N // 2, dtype=torch.bfloat16, device="cuda")
    eng.debug_gemm(path, W, X, 2, h, st)
    g = ref.view(M, N // 128, 2, 64)
    want = (torch.nn.functional.silu(g[:, :, 0]) * g[:, :, 1]).reshape(M, N // 2)
    s = torch.empty(M, N, dtype=torch.bfloat16, device="cuda")
    eng.debug_gemm(path, W, X, 3, s, st)
    torch.cuda.synchronize()
    assert int(st) == 0
    assert _rel(h.float(), want) < 1e-2
    assert _rel(s.float(), torch.nn.functional.silu(ref)) < 1e-2


@pytest.mark.parametrize("path", [1, 3], ids=["tc", "wide"])
@pytest.mark.parametrize("N,K,M", [(1000, 512, 17), (151936, 4096, 17), (151936, 4096, 1), (151936, 4096, 272)])
def test_argmax(eng, path, N, K, M):
    W, X, ref = _inputs(N, K, M, 11 * N + M)
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    out = torch.empty(M, dtype=torch.int32, device="cuda")
    eng.debug_gemm(path, W, X, 4, out, st)
    torch.cuda.synchronize()
    assert int(st) == 0
    top2 = ref.topk(2, dim=1)
    safe = (top2.values[:, 0] - top2.values[:, 1]) > 1e-3
    assert safe.any()
    assert torch.equal(out.long()[safe], top2.indices[:, 0][safe])


def test_persistent_launch_refuses_fewer_than_16_rows(eng):
    """Rows 1-15 never reach the persistent launch: the call is refused on the
    host, before anything is launched (the round routes them to the row-tiled kernel)."""
    from paper_2609_06498_gb300._abi import DFlowError
    W, X, _ = _inputs(4096, 4096, 1, 3)
    out = torch.zeros(1, 4096, device="cuda")
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    with pytest.raises(DFlowError):
        eng.debug_gemm(2, W, X, 0, out, st)
    eng.debug_gemm(1, W, X, 0, out, st)  # the row-tiled kernel takes it
    torch.cuda.synchronize()
    assert int(st) == 0 and _rel(out, X.float() @ W.float().T) <= _tol(4096)
