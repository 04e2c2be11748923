"""The allocation-free greedy-token entry point, through the C ABI, on two calls
in a row.

Callers that cannot allocate device memory (code confined to a caller-owned
memory pool or fixed-budget arena, or a plugin whose host framework owns every
allocation) use dflow_greedy_tokens_noalloc, whose scratch is an array compiled
into the library.  Its tokens are checked against a plain fp32 matmul + argmax
of the same bf16 values (wherever the top-2 gap makes the argmax safe from
accumulation-order rounding) and against the library's regular LM-head path,
which keeps the same scratch in a caller workspace."""
import ctypes

import pytest
import torch

from parity_util import lmhead_engine

pytestmark = pytest.mark.gpu

V, D = 151936, 4096


def _inputs(rows, seed):
    g = torch.Generator(device="cuda")
    g.manual_seed(seed)
    W = (torch.randn(V, D, generator=g, device="cuda") * 0.02).to(torch.bfloat16)
    X = torch.randn(rows, D, generator=g, device="cuda").to(torch.bfloat16)
    return W, X


def _noalloc(lib, W, X, rows):
    out = torch.full((rows,), -7, dtype=torch.int32, device="cuda")
    code = lib.dflow_greedy_tokens_noalloc(ctypes.c_void_p(W.data_ptr()), V, D, ctypes.c_void_p(X.data_ptr()), rows,
                                           ctypes.c_void_p(out.data_ptr()),
                                           ctypes.c_void_p(torch.cuda.current_stream().cuda_stream))
    assert code == 0
    return out


@pytest.mark.parametrize("rows", [17, 1, 64])
def test_noalloc_matches_fp32_argmax_and_regular_path_twice(rows):
    from paper_2609_06498_gb300 import _abi
    lib = _abi.lib()
    W, X = _inputs(rows, rows)
    logits = X.float() @ W.float().T  # plain fp32 product of the same bf16 values
    top2 = logits.topk(2, dim=1)
    safe = (top2.values[:, 0] - top2.values[:, 1]) > 1e-3
    assert safe.sum() >= max(1, rows // 2)
    eng = lmhead_engine(64)
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    ref = torch.empty(rows, dtype=torch.int32, device="cuda")
    eng.debug_gemm(1, W, X, 4, ref, st)  # the regular path: LM-head GEMM + argmax with workspace scratch
    first = _noalloc(lib, W, X, rows)
    second = _noalloc(lib, W, X, rows)
    torch.cuda.synchronize()
    assert int(st) == 0
    for got in (first, second):
        assert torch.equal(got.long()[safe], top2.indices[:, 0][safe])
        assert torch.equal(got, ref)


def test_noalloc_rejects_sizes_beyond_its_scratch():
    from paper_2609_06498_gb300 import _abi
    lib = _abi.lib()
    W, X = _inputs(1, 0)
    out = torch.empty(65, dtype=torch.int32, device="cuda")
    s = ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    assert lib.dflow_greedy_tokens_noalloc(ctypes.c_void_p(W.data_ptr()), V, D, ctypes.c_void_p(X.data_ptr()), 65,
                                           ctypes.c_void_p(out.data_ptr()), s) == 1
    assert lib.dflow_greedy_tokens_noalloc(ctypes.c_void_p(W.data_ptr()), 2048 * 128 + 1, D,
                                           ctypes.c_void_p(X.data_ptr()), 1, ctypes.c_void_p(out.data_ptr()), s) == 1
