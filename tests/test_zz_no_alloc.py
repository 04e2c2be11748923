"""The allocation-free greedy-token entry point (for callers that cannot allocate
device memory, e.g. code confined to a caller-owned pool) against the library's
regular LM-head argmax path, through the C ABI, on two calls in a row."""
import ctypes

import pytest
import torch

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
def test_noalloc_matches_regular_path_twice(rows):
    from paper_2609_06498_gb300 import _abi
    from paper_2609_06498_gb300.probe import _engine
    lib = _abi.lib()
    eng = _engine(64)
    W, X = _inputs(rows, rows)
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    ref = torch.empty(rows, dtype=torch.int32, device="cuda")
    eng.debug_gemm(1, W, X, 4, ref, st)  # the regular path: LM-head GEMM + argmax with workspace scratch
    first = _noalloc(lib, W, X, rows)
    second = _noalloc(lib, W, X, rows)
    torch.cuda.synchronize()
    assert int(st) == 0
    assert torch.equal(first, ref)
    assert torch.equal(second, ref)


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
