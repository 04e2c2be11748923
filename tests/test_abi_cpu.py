"""Host-side checks of the C ABI: the library loads, exports every function the
header declares, its structs match the ctypes mirror, and argument validation
rejects bad calls without touching a GPU."""
import ctypes
import os
import re
import subprocess

import pytest

import synth

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "dflow.h")


@pytest.fixture(scope="module")
def abi():
    from paper_2609_06498_gb300 import build
    build.build()
    from paper_2609_06498_gb300 import _abi
    _abi.lib()
    return _abi


def declared_functions():
    text = open(HEADER).read()
    return sorted(set(re.findall(r"^\s*(?:const\s+char\s*\*|dflow_status)\s*(dflow_\w+)\s*\(", text, re.M)))


def test_every_declared_function_is_exported(abi):
    names = declared_functions()
    assert len(names) >= 12
    lib = abi.lib()
    for n in names:
        assert hasattr(lib, n), n
    assert sorted(abi.EXPORTS) == names


def test_struct_layouts_match_header(abi, tmp_path):
    src = tmp_path / "sz.c"
    src.write_text('#include "dflow.h"\n#include <stdio.h>\n#include <stddef.h>\nint main(void){'
                   'printf("%zu %zu %zu %zu %zu %zu\\n", sizeof(dflow_config), sizeof(dflow_layer_weights),'
                   'sizeof(dflow_weights), sizeof(dflow_state), offsetof(dflow_config, rope_theta),'
                   'offsetof(dflow_state, status)); return 0;}\n')
    exe = tmp_path / "sz"
    subprocess.check_call(["gcc", "-I", os.path.join(ROOT, "include"), str(src), "-o", str(exe)])
    got = [int(x) for x in subprocess.check_output([str(exe)]).split()]
    want = [ctypes.sizeof(abi.Config), ctypes.sizeof(abi.LayerWeights), ctypes.sizeof(abi.Weights),
            ctypes.sizeof(abi.State), abi.Config.rope_theta.offset, abi.State.status.offset]
    assert got == want


def _fake_weights(abi, cfg):
    fake = ctypes.c_void_p(0x1000)
    lw = (abi.LayerWeights * cfg.n_layers)(*[abi.LayerWeights(*([0x1000] * 8)) for _ in range(cfg.n_layers)])
    dw = (abi.LayerWeights * cfg.draft_layers)(*[abi.LayerWeights(*([0x1000] * 8)) for _ in range(cfg.draft_layers)])
    w = abi.Weights(embed=fake, lm_head=fake, final_norm=fake, target=lw, draft=dw, draft_final_norm=fake, w_c=fake,
                    c_norm=fake, e_mask=fake, relay_w1=fake, relay_w2=fake, ln_w=fake, ln_b=fake)
    return w, (lw, dw)


def _config(abi, cfg, **over):
    fl = list(cfg.feat_layers) + [0] * (8 - len(cfg.feat_layers))
    c = abi.Config(dtype=1 if cfg.dtype == "bf16" else 0, d_model=cfg.d, n_layers=cfg.n_layers,
                   n_q_heads=cfg.n_q_heads, n_kv_heads=cfg.n_kv_heads, head_dim=cfg.head_dim, d_inter=cfg.inter,
                   vocab=cfg.vocab, draft_layers=cfg.draft_layers, n_feat=len(cfg.feat_layers),
                   feat_layers=(ctypes.c_int32 * 8)(*fl), block=cfg.block, page_size=cfg.page_size, max_batch=2,
                   max_ctx=cfg.max_ctx(), num_pages=64, rope_theta=cfg.rope_theta, rms_eps=cfg.rms_eps,
                   ln_eps=cfg.ln_eps)
    for k, v in over.items():
        setattr(c, k, v)
    return c


@pytest.mark.parametrize("cfg", [synth.TINY, synth.QWEN3_8B], ids=lambda c: c.name)
def test_create_and_workspace_size_on_host(abi, cfg):
    w, keep = _fake_weights(abi, cfg)
    h = ctypes.c_void_p()
    assert abi.lib().dflow_create(ctypes.byref(_config(abi, cfg)), ctypes.byref(w), ctypes.byref(h)) == 0
    n = ctypes.c_size_t()
    assert abi.lib().dflow_workspace_size(h, ctypes.byref(n)) == 0
    assert n.value > 0
    # calls before a workspace is handed over are rejected
    st = abi.State(batch=1)
    assert abi.lib().dflow_round(h, ctypes.byref(st), None, None, None, 1, None) == 1
    assert abi.lib().dflow_destroy(h) == 0


@pytest.mark.parametrize("field,value,code", [
    ("head_dim", 96, 5), ("d_model", 300, 5), ("dtype", 7, 1), ("n_feat", 0, 1), ("block", 0, 1),
    ("max_ctx", 100, 5),
])
def test_create_rejects_bad_config(abi, field, value, code):
    w, keep = _fake_weights(abi, synth.TINY)
    h = ctypes.c_void_p()
    c = _config(abi, synth.TINY, **{field: value})
    assert abi.lib().dflow_create(ctypes.byref(c), ctypes.byref(w), ctypes.byref(h)) == code
    assert not h.value


def test_create_rejects_null_weights(abi):
    w, keep = _fake_weights(abi, synth.TINY)
    w.relay_w2 = None
    h = ctypes.c_void_p()
    assert abi.lib().dflow_create(ctypes.byref(_config(abi, synth.TINY)), ctypes.byref(w), ctypes.byref(h)) == 1
    assert abi.lib().dflow_create(None, ctypes.byref(w), ctypes.byref(h)) == 1


def test_status_strings(abi):
    for code in range(7):
        assert abi.lib().dflow_status_string(code)
