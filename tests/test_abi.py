"""The C-ABI library builds, loads and exports every function declared in
include/pard.h; host-only entry points validate their arguments without a
GPU."""
import ctypes
import os
import re

import pytest

import synthetic as S

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def declared_functions():
    src = open(os.path.join(ROOT, "include", "pard.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(pard_[a-z_]+)\s*\(", src)))


@pytest.fixture(scope="module")
def lib():
    from paper_2504_18583_gb300 import _build
    _build.build()
    return ctypes.CDLL(_build.LIB)


def test_header_declares_the_decode_step_calls():
    names = declared_functions()
    for required in ("pard_load_weights", "pard_prefill", "pard_draft", "pard_verify", "pard_accept_commit"):
        assert required in names


def test_library_exports_every_declared_symbol(lib):
    missing = [n for n in declared_functions() if not hasattr(lib, n)]
    assert not missing, missing


def test_sizing_is_host_only_and_validates():
    from paper_2504_18583_gb300 import pard
    wl = S.WORKLOADS["8b_greedy"]
    t, d = pard.ModelCfg.of(wl.target), pard.ModelCfg.of(wl.draft)
    lim = pard.Limits(1, 8, 800, 16, 512, 50)
    ws = pard.pard_workspace_bytes(t, d, lim)
    kv = pard.pard_kv_pool_bytes(t, d, lim)
    assert ws > 0
    # KV pool: pages x (target + draft) layers x K/V x kv_heads x page_size x head_dim x bf16
    assert kv == 50 * 2 * 16 * 2 * (32 * 8 * 128 + 16 * 8 * 64)
    bad = pard.ModelCfg.of(wl.target.replace(head_dim=96))
    assert pard.pard_workspace_bytes(bad, d, lim) == 0
    assert pard.pard_workspace_bytes(t, d, pard.Limits(0, 8, 800, 16, 512, 50)) == 0
    assert pard.pard_workspace_bytes(t, d, pard.Limits(1, 8, 800, 16, 100, 50)) == 0


def test_load_rejects_bad_shapes_before_touching_the_device():
    from paper_2504_18583_gb300 import pard
    wl = S.WORKLOADS["tiny"]
    t = pard.ModelCfg.of(wl.target.replace(n_q_heads=3))
    d = pard.ModelCfg.of(wl.draft)
    lim = pard.Limits(1, 4, 64, 16, 64, 8)
    ctx = ctypes.c_void_p()
    w = pard.Weights()
    code = pard.lib().pard_load_weights(ctypes.byref(ctx), ctypes.byref(t), ctypes.byref(w), ctypes.byref(d),
                                        ctypes.byref(w), ctypes.byref(lim), None, 0, None, 0, None, None, None)
    assert code == -2 and "multiple" in pard.pard_last_error()
    code = pard.lib().pard_draft(None, 0, 1.0, 0, 0, None, None, None)
    assert code == -1
    assert pard.lib().pard_draft_sequential(None, 0, 1.0, 0, 0, None, None, None) == -1
    assert pard.lib().pard_set_mask_ids(None, None, 0, None) == -1
    assert pard.lib().pard_selftest_stalled_wait(None, None) == -1
    assert pard.lib().pard_set_attention_split_cap(None, 8) == -1
    bits = ctypes.c_uint32(0)
    assert pard.lib().pard_attention_paths(None, ctypes.byref(bits), None) == -1
    # COD: argument checks happen on the host, before any launch
    for n, K, r, r_min in ((0, 3, 0.5, 0.0), (4097, 3, 0.5, 0.0), (10, 0, 0.5, 0.0), (10, 3, 0.0, 0.0),
                           (10, 3, 1.5, 0.0), (10, 3, 0.5, -0.1)):
        assert pard.lib().pard_cod_select(n, K, r, r_min, 0, 0, None, None, None) == -1


def test_binding_fails_loudly_without_the_library(monkeypatch, tmp_path):
    from paper_2504_18583_gb300 import pard
    monkeypatch.setattr(pard, "LIB", str(tmp_path / "missing.so"))
    monkeypatch.setattr(pard, "_lib", None)
    with pytest.raises(RuntimeError, match="no CPU fallback"):
        pard.lib()
