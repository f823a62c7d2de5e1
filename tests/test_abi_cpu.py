"""C ABI checks that need no GPU: the library loads, exports every function
include/gs.h declares, and rejects bad arguments before touching the device."""
import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def gs():
    from paper_2609_26638_gb300 import build
    build.build()
    from paper_2609_26638_gb300 import gs as binding
    return binding


def declared_functions():
    src = open(os.path.join(ROOT, "include", "gs.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(gs_[a-z_]+)\s*\(", src)))


def test_every_declared_symbol_is_exported(gs):
    names = declared_functions()
    assert len(names) >= 14
    lib = ctypes.CDLL(gs.LIB_PATH)
    for n in names:
        assert hasattr(lib, n), n
    assert set(names) == set(gs.EXPORTED)


def _cfg(gs, **kw):
    c = gs.gs_config()
    vals = dict(n_layers=2, d_model=256, n_heads=4, n_kv_heads=4, head_dim=64, d_ffn=1024,
                vocab=4096, rope_theta=10000.0, rms_eps=1e-6, mask_token_id=4095, eos_token_id=-1,
                max_batch=2, max_ctx=1024, max_K=8, max_prefill=512, kv_pages=0, split_pages=0)
    vals.update(kw)
    for k, v in vals.items():
        setattr(c, k, v)
    return c


def test_workspace_sizing_and_config_validation(gs):
    assert gs.gs_workspace_bytes(_cfg(gs)) > 0
    bigger = gs.gs_workspace_bytes(_cfg(gs, max_batch=4))
    assert bigger > gs.gs_workspace_bytes(_cfg(gs))
    for bad in (dict(head_dim=128), dict(n_heads=3, n_kv_heads=2), dict(d_model=200),
                dict(vocab=4000), dict(mask_token_id=4096), dict(max_batch=0),
                dict(d_ffn=100), dict(max_K=200, n_heads=8, n_kv_heads=2)):
        assert gs.gs_workspace_bytes(_cfg(gs, **bad)) == 0, bad


def test_create_rejects_bad_arguments_without_a_device(gs):
    lib = gs.lib()
    h = ctypes.c_void_p()
    w = gs.gs_weights()
    rc = lib.gs_create(ctypes.byref(_cfg(gs)), ctypes.byref(w), None, 0, None, ctypes.byref(h))
    assert rc == gs.GS_ERR_INVALID_ARG
    assert "weight" in lib.gs_last_error(None).decode()
    rc = lib.gs_create(ctypes.byref(_cfg(gs, head_dim=32)), ctypes.byref(w), None, 0, None,
                       ctypes.byref(h))
    assert rc == gs.GS_ERR_INVALID_ARG and "head_dim" in lib.gs_last_error(None).decode()


def test_entry_points_validate_before_launch(gs):
    lib = gs.lib()
    assert lib.gs_round(None, None, 1, 4, 0, None, None, None, None, None) == gs.GS_ERR_INVALID_ARG
    assert lib.gs_prefill(None, 0, None, 0, None, 0, 1, None) == gs.GS_ERR_INVALID_ARG
    assert lib.gs_destroy(None) == gs.GS_ERR_INVALID_ARG
    # K not a multiple of 64, split not dividing K/64, bad epilogue
    assert lib.gs_linear(8, 8, 8, 4, 128, 100, 0, 1, 8, 1 << 20, None) == gs.GS_ERR_INVALID_ARG
    assert lib.gs_linear(8, 8, 8, 4, 128, 192, 0, 2, 8, 1 << 20, None) == gs.GS_ERR_INVALID_ARG
    assert lib.gs_linear(8, 8, 8, 4, 128, 128, 7, 1, 8, 1 << 20, None) == gs.GS_ERR_INVALID_ARG
    assert lib.gs_attention(2, 8, 8, 1, 8, 1, 8, 1, 5, 16, 8, 8, 8, 1 << 20, 1, None) == \
        gs.GS_ERR_INVALID_ARG
    assert gs.gs_attention_scratch_bytes(2, 17, 16, 8, 40, 2) > 0
    assert gs.gs_attention_scratch_bytes(2, 17, 16, 7, 40, 2) == 0
    # cluster split-K (<= 8 splits at <= 64 rows) needs no partials; 32 splits reduce through scratch
    assert gs.gs_linear_scratch_bytes(17, 2048, 8) == gs.gs_linear_scratch_bytes(17, 2048, 1)
    assert gs.gs_linear_scratch_bytes(17, 2048, 32) > gs.gs_linear_scratch_bytes(17, 2048, 1)
