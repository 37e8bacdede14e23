"""Host-side checks of libkvx.so (no GPU needed).

The library builds for sm_103a, loads, exports every symbol include/kvx.h
declares, and its host-only logic (layer map, argument validation) behaves.
"""
import ctypes
import os
import re

import numpy as np
import pytest

import oracle
import paper_2608_30963_gb300 as kvx
from paper_2608_30963_gb300 import synth

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def lib():
    kvx.build()
    return kvx.lib()


def declared_symbols():
    txt = open(os.path.join(ROOT, "include", "kvx.h")).read()
    return sorted(set(re.findall(r"KVX_API\s+[\w\s\*]+?\b(kvx_\w+)\s*\(", txt)))


def test_header_declares_the_boundary():
    names = declared_symbols()
    for must in ("kvx_translator_create", "kvx_translate", "kvx_destroy", "kvx_build_alignment",
                 "kvx_layer_map_nearest", "kvx_get_device_status", "kvx_last_error"):
        assert must in names


def test_every_declared_symbol_is_exported(lib):
    for name in declared_symbols():
        assert hasattr(lib, name), name
    assert sorted(declared_symbols()) == sorted(kvx.EXPORTS) or set(kvx.EXPORTS) <= set(declared_symbols())


@pytest.mark.parametrize("Ls,Lt", [(4, 2), (28, 28), (28, 26), (80, 28), (1, 3), (5, 1), (3, 7)])
def test_layer_map_matches_oracle(lib, Ls, Lt):
    assert kvx.kvx_layer_map_nearest(Ls, Lt) == list(oracle.layer_map_nearest(Ls, Lt))


def _desc(src, dst, dtype=kvx.KVX_BF16, path=kvx.KVX_PATH_AUTO, layer_map=None):
    return kvx.kvx_translator_desc(kvx.model_geom(src), kvx.model_geom(dst), layer_map, dtype, 0, path)


@pytest.mark.parametrize("src,dst,code", [
    (synth.ModelGeom(2, 3, 128, 1e6), synth.ModelGeom(2, 2, 128, 1e6), kvx.KVX_ERR_UNSUPPORTED),   # 3 vs 2 heads
    (synth.ModelGeom(2, 2, 96, 1e6), synth.ModelGeom(2, 2, 128, 1e6), kvx.KVX_ERR_UNSUPPORTED),    # head_dim 96
    (synth.ModelGeom(2, 32, 128, 1e6), synth.ModelGeom(2, 2, 128, 1e6), kvx.KVX_ERR_UNSUPPORTED),  # in = 2048
    (synth.ModelGeom(0, 2, 128, 1e6), synth.ModelGeom(2, 2, 128, 1e6), kvx.KVX_ERR_INVALID_ARG),
    (synth.ModelGeom(2, 2, 128, 1e6), synth.ModelGeom(200, 2, 128, 1e6), kvx.KVX_ERR_UNSUPPORTED),
    (synth.ModelGeom(2, 2, 128, 1e6, rope_type=3), synth.ModelGeom(2, 2, 128, 1e6), kvx.KVX_ERR_INVALID_ARG),
    (synth.ModelGeom(2, 2, 128, 1e6, rope_type=1, rope_factor=0.0), synth.ModelGeom(2, 2, 128, 1e6),
     kvx.KVX_ERR_INVALID_ARG),
    (synth.ModelGeom(2, 2, 128, 1e6), synth.ModelGeom(2, 2, 128, 1e6, rope_type=2, rope_factor=8.0,
                                                       rope_low_freq_factor=4.0, rope_high_freq_factor=1.0),
     kvx.KVX_ERR_INVALID_ARG),
    # partial rotary: rotary_dim must be 0 or a multiple of 16 in [16, head_dim]
    (synth.ModelGeom(2, 2, 128, 1e6, rotary_dim=24), synth.ModelGeom(2, 2, 128, 1e6), kvx.KVX_ERR_INVALID_ARG),
    (synth.ModelGeom(2, 2, 128, 1e6), synth.ModelGeom(2, 2, 128, 1e6, rotary_dim=256), kvx.KVX_ERR_INVALID_ARG),
    (synth.ModelGeom(2, 2, 128, 1e6), synth.ModelGeom(2, 2, 128, 1e6, rotary_dim=-16), kvx.KVX_ERR_INVALID_ARG),
    (synth.ModelGeom(2, 2, 64, 1e6, rotary_dim=8), synth.ModelGeom(2, 2, 128, 1e6), kvx.KVX_ERR_INVALID_ARG),
])
def test_create_rejects_bad_geometry_without_touching_cuda(lib, src, dst, code):
    h = ctypes.c_void_p()
    w = (ctypes.c_uint16 * 4)()
    st = lib.kvx_translator_create(ctypes.byref(_desc(src, dst)), ctypes.cast(w, ctypes.c_void_p),
                                   ctypes.cast(w, ctypes.c_void_p), 0, ctypes.byref(h))
    assert st == code
    assert h.value is None
    assert kvx.kvx_last_error()


@pytest.mark.parametrize("form,k,with_map,code", [
    (2, 1, False, kvx.KVX_ERR_INVALID_ARG),       # unknown form
    (0, 5, True, kvx.KVX_ERR_INVALID_ARG),        # more than 4 source layers per target layer
    (0, 2, False, kvx.KVX_ERR_INVALID_ARG),       # a group of layers needs an explicit map
    (1, 1, False, kvx.KVX_ERR_UNSUPPORTED),       # dense over 16 heads of 128: in = 2048
])
def test_create_rejects_bad_translator_forms(lib, form, k, with_map, code):
    src, dst = synth.ModelGeom(8, 16, 128, 1e6), synth.ModelGeom(2, 2, 128, 1e6)
    lm = (ctypes.c_int32 * 10)(*range(10))
    d = _desc(src, dst, layer_map=ctypes.cast(lm, kvx.I32P) if with_map else None)
    d.form, d.layers_per_target = form, k
    h = ctypes.c_void_p()
    w = (ctypes.c_uint16 * 4)()
    st = lib.kvx_translator_create(ctypes.byref(d), ctypes.cast(w, ctypes.c_void_p),
                                   ctypes.cast(w, ctypes.c_void_p), 0, ctypes.byref(h))
    assert st == code, kvx.kvx_last_error()
    assert h.value is None


def test_low_rank_create_rejects_bad_rank(lib):
    d = _desc(synth.ModelGeom(2, 4, 128, 1e6), synth.ModelGeom(2, 2, 128, 1e6))
    h = ctypes.c_void_p()
    w = (ctypes.c_uint16 * 4)()
    p = ctypes.cast(w, ctypes.c_void_p)
    for rank in (0, 1025):
        assert lib.kvx_translator_create_low_rank(ctypes.byref(d), rank, p, p, p, p, 0, ctypes.byref(h)) == \
            kvx.KVX_ERR_INVALID_ARG
    assert "rank" in kvx.kvx_last_error()


def test_create_rejects_out_of_range_layer_map(lib):
    lm = (ctypes.c_int32 * 2)(0, 5)
    d = _desc(synth.ModelGeom(4, 2, 64, 1e4), synth.ModelGeom(2, 1, 64, 1e4),
              layer_map=ctypes.cast(lm, kvx.I32P))
    h = ctypes.c_void_p()
    w = (ctypes.c_float * 4)()
    st = lib.kvx_translator_create(ctypes.byref(d), ctypes.cast(w, ctypes.c_void_p),
                                   ctypes.cast(w, ctypes.c_void_p), 0, ctypes.byref(h))
    assert st == kvx.KVX_ERR_INVALID_ARG
    assert "layer_map" in kvx.kvx_last_error()


def test_null_arguments_rejected(lib):
    assert lib.kvx_translate(None, None, None, None, None) == kvx.KVX_ERR_INVALID_ARG
    assert lib.kvx_get_device_status(None, None, None, 0) == kvx.KVX_ERR_INVALID_ARG
    assert lib.kvx_destroy(None) == kvx.KVX_OK
    assert lib.kvx_build_alignment(0, 0, 0, None, None, None, None, None, None, None, None) == \
        kvx.KVX_ERR_INVALID_ARG


def _geom_desc(src, dst, **kw):
    d = _desc(src, dst)
    for k, v in kw.items():
        setattr(d, k, v)
    return d


def test_fit_create_rejects_bad_arguments_without_touching_cuda(lib):
    h = ctypes.c_void_p()
    ok_src, ok_dst = synth.ModelGeom(2, 4, 128, 1e6), synth.ModelGeom(2, 2, 128, 1e6)
    assert lib.kvx_fit_create(None, 0.1, 0, ctypes.byref(h)) == kvx.KVX_ERR_INVALID_ARG
    for lam in (-1.0, float("nan")):
        assert lib.kvx_fit_create(ctypes.byref(_desc(ok_src, ok_dst)), lam, 0, ctypes.byref(h)) == \
            kvx.KVX_ERR_INVALID_ARG
        assert "lambda" in kvx.kvx_last_error()
    for chunk in (-1, (1 << 20) + 1):
        assert lib.kvx_fit_create(ctypes.byref(_desc(ok_src, ok_dst)), 0.1, chunk, ctypes.byref(h)) == \
            kvx.KVX_ERR_INVALID_ARG
        assert "chunk_tokens" in kvx.kvx_last_error()
    # the translator geometry is checked as for kvx_translator_create
    bad = _desc(synth.ModelGeom(2, 4, 128, 1e6, rotary_dim=24), ok_dst)
    assert lib.kvx_fit_create(ctypes.byref(bad), 0.1, 0, ctypes.byref(h)) == kvx.KVX_ERR_INVALID_ARG
    # the fit takes translator inputs up to 512 wide: 8 grouped heads of 128 are 1024
    wide = _desc(synth.ModelGeom(2, 16, 128, 1e6), ok_dst)
    assert lib.kvx_fit_create(ctypes.byref(wide), 0.1, 0, ctypes.byref(h)) == kvx.KVX_ERR_UNSUPPORTED
    assert h.value is None


def test_fit_calls_reject_a_null_fitter(lib):
    assert lib.kvx_fit_accumulate(None, None, None, None, None) == kvx.KVX_ERR_INVALID_ARG
    assert lib.kvx_fit_solve(None, None, None, None, None) == kvx.KVX_ERR_INVALID_ARG
    assert lib.kvx_fit_reset(None, None) == kvx.KVX_ERR_INVALID_ARG
    assert lib.kvx_fit_tokens(None) == 0
    assert lib.kvx_fit_destroy(None) == kvx.KVX_OK


@pytest.mark.parametrize("src,dst,kw,code,words", [
    (synth.ModelGeom(2, 2, 96, 1e6), synth.ModelGeom(2, 2, 128, 1e6), {}, kvx.KVX_ERR_UNSUPPORTED, "head dims"),
    (synth.ModelGeom(2, 3, 128, 1e6), synth.ModelGeom(2, 2, 128, 1e6), {}, kvx.KVX_ERR_UNSUPPORTED, "divides"),
    (synth.ModelGeom(2, 4, 128, 1e6), synth.ModelGeom(2, 2, 128, 1e6), dict(form=kvx.KVX_FORM_DENSE),
     kvx.KVX_ERR_UNSUPPORTED, "per-KV-head"),
    (synth.ModelGeom(2, 4, 128, 1e6), synth.ModelGeom(2, 2, 128, 1e6), dict(layers_per_target=2),
     kvx.KVX_ERR_UNSUPPORTED, "per-KV-head"),
    (synth.ModelGeom(2, 4, 128, 1e6, rotary_dim=40), synth.ModelGeom(2, 2, 128, 1e6), {},
     kvx.KVX_ERR_INVALID_ARG, "rope"),
    (synth.ModelGeom(2, 4, 128, 1e6), synth.ModelGeom(2, 2, 128, 1e6), dict(dtype=7), kvx.KVX_ERR_INVALID_ARG,
     "dtype"),
])
def test_static_entry_rejects_bad_descriptions_without_touching_cuda(lib, src, dst, kw, code, words):
    d = _geom_desc(src, dst, **kw)
    w = (ctypes.c_uint16 * 4)()
    p = ctypes.cast(w, ctypes.c_void_p)
    s, t, o = kvx.kvx_src_kv(), kvx.kvx_tgt_tokens(), kvx.kvx_dst_kv()
    st = lib.kvx_translate_static(ctypes.byref(d), p, p, ctypes.byref(s), ctypes.byref(t), ctypes.byref(o), None,
                                  None)
    assert st == code
    assert words in lib.kvx_static_last_error().decode()
    assert lib.kvx_translate_static(None, p, p, ctypes.byref(s), ctypes.byref(t), ctypes.byref(o), None, None) == \
        kvx.KVX_ERR_INVALID_ARG
