"""The C-ABI library builds, loads and exports every function include/kvg.h
declares; host-side argument checks answer without touching a GPU."""
import ctypes

import pytest

from paper_2607_14431_gb300 import build, kvg


@pytest.fixture(scope="module")
def lib():
    build.build()
    return kvg.lib()


def test_every_declared_function_is_exported(lib):
    names = kvg.header_functions()
    assert len(names) >= 20
    missing = [n for n in names if not hasattr(lib, n)]
    assert not missing, missing
    # and the binding declares a signature for each
    assert set(names) <= set(kvg._SIGNATURES), set(names) - set(kvg._SIGNATURES)


def test_status_strings_and_version(lib):
    assert kvg.kvg_status_string(0) == "ok"
    assert kvg.kvg_status_string(kvg.KVG_ERR_DIGEST) == "digest mismatch"
    assert kvg.kvg_version() >= 0x000100
    assert lib.kvg_launch_count.restype is not None or True


def test_host_checks_reject_bad_geometry_without_a_gpu(lib):
    h = ctypes.c_void_p()
    bad = kvg.make_dims(2, 2, 96, 16)  # head_dim 96 unsupported
    assert lib.kvg_store_create(ctypes.byref(bad), 0, 1 << 20, 0, ctypes.byref(h)) == kvg.KVG_ERR_ARG
    assert "geometry" in kvg.kvg_last_error()
    assert lib.kvg_cache_create(ctypes.byref(bad), 4, 1, 64, 0, ctypes.byref(h)) == kvg.KVG_ERR_ARG
    good = kvg.make_dims(2, 2, 64, 16)
    assert lib.kvg_store_create(ctypes.byref(good), 7, 1 << 20, 0, ctypes.byref(h)) == kvg.KVG_ERR_ARG
    assert lib.kvg_store_create(None, 0, 1 << 20, 0, ctypes.byref(h)) == kvg.KVG_ERR_ARG
    assert lib.kvg_graft(None, 0, None, 0, -1, 0, 0, None, None) == kvg.KVG_ERR_ARG
    assert lib.kvg_store_prefetch(None, 0, None) == kvg.KVG_ERR_ARG
    ends, nc = (ctypes.c_int32 * 2)(), ctypes.c_int32(-1)
    no_events = (ctypes.c_void_p * 2)()
    assert lib.kvg_graft_chunked(None, 0, None, 0, -1, 0, 0, None, None, None, 2, ends,
                                 ctypes.byref(nc)) == kvg.KVG_ERR_ARG  # no event array
    assert lib.kvg_graft_chunked(None, 0, None, 0, -1, 0, 0, None, None, no_events, 2, ends,
                                 ctypes.byref(nc)) == kvg.KVG_ERR_ARG  # null events
    assert "event" in kvg.kvg_last_error()
    assert lib.kvg_graft_chunked(None, 0, None, 0, -1, 0, 0, None, None, no_events, 0, ends,
                                 ctypes.byref(nc)) == kvg.KVG_ERR_ARG  # max_events < 1
    assert lib.kvg_decode_attention(None, 0, None, 1, None, 4, None, ctypes.c_float(1.0), None) == kvg.KVG_ERR_ARG
    assert lib.kvg_decode_attention_range(None, 0, None, 1, None, 4, ctypes.c_float(1.0), 0, 16, 0, None,
                                          None) == kvg.KVG_ERR_ARG
    assert lib.kvg_decode_state_finish(None, 4, 96, None, None) == kvg.KVG_ERR_ARG
    assert lib.kvg_decode_state_finish(None, -1, 64, None, None) == kvg.KVG_ERR_ARG
    assert lib.kvg_decode_state_finish(None, 0, 64, None, None) == kvg.KVG_OK  # nothing to do


def test_host_checks_reject_bad_fp8_dims_without_a_gpu(lib):
    h = ctypes.c_void_p()
    for ks, vs, dt in [(0.0, 1.0, kvg.KVG_KV_E4M3), (1.0, float("inf"), kvg.KVG_KV_E4M3),
                       (-0.5, 1.0, kvg.KVG_KV_E4M3), (1.0, 1.0, 7)]:
        bad = kvg.make_dims(2, 2, 128, 16, kv_dtype=dt, k_scale=ks, v_scale=vs)
        assert lib.kvg_store_create(ctypes.byref(bad), 0, 1 << 20, 0, ctypes.byref(h)) == kvg.KVG_ERR_ARG
        assert lib.kvg_cache_create(ctypes.byref(bad), 4, 1, 64, 0, ctypes.byref(h)) == kvg.KVG_ERR_ARG


def test_struct_layouts_match_header():
    # field offsets the C side relies on
    assert ctypes.sizeof(kvg.kvg_dims) == 40
    assert (kvg.kvg_dims.kv_dtype.offset, kvg.kvg_dims.k_scale.offset, kvg.kvg_dims.v_scale.offset) == (28, 32, 36)
    assert kvg.kvg_block_info.block_digest.offset == 64
    assert ctypes.sizeof(kvg.kvg_graft_report) == 16 + 4 * kvg.KVG_REPORT_MAX_PAGES
    assert ctypes.sizeof(kvg.kvg_cache_view) == 4 * 8 + 2 * 8 + 4 * 4
