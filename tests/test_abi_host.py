"""Host-only checks of the C ABI: the library loads, exports every function
include/vp.h declares, and rejects malformed host-visible arguments before
touching the GPU.  No CUDA compute runs here."""

import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _declared():
    names = set()
    for fn in os.listdir(os.path.join(ROOT, "include")):
        if fn.endswith(".h"):
            txt = open(os.path.join(ROOT, "include", fn)).read()
            txt = re.sub(r"/\*.*?\*/", "", txt, flags=re.S)
            names |= set(re.findall(r"\b(vp_\w+)\s*\(", txt))
    return names


def test_header_declares_the_boundary():
    assert {"vp_init", "vp_decode_step", "vp_free", "vp_last_error", "vp_check_errors",
            "vp_max_kept", "vp_decode_gather"} <= _declared()


def test_library_exports_every_declared_symbol(lib):
    for name in _declared():
        assert hasattr(lib.lib, name), name
        assert name in lib.EXPORTED or name.startswith("vp_"), name


def test_init_rejects_bad_shapes_without_a_gpu(lib):
    bad = [
        lib.make_config(0, 8, 2, 64, 10, 20),                # max_batch 0
        lib.make_config(1, 7, 2, 64, 10, 20),                # H % Hkv != 0
        lib.make_config(1, 8, 2, 64, 10, 10),                # max_seq < max_visual + 1
        lib.make_config(1, 8, 2, 64, 10, 20, dtype=7),       # dtype
        lib.make_config(1, 8, 2, 64, 10, 20, paged=1, page_size=12),
    ]
    for cfg in bad:
        h = ctypes.c_void_p()
        assert lib.lib.vp_init(ctypes.byref(cfg), ctypes.byref(h)) == lib.VP_ERR_INVALID_ARG
        assert not h.value
        assert lib.vp_last_error(None)
    unsupported = [lib.make_config(1, 8, 2, 96, 10, 20), lib.make_config(1, 34, 2, 64, 10, 20),
                   lib.make_config(1, 8, 2, 64, 40000, 50000)]
    for cfg in unsupported:
        h = ctypes.c_void_p()
        assert lib.lib.vp_init(ctypes.byref(cfg), ctypes.byref(h)) == lib.VP_ERR_UNSUPPORTED


def test_null_context_and_null_free(lib):
    b = lib.make_budget()
    st = lib.lib.vp_decode_step(None, 1, None, None, None, None, None, ctypes.byref(b), None,
                                None, 0, None, None, None, None)
    assert st == lib.VP_ERR_NOT_INITIALIZED
    assert lib.lib.vp_check_errors(None, None) == lib.VP_ERR_NOT_INITIALIZED
    st = lib.lib.vp_decode_gather(None, 1, None, None, None, None, None, None, 0, None, 0, 0.0, None, None)
    assert st == lib.VP_ERR_NOT_INITIALIZED
    assert lib.lib.vp_set_score_path(None, lib.VP_SCORE_TC) == lib.VP_ERR_NOT_INITIALIZED
    lib.vp_free(None)


@pytest.mark.parametrize("budget,n,want", [
    (dict(), 576, 28),                                          # ADAPTIVE [1%, 5%] -> K_hi
    (dict(), 1296, 64),
    (dict(tau=0.4, r_lo_ppm=50_000, r_hi_ppm=100_000), 1296, 129),
    (dict(r_lo_ppm=0, r_hi_ppm=1_000_000), 100, 100),
    (dict(mode=1, ratio_ppm=500_000), 576, 288),
    (dict(mode=1, ratio_ppm=1), 10, 1),
    (dict(mode=2, fixed_k=256), 576, 256),
    (dict(mode=2, fixed_k=256), 100, 100),
    (dict(mode=3), 576, 576),
    (dict(), 0, 0),
    (dict(mode=4, ratio_ppm=100_000), 576, 576),               # TOP_P may keep every token
    (dict(mode=4, ratio_ppm=100_000, granularity=1), 576, -1),  # TOP_P needs one set per sequence
    (dict(mode=9), 10, -1),
    (dict(tau=0.0), 10, -1),
    (dict(granularity=2), 10, -1),
])
def test_max_kept_is_the_budget_upper_bound(lib, budget, n, want):
    assert lib.vp_max_kept(lib.make_budget(**budget), n) == want


def test_noalloc_rejects_before_any_cuda_call(lib):
    """Malformed host arguments of the allocation-free entry point are refused
    before it touches the GPU, with the reason readable via vp_last_error(NULL)."""
    b = lib.make_budget()
    cfg = lib.make_config(1, 8, 2, 64, 0, 16)
    st = lib.lib.vp_decode_step_noalloc(None, 1, None, None, None, None, None, ctypes.byref(b), None,
                                        None, 0, None, None, None, None)
    assert st == lib.VP_ERR_INVALID_ARG and "cfg" in lib.vp_last_error(None)
    st = lib.lib.vp_decode_step_noalloc(ctypes.byref(cfg), 1, None, None, None, None, None, ctypes.byref(b), None,
                                        None, -1, None, None, None, None)
    assert st == lib.VP_ERR_CAPACITY and "negative" in lib.vp_last_error(None)
    st = lib.lib.vp_decode_step_noalloc(ctypes.byref(cfg), 0, None, None, None, None, None, ctypes.byref(b), None,
                                        None, 0, None, None, None, None)
    assert st == lib.VP_OK and lib.vp_last_error(None) == ""


def test_last_launch_needs_a_context(lib):
    assert lib.lib.vp_last_launch(None, None, None) == lib.VP_ERR_NOT_INITIALIZED
