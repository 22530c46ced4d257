"""Python binding of libvp (include/vp.h): the same entry points, marshalled
with ctypes.  Every step of the decode path runs in the library's CUDA
kernels; this module only converts torch tensors to raw device pointers.

Importing it loads ``libvp.so`` from this package directory and raises if the
library has not been built (``python -c "import __graft_entry__ as g; g.build()"``):
there is no fallback implementation.
"""

from __future__ import annotations

import ctypes
import os

_LIB_PATH = os.path.join(os.path.dirname(os.path.abspath(__file__)), "libvp.so")
if not os.path.exists(_LIB_PATH):
    raise ImportError(f"{_LIB_PATH} is missing: build it with paper_2605_31457_gb300.build.build()")
lib = ctypes.CDLL(_LIB_PATH)

# vp_status
VP_OK = 0
VP_ERR_INVALID_ARG = 1
VP_ERR_UNSUPPORTED = 2
VP_ERR_CAPACITY = 3
VP_ERR_NOT_INITIALIZED = 4
VP_ERR_CUDA = 5
VP_ERR_DEVICE_PRECOND = 6
# vp_dtype
VP_BF16 = 0
VP_FP32 = 1
# vp_budget_mode
VP_ADAPTIVE = 0
VP_FIXED_RATIO = 1
VP_FIXED_K = 2
VP_DENSE = 3
VP_TOP_P = 4

VP_SCORE_AUTO = 0
VP_SCORE_MMA = 1
VP_SCORE_TC = 2

EXPORTED = ("vp_init", "vp_decode_step", "vp_max_kept", "vp_last_error", "vp_check_errors",
            "vp_timing_enable", "vp_timing_read", "vp_free", "vp_decode_step_noalloc", "vp_decode_gather",
            "vp_set_diagnostics", "vp_set_score_path", "vp_compact_kv", "vp_last_launch")
VP_NOALLOC_SCRATCH_BYTES = 16 << 20


class vp_config(ctypes.Structure):
    _fields_ = [("max_batch", ctypes.c_int32), ("num_q_heads", ctypes.c_int32),
                ("num_kv_heads", ctypes.c_int32), ("head_dim", ctypes.c_int32),
                ("max_visual", ctypes.c_int32), ("max_seq", ctypes.c_int32),
                ("dtype", ctypes.c_int), ("paged", ctypes.c_int32), ("page_size", ctypes.c_int32)]


class vp_kv(ctypes.Structure):
    _fields_ = [("data", ctypes.c_void_p), ("stride_b", ctypes.c_int64), ("stride_h", ctypes.c_int64),
                ("stride_t", ctypes.c_int64), ("block_table", ctypes.c_void_p),
                ("max_pages", ctypes.c_int32), ("num_pages", ctypes.c_int32)]


class vp_span(ctypes.Structure):
    _fields_ = [("vis_start", ctypes.c_void_p), ("vis_len", ctypes.c_void_p)]


class vp_budget(ctypes.Structure):
    _fields_ = [("mode", ctypes.c_int32), ("tau", ctypes.c_float), ("scale", ctypes.c_float),
                ("r_lo_ppm", ctypes.c_int32), ("r_hi_ppm", ctypes.c_int32),
                ("ratio_ppm", ctypes.c_int32), ("fixed_k", ctypes.c_int32),
                ("granularity", ctypes.c_int32)]


_P = ctypes.c_void_p
lib.vp_init.argtypes = [ctypes.POINTER(vp_config), ctypes.POINTER(_P)]
lib.vp_init.restype = ctypes.c_int
lib.vp_decode_step.argtypes = [_P, ctypes.c_int32, _P, ctypes.POINTER(vp_kv), ctypes.POINTER(vp_kv),
                               ctypes.POINTER(vp_span), _P, ctypes.POINTER(vp_budget), _P,
                               _P, ctypes.c_int32, _P, _P, _P, _P]
lib.vp_decode_step.restype = ctypes.c_int
lib.vp_decode_gather.argtypes = [_P, ctypes.c_int32, _P, ctypes.POINTER(vp_kv), ctypes.POINTER(vp_kv),
                                 ctypes.POINTER(vp_span), _P, _P, ctypes.c_int32, _P, ctypes.c_int32,
                                 ctypes.c_float, _P, _P]
lib.vp_decode_gather.restype = ctypes.c_int
lib.vp_set_diagnostics.argtypes = [_P, ctypes.c_float, _P, _P]
lib.vp_set_diagnostics.restype = ctypes.c_int
lib.vp_compact_kv.argtypes = [_P, ctypes.c_int32, ctypes.POINTER(vp_kv), ctypes.POINTER(vp_kv),
                              ctypes.POINTER(vp_span), _P, _P, ctypes.c_int32, _P, _P]
lib.vp_compact_kv.restype = ctypes.c_int
lib.vp_set_score_path.argtypes = [_P, ctypes.c_int32]
lib.vp_set_score_path.restype = ctypes.c_int
lib.vp_last_launch.argtypes = [_P, ctypes.POINTER(ctypes.c_int32), ctypes.POINTER(ctypes.c_int32)]
lib.vp_last_launch.restype = ctypes.c_int
lib.vp_max_kept.argtypes = [ctypes.POINTER(vp_budget), ctypes.c_int32]
lib.vp_max_kept.restype = ctypes.c_int32
lib.vp_last_error.argtypes = [_P]
lib.vp_last_error.restype = ctypes.c_char_p
lib.vp_check_errors.argtypes = [_P, _P]
lib.vp_check_errors.restype = ctypes.c_int
lib.vp_timing_enable.argtypes = [_P, ctypes.c_int32]
lib.vp_timing_enable.restype = ctypes.c_int
lib.vp_timing_read.argtypes = [_P, ctypes.POINTER(ctypes.c_float), ctypes.c_int32, ctypes.POINTER(ctypes.c_int32)]
lib.vp_timing_read.restype = ctypes.c_int
lib.vp_decode_step_noalloc.argtypes = [ctypes.POINTER(vp_config), ctypes.c_int32, _P, ctypes.POINTER(vp_kv),
                                       ctypes.POINTER(vp_kv), ctypes.POINTER(vp_span), _P,
                                       ctypes.POINTER(vp_budget), _P, _P, ctypes.c_int32, _P, _P, _P, _P]
lib.vp_decode_step_noalloc.restype = ctypes.c_int
lib.vp_free.argtypes = [_P]
lib.vp_free.restype = None


class VPError(RuntimeError):
    def __init__(self, status, msg):
        super().__init__(f"vp status {status}: {msg}")
        self.status = status


def _ptr(t):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _check(status, ctx):
    if status != VP_OK:
        raise VPError(status, vp_last_error(ctx))
    return status


# ---------------------------------------------------------------- entry points

def vp_init(cfg: vp_config):
    """Creates a context; returns its handle (raises VPError on failure)."""
    h = _P()
    _check(lib.vp_init(ctypes.byref(cfg), ctypes.byref(h)), None)
    return h


def vp_decode_step(ctx, batch, q, k_cache: vp_kv, v_cache: vp_kv, visual_span: vp_span, text_len,
                   budget: vp_budget, out, kept_idx, kept_cap, kept_count, mass, mass_stats=None,
                   stream=None, check=True):
    """Enqueues one decode step.  Tensors are torch CUDA tensors; ``stream``
    is a torch.cuda.Stream or raw handle (default: torch's current stream)."""
    if stream is None:
        import torch
        stream = torch.cuda.current_stream().cuda_stream
    elif hasattr(stream, "cuda_stream"):
        stream = stream.cuda_stream
    st = lib.vp_decode_step(ctx, int(batch), _ptr(q), ctypes.byref(k_cache), ctypes.byref(v_cache),
                            ctypes.byref(visual_span), _ptr(text_len), ctypes.byref(budget), _ptr(out),
                            _ptr(kept_idx), int(kept_cap), _ptr(kept_count), _ptr(mass),
                            _ptr(mass_stats), ctypes.c_void_p(stream))
    return _check(st, ctx) if check else st


def vp_decode_gather(ctx, batch, q, k_cache: vp_kv, v_cache: vp_kv, visual_span: vp_span, text_len,
                     kept_idx, kept_cap, kept_count, out, granularity=0, scale=0.0, stream=None, check=True):
    """Enqueues the attention of a layer after the anchor layer over every text
    token and the anchor's kept set (kept_idx / kept_count as vp_decode_step
    wrote them).  Tensors are torch CUDA tensors."""
    if stream is None:
        import torch
        stream = torch.cuda.current_stream().cuda_stream
    elif hasattr(stream, "cuda_stream"):
        stream = stream.cuda_stream
    st = lib.vp_decode_gather(ctx, int(batch), _ptr(q), ctypes.byref(k_cache), ctypes.byref(v_cache),
                              ctypes.byref(visual_span), _ptr(text_len), _ptr(kept_idx), int(kept_cap),
                              _ptr(kept_count), int(granularity), float(scale), _ptr(out), ctypes.c_void_p(stream))
    return _check(st, ctx) if check else st


def vp_compact_kv(ctx, batch, src: vp_kv, dst: vp_kv, visual_span: vp_span, text_len, kept_idx, kept_cap,
                  kept_count, stream=None, check=True):
    """Writes into ``dst`` (contiguous) the cache ``src`` with only the kept
    visual rows (FastV prefill pruning followed by VisionPulse)."""
    if stream is None:
        import torch
        stream = torch.cuda.current_stream().cuda_stream
    elif hasattr(stream, "cuda_stream"):
        stream = stream.cuda_stream
    st = lib.vp_compact_kv(ctx, int(batch), ctypes.byref(src), ctypes.byref(dst), ctypes.byref(visual_span),
                           _ptr(text_len), _ptr(kept_idx), int(kept_cap), _ptr(kept_count), ctypes.c_void_p(stream))
    return _check(st, ctx) if check else st


def vp_set_score_path(ctx, path):
    """Score kernel of later vp_decode_step calls: VP_SCORE_AUTO, VP_SCORE_MMA
    or VP_SCORE_TC."""
    return _check(lib.vp_set_score_path(ctx, int(path)), ctx)


def vp_set_diagnostics(ctx, delta, n_act=None, active_bits=None):
    """Turns on (or off, with both arrays None) the N_act(delta) count and the
    OR-accumulated activity bits of later vp_decode_step calls."""
    return _check(lib.vp_set_diagnostics(ctx, float(delta), _ptr(n_act), _ptr(active_bits)), ctx)


def vp_last_launch(ctx):
    """(score kernel, kernels enqueued) of the last decode call on ctx:
    VP_SCORE_TC or VP_SCORE_MMA, and the launch count."""
    path, n = ctypes.c_int32(0), ctypes.c_int32(0)
    _check(lib.vp_last_launch(ctx, ctypes.byref(path), ctypes.byref(n)), ctx)
    return path.value, n.value


def vp_max_kept(budget: vp_budget, n_visual: int) -> int:
    return int(lib.vp_max_kept(ctypes.byref(budget), int(n_visual)))


def vp_last_error(ctx) -> str:
    r = lib.vp_last_error(ctx)
    return r.decode() if r else ""


def vp_check_errors(ctx, stream=None, check=True):
    if stream is None:
        import torch
        stream = torch.cuda.current_stream().cuda_stream
    elif hasattr(stream, "cuda_stream"):
        stream = stream.cuda_stream
    st = lib.vp_check_errors(ctx, ctypes.c_void_p(stream))
    return _check(st, ctx) if check else st


def vp_timing_enable(ctx, slots: int):
    return _check(lib.vp_timing_enable(ctx, int(slots)), ctx)


def vp_timing_read(ctx, max_slots: int):
    """Returns a list of (score_ms, select_ms, gather_ms) per recorded slot."""
    buf = (ctypes.c_float * (3 * max(int(max_slots), 1)))()
    n = ctypes.c_int32(0)
    _check(lib.vp_timing_read(ctx, buf, int(max_slots), ctypes.byref(n)), ctx)
    return [(buf[3 * i], buf[3 * i + 1], buf[3 * i + 2]) for i in range(n.value)]


def vp_free(ctx):
    lib.vp_free(ctx)


def vp_decode_step_noalloc(cfg: vp_config, batch, q, k_cache: vp_kv, v_cache: vp_kv, visual_span: vp_span,
                           text_len, budget: vp_budget, out, kept_idx, kept_cap, kept_count, mass,
                           mass_stats=None, stream=None):
    """The decode step without a context or any device allocation (scratch in
    the library's fixed device array).  For callers that cannot allocate on
    their inference path.  Returns the raw vp_status (0 = VP_OK)."""
    if stream is None:
        import torch
        stream = torch.cuda.current_stream().cuda_stream
    elif hasattr(stream, "cuda_stream"):
        stream = stream.cuda_stream
    return lib.vp_decode_step_noalloc(ctypes.byref(cfg), int(batch), _ptr(q), ctypes.byref(k_cache),
                                      ctypes.byref(v_cache), ctypes.byref(visual_span), _ptr(text_len),
                                      ctypes.byref(budget), _ptr(out), _ptr(kept_idx), int(kept_cap),
                                      _ptr(kept_count), _ptr(mass), _ptr(mass_stats), ctypes.c_void_p(stream))


# ------------------------------------------------------- marshalling helpers

def make_config(max_batch, num_q_heads, num_kv_heads, head_dim, max_visual, max_seq,
                dtype=VP_BF16, paged=0, page_size=16) -> vp_config:
    return vp_config(max_batch, num_q_heads, num_kv_heads, head_dim, max_visual, max_seq,
                     dtype, paged, page_size)


def kv_contiguous(t) -> vp_kv:
    """A [B, Hkv, T, D] tensor (any strides with a contiguous last axis)."""
    assert t.dim() == 4 and t.stride(3) == 1
    return vp_kv(t.data_ptr(), t.stride(0), t.stride(1), t.stride(2), None, 0, 0)


def kv_paged(pool, block_table) -> vp_kv:
    """A [pages, Hkv, page_size, D] pool plus an int32 [B, max_pages] block table."""
    assert pool.dim() == 4 and pool.stride(3) == 1 and block_table.dim() == 2
    return vp_kv(pool.data_ptr(), pool.stride(0), pool.stride(1), pool.stride(2),
                 block_table.data_ptr(), block_table.shape[1], pool.shape[0])


def span(vis_start, vis_len) -> vp_span:
    return vp_span(vis_start.data_ptr(), vis_len.data_ptr())


def make_budget(mode=VP_ADAPTIVE, tau=0.1, scale=0.0, r_lo_ppm=10_000, r_hi_ppm=50_000,
                ratio_ppm=0, fixed_k=0, granularity=0) -> vp_budget:
    return vp_budget(mode, tau, scale, r_lo_ppm, r_hi_ppm, ratio_ppm, fixed_k, granularity)
