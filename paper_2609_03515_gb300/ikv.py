"""Thin ctypes binding of libikv.so (argument marshalling only).

Every function keeps the C name and argument order of ``include/ikv.h``; tensor
arguments may be torch tensors (their ``data_ptr()`` is passed) or raw integer
device pointers.  Nothing here computes: every step runs in the CUDA library,
and importing this module fails loudly if the library was not built.
"""
from __future__ import annotations

import ctypes
import os
from typing import Optional

HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(HERE, "libikv.so")

IKV_OK, IKV_ERR_ARG, IKV_ERR_SHAPE, IKV_ERR_ALIGN, IKV_ERR_WORKSPACE, IKV_ERR_UNSUPPORTED, IKV_ERR_CUDA = range(7)
IKV_F32, IKV_BF16 = 0, 1
IKV_GRAN_SEQ, IKV_GRAN_KVHEAD = 0, 1
IKV_COMPACT_STABLE, IKV_COMPACT_HOLEFILL, IKV_COMPACT_STABLE_SHORT = 0, 1, 2
IKV_INIT_ZERO, IKV_INIT_MEAN = 0, 1
IKV_PATH_CUDA_CORE, IKV_PATH_TENSOR_CORE = 0, 1
IKV_AGG_EMA, IKV_AGG_CUMULATIVE, IKV_AGG_SINGLE_STEP = 0, 1, 2
IKV_SCORE_ATTENTION, IKV_SCORE_VNORM, IKV_SCORE_ENTROPY = 0, 1, 2
IKV_EVICT_STEP, IKV_EVICT_LAYER = 0, 1

P = ctypes.c_void_p
I32 = ctypes.c_int32
F32 = ctypes.c_float
SZ = ctypes.c_size_t


class ikv_shape(ctypes.Structure):
    _fields_ = [("batch", I32), ("layers", I32), ("q_heads", I32), ("kv_heads", I32), ("head_dim", I32),
                ("dtype", I32), ("granularity", I32)]


class ikv_cache(ctypes.Structure):
    _fields_ = [("k", P), ("v", P), ("block_table", P), ("num_pages", I32), ("page_size", I32), ("max_pages", I32),
                ("len", P), ("pos", P), ("next_pos", P), ("max_len", I32), ("start", P), ("dead_slots", I32),
                ("vnorm", P), ("pos_cap", I32)]


class ikv_timing(ctypes.Structure):
    _fields_ = [("begin", P), ("append_end", P), ("attend_end", P), ("combine_end", P), ("score_end", P),
                ("select_end", P), ("end", P)]


class ikv_trace(ctypes.Structure):
    _fields_ = [("raw_top", P), ("ema_top", P), ("n_top", P), ("counts", P)]


class ikv_params(ctypes.Structure):
    _fields_ = [("alpha", F32), ("refresh_period", I32), ("score_free", I32), ("budget", P),
                ("layer_eligible", P), ("compact_mode", I32), ("refresh_init", I32),
                ("timing", ctypes.POINTER(ikv_timing)), ("max_holes", I32), ("agg_mode", I32),
                ("scorer", I32), ("evict_mode", I32), ("trace", ctypes.POINTER(ikv_trace)), ("ws_zeroed", I32)]


class IKVError(RuntimeError):
    def __init__(self, status: int, where: str, msg: str):
        super().__init__(f"{where} failed with status {status}: {msg}")
        self.status = status


def _load():
    if not os.path.exists(LIB_PATH):
        raise ImportError(f"libikv.so not built ({LIB_PATH}); run __graft_entry__.build()")
    lib = ctypes.CDLL(LIB_PATH)
    SP, CP, PP = ctypes.POINTER(ikv_shape), ctypes.POINTER(ikv_cache), ctypes.POINTER(ikv_params)
    sigs = {
        "ikv_last_error": ([], ctypes.c_char_p),
        "ikv_launch_count": ([], ctypes.c_int64),
        "ikv_device_status": ([ctypes.POINTER(ctypes.c_uint32)], I32),
        "ikv_test_stall_next_attention": ([], I32),
        "ikv_attend_path": ([SP, CP, ctypes.POINTER(I32)], I32),
        "ikv_attend_plan": ([SP, CP, I32, I32] + [ctypes.POINTER(I32)] * 5, I32),
        "ikv_attend_workspace_size": ([SP, CP, ctypes.POINTER(SZ)], I32),
        "ikv_decode_attend_score": ([SP, CP, I32, P, P, P, P, F32, P, SZ, P], I32),
        "ikv_static_scratch_bytes": ([], SZ),
        "ikv_decode_attend_score_static": ([SP, CP, I32, P, P, P, P, F32, P], I32),
        "ikv_ema_update": ([I32, I32, P, P, P, I32, F32, P], I32),
        "ikv_value_norms": ([SP, CP, P], I32),
        "ikv_select_budget": ([I32, I32, P, P, I32, P, P, P, P, P], I32),
        "ikv_compact_workspace_size": ([SP, CP, I32, ctypes.POINTER(SZ)], I32),
        "ikv_compact_kv": ([SP, CP, P, P, P, I32, P, SZ, P], I32),
        "ikv_append_token": ([SP, CP, P, P, P, I32, P, SZ, P], I32),
        "ikv_step_workspace_size": ([SP, CP, ctypes.POINTER(SZ)], I32),
        "ikv_step": ([SP, PP, CP, P, I32, P, P, P, P, P, SZ, P], I32),
        "ikv_step_begin": ([SP, PP, CP, P, I32, P, SZ, P], I32),
        "ikv_step_layer": ([SP, PP, CP, P, I32, I32, P, P, P, P, P, SZ, P], I32),
        "ikv_step_end": ([SP, PP, CP, P, I32, P, SZ, P], I32),
    }
    for name, (args, res) in sigs.items():
        f = getattr(lib, name)
        f.argtypes = args
        f.restype = res
    return lib


_lib = _load()


def _p(x) -> Optional[int]:
    if x is None:
        return None
    if isinstance(x, int):
        return x
    return x.data_ptr()


def _stream(s) -> Optional[int]:
    if s is None:
        return None
    if isinstance(s, int):
        return s
    return s.cuda_stream


def _check(status: int, where: str) -> None:
    if status != IKV_OK:
        raise IKVError(status, where, _lib.ikv_last_error().decode())


def ikv_last_error() -> str:
    return _lib.ikv_last_error().decode()


def ikv_launch_count() -> int:
    return int(_lib.ikv_launch_count())


def ikv_device_status() -> int:
    v = ctypes.c_uint32(0)
    _check(_lib.ikv_device_status(ctypes.byref(v)), "ikv_device_status")
    return int(v.value)


def ikv_test_stall_next_attention() -> None:
    _check(_lib.ikv_test_stall_next_attention(), "ikv_test_stall_next_attention")


def ikv_attend_path(shape: ikv_shape, cache: ikv_cache) -> int:
    v = I32(0)
    _check(_lib.ikv_attend_path(ctypes.byref(shape), ctypes.byref(cache), ctypes.byref(v)), "ikv_attend_path")
    return int(v.value)


def ikv_attend_plan(shape: ikv_shape, cache: ikv_cache, n_layers: int, sms: int = 0) -> dict:
    """The partition of one attention launch over n_layers layers (see include/ikv.h)."""
    v = [I32(0) for _ in range(5)]
    _check(_lib.ikv_attend_plan(ctypes.byref(shape), ctypes.byref(cache), n_layers, sms,
                                *[ctypes.byref(x) for x in v]), "ikv_attend_plan")
    keys = ("path", "chunk_tokens", "n_chunks", "passes", "group_sums")
    return {k: int(x.value) for k, x in zip(keys, v)}


def ikv_attend_workspace_size(shape: ikv_shape, cache: ikv_cache) -> int:
    n = SZ(0)
    _check(_lib.ikv_attend_workspace_size(ctypes.byref(shape), ctypes.byref(cache), ctypes.byref(n)),
           "ikv_attend_workspace_size")
    return n.value


def ikv_decode_attend_score(shape, cache, layer, q, out, score, ema, alpha, ws, ws_bytes, stream=None) -> None:
    _check(_lib.ikv_decode_attend_score(ctypes.byref(shape), ctypes.byref(cache), layer, _p(q), _p(out), _p(score),
                                        _p(ema), alpha, _p(ws), ws_bytes, _stream(stream)), "ikv_decode_attend_score")


def ikv_static_scratch_bytes() -> int:
    return int(_lib.ikv_static_scratch_bytes())


def ikv_decode_attend_score_static(shape, cache, layer, q, out, score, ema, alpha, stream=None) -> None:
    _check(_lib.ikv_decode_attend_score_static(ctypes.byref(shape), ctypes.byref(cache), layer, _p(q), _p(out),
                                               _p(score), _p(ema), alpha, _stream(stream)),
           "ikv_decode_attend_score_static")


def ikv_ema_update(rows, cap, ema, score, length, rows_per_seq, alpha, stream=None) -> None:
    _check(_lib.ikv_ema_update(rows, cap, _p(ema), _p(score), _p(length), rows_per_seq, alpha, _stream(stream)),
           "ikv_ema_update")


def ikv_value_norms(shape, cache, stream=None) -> None:
    _check(_lib.ikv_value_norms(ctypes.byref(shape), ctypes.byref(cache), _stream(stream)), "ikv_value_norms")


def ikv_select_budget(rows, cap, util, length, rows_per_seq, budget, pos, keep, keep_len, stream=None) -> None:
    _check(_lib.ikv_select_budget(rows, cap, _p(util), _p(length), rows_per_seq, _p(budget), _p(pos), _p(keep),
                                  _p(keep_len), _stream(stream)), "ikv_select_budget")


def ikv_compact_workspace_size(shape, cache, mode) -> int:
    n = SZ(0)
    _check(_lib.ikv_compact_workspace_size(ctypes.byref(shape), ctypes.byref(cache), mode, ctypes.byref(n)),
           "ikv_compact_workspace_size")
    return n.value


def ikv_compact_kv(shape, cache, keep, keep_len, ema, mode, ws, ws_bytes, stream=None) -> None:
    _check(_lib.ikv_compact_kv(ctypes.byref(shape), ctypes.byref(cache), _p(keep), _p(keep_len), _p(ema), mode,
                               _p(ws), ws_bytes, _stream(stream)), "ikv_compact_kv")


def ikv_append_token(shape, cache, k_new, v_new, ema, init_mean, ws, ws_bytes, stream=None) -> None:
    _check(_lib.ikv_append_token(ctypes.byref(shape), ctypes.byref(cache), _p(k_new), _p(v_new), _p(ema), init_mean,
                                 _p(ws), ws_bytes, _stream(stream)), "ikv_append_token")


def ikv_step_workspace_size(shape, cache) -> int:
    n = SZ(0)
    _check(_lib.ikv_step_workspace_size(ctypes.byref(shape), ctypes.byref(cache), ctypes.byref(n)),
           "ikv_step_workspace_size")
    return n.value


def ikv_step(shape, params, cache, ema, t, q, k_new, v_new, out, ws, ws_bytes, stream=None) -> None:
    _check(_lib.ikv_step(ctypes.byref(shape), ctypes.byref(params), ctypes.byref(cache), _p(ema), t, _p(q), _p(k_new),
                         _p(v_new), _p(out), _p(ws), ws_bytes, _stream(stream)), "ikv_step")


def ikv_step_begin(shape, params, cache, ema, t, ws, ws_bytes, stream=None) -> None:
    _check(_lib.ikv_step_begin(ctypes.byref(shape), ctypes.byref(params), ctypes.byref(cache), _p(ema), t, _p(ws),
                               ws_bytes, _stream(stream)), "ikv_step_begin")


def ikv_step_layer(shape, params, cache, ema, t, layer, q, k_new, v_new, out, ws, ws_bytes, stream=None) -> None:
    _check(_lib.ikv_step_layer(ctypes.byref(shape), ctypes.byref(params), ctypes.byref(cache), _p(ema), t, layer,
                               _p(q), _p(k_new), _p(v_new), _p(out), _p(ws), ws_bytes, _stream(stream)),
           "ikv_step_layer")


def ikv_step_end(shape, params, cache, ema, t, ws, ws_bytes, stream=None) -> None:
    _check(_lib.ikv_step_end(ctypes.byref(shape), ctypes.byref(params), ctypes.byref(cache), _p(ema), t, _p(ws),
                             ws_bytes, _stream(stream)), "ikv_step_end")


def raw_status(fn_name: str, *args) -> int:
    """Call an entry point and return its raw status (used by argument-check tests)."""
    return int(getattr(_lib, fn_name)(*args))
