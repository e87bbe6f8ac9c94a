"""The workspace-free attention entry point, for callers that cannot allocate.

ikv_decode_attend_score_static serves callers with no way to get device
scratch memory (a runtime that owns all device memory after start-up, a hook
inside a framework with its own allocator, a loop that cannot take cudaMalloc's
synchronisation).  It keeps its scratch in a fixed array inside the library.
This test calls it through the C ABI twice in a row and checks each result
against the regular entry point given a caller workspace, within the same
tolerances as the other attention tests.  It also checks that shapes needing
more scratch than the array holds are refused.  Collected last on purpose.
"""
import ctypes

import numpy as np
import pytest
import torch

import gen
from harness import fill_device, make_cache, to_device
from paper_2609_03515_gb300 import ikv

pytestmark = pytest.mark.gpu


def _call_static(c, cch, layer, q, out, score, ema, alpha):
    so = ctypes.CDLL(ikv.LIB_PATH)
    so.ikv_decode_attend_score_static.restype = ctypes.c_int32
    so.ikv_decode_attend_score_static.argtypes = [ctypes.POINTER(ikv.ikv_shape), ctypes.POINTER(ikv.ikv_cache),
                                                  ctypes.c_int32, ctypes.c_void_p, ctypes.c_void_p, ctypes.c_void_p,
                                                  ctypes.c_void_p, ctypes.c_float, ctypes.c_void_p]
    shape = c.shape()
    return so.ikv_decode_attend_score_static(ctypes.byref(shape), ctypes.byref(cch), layer, q.data_ptr(),
                                             out.data_ptr(), score.data_ptr(), ema.data_ptr(), alpha,
                                             torch.cuda.current_stream().cuda_stream)


def test_static_scratch_entry_point_matches_workspace_entry_point():
    import __graft_entry__

    __graft_entry__.build()
    w = gen.Workload("na", 2, 3, 32, 8, 128, [1500, 333], 2, dtype=gen.BF16, seed=77, page_size=64)
    u = w.u_table()
    c = make_cache(w, page_perm_seed=4)
    fill_device(c, w, torch.from_numpy(u).cuda())
    cch = c.cache(max(w.prefill))
    ws = torch.empty(ikv.ikv_attend_workspace_size(c.shape(), cch), dtype=torch.uint8, device="cuda")
    assert ws.numel() <= ikv.ikv_static_scratch_bytes()
    rng = np.random.default_rng(8)
    ema0 = torch.from_numpy(rng.random((c.rows, c.cap)).astype(np.float32)).cuda()
    qs = w.queries(1, 3, u)
    for call, layer in enumerate((1, 2)):     # two calls in a row, different layers and queries
        q = to_device(qs[call, layer], w)
        out_a = torch.empty((w.batch, w.q_heads, w.head_dim), dtype=torch.bfloat16, device="cuda")
        out_b = torch.empty_like(out_a)
        sc_a = torch.zeros((c.rows, c.cap), device="cuda")
        sc_b = torch.zeros_like(sc_a)
        em_a, em_b = ema0.clone(), ema0.clone()
        ikv.ikv_decode_attend_score(c.shape(), cch, layer, q, out_a, sc_a, em_a, 0.9, ws, ws.numel())
        assert _call_static(c, cch, layer, q, out_b, sc_b, em_b, 0.9) == ikv.IKV_OK, ikv.ikv_last_error()
        torch.cuda.synchronize()
        assert (out_a.float() - out_b.float()).abs().max().item() < 2e-2
        for b, L in enumerate(w.prefill):
            assert (sc_a[b, :L] - sc_b[b, :L]).abs().max().item() < 2e-5
            assert (em_a[b, :L] - em_b[b, :L]).abs().max().item() < 2e-5
        ema0 = em_b


def test_static_scratch_entry_point_refuses_oversized_shapes():
    w = gen.Workload("big", 8, 1, 32, 8, 128, [40000], 1, dtype=gen.BF16, seed=1, page_size=64)
    c = make_cache(w.with_(batch=1), page_perm_seed=None)
    big = ikv.ikv_shape(8, 1, 32, 8, 128, ikv.IKV_BF16, ikv.IKV_GRAN_SEQ)   # scratch of 8 x 32 x 40k floats
    cch = c.cache(100)
    need = ikv.ikv_attend_workspace_size(big, cch)
    assert need > ikv.ikv_static_scratch_bytes()
    so = ctypes.CDLL(ikv.LIB_PATH)
    so.ikv_decode_attend_score_static.restype = ctypes.c_int32
    t = torch.zeros(16, device="cuda")
    st = so.ikv_decode_attend_score_static(ctypes.byref(big), ctypes.byref(cch), 0, ctypes.c_void_p(t.data_ptr()),
                                           ctypes.c_void_p(t.data_ptr()), None, None, ctypes.c_float(0.9), None)
    assert st == ikv.IKV_ERR_WORKSPACE
    assert "scratch" in ikv.ikv_last_error()
