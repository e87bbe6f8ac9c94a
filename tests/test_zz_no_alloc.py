"""The workspace-free attention entry point, for callers that cannot allocate.

ikv_decode_attend_score_static serves callers with no way to get device
scratch memory (a runtime that owns all device memory after start-up, a hook
inside a framework with its own allocator, a loop that cannot take cudaMalloc's
synchronisation).  It keeps its scratch in a fixed array inside the library.
These tests call it through the C ABI several times in a row, on the tensor-core
attention path and on the CUDA-core one, and check each result
  - bit for bit against the regular entry point given a caller workspace (both
    run the same kernels on the same plan, so any difference is a scratch fault),
  - against the CPU oracle at the tolerances of the other attention tests,
and that the calls leave the device's free memory unchanged.  They also check
that shapes needing more scratch than the array holds are refused.  Collected
last on purpose.
"""
import ctypes

import numpy as np
import pytest
import torch

import gen
import oracle as O
from harness import as_f64, fill_device, make_cache, to_device
from paper_2609_03515_gb300 import ikv

pytestmark = pytest.mark.gpu


def _static_fn():
    so = ctypes.CDLL(ikv.LIB_PATH)
    f = so.ikv_decode_attend_score_static
    f.restype = ctypes.c_int32
    f.argtypes = [ctypes.POINTER(ikv.ikv_shape), ctypes.POINTER(ikv.ikv_cache), ctypes.c_int32, ctypes.c_void_p,
                  ctypes.c_void_p, ctypes.c_void_p, ctypes.c_void_p, ctypes.c_float, ctypes.c_void_p]
    return f


def _call_static(f, c, cch, layer, q, out, score, ema, alpha):
    shape = c.shape()
    return f(ctypes.byref(shape), ctypes.byref(cch), layer, q.data_ptr(), out.data_ptr(), score.data_ptr(),
             ema.data_ptr(), alpha, torch.cuda.current_stream().cuda_stream)


# (page size, lengths): page 64 runs the tensor-core kernel (several chunks per unit for
# the longer sequence), page 48 the CUDA-core split kernel and its combine
@pytest.mark.parametrize("ps,lens", [(64, [1500, 333]), (48, [700, 1501])], ids=["tensor_core", "cuda_core"])
def test_static_scratch_entry_point_matches_workspace_entry_point_and_oracle(ps, lens):
    import __graft_entry__

    __graft_entry__.build()
    f = _static_fn()
    w = gen.Workload("na", len(lens), 3, 32, 8, 128, lens, 2, dtype=gen.BF16, seed=77, page_size=ps)
    u = w.u_table()
    c = make_cache(w, page_perm_seed=4)
    fill_device(c, w, torch.from_numpy(u).cuda())
    cch = c.cache(max(w.prefill))
    want_path = ikv.IKV_PATH_TENSOR_CORE if ps == 64 else ikv.IKV_PATH_CUDA_CORE
    assert ikv.ikv_attend_path(c.shape(), cch) == want_path
    ws = torch.empty(ikv.ikv_attend_workspace_size(c.shape(), cch), dtype=torch.uint8, device="cuda")
    assert ws.numel() <= ikv.ikv_static_scratch_bytes()
    rng = np.random.default_rng(8)
    ema0 = torch.from_numpy(rng.random((c.rows, c.cap)).astype(np.float32)).cuda()
    qs = w.queries(1, 3, u)
    alpha = 0.9
    # every buffer of the calls exists before the free-memory reading; calls in a row on
    # different layers and queries
    calls = []
    for call, layer in ((0, 1), (1, 2), (1, 1)):
        calls.append(dict(layer=layer, q_h=qs[call, layer], q=to_device(qs[call, layer], w),
                          out_a=torch.empty((w.batch, w.q_heads, w.head_dim), dtype=torch.bfloat16, device="cuda"),
                          out_b=torch.empty((w.batch, w.q_heads, w.head_dim), dtype=torch.bfloat16, device="cuda"),
                          sc_a=torch.zeros((c.rows, c.cap), device="cuda"),
                          sc_b=torch.zeros((c.rows, c.cap), device="cuda")))
    em_a, em_b = ema0.clone(), ema0.clone()
    # The first call sets the array's address up on this device.  The free-memory reading is
    # taken once the first round of calls and checks has run (every kernel and module they
    # use is loaded by then) and must not move afterwards.
    free0 = None
    m_prev = ema0.double().cpu().numpy()
    for i, k in enumerate(calls):
        ikv.ikv_decode_attend_score(c.shape(), cch, k["layer"], k["q"], k["out_a"], k["sc_a"], em_a, alpha, ws,
                                    ws.numel())
        assert _call_static(f, c, cch, k["layer"], k["q"], k["out_b"], k["sc_b"], em_b, alpha) == ikv.IKV_OK, \
            ikv.ikv_last_error()
        torch.cuda.synchronize()
        if free0 is not None:
            assert torch.cuda.mem_get_info()[0] == free0     # the static calls allocated nothing
        assert ikv.ikv_device_status() == 0
        # bit for bit the workspace entry point's results
        assert torch.equal(k["out_a"], k["out_b"])
        assert torch.equal(k["sc_a"], k["sc_b"])
        assert torch.equal(em_a, em_b)
        # and the oracle's, at the attention tests' tolerances
        q64 = as_f64(k["q_h"], w)
        em_h = em_b.cpu().numpy()
        for b, L in enumerate(w.prefill):
            kk, vv = w.kv_block(b, k["layer"], 0, L, u)
            a, o = O.last_query_attention(q64[b], [x.astype(np.float64) for x in kk],
                                          [x.astype(np.float64) for x in vv])
            assert np.max(np.abs(k["out_b"][b].cpu().float().numpy() - o)) < 2e-2
            s = O.pooled_score(a, O.GRAN_SEQ, w.kv_heads)[0]
            assert np.max(np.abs(k["sc_b"][b, :L].cpu().numpy() - s)) < 2e-5
            want = O.ema_update(m_prev[b, :L], s, alpha)
            assert np.max(np.abs(em_h[b, :L] - want)) < 2e-5
            m_prev[b, :L] = em_h[b, :L]
        if free0 is None:
            torch.cuda.synchronize()
            free0 = torch.cuda.mem_get_info()[0]


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
