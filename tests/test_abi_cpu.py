"""C-ABI checks that need no GPU: the library loads, exports every entry point
declared in include/*.h, and rejects bad arguments on the host before any launch."""
import ctypes
import glob
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def lib():
    import __graft_entry__

    __graft_entry__.build()
    from paper_2609_03515_gb300 import ikv

    return ikv


def declared_symbols():
    names = set()
    for h in glob.glob(os.path.join(ROOT, "include", "*.h")):
        src = open(h).read()
        src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
        for m in re.finditer(r"^\s*(?:const\s+)?[A-Za-z_][A-Za-z0-9_]*\s*\*?\s*(ikv_[a-z0-9_]+)\s*\(", src, re.M):
            names.add(m.group(1))
    return sorted(names)


def test_header_declares_the_entry_points():
    names = declared_symbols()
    for must in ("ikv_decode_attend_score", "ikv_ema_update", "ikv_select_budget", "ikv_compact_kv", "ikv_step"):
        assert must in names


def test_library_exports_every_declared_symbol(lib):
    so = ctypes.CDLL(lib.LIB_PATH)
    missing = [n for n in declared_symbols() if not hasattr(so, n)]
    assert not missing, missing


def _shape(lib, **kw):
    d = dict(batch=1, layers=2, q_heads=4, kv_heads=2, head_dim=64, dtype=lib.IKV_F32, granularity=lib.IKV_GRAN_SEQ)
    d.update(kw)
    return lib.ikv_shape(**d)


def _cache(lib, **kw):
    d = dict(k=16, v=16, block_table=16, num_pages=4, page_size=64, max_pages=4, len=16, pos=16, next_pos=16,
             max_len=100)
    d.update(kw)
    return lib.ikv_cache(**d)


def test_argument_checks_fail_before_launch(lib):
    n = lib.SZ(0)
    bad = [
        (_shape(lib, head_dim=96), _cache(lib), lib.IKV_ERR_UNSUPPORTED),
        (_shape(lib, q_heads=6, kv_heads=2), _cache(lib), lib.IKV_ERR_UNSUPPORTED),   # group 3
        (_shape(lib, q_heads=5, kv_heads=2), _cache(lib), lib.IKV_ERR_SHAPE),
        (_shape(lib, dtype=7), _cache(lib), lib.IKV_ERR_ARG),
        (_shape(lib), _cache(lib, k=0), lib.IKV_ERR_ARG),
        (_shape(lib), _cache(lib, k=8), lib.IKV_ERR_ALIGN),
        (_shape(lib), _cache(lib, max_len=10_000), lib.IKV_ERR_SHAPE),
        (_shape(lib), _cache(lib, page_size=0), lib.IKV_ERR_SHAPE),
    ]
    for shp, cch, want in bad:
        st = lib.raw_status("ikv_step_workspace_size", ctypes.byref(shp), ctypes.byref(cch), ctypes.byref(n))
        assert st == want, (st, want, lib.ikv_last_error())
        assert lib.ikv_last_error() != ""
    st = lib.raw_status("ikv_step_workspace_size", ctypes.byref(_shape(lib)), ctypes.byref(_cache(lib)),
                        ctypes.byref(n))
    assert st == lib.IKV_OK and n.value > 0


def test_step_rejects_bad_schedule_and_workspace(lib):
    shp, cch = _shape(lib), _cache(lib)
    p = lib.ikv_params()
    p.alpha, p.refresh_period, p.budget = 0.9, 1, 16
    args = lambda t, ws, wsb: (ctypes.byref(shp), ctypes.byref(p), ctypes.byref(cch), 16, t, 16, 16, 16, 16, ws, wsb,
                               None)
    assert lib.raw_status("ikv_step", *args(0, 16, 1 << 40)) == lib.IKV_ERR_ARG          # t is 1-based
    assert lib.raw_status("ikv_step", *args(1, 0, 0)) == lib.IKV_ERR_WORKSPACE
    assert lib.raw_status("ikv_step", *args(1, 16, 10)) == lib.IKV_ERR_WORKSPACE
    p.refresh_period = 0
    assert lib.raw_status("ikv_step", *args(1, 16, 1 << 40)) == lib.IKV_ERR_ARG
    p.refresh_period, p.alpha = 1, 1.5
    assert lib.raw_status("ikv_step", *args(1, 16, 1 << 40)) == lib.IKV_ERR_ARG
    p.alpha, p.compact_mode = 0.9, 9
    assert lib.raw_status("ikv_step", *args(1, 16, 1 << 40)) == lib.IKV_ERR_ARG
    p.compact_mode = 0
    full = _cache(lib, max_len=256)  # no free slot for the append
    assert lib.raw_status("ikv_step", ctypes.byref(shp), ctypes.byref(p), ctypes.byref(full), 16, 1, 16, 16, 16, 16,
                          16, 1 << 40, None) == lib.IKV_ERR_SHAPE


def test_split_step_rejects_bad_arguments(lib):
    """ikv_step_begin / _layer / _end check what ikv_step checks, plus the layer index."""
    shp, cch = _shape(lib), _cache(lib)
    p = lib.ikv_params()
    p.alpha, p.refresh_period, p.budget = 0.9, 1, 16
    P, S, C = ctypes.byref(p), ctypes.byref(shp), ctypes.byref(cch)
    big = 1 << 40
    assert lib.raw_status("ikv_step_begin", S, P, C, 16, 0, 16, big, None) == lib.IKV_ERR_ARG    # t is 1-based
    assert lib.raw_status("ikv_step_begin", S, P, C, None, 1, 16, big, None) == lib.IKV_ERR_ARG  # no ema
    assert lib.raw_status("ikv_step_begin", S, P, C, 16, 1, 16, 10, None) == lib.IKV_ERR_WORKSPACE
    assert lib.raw_status("ikv_step_end", S, P, C, 16, 1, 0, 0, None) == lib.IKV_ERR_WORKSPACE
    layer = lambda l, q=16, kn=16, out=16: lib.raw_status("ikv_step_layer", S, P, C, 16, 1, l, q, kn, 16, out, 16,
                                                          big, None)
    assert layer(2) == lib.IKV_ERR_ARG      # two layers: 0 and 1
    assert layer(-1) == lib.IKV_ERR_ARG
    assert layer(0, q=None) == lib.IKV_ERR_ARG
    assert layer(0, kn=None) == lib.IKV_ERR_ARG
    assert layer(1, out=8) == lib.IKV_ERR_ALIGN
    p.refresh_period = 0
    for fn in ("ikv_step_begin", "ikv_step_end"):
        assert lib.raw_status(fn, S, P, C, 16, 1, 16, big, None) == lib.IKV_ERR_ARG
    assert layer(0) == lib.IKV_ERR_ARG
    p.refresh_period = 1
    full = _cache(lib, max_len=256)  # no free slot for the new token
    assert lib.raw_status("ikv_step_begin", S, P, ctypes.byref(full), 16, 1, 16, big, None) == lib.IKV_ERR_SHAPE


def test_per_layer_eviction_arguments(lib):
    """IKV_EVICT_LAYER supports one configuration of the other options; the rest are refused
    on the host."""
    shp = _shape(lib)
    cch = _cache(lib, pos_cap=200)
    p = lib.ikv_params()
    p.alpha, p.refresh_period, p.budget, p.evict_mode = 0.9, 1, 16, lib.IKV_EVICT_LAYER
    call = lambda s, c: lib.raw_status("ikv_step", ctypes.byref(s), ctypes.byref(p), ctypes.byref(c), 16, 1, 16, 16,
                                       16, 16, 16, 1 << 40, None)
    p.max_holes = 4
    assert call(shp, cch) == lib.IKV_ERR_UNSUPPORTED
    p.max_holes, p.scorer = 0, lib.IKV_SCORE_ENTROPY
    assert call(shp, cch) == lib.IKV_ERR_UNSUPPORTED
    p.scorer = lib.IKV_SCORE_ATTENTION
    assert call(_shape(lib, granularity=lib.IKV_GRAN_KVHEAD), cch) == lib.IKV_ERR_UNSUPPORTED
    assert call(shp, _cache(lib)) == lib.IKV_ERR_ARG             # pos_cap 0
    p.evict_mode = 7
    assert call(shp, cch) == lib.IKV_ERR_ARG
    # the workspace grows with the position capacity
    n0, n1 = lib.SZ(0), lib.SZ(0)
    lib.raw_status("ikv_step_workspace_size", ctypes.byref(shp), ctypes.byref(_cache(lib)), ctypes.byref(n0))
    lib.raw_status("ikv_step_workspace_size", ctypes.byref(shp), ctypes.byref(cch), ctypes.byref(n1))
    assert n1.value >= n0.value + 200 * 4


def test_rank_trace_arguments(lib):
    shp, cch = _shape(lib), _cache(lib)
    p = lib.ikv_params()
    p.alpha, p.refresh_period, p.budget = 0.9, 1, 16
    tr = lib.ikv_trace(16, 16, 16, None)
    p.trace = ctypes.pointer(tr)
    call = lambda: lib.raw_status("ikv_step", ctypes.byref(shp), ctypes.byref(p), ctypes.byref(cch), 16, 1, 16, 16,
                                  16, 16, 16, 1 << 40, None)
    assert call() == lib.IKV_ERR_ARG                 # counts is NULL
    tr.counts = 16
    p.scorer = lib.IKV_SCORE_ENTROPY
    assert call() == lib.IKV_ERR_UNSUPPORTED
    p.scorer, p.evict_mode = lib.IKV_SCORE_ATTENTION, lib.IKV_EVICT_LAYER
    cch.pos_cap = 100
    assert call() == lib.IKV_ERR_UNSUPPORTED


def test_deferred_compaction_arguments(lib):
    shp, cch = _shape(lib), _cache(lib)
    p = lib.ikv_params()
    p.alpha, p.refresh_period, p.budget, p.max_holes = 0.9, 1, 16, -1
    assert lib.raw_status("ikv_step", ctypes.byref(shp), ctypes.byref(p), ctypes.byref(cch), 16, 1, 16, 16, 16, 16,
                          16, 1 << 40, None) == lib.IKV_ERR_ARG
    p.max_holes, p.agg_mode = 0, 3   # no such aggregation rule
    assert lib.raw_status("ikv_step", ctypes.byref(shp), ctypes.byref(p), ctypes.byref(cch), 16, 1, 16, 16, 16, 16,
                          16, 1 << 40, None) == lib.IKV_ERR_ARG
    p.agg_mode, p.scorer = 0, 5   # no such scorer
    assert lib.raw_status("ikv_step", ctypes.byref(shp), ctypes.byref(p), ctypes.byref(cch), 16, 1, 16, 16, 16, 16,
                          16, 1 << 40, None) == lib.IKV_ERR_ARG
    p.scorer = lib.IKV_SCORE_VNORM   # VNorm without value norms in the cache
    assert lib.raw_status("ikv_step", ctypes.byref(shp), ctypes.byref(p), ctypes.byref(cch), 16, 1, 16, 16, 16, 16,
                          16, 1 << 40, None) == lib.IKV_ERR_ARG
    assert lib.raw_status("ikv_value_norms", ctypes.byref(shp), ctypes.byref(cch), None) == lib.IKV_ERR_ARG
    nopos = _cache(lib, pos=0, dead_slots=1)
    n = lib.SZ(0)
    assert lib.raw_status("ikv_attend_workspace_size", ctypes.byref(shp), ctypes.byref(nopos),
                          ctypes.byref(n)) == lib.IKV_ERR_ARG


def test_auto_max_holes():
    """The deferred-compaction threshold minimises masked reads plus amortised compaction."""
    from paper_2609_03515_gb300 import auto_max_holes
    import math
    for b in (51, 615, 1638, 3277, 6554):
        mh = auto_max_holes([b])
        assert mh % 8 == 0 and mh >= 8
        cost = lambda m: m / 2 + 2 * b / m
        assert cost(mh) <= 1.05 * cost(2 * math.sqrt(b))   # within 5 % of the continuous optimum
    assert auto_max_holes([3277]) == 112 and auto_max_holes([6554]) == 160


def test_step_lengths_mirror():
    """Host bookkeeping of len (dead slots included) and live slots across steps."""
    from paper_2609_03515_gb300 import step_lengths
    # compact every step: len = live = min(L + 1, B)
    assert step_lengths([100, 10], [100, 10], [50, 20]) == ([50, 11], [50, 11])
    # deferred: one eviction per step adds a dead slot until more than max_holes would be dead
    lens, live = [50], [50]
    seen = []
    for _ in range(7):
        lens, live = step_lengths(lens, live, [50], max_holes=3)
        seen.append(lens[0])
        assert live == [50]
    assert seen == [51, 52, 53, 50, 51, 52, 53]
    # the first step evicts far more than max_holes: compacted at once
    assert step_lengths([1000], [1000], [100], max_holes=8) == ([100], [100])
    # below the budget nothing is evicted or marked
    assert step_lengths([10], [10], [100], max_holes=8) == ([11], [11])


def test_other_entry_points_reject_nulls(lib):
    assert lib.raw_status("ikv_select_budget", 2, 8, None, 16, 1, 16, None, 16, 16, None) == lib.IKV_ERR_ARG
    assert lib.raw_status("ikv_select_budget", -1, 8, 16, 16, 1, 16, None, 16, 16, None) == lib.IKV_ERR_SHAPE
    assert lib.raw_status("ikv_ema_update", 2, 8, 16, None, 16, 1, ctypes.c_float(0.5), None) == lib.IKV_ERR_ARG
    assert lib.raw_status("ikv_ema_update", 2, 8, 16, 16, 16, 1, ctypes.c_float(-0.5), None) == lib.IKV_ERR_ARG
    shp, cch = _shape(lib), _cache(lib)
    assert lib.raw_status("ikv_compact_kv", ctypes.byref(shp), ctypes.byref(cch), None, 16, None, 0, None, 0,
                          None) == lib.IKV_ERR_ARG
    assert lib.raw_status("ikv_compact_kv", ctypes.byref(shp), ctypes.byref(cch), 16, 16, None, 1, None, 0,
                          None) == lib.IKV_ERR_WORKSPACE
    assert lib.raw_status("ikv_decode_attend_score", ctypes.byref(shp), ctypes.byref(cch), 5, 16, 16, None, None,
                          ctypes.c_float(0.9), 16, 1 << 40, None) == lib.IKV_ERR_ARG   # layer out of range
    assert lib.raw_status("ikv_decode_attend_score", ctypes.byref(shp), ctypes.byref(cch), 0, 8, 16, None, None,
                          ctypes.c_float(0.9), 16, 1 << 40, None) == lib.IKV_ERR_ALIGN
    assert lib.raw_status("ikv_append_token", ctypes.byref(shp), ctypes.byref(cch), 16, 16, None, 0, None, 0,
                          None) == lib.IKV_ERR_WORKSPACE


def test_attend_path_query(lib):
    """Which attention kernel a shape gets is decided on the host (no launch)."""
    def path(shape_kw, cache_kw):
        return lib.ikv_attend_path(_shape(lib, **shape_kw), _cache(lib, **cache_kw))
    bf = dict(dtype=lib.IKV_BF16, head_dim=128, q_heads=32, kv_heads=8)
    assert path({}, {}) == lib.IKV_PATH_CUDA_CORE                                  # fp32, d = 64
    assert path(bf, {}) == lib.IKV_PATH_TENSOR_CORE                                # bf16, d = 128, G = 4, page 64
    assert path(dict(bf, q_heads=28, kv_heads=4), {}) == lib.IKV_PATH_TENSOR_CORE  # G = 7
    assert path(bf, dict(page_size=256, max_pages=1)) == lib.IKV_PATH_TENSOR_CORE
    assert path(bf, dict(page_size=48, max_pages=4, max_len=100)) == lib.IKV_PATH_CUDA_CORE
    assert path(dict(bf, head_dim=64), {}) == lib.IKV_PATH_CUDA_CORE               # bf16, d = 64
    with pytest.raises(lib.IKVError):
        path(dict(bf, q_heads=5, kv_heads=2), {})


def test_attend_plan_query(lib):
    """How each workload's attention launch is partitioned is decided on the host (152 SMs):
    chunk size and count per (sequence, layer, KV head) unit, the passes one CTA takes, and
    whether the launch hands the score pass group sums."""
    def plan(batch, layers, H, Hkv, max_len, n_layers, dtype=lib.IKV_BF16, d=128, sms=152):
        pages = (max_len + 1 + 63) // 64 + 1
        shp = _shape(lib, batch=batch, layers=layers, q_heads=H, kv_heads=Hkv, head_dim=d, dtype=dtype)
        cch = _cache(lib, num_pages=batch * pages, max_pages=pages, max_len=max_len)
        return lib.ikv_attend_plan(shp, cch, n_layers, sms)
    tc, cc = lib.IKV_PATH_TENSOR_CORE, lib.IKV_PATH_CUDA_CORE
    # Llama b = 1, 3278 slots (+ one decode token): 256 units of 27 tiles fill 256 of 304
    # slots, so each CTA takes its unit's two 15-tile chunks in turn
    assert plan(1, 32, 32, 8, 3279, 32) == dict(path=tc, chunk_tokens=1920, n_chunks=2, passes=2, group_sums=0)
    # ... and one layer of it (split step): 8 units, the shortest chunks that fill one wave
    assert plan(1, 32, 32, 8, 3279, 1) == dict(path=tc, chunk_tokens=256, n_chunks=14, passes=1, group_sums=0)
    # Llama b = 8, 6554 slots: 2048 units, one wave's worth of 15-tile chunks, merged
    assert plan(8, 32, 32, 8, 6555, 32) == dict(path=tc, chunk_tokens=1920, n_chunks=4, passes=1, group_sums=0)
    # Llama b = 16 at ~800 slots and Qwen b = 32 at 1638: every unit one chunk -> group sums
    assert plan(16, 32, 32, 8, 820, 32) == dict(path=tc, chunk_tokens=1920, n_chunks=1, passes=1, group_sums=1)
    assert plan(32, 28, 28, 4, 1639, 28) == dict(path=tc, chunk_tokens=1920, n_chunks=1, passes=1, group_sums=1)
    # units that overfill the wave take no passes
    assert plan(2, 32, 32, 8, 3279, 32)["passes"] == 1
    # the CUDA-core kernel (fp32, d = 64): split-K, no passes, logits
    r = plan(1, 2, 4, 2, 100, 2, dtype=lib.IKV_F32, d=64)
    assert r["path"] == cc and r["passes"] == 1 and r["group_sums"] == 0 and r["n_chunks"] * r["chunk_tokens"] >= 100
    for bad in (0, 33):
        with pytest.raises(lib.IKVError):
            plan(1, 32, 32, 8, 3279, bad)
    with pytest.raises(lib.IKVError):
        plan(1, 32, 32, 8, 3279, 32, sms=-1)


def test_attend_plan_properties(lib):
    """For random shapes and lengths the plan covers every slot (plus a start offset's
    slack on the tensor-core kernel), keeps chunks within TMEM and the partial buffers,
    gives a CTA either one chunk or all of its unit's, and hands over group sums only
    when every unit is one chunk."""
    import random

    rng = random.Random(7)
    for _ in range(400):
        G = rng.choice([1, 2, 4, 7, 8])
        Hkv = rng.choice([1, 2, 4, 8])
        layers = rng.randint(1, 80)
        batch = rng.randint(1, 64)
        max_len = rng.randint(1, 200000)
        ps = rng.choice([16, 64, 128, 256])
        sms = rng.choice([1, 8, 148, 152, 160])
        n_layers = rng.choice([1, layers])
        pages = (max_len + ps) // ps + 1
        shp = _shape(lib, batch=batch, layers=layers, q_heads=G * Hkv, kv_heads=Hkv, head_dim=128, dtype=lib.IKV_BF16)
        cch = _cache(lib, num_pages=min(batch * pages, 1 << 20), page_size=ps, max_pages=pages, max_len=max_len)
        r = lib.ikv_attend_plan(shp, cch, n_layers, sms)
        slack = 127 if r["path"] == lib.IKV_PATH_TENSOR_CORE else 0
        assert r["n_chunks"] * r["chunk_tokens"] >= max_len + slack, r
        assert 1 <= r["n_chunks"] <= 128, r
        assert r["passes"] in (1, r["n_chunks"]), r
        if r["path"] == lib.IKV_PATH_TENSOR_CORE:
            assert r["chunk_tokens"] % 128 == 0 and r["chunk_tokens"] <= 15 * 128, r
            units = batch * n_layers * Hkv
            if r["passes"] > 1:                      # one CTA per unit, one wave of two per SM
                assert 4 * units >= 3 * 2 * sms and units <= 2 * sms, (r, units)
        else:
            assert r["passes"] == 1 and r["group_sums"] == 0, r
        if r["group_sums"]:
            assert r["n_chunks"] == 1, r


def test_product_package_does_not_reference_the_oracle():
    """The CUDA path and its binding never import or link the CPU oracle."""
    pkg = os.path.join(ROOT, "paper_2609_03515_gb300")
    for path in glob.glob(os.path.join(pkg, "**", "*.*"), recursive=True):
        if path.endswith((".py", ".cu", ".cuh", ".h")):
            src = open(path).read()
            assert "oracle" not in src.replace("oracle-free", ""), path
