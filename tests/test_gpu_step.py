"""Whole decode steps (ikv_step, or its begin / per-layer / end split) in lock-step
with the oracle (GPU only).

Each case runs several decode steps, with eviction on every step, and checks
per step: attention outputs (bf16: 2e-2, fp32: 1e-4 absolute), utilities of
the kept tokens (1e-3 absolute, fp32 vs fp64), the retained set under the
boundary rule (gap 1e-4 around the oracle's B-th utility), and the compacted
K/V rows bit for bit.
"""
import numpy as np
import pytest
import torch

import gen
from harness import decode_step, make_cache, fill_prefill, run_lockstep, to_device
from paper_2609_03515_gb300 import ikv

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    import __graft_entry__

    __graft_entry__.build()


def _assert(reps, tol_out, strict_fraction=0.0):
    for r in reps:
        assert r.set_ok, r
        assert r.out_err < tol_out, r
        assert r.m_err < 1e-3, r
        assert r.kv_err == 0.0, r
    if strict_fraction:
        assert np.mean([r.strict_set_equal for r in reps]) >= strict_fraction


def small_llama(**kw):
    base = dict(name="llama-small", batch=3, layers=3, q_heads=32, kv_heads=8, head_dim=128,
                prefill=[300, 777, 1200], steps=10, dtype=gen.BF16, alpha=0.9, seed=5, page_size=64)
    base.update(kw)
    return gen.Workload(**base)


def test_config0_full_trajectory():
    """The tiny fp32 workload end to end: 16 steps, full refresh, alpha 0.9, B = 51."""
    w = gen.config(0)
    reps = run_lockstep(w)
    _assert(reps, 1e-4, strict_fraction=1.0)


def test_small_llama_full_refresh():
    _assert(run_lockstep(small_llama()), 2e-2)


def test_small_llama_lazy_refresh():
    _assert(run_lockstep(small_llama(refresh_period=3, steps=9)), 2e-2)


def test_small_llama_score_free():
    _assert(run_lockstep(small_llama(score_free=True, steps=8)), 2e-2)


def test_small_llama_kvhead_rows():
    _assert(run_lockstep(small_llama(steps=6), gran=ikv.IKV_GRAN_KVHEAD), 2e-2)


def test_holefill_keeps_the_same_sets():
    _assert(run_lockstep(small_llama(steps=6), compact_mode=ikv.IKV_COMPACT_HOLEFILL), 2e-2)


def test_short_side_compaction_trajectory():
    """Shorter-side stable compaction moves start, so the attention sees tiles that do
    not start at slot 0 of the slot space; results must not change."""
    _assert(run_lockstep(small_llama(steps=10), compact_mode=ikv.IKV_COMPACT_STABLE_SHORT), 2e-2)
    _assert(run_lockstep(gen.config(0), compact_mode=ikv.IKV_COMPACT_STABLE_SHORT), 1e-4, strict_fraction=1.0)
    _assert(run_lockstep(small_llama(steps=6, score_free=True, page_size=16),
                         compact_mode=ikv.IKV_COMPACT_STABLE_SHORT), 2e-2)


def test_sparse_layer_mask_and_mean_init_on_refresh():
    w = small_llama(steps=5, layers=4)
    _assert(run_lockstep(w, layer_eligible=[1, 0, 1, 0], refresh_init=ikv.IKV_INIT_MEAN), 2e-2)


def test_qwen_group7():
    w = gen.Workload("qwen-small", 2, 2, 28, 4, 128, [2000, 513], 6, dtype=gen.BF16, seed=6, alpha=0.5)
    _assert(run_lockstep(w), 2e-2)


def test_budget_edges():
    # no eviction ever (B >= L0 + steps), and a budget of one token
    w = small_llama(batch=2, prefill=[100, 200], steps=4, budget_frac=1.0, layers=2)
    _assert(run_lockstep(w, steps=4), 2e-2)
    w1 = small_llama(batch=1, prefill=[90], steps=4, budget_frac=0.011, layers=2)
    assert w1.budgets() == [1]
    _assert(run_lockstep(w1), 2e-2)


def test_alpha_zero_and_one():
    _assert(run_lockstep(small_llama(alpha=0.0, steps=3, layers=2)), 2e-2)
    _assert(run_lockstep(small_llama(alpha=1.0, steps=3, layers=2)), 2e-2)


def test_deferred_compaction_trajectories():
    """max_holes > 0: evicted slots are only marked dead until the sequence holds more
    than max_holes of them, then the cache is compacted.  The kept set, its order, the
    utilities and the outputs must match the oracle (which compacts every step) on every
    step, across compactions and under every schedule and compaction mode."""
    _assert(run_lockstep(gen.config(0), max_holes=3), 1e-4, strict_fraction=1.0)
    _assert(run_lockstep(small_llama(steps=12), max_holes=4), 2e-2)
    _assert(run_lockstep(small_llama(steps=12, refresh_period=3), compact_mode=ikv.IKV_COMPACT_STABLE_SHORT,
                         max_holes=5), 2e-2)
    _assert(run_lockstep(small_llama(steps=10, score_free=True, page_size=16), max_holes=3), 2e-2)
    _assert(run_lockstep(small_llama(steps=8), gran=ikv.IKV_GRAN_KVHEAD, max_holes=3), 2e-2)
    _assert(run_lockstep(small_llama(steps=8), compact_mode=ikv.IKV_COMPACT_HOLEFILL, max_holes=3), 2e-2)
    _assert(run_lockstep(small_llama(steps=8, refresh_period=2), refresh_init=ikv.IKV_INIT_MEAN, max_holes=64), 2e-2)


def test_multi_pass_trajectories():
    """256 (sequence, layer, kv head) units of 16-31 tiles: the units nearly fill one wave of
    resident CTAs, so each CTA takes its unit's 15-tile chunks as passes, merged in registers.
    A 90% budget keeps the units long on every step; ragged lengths, deferred compaction
    (dead slots inside the passes), the KV-head granularity and the VNorm scorer; and the
    split step, whose per-layer launches are multi-pass and store the new rows themselves."""
    rng = np.random.default_rng(41)
    prefill = [int(x) for x in rng.integers(1900, 3800, size=16)]
    w = small_llama(batch=16, layers=2, prefill=prefill, steps=4, budget_frac=0.9)
    # the whole step's launch (2 layers x 16 sequences x 8 KV heads) is multi-pass on this device
    c0 = make_cache(w)
    assert ikv.ikv_attend_plan(c0.shape(), c0.cache(max(prefill) + 1), w.layers, 0)["passes"] > 1
    del c0
    _assert(run_lockstep(w), 2e-2)
    _assert(run_lockstep(w, max_holes=64, compact_mode=ikv.IKV_COMPACT_STABLE_SHORT), 2e-2)
    _assert(run_lockstep(w.with_(steps=3), gran=ikv.IKV_GRAN_KVHEAD), 2e-2)
    _assert(run_lockstep(w.with_(steps=3), scorer=ikv.IKV_SCORE_VNORM), 2e-2)
    # the split step: each layer call is itself a multi-pass launch (32 sequences x 8 KV
    # heads = 256 units of 16-31 tiles) whose CTAs also store the layer's new rows
    w32 = small_llama(batch=32, layers=2, prefill=[int(x) for x in rng.integers(1900, 3800, size=32)], steps=3,
                      budget_frac=0.9)
    c0 = make_cache(w32)
    assert ikv.ikv_attend_plan(c0.shape(), c0.cache(max(w32.prefill) + 1), 1, 0)["passes"] > 1
    del c0
    _assert(run_lockstep(w32, per_layer=True), 2e-2)
    _assert(run_lockstep(w32, per_layer=True, max_holes=64, compact_mode=ikv.IKV_COMPACT_STABLE_SHORT,
                         scorer=ikv.IKV_SCORE_VNORM), 2e-2)


def test_cumulative_and_single_step_aggregation():
    """Eq. 3 (cumulative) and Eq. 2 (single-step) in place of the EMA, under full refresh,
    Lazy refresh and deferred compaction."""
    cum, single = ikv.IKV_AGG_CUMULATIVE, ikv.IKV_AGG_SINGLE_STEP
    _assert(run_lockstep(gen.config(0), agg_mode=cum), 1e-4, strict_fraction=1.0)
    _assert(run_lockstep(small_llama(steps=8), agg_mode=cum), 2e-2)
    _assert(run_lockstep(small_llama(steps=8, refresh_period=3), agg_mode=cum, max_holes=4), 2e-2)
    _assert(run_lockstep(small_llama(steps=6), agg_mode=single), 2e-2)
    _assert(run_lockstep(small_llama(steps=6), gran=ikv.IKV_GRAN_KVHEAD, agg_mode=single,
                         compact_mode=ikv.IKV_COMPACT_STABLE_SHORT), 2e-2)


def test_vnorm_and_entropy_scorers():
    """The Appendix's VNorm and entropy-weighted scorers in place of Eq. 1, in lock-step with
    the oracle.  VNorm reads value-row norms that the append stores and the compaction moves
    (stable, shorter-side, hole-fill and deferred), so the trajectories also check those."""
    vn, ent = ikv.IKV_SCORE_VNORM, ikv.IKV_SCORE_ENTROPY
    _assert(run_lockstep(gen.config(0), scorer=vn), 1e-4, strict_fraction=1.0)
    _assert(run_lockstep(gen.config(0), scorer=ent), 1e-4, strict_fraction=1.0)
    _assert(run_lockstep(small_llama(steps=8), scorer=vn), 2e-2)
    _assert(run_lockstep(small_llama(steps=8, refresh_period=3), scorer=vn, compact_mode=ikv.IKV_COMPACT_STABLE_SHORT,
                         max_holes=3), 2e-2)
    _assert(run_lockstep(small_llama(steps=6), scorer=vn, gran=ikv.IKV_GRAN_KVHEAD,
                         compact_mode=ikv.IKV_COMPACT_HOLEFILL), 2e-2)
    _assert(run_lockstep(small_llama(steps=8), scorer=ent), 2e-2)
    _assert(run_lockstep(small_llama(steps=8, score_free=True), scorer=ent, max_holes=4), 2e-2)
    _assert(run_lockstep(small_llama(steps=6), scorer=ent, gran=ikv.IKV_GRAN_KVHEAD,
                         agg_mode=ikv.IKV_AGG_CUMULATIVE), 2e-2)


def test_per_layer_split_trajectories():
    """ikv_step_begin, one ikv_step_layer per layer, ikv_step_end: the model-integration
    form of the step (Appendix "Layer scoring": scores folded layer by layer inside the
    forward pass), in lock-step with the oracle across schedules, row granularities,
    compaction modes, deferral, aggregation rules and scorers."""
    vn, ent = ikv.IKV_SCORE_VNORM, ikv.IKV_SCORE_ENTROPY
    _assert(run_lockstep(gen.config(0), per_layer=True), 1e-4, strict_fraction=1.0)
    _assert(run_lockstep(gen.config(0), max_holes=3, scorer=ent, per_layer=True), 1e-4, strict_fraction=1.0)
    _assert(run_lockstep(small_llama(steps=8), per_layer=True), 2e-2)
    _assert(run_lockstep(small_llama(steps=9, refresh_period=4), compact_mode=ikv.IKV_COMPACT_STABLE_SHORT,
                         max_holes=3, per_layer=True), 2e-2)
    _assert(run_lockstep(small_llama(steps=6, score_free=True, page_size=16), max_holes=4, per_layer=True), 2e-2)
    _assert(run_lockstep(small_llama(steps=6), gran=ikv.IKV_GRAN_KVHEAD, compact_mode=ikv.IKV_COMPACT_HOLEFILL,
                         per_layer=True), 2e-2)
    _assert(run_lockstep(small_llama(steps=6, layers=4), layer_eligible=[0, 1, 1, 0],
                         refresh_init=ikv.IKV_INIT_MEAN, agg_mode=ikv.IKV_AGG_CUMULATIVE, per_layer=True), 2e-2)
    _assert(run_lockstep(small_llama(steps=6), scorer=vn, max_holes=3, per_layer=True), 2e-2)
    _assert(run_lockstep(small_llama(steps=6, refresh_period=2), scorer=ent, per_layer=True), 2e-2)
    w = gen.Workload(name="qwen-small", batch=2, layers=2, q_heads=28, kv_heads=4, head_dim=128, prefill=[700, 260],
                     steps=5, dtype=gen.BF16, alpha=0.9, seed=9, page_size=32)
    _assert(run_lockstep(w, per_layer=True), 2e-2)


def test_per_layer_split_equals_whole_step():
    """The split step and ikv_step on the same inputs give bit-identical caches, utilities
    and outputs when the attention is partitioned alike: at these lengths (at most 3 tiles
    of 128 slots per unit) both give every tile its own split, so the two differ only in
    how the launches are cut."""
    w = small_llama(steps=6, refresh_period=2, prefill=[100, 180, 250])
    u = w.u_table()
    caches = []
    for per_layer in (False, True):
        c = make_cache(w)
        fill_prefill(c, w, u)
        caches.append(c)
    p = [c.params(w.alpha, w.refresh_period, False, ikv.IKV_COMPACT_STABLE_SHORT, max_holes=3) for c in caches]
    ws = [c.step_workspace() for c in caches]
    qs = w.queries(1, w.steps + 1, u)
    outs = [torch.empty((w.layers, w.batch, w.q_heads, w.head_dim), dtype=torch.bfloat16, device="cuda")
            for _ in caches]
    max_len = max(w.prefill)
    for t in range(1, w.steps + 1):
        kn, vn = w.new_tokens(t, u)
        for i, c in enumerate(caches):
            decode_step(c, p[i], c.cache(max_len), t, to_device(qs[t - 1], w), to_device(kn, w), to_device(vn, w),
                        outs[i], ws[i], per_layer=i == 1)
        torch.cuda.synchronize()
        a, b = caches
        assert torch.equal(a.len, b.len) and torch.equal(a.start, b.start) and torch.equal(a.pos, b.pos), t
        assert torch.equal(a.next_pos, b.next_pos), t
        assert torch.equal(a.k, b.k) and torch.equal(a.v, b.v), t
        assert torch.equal(a.ema, b.ema), t
        assert torch.equal(outs[0], outs[1]), t
        max_len = int(a.len.max())
    assert ikv.ikv_device_status() == 0


def test_per_layer_immediate_eviction_trajectories():
    """IKV_EVICT_LAYER: each layer evicts right after folding its score into the
    position-indexed state (reading R10), through ikv_step and through the begin /
    per-layer / end split, in lock-step with the oracle's decode_step_layerwise."""
    from harness import run_lockstep_layerwise

    _assert(run_lockstep_layerwise(gen.config(0)), 1e-4, strict_fraction=1.0)
    _assert(run_lockstep_layerwise(gen.config(0), per_layer=True), 1e-4, strict_fraction=1.0)
    _assert(run_lockstep_layerwise(gen.config(0).with_(refresh_period=3), refresh_init=ikv.IKV_INIT_MEAN),
            1e-4, strict_fraction=1.0)
    _assert(run_lockstep_layerwise(small_llama(steps=8)), 2e-2)
    _assert(run_lockstep_layerwise(small_llama(steps=8), per_layer=True), 2e-2)
    _assert(run_lockstep_layerwise(small_llama(steps=9, refresh_period=4)), 2e-2)
    _assert(run_lockstep_layerwise(small_llama(steps=6, score_free=True, page_size=16), per_layer=True), 2e-2)
    _assert(run_lockstep_layerwise(small_llama(steps=6, layers=4), layer_eligible=[0, 1, 1, 0],
                                   refresh_init=ikv.IKV_INIT_MEAN), 2e-2)
    _assert(run_lockstep_layerwise(small_llama(steps=8), compact_mode=ikv.IKV_COMPACT_HOLEFILL), 2e-2)
    _assert(run_lockstep_layerwise(small_llama(steps=6, refresh_period=2), compact_mode=ikv.IKV_COMPACT_STABLE_SHORT,
                                   per_layer=True), 2e-2)
    _assert(run_lockstep_layerwise(gen.config(0), compact_mode=ikv.IKV_COMPACT_HOLEFILL), 1e-4)
    w = gen.Workload(name="qwen-small", batch=2, layers=2, q_heads=28, kv_heads=4, head_dim=128, prefill=[700, 260],
                     steps=5, dtype=gen.BF16, alpha=0.9, seed=9, page_size=32)
    _assert(run_lockstep_layerwise(w, per_layer=True), 2e-2)


def test_rank_trace_diagnostics():
    """The step's rank trace (reading R11): the EMA top-k equals the kept positions, the raw
    top-k is a valid top-B of the oracle's single-step score under the boundary rule, and
    the overlap counts equal the set intersections of this and the previous traced step;
    across schedules, granularities, compaction modes, deferral and the split step."""
    _assert(run_lockstep(gen.config(0), trace=True), 1e-4, strict_fraction=1.0)
    _assert(run_lockstep(small_llama(steps=8), trace=True), 2e-2)
    _assert(run_lockstep(small_llama(steps=9, refresh_period=3), trace=True, max_holes=3,
                         compact_mode=ikv.IKV_COMPACT_STABLE_SHORT), 2e-2)
    _assert(run_lockstep(small_llama(steps=6), gran=ikv.IKV_GRAN_KVHEAD, compact_mode=ikv.IKV_COMPACT_HOLEFILL,
                         trace=True), 2e-2)
    _assert(run_lockstep(small_llama(steps=6), scorer=ikv.IKV_SCORE_VNORM, trace=True, per_layer=True), 2e-2)


def test_workspace_kept_zero_across_steps():
    """ikv_params.ws_zeroed: with a zero-filled workspace every step leaves its counters zero,
    so steps that skip re-zeroing them give the same trajectories (whole step with
    multi-chunk attention units and the fused selection, deferral, the split step)."""
    _assert(run_lockstep(gen.config(0), ws_zeroed=True), 1e-4, strict_fraction=1.0)
    _assert(run_lockstep(small_llama(steps=8, prefill=[300, 2000, 1200]), ws_zeroed=True), 2e-2)
    _assert(run_lockstep(small_llama(steps=9, refresh_period=3), max_holes=3, ws_zeroed=True,
                         compact_mode=ikv.IKV_COMPACT_STABLE_SHORT), 2e-2)
    _assert(run_lockstep(small_llama(steps=6), per_layer=True, ws_zeroed=True), 2e-2)


@pytest.mark.parametrize("case", [
    dict(compact_mode=ikv.IKV_COMPACT_STABLE_SHORT, max_holes=2),     # prefix moves right, start advances
    dict(compact_mode=ikv.IKV_COMPACT_STABLE_SHORT, tight=True),      # append at cap - 1, relocation to slot 0
    dict(compact_mode=ikv.IKV_COMPACT_HOLEFILL, scorer=ikv.IKV_SCORE_VNORM),
    dict(compact_mode=ikv.IKV_COMPACT_STABLE, gran=ikv.IKV_GRAN_KVHEAD),
    dict(compact_mode=ikv.IKV_COMPACT_STABLE_SHORT, max_holes=3, per_layer=True),
    dict(compact_mode=ikv.IKV_COMPACT_STABLE_SHORT, max_holes=2, strided=True),
], ids=["short_deferred", "short_tight_cap", "holefill_vnorm", "stable_kvhead", "split_step", "short_strided"])
def test_nothing_written_outside_the_buffers(case):
    """Canaries around every buffer (spare pool pages among the used ones, tails after pos,
    ema, vnorm and the workspace) stay intact through lock-step runs that exercise the
    shorter-side moves (right moves, relocation to slot 0), an append into the last slot of
    the slot space, hole-fill with value norms, KV-head rows, the split step, and the
    compaction's grid-stride form (16 sequences x 33 items: more than one wave of its CTAs)."""
    case = dict(case)
    tight = case.pop("tight", False)
    strided = case.pop("strided", False)
    if strided:
        w = small_llama(batch=16, layers=4, steps=6,
                        prefill=[150 + 29 * i for i in range(16)])
    elif tight:
        # cap = 320 slots: sequence 0's first append lands in slot 319, and the shorter-side
        # compaction runs out of room on the right
        w = small_llama(prefill=[319, 200], batch=2, steps=8, budget_frac=0.5)
    else:
        w = small_llama(steps=6)
    _assert(run_lockstep(w, canaries=True, **case), 2e-2)
