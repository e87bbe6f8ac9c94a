"""Parity at the five workloads' full sizes (GPU only).

The GPU runs each workload at its real shape in the benchmark's launch
configuration; the streaming oracle (oracle.decode_step_streaming, pinned bit for
bit to oracle.decode_step) follows sampled sequences (sequences are independent)
for the first decode steps, including step 1, which scores the whole prefill
and evicts ~90% of it.  Per step: attention outputs of every layer and head
(bf16: 2e-2), the kept set under the 1e-4 boundary rule and under the relative
rule (gap 1e-4 theta), the kept utilities (1e-3 absolute and 1e-3 relative),
and the compacted K/V rows of the first and last layer bit for bit.  The
fraction of steps whose kept set equals the oracle's own top-B is printed.

The last tests replay the benchmark's own timed loop (bench.run_mode_graph: one
CUDA graph per step, workspace counters kept zero, deferred shorter-side
compaction) through a compaction of the dead slots, checking every step.
"""
import os
import sys

import pytest

import gen
from harness import SampledOracle, run_fullsize_sampled, run_fullsize_sampled_layerwise
from paper_2609_03515_gb300 import ikv

pytestmark = pytest.mark.gpu


def _check(reps, label=""):
    for r in reps:
        assert r.set_ok, r
        assert r.rel_set_ok, r
        assert r.out_err < 2e-2, r
        assert r.m_err < 1e-3, r
        assert r.m_rel_err < 1e-3, r
        assert r.kv_err == 0.0, r
    strict = sum(r.strict_set_equal for r in reps) / max(1, len(reps))
    print(f"\n{label} steps {len(reps)}: strict-set fraction {strict:.3f}, max rel utility error "
          f"{max(r.m_rel_err for r in reps):.2e}, max out error {max(r.out_err for r in reps):.2e}")


# The benchmark's configuration: shorter-side stable compaction, deferred while a
# sequence holds at most 128 dead slots.
SHORT = ikv.IKV_COMPACT_STABLE_SHORT


def bench_holes(w):
    return 128


@pytest.mark.timeout(1200)
def test_config1_llama_b1_32k_full_refresh():
    w = gen.config(1)
    _check(run_fullsize_sampled(w, seqs=[0], steps=4, compact_mode=SHORT, max_holes=bench_holes(w)))


@pytest.mark.timeout(1200)
def test_config1_deferred_compaction_crossing():
    # max_holes 3: steps 2-4 mark their evictions dead, step 5 compacts them away, 6-7 mark again
    _check(run_fullsize_sampled(gen.config(1), seqs=[0], steps=7, compact_mode=SHORT, max_holes=3))


@pytest.mark.timeout(1200)
def test_config2_llama_b16_ragged_lazy4():
    # steps 1 and 5 refresh, 2-4 carry the state (Eq. 6); two of the sixteen sequences followed
    w = gen.config(2)
    _check(run_fullsize_sampled(w, seqs=[0, 11], steps=5, compact_mode=SHORT, max_holes=bench_holes(w)))


@pytest.mark.timeout(1200)
def test_config3_llama_b8_64k_score_free():
    w = gen.config(3)
    _check(run_fullsize_sampled(w, seqs=[5], steps=3, compact_mode=SHORT, max_holes=bench_holes(w)))


@pytest.mark.timeout(1200)
def test_config4_qwen_b32_16k_sweep_point():
    # one point of the sweep: budget 25%, alpha 0.5, Lazy refresh period 2
    w = gen.config(4).with_(budget_frac=0.25, alpha=0.5, refresh_period=2)
    _check(run_fullsize_sampled(w, seqs=[31], steps=3, compact_mode=SHORT, max_holes=bench_holes(w)))


@pytest.mark.timeout(1200)
def test_config4_every_step_compaction():
    # the same workload with compaction on every eviction and the always-left stable shift
    w = gen.config(4).with_(budget_frac=0.1)
    _check(run_fullsize_sampled(w, seqs=[0], steps=3, compact_mode=ikv.IKV_COMPACT_STABLE))


@pytest.mark.timeout(1200)
def test_config2_per_layer_split():
    # the same workload stepped through ikv_step_begin / one ikv_step_layer per layer / ikv_step_end
    w = gen.config(2)
    _check(run_fullsize_sampled(w, seqs=[3], steps=5, compact_mode=SHORT, max_holes=bench_holes(w), per_layer=True))


@pytest.mark.timeout(1200)
def test_config1_per_layer_split():
    _check(run_fullsize_sampled(gen.config(1), seqs=[0], steps=3, compact_mode=SHORT, max_holes=3, per_layer=True))


@pytest.mark.timeout(1200)
def test_config1_per_layer_immediate_eviction():
    # every layer evicts right after its own update (step 1 drops ~90% of each layer's prefill)
    _check(run_fullsize_sampled_layerwise(gen.config(1), seqs=[0], steps=3))


@pytest.mark.timeout(1200)
def test_config2_per_layer_immediate_eviction_split_lazy4():
    _check(run_fullsize_sampled_layerwise(gen.config(2), seqs=[5], steps=5, per_layer=True))


def _bench_path(cfg: int, seqs, warmup: int, steps: int, **kw):
    """The benchmark's timed loop for workload cfg, every step checked against the oracle."""
    import torch

    sys.path.insert(0, os.path.dirname(os.path.dirname(os.path.abspath(__file__))))
    import bench

    w = gen.config(cfg).with_(**kw)
    if warmup + steps > w.steps:
        w = w.with_(steps=warmup + steps)
    args = type("A", (), {"warmup": warmup, "steps": steps})()
    dev = torch.device("cuda", 0)
    c = bench.setup(w, dev, ikv.IKV_COMPACT_STABLE_SHORT, warmup + steps)
    u = w.u_table()
    u_dev = torch.from_numpy(u).to(dev)
    ws = c.step_workspace()
    qs_dev, kn_dev, vn_dev = bench.device_inputs(w, u, u_dev, warmup + steps, dev)
    chk = SampledOracle(w, c, seqs, u, ikv.IKV_COMPACT_STABLE_SHORT)
    res = bench.run_mode_graph(args, w, c, u_dev, qs_dev, kn_dev, vn_dev, ws, ikv.IKV_COMPACT_STABLE_SHORT, None,
                               False, 128, after_step=lambda t, out: chk.check(t, out))
    assert res["launches"] > 0
    assert ikv.ikv_device_status() == 0
    return chk.reports


@pytest.mark.timeout(1800)
def test_config1_bench_path_graph_replay_across_deferred_compaction():
    # decode steps 1-5 eager (step 1 evicts ~90% of the prefill), 6-145 replayed from
    # per-step graphs with ws_zeroed; the dead slots reach 129 at step 130, which compacts
    reps = _bench_path(1, [0], 5, 140)
    assert len(reps) == 145
    _check(reps, "config 1 bench path")


@pytest.mark.timeout(1800)
def test_config2_bench_path_lazy4_graph_replay_across_deferred_compaction():
    reps = _bench_path(2, [0, 9], 5, 135)
    _check(reps, "config 2 bench path")
