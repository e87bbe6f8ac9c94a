"""Pins the CPU oracle to what the paper and the mathematics fix (no GPU needed).

Each test checks the oracle against something other than itself: a closed form
the paper states, a textbook routine, brute force on tiny inputs, or an
invariant of the method.  A plausible slip in the oracle (dropped term, wrong
sign, wrong index, transposed operand, wrong layer order, wrong schedule)
fails at least one of them.
"""
import itertools
import json
import math
import os

import numpy as np
import pytest
import torch

import oracle as O

GOLD = os.path.join(os.path.dirname(__file__), "golden")


def _load(name):
    with open(os.path.join(GOLD, name)) as f:
        return json.load(f)


def _num(x):
    return float(x) if not isinstance(x, str) else float(x.replace("inf", "inf"))


def _rand_state(rng, layers=3, kv=2, L0=40, d=8, budget=12, gran=O.GRAN_SEQ, heavy=True):
    K = [[rng.standard_normal((L0, d)) for _ in range(kv)] for _ in range(layers)]
    V = [[rng.standard_normal((L0, d)) for _ in range(kv)] for _ in range(layers)]
    if heavy:  # a few strongly attended tokens so rankings are not pure noise
        for l in range(layers):
            for g in range(kv):
                K[l][g][::7] *= 3.0
    return O.prefill_state(K, V, budget, gran)


def _rand_inputs(rng, T, layers=3, H=4, kv=2, d=8):
    q = rng.standard_normal((T, layers, H, d))
    kn = rng.standard_normal((T, layers, kv, d))
    vn = rng.standard_normal((T, layers, kv, d))
    return q, kn, vn


def _clone(st):
    return O.SeqState(K=[[k.copy() for k in row] for row in st.K], V=[[v.copy() for v in row] for row in st.V],
                      m=st.m.copy(), pos=st.pos.copy(), budget=st.budget, next_pos=st.next_pos,
                      granularity=st.granularity)


# ---------------------------------------------------------------- attention
def test_softmax_rows_sum_to_one():
    rng = np.random.default_rng(0)
    z = rng.standard_normal((50, 300)) * 30
    a = O.softmax(z)
    assert np.all(a >= 0)
    assert np.max(np.abs(a.sum(-1) - 1.0)) < 1e-12


def test_attention_golden_two_tokens():
    g = _load("attention_two_tokens.json")
    a, out = O.last_query_attention(np.array(g["q"]), [np.array(k) for k in g["K"]], [np.array(v) for v in g["V"]])
    assert np.allclose(a, g["a"], atol=1e-15, rtol=0)
    assert np.allclose(out, g["out"], atol=1e-14, rtol=0)


def test_attention_matches_library_sdpa_gqa():
    """GQA last-query attention equals torch's fp64 scaled_dot_product_attention
    with the KV heads repeated over their query groups (textbook special case)."""
    rng = np.random.default_rng(1)
    H, kv, L, d = 8, 2, 37, 16
    q = rng.standard_normal((H, d))
    K = [rng.standard_normal((L, d)) for _ in range(kv)]
    V = [rng.standard_normal((L, d)) for _ in range(kv)]
    _, out = O.last_query_attention(q, K, V)
    Kt = torch.tensor(np.stack(K)).repeat_interleave(H // kv, 0)[None]
    Vt = torch.tensor(np.stack(V)).repeat_interleave(H // kv, 0)[None]
    ref = torch.nn.functional.scaled_dot_product_attention(torch.tensor(q)[None, :, None], Kt, Vt)[0, :, 0]
    assert np.max(np.abs(out - ref.numpy())) < 1e-12


def test_attention_bruteforce_loops():
    rng = np.random.default_rng(2)
    H, kv, L, d = 4, 2, 5, 3
    q = rng.standard_normal((H, d))
    K = [rng.standard_normal((L, d)) for _ in range(kv)]
    V = [rng.standard_normal((L, d)) for _ in range(kv)]
    a, out = O.last_query_attention(q, K, V)
    for h in range(H):
        g = h // 2
        z = [sum(q[h][e] * K[g][i][e] for e in range(d)) / math.sqrt(d) for i in range(L)]
        den = sum(math.exp(x) for x in z)
        for i in range(L):
            assert abs(a[h][i] - math.exp(z[i]) / den) < 1e-14
        for e in range(d):
            assert abs(out[h][e] - sum(math.exp(z[i]) / den * V[g][i][e] for i in range(L))) < 1e-13


def test_pooled_score_granularities_bruteforce():
    rng = np.random.default_rng(3)
    a = rng.random((6, 9))
    s_seq = O.pooled_score(a, O.GRAN_SEQ, 3)
    s_kv = O.pooled_score(a, O.GRAN_KVHEAD, 3)
    assert s_seq.shape == (1, 9) and s_kv.shape == (3, 9)
    for i in range(9):
        assert abs(s_seq[0, i] - sum(a[h, i] for h in range(6)) / 6) < 1e-15
        for g in range(3):
            assert abs(s_kv[g, i] - (a[2 * g, i] + a[2 * g + 1, i]) / 2) < 1e-15


# ---------------------------------------------------------------- EMA
def test_layer_weights_golden():
    """Appendix 'Layer scoring': prior weight alpha^K, layer l weight (1-alpha) alpha^(K-l)."""
    for c in _load("layer_weights.json")["cases"]:
        K, alpha = c["K"], c["alpha"]
        # one-hot probes recover each weight from the recurrence
        prior = O.layer_sequential_ema(np.array([1.0]), [np.array([0.0])] * K, alpha)[0]
        assert abs(prior - c["prior"]) < 1e-12
        for l in range(K):
            s = [np.array([1.0 if j == l else 0.0]) for j in range(K)]
            w = O.layer_sequential_ema(np.array([0.0]), s, alpha)[0]
            assert abs(w - c["layer"][l]) < 1e-12
        assert abs(c["prior"] + sum(c["layer"]) - 1.0) < 1e-12


def test_layer_sequential_matches_closed_form_weights():
    rng = np.random.default_rng(4)
    K, alpha = 7, 0.73
    m0 = rng.random(11)
    S = [rng.random(11) for _ in range(K)]
    got = O.layer_sequential_ema(m0, S, alpha)
    want = alpha ** K * m0 + sum((1 - alpha) * alpha ** (K - 1 - l) * S[l] for l in range(K))
    assert np.max(np.abs(got - want)) < 1e-14


def test_momentum_dominance_golden():
    g = _load("momentum_dominance.json")
    rng = np.random.default_rng(5)
    s = rng.random(64)
    delta = rng.standard_normal(64)
    delta *= g["rel_perturbation"] * np.linalg.norm(s) / np.linalg.norm(delta)
    m = rng.random(64)
    rel = np.linalg.norm(O.ema_update(m, s + delta, g["alpha"]) - O.ema_update(m, s, g["alpha"])) / np.linalg.norm(s)
    assert abs(rel - g["expected_rel_change"]) < 1e-12
    assert round(100 * rel) == g["paper_rounded_percent"]


def test_prop1a_expectation_closed_form():
    """Prop. 1(a) proof: E[mu_T] = (1 - alpha^T) s_bar from mu_0 = 0."""
    rng = np.random.default_rng(6)
    alpha, T, n = 0.8, 12, 400000
    s = rng.random((T, n))  # iid U[0,1], mean 1/2
    mu = np.zeros(n)
    for t in range(T):
        mu = O.ema_update(mu, s[t], alpha)
    want = (1 - alpha ** T) * 0.5
    se = np.std(mu) / np.sqrt(n)
    assert abs(mu.mean() - want) < 5 * se


def test_prop1b_variance_bound_monte_carlo():
    """Prop. 1(b): Var[mu_T(i) - mu_T(j)] <= 2(1-alpha)/(1+alpha) sigma^2, and for iid
    scores the finite-T value is that bound times (1 - alpha^(2T))."""
    rng = np.random.default_rng(7)
    for alpha in (0.5, 0.8, 0.95):
        T, n = 60, 200000
        sigma2 = 1.0 / 12.0
        mi = np.zeros(n)
        mj = np.zeros(n)
        for _ in range(T):
            mi = O.ema_update(mi, rng.random(n) + 0.1, alpha)
            mj = O.ema_update(mj, rng.random(n), alpha)
        var = np.var(mi - mj)
        bound = 2 * (1 - alpha) / (1 + alpha) * sigma2
        exact = bound * (1 - alpha ** (2 * T))
        assert abs(var - exact) / exact < 0.02
        assert var <= bound * 1.02


def test_ema_constant_stream_through_decode_loop():
    """Uniform attention (all-zero keys) gives a constant score s = 1/L at every layer and
    step; with B = L0 the prefill tokens survive and end at m = (1 - alpha^(K T)) / L
    (geometric series, Prop. 1 proof with mu_0 = 0)."""
    layers, kv, H, d, L0, T, alpha = 3, 2, 4, 8, 20, 5, 0.7
    K = [[np.zeros((L0, d)) for _ in range(kv)] for _ in range(layers)]
    V = [[np.ones((L0, d)) for _ in range(kv)] for _ in range(layers)]
    st = O.prefill_state(K, V, budget=L0)
    p = O.Params(alpha=alpha)
    rng = np.random.default_rng(8)
    for t in range(1, T + 1):
        q = rng.standard_normal((layers, H, d))
        out = O.decode_step(st, t, q, np.zeros((layers, kv, d)), np.ones((layers, kv, d)), p)
        assert np.allclose(out, 1.0, atol=1e-14)
        assert st.length == L0
    assert np.array_equal(st.pos[0], np.arange(L0))
    want = (1 - alpha ** (layers * T)) / (L0 + 1)
    assert np.max(np.abs(st.m[0] - want)) < 1e-15


def _spike_layers(layers, kv, H, d, L0, spikes, z_spike):
    """Keys zero except one token per layer (spikes[l]) aligned with the query,
    giving that token logit z_spike and every other token logit 0."""
    K = [[np.zeros((L0, d)) for _ in range(kv)] for _ in range(layers)]
    for l in range(layers):
        for g in range(kv):
            K[l][g][spikes[l], 0] = z_spike * math.sqrt(d)
    V = [[np.zeros((L0, d)) for _ in range(kv)] for _ in range(layers)]
    q = np.zeros((layers, H, d))
    q[:, :, 0] = 1.0
    return K, V, q


def test_layer_order_through_decode_step():
    """One refresh step where each layer spikes on a different token: the resulting
    state must carry the paper's layer weights in layer order."""
    layers, kv, H, d, L0, alpha, zs = 4, 2, 4, 4, 10, 0.6, 2.0
    spikes = [1, 4, 6, 8]
    K, V, q = _spike_layers(layers, kv, H, d, L0, spikes, zs)
    st = O.prefill_state(K, V, budget=L0 + 1)
    O.decode_step(st, 1, q, np.zeros((layers, kv, d)), np.zeros((layers, kv, d)), O.Params(alpha=alpha))
    L = L0 + 1
    den = math.exp(zs) + L - 1
    for i in range(L):
        want = 0.0
        for l in range(layers):
            s = math.exp(zs) / den if i == spikes[l] else 1.0 / den
            want += (1 - alpha) * alpha ** (layers - 1 - l) * s
        assert abs(st.m[0, i] - want) < 1e-15


def test_alpha_zero_keeps_only_last_eligible_layer():
    """Sec. 5.1: alpha = 0 retains only the last processed layer."""
    layers, kv, H, d, L0, zs = 3, 1, 2, 4, 8, 1.5
    spikes = [0, 3, 5]
    K, V, q = _spike_layers(layers, kv, H, d, L0, spikes, zs)
    for mask, last in (([True, True, True], 2), ([True, True, False], 1)):
        st = O.prefill_state(K, V, budget=L0 + 1)
        O.decode_step(st, 1, q, np.zeros((layers, kv, d)), np.zeros((layers, kv, d)),
                      O.Params(alpha=0.0, layer_mask=mask))
        den = math.exp(zs) + L0
        want = np.full(L0 + 1, 1.0 / den)
        want[spikes[last]] = math.exp(zs) / den
        assert np.max(np.abs(st.m[0] - want)) < 1e-15


def test_cumulative_constant_stream_through_decode_loop():
    """Eq. 3 under the layer-sequential update: uniform attention gives s = 1/L at every
    layer and step, so after T refresh steps the surviving prefill tokens hold K T / L
    (no forgetting), and the new token (K / L after its own step) is the one evicted."""
    layers, kv, H, d, L0, T = 3, 2, 4, 8, 20, 5
    K = [[np.zeros((L0, d)) for _ in range(kv)] for _ in range(layers)]
    V = [[np.ones((L0, d)) for _ in range(kv)] for _ in range(layers)]
    st = O.prefill_state(K, V, budget=L0)
    p = O.Params(aggregation="cumulative")
    rng = np.random.default_rng(9)
    for t in range(1, T + 1):
        q = rng.standard_normal((layers, H, d))
        O.decode_step(st, t, q, np.zeros((layers, kv, d)), np.ones((layers, kv, d)), p)
        assert st.length == L0
    assert np.array_equal(st.pos[0], np.arange(L0))
    assert np.max(np.abs(st.m[0] - layers * T / (L0 + 1))) < 1e-13


def test_single_step_keeps_last_layer_and_equals_alpha_zero():
    """Eq. 2: the utility is the last eligible layer's score -- the same as EMA with
    alpha = 0 (bit for bit) -- whatever the earlier layers or steps contributed."""
    layers, kv, H, d, L0, zs = 3, 1, 2, 4, 8, 1.5
    spikes = [0, 3, 5]
    K, V, q = _spike_layers(layers, kv, H, d, L0, spikes, zs)
    for mask, last in (([True, True, True], 2), ([True, False, False], 0)):
        st = O.prefill_state(K, V, budget=L0 + 1)
        st.m[:] = 7.0  # any earlier state is discarded
        ref = _clone(st)
        O.decode_step(st, 1, q, np.zeros((layers, kv, d)), np.zeros((layers, kv, d)),
                      O.Params(aggregation="single", layer_mask=mask))
        O.decode_step(ref, 1, q, np.zeros((layers, kv, d)), np.zeros((layers, kv, d)),
                      O.Params(alpha=0.0, layer_mask=mask))
        den = math.exp(zs) + L0
        want = np.full(L0 + 1, 1.0 / den)
        want[spikes[last]] = math.exp(zs) / den
        assert np.max(np.abs(st.m[0] - want)) < 1e-15
        assert np.array_equal(st.m, ref.m)


def test_vnorm_weights_bruteforce_and_invariances():
    """VNorm (Appendix "Per-step scoring"): pure-Python norms and means; unit-norm values
    leave Eq. 1 unchanged; scaling a KV head's values does not change the score."""
    rng = np.random.default_rng(21)
    H, kv, L, d = 6, 3, 9, 5
    V = [rng.standard_normal((L, d)) for _ in range(kv)]
    a = rng.random((H, L))
    a /= a.sum(axis=1, keepdims=True)
    got = O.vnorm_score(a, V, O.GRAN_SEQ, kv)[0]
    G = H // kv
    for i in range(L):
        acc = 0.0
        for h in range(H):
            g = h // G
            norms = [math.sqrt(sum(x * x for x in V[g][j])) for j in range(L)]
            acc += a[h, i] * norms[i] / (sum(norms) / L)
        assert abs(got[i] - acc / H) < 1e-14
    unit = [v / np.linalg.norm(v, axis=1, keepdims=True) for v in V]
    assert np.max(np.abs(O.vnorm_score(a, unit, O.GRAN_KVHEAD, kv) - O.pooled_score(a, O.GRAN_KVHEAD, kv))) < 1e-14
    scaled = [v * c for v, c in zip(V, (0.5, 3.0, 7.0))]
    assert np.max(np.abs(O.vnorm_score(a, scaled, O.GRAN_SEQ, kv) - got)) < 1e-14


def test_entropy_weight_closed_forms():
    """Entropy weighting: uniform scores have normalized entropy 1 (no change), a one-hot
    distribution 0, and a two-point distribution (p, 1-p) over n tokens has
    -(p ln p + (1-p) ln(1-p)) / ln n; brute force with math.log."""
    assert abs(O.entropy_weight(np.full(37, 1 / 37)) - 1.0) < 1e-14
    assert O.entropy_weight(np.eye(1, 12)[0]) == 0.0
    assert O.entropy_weight(np.array([1.0])) == 1.0
    p, n = 0.3, 8
    s = np.zeros(n)
    s[2], s[5] = p, 1 - p
    assert abs(O.entropy_weight(s) - (-(p * math.log(p) + (1 - p) * math.log(1 - p)) / math.log(n))) < 1e-15
    rng = np.random.default_rng(3)
    r = rng.random(15)
    r /= r.sum()
    assert abs(O.entropy_weight(r) - sum(-x * math.log(x) for x in r) / math.log(15)) < 1e-14


def test_entropy_scorer_through_decode_step():
    """Uniform attention: entropy weight 1, so the step equals the plain scorer bit for
    bit; a spiked layer contributes its score times its normalized entropy."""
    layers, kv, H, d, L0, alpha = 2, 1, 2, 4, 10, 0.6
    K = [[np.zeros((L0, d)) for _ in range(kv)] for _ in range(layers)]
    V = [[np.ones((L0, d)) for _ in range(kv)] for _ in range(layers)]
    q = np.ones((layers, H, d))
    st, ref = O.prefill_state(K, V, budget=L0 + 1), O.prefill_state(K, V, budget=L0 + 1)
    O.decode_step(st, 1, q, np.zeros((layers, kv, d)), np.ones((layers, kv, d)), O.Params(alpha=alpha, scorer="entropy"))
    O.decode_step(ref, 1, q, np.zeros((layers, kv, d)), np.ones((layers, kv, d)), O.Params(alpha=alpha))
    assert np.max(np.abs(st.m - ref.m)) < 1e-15
    zs = 3.0
    K2, V2, q2 = _spike_layers(1, 1, 2, 4, L0, [4], zs)
    st2 = O.prefill_state(K2, V2, budget=L0 + 1)
    O.decode_step(st2, 1, q2, np.zeros((1, 1, 4)), np.zeros((1, 1, 4)), O.Params(alpha=alpha, scorer="entropy"))
    L = L0 + 1
    s = np.full(L, 1.0 / (math.exp(zs) + L - 1))
    s[4] = math.exp(zs) / (math.exp(zs) + L - 1)
    w = -sum(x * math.log(x) for x in s) / math.log(L)
    assert np.max(np.abs(st2.m[0] - (1 - alpha) * w * s)) < 1e-15


def test_vnorm_scorer_through_decode_step():
    """VNorm inside the decode loop: value rows of equal norm give the plain scores; one
    value row twice as long doubles its token's weight relative to the mean norm."""
    layers, kv, H, d, L0, alpha = 1, 1, 2, 4, 6, 0.5
    K = [[np.zeros((L0, d))]]
    V = [[np.ones((L0, d))]]
    V[0][0][3] *= 2.0
    q = np.ones((layers, H, d))
    st = O.prefill_state(K, V, budget=L0 + 1)
    O.decode_step(st, 1, q, np.zeros((layers, kv, d)), np.ones((layers, kv, d)), O.Params(alpha=alpha, scorer="vnorm"))
    L = L0 + 1
    norms = np.full(L, 2.0)
    norms[3] = 4.0
    want = (1 - alpha) * (1.0 / L) * norms / norms.mean()
    assert np.max(np.abs(st.m[0] - want)) < 1e-15


# ---------------------------------------------------------------- schedule
def test_refresh_sets():
    assert [t for t in range(1, 14) if O.is_refresh(t, 4, False)] == [1, 5, 9, 13]
    assert [t for t in range(1, 6) if O.is_refresh(t, 1, False)] == [1, 2, 3, 4, 5]
    assert [t for t in range(1, 9) if O.is_refresh(t, 3, True)] == [1]


def _run(st, q, kn, vn, p, T0=1):
    outs = []
    for i in range(q.shape[0]):
        outs.append(O.decode_step(st, T0 + i, q[i], kn[i], vn[i], p))
    return outs


@pytest.mark.parametrize("gran", [O.GRAN_SEQ, O.GRAN_KVHEAD])
def test_lazy_r1_equals_full_refresh(gran):
    rng = np.random.default_rng(9)
    st = _rand_state(rng, gran=gran)
    q, kn, vn = _rand_inputs(rng, 10)
    a, b = _clone(st), _clone(st)
    oa = _run(a, q, kn, vn, O.Params(alpha=0.8, refresh_period=1, granularity=gran))
    ob = _run(b, q, kn, vn, O.Params(alpha=0.8, granularity=gran))
    assert all(np.array_equal(x, y) for x, y in zip(oa, ob))
    assert np.array_equal(a.m, b.m) and np.array_equal(a.pos, b.pos)


def test_lazy_off_refresh_state_carried_and_mean_init():
    """Eq. 6: off-refresh m_t = m_{t-1} (survivors bit-unchanged); the new token gets the
    mean of the existing L_t - 1 tokens (Appendix 'New token insertion')."""
    rng = np.random.default_rng(10)
    st = _rand_state(rng)
    q, kn, vn = _rand_inputs(rng, 9)
    p = O.Params(alpha=0.8, refresh_period=3)
    for i in range(9):
        t = i + 1
        before = dict(zip(st.pos[0].tolist(), st.m[0].tolist()))
        mean_before = float(np.mean(st.m[0]))
        new_pos = st.next_pos
        O.decode_step(st, t, q[i], kn[i], vn[i], p)
        if not O.is_refresh(t, 3, False):
            for pos, m in zip(st.pos[0].tolist(), st.m[0].tolist()):
                if pos == new_pos:
                    assert m == mean_before
                else:
                    assert m == before[pos]
        assert st.length == min(st.budget, st.length)


def test_score_free_equals_lazy_with_long_period():
    rng = np.random.default_rng(11)
    st = _rand_state(rng)
    q, kn, vn = _rand_inputs(rng, 8)
    a, b, c = _clone(st), _clone(st), _clone(st)
    oa = _run(a, q, kn, vn, O.Params(alpha=0.9, score_free=True))
    ob = _run(b, q, kn, vn, O.Params(alpha=0.9, refresh_period=100))
    assert all(np.array_equal(x, y) for x, y in zip(oa, ob))
    assert np.array_equal(a.m, b.m) and np.array_equal(a.pos, b.pos)
    # step 1 of Score-Free equals step 1 of full refresh
    O.decode_step(c, 1, q[0], kn[0], vn[0], O.Params(alpha=0.9))
    d = _clone(st)
    O.decode_step(d, 1, q[0], kn[0], vn[0], O.Params(alpha=0.9, score_free=True))
    assert np.array_equal(c.m, d.m) and np.array_equal(c.pos, d.pos)


def test_score_free_freezes_prefill_ranking():
    rng = np.random.default_rng(12)
    st = _rand_state(rng, L0=60, budget=20)
    q, kn, vn = _rand_inputs(rng, 10)
    p = O.Params(alpha=0.9, score_free=True)
    O.decode_step(st, 1, q[0], kn[0], vn[0], p)
    frozen = {pos: m for pos, m in zip(st.pos[0].tolist(), st.m[0].tolist()) if pos < 60}
    for i in range(1, 10):
        O.decode_step(st, i + 1, q[i], kn[i], vn[i], p)
        for pos, m in zip(st.pos[0].tolist(), st.m[0].tolist()):
            if pos < 60:
                assert m == frozen[pos]


# ---------------------------------------------------------------- selection / eviction
def _valid_by_definition(m, keep, B):
    """Brute-force check of Sec. 3's rule with the tie reading: every kept token ranks
    above every evicted one under (NaN lowest, m descending, slot ascending)."""
    def rank_key(i):
        x = m[i]
        return (0 if math.isnan(x) else 1, -math.inf if math.isnan(x) else x, -i)
    ks = set(keep)
    if len(ks) != min(B, len(m)):
        return False
    return all(rank_key(i) > rank_key(j) for i in ks for j in range(len(m)) if j not in ks)


def test_selection_golden():
    for c in _load("selection_cases.json")["cases"]:
        m = np.array([float(x) for x in c["m"]])
        keep = O.select_keep(m, c["B"])
        assert keep.tolist() == c["keep"], c


def test_selection_bruteforce_subsets():
    rng = np.random.default_rng(13)
    pool = [0.0, -0.0, 0.25, 0.5, 1.0, -1.0, np.inf, -np.inf, np.nan, 1e-300]
    for trial in range(300):
        L = int(rng.integers(1, 8))
        m = np.array([pool[int(i)] for i in rng.integers(0, len(pool), L)])
        for B in range(0, L + 2):
            keep = O.select_keep(m, B).tolist()
            valid = [list(S) for S in itertools.combinations(range(L), min(B, L))
                     if _valid_by_definition(m, list(S), B)]
            assert valid == [keep], (m, B, keep, valid)


def test_selection_positive_scale_invariance():
    """Corollary 2: uniform positive scaling is invisible to the ranking."""
    rng = np.random.default_rng(14)
    for _ in range(50):
        m = rng.random(200) ** 3
        B = int(rng.integers(1, 200))
        for c in (3.7, 1e-6, 2.0 ** 40):
            assert np.array_equal(O.select_keep(m, B), O.select_keep(c * m, B))


@pytest.mark.parametrize("r,sf", [(1, False), (4, False), (1, True)])
def test_budget_always_holds_and_compaction_is_stable(r, sf):
    """Appendix 'Eviction on non-refresh steps': |cache| <= B on every step; kept rows are
    the previous rows at the kept slots, in ascending slot order (stable)."""
    rng = np.random.default_rng(15)
    st = _rand_state(rng, L0=50, budget=17)
    q, kn, vn = _rand_inputs(rng, 12)
    p = O.Params(alpha=0.85, refresh_period=r, score_free=sf)
    for i in range(12):
        t = i + 1
        refresh = O.is_refresh(t, r, sf)
        O.append_token(st, kn[i], vn[i], refresh, p)
        O.attend_and_score(st, q[i], refresh, p)
        snap = _clone(st)
        keeps = O.evict(st)
        assert st.length == min(snap.length, st.budget)
        k = keeps[0]
        assert np.all(np.diff(k) > 0)
        assert _valid_by_definition(snap.m[0].tolist(), k.tolist(), st.budget)
        assert np.array_equal(st.pos[0], snap.pos[0][k])
        assert np.array_equal(st.m[0], snap.m[0][k])
        for l in range(st.layers):
            for g in range(st.kv_heads):
                assert np.array_equal(st.K[l][g], snap.K[l][g][k])
                assert np.array_equal(st.V[l][g], snap.V[l][g][k])


def test_kvhead_rows_select_independently():
    rng = np.random.default_rng(16)
    st = _rand_state(rng, gran=O.GRAN_KVHEAD, L0=30, budget=9)
    q, kn, vn = _rand_inputs(rng, 3)
    p = O.Params(alpha=0.8, granularity=O.GRAN_KVHEAD)
    O.append_token(st, kn[0], vn[0], True, p)
    O.attend_and_score(st, q[0], True, p)
    snap = _clone(st)
    O.evict(st)
    for g in range(st.kv_heads):
        k = O.select_keep(snap.m[g], 9)
        assert np.array_equal(st.pos[g], snap.pos[g][k])
        for l in range(st.layers):
            assert np.array_equal(st.K[l][g], snap.K[l][g][k])
    assert not np.array_equal(st.pos[0], st.pos[1])


def test_new_token_can_be_evicted_same_step():
    """Appendix: the new token may be evicted on the step it arrives (non-refresh, mean init
    below every survivor when the existing state is uniform except one low token)."""
    K = [[np.zeros((4, 2))]]
    V = [[np.zeros((4, 2))]]
    st = O.prefill_state(K, V, budget=4)
    st.m[0] = np.array([1.0, 1.0, 1.0, 0.2])   # mean 0.8 < 1.0 but > 0.2
    O.append_token(st, np.zeros((1, 1, 2)), np.zeros((1, 1, 2)), False, O.Params())
    assert st.m[0, -1] == pytest.approx(0.8)
    O.evict(st)
    assert st.pos[0].tolist() == [0, 1, 2, 4]
    st.m[0] = np.array([1.0, 1.0, 1.0, 1.0])
    O.append_token(st, np.zeros((1, 1, 2)), np.zeros((1, 1, 2)), False, O.Params())
    O.evict(st)  # mean 1.0 ties every survivor; the new token holds the highest slot
    assert st.pos[0].tolist() == [0, 1, 2, 4]


# ------------------------------------------------ per-layer immediate eviction (R10)
def _layerwise_from(st):
    return O.layerwise_prefill_state([[k.copy() for k in row] for row in st.K],
                                     [[v.copy() for v in row] for row in st.V], st.budget)


@pytest.mark.parametrize("r,sf", [(1, False), (3, False), (1, True)])
def test_layerwise_with_one_layer_is_the_base_method(r, sf):
    """One layer: the per-layer eviction after the layer's update is the step-end eviction,
    and every live position is held by that layer -- identical to decode_step."""
    rng = np.random.default_rng(11)
    base = _rand_state(rng, layers=1, kv=2, L0=30, budget=9)
    lw = _layerwise_from(base)
    p = O.Params(alpha=0.8, refresh_period=r, score_free=sf)
    q, kn, vn = _rand_inputs(rng, 8, layers=1)
    for t in range(1, 9):
        o_base = O.decode_step(base, t, q[t - 1], kn[t - 1], vn[t - 1], p)
        o_lw, _ = O.decode_step_layerwise(lw, t, q[t - 1], kn[t - 1], vn[t - 1], p)
        assert np.array_equal(o_base, o_lw)
        assert np.array_equal(base.pos[0], lw.pos[0])
        assert np.array_equal(base.m[0], lw.m[lw.pos[0]])


def _worked_example(refresh_period):
    """Two layers, one head, d = 1, q = 1 (so each logit is the key itself), budget 2,
    alpha 1/2, prefill positions 0 and 1; tokens 2 and 3 arrive at steps 1 and 2.
    Keys are logs of small integers, so every softmax is a ratio of integers:
        layer 0: positions 0..3 -> ln 1, ln 2, ln 3, ln 1
        layer 1: positions 0..3 -> ln 3, ln 2, ln 2, ln 6
    Values: v = 10 * layer + position (one dimension)."""
    lnk = [[math.log(1), math.log(2), math.log(3), math.log(1)], [math.log(3), math.log(2), math.log(2), math.log(6)]]
    K = [[np.array([[lnk[l][0]], [lnk[l][1]]])] for l in range(2)]
    V = [[np.array([[10.0 * l + 0], [10.0 * l + 1]])] for l in range(2)]
    st = O.layerwise_prefill_state(K, V, budget=2)
    p = O.Params(alpha=0.5, refresh_period=refresh_period)
    steps = []
    for t, newp in ((1, 2), (2, 3)):
        q = np.ones((2, 1, 1))
        kn = np.array([[[lnk[l][newp]]] for l in range(2)])
        vn = np.array([[[10.0 * l + newp]] for l in range(2)])
        out, tr = O.decode_step_layerwise(st, t, q, kn, vn, p)
        steps.append((out, tr, [x.copy() for x in st.pos], st.m.copy()))
    return steps


def test_layerwise_worked_example_full_refresh():
    """Hand-derived from Eq. 1, Eq. 4 and reading R10.
    Step 1, layer 0 attends [0,1,2] with weights 1:2:3, so m = (1/12, 2/12, 3/12) and it keeps
    {1, 2}.  Layer 1 attends [0,1,2] with 3:2:2 (the position layer 0 dropped is still live
    through layer 1): m = m/2 + (3/14, 1/7, 1/7) = (43, 38, 45)/168; it keeps {0, 2}.
    Step 2 appends 3 with m = 0.  Layer 0 attends [1,2,3] with 2:3:1; position 0 (held only by
    layer 1) gets score 0 and decays: m = (43, 94, 129, 28)/336; layer 0 keeps {1, 2}.
    Layer 1 attends [0,2,3] with 3:2:6 (position 1, held only by layer 0, decays):
    m = (1481, 1034, 2091, 2324)/7392; layer 1 keeps {2, 3}."""
    (o1, tr1, pos1, m1), (o2, tr2, pos2, m2) = _worked_example(1)
    assert [list(x) for x in pos1] == [[1, 2], [0, 2]]
    np.testing.assert_allclose(tr1[0].m, np.array([1, 2, 3]) / 12, rtol=1e-15)
    np.testing.assert_allclose(m1, np.array([43, 38, 45]) / 168, rtol=1e-15)
    assert [list(x) for x in pos2] == [[1, 2], [2, 3]]
    np.testing.assert_allclose(tr2[0].m, np.array([94, 129, 28]) / 336, rtol=1e-15)
    np.testing.assert_allclose(m2, np.array([1481, 1034, 2091, 2324]) / 7392, rtol=1e-15)
    # outputs: softmax-weighted values of each layer's held tokens at attention time
    np.testing.assert_allclose(o1[0, 0, 0], (1 * 0 + 2 * 1 + 3 * 2) / 6, rtol=1e-15)
    np.testing.assert_allclose(o1[1, 0, 0], (3 * 10 + 2 * 11 + 2 * 12) / 7, rtol=1e-15)
    np.testing.assert_allclose(o2[0, 0, 0], (2 * 1 + 3 * 2 + 1 * 3) / 6, rtol=1e-15)
    np.testing.assert_allclose(o2[1, 0, 0], (3 * 10 + 2 * 12 + 6 * 13) / 11, rtol=1e-15)


def test_layerwise_worked_example_lazy_mean_init():
    """Refresh period 2: step 2 carries the state; the new token starts at the mean over the
    live positions {0, 1, 2} (position 0 is held by layer 1 only): (43+38+45)/(3*168) = 42/168.
    Layer 0 then keeps {2, 3} from (38, 45, 42)/168 and layer 1 keeps {0, 2} from (43, 45, 42)/168."""
    (_, _, pos1, m1), (_, tr2, pos2, m2) = _worked_example(2)
    assert [list(x) for x in pos1] == [[1, 2], [0, 2]]
    np.testing.assert_allclose(m2, np.array([43, 38, 45, 42]) / 168, rtol=1e-15)
    assert [list(x) for x in pos2] == [[2, 3], [0, 2]]
    np.testing.assert_allclose(tr2[1].m, np.array([43, 45, 42]) / 168, rtol=1e-15)


def test_layerwise_alpha_one_keeps_the_oldest_everywhere():
    """alpha = 1: Eq. 4 never moves the state, refresh steps give new tokens 0, so every layer
    ranks all-equal utilities and keeps its lowest slots (R4) -- the B oldest positions, in
    every layer, as the base method does."""
    rng = np.random.default_rng(5)
    base = _rand_state(rng, layers=3, kv=2, L0=20, budget=7)
    lw = _layerwise_from(base)
    p = O.Params(alpha=1.0)
    q, kn, vn = _rand_inputs(rng, 5, layers=3)
    for t in range(1, 6):
        O.decode_step(base, t, q[t - 1], kn[t - 1], vn[t - 1], p)
        O.decode_step_layerwise(lw, t, q[t - 1], kn[t - 1], vn[t - 1], p)
        for l in range(3):
            assert list(lw.pos[l]) == list(range(7)) == list(base.pos[0])


def test_layerwise_invariants():
    """Every layer holds min(L, B) tokens in ascending position order, drawn from what it held
    plus the new token; each layer's choice is the top B of its held tokens by the state it
    saw (R4 ties); live positions are exactly the union of the layers' sets."""
    rng = np.random.default_rng(8)
    base = _rand_state(rng, layers=4, kv=2, L0=25, budget=8)
    lw = _layerwise_from(base)
    p = O.Params(alpha=0.7, refresh_period=2)
    q, kn, vn = _rand_inputs(rng, 10, layers=4)
    diverged = False
    for t in range(1, 11):
        before = [set(x.tolist()) | {lw.next_pos} for x in lw.pos]
        _, tr = O.decode_step_layerwise(lw, t, q[t - 1], kn[t - 1], vn[t - 1], p)
        for l in range(4):
            held = lw.pos[l]
            assert len(held) == 8 and np.all(np.diff(held) > 0)
            assert set(held.tolist()) <= before[l]
            order = sorted(range(len(tr[l].m)), key=lambda i: (-tr[l].m[i], i))[:8]
            assert set(tr[l].pos[order].tolist()) == set(held.tolist())
        assert set(lw.live().tolist()) == set().union(*[set(x.tolist()) for x in lw.pos])
        diverged |= len({tuple(x) for x in lw.pos}) > 1
    assert diverged  # the layers' sets do part ways on this input


# ------------------------------------------------------- rank-trace diagnostics (R11)
def test_rank_trace_set_measures_closed_forms():
    assert O.churn(np.array([1, 2, 3, 4]), np.array([1, 2, 3, 4])) == 0.0
    assert O.churn(np.array([1, 2, 3, 4]), np.array([5, 6, 7, 8])) == 1.0
    assert O.churn(np.array([1, 2, 3, 4]), np.array([0, 2, 3, 9])) == 0.5
    assert O.jaccard(np.array([1, 2, 3]), np.array([2, 3, 4])) == 0.5
    assert O.raw_top_evicted(np.array([1, 2, 3, 4]), np.array([2, 4, 6, 8])) == 0.5
    # ties go to the lower slot (R4), the result is in position order
    assert list(O.topk_positions(np.array([0.5, 0.2, 0.5, 0.9]), np.array([40, 10, 30, 20]), 2)) == [20, 40]


def test_rank_trace_alpha_zero_raw_equals_ema():
    """alpha = 0: the state after a refresh step is the last eligible layer's score (Eq. 4),
    i.e. the raw score itself, so the kept set is the raw top-k: Jaccard 1, nothing of the
    raw top-k evicted, equal churns."""
    rng = np.random.default_rng(21)
    st = _rand_state(rng, layers=3, kv=2, L0=30, budget=9)
    p = O.Params(alpha=0.0)
    q, kn, vn = _rand_inputs(rng, 6, layers=3)
    prev = None
    for t in range(1, 7):
        _, sets = O.decode_step_traced(st, t, q[t - 1], kn[t - 1], vn[t - 1], p)
        R, E = sets[0]
        assert O.jaccard(R, E) == 1.0 and O.raw_top_evicted(R, E) == 0.0
        if prev is not None:
            assert O.churn(R, prev[0]) == O.churn(E, prev[1])
        prev = (R, E)


def test_rank_trace_alpha_one_freezes_the_kept_set():
    """alpha = 1: utilities never move and new tokens start at 0 on refresh steps, so every
    step evicts the new token and the EMA top-k never changes (churn 0), while the raw
    top-k follows the queries."""
    rng = np.random.default_rng(22)
    st = _rand_state(rng, layers=2, kv=2, L0=24, budget=8)
    p = O.Params(alpha=1.0)
    q, kn, vn = _rand_inputs(rng, 6, layers=2)
    prev = None
    raw_churns = []
    for t in range(1, 7):
        _, sets = O.decode_step_traced(st, t, q[t - 1], kn[t - 1], vn[t - 1], p)
        R, E = sets[0]
        if prev is not None:
            assert O.churn(E, prev[1]) == 0.0
            raw_churns.append(O.churn(R, prev[0]))
        prev = (R, E)
    assert max(raw_churns) > 0.0


def test_rank_trace_raw_is_last_eligible_layer_score():
    """The traced raw score is the last eligible layer's Eq. 1 score, which single-step
    aggregation (Eq. 2) also leaves as the utility."""
    rng = np.random.default_rng(23)
    a = _rand_state(rng, layers=3, kv=2, L0=20, budget=30)   # no eviction: compare full rows
    b = _clone(a)
    q, kn, vn = _rand_inputs(rng, 1, layers=3)
    O.decode_step(a, 1, q[0], kn[0], vn[0], O.Params(alpha=0.8, layer_mask=[True, True, False]))
    O.decode_step(b, 1, q[0], kn[0], vn[0], O.Params(aggregation="single", layer_mask=[True, True, False]))
    np.testing.assert_array_equal(a.raw, b.m)


# ------------------------------------- the step with rows fetched by position
def _position_table(rng, layers, kv, n_pos, d, heavy=True):
    """K/V rows of every (layer, KV head, original position): the cache a sequence would
    hold, addressed by position."""
    K = rng.standard_normal((layers, kv, n_pos, d))
    V = rng.standard_normal((layers, kv, n_pos, d))
    if heavy:
        K[:, :, ::7] *= 3.0
    return K, V


_STREAM_CASES = [
    dict(),                                                     # full refresh, Eq. 4
    dict(refresh_period=3),                                     # Lazy-3 (Eq. 6)
    dict(score_free=True),                                      # Score-Free
    dict(refresh_init="mean", layer_mask=[True, False, True]),  # mean init, sparse layer mask
    dict(gran=O.GRAN_KVHEAD, refresh_period=2),                 # one row per KV head
    dict(scorer="vnorm"),
    dict(scorer="entropy", refresh_period=2),
    dict(aggregation="cumulative"),
    dict(aggregation="single"),
]


@pytest.mark.parametrize("case", _STREAM_CASES, ids=[str(i) for i in range(len(_STREAM_CASES))])
def test_streaming_step_equals_cache_holding_step(case):
    """decode_step_streaming keeps only (positions, utilities) and fetches rows by position;
    on the same sequence it gives decode_step's outputs, utilities and kept positions bit
    for bit over a run that evicts every step (positions are the rows' identity, so the
    position bookkeeping is what this pins)."""
    case = dict(case)
    gran = case.pop("gran", O.GRAN_SEQ)
    rng = np.random.default_rng(31)
    layers, kv, H, d, L0, B, T = 3, 2, 4, 8, 30, 10, 9
    Kt, Vt = _position_table(rng, layers, kv, L0 + T, d)
    held = O.prefill_state([[Kt[l, g, :L0] for g in range(kv)] for l in range(layers)],
                           [[Vt[l, g, :L0] for g in range(kv)] for l in range(layers)], B, gran)
    st = O.stream_prefill_state(L0, B, layers, kv, gran)
    p = O.Params(alpha=0.8, **case)
    q = rng.standard_normal((T, layers, H, d))
    fetched = []

    def rows(l, g, positions):
        fetched.append(len(positions))
        return Kt[l, g, positions], Vt[l, g, positions]

    for t in range(1, T + 1):
        newp = L0 + t - 1
        o_held = O.decode_step(held, t, q[t - 1], Kt[:, :, newp], Vt[:, :, newp], p)
        o_st = O.decode_step_streaming(st, t, q[t - 1], rows, p)
        assert np.array_equal(o_held, o_st), t
        assert np.array_equal(held.m, st.m), t
        assert np.array_equal(held.pos, st.pos), t
        assert st.length == min(L0 + t, B)
    assert min(fetched) == B + 1  # steady state: the budget plus the new token


def test_streaming_step_adopts_an_override_like_evict():
    """keep_override replaces the row's own choice exactly as evict(keep_override=...) does."""
    rng = np.random.default_rng(32)
    layers, kv, H, d, L0, B, T = 2, 2, 4, 8, 20, 6, 4
    Kt, Vt = _position_table(rng, layers, kv, L0 + T, d)
    held = O.prefill_state([[Kt[l, g, :L0] for g in range(kv)] for l in range(layers)],
                           [[Vt[l, g, :L0] for g in range(kv)] for l in range(layers)], B)
    st = O.stream_prefill_state(L0, B, layers, kv)
    p = O.Params(alpha=0.5)
    q = rng.standard_normal((T, layers, H, d))
    seen = []

    def pick(r, m_row, pos_row):  # any B slots: here the oldest ones
        seen.append((m_row.copy(), pos_row.copy()))
        return np.arange(min(B, len(m_row)))

    for t in range(1, T + 1):
        newp = L0 + t - 1
        O.append_token(held, Kt[:, :, newp], Vt[:, :, newp], O.is_refresh(t, 1, False), p)
        o_held = O.attend_and_score(held, q[t - 1], True, p)
        m_before = held.m[0].copy()
        O.evict(held, keep_override=[np.arange(min(B, held.length))])
        o_st = O.decode_step_streaming(st, t, q[t - 1], lambda l, g, ps: (Kt[l, g, ps], Vt[l, g, ps]), p,
                                       keep_override=pick)
        assert np.array_equal(o_held, o_st)
        assert np.array_equal(seen[-1][0], m_before)       # the override sees the state the selection sees
        assert np.array_equal(held.pos, st.pos) and np.array_equal(held.m, st.m)
    assert st.pos[0].tolist() == list(range(B))


def test_streaming_step_with_generator_rows_by_position():
    """The workload generator's rows at arbitrary positions are the rows of its prefill
    block and of its appended tokens, so the streaming oracle driven by kv_rows follows the
    cache-holding oracle on a generated (bf16) workload."""
    import gen

    w = gen.Workload("pin", 2, 2, 8, 2, 64, [90, 70], 5, dtype=gen.BF16, seed=12, page_size=16)
    u = w.u_table()
    qs = w.queries(1, w.steps + 1, u)
    q64 = gen.bf16_to_f32(qs).astype(np.float64)
    p = O.Params(alpha=0.9, refresh_period=2)
    B = w.budgets()
    for b in range(w.batch):
        K, V = [], []
        for l in range(w.layers):
            k, v = w.kv_block(b, l, 0, w.prefill[b], u)
            K.append([k[g].astype(np.float64) for g in range(w.kv_heads)])
            V.append([v[g].astype(np.float64) for g in range(w.kv_heads)])
        held = O.prefill_state(K, V, B[b])
        st = O.stream_prefill_state(w.prefill[b], B[b], w.layers, w.kv_heads)

        def rows(l, g, positions, b=b):
            k, v = w.kv_rows(b, l, positions, u)
            return k[g], v[g]

        for t in range(1, w.steps + 1):
            kn, vn = w.new_tokens(t, u)
            o_held = O.decode_step(held, t, q64[t - 1][:, b], kn[:, b], vn[:, b], p)
            o_st = O.decode_step_streaming(st, t, q64[t - 1][:, b], rows, p)
            assert np.array_equal(o_held, o_st), (b, t)
            assert np.array_equal(held.m, st.m) and np.array_equal(held.pos, st.pos), (b, t)


@pytest.mark.parametrize("case", [dict(), dict(refresh_period=3), dict(score_free=True),
                                  dict(refresh_init="mean", layer_mask=[False, True, True, False])],
                         ids=["full", "lazy3", "score_free", "mean_sparse"])
def test_layerwise_streaming_equals_cache_holding_step(case):
    """decode_step_layerwise_streaming (reading R10 with rows fetched by position) gives
    decode_step_layerwise's outputs, per-layer kept positions, states and traces bit for bit."""
    rng = np.random.default_rng(33)
    layers, kv, H, d, L0, B, T = 4, 2, 4, 8, 26, 8, 8
    Kt, Vt = _position_table(rng, layers, kv, L0 + T, d)
    held = O.layerwise_prefill_state([[Kt[l, g, :L0] for g in range(kv)] for l in range(layers)],
                                     [[Vt[l, g, :L0] for g in range(kv)] for l in range(layers)], B)
    st = O.layerwise_stream_prefill_state(L0, B, layers, kv)
    p = O.Params(alpha=0.7, **case)
    q = rng.standard_normal((T, layers, H, d))
    diverged = False
    for t in range(1, T + 1):
        newp = L0 + t - 1
        o_held, tr_h = O.decode_step_layerwise(held, t, q[t - 1], Kt[:, :, newp], Vt[:, :, newp], p)
        o_st, tr_s = O.decode_step_layerwise_streaming(st, t, q[t - 1],
                                                       lambda l, g, ps: (Kt[l, g, ps], Vt[l, g, ps]), p)
        assert np.array_equal(o_held, o_st), t
        assert np.array_equal(held.m, st.m), t
        for l in range(layers):
            assert np.array_equal(held.pos[l], st.pos[l]), (t, l)
            assert np.array_equal(tr_h[l].m, tr_s[l].m) and np.array_equal(tr_h[l].kept, tr_s[l].kept)
        diverged |= any(not np.array_equal(st.pos[0], st.pos[l]) for l in range(1, layers))
    if not case:
        assert diverged  # the layers' sets do differ, so every layer's bookkeeping is exercised
