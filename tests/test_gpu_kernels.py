"""Per-entry-point parity of the CUDA library against the CPU oracle (GPU only).

Inputs: seeded draws from ``gen``.  Expected values: ``oracle`` only.
Sizes span several 64-token tiles, several split-K partitions and ragged tails.
"""
import ctypes

import numpy as np
import pytest
import torch

import gen
import oracle as O
from harness import as_f64, fill_device, make_cache, to_device
from paper_2609_03515_gb300 import DecodeCache, ikv

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    import __graft_entry__

    __graft_entry__.build()


# ------------------------------------------------------------------ generator
def test_device_generator_matches_host_bits():
    w = gen.Workload("t", 3, 2, 8, 2, 128, [100, 257, 64], 4, dtype=gen.BF16, seed=11, page_size=32)
    u = w.u_table()
    c = make_cache(w, page_perm_seed=3)
    fill_device(c, w, torch.from_numpy(u).cuda())
    torch.cuda.synchronize()
    for b in range(w.batch):
        for l in range(w.layers):
            k, v = w.kv_block(b, l, 0, w.prefill[b], u)
            for g in range(w.kv_heads):
                gk = c.gather(c.k, b, l, g, w.prefill[b]).float().cpu().numpy()
                gv = c.gather(c.v, b, l, g, w.prefill[b]).float().cpu().numpy()
                assert np.array_equal(gk, k[g]) and np.array_equal(gv, v[g])
    # appended tokens and raw normals
    L0 = torch.tensor(w.prefill, dtype=torch.int32, device="cuda")
    kk = torch.empty((2, w.layers, w.batch, w.kv_heads, w.head_dim), dtype=torch.bfloat16, device="cuda")
    vv = torch.empty_like(kk)
    sp = w.spec()
    assert gen.cuda_lib().ikvgen_fill_tokens_cuda(ctypes.byref(sp), torch.from_numpy(u).cuda().data_ptr(),
                                                  L0.data_ptr(), 3, 5, w.dtype, kk.data_ptr(), vv.data_ptr(),
                                                  torch.cuda.current_stream().cuda_stream) == 0
    torch.cuda.synchronize()
    for i, t in enumerate((3, 4)):
        K, V = w.new_tokens(t, u)
        assert np.array_equal(kk[i].float().cpu().numpy(), K) and np.array_equal(vv[i].float().cpu().numpy(), V)
    n = 1 << 20
    dn = torch.empty(n, dtype=torch.float32, device="cuda")
    gen.cuda_lib().ikvgen_normals_cuda(5, 1, n, dn.data_ptr(), torch.cuda.current_stream().cuda_stream)
    hn = np.empty(n, np.float32)
    gen.host_lib().ikvgen_normals(5, 1, n, hn.ctypes.data)
    assert np.array_equal(dn.cpu().numpy(), hn)


# ------------------------------------------------------------------ attention + score
ATT_CASES = [
    # dtype, d, H, Hkv, lengths, gran, page_size   (bf16 / d=128 / page 8..128 | 128k -> tensor-core kernel)
    (gen.F32, 64, 4, 2, [512, 37, 1], ikv.IKV_GRAN_SEQ, 64),
    (gen.BF16, 128, 32, 8, [700, 64, 1500], ikv.IKV_GRAN_SEQ, 64),
    (gen.BF16, 128, 32, 8, [700, 129, 4100], ikv.IKV_GRAN_SEQ, 16),
    (gen.BF16, 128, 32, 8, [1, 127, 128, 2000], ikv.IKV_GRAN_SEQ, 256),
    (gen.BF16, 128, 32, 8, [700, 64, 1500], ikv.IKV_GRAN_SEQ, 48),      # page size 48: CUDA-core kernel
    (gen.BF16, 128, 28, 4, [333, 1025], ikv.IKV_GRAN_SEQ, 64),
    (gen.BF16, 128, 28, 4, [333, 1025], ikv.IKV_GRAN_KVHEAD, 32),
    (gen.BF16, 64, 8, 8, [129, 3000], ikv.IKV_GRAN_SEQ, 64),
    (gen.F32, 128, 16, 2, [65, 2100], ikv.IKV_GRAN_KVHEAD, 64),
    (gen.BF16, 128, 16, 16, [5000], ikv.IKV_GRAN_SEQ, 64),
    (gen.BF16, 128, 16, 8, [30000], ikv.IKV_GRAN_SEQ, 128),            # 2 heads per group, long split
]


@pytest.mark.parametrize("dt,d,H,Hkv,lens,gran,ps", ATT_CASES)
def test_decode_attend_score_matches_oracle(dt, d, H, Hkv, lens, gran, ps):
    w = gen.Workload("a", len(lens), 3, H, Hkv, d, lens, 1, dtype=dt, seed=21, page_size=ps)
    u = w.u_table()
    c = make_cache(w, gran, page_perm_seed=5)
    fill_device(c, w, torch.from_numpy(u).cuda())
    layer = 2
    q_h = w.queries(1, 2, u)[0, layer]                     # [batch][H][d]
    q = to_device(q_h, w)
    out = torch.empty((w.batch, H, d), dtype=q.dtype, device="cuda")
    score = torch.full((c.rows, c.cap), -7.0, device="cuda")
    rng = np.random.default_rng(3)
    ema0 = torch.from_numpy(rng.random((c.rows, c.cap)).astype(np.float32)).cuda()
    ema = ema0.clone()
    cch = c.cache(max(lens))
    ws = torch.empty(ikv.ikv_attend_workspace_size(c.shape(), cch), dtype=torch.uint8, device="cuda")
    alpha = 0.85
    ikv.ikv_decode_attend_score(c.shape(), cch, layer, q, out, score, ema, alpha, ws, ws.numel())
    torch.cuda.synchronize()
    assert ikv.ikv_device_status() == 0
    q64 = as_f64(q_h, w)
    tol_out = 2e-2 if dt == gen.BF16 else 1e-4
    R = c.rows_per_seq
    for b, L in enumerate(lens):
        k, v = w.kv_block(b, layer, 0, L, u)
        K = [k[g].astype(np.float64) for g in range(Hkv)]
        V = [v[g].astype(np.float64) for g in range(Hkv)]
        a, o = O.last_query_attention(q64[b], K, V)
        assert np.max(np.abs(out[b].float().cpu().numpy() - o)) < tol_out
        s = O.pooled_score(a, O.GRAN_SEQ if gran == ikv.IKV_GRAN_SEQ else O.GRAN_KVHEAD, Hkv)
        for rr in range(R):
            r = b * R + rr
            gs = score[r, :L].cpu().numpy()
            assert np.max(np.abs(gs - s[rr])) < 2e-5
            want = O.ema_update(ema0[r, :L].double().cpu().numpy(), s[rr], alpha)
            assert np.max(np.abs(ema[r, :L].cpu().numpy() - want)) < 2e-5
            assert torch.all(score[r, L:] == -7.0)       # nothing written past len
            assert torch.equal(ema[r, L:], ema0[r, L:])


@pytest.mark.parametrize("ps,starts,lens", [
    (64, [37, 128, 1000, 0], [700, 129, 4100, 1]),    # tensor-core kernel, chunks cut physical tiles
    (16, [5, 250], [2000, 17]),
    (48, [100, 3], [1500, 64]),                          # CUDA-core kernel
])
def test_decode_attend_score_with_start_offset(ps, starts, lens):
    """Logical slot j of sequence b lives at physical slot start[b] + j; scores land at j."""
    fill = [s + L for s, L in zip(starts, lens)]
    w = gen.Workload("a", len(lens), 2, 32, 8, 128, fill, 1, dtype=gen.BF16, seed=22, page_size=ps)
    u = w.u_table()
    c = make_cache(w, page_perm_seed=9)
    fill_device(c, w, torch.from_numpy(u).cuda())      # physical slot p holds position p
    c.start.copy_(torch.tensor(starts, dtype=torch.int32))
    c.len.copy_(torch.tensor(lens, dtype=torch.int32))
    layer = 1
    q_h = w.queries(1, 2, u)[0, layer]
    q = to_device(q_h, w)
    out = torch.empty((w.batch, 32, 128), dtype=q.dtype, device="cuda")
    score = torch.full((c.rows, c.cap), -7.0, device="cuda")
    ema = torch.zeros((c.rows, c.cap), device="cuda")
    cch = c.cache(max(lens))
    ws = torch.empty(ikv.ikv_attend_workspace_size(c.shape(), cch), dtype=torch.uint8, device="cuda")
    ikv.ikv_decode_attend_score(c.shape(), cch, layer, q, out, score, ema, 0.5, ws, ws.numel())
    torch.cuda.synchronize()
    assert ikv.ikv_device_status() == 0
    q64 = as_f64(q_h, w)
    for b, (S, L) in enumerate(zip(starts, lens)):
        k, v = w.kv_block(b, layer, S, L, u)
        a, o = O.last_query_attention(q64[b], [x.astype(np.float64) for x in k], [x.astype(np.float64) for x in v])
        assert np.max(np.abs(out[b].float().cpu().numpy() - o)) < 2e-2
        sc = O.pooled_score(a, O.GRAN_SEQ, 8)[0]
        assert np.max(np.abs(score[b, :L].cpu().numpy() - sc)) < 2e-5
        assert torch.all(score[b, L:] == -7.0)


@pytest.mark.parametrize("ps", [64, 48])   # tensor-core kernel, CUDA-core kernel
def test_decode_attend_score_skips_dead_slots(ps):
    """Dead slots (pos < 0) leave the softmax: the output and scores are the oracle's over
    the live slots, dead slots score 0.  Sequence 0 has every chunk of its first 4000 slots
    dead, sequence 1 keeps a single live slot, sequence 2 scattered holes."""
    lens = [6000, 900, 3000]
    w = gen.Workload("a", 3, 2, 32, 8, 128, lens, 1, dtype=gen.BF16, seed=23, page_size=ps)
    u = w.u_table()
    c = make_cache(w, page_perm_seed=4)
    fill_device(c, w, torch.from_numpy(u).cuda())
    rng = np.random.default_rng(15)
    pos = c.pos.cpu().numpy()
    pos[0, :4000] = -1
    pos[1, :900] = -1
    pos[1, 457] = 457
    pos[2, :3000][rng.random(3000) < 0.2] = -1
    c.pos.copy_(torch.from_numpy(pos).cuda())
    layer = 1
    q_h = w.queries(1, 2, u)[0, layer]
    q = to_device(q_h, w)
    out = torch.empty((3, 32, 128), dtype=q.dtype, device="cuda")
    score = torch.full((c.rows, c.cap), -7.0, device="cuda")
    ema0 = torch.from_numpy(rng.random((c.rows, c.cap)).astype(np.float32)).cuda()
    ema = ema0.clone()
    cch = c.cache(max(lens), dead_slots=True)
    ws = torch.empty(ikv.ikv_attend_workspace_size(c.shape(), cch), dtype=torch.uint8, device="cuda")
    alpha = 0.75
    ikv.ikv_decode_attend_score(c.shape(), cch, layer, q, out, score, ema, alpha, ws, ws.numel())
    torch.cuda.synchronize()
    assert ikv.ikv_device_status() == 0
    q64 = as_f64(q_h, w)
    for b, L in enumerate(lens):
        live = np.nonzero(pos[b, :L] >= 0)[0]
        k, v = w.kv_rows(b, layer, live, u)
        a_, o = O.last_query_attention(q64[b], [x.astype(np.float64) for x in k], [x.astype(np.float64) for x in v])
        assert np.max(np.abs(out[b].float().cpu().numpy() - o)) < 2e-2
        sc = O.pooled_score(a_, O.GRAN_SEQ, 8)[0]
        got = score[b, :L].cpu().numpy()
        assert np.max(np.abs(got[live] - sc)) < 2e-5
        dead = pos[b, :L] < 0
        assert np.all(got[dead] == 0.0)
        e0 = ema0[b, :L].cpu().numpy()
        assert np.array_equal(ema[b, :L].cpu().numpy()[dead], (np.float32(alpha) * e0[dead]).astype(np.float32))


@pytest.mark.parametrize("H,Hkv,batch", [(32, 8, 32), (28, 4, 64), (64, 8, 32), (16, 8, 32), (8, 8, 32)])
def test_attend_multi_pass_units(H, Hkv, batch):
    """256 (sequence, kv head) units of up to 30 tiles, G = 4, 7, 8, 2 and 1: the units nearly
    fill one wave of resident CTAs but their 15-tile chunks do not, so each CTA takes its
    unit's chunks as consecutive passes.  Ragged lengths (one chunk, two, an empty
    sequence), a sequence whose first chunk is all dead, one whose second chunk is all dead
    and one whose only live slot sits in its second chunk."""
    rng = np.random.default_rng(31)
    lens = [int(x) for x in rng.integers(1, 3841, size=batch)]
    lens[:6] = [3840, 3840, 3000, 0, 1920, 1921]
    w = gen.Workload("a", batch, 2, H, Hkv, 128, lens, 1, dtype=gen.BF16, seed=27, page_size=64)
    u = w.u_table()
    c = make_cache(w, page_perm_seed=8)
    fill_device(c, w, torch.from_numpy(u).cuda())
    pos = c.pos.cpu().numpy()
    pos[0, :1920] = -1          # first chunk dead
    pos[1, 1920:3840] = -1      # second chunk dead
    pos[2, :3000] = -1
    pos[2, 2500] = 2500         # one live slot, in the second chunk
    pos[6, :lens[6]][rng.random(lens[6]) < 0.3] = -1
    c.pos.copy_(torch.from_numpy(pos).cuda())
    layer = 1
    q_h = w.queries(1, 2, u)[0, layer]
    q = to_device(q_h, w)
    out = torch.full((batch, H, 128), 7.0, dtype=q.dtype, device="cuda")
    score = torch.full((c.rows, c.cap), -7.0, device="cuda")
    ema0 = torch.from_numpy(rng.random((c.rows, c.cap)).astype(np.float32)).cuda()
    ema = ema0.clone()
    cch = c.cache(max(lens), dead_slots=True)
    # the plan this device runs really is multi-pass (one layer per call)
    assert ikv.ikv_attend_plan(c.shape(), cch, 1, 0)["passes"] > 1
    ws = torch.empty(ikv.ikv_attend_workspace_size(c.shape(), cch), dtype=torch.uint8, device="cuda")
    alpha = 0.6
    ikv.ikv_decode_attend_score(c.shape(), cch, layer, q, out, score, ema, alpha, ws, ws.numel())
    torch.cuda.synchronize()
    assert ikv.ikv_device_status() == 0
    q64 = as_f64(q_h, w)
    for b, L in enumerate(lens):
        if L == 0:
            assert torch.all(out[b] == 0)
            continue
        live = np.nonzero(pos[b, :L] >= 0)[0]
        k, v = w.kv_rows(b, layer, live, u)
        a_, o = O.last_query_attention(q64[b], [x.astype(np.float64) for x in k], [x.astype(np.float64) for x in v])
        assert np.max(np.abs(out[b].float().cpu().numpy() - o)) < 2e-2, b
        sc = O.pooled_score(a_, O.GRAN_SEQ, Hkv)[0]
        got = score[b, :L].cpu().numpy()
        assert np.max(np.abs(got[live] - sc)) < 2e-5, b
        assert np.all(got[pos[b, :L] < 0] == 0.0), b
        want = O.ema_update(ema0[b, :L].double().cpu().numpy(), np.where(pos[b, :L] >= 0, 0.0, 0.0), alpha)
        want[live] = O.ema_update(ema0[b, :L].double().cpu().numpy()[live], sc, alpha)
        assert np.max(np.abs(ema[b, :L].cpu().numpy() - want)) < 2e-5, b


def _attend_case(w, c, layer, kv=None, u=None, alpha=0.5):
    """Run one attention layer through the ABI and compare it with the oracle (GRAN_SEQ)."""
    u = w.u_table() if u is None else u
    q_h = w.queries(1, 2, u)[0, layer]
    q = to_device(q_h, w)
    out = torch.empty((w.batch, w.q_heads, w.head_dim), dtype=q.dtype, device="cuda")
    score = torch.full((c.rows, c.cap), -7.0, device="cuda")
    ema = torch.zeros((c.rows, c.cap), device="cuda")
    cch = c.cache(max(w.prefill))
    ws = torch.empty(ikv.ikv_attend_workspace_size(c.shape(), cch), dtype=torch.uint8, device="cuda")
    ikv.ikv_decode_attend_score(c.shape(), cch, layer, q, out, score, ema, alpha, ws, ws.numel())
    torch.cuda.synchronize()
    assert ikv.ikv_device_status() == 0
    q64 = as_f64(q_h, w)
    for b, L in enumerate(w.prefill):
        k, v = kv[b] if kv is not None else w.kv_block(b, layer, 0, L, u)
        a_, o = O.last_query_attention(q64[b], [x.astype(np.float64) for x in k], [x.astype(np.float64) for x in v])
        assert np.max(np.abs(out[b].float().cpu().numpy() - o)) < 2e-2, b
        sc = O.pooled_score(a_, O.GRAN_SEQ, w.kv_heads)[0]
        assert np.max(np.abs(score[b, :L].cpu().numpy() - sc)) < 2e-5, b


def test_attend_dominant_late_logits():
    """Keys deep inside long units are set along their head's query, so their logits
    exceed every other by ~80 (log2 units): one slot takes nearly all of the softmax,
    in a late chunk of the split, far from the first tiles."""
    w = gen.Workload("r", 1, 2, 32, 8, 128, [40000], 1, dtype=gen.BF16, seed=24, page_size=64)
    u = w.u_table()
    c = make_cache(w, page_perm_seed=6)
    fill_device(c, w, torch.from_numpy(u).cuda())
    layer = 1
    q_h = w.queries(1, 2, u)[0, layer]                      # [batch][H][d] bf16 bits
    qf = gen.bf16_to_f32(q_h)
    k, v = w.kv_block(0, layer, 0, 40000, u)
    for slot, g in ((9000, 0), (21000, 3), (33333, 5), (39990, 7)):
        k[g][slot] = gen.bf16_to_f32(gen.f32_to_bf16_bits((5.0 * qf[0, g * 4]).astype(np.float32)))
    for g in range(8):
        c.scatter(c.k, 0, layer, g, torch.from_numpy(k[g]).cuda())
    _attend_case(w, c, layer, kv=[(k, v)], u=u)


def test_attend_many_tiny_units():
    """Units of 0..3 slots next to longer ones: one-tile chunks, mostly-masked tiles and an
    empty sequence (zero output)."""
    lens = [1, 2, 3, 0, 130, 1, 64]
    w = gen.Workload("t", len(lens), 3, 16, 8, 128, lens, 1, dtype=gen.BF16, seed=26, page_size=16)
    u = w.u_table()
    c = make_cache(w, page_perm_seed=2)
    fill_device(c, w, torch.from_numpy(u).cuda())
    q_h = w.queries(1, 2, u)[0, 2]
    q = to_device(q_h, w)
    out = torch.full((w.batch, 16, 128), 7.0, dtype=q.dtype, device="cuda")
    cch = c.cache(max(lens))
    ws = torch.empty(ikv.ikv_attend_workspace_size(c.shape(), cch), dtype=torch.uint8, device="cuda")
    ikv.ikv_decode_attend_score(c.shape(), cch, 2, q, out, None, None, 0.5, ws, ws.numel())
    torch.cuda.synchronize()
    assert ikv.ikv_device_status() == 0
    q64 = as_f64(q_h, w)
    for b, L in enumerate(lens):
        if L == 0:
            assert torch.all(out[b] == 0)
            continue
        k, v = w.kv_block(b, 2, 0, L, u)
        _, o = O.last_query_attention(q64[b], [x.astype(np.float64) for x in k], [x.astype(np.float64) for x in v])
        assert np.max(np.abs(out[b].float().cpu().numpy() - o)) < 2e-2, b


def test_decode_attend_without_score_leaves_state():
    w = gen.Workload("a", 2, 1, 32, 8, 128, [900, 50], 1, dtype=gen.BF16, seed=2)
    u = w.u_table()
    c = make_cache(w)
    fill_device(c, w, torch.from_numpy(u).cuda())
    q_h = w.queries(1, 2, u)[0, 0]
    out = torch.empty((2, 32, 128), dtype=torch.bfloat16, device="cuda")
    cch = c.cache(900)
    ws = torch.empty(ikv.ikv_attend_workspace_size(c.shape(), cch), dtype=torch.uint8, device="cuda")
    ikv.ikv_decode_attend_score(c.shape(), cch, 0, to_device(q_h, w), out, None, None, 0.9, ws, ws.numel())
    torch.cuda.synchronize()
    for b, L in enumerate(w.prefill):
        k, v = w.kv_block(b, 0, 0, L, u)
        _, o = O.last_query_attention(as_f64(q_h, w)[b], [x.astype(np.float64) for x in k],
                                      [x.astype(np.float64) for x in v])
        assert np.max(np.abs(out[b].float().cpu().numpy() - o)) < 2e-2


def test_value_norms_match_numpy():
    """ikv_value_norms: the l2 norm of every cached value row, through start and a permuted
    block table, for both dtypes."""
    for dt, d, ps in ((gen.BF16, 128, 64), (gen.F32, 64, 16)):
        w = gen.Workload("n", 3, 2, 8, 4, d, [300, 1, 777], 1, dtype=dt, seed=27, page_size=ps)
        u = w.u_table()
        c = make_cache(w, page_perm_seed=3, value_norms=True)
        fill_device(c, w, torch.from_numpy(u).cuda())
        ikv.ikv_value_norms(c.shape(), c.cache(777))
        torch.cuda.synchronize()
        got = c.vnorm.cpu().numpy()
        for b, L in enumerate(w.prefill):
            for l in range(2):
                _, v = w.kv_block(b, l, 0, L, u)
                for g in range(4):
                    want = np.sqrt(np.sum(v[g].astype(np.float64) ** 2, axis=1))
                    assert np.max(np.abs(got[l, b, g, :L] - want) / want) < 1e-5


def test_ema_update_matches_eq4():
    rng = np.random.default_rng(4)
    rows, cap = 5, 1000
    m0 = rng.random((rows, cap)).astype(np.float32)
    s = rng.random((rows, cap)).astype(np.float32)
    lens = np.array([1000, 3, 0, 999, 500], np.int32)
    ema = torch.from_numpy(m0).cuda()
    ikv.ikv_ema_update(rows, cap, ema, torch.from_numpy(s).cuda(), torch.from_numpy(lens).cuda(), 1, 0.7)
    torch.cuda.synchronize()
    got = ema.cpu().numpy()
    for r in range(rows):
        L = lens[r]
        assert np.max(np.abs(got[r, :L] - O.ema_update(m0[r, :L].astype(np.float64), s[r, :L], 0.7)), initial=0) < 1e-6
        assert np.array_equal(got[r, L:], m0[r, L:])


# ------------------------------------------------------------------ selection
def _select_gpu(util: np.ndarray, lens, budgets, rps=1, pos=None):
    rows, cap = util.shape
    keep = torch.full((rows, cap), -1, dtype=torch.int32, device="cuda")
    keep_len = torch.full((rows,), -1, dtype=torch.int32, device="cuda")
    pos_d = None if pos is None else torch.from_numpy(np.ascontiguousarray(pos, dtype=np.int32)).cuda()
    ikv.ikv_select_budget(rows, cap, torch.from_numpy(util).cuda(), torch.tensor(lens, dtype=torch.int32).cuda(), rps,
                          torch.tensor(budgets, dtype=torch.int32).cuda(), pos_d, keep, keep_len)
    torch.cuda.synchronize()
    return keep.cpu().numpy(), keep_len.cpu().numpy()


def _check_select(util, lens, budgets, rps=1):
    keep, keep_len = _select_gpu(util, lens, budgets, rps)
    for r in range(util.shape[0]):
        L, B = lens[r // rps], budgets[r // rps]
        want = O.select_keep(util[r, :L].astype(np.float64), B)
        assert keep_len[r] == len(want), (r, keep_len[r], len(want))
        assert np.array_equal(keep[r, :len(want)], want), r


@pytest.mark.parametrize("seed", [0, 1, 2])
def test_select_bit_exact_random(seed):
    rng = np.random.default_rng(seed)
    cap = 70000
    lens = [32769, 3278, 65537, 1, 7, 2049, 5000, 6555]
    budgets = [3277, 3277, 6554, 1, 0, 2048, 5000, 6554]
    util = (rng.random((len(lens), cap)) ** 4).astype(np.float32)
    _check_select(util, lens, budgets)


def test_select_ties_and_special_values():
    rng = np.random.default_rng(9)
    cap = 5000
    pool = np.array([0.0, -0.0, 0.25, 0.5, 1.0, -1.0, np.inf, -np.inf, np.nan, 1e-30, 1e-38], np.float32)
    rows = 12
    util = pool[rng.integers(0, len(pool), (rows, cap))]
    lens = [cap, cap, 4000, 1000, 11, 12, 2, 4097, 4096, 3000, 5, cap]
    budgets = [2500, 1, 3999, 999, 3, 12, 1, 4096, 4096, 2999, 0, cap - 1]
    _check_select(util, lens, budgets)
    # all equal: the lowest slots survive
    _check_select(np.full((2, 3000), 0.125, np.float32), [3000, 2999], [100, 2998])


def test_select_skips_dead_slots():
    """Dead slots (pos < 0, deferred compaction) are never kept and not counted: the kept
    set is the oracle's selection over the live slots, mapped back to their slots."""
    rng = np.random.default_rng(12)
    cap = 9000
    pool = np.array([0.0, 0.25, 0.5, 1.0, -np.inf, np.nan, 1e-30], np.float32)
    lens = [8000, 8000, 8000, 3278, 3278, 300, 5, 4097]
    dead_frac = [0.01, 0.3, 0.0, 0.02, 0.5, 0.9, 0.4, 0.25]
    rows = len(lens)
    util = (rng.random((rows, cap)) ** 4).astype(np.float32)
    util[1] = pool[rng.integers(0, len(pool), cap)]            # ties and special values among live slots
    pos = np.tile(np.arange(cap, dtype=np.int32), (rows, 1))
    n_live = []
    for r in range(rows):
        dead = rng.random(lens[r]) < dead_frac[r]
        pos[r, :lens[r]][dead] = -1
        n_live.append(int((~dead).sum()))
    # budgets: more than the live count, exactly one too many, and the general case
    budgets = [n_live[0] - 1, 1000, n_live[2] - 1, 3277, n_live[4] + 5, 10, n_live[6] - 1, 100]
    keep, keep_len = _select_gpu(util, lens, budgets, 1, pos)
    for r in range(rows):
        live = np.nonzero(pos[r, :lens[r]] >= 0)[0]
        want = live[O.select_keep(util[r, live].astype(np.float64), budgets[r])]
        assert keep_len[r] == len(want), (r, keep_len[r], len(want))
        assert np.array_equal(keep[r, :len(want)], np.sort(want)), r


def test_select_scale_invariance_on_gpu():
    """Corollary 2: uniform positive scaling does not change the kept set."""
    rng = np.random.default_rng(10)
    util = (rng.random((3, 4000)) ** 3).astype(np.float32)
    lens, budgets = [4000, 3000, 2000], [400, 2999, 7]
    k1, _ = _select_gpu(util, lens, budgets)
    k2, _ = _select_gpu((util * np.float32(4.0)).astype(np.float32), lens, budgets)   # exact power-of-two scale
    assert np.array_equal(k1, k2)


def test_select_kvhead_rows_share_length():
    rng = np.random.default_rng(11)
    util = rng.random((6, 800)).astype(np.float32)
    _check_select(util, [800, 500], [300, 10], rps=3)


# ------------------------------------------------------------------ compaction and append
@pytest.mark.parametrize("mode", [ikv.IKV_COMPACT_STABLE, ikv.IKV_COMPACT_HOLEFILL, ikv.IKV_COMPACT_STABLE_SHORT])
@pytest.mark.parametrize("gran", [ikv.IKV_GRAN_SEQ, ikv.IKV_GRAN_KVHEAD])
def test_compact_matches_oracle_eviction(mode, gran):
    w = gen.Workload("c", 3, 2, 8, 2, 128, [1000, 3278, 70], 1, dtype=gen.BF16, seed=31, page_size=16)
    u = w.u_table()
    c = make_cache(w, gran, page_perm_seed=9)
    fill_device(c, w, torch.from_numpy(u).cuda())
    rng = np.random.default_rng(12)
    util = rng.random((c.rows, c.cap)).astype(np.float32)
    if True:  # one sequence in steady state: a single eviction
        util[c.rows_per_seq:2 * c.rows_per_seq, :3278] = rng.random((c.rows_per_seq, 3278))
    c.ema.copy_(torch.from_numpy(util).cuda())
    budgets = [100, 3277, 70]
    c.budget.copy_(torch.tensor(budgets, dtype=torch.int32).cuda())
    keep = torch.empty((c.rows, c.cap), dtype=torch.int32, device="cuda")
    keep_len = torch.empty((c.rows,), dtype=torch.int32, device="cuda")
    ikv.ikv_select_budget(c.rows, c.cap, c.ema, c.len, c.rows_per_seq, c.budget, None, keep, keep_len)
    cch = c.cache(3278)
    nws = ikv.ikv_compact_workspace_size(c.shape(), cch, mode)
    ws = torch.empty(max(nws, 1), dtype=torch.uint8, device="cuda")
    ikv.ikv_compact_kv(c.shape(), cch, keep, keep_len, c.ema, mode, ws, nws)
    torch.cuda.synchronize()
    R = c.rows_per_seq
    pos = c.pos.cpu().numpy()
    ema = c.ema.cpu().numpy()
    assert c.len.cpu().tolist() == [min(L, B) for L, B in zip(w.prefill, budgets)]
    for b in range(w.batch):
        L = w.prefill[b]
        K = [[None] * w.kv_heads for _ in range(w.layers)]
        V = [[None] * w.kv_heads for _ in range(w.layers)]
        for l in range(w.layers):
            k, v = w.kv_block(b, l, 0, L, u)
            for g in range(w.kv_heads):
                K[l][g], V[l][g] = k[g].astype(np.float64), v[g].astype(np.float64)
        st = O.prefill_state(K, V, budgets[b], O.GRAN_SEQ if gran == ikv.IKV_GRAN_SEQ else O.GRAN_KVHEAD)
        st.m = util[b * R:(b + 1) * R, :L].astype(np.float64)
        O.evict(st)
        n = st.length
        for rr in range(R):
            gp = pos[b * R + rr, :n]
            if mode != ikv.IKV_COMPACT_HOLEFILL:
                assert np.array_equal(gp, st.pos[rr])
                assert np.array_equal(ema[b * R + rr, :n], st.m[rr].astype(np.float32))
            else:
                assert set(gp.tolist()) == set(st.pos[rr].tolist())
                order = np.argsort(gp)
                assert np.array_equal(ema[b * R + rr, :n][order], st.m[rr].astype(np.float32))
        for l in range(w.layers):
            for g in range(w.kv_heads):
                rr = 0 if R == 1 else g
                gp = pos[b * R + rr, :n]
                rank = np.argsort(np.argsort(gp))
                gk = c.gather(c.k, b, l, g, n).float().cpu().numpy()
                gv = c.gather(c.v, b, l, g, n).float().cpu().numpy()
                assert np.array_equal(gk, st.K[l][g][rank]) and np.array_equal(gv, st.V[l][g][rank])


@pytest.mark.parametrize("init_mean", [0, 1])
def test_append_token(init_mean):
    w = gen.Workload("p", 2, 3, 8, 2, 64, [130, 5], 1, dtype=gen.F32, seed=41, page_size=64)
    u = w.u_table()
    c = make_cache(w, ikv.IKV_GRAN_KVHEAD)
    fill_device(c, w, torch.from_numpy(u).cuda())
    rng = np.random.default_rng(13)
    m0 = rng.random((c.rows, c.cap)).astype(np.float32)
    c.ema.copy_(torch.from_numpy(m0).cuda())
    kn, vn = w.new_tokens(1, u)
    ws = torch.empty(4096, dtype=torch.uint8, device="cuda")
    ikv.ikv_append_token(c.shape(), c.cache(130), to_device(kn, w), to_device(vn, w), c.ema, init_mean, ws, 4096)
    torch.cuda.synchronize()
    assert c.len.cpu().tolist() == [131, 6] and c.next_pos.cpu().tolist() == [131, 6]
    for b, L in enumerate(w.prefill):
        for g in range(w.kv_heads):
            r = b * w.kv_heads + g
            want = O.new_token_state(m0[r, :L].astype(np.float64), refresh=not init_mean, refresh_init="zero")
            assert abs(float(c.ema[r, L]) - want) < 1e-6
            assert int(c.pos[r, L]) == L
            for l in range(w.layers):
                assert np.array_equal(c.gather(c.k, b, l, g, L + 1)[L].cpu().numpy(), kn[l, b, g])
                assert np.array_equal(c.gather(c.v, b, l, g, L + 1)[L].cpu().numpy(), vn[l, b, g])


def test_append_mean_skips_dead_slots():
    """With dead slots the new token's utility is the mean over the live slots only."""
    w = gen.Workload("p", 2, 2, 8, 2, 64, [300, 40], 1, dtype=gen.F32, seed=42, page_size=64)
    u = w.u_table()
    c = make_cache(w, ikv.IKV_GRAN_KVHEAD)
    fill_device(c, w, torch.from_numpy(u).cuda())
    rng = np.random.default_rng(14)
    m0 = rng.random((c.rows, c.cap)).astype(np.float32)
    pos = c.pos.cpu().numpy()
    for r in range(c.rows):
        pos[r, :w.prefill[r // w.kv_heads]][rng.random(w.prefill[r // w.kv_heads]) < 0.3] = -1
    c.pos.copy_(torch.from_numpy(pos).cuda())
    c.ema.copy_(torch.from_numpy(m0).cuda())
    kn, vn = w.new_tokens(1, u)
    ws = torch.empty(4096, dtype=torch.uint8, device="cuda")
    ikv.ikv_append_token(c.shape(), c.cache(300, dead_slots=True), to_device(kn, w), to_device(vn, w), c.ema, 1, ws,
                         4096)
    torch.cuda.synchronize()
    assert c.len.cpu().tolist() == [301, 41]
    for r in range(c.rows):
        L = w.prefill[r // w.kv_heads]
        live = pos[r, :L] >= 0
        want = O.new_token_state(m0[r, :L][live].astype(np.float64), refresh=False, refresh_init="zero")
        assert abs(float(c.ema[r, L]) - want) < 1e-6
        assert int(c.pos[r, L]) == L


def test_compact_short_side_moves_the_prefix():
    """Shorter-side stable compaction: an eviction near the front moves the prefix right
    and advances start; one near the back moves the suffix left; order is kept."""
    w = gen.Workload("c", 2, 2, 8, 2, 128, [3278, 3278], 1, dtype=gen.BF16, seed=33, page_size=64)
    u = w.u_table()
    c = make_cache(w, page_perm_seed=2)
    fill_device(c, w, torch.from_numpy(u).cuda())
    util = np.ones((2, c.cap), np.float32)
    util[0, 5] = 0.0       # evict slot 5 of sequence 0: 5 rows before it, 3272 after
    util[1, 3000] = 0.0    # evict slot 3000 of sequence 1: 277 rows after it
    c.ema.copy_(torch.from_numpy(util).cuda())
    c.budget.fill_(3277)
    keep = torch.empty((2, c.cap), dtype=torch.int32, device="cuda")
    keep_len = torch.empty((2,), dtype=torch.int32, device="cuda")
    ikv.ikv_select_budget(2, c.cap, c.ema, c.len, 1, c.budget, None, keep, keep_len)
    cch = c.cache(3278)
    nws = ikv.ikv_compact_workspace_size(c.shape(), cch, ikv.IKV_COMPACT_STABLE_SHORT)
    ws = torch.empty(nws, dtype=torch.uint8, device="cuda")
    ikv.ikv_compact_kv(c.shape(), cch, keep, keep_len, c.ema, ikv.IKV_COMPACT_STABLE_SHORT, ws, nws)
    torch.cuda.synchronize()
    assert c.start.cpu().tolist() == [1, 0] and c.len.cpu().tolist() == [3277, 3277]
    for b, ev in ((0, 5), (1, 3000)):
        want_pos = [p for p in range(3278) if p != ev]
        assert c.pos[b, :3277].cpu().tolist() == want_pos
        for l in range(2):
            k, v = w.kv_rows(b, l, np.array(want_pos), u)
            for g in range(2):
                assert np.array_equal(c.gather(c.k, b, l, g, 3277).float().cpu().numpy(), k[g])
                assert np.array_equal(c.gather(c.v, b, l, g, 3277).float().cpu().numpy(), v[g])


def test_compact_short_side_relocates_and_skips_in_place():
    """Shorter-side compaction at the end of the slot space: (0) the prefix would move right
    but has no room, so every row moves to slot 0 once; (1) the oldest row is evicted, so
    start advances with no row moved; (2) no room and too little slack to relocate, so the
    suffix moves left and start stays."""
    w = gen.Workload("c", 3, 2, 8, 2, 128, [3520] * 3, 1, dtype=gen.BF16, seed=34, page_size=64)
    u = w.u_table()
    c = DecodeCache(3, 2, 8, 2, 128, 3520, dtype=ikv.IKV_BF16, page_size=64, page_perm_seed=5)
    assert c.cap == 3520
    fill_device(c, w, torch.from_numpy(u).cuda())  # physical slot p holds position p
    S, L, ev = [244, 100, 70], [3276, 3276, 3450], [5, 0, 5]
    c.start.copy_(torch.tensor(S, dtype=torch.int32))
    c.len.copy_(torch.tensor(L, dtype=torch.int32))
    c.budget.copy_(torch.tensor([x - 1 for x in L], dtype=torch.int32))
    util = np.ones((3, c.cap), np.float32)
    pos = np.zeros((3, c.cap), np.int32)
    for b in range(3):
        util[b, ev[b]] = 0.0
        pos[b, :L[b]] = np.arange(S[b], S[b] + L[b])
    c.ema.copy_(torch.from_numpy(util).cuda())
    c.pos.copy_(torch.from_numpy(pos).cuda())
    keep = torch.empty((3, c.cap), dtype=torch.int32, device="cuda")
    keep_len = torch.empty((3,), dtype=torch.int32, device="cuda")
    ikv.ikv_select_budget(3, c.cap, c.ema, c.len, 1, c.budget, None, keep, keep_len)
    cch = c.cache(max(L))
    nws = ikv.ikv_compact_workspace_size(c.shape(), cch, ikv.IKV_COMPACT_STABLE_SHORT)
    ws = torch.empty(nws, dtype=torch.uint8, device="cuda")
    ikv.ikv_compact_kv(c.shape(), cch, keep, keep_len, c.ema, ikv.IKV_COMPACT_STABLE_SHORT, ws, nws)
    torch.cuda.synchronize()
    assert c.start.cpu().tolist() == [0, 101, 70]
    assert c.len.cpu().tolist() == [x - 1 for x in L]
    for b in range(3):
        n = L[b] - 1
        want_pos = [S[b] + j for j in range(L[b]) if j != ev[b]]
        assert c.pos[b, :n].cpu().tolist() == want_pos
        for l in range(2):
            k, v = w.kv_rows(b, l, np.array(want_pos), u)
            for g in range(2):
                assert np.array_equal(c.gather(c.k, b, l, g, n).float().cpu().numpy(), k[g])
                assert np.array_equal(c.gather(c.v, b, l, g, n).float().cpu().numpy(), v[g])


def test_bounded_wait_runs_out_and_the_next_launch_is_correct():
    """The tensor-core kernel's waits are bounded.  ikv_test_stall_next_attention makes the
    next launch start with a wait (10 us) on a barrier nothing arrives at: every CTA takes its
    timeout path (abort flag, in-flight copies drained, TMEM freed, no fault), the device
    error word reports bit 0, and the following launch on the same inputs is correct."""
    w = gen.Workload("stall", 2, 2, 32, 8, 128, [700, 200], 1, dtype=gen.BF16, seed=29, page_size=64)
    u = w.u_table()
    c = make_cache(w, page_perm_seed=3)
    fill_device(c, w, torch.from_numpy(u).cuda())
    cch = c.cache(max(w.prefill))
    assert ikv.ikv_attend_path(c.shape(), cch) == ikv.IKV_PATH_TENSOR_CORE
    layer = 1
    q_h = w.queries(1, 2, u)[0, layer]
    q = to_device(q_h, w)
    ws = torch.empty(ikv.ikv_attend_workspace_size(c.shape(), cch), dtype=torch.uint8, device="cuda")
    out = torch.empty((w.batch, w.q_heads, w.head_dim), dtype=torch.bfloat16, device="cuda")
    score = torch.zeros((c.rows, c.cap), device="cuda")
    assert ikv.ikv_device_status() == 0
    ikv.ikv_test_stall_next_attention()
    ikv.ikv_decode_attend_score(c.shape(), cch, layer, q, out, score, None, 0.0, ws, ws.numel())
    torch.cuda.synchronize()
    assert ikv.ikv_device_status() & 1          # the wait ran out; the context is intact
    assert ikv.ikv_device_status() == 0         # and the word was cleared
    ikv.ikv_decode_attend_score(c.shape(), cch, layer, q, out, score, None, 0.0, ws, ws.numel())
    torch.cuda.synchronize()
    assert ikv.ikv_device_status() == 0
    q64 = as_f64(q_h, w)
    for b, L in enumerate(w.prefill):
        k, v = w.kv_block(b, layer, 0, L, u)
        a, o = O.last_query_attention(q64[b], [x.astype(np.float64) for x in k], [x.astype(np.float64) for x in v])
        assert np.max(np.abs(out[b].cpu().float().numpy() - o)) < 2e-2
        assert np.max(np.abs(score[b, :L].cpu().numpy() - O.pooled_score(a, O.GRAN_SEQ, w.kv_heads)[0])) < 2e-5
