"""Shared test plumbing: build a device cache from a workload, mirror it in the
oracle, and step both in lock-step.

Inputs come only from ``gen`` (host draws uploaded, or the device generator
whose bits are tested equal to the host's).  Expected values come only from
``oracle``.  After each step the oracle adopts the GPU's kept set when that set
is valid under the boundary rule (every token above theta + gap kept, every
token below theta - gap evicted), so legal near-tie choices cannot make the
trajectories diverge.
"""
from __future__ import annotations

import ctypes
from dataclasses import dataclass, field
from typing import List, Optional

import numpy as np
import torch

import gen
import oracle as O
from paper_2609_03515_gb300 import DecodeCache, ikv, step_lengths

GAP = 1e-4          # retained-set boundary rule
TOL_M = 1e-3        # utilities, fp32 vs fp64
TOL_OUT_BF16 = 2e-2
TOL_OUT_F32 = 1e-4


def torch_dtype(w: gen.Workload):
    return torch.bfloat16 if w.dtype == gen.BF16 else torch.float32


def make_cache(w: gen.Workload, gran: int = ikv.IKV_GRAN_SEQ, page_perm_seed: Optional[int] = 7,
               extra_cap: int = 0, value_norms: bool = False) -> DecodeCache:
    c = DecodeCache(w.batch, w.layers, w.q_heads, w.kv_heads, w.head_dim, w.cap + extra_cap,
                    dtype=ikv.IKV_BF16 if w.dtype == gen.BF16 else ikv.IKV_F32, page_size=w.page_size,
                    granularity=gran, page_perm_seed=page_perm_seed, value_norms=value_norms)
    c.set_prefill(w.prefill, w.budgets())
    return c


def fill_prefill(c: DecodeCache, w: gen.Workload, u: np.ndarray):
    """Write the prefill K/V into the device pools with the device generator and return the
    host generator's draws of the same rows for the oracle, [b][l] -> (K[g], V[g]) float64
    (the two halves agree bit for bit: test_generator_bits_host_equals_device)."""
    fill_device(c, w, torch.from_numpy(u).cuda())
    kv = []
    for b in range(w.batch):
        per_l = []
        for l in range(w.layers):
            k, v = w.kv_block(b, l, 0, w.prefill[b], u)
            per_l.append((k.astype(np.float64), v.astype(np.float64)))
        kv.append(per_l)
    return kv


class HostPools:
    """The K/V pools and the slot map copied to the host once, gathered there (the small
    lock-step checks launch no indexing kernels this way)."""

    def __init__(self, c: DecodeCache):
        self.c = c
        self.k = c.k.cpu().float().numpy()
        self.v = c.v.cpu().float().numpy()
        self.bt = c.block_table.cpu().numpy()
        self.start = c.start.cpu().numpy()

    def rows(self, pool: np.ndarray, b: int, l: int, g: int, n: int) -> np.ndarray:
        slots = np.arange(n) + int(self.start[b])
        pages = self.bt[b, slots // self.c.page_size]
        return pool[l, pages, g, slots % self.c.page_size]


def fill_device(c: DecodeCache, w: gen.Workload, u_dev: torch.Tensor) -> None:
    sp = w.spec()
    L0 = torch.tensor(w.prefill, dtype=torch.int32, device="cuda")
    st = torch.cuda.current_stream().cuda_stream
    rc = gen.cuda_lib().ikvgen_fill_paged_cuda(ctypes.byref(sp), u_dev.data_ptr(), c.k.data_ptr(), c.v.data_ptr(),
                                               c.block_table.data_ptr(), L0.data_ptr(), c.num_pages, c.page_size,
                                               c.max_pages, max(w.prefill), w.dtype, st)
    assert rc == 0, rc


def oracle_states(w: gen.Workload, kv, gran: int) -> List[O.SeqState]:
    sts = []
    for b in range(w.batch):
        K = [[kv[b][l][0][g] for g in range(w.kv_heads)] for l in range(w.layers)]
        V = [[kv[b][l][1][g] for g in range(w.kv_heads)] for l in range(w.layers)]
        sts.append(O.prefill_state(K, V, w.budgets()[b], O.GRAN_SEQ if gran == ikv.IKV_GRAN_SEQ else O.GRAN_KVHEAD))
    return sts


def as_f64(x: np.ndarray, w: gen.Workload) -> np.ndarray:
    if w.dtype == gen.BF16:
        return gen.bf16_to_f32(x).astype(np.float64)
    return x.astype(np.float64)


def to_device(x: np.ndarray, w: gen.Workload) -> torch.Tensor:
    """Host array (bf16 bits or fp32) -> device tensor of the workload dtype."""
    if w.dtype == gen.BF16:
        if x.dtype != np.uint16:
            x = gen.f32_to_bf16_bits(x)
        return torch.from_numpy(x.view(np.int16)).cuda().view(torch.bfloat16)
    return torch.from_numpy(np.ascontiguousarray(x, np.float32)).cuda()


def boundary_ok(m_o: np.ndarray, kept_mask: np.ndarray, budget: int, gap: float = GAP, relative: bool = False):
    """Retained-set rule against the oracle's utilities m_o (one row): with theta the
    oracle's B-th largest utility, every token above theta + gap is kept and every token
    below theta - gap evicted.  relative: the gap is gap * theta (the stricter rule for
    utilities far below 1)."""
    L = m_o.shape[0]
    if L <= budget:
        return bool(kept_mask.all()), 0.0
    theta = np.sort(m_o)[::-1][budget - 1]
    if relative:
        gap = gap * abs(theta)
    must_keep = m_o > theta + gap
    must_drop = m_o < theta - gap
    ok = bool(np.all(kept_mask[must_keep]) and not np.any(kept_mask[must_drop]) and kept_mask.sum() == budget)
    return ok, float(theta)


class Canaries:
    """Guard regions around every buffer a step writes, each holding a fixed bit pattern
    that no call may change (the substitute for a memory checker on this GPU pool):
      - spare pages in the K/V pools, interleaved at random with the used pages and never
        named by the block table;
      - tails after pos, ema and (with VNorm) vnorm;
      - a tail after the workspace.
    Install on a fresh DecodeCache before its prefill is written; check() after each call."""

    TAIL = 1024  # elements (bytes for the workspace)

    def __init__(self, c: DecodeCache, ws_bytes: int, seed: int = 11):
        self.c = c
        dev = c.k.device
        P = c.num_pages
        S = max(2, P // 3)
        rng = np.random.default_rng(seed)
        perm = rng.permutation(P + S)
        self.spare = torch.from_numpy(np.sort(perm[P:]).astype(np.int64)).to(dev)
        bt = perm[:P][c.block_table.cpu().numpy()]
        shp = list(c.k.shape)
        shp[1] = P + S
        self.ik = torch.int16 if c.k.dtype == torch.bfloat16 else torch.int32
        self.kpat = 0x7F7F if self.ik == torch.int16 else 0x7F7F7F7F  # finite values, never read
        for name in ("k", "v"):
            pool = torch.empty(shp, dtype=c.k.dtype, device=dev)
            pool.view(self.ik).fill_(self.kpat)
            used = torch.from_numpy(perm[:P].astype(np.int64)).to(dev)
            pool[:, used] = getattr(c, name)
            setattr(c, name, pool)
        c.block_table = torch.from_numpy(bt.astype(np.int32)).to(dev)
        c.num_pages = P + S
        self.tails = {}
        for name in ("pos", "ema", "vnorm"):
            t = getattr(c, name)
            if t is None:
                continue
            n = t.numel()
            big = torch.empty(n + self.TAIL, dtype=t.dtype, device=dev)
            big.view(torch.int32).fill_(0x5A5AA5A5)
            big[:n].copy_(t.reshape(-1))
            setattr(c, name, big[:n].view(t.shape))
            self.tails[name] = big[n:]
        self.ws_big = torch.zeros(ws_bytes + self.TAIL, dtype=torch.uint8, device=dev)
        self.ws_big[ws_bytes:].fill_(0xA5)
        self.ws = self.ws_big[:ws_bytes]
        self.ws_bytes = ws_bytes

    def check(self, where=""):
        c = self.c
        for name in ("k", "v"):
            pages = getattr(c, name)[:, self.spare].contiguous().view(self.ik)
            assert bool((pages == self.kpat).all()), f"{where}: a spare {name} page was written"
        for name, t in self.tails.items():
            assert bool((t.view(torch.int32) == 0x5A5AA5A5).all()), f"{where}: the tail after {name} was written"
        assert bool((self.ws_big[self.ws_bytes:] == 0xA5).all()), f"{where}: the tail after the workspace was written"


@dataclass
class StepReport:
    t: int
    out_err: float = 0.0
    m_err: float = 0.0           # kept utilities, absolute error against the oracle
    m_rel_err: float = 0.0       # the same, relative (full-size runs)
    kv_err: float = 0.0
    set_ok: bool = True          # boundary rule, absolute gap
    rel_set_ok: bool = True      # boundary rule, relative gap (full-size runs)
    strict_set_equal: bool = True
    refresh: bool = True


STABLE_MODES = (ikv.IKV_COMPACT_STABLE, ikv.IKV_COMPACT_STABLE_SHORT)


def live_slots(pos_row: np.ndarray, n: int) -> np.ndarray:
    """Logical slots below n that hold a live token (pos >= 0; -1 marks a dead slot)."""
    return np.nonzero(pos_row[:n] >= 0)[0]


def decode_step(c: DecodeCache, p, cache, t: int, q, kn, vn, out, ws, per_layer: bool = False) -> None:
    """One decode step through the C ABI: ikv_step, or its begin / per-layer / end split
    (q, kn, vn, out: [layers][batch][...] device tensors)."""
    m = c.utility(p.evict_mode)
    if not per_layer:
        ikv.ikv_step(c.shape(), p, cache, m, t, q, kn, vn, out, ws, ws.numel())
        return
    ikv.ikv_step_begin(c.shape(), p, cache, m, t, ws, ws.numel())
    for l in range(c.layers):
        ikv.ikv_step_layer(c.shape(), p, cache, m, t, l, q[l], kn[l], vn[l], out[l], ws, ws.numel())
    ikv.ikv_step_end(c.shape(), p, cache, m, t, ws, ws.numel())


def run_lockstep(w: gen.Workload, gran: int = ikv.IKV_GRAN_SEQ, compact_mode: int = ikv.IKV_COMPACT_STABLE,
                 steps: Optional[int] = None, kv_check_layers=(0, -1), page_perm_seed: Optional[int] = 7,
                 refresh_init: int = ikv.IKV_INIT_ZERO, layer_eligible=None, max_holes: int = 0,
                 agg_mode: int = ikv.IKV_AGG_EMA, scorer: int = ikv.IKV_SCORE_ATTENTION,
                 per_layer: bool = False, trace: bool = False, ws_zeroed: bool = False,
                 canaries: bool = False) -> List[StepReport]:
    T = w.steps if steps is None else steps
    u = w.u_table()
    c = make_cache(w, gran, page_perm_seed, value_norms=scorer == ikv.IKV_SCORE_VNORM)
    guard = Canaries(c, c.step_workspace().numel()) if canaries else None
    kv = fill_prefill(c, w, u)
    if c.vnorm is not None:
        ikv.ikv_value_norms(c.shape(), c.cache(max(w.prefill)))
    sts = oracle_states(w, kv, gran)
    op = O.Params(alpha=w.alpha, refresh_period=w.refresh_period, score_free=w.score_free,
                  granularity=O.GRAN_SEQ if gran == ikv.IKV_GRAN_SEQ else O.GRAN_KVHEAD,
                  layer_mask=None if layer_eligible is None else [bool(x) for x in layer_eligible],
                  refresh_init="zero" if refresh_init == ikv.IKV_INIT_ZERO else "mean",
                  aggregation={ikv.IKV_AGG_EMA: "ema", ikv.IKV_AGG_CUMULATIVE: "cumulative",
                               ikv.IKV_AGG_SINGLE_STEP: "single"}[agg_mode],
                  scorer={ikv.IKV_SCORE_ATTENTION: "attention", ikv.IKV_SCORE_VNORM: "vnorm",
                          ikv.IKV_SCORE_ENTROPY: "entropy"}[scorer])
    from paper_2609_03515_gb300 import RankTrace

    tr = RankTrace(c) if trace else None
    p = c.params(w.alpha, w.refresh_period, w.score_free, compact_mode, refresh_init, layer_eligible, max_holes,
                 agg_mode, scorer, trace=tr, ws_zeroed=ws_zeroed)
    ws = c.step_workspace() if guard is None else guard.ws
    qs = w.queries(1, T + 1, u)
    prev_sets = [(np.zeros(0, np.int64), np.zeros(0, np.int64))] * (w.batch * c.rows_per_seq)
    budgets = w.budgets()
    lens, live = list(w.prefill), list(w.prefill)
    out = torch.empty((w.layers, w.batch, w.q_heads, w.head_dim), dtype=torch_dtype(w), device="cuda")
    tol_out = TOL_OUT_BF16 if w.dtype == gen.BF16 else TOL_OUT_F32
    reports = []
    R = c.rows_per_seq
    for t in range(1, T + 1):
        kn, vn = w.new_tokens(t, u)
        decode_step(c, p, c.cache(max(lens)), t, to_device(qs[t - 1], w), to_device(kn, w), to_device(vn, w), out,
                    ws, per_layer)
        lens, live = step_lengths(lens, live, budgets, max_holes)
        torch.cuda.synchronize()
        if guard is not None:
            guard.check(f"step {t}")
        out_h = out.cpu().float().numpy()
        ema_h = c.ema.cpu().numpy()
        pos_h = c.pos.cpu().numpy()
        len_h = c.len.cpu().numpy()
        refresh = O.is_refresh(t, w.refresh_period, w.score_free)
        if tr is not None:
            cnt_h = tr.counts.cpu().numpy()
            ntop_h = tr.n_top.cpu().numpy()
            rawtop_h = tr.raw_top.cpu().numpy()
            ematop_h = tr.ema_top.cpu().numpy()
        rep = StepReport(t=t, refresh=refresh)
        q64 = as_f64(qs[t - 1], w)
        hp = HostPools(c) if kv_check_layers else None
        for b, st in enumerate(sts):
            st.raw = None
            O.append_token(st, kn[:, b], vn[:, b], refresh, op)
            o_out = O.attend_and_score(st, q64[:, b], refresh, op)
            rep.out_err = max(rep.out_err, float(np.max(np.abs(out_h[:, b] - o_out))))
            assert len_h[b] == lens[b], (t, b, len_h[b], lens[b])
            keeps = []
            for rr in range(R):
                r = b * R + rr
                ls = live_slots(pos_h[r], int(len_h[b]))
                n = len(ls)
                assert n == min(st.length, budgets[b]), (t, b, n, st.length)
                gpos = pos_h[r, ls]
                gm = ema_h[r, ls]
                if compact_mode in STABLE_MODES:  # survivors keep their order (R5)
                    assert np.all(np.diff(gpos) > 0), (t, b, rr)
                slot_of = {int(pp): i for i, pp in enumerate(st.pos[rr])}
                assert len(set(gpos.tolist())) == n
                oslots = np.array([slot_of[int(pp)] for pp in gpos])
                kept_mask = np.zeros(st.length, bool)
                kept_mask[oslots] = True
                ok, _ = boundary_ok(st.m[rr], kept_mask, budgets[b])
                rep.set_ok &= ok
                own = set(O.select_keep(st.m[rr], budgets[b]).tolist())
                rep.strict_set_equal &= own == set(oslots.tolist())
                if tr is not None:  # rank trace of this row (reading R11)
                    Et = np.sort(gpos.astype(np.int64))
                    nR, nE = int(ntop_h[r, 0]), int(ntop_h[r, 1])
                    assert nE == len(Et) and np.array_equal(ematop_h[r, :nE], Et), (t, b, rr)
                    Rp, Ep = prev_sets[r]
                    c5 = cnt_h[r]
                    assert c5[1] == len(set(Et.tolist()) & set(Ep.tolist())) and c5[4] == len(Et), (t, b, rr, c5)
                    if refresh:
                        Rt = rawtop_h[r, :nR].astype(np.int64)
                        assert np.all(np.diff(Rt) > 0) and nR == min(st.length, budgets[b])
                        rmask = np.isin(st.pos[rr], Rt)  # the oracle's raw score decides validity
                        ok_r, _ = boundary_ok(st.raw[rr], rmask, budgets[b])
                        rep.set_ok &= ok_r
                        assert c5[3] == nR and c5[0] == len(set(Rt.tolist()) & set(Rp.tolist())), (t, b, rr, c5)
                        assert c5[2] == len(set(Rt.tolist()) & set(Et.tolist())), (t, b, rr, c5)
                        prev_sets[r] = (Rt, Et)
                    else:
                        assert c5[0] == -1 and c5[2] == -1 and c5[3] == -1
                        prev_sets[r] = (Rp, Et)
                rep.m_err = max(rep.m_err, float(np.max(np.abs(gm - st.m[rr][oslots]))))
                keeps.append(np.sort(oslots))
            O.evict(st, keep_override=keeps)
            # compacted K/V rows equal the oracle's rows at the same positions
            for l in kv_check_layers:
                for g in range(w.kv_heads):
                    rr = 0 if R == 1 else g
                    ls = live_slots(pos_h[b * R + rr], int(len_h[b]))
                    gk = hp.rows(hp.k, b, l % w.layers, g, int(len_h[b]))[ls]
                    gv = hp.rows(hp.v, b, l % w.layers, g, int(len_h[b]))[ls]
                    order = np.argsort(np.argsort(pos_h[b * R + rr, ls]))  # gpu live slot -> rank by position
                    ok_rows = st.K[l][g][order]
                    ov_rows = st.V[l][g][order]
                    rep.kv_err = max(rep.kv_err, float(np.max(np.abs(gk - ok_rows))), float(np.max(np.abs(gv - ov_rows))))
        reports.append(rep)
    assert ikv.ikv_device_status() == 0
    return reports


class KVRowsByPosition:
    """kv_rows(l, g, positions) for the streaming oracle of sequence b: the workload
    generator's K/V rows at those original positions (exactly the values the device
    generator wrote into the cache).  Each layer's last answer is memoised, so a step that
    keeps most positions regenerates only the new ones."""

    def __init__(self, w: gen.Workload, b: int, u: np.ndarray):
        self.w, self.b, self.u = w, b, u
        self.memo = {}

    def __call__(self, l: int, g: int, positions):
        P = np.asarray(positions, dtype=np.int64)
        ent = self.memo.get(l)
        if ent is None or ent[0].shape != P.shape or not np.array_equal(ent[0], P):
            ent = self._fetch(l, P, ent)
            self.memo[l] = ent
        return ent[1][g], ent[2][g]

    def _fetch(self, l, P, old):
        w = self.w
        K = np.empty((w.kv_heads, P.shape[0], w.head_dim), np.float32)
        V = np.empty_like(K)
        miss = np.ones(P.shape[0], bool)
        if old is not None and old[0].size:
            order = np.argsort(old[0], kind="stable")
            sp = old[0][order]
            i = np.minimum(np.searchsorted(sp, P), sp.shape[0] - 1)
            found = sp[i] == P
            src = order[i[found]]
            K[:, found] = old[1][:, src]
            V[:, found] = old[2][:, src]
            miss = ~found
        if miss.any():
            k, v = w.kv_rows(self.b, l, P[miss], self.u)
            K[:, miss] = k
            V[:, miss] = v
        return P.copy(), K, V


def rel_err(g: np.ndarray, o: np.ndarray) -> float:
    """Largest relative error of g against the oracle's o (entries where o is 0 compare absolutely)."""
    if g.size == 0:
        return 0.0
    den = np.where(o != 0, np.abs(o), 1.0)
    return float(np.max(np.abs(g - o) / den))


class SampledOracle:
    """The streaming oracle (oracle.decode_step_streaming) following a few sequences of a
    full-size GPU run in lock-step (GRAN_SEQ).  Each sampled sequence keeps only its
    positions and utilities; its K/V rows are regenerated by position.  Sequences are
    independent, so sampling them checks the whole batch.  check(t, out) runs after the
    GPU finished step t and compares, per sampled sequence:
      - every layer's and head's attention output;
      - the kept set under the 1e-4 boundary rule and under the relative one (1e-4 theta);
        whether it equals the oracle's own top-B (strict); the oracle then adopts it;
      - the kept utilities, absolute and relative error;
      - the K/V rows of check_layers at the live slots, bit for bit."""

    def __init__(self, w: gen.Workload, c: DecodeCache, seqs, u: np.ndarray, compact_mode: int,
                 check_layers=(0, -1), refresh_init: int = ikv.IKV_INIT_ZERO):
        self.w, self.c, self.seqs, self.u = w, c, list(seqs), u
        self.compact_mode, self.check_layers = compact_mode, check_layers
        self.op = O.Params(alpha=w.alpha, refresh_period=w.refresh_period, score_free=w.score_free,
                           refresh_init="zero" if refresh_init == ikv.IKV_INIT_ZERO else "mean")
        B = w.budgets()
        self.states = {b: O.stream_prefill_state(w.prefill[b], B[b], w.layers, w.kv_heads) for b in self.seqs}
        self.rows = {b: KVRowsByPosition(w, b, u) for b in self.seqs}
        self.reports: List[StepReport] = []

    def check(self, t: int, out: torch.Tensor) -> StepReport:
        w, c = self.w, self.c
        torch.cuda.synchronize()
        rep = StepReport(t=t, refresh=O.is_refresh(t, w.refresh_period, w.score_free))
        q64 = as_f64(w.queries(t, t + 1, self.u)[0], w)
        len_h = c.len.cpu().numpy()
        for b in self.seqs:
            n_b = int(len_h[b])
            pos_b = c.pos[b, :n_b].cpu().numpy().astype(np.int64)
            ema_b = c.ema[b, :n_b].cpu().numpy()
            ls = live_slots(pos_b, n_b)
            gpos, gm = pos_b[ls], ema_b[ls]
            if self.compact_mode in STABLE_MODES:  # survivors keep their order (R5)
                assert np.all(np.diff(gpos) > 0), (t, b)
            assert len(set(gpos.tolist())) == len(gpos), (t, b)
            B = self.states[b].budget

            def adopt(r, m_row, pos_row, rep=rep, gpos=gpos, gm=gm, B=B, b=b):
                slot_of = {int(pp): i for i, pp in enumerate(pos_row)}
                assert len(gpos) == min(len(pos_row), B), (t, b, len(gpos), len(pos_row))
                oslots = np.array([slot_of[int(pp)] for pp in gpos], dtype=np.int64)
                kept = np.zeros(len(pos_row), bool)
                kept[oslots] = True
                ok, _ = boundary_ok(m_row, kept, B)
                rok, _ = boundary_ok(m_row, kept, B, relative=True)
                rep.set_ok &= ok
                rep.rel_set_ok &= rok
                rep.strict_set_equal &= set(O.select_keep(m_row, B).tolist()) == set(oslots.tolist())
                rep.m_err = max(rep.m_err, float(np.max(np.abs(gm - m_row[oslots]))) if len(gm) else 0.0)
                rep.m_rel_err = max(rep.m_rel_err, rel_err(gm, m_row[oslots]))
                return np.sort(oslots)

            o_out = O.decode_step_streaming(self.states[b], t, q64[:, b], self.rows[b], self.op, keep_override=adopt)
            out_b = out[:, b].float().cpu().numpy()
            rep.out_err = max(rep.out_err, float(np.max(np.abs(out_b - o_out))))
            for l in self.check_layers:
                lk, lv = w.kv_rows(b, l % w.layers, gpos, self.u)
                for g in range(w.kv_heads):
                    gk = c.gather(c.k, b, l % w.layers, g, n_b).float().cpu().numpy()[ls]
                    gv = c.gather(c.v, b, l % w.layers, g, n_b).float().cpu().numpy()[ls]
                    rep.kv_err = max(rep.kv_err, float(np.max(np.abs(gk - lk[g]))), float(np.max(np.abs(gv - lv[g]))))
        self.reports.append(rep)
        return rep


def fullsize_cache(w: gen.Workload, page_perm_seed: Optional[int] = 7, pos_cap: int = 0):
    """The workload's device cache with its prefill written by the device generator."""
    u = w.u_table()
    c = DecodeCache(w.batch, w.layers, w.q_heads, w.kv_heads, w.head_dim, w.cap,
                    dtype=ikv.IKV_BF16 if w.dtype == gen.BF16 else ikv.IKV_F32, page_size=w.page_size,
                    page_perm_seed=page_perm_seed, pos_cap=pos_cap)
    c.set_prefill(w.prefill, w.budgets())
    fill_device(c, w, torch.from_numpy(u).cuda())
    return c, u


def device_new_tokens(w: gen.Workload, u: np.ndarray, t: int):
    """k_new, v_new of decode step t ([layers][batch][kv_heads][d]) from the device generator."""
    sp = w.spec()
    u_dev = torch.from_numpy(u).cuda()
    L0_dev = torch.tensor(w.prefill, dtype=torch.int32, device="cuda")
    kn = torch.empty((1, w.layers, w.batch, w.kv_heads, w.head_dim), dtype=torch_dtype(w), device="cuda")
    vn = torch.empty_like(kn)
    assert gen.cuda_lib().ikvgen_fill_tokens_cuda(ctypes.byref(sp), u_dev.data_ptr(), L0_dev.data_ptr(), t, t + 1,
                                                  w.dtype, kn.data_ptr(), vn.data_ptr(),
                                                  torch.cuda.current_stream().cuda_stream) == 0
    return kn[0], vn[0]


def run_fullsize_sampled(w: gen.Workload, seqs, steps: int, check_layers=(0, -1), page_perm_seed: Optional[int] = 7,
                         compact_mode: int = ikv.IKV_COMPACT_STABLE, max_holes: int = 0, per_layer: bool = False):
    """Full-size lock-step for a few sequences of a workload (GRAN_SEQ), eager calls.

    The GPU decodes the whole batch at its real size (device-generated prefill, the same
    launch configuration as the benchmark); SampledOracle follows the sampled sequences."""
    c, u = fullsize_cache(w, page_perm_seed)
    chk = SampledOracle(w, c, seqs, u, compact_mode, check_layers)
    p = c.params(w.alpha, w.refresh_period, w.score_free, compact_mode, max_holes=max_holes)
    ws = c.step_workspace()
    qs = w.queries(1, steps + 1, u)
    budgets = w.budgets()
    lens, live = list(w.prefill), list(w.prefill)
    out = torch.empty((w.layers, w.batch, w.q_heads, w.head_dim), dtype=torch_dtype(w), device="cuda")
    for t in range(1, steps + 1):
        kn, vn = device_new_tokens(w, u, t)
        decode_step(c, p, c.cache(max(lens)), t, to_device(qs[t - 1], w), kn, vn, out, ws, per_layer)
        lens, live = step_lengths(lens, live, budgets, max_holes)
        torch.cuda.synchronize()
        assert list(c.len.cpu().numpy()) == lens, t
        chk.check(t, out)
    assert ikv.ikv_device_status() == 0
    return chk.reports


def run_lockstep_layerwise(w: gen.Workload, steps: Optional[int] = None, page_perm_seed: Optional[int] = 7,
                           refresh_init: int = ikv.IKV_INIT_ZERO, layer_eligible=None, per_layer: bool = False,
                           compact_mode: int = ikv.IKV_COMPACT_STABLE):
    """Per-layer immediate eviction (IKV_EVICT_LAYER) in lock-step with the oracle's
    decode_step_layerwise.  Per step: every layer's attention output, every layer's kept
    positions under the boundary rule against the oracle's utilities at that layer's
    eviction (the oracle then adopts the GPU's set), the state at every live position
    (1e-3), and each layer's K/V rows bit for bit."""
    T = w.steps if steps is None else steps
    u = w.u_table()
    pos_cap = max(w.prefill) + T + 1
    c = DecodeCache(w.batch, w.layers, w.q_heads, w.kv_heads, w.head_dim, w.cap,
                    dtype=ikv.IKV_BF16 if w.dtype == gen.BF16 else ikv.IKV_F32, page_size=w.page_size,
                    page_perm_seed=page_perm_seed, pos_cap=pos_cap)
    c.set_prefill(w.prefill, w.budgets())
    kv = fill_prefill(c, w, u)
    budgets = w.budgets()
    sts = []
    for b in range(w.batch):
        K = [[kv[b][l][0][g] for g in range(w.kv_heads)] for l in range(w.layers)]
        V = [[kv[b][l][1][g] for g in range(w.kv_heads)] for l in range(w.layers)]
        sts.append(O.layerwise_prefill_state(K, V, budgets[b]))
    op = O.Params(alpha=w.alpha, refresh_period=w.refresh_period, score_free=w.score_free,
                  layer_mask=None if layer_eligible is None else [bool(x) for x in layer_eligible],
                  refresh_init="zero" if refresh_init == ikv.IKV_INIT_ZERO else "mean")
    p = c.params(w.alpha, w.refresh_period, w.score_free, compact_mode, refresh_init, layer_eligible,
                 evict_mode=ikv.IKV_EVICT_LAYER)
    ws = c.step_workspace()
    qs = w.queries(1, T + 1, u)
    out = torch.empty((w.layers, w.batch, w.q_heads, w.head_dim), dtype=torch_dtype(w), device="cuda")
    reports = []
    lens = list(w.prefill)
    for t in range(1, T + 1):
        kn, vn = w.new_tokens(t, u)
        decode_step(c, p, c.cache(max(lens)), t, to_device(qs[t - 1], w), to_device(kn, w), to_device(vn, w), out,
                    ws, per_layer)
        lens = [min(L + 1, B) for L, B in zip(lens, budgets)]
        torch.cuda.synchronize()
        out_h = out.float().cpu().numpy()
        m_h = c.pos_state.cpu().numpy()
        pos_h = c.pos.cpu().numpy()
        len_h = c.len.cpu().numpy()
        rep = StepReport(t=t, refresh=O.is_refresh(t, w.refresh_period, w.score_free))
        q64 = as_f64(qs[t - 1], w)
        for b, st in enumerate(sts):
            assert len_h[b] == lens[b], (t, b, len_h[b], lens[b])
            gpu_slots = [pos_h[b * w.layers + l, :lens[b]].astype(np.int64) for l in range(w.layers)]
            if compact_mode in STABLE_MODES:                    # survivors keep their order (R5)
                for l in range(w.layers):
                    assert np.all(np.diff(gpu_slots[l]) > 0), (t, b, l)
            gpu_kept = [np.sort(x) for x in gpu_slots]

            def adopt(l, tr, b=b):
                kept = gpu_kept[l]
                assert len(np.unique(kept)) == len(kept), (t, b, l)
                mask = np.isin(tr.pos, kept)
                assert mask.sum() == len(kept), (t, b, l)      # kept positions were held by the layer
                ok, _ = boundary_ok(tr.m, mask, budgets[b])
                rep.set_ok &= ok
                rep.strict_set_equal &= set(tr.kept.tolist()) == set(kept.tolist())
                return kept

            o_out, _ = O.decode_step_layerwise(st, t, q64[:, b], kn[:, b], vn[:, b], op, keep_override=adopt)
            rep.out_err = max(rep.out_err, float(np.max(np.abs(out_h[:, b] - o_out))))
            live = st.live()
            rep.m_err = max(rep.m_err, float(np.max(np.abs(m_h[b, live] - st.m[live]))))
            for l in range(w.layers):
                assert np.array_equal(gpu_kept[l], st.pos[l]), (t, b, l)
                order = np.argsort(gpu_slots[l])  # GPU slot order -> ascending positions
                for g in range(w.kv_heads):
                    gk = c.gather(c.k, b, l, g, lens[b]).float().cpu().numpy()[order]
                    gv = c.gather(c.v, b, l, g, lens[b]).float().cpu().numpy()[order]
                    rep.kv_err = max(rep.kv_err, float(np.max(np.abs(gk - st.K[l][g]))),
                                     float(np.max(np.abs(gv - st.V[l][g]))))
        reports.append(rep)
    assert ikv.ikv_device_status() == 0
    return reports


def run_fullsize_sampled_layerwise(w: gen.Workload, seqs, steps: int, check_layers=(0, -1),
                                   page_perm_seed: Optional[int] = 7, per_layer: bool = False):
    """Full-size lock-step of per-layer immediate eviction for a few sequences (GRAN_SEQ),
    against oracle.decode_step_layerwise_streaming (reading R10 with every layer's K/V rows
    regenerated by position)."""
    T = steps
    c, u = fullsize_cache(w, page_perm_seed, pos_cap=max(w.prefill) + T + 1)
    op = O.Params(alpha=w.alpha, refresh_period=w.refresh_period, score_free=w.score_free)
    p = c.params(w.alpha, w.refresh_period, w.score_free, ikv.IKV_COMPACT_STABLE, evict_mode=ikv.IKV_EVICT_LAYER)
    ws = c.step_workspace()
    qs = w.queries(1, T + 1, u)
    budgets = w.budgets()
    lens = list(w.prefill)
    out = torch.empty((w.layers, w.batch, w.q_heads, w.head_dim), dtype=torch_dtype(w), device="cuda")
    states = {b: O.layerwise_stream_prefill_state(w.prefill[b], budgets[b], w.layers, w.kv_heads) for b in seqs}
    rows = {b: {l: KVRowsByPosition(w, b, u) for l in range(w.layers)} for b in seqs}
    reports = []
    for t in range(1, T + 1):
        kn, vn = device_new_tokens(w, u, t)
        decode_step(c, p, c.cache(max(lens)), t, to_device(qs[t - 1], w), kn, vn, out, ws, per_layer)
        lens = [min(L + 1, B) for L, B in zip(lens, budgets)]
        torch.cuda.synchronize()
        rep = StepReport(t=t, refresh=O.is_refresh(t, w.refresh_period, w.score_free))
        q64 = as_f64(qs[t - 1], w)
        len_h = c.len.cpu().numpy()
        pos_h = c.pos.cpu().numpy()
        m_h = c.pos_state.cpu().numpy()
        for b in seqs:
            assert len_h[b] == lens[b]
            gpu_kept = [np.sort(pos_h[b * w.layers + l, :lens[b]].astype(np.int64)) for l in range(w.layers)]
            for l in range(w.layers):
                assert np.all(np.diff(pos_h[b * w.layers + l, :lens[b]]) > 0), (t, b, l)

            def adopt(l, tr, b=b, rep=rep):
                kept = gpu_kept[l]
                mask = np.isin(tr.pos, kept)
                assert mask.sum() == len(kept), (t, b, l)      # kept positions were held by the layer
                ok, _ = boundary_ok(tr.m, mask, budgets[b])
                rok, _ = boundary_ok(tr.m, mask, budgets[b], relative=True)
                rep.set_ok &= ok
                rep.rel_set_ok &= rok
                rep.strict_set_equal &= set(tr.kept.tolist()) == set(kept.tolist())
                return kept

            st = states[b]
            # every layer's rows by position (the layers hold different sets: one memo per layer)
            o_out, _ = O.decode_step_layerwise_streaming(st, t, q64[:, b],
                                                         lambda l, g, ps, b=b: rows[b][l](l, g, ps), op,
                                                         keep_override=adopt)
            out_b = out[:, b].float().cpu().numpy()
            rep.out_err = max(rep.out_err, float(np.max(np.abs(out_b - o_out))))
            live = st.live()
            rep.m_err = max(rep.m_err, float(np.max(np.abs(m_h[b, live] - st.m[live]))))
            rep.m_rel_err = max(rep.m_rel_err, rel_err(m_h[b, live], st.m[live]))
            for l in check_layers:
                ll = l % w.layers
                assert np.array_equal(gpu_kept[ll], st.pos[ll])
                lk, lv = w.kv_rows(b, ll, st.pos[ll], u)
                for g in range(w.kv_heads):
                    gk = c.gather(c.k, b, ll, g, lens[b]).float().cpu().numpy()
                    gv = c.gather(c.v, b, ll, g, lens[b]).float().cpu().numpy()
                    rep.kv_err = max(rep.kv_err, float(np.max(np.abs(gk - lk[g]))), float(np.max(np.abs(gv - lv[g]))))
        reports.append(rep)
    assert ikv.ikv_device_status() == 0
    return reports
