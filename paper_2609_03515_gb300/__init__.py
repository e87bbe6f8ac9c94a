"""InertiaKV decode-step eviction path on GB300 (sm_103a): Python side.

``ikv`` binds the C ABI of ``libikv.so`` (include/ikv.h).  ``DecodeCache``
allocates the device tensors a caller hands to that ABI -- paged K/V pools,
block table, lengths, positions, utilities, budgets and workspace -- using
PyTorch purely as the device allocator.  All arithmetic of the path runs in
the CUDA library.
"""
from __future__ import annotations

from typing import Optional, Sequence

import torch

from . import ikv

__all__ = ["ikv", "DecodeCache", "RankTrace", "step_lengths", "auto_max_holes"]


def auto_max_holes(budgets: Sequence[int]) -> int:
    """A deferred-compaction threshold (ikv_params.max_holes) for sequences with these
    budgets.  Holding on average max_holes / 2 dead slots makes the attention read that
    many masked rows per step, and one compaction of about B rows (read + write) is
    spread over max_holes steps; max_holes / 2 + 2 B / max_holes is smallest at
    max_holes = 2 sqrt(B).  Rounded to a multiple of 8, at least 8."""
    import math

    b = sum(budgets) / max(1, len(budgets))
    return max(8, int(round(2 * math.sqrt(b) / 8)) * 8)


def step_lengths(lens: Sequence[int], live: Sequence[int], budgets: Sequence[int], max_holes: int = 0):
    """Host mirror of one ikv_step's length bookkeeping, for sizing max_len.

    lens: slots in use per sequence (len[b], dead slots included); live: live slots.
    The step appends one token; if more than budget[b] slots are then live, it keeps
    budget[b] of them.  The evicted slots are only marked dead while the dead slots
    stay <= max_holes (> 0); otherwise the sequence is compacted to its live slots.
    Returns the (lens, live) after the step."""
    out_l, out_v = [], []
    for L, n, B in zip(lens, live, budgets):
        L, n = L + 1, n + 1
        kept = min(n, B)
        if max_holes > 0 and L - kept <= max_holes:
            out_l.append(L)
        else:
            out_l.append(kept)
        out_v.append(kept)
    return out_l, out_v


class DecodeCache:
    """Device buffers of one batch of decode sequences.

    k, v:        [layers][num_pages][kv_heads][page_size][head_dim] (bf16 or fp32)
    block_table: [batch][max_pages] int32 physical page of each logical page
    len:         [batch] int32 slots in use (dead slots included);  next_pos: [batch] int32
    pos, ema:    [rows][cap] int32 / fp32, rows = batch (per-sequence state) or batch * kv_heads;
                 pos = -1 marks a dead slot (deferred compaction).  With pos_cap > 0 (per-layer
                 eviction): pos has batch * layers rows (row b * layers + l: layer l's positions)
                 and pos_state [batch][pos_cap] is the utility by token position
    budget:      [batch] int32
    """

    def __init__(self, batch: int, layers: int, q_heads: int, kv_heads: int, head_dim: int, cap_tokens: int,
                 dtype: int = ikv.IKV_BF16, page_size: int = 64, granularity: int = ikv.IKV_GRAN_SEQ,
                 device: str = "cuda", page_perm_seed: Optional[int] = None, value_norms: bool = False,
                 pos_cap: int = 0):
        self.batch, self.layers, self.q_heads, self.kv_heads, self.head_dim = batch, layers, q_heads, kv_heads, head_dim
        self.dtype, self.granularity, self.page_size = dtype, granularity, page_size
        self.max_pages = (cap_tokens + page_size - 1) // page_size
        self.cap = self.max_pages * page_size
        self.num_pages = batch * self.max_pages
        tdt = torch.bfloat16 if dtype == ikv.IKV_BF16 else torch.float32
        self.torch_dtype = tdt
        shp = (layers, self.num_pages, kv_heads, page_size, head_dim)
        self.k = torch.zeros(shp, dtype=tdt, device=device)
        self.v = torch.zeros(shp, dtype=tdt, device=device)
        pages = torch.arange(self.num_pages, dtype=torch.int32)
        if page_perm_seed is not None:
            g = torch.Generator().manual_seed(page_perm_seed)
            pages = pages[torch.randperm(self.num_pages, generator=g)]
        self.block_table = pages.view(batch, self.max_pages).to(device)
        self.rows = batch if granularity == ikv.IKV_GRAN_SEQ else batch * kv_heads
        self.len = torch.zeros(batch, dtype=torch.int32, device=device)
        self.next_pos = torch.zeros(batch, dtype=torch.int32, device=device)
        # per-layer eviction (pos_cap > 0): a position row per (sequence, layer) and the
        # utility state indexed by token position (pos_state); the step-end mode reads
        # the first `rows` position rows and ema
        self.pos_cap = pos_cap
        pos_rows = max(self.rows, batch * layers) if pos_cap > 0 else self.rows
        self.pos = torch.zeros((pos_rows, self.cap), dtype=torch.int32, device=device)
        self.ema = torch.zeros((self.rows, self.cap), dtype=torch.float32, device=device)
        self.pos_state = (torch.zeros((batch, pos_cap), dtype=torch.float32, device=device) if pos_cap > 0
                          else None)
        self.budget = torch.zeros(batch, dtype=torch.int32, device=device)
        self.start = torch.zeros(batch, dtype=torch.int32, device=device)
        # per-slot value-row norms, for the VNorm scorer
        self.vnorm = (torch.zeros((layers, batch, kv_heads, self.cap), dtype=torch.float32, device=device)
                      if value_norms else None)
        self.max_len = 0

    # ---- ABI structs ------------------------------------------------------
    def shape(self) -> ikv.ikv_shape:
        return ikv.ikv_shape(self.batch, self.layers, self.q_heads, self.kv_heads, self.head_dim, self.dtype,
                             self.granularity)

    def cache(self, max_len: Optional[int] = None, dead_slots: bool = False) -> ikv.ikv_cache:
        ml = self.max_len if max_len is None else max_len
        return ikv.ikv_cache(self.k.data_ptr(), self.v.data_ptr(), self.block_table.data_ptr(), self.num_pages,
                             self.page_size, self.max_pages, self.len.data_ptr(), self.pos.data_ptr(),
                             self.next_pos.data_ptr(), ml, self.start.data_ptr(), 1 if dead_slots else 0,
                             self.vnorm.data_ptr() if self.vnorm is not None else None, self.pos_cap)

    @property
    def rows_per_seq(self) -> int:
        return 1 if self.granularity == ikv.IKV_GRAN_SEQ else self.kv_heads

    # ---- host-side helpers (setup / inspection) ----------------------------
    def set_prefill(self, lengths: Sequence[int], budgets: Sequence[int]) -> None:
        """Mark slots [0, L0_b) as holding positions 0..L0_b-1 with utility 0 (m_0 = 0)."""
        dev = self.len.device
        self.len.copy_(torch.tensor(list(lengths), dtype=torch.int32, device=dev))
        self.next_pos.copy_(self.len)
        self.budget.copy_(torch.tensor(list(budgets), dtype=torch.int32, device=dev))
        ar = torch.arange(self.cap, dtype=torch.int32, device=dev)
        self.pos.copy_(ar.expand(self.pos.shape[0], self.cap))
        self.ema.zero_()
        if self.pos_state is not None:
            self.pos_state.zero_()
        self.start.zero_()
        self.max_len = max(lengths)

    def slot_rows(self, b: int, layer: int, g: int, n: int):
        """(pages, offsets) of cache slots 0..n-1 of sequence b (through start and the block table)."""
        slots = torch.arange(n, device=self.k.device) + int(self.start[b].item())
        pages = self.block_table[b, (slots // self.page_size).long()].long()
        return pages, slots % self.page_size

    def gather(self, pool: torch.Tensor, b: int, layer: int, g: int, n: int) -> torch.Tensor:
        pages, off = self.slot_rows(b, layer, g, n)
        return pool[layer, pages, g, off]

    def scatter(self, pool: torch.Tensor, b: int, layer: int, g: int, rows: torch.Tensor, start: int = 0) -> None:
        n = rows.shape[0]
        s0 = start + int(self.start[b].item())
        slots = torch.arange(s0, s0 + n, device=pool.device)
        pages = self.block_table[b, (slots // self.page_size).long()].long()
        pool[layer, pages, g, slots % self.page_size] = rows.to(pool.dtype)

    def utility(self, evict_mode: int = ikv.IKV_EVICT_STEP) -> torch.Tensor:
        """The utility array a step of this eviction mode updates (ema or pos_state)."""
        return self.pos_state if evict_mode == ikv.IKV_EVICT_LAYER else self.ema

    def step_workspace(self) -> torch.Tensor:
        """Zero-filled, so steps may run with ikv_params.ws_zeroed from the first one."""
        n = ikv.ikv_step_workspace_size(self.shape(), self.cache(self.cap - 1))
        return torch.zeros(n, dtype=torch.uint8, device=self.k.device)

    def params(self, alpha: float, refresh_period: int = 1, score_free: bool = False,
               compact_mode: int = ikv.IKV_COMPACT_STABLE, refresh_init: int = ikv.IKV_INIT_ZERO,
               layer_eligible: Optional[Sequence[int]] = None, max_holes: int = 0,
               agg_mode: int = ikv.IKV_AGG_EMA, scorer: int = ikv.IKV_SCORE_ATTENTION,
               evict_mode: int = ikv.IKV_EVICT_STEP, trace: "Optional[RankTrace]" = None,
               ws_zeroed: bool = False) -> ikv.ikv_params:
        p = ikv.ikv_params()
        p.alpha = alpha
        p.refresh_period = refresh_period
        p.score_free = 1 if score_free else 0
        p.budget = self.budget.data_ptr()
        if layer_eligible is not None:
            self._elig = (ctypes_u8 * self.layers)(*[1 if x else 0 for x in layer_eligible])
            p.layer_eligible = ctypes_addr(self._elig)
        p.compact_mode = compact_mode
        p.refresh_init = refresh_init
        p.max_holes = max_holes
        p.agg_mode = agg_mode
        p.scorer = scorer
        p.evict_mode = evict_mode
        p.ws_zeroed = 1 if ws_zeroed else 0
        if trace is not None:
            p.trace = _ct.pointer(trace.struct)
            self._trace = trace
        return p


import ctypes as _ct  # noqa: E402

ctypes_u8 = _ct.c_uint8


def ctypes_addr(x) -> int:
    return _ct.addressof(x)


class RankTrace:
    """Device buffers of the rank-trace diagnostics (ikv_trace) for one DecodeCache: each
    utility row's previous raw / EMA top-k positions, their sizes and the last step's
    overlap counts {|R & R_prev|, |E & E_prev|, |R & E|, |R|, |E|}."""

    def __init__(self, c: DecodeCache):
        dev = c.k.device
        self.raw_top = torch.zeros((c.rows, c.cap), dtype=torch.int32, device=dev)
        self.ema_top = torch.zeros((c.rows, c.cap), dtype=torch.int32, device=dev)
        self.n_top = torch.zeros((c.rows, 2), dtype=torch.int32, device=dev)
        self.counts = torch.zeros((c.rows, 5), dtype=torch.int32, device=dev)
        self.struct = ikv.ikv_trace(self.raw_top.data_ptr(), self.ema_top.data_ptr(), self.n_top.data_ptr(),
                                    self.counts.data_ptr())

    def reset(self) -> None:
        self.n_top.zero_()
