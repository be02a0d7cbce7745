"""GB300-native CacheBack receiver-conditioned KV filtering.

    score   (App. C.1, App. D.2)  every cached sender position by the attention it
            receives from the receiver's query tokens: S_t = Q_t * C_{p,t}^alpha
    select  (App. C.2)            B = ceil(keep * T) positions by the span rule
    compact                       the selected K/V rows of every layer into one
                                  contiguous send buffer (fan-in senders concatenated)

The compute runs in hand-written sm_103a CUDA kernels behind the C-ABI of
include/cacheback.h (libcacheback.so); this package is the Python binding.
"""
from __future__ import annotations

from typing import List, Optional, Sequence

from .binding import (CB_EBUDGET, CB_ECUDA, CB_EDEVICE, CB_EINVAL, CB_ENOMEM, CB_ESHAPE, CB_ETIMEOUT, CB_OK, EXPORTED,
                      LIB_PATH, CacheBack, CBError, PagedKV, budget, chain_budget, load_library)

__all__ = ["CacheBack", "CBError", "PagedKV", "budget", "chain_budget", "load_library", "LIB_PATH", "EXPORTED",
           "Filter", "Chain",
           "CB_OK", "CB_EINVAL", "CB_ESHAPE", "CB_EBUDGET", "CB_ENOMEM", "CB_ECUDA", "CB_ETIMEOUT", "CB_EDEVICE"]


class Filter:
    """Score -> select -> compact for a fixed batch of senders, outputs allocated once.

    senders: list of (K, V) bf16 [nL][Hkv][T_i][d] device tensors, or PagedKV caches (block-table
             layout); one (K, V) may appear several
             times, each with its own query (multi-query serving: one launch scores the state
             for every receiver query, and each query gets its own message)
    queries: list of Q bf16 [nL][m_i][Hq][d] device tensors, one per sender (may repeat)
    keep:    keep ratio; budgets B_i = max(ceil(keep * T_i), min(T_i, n_sink + n_latent))
    The send buffer holds every sender's rows back to back: sender i at offset sum_{j<i} B_j.
    """

    def __init__(self, cb: CacheBack, senders: Sequence, queries: Sequence, keep: float, device=None,
                 query_keys: Optional[Sequence] = None):
        import torch
        self.cb = cb
        # a PagedKV stands for both K and V of its sender
        senders = [(s, s) if isinstance(s, PagedKV) else s for s in senders]
        self.Ks = [k for k, _ in senders]
        self.Vs = [v for _, v in senders]
        self.Qs = list(queries)
        # optional: the query tokens' own keys [nL][m][Hkv][d] per sender (None: sender positions only)
        self.Kqs = list(query_keys) if query_keys is not None else [None] * len(self.Ks)
        dev = device or self.Ks[0].device
        self.Ts = [int(K.shape[2]) for K in self.Ks]
        # B_i = ceil(keep * T_i), raised to the forced count when that is larger (App. C.2: the
        # forced first and latent positions count toward B and every budget holds them)
        forced = cb.cfg.n_sink + cb.cfg.n_latent
        self.budgets = [max(budget(T, keep), min(T, forced)) for T in self.Ts]
        self.offsets = []
        off = 0
        for b in self.budgets:
            self.offsets.append(off)
            off += b
        self.capacity = off
        nL, Hkv, _, d = self.Ks[0].shape
        self.scores = [torch.empty(T, dtype=torch.float32, device=dev) for T in self.Ts]
        self.idx = [torch.empty(max(b, 1), dtype=torch.int32, device=dev) for b in self.budgets]
        self.k_out = torch.empty(nL, Hkv, max(self.capacity, 1), d, dtype=self.Ks[0].dtype, device=dev)
        self.v_out = torch.empty_like(self.k_out)

    def score(self, stream=None):
        self.cb.score(self.Ks, self.Qs, self.scores, stream, self.Kqs)

    def select(self, stream=None):
        self.cb.select(self.scores, self.Ts, self.budgets, self.idx, stream)

    def compact(self, stream=None, rope: Optional[dict] = None):
        """rope = dict(base=..., style=0 or 1, pos0=...): also move K to receiver positions
        pos0 + (row of the send buffer) with the receiver's rotary embedding."""
        if rope is None:
            self.cb.compact(self.Ks, self.Vs, self.idx, self.budgets, self.k_out, self.v_out, self.offsets, stream)
        else:
            self.cb.compact_rope(self.Ks, self.Vs, self.idx, self.budgets, self.k_out, self.v_out, self.offsets,
                                 rope["base"], rope.get("style", 0), rope.get("pos0", 0), stream)

    def run(self, stream=None, wave: Optional[int] = None):
        """The whole path.  wave = None: score, select and compact every sender in turn on
        `stream`.  wave = w: senders go in waves of w; a wave's selection and compaction run on a
        second stream while the next wave is scored (compaction is bound by HBM bandwidth, the
        scoring by the tensor pipe and exp2 throughput), and `stream` waits for both at the end.
        Results are identical either way."""
        n = len(self.Ks)
        if not wave or wave >= n:
            self.score(stream)
            self.select(stream)
            self.compact(stream)
            return self
        import torch
        main = stream if stream is not None else torch.cuda.current_stream(self.Ks[0].device)
        side = self._side_stream(main.device)
        side.wait_stream(main)                       # inputs written on the caller's stream
        for a in range(0, n, wave):
            b = min(n, a + wave)
            sl = slice(a, b)
            self.cb.score(self.Ks[sl], self.Qs[sl], self.scores[sl], main, self.Kqs[sl])
            done = torch.cuda.Event()
            done.record(main)
            side.wait_event(done)
            self.cb.select(self.scores[sl], self.Ts[sl], self.budgets[sl], self.idx[sl], side)
            self.cb.compact(self.Ks[sl], self.Vs[sl], self.idx[sl], self.budgets[sl], self.k_out, self.v_out,
                            self.offsets[sl], side)
        main.wait_stream(side)
        return self

    def _side_stream(self, device):
        import torch
        if getattr(self, "_side", None) is None:
            self._side = torch.cuda.Stream(device=device)
        return self._side

    def indices(self) -> List:
        return [x[:b] for x, b in zip(self.idx, self.budgets)]

    # -- message encodings (Sec. 3.1 "State Representation", App. C.3) ------------------
    def message_rows(self, tables: Sequence, stream=None):
        """Continuous-row encoding: every selected position as one row of the sender's
        per-position table (e.g. hidden states [T_i][hidden]); senders back to back."""
        import torch
        out = torch.empty((max(self.capacity, 1),) + tuple(tables[0].shape[1:]), dtype=tables[0].dtype,
                          device=tables[0].device)
        self.cb.gather(tables, self.idx, self.budgets, out, self.offsets, stream)
        return out[:self.capacity]

    def message_token_ids(self, token_ids: Sequence, tables: Sequence, stream=None):
        """Token-ID encoding: the selected source positions as token IDs (int32 [T_i] tables), the
        latent positions (the last n_latent, always selected) as continuous rows.  Returns
        (ids [sum_i (B_i - L_i)], rows [sum_i L_i][...]) with L_i = min(T_i, n_latent)."""
        import torch
        lat = [min(T, self.cb.cfg.n_latent) for T in self.Ts]
        n_src = [b - l for b, l in zip(self.budgets, lat)]
        id_off, row_off = [], []
        a = r = 0
        for ns, nl in zip(n_src, lat):
            id_off.append(a); row_off.append(r)
            a += ns; r += nl
        dev = tables[0].device
        ids = torch.empty(max(a, 1), dtype=torch.int32, device=dev)
        rows = torch.empty((max(r, 1),) + tuple(tables[0].shape[1:]), dtype=tables[0].dtype, device=dev)
        tabs = [t.view(-1, 1) for t in token_ids]
        self.cb.gather(tabs, [x[:max(ns, 1)] for x, ns in zip(self.idx, n_src)], n_src, ids.view(-1, 1), id_off,
                       stream)
        self.cb.gather(tables, [x[ns:] for x, ns in zip(self.idx, n_src)], lat, rows, row_off, stream)
        return ids[:a], rows[:r]


def _copy_rows(dst, src):
    """dst.copy_(src) for [nL][Hkv][T][d] bf16 views whose rows are contiguous: moved as 8-byte
    words (a strided copy of 2-byte elements runs at a third of the bandwidth)."""
    import torch
    if dst.dtype == src.dtype and dst.element_size() == 2 and dst.shape[-1] % 4 == 0 and \
            dst.stride(-1) == 1 and src.stride(-1) == 1:
        try:
            dst.view(torch.int64).copy_(src.view(torch.int64))
            return
        except RuntimeError:
            pass
    dst.copy_(src)


class Chain:
    """Sequential communication (App. C.2; the LongBench hops of Sec. 4): hop i's sender cache is
    the previous hop's message (its selected K/V rows, in source order) followed by the hop's new
    prompt and latent positions.  Each hop scores that whole cache against its receiver query,
    selects B_i positions under the chain budget (inherited and new positions ranked together;
    only the first and the current n_latent positions forced, so inherited latent positions may be
    dropped) and compacts them into the front of the other of two cache buffers, which the next
    hop extends.  Nothing is copied besides the compaction.

    cb:        CacheBack sized for one sender with max_positions >= capacity
    capacity:  the largest T_old + T_new of any hop
    mode:      "relative" (B = T_old + ceil(keep T_new)) or "fixed" (B = min(B_max, T_old + T_new))
    """

    def __init__(self, cb: CacheBack, capacity: int, keep: float = 0.25, mode: str = "relative",
                 B_max: int = 0, device=None):
        import torch
        self.cb, self.capacity, self.keep, self.mode, self.B_max = cb, int(capacity), keep, mode, B_max
        c = cb.cfg
        shape = (c.n_layers, c.n_kv_heads, self.capacity, c.head_dim)
        self.K = [torch.empty(shape, dtype=torch.bfloat16, device=device) for _ in range(2)]
        self.V = [torch.empty(shape, dtype=torch.bfloat16, device=device) for _ in range(2)]
        self.cur = 0
        self.T_old = 0

    def reset(self):
        """Start a new chain over the same buffers (the next hop inherits no message)."""
        self.cur = 0
        self.T_old = 0

    def new_slot(self, T_new: int):
        """Views of the current buffer where the hop's T_new new positions go (after the message)."""
        a, b = self.T_old, self.T_old + int(T_new)
        if b > self.capacity:
            raise ValueError("hop of %d positions exceeds the chain capacity %d" % (b, self.capacity))
        return self.K[self.cur][:, :, a:b], self.V[self.cur][:, :, a:b]

    def hop(self, Q, K_new=None, V_new=None, T_new: Optional[int] = None, stream=None) -> dict:
        """One hop: K_new / V_new (or T_new positions already written through new_slot) join the
        inherited message; returns the hop's cache views, scores, budget and selected indices."""
        import torch
        if K_new is not None:
            T_new = int(K_new.shape[2])
            k, v = self.new_slot(T_new)
            _copy_rows(k, K_new)
            _copy_rows(v, V_new)
        T_old, T = self.T_old, self.T_old + int(T_new)
        c = self.cb.cfg
        B = chain_budget(T_old, T_new, self.keep, self.mode, self.B_max)
        B = max(B, min(T, c.n_sink + c.n_latent))          # the forced positions always fit
        Kv, Vv = self.K[self.cur][:, :, :T], self.V[self.cur][:, :, :T]
        scores = torch.empty(T, dtype=torch.float32, device=Kv.device)
        idx = torch.empty(max(B, 1), dtype=torch.int32, device=Kv.device)
        self.cb.score([Kv], [Q], [scores], stream)
        self.cb.select([scores], [T], [B], [idx], stream)
        nxt = 1 - self.cur
        self.cb.compact([Kv], [Vv], [idx], [B], self.K[nxt], self.V[nxt], [0], stream)
        out = {"K": Kv, "V": Vv, "T_old": T_old, "T": T, "B": B, "scores": scores, "idx": idx[:B],
               "message_K": self.K[nxt][:, :, :B], "message_V": self.V[nxt][:, :, :B]}
        self.cur, self.T_old = nxt, B
        return out

