"""Thin Python binding of include/cacheback.h (argument marshalling only).

Every step of the path runs in libcacheback.so's CUDA kernels; this module only
turns torch tensors into pointers, sizes and strides.  If the library is missing
the import of `CacheBack` fails loudly: there is no CPU fallback.
"""
from __future__ import annotations

import ctypes
import math
import os
from typing import Optional, Sequence

PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(PKG, "libcacheback.so")

CB_OK, CB_EINVAL, CB_ESHAPE, CB_EBUDGET, CB_ENOMEM, CB_ECUDA, CB_ETIMEOUT, CB_EDEVICE = range(8)
STATUS_NAMES = ["CB_OK", "CB_EINVAL", "CB_ESHAPE", "CB_EBUDGET", "CB_ENOMEM", "CB_ECUDA", "CB_ETIMEOUT",
                "CB_EDEVICE"]

# Every entry point include/cacheback.h declares (checked by the tests).
EXPORTED = ["cb_config_init", "cb_create", "cb_score", "cb_budget", "cb_select", "cb_compact",
            "cb_sync_status", "cb_destroy", "cb_last_error", "cb_scratch_bytes", "cb_score_path", "cb_select_noalloc",
            "cb_select_noalloc_status", "cb_gather", "cb_chain_budget", "cb_compact_rope",
            "cb_enable_stage_timing", "cb_stage_times", "cb_set_wait_limit", "cb_set_score_sms"]


class CBError(RuntimeError):
    def __init__(self, status: int, message: str):
        name = STATUS_NAMES[status] if 0 <= status < len(STATUS_NAMES) else str(status)
        super().__init__("%s: %s" % (name, message))
        self.status = status


class cb_config(ctypes.Structure):
    _fields_ = [("n_layers", ctypes.c_int32), ("n_q_heads", ctypes.c_int32), ("n_kv_heads", ctypes.c_int32),
                ("head_dim", ctypes.c_int32), ("max_query_tokens", ctypes.c_int32),
                ("max_positions", ctypes.c_int64), ("max_senders", ctypes.c_int32),
                ("softmax_scale", ctypes.c_float), ("p", ctypes.c_float), ("alpha", ctypes.c_float),
                ("pool_width", ctypes.c_int32), ("span_width", ctypes.c_int32),
                ("n_sink", ctypes.c_int32), ("n_latent", ctypes.c_int32), ("score_kernel", ctypes.c_int32)]


class cb_kv(ctypes.Structure):
    _fields_ = [("k", ctypes.c_void_p), ("v", ctypes.c_void_p), ("T", ctypes.c_int64),
                ("s_layer", ctypes.c_int64), ("s_head", ctypes.c_int64), ("s_pos", ctypes.c_int64),
                ("pages", ctypes.c_void_p), ("page_size", ctypes.c_int32), ("s_page", ctypes.c_int64),
                ("n_pages", ctypes.c_int64)]


class cb_query(ctypes.Structure):
    _fields_ = [("q", ctypes.c_void_p), ("m", ctypes.c_int32), ("s_layer", ctypes.c_int64),
                ("s_tok", ctypes.c_int64), ("s_head", ctypes.c_int64), ("k_self", ctypes.c_void_p),
                ("ks_layer", ctypes.c_int64), ("ks_tok", ctypes.c_int64), ("ks_head", ctypes.c_int64)]


_LIB = None


def load_library(path: Optional[str] = None) -> ctypes.CDLL:
    """Load libcacheback.so (built by paper_2609_32046_gb300.build); raises if absent."""
    global _LIB
    if _LIB is not None and path is None:
        return _LIB
    p = path or LIB_PATH
    if not os.path.exists(p):
        raise ImportError("libcacheback.so is not built (%s); run `python -m paper_2609_32046_gb300.build` "
                          "or __graft_entry__.build()" % p)
    lib = ctypes.CDLL(p)
    P = ctypes.c_void_p
    lib.cb_config_init.argtypes = [ctypes.POINTER(cb_config)]
    lib.cb_config_init.restype = None
    lib.cb_create.argtypes = [ctypes.POINTER(cb_config), ctypes.POINTER(P)]
    lib.cb_create.restype = ctypes.c_int
    lib.cb_score.argtypes = [P, ctypes.c_int32, ctypes.POINTER(cb_kv), ctypes.POINTER(cb_query), P, P]
    lib.cb_score.restype = ctypes.c_int
    lib.cb_budget.argtypes = [ctypes.c_int64, ctypes.c_double]
    lib.cb_budget.restype = ctypes.c_int64
    lib.cb_chain_budget.argtypes = [ctypes.c_int64, ctypes.c_int64, ctypes.c_double, ctypes.c_int32, ctypes.c_int64]
    lib.cb_chain_budget.restype = ctypes.c_int64
    lib.cb_select.argtypes = [P, ctypes.c_int32, P, P, P, P, P]
    lib.cb_select.restype = ctypes.c_int
    lib.cb_compact.argtypes = [P, ctypes.c_int32, ctypes.POINTER(cb_kv), P, P, P, P, ctypes.c_int64, P,
                               ctypes.c_int64, ctypes.c_int64, P]
    lib.cb_compact.restype = ctypes.c_int
    lib.cb_compact_rope.argtypes = [P, ctypes.c_int32, ctypes.POINTER(cb_kv), P, P, P, P, ctypes.c_int64, P,
                                    ctypes.c_int64, ctypes.c_int64, ctypes.c_double, ctypes.c_int32,
                                    ctypes.c_int64, P]
    lib.cb_compact_rope.restype = ctypes.c_int
    lib.cb_gather.argtypes = [P, ctypes.c_int32, P, P, ctypes.c_int64, ctypes.c_int64, P, P, P, ctypes.c_int64, P,
                              ctypes.c_int64, P]
    lib.cb_gather.restype = ctypes.c_int
    lib.cb_sync_status.argtypes = [P, P]
    lib.cb_sync_status.restype = ctypes.c_int
    lib.cb_destroy.argtypes = [P]
    lib.cb_destroy.restype = None
    lib.cb_last_error.argtypes = [P]
    lib.cb_last_error.restype = ctypes.c_char_p
    lib.cb_scratch_bytes.argtypes = [P]
    lib.cb_scratch_bytes.restype = ctypes.c_int64
    lib.cb_score_path.argtypes = [P]
    lib.cb_score_path.restype = ctypes.c_int32
    lib.cb_select_noalloc.argtypes = [ctypes.c_int32, P, P, P, P, ctypes.c_int32, ctypes.c_int32, ctypes.c_int32, P]
    lib.cb_select_noalloc.restype = ctypes.c_int
    lib.cb_set_wait_limit.argtypes = [P, ctypes.c_int64, ctypes.c_int32]
    lib.cb_set_wait_limit.restype = ctypes.c_int
    lib.cb_set_score_sms.argtypes = [P, ctypes.c_int32]
    lib.cb_set_score_sms.restype = ctypes.c_int
    lib.cb_select_noalloc_status.argtypes = [P]
    lib.cb_select_noalloc_status.restype = ctypes.c_int
    lib.cb_enable_stage_timing.argtypes = [P, ctypes.c_int32]
    lib.cb_enable_stage_timing.restype = ctypes.c_int
    lib.cb_stage_times.argtypes = [P, ctypes.POINTER(ctypes.c_float), ctypes.POINTER(ctypes.c_int32)]
    lib.cb_stage_times.restype = ctypes.c_int
    if path is None:
        _LIB = lib
    return lib


def budget(T: int, keep: float) -> int:
    """ceil(keep * T) in double, clamped to [0, T] (App. C.2), computed by the library."""
    return int(load_library().cb_budget(int(T), float(keep)))


def chain_budget(T_old: int, T_new: int, keep: float = 0.0, mode: str = "relative", B_max: int = 0) -> int:
    """Budget of one hop of a sequential chain (App. C.2): relative T_old + ceil(keep T_new) or
    fixed min(B_max, T_old + T_new), computed by the library."""
    m = {"relative": 0, "fixed": 1}[mode]
    b = int(load_library().cb_chain_budget(int(T_old), int(T_new), float(keep), m, int(B_max)))
    if b < 0:
        raise ValueError("invalid chain budget arguments")
    return b


def select_noalloc(scores: Sequence, Ts: Sequence[int], budgets: Sequence[int], idx: Sequence, n_sink: int = 1,
                   n_latent: int = 40, span_width: int = 16, stream=None):
    """cb_select_noalloc: selection without a context and without device allocation."""
    lib = load_library()
    n = len(scores)
    st = lib.cb_select_noalloc(n, _ptr_array([s.data_ptr() for s in scores]),
                               _ptr_array([int(t) for t in Ts], ctypes.c_int64),
                               _ptr_array([int(b) for b in budgets], ctypes.c_int64),
                               _ptr_array([x.data_ptr() for x in idx]), n_sink, n_latent, span_width,
                               _stream_handle(stream))
    if st != CB_OK:
        raise CBError(st, lib.cb_last_error(None).decode())


def select_noalloc_status(stream=None):
    """cb_select_noalloc_status: wait for the stream and raise if the allocation-free selection's
    kernel check failed since the last read."""
    lib = load_library()
    st = lib.cb_select_noalloc_status(_stream_handle(stream))
    if st != CB_OK:
        raise CBError(st, lib.cb_last_error(None).decode())


def _ptr_array(values, ctype=ctypes.c_void_p):
    arr = (ctype * len(values))(*values)
    return arr


def _stream_handle(stream) -> int:
    if stream is None:
        import torch
        return torch.cuda.current_stream().cuda_stream
    if isinstance(stream, int):
        return stream
    return stream.cuda_stream


class PagedKV:
    """A sender cache in the paged (block-table) layout of a vLLM-style server (App. F).

    k_pool, v_pool: bf16 tensors indexed [l][page][row][g][k] (vLLM's per-layer
                    [n_pages][page_size][Hkv][d] caches stacked over layers, or any view with
                    that index order and a unit head-dim stride; both with the same strides)
    pages:          int32 device tensor, pages[b] = the page holding positions
                    b * page_size .. b * page_size + page_size - 1 (the sequence's block table)
    T:              positions cached
    Quacks like the [nL][Hkv][T][d] tensor it stands for (shape, dtype, device), so it can be
    passed wherever a sender's K is expected; kv_desc(p) describes both pools.
    """

    def __init__(self, k_pool, v_pool, pages, T: int):
        assert k_pool.dim() == 5 and k_pool.dtype.itemsize == 2 and k_pool.stride(4) == 1
        assert v_pool.shape == k_pool.shape and v_pool.stride() == k_pool.stride()
        nL, n_pages, P, Hkv, d = k_pool.shape
        assert P & (P - 1) == 0, "page_size must be a power of two"
        assert pages.dtype.itemsize == 4 and pages.is_contiguous() and pages.numel() >= (T + P - 1) // P
        self.k_pool, self.v_pool, self.pages, self.T = k_pool, v_pool, pages, int(T)
        self.page_size, self.n_pages = P, n_pages
        self.shape = (nL, Hkv, int(T), d)
        self.dtype = k_pool.dtype
        self.device = k_pool.device

    def desc(self) -> cb_kv:
        k = self.k_pool
        return cb_kv(k.data_ptr(), self.v_pool.data_ptr(), self.T, k.stride(0), k.stride(3), k.stride(2),
                     self.pages.data_ptr(), self.page_size, k.stride(1), self.n_pages)


def kv_desc(K, V=None) -> cb_kv:
    """K, V: bf16 [nL][Hkv][T][d] (any strides with unit head-dim stride), or K a PagedKV
    (V ignored: the PagedKV holds both pools)."""
    if isinstance(K, PagedKV):
        return K.desc()
    assert K.dtype.itemsize == 2 and K.stride(3) == 1
    if V is not None:
        assert V.shape == K.shape and V.stride() == K.stride()
    return cb_kv(K.data_ptr(), V.data_ptr() if V is not None else None, K.shape[2],
                 K.stride(0), K.stride(1), K.stride(2))


def query_desc(Q, Kself=None) -> cb_query:
    """Q: bf16 [nL][m][Hq][d]; Kself (optional): the query tokens' own keys, bf16 [nL][m][Hkv][d]."""
    assert Q.dtype.itemsize == 2 and Q.stride(3) == 1
    if Kself is None:
        return cb_query(Q.data_ptr(), Q.shape[1], Q.stride(0), Q.stride(1), Q.stride(2), None, 0, 0, 0)
    assert Kself.dtype.itemsize == 2 and Kself.stride(3) == 1 and Kself.shape[1] == Q.shape[1]
    return cb_query(Q.data_ptr(), Q.shape[1], Q.stride(0), Q.stride(1), Q.stride(2), Kself.data_ptr(),
                    Kself.stride(0), Kself.stride(1), Kself.stride(2))


class CacheBack:
    """One cb_ctx.  Methods enqueue work on a CUDA stream (default: torch's current stream)."""

    def __init__(self, n_layers: int, n_q_heads: int, n_kv_heads: int, head_dim: int, max_query_tokens: int,
                 max_positions: int, max_senders: int = 1, p: float = 2.0, alpha: float = 2.0,
                 pool_width: int = 7, span_width: int = 16, n_sink: int = 1, n_latent: int = 40,
                 softmax_scale: float = 0.0, score_kernel: int = 0, lib_path: Optional[str] = None):
        self.lib = load_library(lib_path)
        cfg = cb_config()
        self.lib.cb_config_init(ctypes.byref(cfg))
        cfg.n_layers, cfg.n_q_heads, cfg.n_kv_heads, cfg.head_dim = n_layers, n_q_heads, n_kv_heads, head_dim
        cfg.max_query_tokens, cfg.max_positions, cfg.max_senders = max_query_tokens, max_positions, max_senders
        cfg.softmax_scale, cfg.p, cfg.alpha = softmax_scale, p, alpha
        cfg.pool_width, cfg.span_width, cfg.n_sink, cfg.n_latent = pool_width, span_width, n_sink, n_latent
        cfg.score_kernel = score_kernel
        self.cfg = cfg
        h = ctypes.c_void_p()
        st = self.lib.cb_create(ctypes.byref(cfg), ctypes.byref(h))
        if st != CB_OK:
            raise CBError(st, self.lib.cb_last_error(None).decode())
        self.h = h

    def close(self):
        if getattr(self, "h", None):
            self.lib.cb_destroy(self.h)
            self.h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def _check(self, st: int):
        if st != CB_OK:
            raise CBError(st, self.lib.cb_last_error(self.h).decode())

    @property
    def scratch_bytes(self) -> int:
        return int(self.lib.cb_scratch_bytes(self.h))

    def score_path(self) -> int:
        """Logit-pass kernels of the last score call: 2 tcgen05, 1 mma.sync, 0 none yet."""
        return int(self.lib.cb_score_path(self.h))

    # -- the three steps ----------------------------------------------------
    def score(self, Ks: Sequence, Qs: Sequence, scores: Sequence, stream=None, Kselfs: Optional[Sequence] = None):
        """Kselfs (optional): per sender, the query tokens' own keys (or None) that join each
        query token's softmax causally."""
        n = len(Ks)
        kv = (cb_kv * n)(*[kv_desc(K) for K in Ks])
        Kselfs = Kselfs or [None] * n
        qq = (cb_query * n)(*[query_desc(Q, Kq) for Q, Kq in zip(Qs, Kselfs)])
        out = _ptr_array([s.data_ptr() for s in scores])
        self._check(self.lib.cb_score(self.h, n, kv, qq, out, _stream_handle(stream)))

    def select(self, scores: Sequence, Ts: Sequence[int], budgets: Sequence[int], idx: Sequence, stream=None):
        n = len(scores)
        sp = _ptr_array([s.data_ptr() for s in scores])
        Ta = _ptr_array([int(t) for t in Ts], ctypes.c_int64)
        Ba = _ptr_array([int(b) for b in budgets], ctypes.c_int64)
        ip = _ptr_array([x.data_ptr() for x in idx])
        self._check(self.lib.cb_select(self.h, n, sp, Ta, Ba, ip, _stream_handle(stream)))

    def compact(self, Ks: Sequence, Vs: Sequence, idx: Sequence, budgets: Sequence[int], k_out, v_out,
                offsets: Sequence[int], stream=None):
        """k_out, v_out: bf16 [nL][Hkv][capacity][d] (contiguous rows)."""
        n = len(Ks)
        kv = (cb_kv * n)(*[kv_desc(K, V) for K, V in zip(Ks, Vs)])
        ip = _ptr_array([x.data_ptr() for x in idx])
        Ba = _ptr_array([int(b) for b in budgets], ctypes.c_int64)
        Oa = _ptr_array([int(o) for o in offsets], ctypes.c_int64)
        assert k_out.stride(3) == 1 and k_out.stride(2) == k_out.shape[3] and v_out.stride() == k_out.stride()
        self._check(self.lib.cb_compact(self.h, n, kv, ip, Ba, k_out.data_ptr(), v_out.data_ptr(),
                                        k_out.shape[2], Oa, k_out.stride(0), k_out.stride(1),
                                        _stream_handle(stream)))

    def compact_rope(self, Ks: Sequence, Vs: Sequence, idx: Sequence, budgets: Sequence[int], k_out, v_out,
                     offsets: Sequence[int], base: float, style: int = 0, pos0: int = 0, stream=None):
        """compact with K moved to receiver positions pos0 + offset + j by the rotary embedding
        (style 0: pairs (k, k + d/2); 1: pairs (2k, 2k + 1))."""
        n = len(Ks)
        kv = (cb_kv * n)(*[kv_desc(K, V) for K, V in zip(Ks, Vs)])
        ip = _ptr_array([x.data_ptr() for x in idx])
        Ba = _ptr_array([int(b) for b in budgets], ctypes.c_int64)
        Oa = _ptr_array([int(o) for o in offsets], ctypes.c_int64)
        assert k_out.stride(3) == 1 and k_out.stride(2) == k_out.shape[3] and v_out.stride() == k_out.stride()
        self._check(self.lib.cb_compact_rope(self.h, n, kv, ip, Ba, k_out.data_ptr(), v_out.data_ptr(),
                                             k_out.shape[2], Oa, k_out.stride(0), k_out.stride(1), float(base),
                                             int(style), int(pos0), _stream_handle(stream)))

    def gather(self, tables: Sequence, idx: Sequence, counts: Sequence[int], out, offsets: Sequence[int],
               stream=None):
        """Message rows (App. C.3): out row offsets[i] + j = tables[i][idx[i][j]], j < counts[i].
        tables: per-sender [T_i][...] device tensors with one row per position (same row size and
        row stride); out: [capacity][...] with the same row size; idx: int32 device tensors."""
        n = len(tables)
        row_bytes = tables[0][0].numel() * tables[0].element_size()
        src_stride = tables[0].stride(0) * tables[0].element_size()
        for t in tables:
            assert t[0].is_contiguous() and t.stride(0) * t.element_size() == src_stride
            assert t[0].numel() * t.element_size() == row_bytes
        assert out[0].numel() * out.element_size() == row_bytes and out[0].is_contiguous()
        sp = _ptr_array([t.data_ptr() for t in tables])
        Ta = _ptr_array([int(t.shape[0]) for t in tables], ctypes.c_int64)
        ip = _ptr_array([x.data_ptr() for x in idx])
        Ca = _ptr_array([int(c) for c in counts], ctypes.c_int64)
        Oa = _ptr_array([int(o) for o in offsets], ctypes.c_int64)
        self._check(self.lib.cb_gather(self.h, n, sp, Ta, src_stride, row_bytes, ip, Ca, out.data_ptr(),
                                       out.shape[0], Oa, out.stride(0) * out.element_size(),
                                       _stream_handle(stream)))

    def set_wait_limit(self, limit_ns: int = 0, stall_next_score: bool = False):
        """cb_set_wait_limit: limit of one bounded device wait (0: the 1 s default); with
        stall_next_score the next tcgen05 cb_score makes one wait run out (failure-detection test)."""
        self._check(self.lib.cb_set_wait_limit(self.h, int(limit_ns), 1 if stall_next_score else 0))

    def set_score_sms(self, n_sms: int = 0):
        """cb_set_score_sms: SMs the persistent score kernels occupy (0: all)."""
        self._check(self.lib.cb_set_score_sms(self.h, int(n_sms)))

    STAGES = ("row_statistics", "statistics_combine", "normalised_accumulation", "finalize")

    def enable_stage_timing(self, enable=True):
        """True / 1: time every score kernel; 2: only the second logit pass; False / 0: off."""
        mode = int(enable) if not isinstance(enable, bool) else (1 if enable else 0)
        self._check(self.lib.cb_enable_stage_timing(self.h, mode))

    def stage_times(self):
        """(dict stage -> summed ms, number of cb_score calls) since the previous read."""
        ms = (ctypes.c_float * 4)()
        calls = ctypes.c_int32()
        self._check(self.lib.cb_stage_times(self.h, ms, ctypes.byref(calls)))
        return dict(zip(self.STAGES, list(ms))), int(calls.value)

    def sync_status(self, stream=None):
        self._check(self.lib.cb_sync_status(self.h, _stream_handle(stream)))
