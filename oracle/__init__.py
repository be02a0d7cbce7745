"""CPU oracle for CacheBack's score -> select -> compact path (fp64).

TEST INFRASTRUCTURE, NOT PRODUCT CODE.  Only `tests/`, `__graft_entry__.smoke()`
and the CPU-baseline / reference leg of `bench.py` may import this package.
It shares nothing with the CUDA path: the arithmetic lives in `cb_oracle.c`
(plain C, fp64, OpenMP over KV-head groups with a fixed-order final sum), built
here with gcc; `brute.py` is a second, literal numpy restatement used only on
tiny inputs.

Functions (each follows the paper's App. C.1 / C.2 in its own order):
  score(K, Q, ...)        -> dict of fp64 [T] arrays: S, Q, C, U, N, D
  attention(K, Q, scale)  -> a[l][h][r][t]
  select(S, B, ...)       -> int32 indices, ascending
  compact(K, V, idx, ...) -> gathered K, V rows
  budget(T, keep)         -> ceil(keep * T) in double, clamped to [0, T]
"""
from __future__ import annotations

import ctypes
import math
import os
import subprocess
from typing import Optional

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "cb_oracle.c")
_LIB_PATH = os.path.join(_HERE, "libcb_oracle.so")
CFLAGS = ["-O2", "-ffp-contract=off", "-fopenmp", "-fPIC", "-shared", "-Wall", "-Wextra"]

OK, EINVAL, ESHAPE, EBUDGET, ENOMEM = 0, 1, 2, 3, 4


def build(src: str = _SRC, out: str = _LIB_PATH, force: bool = False) -> str:
    """Compile the oracle with gcc (no nvcc, no CUDA)."""
    if not force and os.path.exists(out) and os.path.getmtime(out) >= os.path.getmtime(src):
        return out
    tmp = out + ".tmp%d" % os.getpid()
    subprocess.check_call(["gcc", *CFLAGS, "-o", tmp, src, "-lm"])
    os.replace(tmp, out)
    return out


class _Dims(ctypes.Structure):
    _fields_ = [
        ("n_layers", ctypes.c_int32), ("n_q_heads", ctypes.c_int32), ("n_kv_heads", ctypes.c_int32),
        ("head_dim", ctypes.c_int32), ("m", ctypes.c_int32), ("T", ctypes.c_int64),
        ("k_layer", ctypes.c_int64), ("k_head", ctypes.c_int64), ("k_pos", ctypes.c_int64),
        ("q_layer", ctypes.c_int64), ("q_tok", ctypes.c_int64), ("q_head", ctypes.c_int64),
        ("s_layer", ctypes.c_int64), ("s_tok", ctypes.c_int64), ("s_head", ctypes.c_int64),
    ]


_P = ctypes.c_void_p


class Oracle:
    """ctypes view of one build of cb_oracle.c (the default build, or a test's variant)."""

    def __init__(self, path: Optional[str] = None):
        self.path = path or build()
        lib = ctypes.CDLL(self.path)
        lib.cbo_score.argtypes = [ctypes.POINTER(_Dims), _P, _P, ctypes.c_double, ctypes.c_double,
                                  ctypes.c_double, ctypes.c_int32, ctypes.c_int32, _P, _P, _P, _P, _P, _P]
        lib.cbo_score.restype = ctypes.c_int
        lib.cbo_attention.argtypes = [ctypes.POINTER(_Dims), _P, _P, ctypes.c_double, _P]
        lib.cbo_attention.restype = ctypes.c_int
        lib.cbo_score_self.argtypes = [ctypes.POINTER(_Dims), _P, _P, _P, ctypes.c_double, ctypes.c_double,
                                       ctypes.c_double, ctypes.c_int32, ctypes.c_int32, _P, _P, _P, _P, _P, _P]
        lib.cbo_score_self.restype = ctypes.c_int
        lib.cbo_attention_self.argtypes = [ctypes.POINTER(_Dims), _P, _P, _P, ctypes.c_double, _P]
        lib.cbo_attention_self.restype = ctypes.c_int
        for name, ptr_t in (("cbo_select_f64", _P), ("cbo_select_f32", _P)):
            f = getattr(lib, name)
            f.argtypes = [ctypes.c_int64, ptr_t, ctypes.c_int64, ctypes.c_int32, ctypes.c_int32,
                          ctypes.c_int32, _P]
            f.restype = ctypes.c_int64
        lib.cbo_compact.argtypes = [ctypes.POINTER(_Dims), _P, _P, _P, ctypes.c_int64, _P, _P,
                                    ctypes.c_int64, ctypes.c_int64, ctypes.c_int64]
        lib.cbo_compact.restype = ctypes.c_int
        lib.cbo_compact_rope.argtypes = [ctypes.POINTER(_Dims), _P, _P, _P, ctypes.c_int64, _P, _P, ctypes.c_int64,
                                         ctypes.c_int64, ctypes.c_int64, ctypes.c_double, ctypes.c_int32,
                                         ctypes.c_int64]
        lib.cbo_compact_rope.restype = ctypes.c_int
        lib.cbo_gather.argtypes = [_P, ctypes.c_int64, ctypes.c_int64, ctypes.c_int64, _P, ctypes.c_int64, _P,
                                   ctypes.c_int64, ctypes.c_int64]
        lib.cbo_gather.restype = ctypes.c_int
        i32, i64 = ctypes.c_int32, ctypes.c_int64
        lib.cbo_unpage.argtypes = [_P, i32, i32, i32, i64, _P, i64, i64, i64, i64, i64, i64, _P]
        lib.cbo_unpage.restype = ctypes.c_int
        lib.cbo_pool.argtypes = [_P, _P, ctypes.c_int64, ctypes.c_int32]
        lib.cbo_pool.restype = None
        lib.cbo_max_threads.restype = ctypes.c_int
        self.lib = lib

    # -- helpers -----------------------------------------------------------
    @staticmethod
    def _bits(x) -> np.ndarray:
        """bf16 tensor/array -> contiguous uint16 bit array (host)."""
        try:
            import torch
            if isinstance(x, torch.Tensor):
                return x.detach().cpu().contiguous().view(torch.int16).numpy().view(np.uint16)
        except ImportError:  # pragma: no cover
            pass
        a = np.ascontiguousarray(x)
        if a.dtype != np.uint16:
            raise TypeError("expected bf16 bits as uint16")
        return a

    @staticmethod
    def _dims(Kb: np.ndarray, Qb: np.ndarray) -> _Dims:
        nL, Hkv, T, d = Kb.shape
        nL2, m, Hq, d2 = Qb.shape
        if nL2 != nL or d2 != d:
            raise ValueError("K and Q disagree on layers or head_dim")
        return _Dims(nL, Hq, Hkv, d, m, T, Hkv * T * d, T * d, d, m * Hq * d, Hq * d, d)

    def max_threads(self) -> int:
        return int(self.lib.cbo_max_threads())

    # -- App. C.1 ------------------------------------------------------------
    def _self_keys(self, dm: _Dims, Kself):
        """Bits of the query's own keys [nL][m][Hkv][d] (or None) with their strides set in dm."""
        if Kself is None:
            return None
        Ksb = self._bits(Kself)
        if Ksb.shape != (dm.n_layers, dm.m, dm.n_kv_heads, dm.head_dim):
            raise ValueError("the query's own keys must be [nL][m][Hkv][d]")
        dm.s_layer, dm.s_tok, dm.s_head = dm.m * dm.n_kv_heads * dm.head_dim, dm.n_kv_heads * dm.head_dim, dm.head_dim
        return Ksb

    def score(self, K, Q, p: float = 2.0, alpha: float = 2.0, pool_w: int = 7,
              scale: Optional[float] = None, n_threads: int = 0, Kself=None) -> dict:
        """Kself: the query tokens' own keys [nL][m][Hkv][d]; each query token's softmax then
        also runs over the keys of query tokens 0..r (None: sender positions only)."""
        Kb, Qb = self._bits(K), self._bits(Q)
        dm = self._dims(Kb, Qb)
        Ksb = self._self_keys(dm, Kself)
        T = dm.T
        if scale is None:
            scale = 1.0 / math.sqrt(dm.head_dim)
        out = {k: np.zeros(T, dtype=np.float64) for k in ("S", "Q", "C", "U", "N", "D")}
        st = self.lib.cbo_score_self(ctypes.byref(dm), Kb.ctypes.data, Qb.ctypes.data,
                                     None if Ksb is None else Ksb.ctypes.data, scale, p, alpha, pool_w, n_threads,
                                     *(out[k].ctypes.data for k in ("S", "Q", "C", "U", "N", "D")))
        if st != OK:
            raise RuntimeError("cbo_score failed with status %d" % st)
        return out

    def attention(self, K, Q, scale: Optional[float] = None, Kself=None) -> np.ndarray:
        Kb, Qb = self._bits(K), self._bits(Q)
        dm = self._dims(Kb, Qb)
        Ksb = self._self_keys(dm, Kself)
        if scale is None:
            scale = 1.0 / math.sqrt(dm.head_dim)
        a = np.zeros((dm.n_layers, dm.n_q_heads, dm.m, dm.T), dtype=np.float64)
        st = self.lib.cbo_attention_self(ctypes.byref(dm), Kb.ctypes.data, Qb.ctypes.data,
                                         None if Ksb is None else Ksb.ctypes.data, scale, a.ctypes.data)
        if st != OK:
            raise RuntimeError("cbo_attention failed with status %d" % st)
        return a

    def pool(self, x, w: int = 7) -> np.ndarray:
        x = np.ascontiguousarray(x, dtype=np.float64)
        y = np.empty_like(x)
        self.lib.cbo_pool(x.ctypes.data, y.ctypes.data, x.shape[0], w)
        return y

    # -- App. C.2 ------------------------------------------------------------
    def select(self, S, B: int, n_sink: int = 1, n_latent: int = 40, span_w: int = 16) -> np.ndarray:
        """Span selection.  fp32 scores are ranked in fp32, fp64 scores in fp64."""
        S = np.asarray(S)
        T = S.shape[0]
        idx = np.zeros(max(B, 1), dtype=np.int32)
        if S.dtype == np.float32:
            S = np.ascontiguousarray(S)
            n = self.lib.cbo_select_f32(T, S.ctypes.data, B, n_sink, n_latent, span_w, idx.ctypes.data)
        else:
            S = np.ascontiguousarray(S, dtype=np.float64)
            n = self.lib.cbo_select_f64(T, S.ctypes.data, B, n_sink, n_latent, span_w, idx.ctypes.data)
        if n < 0:
            raise ValueError("cbo_select failed with status %d" % (-n))
        return idx[:n]

    def compact(self, K, V, idx, out_k=None, out_v=None, offset: int = 0):
        Kb, Vb = self._bits(K), self._bits(V)
        nL, Hkv, T, d = Kb.shape
        idx = np.ascontiguousarray(idx, dtype=np.int32)
        B = idx.shape[0]
        if out_k is None:
            out_k = np.zeros((nL, Hkv, offset + B, d), dtype=np.uint16)
            out_v = np.zeros_like(out_k)
        cap = out_k.shape[2]
        dm = _Dims(nL, Hkv, Hkv, d, 1, T, Hkv * T * d, T * d, d, 0, 0, 0)
        st = self.lib.cbo_compact(ctypes.byref(dm), Kb.ctypes.data, Vb.ctypes.data, idx.ctypes.data, B,
                                  out_k.ctypes.data, out_v.ctypes.data, offset, Hkv * cap * d, cap * d)
        if st != OK:
            raise RuntimeError("cbo_compact failed with status %d" % st)
        return out_k, out_v


    def compact_rope(self, K, V, idx, base: float, style: int = 0, pos0: int = 0, out_k=None, out_v=None,
                     offset: int = 0):
        """Compaction with K moved from its sender positions idx[j] to receiver positions
        pos0 + offset + j by the rotary embedding (style 0: halves, 1: interleaved pairs)."""
        Kb, Vb = self._bits(K), self._bits(V)
        nL, Hkv, T, d = Kb.shape
        idx = np.ascontiguousarray(idx, dtype=np.int32)
        B = idx.shape[0]
        if out_k is None:
            out_k = np.zeros((nL, Hkv, offset + B, d), dtype=np.uint16)
            out_v = np.zeros_like(out_k)
        cap = out_k.shape[2]
        dm = _Dims(nL, Hkv, Hkv, d, 1, T, Hkv * T * d, T * d, d, 0, 0, 0)
        st = self.lib.cbo_compact_rope(ctypes.byref(dm), Kb.ctypes.data, Vb.ctypes.data, idx.ctypes.data, B,
                                       out_k.ctypes.data, out_v.ctypes.data, offset, Hkv * cap * d, cap * d,
                                       base, style, pos0)
        if st != OK:
            raise RuntimeError("cbo_compact_rope failed with status %d" % st)
        return out_k, out_v

    def gather(self, table, idx, out=None, offset: int = 0) -> np.ndarray:
        """Message rows (App. C.3): out[offset + j] = table[idx[j]] as raw bytes.  table: numpy
        array or tensor with one row per position (its leading axis)."""
        tb = np.ascontiguousarray(self._raw(table))
        T = tb.shape[0]
        row_bytes = tb[0].nbytes if T else 0
        idx = np.ascontiguousarray(idx, dtype=np.int32)
        if out is None:
            out = np.zeros((offset + idx.shape[0],) + tb.shape[1:], dtype=tb.dtype)
        assert out.flags.c_contiguous and out.dtype == tb.dtype and out.shape[1:] == tb.shape[1:]
        st = self.lib.cbo_gather(tb.ctypes.data, T, row_bytes, row_bytes, idx.ctypes.data, idx.shape[0],
                                 out.ctypes.data, offset, row_bytes)
        if st != OK:
            raise RuntimeError("cbo_gather failed with status %d" % st)
        return out

    def unpage(self, pool, pages, T: int) -> np.ndarray:
        """Paged cache layout (App. F, vLLM's block table): pool indexed [l][page][row][g][k]
        (P = rows per page), pages[b] = the page holding positions b*P .. b*P + P - 1.  Returns the
        contiguous cache [nL][Hkv][T][d] as bf16 bits."""
        pl = np.ascontiguousarray(self._raw(pool))
        nL, n_pages, P, Hkv, d = pl.shape
        pg = np.ascontiguousarray(pages, dtype=np.int32)
        out = np.zeros((nL, Hkv, T, d), dtype=pl.dtype)
        st = self.lib.cbo_unpage(pl.ctypes.data, nL, Hkv, d, T, pg.ctypes.data, P, n_pages,
                                 n_pages * P * Hkv * d, P * Hkv * d, Hkv * d, d, out.ctypes.data)
        if st != OK:
            raise RuntimeError("cbo_unpage failed with status %d" % st)
        return out

    @staticmethod
    def _raw(x) -> np.ndarray:
        if isinstance(x, np.ndarray):
            return x
        import torch
        x = x.detach().cpu().contiguous()
        if x.dtype in (torch.bfloat16, torch.float16):
            return x.view(torch.int16).numpy().view(np.uint16)
        return x.numpy()


def budget(T: int, keep: float) -> int:
    """B = ceil(keep * T) in double, clamped to [0, T] (App. C.2: B_i = ceil(T_i / r), keep = 1/r)."""
    return int(min(T, max(0, math.ceil(keep * T))))


def chain_budget(T_old: int, T_new: int, keep: float = 0.0, mode: str = "relative", B_max: int = 0) -> int:
    """One hop of a sequential chain (App. C.2): relative B = T_old + ceil(T_new / r) with r = 1/keep,
    fixed B = min(B_max, T_old + T_new); at most T_old + T_new."""
    T = T_old + T_new
    if mode == "relative":
        B = T_old + budget(T_new, keep)
    elif mode == "fixed":
        B = min(B_max, T)
    else:
        raise ValueError(mode)
    return min(T, max(0, B))


_DEFAULT: Optional[Oracle] = None


def default() -> Oracle:
    global _DEFAULT
    if _DEFAULT is None:
        _DEFAULT = Oracle()
    return _DEFAULT
