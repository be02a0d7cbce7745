"""cb_select_noalloc, the selection entry point for callers that cannot allocate device memory.

Such callers (code running inside a memory pool or arena it does not own, hosts
that forbid cudaMalloc after start-up, engines whose allocator is busy at the
point of the call) cannot create a cb_ctx, so this entry point keeps its scratch
in an array compiled into the library.  The selection kernel keeps the span
means of senders with at most 8192 spans in shared memory; longer senders
(more than 131072 positions at span width 16) keep them in that array.  These
tests call the entry point through the C-ABI and check that it returns exactly
what cb_select returns, on calls in a row that share the array: two calls whose
long senders sit at different places in it, and a call of more than 64 senders,
which the library launches in two groups that each place their long senders from
the start of the array.  Collected last so that a failure here never hides
another test's result.
"""
import ctypes

import pytest
import torch

import paper_2609_32046_gb300 as cb
from paper_2609_32046_gb300 import binding
from paper_2609_32046_gb300.build import build

pytestmark = pytest.mark.gpu


def _inputs(seed, Ts):
    g = torch.Generator().manual_seed(seed)
    scores = []
    for k, T in enumerate(Ts):
        x = torch.rand(T, generator=g)
        if k % 3 == 1:
            x = torch.round(x * 3)          # many equal span means: exercises the tie-break
        scores.append(x.to(torch.float32).cuda())
    return scores


def _call_noalloc(lib, scores, Ts, Bs, idx, n_sink=1, n_latent=40, span_w=16):
    n = len(scores)
    P = ctypes.c_void_p
    st = lib.cb_select_noalloc(n, (P * n)(*[s.data_ptr() for s in scores]),
                               (ctypes.c_int64 * n)(*Ts), (ctypes.c_int64 * n)(*Bs),
                               (P * n)(*[x.data_ptr() for x in idx]), n_sink, n_latent, span_w,
                               torch.cuda.current_stream().cuda_stream)
    return st


def _compare(lib, ctx, seed, Ts, keep=0.25):
    scores = _inputs(seed, Ts)
    Bs = [max(cb.budget(T, keep), min(T, 41)) for T in Ts]
    ref = [torch.empty(B, dtype=torch.int32, device="cuda") for B in Bs]
    ctx.select(scores, Ts, Bs, ref)
    ctx.sync_status()
    got = [torch.full((B,), -1, dtype=torch.int32, device="cuda") for B in Bs]
    assert _call_noalloc(lib, scores, Ts, Bs, got) == binding.CB_OK, lib.cb_last_error(None)
    st = lib.cb_select_noalloc_status(ctypes.c_void_p(torch.cuda.current_stream().cuda_stream))
    assert st == binding.CB_OK, lib.cb_last_error(None)
    for a, b in zip(ref, got):
        assert torch.equal(a, b)            # integer output: bit-exact


def test_noalloc_select_matches_cb_select_on_calls_in_a_row():
    build()
    lib = binding.load_library()
    # senders above 8192 spans use the array: 200000 (12500 slots) first at slot 0, then
    # 150000 and 140000 (9375 + 8750 slots) at slots 0 and 9375 over the first call's contents
    ctx = cb.CacheBack(1, 1, 1, 64, 1, 200000, 3)
    _compare(lib, ctx, 1, [200000, 300, 8192])
    _compare(lib, ctx, 2, [150000, 140000, 999])
    ctx.close()
    # 130 senders: launched as 64 + 64 + 2; none has more than 8192 spans, so no slot is used
    ctx = cb.CacheBack(1, 1, 1, 64, 1, 8192, 130)
    _compare(lib, ctx, 3, [8192 - 37 * (k % 5) for k in range(130)])
    ctx.close()


def test_noalloc_select_rejects_oversized_calls_and_bad_budgets():
    build()
    lib = binding.load_library()
    Ts = [70000 * 16]                          # 70000 spans > 65536 slots
    scores = [torch.zeros(Ts[0], dtype=torch.float32, device="cuda")]
    idx = [torch.empty(100, dtype=torch.int32, device="cuda")]
    assert _call_noalloc(lib, scores, Ts, [100], idx) == binding.CB_ESHAPE
    assert b"span slots" in lib.cb_last_error(None)
    small = [torch.zeros(512, dtype=torch.float32, device="cuda")]
    assert _call_noalloc(lib, small, [512], [40], idx) == binding.CB_EBUDGET
    assert _call_noalloc(lib, [torch.zeros(512)], [512], [64], idx) == binding.CB_EINVAL  # host memory
    # a refused call leaves the error text; a good call clears it
    assert _call_noalloc(lib, small, [512], [64], idx) == binding.CB_OK
    assert lib.cb_last_error(None) == b""
    assert lib.cb_select_noalloc_status(ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)) == binding.CB_OK
