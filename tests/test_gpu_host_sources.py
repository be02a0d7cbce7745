"""Row sources in pinned host memory (GPU).

A sender cache may stay on the host: K is copied to the device for scoring, while compaction
reads only the selected K/V rows from pinned host memory across the link, and message gathers
read their rows from a pinned host table.  Results must equal the all-device path bit for bit
and the oracle; pageable host memory is refused, never dereferenced.
"""
import numpy as np
import pytest
import torch

import oracle
import paper_2609_32046_gb300 as cb
import synth
from gpu_helpers import assert_compact_exact, make_cb

pytestmark = pytest.mark.gpu


def _setup():
    w = synth.custom_workload(synth.Shape(2, 8, 2, 128), [700, 333], 12, seed=41, n_planted_spans=2)
    c = make_cb(w.spec.shape, 700, 12, 2)
    Q = w.queries[0].cuda()
    dev = [(s.K.cuda(), s.V.cuda()) for s in w.senders]
    f = cb.Filter(c, dev, [Q, Q], 0.25).run()
    c.sync_status()
    return w, c, f, dev


def test_compaction_reads_pinned_host_rows():
    w, c, f, dev = _setup()
    for where in ("v", "kv"):
        Ks = [s.K.pin_memory() if where == "kv" else K for s, (K, _) in zip(w.senders, dev)]
        Vs = [s.V.pin_memory() for s in w.senders]
        ko = torch.zeros_like(f.k_out)
        vo = torch.zeros_like(f.v_out)
        c.compact(Ks, Vs, f.idx, f.budgets, ko, vo, f.offsets)
        c.sync_status()
        assert torch.equal(ko.view(torch.int16), f.k_out.view(torch.int16)), where
        assert torch.equal(vo.view(torch.int16), f.v_out.view(torch.int16)), where
    for i, s in enumerate(w.senders):
        assert_compact_exact(f, i, s.K, s.V, f.idx[i][:f.budgets[i]])


def test_rows_inside_a_larger_pinned_allocation():
    """A host source that starts inside its allocation (here 128 bytes in) maps to the same rows."""
    w, c, f, dev = _setup()
    Vs = []
    for s in w.senders:
        big = torch.zeros(s.V.numel() + 64, dtype=torch.bfloat16).pin_memory()
        view = big[64:].view(s.V.shape)
        view.copy_(s.V)
        Vs.append(view)
    ko, vo = torch.zeros_like(f.k_out), torch.zeros_like(f.v_out)
    c.compact([K for K, _ in dev], Vs, f.idx, f.budgets, ko, vo, f.offsets)
    c.sync_status()
    assert torch.equal(vo.view(torch.int16), f.v_out.view(torch.int16))


def test_rope_compaction_reads_pinned_host_rows():
    w, c, f, dev = _setup()
    ref_k, ref_v = torch.zeros_like(f.k_out), torch.zeros_like(f.v_out)
    c.compact_rope([K for K, _ in dev], [V for _, V in dev], f.idx, f.budgets, ref_k, ref_v, f.offsets, 1e6, 0, 300)
    ko, vo = torch.zeros_like(f.k_out), torch.zeros_like(f.v_out)
    c.compact_rope([s.K.pin_memory() for s in w.senders], [s.V.pin_memory() for s in w.senders], f.idx,
                   f.budgets, ko, vo, f.offsets, 1e6, 0, 300)
    c.sync_status()
    assert torch.equal(ko.view(torch.int16), ref_k.view(torch.int16))
    assert torch.equal(vo.view(torch.int16), ref_v.view(torch.int16))


def test_gather_reads_a_pinned_host_table():
    w, c, f, dev = _setup()
    g = torch.Generator().manual_seed(5)
    tables = [torch.randn(T, 4096, generator=g).to(torch.bfloat16).pin_memory() for T in f.Ts]
    out = torch.zeros(f.capacity, 4096, dtype=torch.bfloat16, device="cuda")
    c.gather(tables, f.idx, f.budgets, out, f.offsets)
    c.sync_status()
    o = oracle.default()
    ref = np.zeros((f.capacity, 4096), dtype=np.uint16)
    for i in range(len(f.Ts)):
        o.gather(tables[i], f.idx[i][:f.budgets[i]].cpu().numpy(), out=ref, offset=f.offsets[i])
    assert np.array_equal(out.cpu().view(torch.int16).numpy().view(np.uint16), ref)


def test_pageable_host_memory_is_refused():
    w, c, f, dev = _setup()
    ko, vo = torch.zeros_like(f.k_out), torch.zeros_like(f.v_out)
    with pytest.raises(cb.CBError) as e:
        c.compact([K for K, _ in dev], [s.V for s in w.senders], f.idx, f.budgets, ko, vo, f.offsets)
    assert e.value.status == cb.CB_EINVAL
    with pytest.raises(cb.CBError) as e:
        c.gather([torch.zeros(T, 8, dtype=torch.int32) for T in f.Ts], f.idx, f.budgets,
                 torch.zeros(f.capacity, 8, dtype=torch.int32, device="cuda"), f.offsets)
    assert e.value.status == cb.CB_EINVAL
    with pytest.raises(cb.CBError) as e:            # cb_score needs K on the device (tensor maps)
        c.score([w.senders[0].K.pin_memory()], [w.queries[0].cuda()], [f.scores[0]])
    assert e.value.status == cb.CB_EINVAL
