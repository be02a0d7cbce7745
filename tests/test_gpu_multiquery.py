"""Multi-query serving: one sender state scored against many receiver queries in one launch (GPU).

The batch names the same K/V tensors once per query, each entry with its own query (different
token counts, optionally with the query's own keys).  Every (sender, query) pair must match the
oracle on its own, and must equal the same pair run alone bit for bit: a pair's arithmetic does
not depend on what else shares the launch.
"""
import dataclasses

import numpy as np
import pytest
import torch

import paper_2609_32046_gb300 as cb
import synth
from gpu_helpers import check_sender, make_cb

pytestmark = pytest.mark.gpu

SHAPE = synth.Shape(2, 32, 8, 128)
MS = [64, 40, 17, 128, 64]


def _state_and_queries(T=700, seed=23):
    w = synth.custom_workload(SHAPE, [T], max(MS), seed=seed, n_planted_spans=3)
    snd = w.senders[0]
    qs = []
    for j, m in enumerate(MS):
        spec = dataclasses.replace(w.spec, m=m)
        qs.append(synth.make_query(spec, seed + 100, j))
    kq = synth.make_query_keys(dataclasses.replace(w.spec, m=MS[1]), seed + 100, 1)
    return snd, qs, kq


def _run(c, K, V, qs, kqs, keep):
    f = cb.Filter(c, [(K, V)] * len(qs), qs, keep, query_keys=kqs)
    f.run()
    c.sync_status()
    torch.cuda.synchronize()
    return f


@pytest.mark.parametrize("kernel", [1, 2], ids=["mma_sync", "tcgen05"])
def test_one_state_many_queries(kernel):
    snd, qs, kq = _state_and_queries()
    K, V = snd.K.cuda(), snd.V.cuda()
    qd = [q.cuda() for q in qs]
    kqs = [None, kq.cuda(), None, None, None]          # the second query brings its own keys
    c = make_cb(SHAPE, snd.T, max(MS), len(qs), score_kernel=kernel)
    f = _run(c, K, V, qd, kqs, 0.25)
    assert c.score_path() == kernel
    for j in range(len(qs)):
        check_sender(f, j, snd.K, snd.V, qs[j], Kself=None if kqs[j] is None else kq)
    # the two m = 64 queries differ, so their messages must too
    assert not torch.equal(f.scores[0], f.scores[4])
    # each pair equals the same pair run alone
    for j in range(len(qs)):
        c1 = make_cb(SHAPE, snd.T, MS[j], 1, score_kernel=kernel)
        g = _run(c1, K, V, [qd[j]], [kqs[j]], 0.25)
        assert torch.equal(g.scores[0].view(torch.int32), f.scores[j].view(torch.int32)), j
        B = f.budgets[j]
        assert torch.equal(g.idx[0][:B], f.idx[j][:B]), j
        o = f.offsets[j]
        assert torch.equal(g.k_out[:, :, :B].view(torch.int16), f.k_out[:, :, o:o + B].view(torch.int16)), j


def test_full_size_queries_share_the_state():
    """Qwen3-8B-shaped state (36 layers, 8 KV heads, T = 8192) against three of the workload's
    64-token queries in one launch: each pair equals its single-pair run bit for bit (the
    single-pair path is checked against the oracle at this size in the full-size tests)."""
    w = synth.make_workload("multiquery", device="cuda", senders=[0, 5, 7])
    c = make_cb(w.spec.shape, 8192, 64, 3)
    f = cb.Filter(c, [(s.K, s.V) for s in w.senders], [w.queries[s.task] for s in w.senders], 0.25)
    f.run()
    c.sync_status()
    assert c.score_path() == 2
    for j, s in enumerate(w.senders):
        c1 = make_cb(w.spec.shape, 8192, 64, 1)
        g = cb.Filter(c1, [(s.K, s.V)], [w.queries[s.task]], 0.25).run()
        c1.sync_status()
        assert torch.equal(g.scores[0].view(torch.int32), f.scores[j].view(torch.int32)), j
        assert torch.equal(g.idx[0], f.idx[j][:f.budgets[j]]), j
        S = f.scores[j].cpu().numpy()
        assert np.all(np.isfinite(S)) and np.all(S > 0)
