"""The whole path captured into a CUDA graph (GPU).

score -> select -> compact allocate nothing and enqueue only kernels and events, so a caller can
capture a step once and replay it.  Replays must give the same bytes as direct calls, and the
stage timer's events, captured with the step, must time every replay.
"""
import pytest
import torch

import paper_2609_32046_gb300 as cb
import synth
from gpu_helpers import make_cb

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("kernel", [1, 2], ids=["mma_sync", "tcgen05"])
def test_graph_replay_matches_direct_calls(kernel):
    w = synth.custom_workload(synth.Shape(2, 16, 4, 128), [700, 333], 24, seed=12, n_planted_spans=2)
    pairs = [(s.K.cuda(), s.V.cuda()) for s in w.senders]
    Q = w.queries[0].cuda()
    c = make_cb(w.spec.shape, 700, 24, 2, score_kernel=kernel)
    f = cb.Filter(c, pairs, [Q, Q], 0.25)
    st = torch.cuda.Stream()
    f.run(st)                                   # direct (also sizes every scratch lazily used)
    c.sync_status(st)
    torch.cuda.synchronize()
    want = ([x.clone() for x in f.scores], [x.clone() for x in f.idx], f.k_out.clone(), f.v_out.clone())
    for x in f.scores + f.idx:
        x.zero_()
    f.k_out.zero_()
    f.v_out.zero_()
    c.enable_stage_timing(2)
    c.stage_times()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=st):
        f.run(st)
        f.run(st)
    with torch.cuda.stream(st):
        g.replay()
    torch.cuda.synchronize()
    c.sync_status(st)
    for a, b in zip(want[0], f.scores):
        assert torch.equal(a.view(torch.int32), b.view(torch.int32))
    for a, b in zip(want[1], f.idx):
        assert torch.equal(a, b)
    assert torch.equal(want[2].view(torch.int16), f.k_out.view(torch.int16))
    assert torch.equal(want[3].view(torch.int16), f.v_out.view(torch.int16))
    ms, calls = c.stage_times()
    assert calls == 2 and ms["normalised_accumulation"] > 0, (ms, calls)
    del g
    c.enable_stage_timing(False)
