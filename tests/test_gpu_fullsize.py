"""Full-size workloads through the same calls bench.py times, against the CPU oracle (GPU).

Inputs are drawn on the GPU by the counter-based generator; the senders the oracle
checks are drawn again on the CPU (bit-identical by construction, and checked).
Where a workload has many senders the oracle checks a sample of them; every
sender's selection is still checked for its invariants and every sender's
compacted rows against the oracle's gather with the GPU's indices.
"""
import numpy as np
import pytest
import torch

import oracle
import paper_2609_32046_gb300 as cb
import synth
from gpu_helpers import assert_compact_exact, assert_scores_close, assert_selection_matches

pytestmark = pytest.mark.gpu


def _run(name, keep, senders=None):
    spec = synth.SPECS[name]
    w = synth.make_workload(name, seed=0, device="cuda", senders=senders)
    pairs = [(s.K, s.V) for s in w.senders]
    queries = [w.queries[s.task] for s in w.senders]
    sh = spec.shape
    c = cb.CacheBack(sh.n_layers, sh.n_q_heads, sh.n_kv_heads, sh.head_dim, spec.m, max(spec.T), len(pairs))
    f = cb.Filter(c, pairs, queries, keep)
    f.run()
    c.sync_status()
    torch.cuda.synchronize()
    assert c.score_path() == 2, "full-size workloads run the tcgen05 logit passes"
    return spec, w, f


def _check_sampled(spec, w, f, sample):
    o = oracle.default()
    for i in sample:
        snd = synth.make_sender(spec, 0, i, synth.make_query(spec, 0, i // spec.senders_per_task, "cpu"), "cpu")
        assert torch.equal(snd.K.view(torch.int16), w.senders[i].K.cpu().view(torch.int16)), "generator mismatch"
        Q = synth.make_query(spec, 0, i // spec.senders_per_task, "cpu")
        ref = o.score(snd.K, Q)
        assert_scores_close(f.scores[i].cpu().numpy(), ref["S"])
        B = f.budgets[i]
        ridx = o.select(ref["S"], B)
        assert_selection_matches(f.idx[i][:B].cpu().numpy(), ridx, ref["S"], B)
        # same fp32 scores ranked in fp32: identical indices
        assert f.idx[i][:B].cpu().numpy().tolist() == o.select(f.scores[i].cpu().numpy(), B).tolist()


def _check_all_compacted(w, f, oracle_sample):
    """Every sender: selection invariants and compacted rows equal to their source rows
    (the oracle's gather for the sampled senders, a device gather for the others)."""
    for i, s in enumerate(w.senders):
        B = f.budgets[i]
        idx_d = f.idx[i][:B]
        idx = idx_d.cpu().numpy()
        assert len(idx) == B and np.all(np.diff(idx) > 0)
        assert idx[0] == 0 and np.array_equal(idx[-40:], np.arange(s.T - 40, s.T))
        if i in oracle_sample:
            assert_compact_exact(f, i, s.K, s.V, idx_d)
        else:
            off = f.offsets[i]
            rows = idx_d.long()
            assert torch.equal(f.k_out[:, :, off:off + B].view(torch.int16), s.K[:, :, rows].view(torch.int16))
            assert torch.equal(f.v_out[:, :, off:off + B].view(torch.int16), s.V[:, :, rows].view(torch.int16))


def test_qwen8b_full():
    spec, w, f = _run("qwen8b", 0.25)
    assert f.budgets == [2048]
    _check_sampled(spec, w, f, [0])
    _check_all_compacted(w, f, [0])


def test_fanin_full():
    spec, w, f = _run("fanin", 0.25)
    assert f.budgets == [4096] * 3 and f.offsets == [0, 4096, 8192] and f.capacity == 12288
    _check_sampled(spec, w, f, [0])
    _check_all_compacted(w, f, [0, 1, 2])


def test_hybrid_full():
    spec, w, f = _run("hybrid", 0.10)
    assert f.budgets == [6554]
    _check_sampled(spec, w, f, [0])
    _check_all_compacted(w, f, [0])


@pytest.mark.parametrize("keep", [0.10, 0.25, 0.50])
def test_sweep_full(keep):
    spec, w, f = _run("sweep", keep)
    assert len(f.budgets) == 48
    assert f.budgets[0] == {0.10: 820, 0.25: 2048, 0.50: 4096}[keep]
    sample = [0] if keep != 0.25 else [0, 47]
    _check_sampled(spec, w, f, sample)
    _check_all_compacted(w, f, sample)
