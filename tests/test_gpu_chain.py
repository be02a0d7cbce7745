"""Sequential chains (App. C.2): each hop scores its inherited message plus its new positions,
selects under the chain budget and compacts into the next hop's cache (GPU).

Every hop is checked against the oracle on that hop's own cache (scores, the selection rule,
the budget) and the message it hands on is checked byte for byte against its source rows.
"""
import numpy as np
import pytest
import torch

import oracle
import paper_2609_32046_gb300 as cb
import synth
from gpu_helpers import assert_scores_close, assert_selection_matches, make_cb

pytestmark = pytest.mark.gpu


def _hops(shape, T_news, m, seed):
    w = synth.custom_workload(synth.Shape(*shape), T_news, m, seed=seed, n_planted_spans=2, shared_query=False)
    return [(s.K.cuda(), s.V.cuda(), w.queries[s.task].cuda()) for s in w.senders]


@pytest.mark.parametrize("mode,keep,B_max", [("relative", 0.25, 0), ("fixed", 0.0, 180)])
def test_three_hop_chain(mode, keep, B_max):
    shape, T_news, m = (2, 8, 2, 128), [300, 200, 260], 12
    hops = _hops(shape, T_news, m, seed=11)
    cap = sum(T_news)
    c = make_cb(synth.Shape(*shape), cap, m, 1)
    chain = cb.Chain(c, cap, keep=keep, mode=mode, B_max=B_max, device="cuda")
    o = oracle.default()
    T_old = 0
    for K_new, V_new, Q in hops:
        prev = None if T_old == 0 else chain.K[chain.cur][:, :, :T_old].clone()
        r = chain.hop(Q, K_new, V_new)
        c.sync_status()
        torch.cuda.synchronize()
        T_new = K_new.shape[2]
        assert r["T_old"] == T_old and r["T"] == T_old + T_new
        assert r["B"] == max(oracle.chain_budget(T_old, T_new, keep, mode, B_max), min(r["T"], 41))
        # the cache is the inherited message followed by the new positions
        if prev is not None:
            assert torch.equal(r["K"][:, :, :T_old].view(torch.int16), prev.view(torch.int16))
        assert torch.equal(r["K"][:, :, T_old:].view(torch.int16), K_new.view(torch.int16))
        Kc, Vc = r["K"].cpu().contiguous(), r["V"].cpu().contiguous()
        ref = o.score(Kc, Q.cpu())
        assert_scores_close(r["scores"].cpu().numpy(), ref["S"])
        B = r["B"]
        gidx = r["idx"].cpu().numpy()
        assert_selection_matches(gidx, o.select(ref["S"], B), ref["S"], B)
        # only the first and the last 40 positions are forced: inherited latent rows may go
        assert gidx[0] == 0 and np.array_equal(gidx[-40:], np.arange(r["T"] - 40, r["T"]))
        ko, vo = o.compact(Kc, Vc, gidx)
        assert np.array_equal(r["message_K"].cpu().contiguous().view(torch.int16).numpy().view(np.uint16), ko)
        assert np.array_equal(r["message_V"].cpu().contiguous().view(torch.int16).numpy().view(np.uint16), vo)
        T_old = B
    assert chain.T_old == T_old


def test_chain_rejects_overflow():
    shape = (1, 4, 2, 128)
    c = make_cb(synth.Shape(*shape), 200, 4, 1)
    chain = cb.Chain(c, 200, keep=0.5, device="cuda")
    with pytest.raises(ValueError):
        chain.new_slot(201)
