"""Message encodings (Sec. 3.1 "State Representation", App. C.3) through cb_gather (GPU).

The continuous-row encoding sends one hidden-state row per selected position; the token-ID
encoding sends token IDs for the selected source positions and continuous rows for the latent
positions.  Both must equal the oracle's gather of the same rows byte for byte.
"""
import numpy as np
import pytest
import torch

import oracle
import paper_2609_32046_gb300 as cb
import synth
from gpu_helpers import make_cb

pytestmark = pytest.mark.gpu


def _filter(n_latent=40):
    w = synth.custom_workload(synth.Shape(2, 8, 2, 128), [300, 517, 64], 12, seed=31, n_planted_spans=2)
    c = make_cb(w.spec.shape, 517, 12, 3, n_latent=n_latent)
    pairs = [(s.K.cuda(), s.V.cuda()) for s in w.senders]
    qs = [w.queries[s.task].cuda() for s in w.senders]
    f = cb.Filter(c, pairs, qs, 0.25).run()
    c.sync_status()
    return c, f


def _tables(Ts, hidden, seed):
    g = torch.Generator().manual_seed(seed)
    rows = [torch.randn(T, hidden, generator=g).to(torch.bfloat16).cuda() for T in Ts]
    ids = [torch.randint(0, 151936, (T,), generator=g, dtype=torch.int32).cuda() for T in Ts]
    return rows, ids


def test_continuous_rows_match_oracle():
    c, f = _filter()
    rows, _ = _tables(f.Ts, 4096, 1)                  # 8 KiB rows, as for Qwen3-8B
    msg = f.message_rows(rows)
    c.sync_status()
    o = oracle.default()
    ref = np.zeros((f.capacity, 4096), dtype=np.uint16)
    for i in range(len(f.Ts)):
        o.gather(rows[i], f.idx[i][:f.budgets[i]].cpu().numpy(), out=ref, offset=f.offsets[i])
    assert np.array_equal(msg.cpu().view(torch.int16).numpy().view(np.uint16), ref)


def test_token_id_encoding_matches_oracle():
    c, f = _filter()
    rows, ids = _tables(f.Ts, 4096, 2)
    got_ids, got_rows = f.message_token_ids(ids, rows)
    c.sync_status()
    o = oracle.default()
    want_ids, want_rows = [], []
    for i, T in enumerate(f.Ts):
        sel = f.idx[i][:f.budgets[i]].cpu().numpy()
        L = min(T, 40)
        assert np.array_equal(sel[-L:], np.arange(T - L, T))   # the latent positions close every message
        want_ids.append(o.gather(ids[i], sel[:-L]))
        want_rows.append(o.gather(rows[i], sel[-L:]))
    assert np.array_equal(got_ids.cpu().numpy(), np.concatenate(want_ids))
    assert np.array_equal(got_rows.cpu().view(torch.int16).numpy().view(np.uint16), np.concatenate(want_rows))


def test_unaligned_rows_take_the_word_path():
    """Rows of 12 bytes in a 20-byte stride: the 4-byte-word kernel, still exact."""
    c, f = _filter()
    g = torch.Generator().manual_seed(3)
    base = [torch.randint(-2**31, 2**31 - 1, (T, 5), generator=g, dtype=torch.int32).cuda() for T in f.Ts]
    tables = [b[:, :3] for b in base]
    out = torch.full((f.capacity, 3), -1, dtype=torch.int32, device="cuda")
    c.gather(tables, f.idx, f.budgets, out, f.offsets)
    c.sync_status()
    o = oracle.default()
    for i in range(len(f.Ts)):
        sel = f.idx[i][:f.budgets[i]].cpu().numpy()
        want = o.gather(np.ascontiguousarray(tables[i].cpu().numpy()), sel)
        assert np.array_equal(out[f.offsets[i]:f.offsets[i] + f.budgets[i]].cpu().numpy(), want)


def test_empty_and_bad_indices():
    c, f = _filter()
    rows, _ = _tables(f.Ts, 256, 4)
    out = torch.zeros((8, 256), dtype=torch.bfloat16, device="cuda")
    idx = torch.tensor([0, 5, 10**6, 7], dtype=torch.int32, device="cuda")
    c.gather([rows[0], rows[1]], [idx, idx], [0, 4], out, [0, 2])     # sender 0 sends nothing
    with pytest.raises(cb.CBError, match="CB_EDEVICE"):
        c.sync_status()
    torch.cuda.synchronize()
    assert torch.equal(out[2], rows[1][0]) and torch.equal(out[3], rows[1][5]) and torch.equal(out[5], rows[1][7])
    assert not out[4].any() and not out[0].any()                      # the bad row was skipped
    with pytest.raises(cb.CBError, match="CB_EBUDGET"):
        c.gather([rows[0]], [idx], [4], out, [6])                     # rows past the capacity
