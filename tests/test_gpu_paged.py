"""Paged (block-table) sender caches on both score paths (GPU).

App. F serves the agents with vLLM, whose KV cache lives in fixed-size pages named by a
per-sequence block table.  Each sender's cache is scattered over a pool of pages in a random
order, with unused pages in between; the oracle unpages the pool by its definition and scores
the result.  The CUDA path reads the pages through the block table and must match the oracle
(scores within the tolerance, selection and compaction as the parity rules say), and must equal
the same sender in the strided layout bit for bit.  A block-table entry outside the pool is
never dereferenced: the call reports CB_EDEVICE.
"""
import ctypes
import math
import zlib

import numpy as np
import pytest
import torch

import oracle
import paper_2609_32046_gb300 as cb
import synth
from gpu_helpers import check_sender, make_cb

pytestmark = pytest.mark.gpu


def _page(K, V, P, n_extra, seed, head_major=False):
    """Scatter K, V [nL][Hkv][T][d] over a pool of pages in a random order.  Returns the PagedKV
    and the pool tensors; unused pages and rows hold unrelated values."""
    nL, Hkv, T, d = K.shape
    nb = (T + P - 1) // P
    n_pages = nb + n_extra
    g = torch.Generator().manual_seed(seed)
    order = torch.randperm(n_pages, generator=g)[:nb]                  # page of block b
    shape = (nL, n_pages, Hkv, P, d) if head_major else (nL, n_pages, P, Hkv, d)
    pools = []
    for X in (K, V):
        pool = torch.randn(shape, generator=g).to(torch.bfloat16).to(K.device)
        Xp = torch.cat([X, X.new_zeros(nL, Hkv, nb * P - T, d)], dim=2).view(nL, Hkv, nb, P, d)
        if head_major:
            pool[:, order.to(K.device)] = Xp.permute(0, 2, 1, 3, 4)      # [l][b][g][row][k]
        else:
            pool[:, order.to(K.device)] = Xp.permute(0, 2, 3, 1, 4)      # [l][b][row][g][k]
        pools.append(pool)
    kp, vp = pools
    if head_major:      # index order [l][page][row][g][k] as a view
        kp, vp = kp.permute(0, 1, 3, 2, 4), vp.permute(0, 1, 3, 2, 4)
    pages = order.to(torch.int32).to(K.device)
    return cb.PagedKV(kp, vp, pages, T)


def _bf16_tensor(bits):
    return torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).view(torch.bfloat16)


CASES = [
    # name, shape (nL, Hq, Hkv, d), T list, m, page size, head-major pool
    ("g4_p16_fanin", (2, 32, 8, 128), [700, 333], 40, 16, False),
    ("g2_p1_head_major", (1, 8, 4, 128), [517], 12, 1, True),
    ("g4_p256_few_pages", (1, 16, 4, 128), [1000], 20, 256, False),
    ("g2_d64_p64", (2, 8, 4, 64), [611], 17, 64, True),
]


def _tc_ok(shape, m):
    nL, Hq, Hkv, d = shape
    return d == 128 and m * (Hq // Hkv) <= 512


@pytest.mark.parametrize("kernel", [1, 2], ids=["mma_sync", "tcgen05"])
@pytest.mark.parametrize("case", CASES, ids=[c[0] for c in CASES])
def test_paged_matches_oracle_and_strided(case, kernel):
    name, shape, Ts, m, P, head_major = case
    if kernel == 2 and not _tc_ok(shape, m):
        pytest.skip("shape outside the tcgen05 score path")
    seed = zlib.crc32(name.encode()) % 1000
    w = synth.custom_workload(synth.Shape(*shape), Ts, m, seed=seed, n_planted_spans=2)
    Q = w.queries[0].cuda()
    Ks = [s.K.cuda() for s in w.senders]
    Vs = [s.V.cuda() for s in w.senders]
    paged = [_page(K, V, P, 3, seed + i, head_major) for i, (K, V) in enumerate(zip(Ks, Vs))]
    c = make_cb(w.spec.shape, max(Ts), m, len(Ts), score_kernel=kernel)
    f = cb.Filter(c, paged, [Q] * len(Ts), 0.3).run()
    c.sync_status()
    assert c.score_path() == kernel
    o = oracle.default()
    for i, pk in enumerate(paged):
        Ku = o.unpage(pk.k_pool.cpu(), pk.pages.cpu().numpy(), pk.T)
        Vu = o.unpage(pk.v_pool.cpu(), pk.pages.cpu().numpy(), pk.T)
        # the pool holds the sender's cache (checks the scatter above against the oracle's reading)
        assert np.array_equal(Ku, w.senders[i].K.view(torch.int16).numpy().view(np.uint16))
        check_sender(f, i, _bf16_tensor(Ku), _bf16_tensor(Vu), w.queries[0])
    # the strided layout gives the same bits
    c2 = make_cb(w.spec.shape, max(Ts), m, len(Ts), score_kernel=kernel)
    g = cb.Filter(c2, list(zip(Ks, Vs)), [Q] * len(Ts), 0.3).run()
    c2.sync_status()
    for i in range(len(Ts)):
        assert torch.equal(g.scores[i].view(torch.int32), f.scores[i].view(torch.int32)), i
        assert torch.equal(g.idx[i], f.idx[i]), i
    assert torch.equal(g.k_out.view(torch.int16), f.k_out.view(torch.int16))
    assert torch.equal(g.v_out.view(torch.int16), f.v_out.view(torch.int16))


def test_paged_and_strided_senders_in_one_call():
    """A call may mix layouts sender by sender (the tcgen05 passes batch them apart)."""
    w = synth.custom_workload(synth.Shape(1, 8, 2, 128), [300, 450, 129], 16, seed=3, n_planted_spans=2)
    Q = w.queries[0].cuda()
    pairs = [(s.K.cuda(), s.V.cuda()) for s in w.senders]
    mixed = [pairs[0], _page(*pairs[1], 16, 2, 5), pairs[2]]
    c = make_cb(w.spec.shape, 450, 16, 3)
    f = cb.Filter(c, mixed, [Q] * 3, 0.25).run()
    c.sync_status()
    c2 = make_cb(w.spec.shape, 450, 16, 3)
    g = cb.Filter(c2, pairs, [Q] * 3, 0.25).run()
    c2.sync_status()
    for i in range(3):
        assert torch.equal(g.scores[i].view(torch.int32), f.scores[i].view(torch.int32)), i
    assert torch.equal(g.k_out.view(torch.int16), f.k_out.view(torch.int16))


@pytest.mark.parametrize("kernel", [1, 2], ids=["mma_sync", "tcgen05"])
def test_bad_block_table_is_reported_not_read(kernel):
    w = synth.custom_workload(synth.Shape(1, 8, 2, 128), [300], 16, seed=9, n_planted_spans=2)
    K, V = w.senders[0].K.cuda(), w.senders[0].V.cuda()
    pk = _page(K, V, 16, 1, 9)
    for bad in (pk.n_pages, -1, 1 << 30):
        pages = pk.pages.clone()
        pages[5] = bad
        bad_kv = cb.PagedKV(pk.k_pool, pk.v_pool, pages, pk.T)
        c = make_cb(w.spec.shape, 300, 16, 1, score_kernel=kernel)
        f = cb.Filter(c, [bad_kv], [w.queries[0].cuda()], 0.25)
        f.score()
        with pytest.raises(cb.CBError, match="CB_EDEVICE"):
            c.sync_status()
        idx = torch.arange(70, 100, dtype=torch.int32, device="cuda")         # positions 80..95 sit in block 5
        ko = torch.full((1, 2, 30, 128), 7, dtype=torch.bfloat16, device="cuda")
        vo = ko.clone()
        c.compact([bad_kv], [bad_kv], [idx], [30], ko, vo, [0])
        with pytest.raises(cb.CBError, match="CB_EDEVICE"):
            c.sync_status()
        torch.cuda.synchronize()
        assert torch.equal(ko[:, :, :10], K[:, :, 70:80]) and torch.equal(ko[:, :, 26:], K[:, :, 96:100])
        assert bool((ko[:, :, 10:26] == 7).all())                             # rows of the bad page untouched


def test_bad_page_arguments_are_rejected():
    w = synth.custom_workload(synth.Shape(1, 8, 2, 128), [300], 16, seed=9, n_planted_spans=2)
    K, V = w.senders[0].K.cuda(), w.senders[0].V.cuda()
    pk = _page(K, V, 16, 1, 9)
    c = make_cb(w.spec.shape, 300, 16, 1)
    S = torch.empty(300, dtype=torch.float32, device="cuda")
    qd = cb.binding.query_desc(w.queries[0].cuda())
    for field, value in (("page_size", 12), ("page_size", 0), ("page_size", 1 << 17), ("s_page", 12),
                         ("n_pages", 0)):
        kv = pk.desc()
        setattr(kv, field, value)
        kva = (cb.binding.cb_kv * 1)(kv)
        qa = (cb.binding.cb_query * 1)(qd)
        out = (ctypes.c_void_p * 1)(S.data_ptr())
        st = c.lib.cb_score(c.h, 1, kva, qa, out, torch.cuda.current_stream().cuda_stream)
        assert st == cb.CB_EINVAL, (field, value, st)
