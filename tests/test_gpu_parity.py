"""CUDA path vs the CPU oracle on sizes the oracle finishes in seconds (GPU).

Shapes span several tiles and ragged tails: 256-position stats chunks,
128-position accumulation chunks, 8-token query blocks, 64-token slabs.
"""
import zlib

import numpy as np
import pytest
import torch

import oracle
import paper_2609_32046_gb300 as cb
import synth
from gpu_helpers import (assert_scores_close, check_sender, make_cb, oracle_scores, run_path)

pytestmark = pytest.mark.gpu

CASES = [
    # name, shape (nL, Hq, Hkv, d), T list, m, keep, extra config
    ("tiny_spec", None, None, None, 0.25, {}),
    ("g4_d128_ragged", (2, 32, 8, 128), [1000], 64, 0.25, {}),
    ("g2_d64_odd_m", (3, 8, 4, 64), [777], 20, 0.30, {}),
    ("mha_d128", (2, 4, 4, 128), [300], 3, 0.40, {}),
    ("two_slabs", (1, 8, 2, 128), [700], 100, 0.25, {}),
    ("below_one_tile", (2, 8, 2, 64), [47], 5, 0.9, {}),
    ("p3_alpha1_pool5", (2, 8, 2, 64), [600], 12, 0.2, dict(p=3.0, alpha=1.0, pool_width=5)),
    ("mean_query_attention", (2, 8, 2, 64), [600], 12, 0.2, dict(alpha=0.0)),
    ("no_pooling", (2, 8, 2, 64), [600], 12, 0.2, dict(pool_width=1)),
    ("per_position_spans", (2, 8, 2, 64), [600], 12, 0.2, dict(span_width=1)),
    ("width8_spans_p1_5", (1, 8, 4, 128), [611], 9, 0.35, dict(span_width=8, p=1.5, alpha=4.0)),
    ("fan_in_ragged", (2, 16, 4, 128), [300, 513, 129], 33, 0.25, {}),
    ("m128_two_chunks", (2, 32, 8, 128), [900], 128, 0.25, {}),
    # 384 rows with G = 4: the last 256-row chunk has only its first column half
    ("g4_m96_three_halves", (2, 32, 8, 128), [1100], 96, 0.25, {}),
    ("g2_m200", (1, 8, 4, 128), [555], 200, 0.25, {}),
    ("g1_m300", (1, 2, 2, 128), [400], 300, 0.5, {}),
    ("pool3", (1, 8, 2, 128), [500], 40, 0.3, dict(pool_width=3)),
    ("pool5_p3", (1, 8, 2, 128), [500], 40, 0.3, dict(pool_width=5, p=3.0)),
    ("tail_1_position", (1, 8, 2, 128), [123], 8, 0.5, {}),
    # degenerate sizes: a single position, fewer positions than the forced 41, exactly 41
    ("degenerate_T", (2, 8, 2, 128), [1, 2, 40, 41, 129], 3, 0.5, {}),
    ("keep_everything", (1, 8, 2, 128), [300, 77], 5, 1.0, {}),
    ("keep_forced_only", (1, 8, 2, 64), [500], 4, 0.01, {}),
    # p = infinity (App. D.2): maxima instead of sums of powers
    ("p_inf_g4", (2, 32, 8, 128), [700], 40, 0.25, dict(p=float("inf"))),
    ("p_inf_g2_pool5", (2, 8, 4, 128), [611], 20, 0.3, dict(p=float("inf"), pool_width=5, alpha=3.0)),
    ("p_inf_d64", (2, 8, 2, 64), [600], 12, 0.2, dict(p=float("inf"))),
    ("p_inf_m128_four_halves", (1, 32, 8, 128), [700], 128, 0.3, dict(p=float("inf"))),
    # the query tokens' own keys join the softmax causally
    ("self_keys_g4", (2, 32, 8, 128), [700], 40, 0.25, dict(self_keys=True)),
    ("self_keys_g2_d64", (2, 8, 4, 64), [333], 17, 0.3, dict(self_keys=True)),
    ("self_keys_fan_in_m128", (1, 16, 4, 128), [300, 129], 128, 0.25, dict(self_keys=True)),
    # 100 query tokens: the staged self keys come in a chunk of 64 and one of 36
    ("self_keys_m100_two_chunks", (2, 8, 2, 128), [500], 100, 0.3, dict(self_keys=True)),
    # more senders than one tcgen05 launch takes (32): two launches per pass
    ("forty_senders", (1, 8, 2, 128), [97 + 13 * i for i in range(40)], 8, 0.3, {}),
]


def _workload(name, shape, Ts, m):
    if shape is None:
        return synth.make_workload("tiny")
    return synth.custom_workload(synth.Shape(*shape), Ts, m, seed=zlib.crc32(name.encode()) % 1000, n_planted_spans=2)


def _tc_supported(shape, m, extra):
    if shape is None:
        return False                      # the tiny workload has head_dim 64
    nL, Hq, Hkv, d = shape
    return d == 128 and extra.get("pool_width", 7) <= 7 and m * (Hq // Hkv) <= 512


@pytest.mark.parametrize("kernel", [1, 2], ids=["mma_sync", "tcgen05"])
@pytest.mark.parametrize("case", CASES, ids=[c[0] for c in CASES])
def test_parity(case, kernel):
    name, shape, Ts, m, keep, extra = case
    if kernel == 2 and not _tc_supported(shape, m, extra):
        pytest.skip("shape outside the tcgen05 score path")
    w = _workload(name, shape, Ts, m)
    extra = dict(extra)
    qk = None
    if extra.pop("self_keys", False):
        qk = [synth.make_query_keys(w.spec, 5, s.task) for s in w.senders]
    f = run_path(w, keep, score_kernel=kernel, query_keys=qk, **extra)
    assert f.cb.score_path() == kernel, "the requested logit-pass kernels did not run"
    kw = dict(p=extra.get("p", 2.0), alpha=extra.get("alpha", 2.0), pool_w=extra.get("pool_width", 7),
              span_w=extra.get("span_width", 16))
    for i, s in enumerate(w.senders):
        check_sender(f, i, s.K, s.V, w.queries[s.task], Kself=None if qk is None else qk[i], **kw)


def test_select_on_oracle_scores_is_exact():
    """Both sides rank the same fp32 scores in fp32: indices must be identical."""
    o = oracle.default()
    w = synth.custom_workload(synth.Shape(2, 8, 2, 64), [2000, 777, 65], 16, seed=5)
    c = make_cb(w.spec.shape, 2000, 16, 3)
    scores, Ts, Bs, idx = [], [], [], []
    for s in w.senders:
        S = o.score(s.K, w.queries[0])["S"].astype(np.float32)
        scores.append(torch.from_numpy(S).cuda())
        Ts.append(s.T)
        Bs.append(max(cb.budget(s.T, 0.3), min(s.T, 41)))
        idx.append(torch.empty(Bs[-1], dtype=torch.int32, device="cuda"))
    c.select(scores, Ts, Bs, idx)
    c.sync_status()
    for S, B, x in zip(scores, Bs, idx):
        want = o.select(S.cpu().numpy(), B)
        assert x.cpu().numpy().tolist() == want.tolist()


def test_select_ties_and_edge_budgets_exact():
    o = oracle.default()
    c = cb.CacheBack(1, 1, 1, 64, 1, 5000, 1)
    rng = np.random.default_rng(3)
    cases = [
        np.ones(1000, np.float32),                                # all spans tie
        np.round(rng.random(999) * 4).astype(np.float32),         # many ties, ragged last span
        np.zeros(300, np.float32),
        rng.random(41).astype(np.float32),                        # everything forced
        rng.random(4096).astype(np.float32),
    ]
    for S in cases:
        T = len(S)
        forced = min(T, 41)
        for B in sorted({forced, min(T, forced + 1), min(T, forced + 15), min(T, forced + 16), (T + forced) // 2, T}):
            x = torch.empty(max(B, 1), dtype=torch.int32, device="cuda")
            c.select([torch.from_numpy(S).cuda()], [T], [B], [x])
            c.sync_status()
            assert x[:B].cpu().numpy().tolist() == o.select(S, B).tolist(), (T, B)


def test_strided_inputs():
    """K/V stored position-major [T][nL][Hkv][d] and Q [m][nL][Hq][d]: strides, not copies."""
    w = synth.custom_workload(synth.Shape(2, 8, 2, 128), [513], 16, seed=9)
    s = w.senders[0]
    Kt = s.K.permute(2, 0, 1, 3).contiguous().cuda()   # [T][nL][Hkv][d]
    Vt = s.V.permute(2, 0, 1, 3).contiguous().cuda()
    Qt = w.queries[0].permute(1, 0, 2, 3).contiguous().cuda()
    K, V, Q = Kt.permute(1, 2, 0, 3), Vt.permute(1, 2, 0, 3), Qt.permute(1, 0, 2, 3)
    c = make_cb(w.spec.shape, 513, 16, 1)
    f = cb.Filter(c, [(K, V)], [Q], 0.25)
    f.run()
    c.sync_status()
    check_sender(f, 0, s.K, s.V, w.queries[0])


def test_deterministic_across_runs_and_streams():
    w = synth.custom_workload(synth.Shape(2, 16, 4, 128), [900, 400], 24, seed=2)
    f1 = run_path(w, 0.25)
    side = torch.cuda.Stream()
    with torch.cuda.stream(side):
        f2 = run_path(w, 0.25)
    torch.cuda.synchronize()
    for a, b in zip(f1.scores, f2.scores):
        assert torch.equal(a.view(torch.int32), b.view(torch.int32))
    assert torch.equal(f1.k_out.view(torch.int16), f2.k_out.view(torch.int16))


def test_scores_depend_on_the_query():
    """Sec. 4.2 query ablation: an unrelated query changes the selection."""
    w = synth.make_workload("tiny")
    s = w.senders[0]
    other = synth.make_query(w.spec, seed=99, task=0).cuda()
    c = make_cb(w.spec.shape, 512, 16, 2)
    f = cb.Filter(c, [(s.K.cuda(), s.V.cuda())] * 2, [w.queries[0].cuda(), other], 0.25)
    f.run()
    c.sync_status()
    a, b = f.indices()
    assert set(a.cpu().tolist()) != set(b.cpu().tolist())
    planted = {j for j in s.planted_spans}
    got = {int(t) // 16 for t in a.cpu().tolist()}
    assert planted <= got, "planted spans missed by the matching query"


def test_error_paths():
    w = synth.make_workload("tiny")
    s = w.senders[0]
    K, V, Q = s.K.cuda(), s.V.cuda(), w.queries[0].cuda()
    c = make_cb(w.spec.shape, 512, 16, 1)
    S = torch.empty(512, dtype=torch.float32, device="cuda")
    with pytest.raises(cb.CBError) as e:       # host memory is rejected, not dereferenced
        c.score([s.K], [Q], [S])
    assert e.value.status == cb.CB_EINVAL
    buf = torch.zeros(K.numel() + 8, dtype=torch.bfloat16, device="cuda")
    Kmis = buf[1:1 + K.numel()].view(K.shape)  # 2 bytes off a 16-byte boundary
    with pytest.raises(cb.CBError) as e:
        c.score([Kmis], [Q], [S])
    assert e.value.status == cb.CB_EINVAL
    with pytest.raises(cb.CBError) as e:       # T above the creation limit
        big = torch.zeros(2, 2, 600, 64, dtype=torch.bfloat16, device="cuda")
        c.score([big], [Q], [torch.empty(600, device="cuda")])
    assert e.value.status == cb.CB_ESHAPE
    c.score([K], [Q], [S])
    idx = torch.empty(128, dtype=torch.int32, device="cuda")
    with pytest.raises(cb.CBError) as e:       # budget below the 41 forced positions
        c.select([S], [512], [40], [idx])
    assert e.value.status == cb.CB_EBUDGET
    with pytest.raises(cb.CBError) as e:       # budget above T
        c.select([S], [512], [513], [idx])
    assert e.value.status == cb.CB_EBUDGET
    ko = torch.empty(2, 2, 100, 64, dtype=torch.bfloat16, device="cuda")
    with pytest.raises(cb.CBError) as e:       # capacity overflow
        c.compact([K], [V], [idx], [128], ko, torch.empty_like(ko), [0])
    assert e.value.status == cb.CB_EBUDGET
    bad = torch.full((128,), 7, dtype=torch.int32, device="cuda")
    bad[5] = 600                                # outside [0, T): skipped by the kernel, reported
    ko = torch.zeros(2, 2, 128, 64, dtype=torch.bfloat16, device="cuda")
    c.compact([K], [V], [bad], [128], ko, torch.empty_like(ko), [0])
    with pytest.raises(cb.CBError) as e:
        c.sync_status()
    assert e.value.status == cb.CB_EDEVICE
    c.sync_status()                             # the error word was cleared
    assert torch.equal(ko[:, :, 4], K[:, :, 7])
    assert not ko[:, :, 5].any()


def test_stage_timing_counts_calls_across_sender_batches():
    """Stage timing covers every sender batch of a call and counts cb_score calls, not batches."""
    name, shape, Ts, m, keep, extra = [c for c in CASES if c[0] == "forty_senders"][0]
    w = _workload(name, shape, Ts, m)
    c = make_cb(w.spec.shape, max(Ts), m, len(Ts), score_kernel=2)
    Ks = [s.K.cuda() for s in w.senders]
    Qs = [w.queries[s.task].cuda() for s in w.senders]
    S = [torch.empty(s.T, device="cuda") for s in w.senders]
    c.enable_stage_timing(True)
    c.stage_times()
    for _ in range(3):
        c.score(Ks, Qs, S)
    st, calls = c.stage_times()
    c.sync_status()
    assert c.score_path() == 2
    assert calls == 3
    assert all(v > 0 for v in st.values()), st
    # mode 2: only the second logit pass is bracketed (both sub-batches of each call)
    c.enable_stage_timing(2)
    c.stage_times()
    for _ in range(3):
        c.score(Ks, Qs, S)
    st2, calls2 = c.stage_times()
    assert calls2 == 3 and st2["normalised_accumulation"] > 0, st2
    assert st2["row_statistics"] == st2["statistics_combine"] == st2["finalize"] == 0.0, st2
    # about the same time for that kernel either way (a loose bound: timing noise)
    assert 0.5 < st2["normalised_accumulation"] / st["normalised_accumulation"] < 2.0
    with pytest.raises(cb.CBError) as e:
        c.enable_stage_timing(3)
    assert e.value.status == cb.CB_EINVAL
    c.enable_stage_timing(False)


def test_wave_schedule_matches_sequential():
    """Selection and compaction on a second stream under the next wave's scoring: same bytes."""
    name, shape, Ts, m, keep, extra = [c for c in CASES if c[0] == "forty_senders"][0]
    w = _workload(name, shape, Ts, m)
    c = make_cb(w.spec.shape, max(Ts), m, len(Ts), score_kernel=2)
    pairs = [(s.K.cuda(), s.V.cuda()) for s in w.senders]
    qs = [w.queries[s.task].cuda() for s in w.senders]
    ref = cb.Filter(c, pairs, qs, keep).run()
    got = cb.Filter(c, pairs, qs, keep).run(wave=7)
    c.sync_status()
    torch.cuda.synchronize()
    for a, b in zip(ref.scores, got.scores):
        assert torch.equal(a, b)
    for a, b, B in zip(ref.idx, got.idx, ref.budgets):
        assert torch.equal(a[:B], b[:B])
    assert torch.equal(ref.k_out.view(torch.int16), got.k_out.view(torch.int16))
    assert torch.equal(ref.v_out.view(torch.int16), got.v_out.view(torch.int16))



def test_results_do_not_depend_on_the_score_sms():
    """cb_set_score_sms: the tcgen05 passes on fewer SMs (a smaller persistent grid, so other
    contiguous work ranges) give the same bytes, and the wave schedule beside it too."""
    name, shape, Ts, m, keep, extra = [c for c in CASES if c[0] == "forty_senders"][0]
    w = _workload(name, shape, Ts, m)
    pairs = [(s.K.cuda(), s.V.cuda()) for s in w.senders]
    qs = [w.queries[s.task].cuda() for s in w.senders]
    c = make_cb(w.spec.shape, max(Ts), m, len(Ts), score_kernel=2)
    ref = cb.Filter(c, pairs, qs, keep).run()
    c.sync_status()
    for n_sms in (97, 16, 1):
        c.set_score_sms(n_sms)
        got = cb.Filter(c, pairs, qs, keep).run(wave=9)
        c.sync_status()
        assert c.score_path() == 2
        for a, b in zip(ref.scores, got.scores):
            assert torch.equal(a.view(torch.int32), b.view(torch.int32)), n_sms
        for a, b, B in zip(ref.idx, got.idx, ref.budgets):
            assert torch.equal(a[:B], b[:B]), n_sms
        assert torch.equal(ref.k_out.view(torch.int16), got.k_out.view(torch.int16)), n_sms
        assert torch.equal(ref.v_out.view(torch.int16), got.v_out.view(torch.int16)), n_sms
    c.set_score_sms(0)
    with pytest.raises(cb.CBError):
        c.set_score_sms(-1)


@pytest.mark.parametrize("kernel", [1, 2], ids=["mma_sync", "tcgen05"])
@pytest.mark.parametrize("scale", [70.0, 150.0], ids=["large_finite", "overflowing"])
def test_extreme_logit_rows(kernel, scale):
    """One query row meets keys far above the rest of its chunk: c*z - m about 100 log2 units stays
    in fp32 range on the fast path, about 210 overflows pass 1's exp2 and the combine kernel
    recomputes that row's statistics from Q and K.  Scores must still match the oracle."""
    w = synth.custom_workload(synth.Shape(2, 8, 2, 128), [700], 8, seed=77, n_planted_spans=2)
    s = w.senders[0]
    K, V, Q = s.K.clone(), s.V, w.queries[0]
    l, r, h = 1, 3, 5
    g = h // 4
    q = Q[l, r, h].float()
    K[l, g, 300:304] = (q / q.norm() * scale).to(torch.bfloat16)
    c = make_cb(w.spec.shape, 700, 8, 1, score_kernel=kernel)
    f = cb.Filter(c, [(K.cuda(), V.cuda())], [Q.cuda()], 0.25).run()
    c.sync_status()
    assert c.score_path() == kernel
    check_sender(f, 0, K, V, Q)


# Every pass-2 instantiation the tcgen05 path admits: k_accum_tc<G, pool_width / 2, p == 2>, G in
# {1, 2, 4}, pool widths 1, 3, 5, 7 and p = 2 or not (p = 3 for the general power).
TC_INSTANCES = [(G, pw, p) for G in (1, 2, 4) for pw in (1, 3, 5, 7) for p in (2.0, 3.0)]


@pytest.mark.parametrize("G,pool_width,p", TC_INSTANCES,
                         ids=["g%d_pool%d_p%g" % c for c in TC_INSTANCES])
def test_tcgen05_every_instantiation(G, pool_width, p):
    Hkv = 4
    m = {1: 61, 2: 45, 4: 33}[G]            # 61, 90 and 132 query rows: one and two 128-row halves
    w = synth.custom_workload(synth.Shape(2, G * Hkv, Hkv, 128), [431], m,
                              seed=100 * G + 10 * pool_width + int(p), n_planted_spans=2)
    extra = dict(pool_width=pool_width, p=p)
    f = run_path(w, 0.3, score_kernel=2, **extra)
    assert f.cb.score_path() == 2
    s = w.senders[0]
    check_sender(f, 0, s.K, s.V, w.queries[0], p=p, pool_w=pool_width)


@pytest.mark.parametrize("G", [1, 2, 4])
def test_tcgen05_unpooled_variance_identity(G):
    """App. C.1: at p = 2 without pooling, C_t = 1 + sum_s Var_r(b) / sum_s (mean_r b)^2, and with
    alpha = 1, S_t = Q_t C_t where Q_t = sum_s mean over (r, h) of a is the unpooled mean query
    attention.  b comes from torch's fp64 softmax (not from the oracle), and the GPU scores of the
    tcgen05 passes must satisfy the identity within the score tolerance."""
    import math
    nL, Hkv, T, m = 2, 4, 517, {1: 50, 2: 37, 4: 29}[G]
    Hq = G * Hkv
    w = synth.custom_workload(synth.Shape(nL, Hq, Hkv, 128), [T], m, seed=31 + G, n_planted_spans=3)
    f = run_path(w, 0.25, score_kernel=2, pool_width=1, p=2.0, alpha=1.0)
    assert f.cb.score_path() == 2
    K, Q = w.senders[0].K, w.queries[0]
    Qd = Q.to(torch.float64).permute(0, 2, 1, 3)                                  # [nL][Hq][m][d]
    eye = torch.eye(T, dtype=torch.float64).expand(nL, Hkv, T, T)
    a = torch.nn.functional.scaled_dot_product_attention(
        Qd, K.to(torch.float64), eye, scale=1.0 / math.sqrt(128), enable_gqa=True).numpy()   # [nL][Hq][m][T]
    b = a.reshape(nL, Hkv, G, m, T).mean(axis=2)                                  # [nL][Hkv][m][T]
    C = 1.0 + b.var(axis=2).sum(axis=(0, 1)) / (b.mean(axis=2) ** 2).sum(axis=(0, 1))
    U = a.sum(axis=(1, 2)).sum(axis=0) / (m * Hq)
    assert_scores_close(f.scores[0].cpu().numpy(), U * C)


def test_tcgen05_bounded_wait_gives_up_and_context_recovers():
    """Failure detection without a GPU fault: one wait of the row-statistics kernel is made to
    wait on a barrier nothing arrives on.  After the configured limit it gives up, the kernel
    drains its copies and MMAs, frees its tensor memory and returns; the host reads CB_ETIMEOUT.
    The same context then scores correctly."""
    w = synth.custom_workload(synth.Shape(2, 32, 8, 128), [3000], 64, seed=41, n_planted_spans=2)
    s = w.senders[0]
    K, V, Q = s.K.cuda(), s.V.cuda(), w.queries[0].cuda()
    c = make_cb(w.spec.shape, 3000, 64, 1, score_kernel=2)
    S = torch.empty(3000, device="cuda")
    c.set_wait_limit(20_000_000, stall_next_score=True)        # 20 ms
    c.score([K], [Q], [S])
    with pytest.raises(cb.CBError) as e:
        c.sync_status()
    assert e.value.status == cb.CB_ETIMEOUT
    assert "gave up" in str(e.value)
    c.sync_status()                                            # cleared
    # the stall was for one call; the short limit stays and ordinary waits stay far below it
    f = cb.Filter(c, [(K, V)], [Q], 0.25).run()
    c.sync_status()
    check_sender(f, 0, s.K, s.V, w.queries[0])
    c.set_wait_limit(0)
    with pytest.raises(cb.CBError) as e:
        c.set_wait_limit(10)                                   # below 1 microsecond
    assert e.value.status == cb.CB_EINVAL
