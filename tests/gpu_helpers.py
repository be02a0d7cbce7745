"""Shared helpers of the GPU parity tests: run the CUDA path, run the oracle, compare.

Tolerances (stated by the workload's acceptance rule, bf16 inputs, fp32 accumulation):
  scores      max relative error per position <= 2e-3 against the fp64 oracle
  selection   same count; a position may differ only inside a span whose oracle mean
              lies within 2e-3 * tau of tau, tau = the lowest mean among the spans the
              oracle admitted (the span where the budget ran out); with the oracle's
              scores cast to fp32 both sides rank in fp32 and must agree exactly
  compaction  bit-exact against the oracle's gather with the GPU's indices
"""
from __future__ import annotations

import math

import numpy as np
import torch

import oracle
import paper_2609_32046_gb300 as cb

SCORE_RTOL = 2e-3
SELECT_RTOL = 2e-3


def make_cb(shape, max_positions, m, n_senders=1, **kw):
    return cb.CacheBack(shape.n_layers, shape.n_q_heads, shape.n_kv_heads, shape.head_dim, m,
                        max_positions, n_senders, **kw)


def run_path(workload, keep, device="cuda", query_keys=None, **kw):
    """CUDA path over every sender of the workload: returns the Filter (results on device).
    query_keys: optional per-sender query self-keys (joining the softmax causally)."""
    spec = workload.spec
    senders = [(s.K.to(device), s.V.to(device)) for s in workload.senders]
    queries = [workload.queries[s.task].to(device) for s in workload.senders]
    m = max(q.shape[1] for q in queries)
    c = make_cb(spec.shape, max(s.T for s in workload.senders), m, len(senders), **kw)
    qk = None if query_keys is None else [k.to(device) for k in query_keys]
    f = cb.Filter(c, senders, queries, keep, query_keys=qk)
    f.run()
    c.sync_status()
    torch.cuda.synchronize()
    return f


def oracle_scores(o, K, Q, p=2.0, alpha=2.0, pool_w=7, scale=None, Kself=None):
    return o.score(K.cpu(), Q.cpu(), p=p, alpha=alpha, pool_w=pool_w, scale=scale,
                   Kself=None if Kself is None else Kself.cpu())


def assert_scores_close(gpu_S, ref_S, rtol=SCORE_RTOL):
    g = np.asarray(gpu_S, dtype=np.float64)
    r = np.asarray(ref_S, dtype=np.float64)
    assert g.shape == r.shape
    assert np.all(np.isfinite(g))
    rel = np.abs(g - r) / np.maximum(np.abs(r), 1e-30)
    worst = int(np.argmax(rel))
    assert rel[worst] <= rtol, "score rel err %.3e at t=%d (gpu %.9e, oracle %.9e)" % (rel[worst], worst, g[worst], r[worst])
    return float(rel.max())


def span_means(S, w, n_sink):
    S = np.asarray(S, dtype=np.float64).copy()
    if n_sink > 0:
        S[0] = S.max()
    T = len(S)
    return np.array([S[j:min(T, j + w)].mean() for j in range(0, T, w)])


def assert_selection_matches(gpu_idx, ref_idx, ref_S, B, span_w=16, n_sink=1, n_latent=40, rtol=SELECT_RTOL):
    g = np.asarray(gpu_idx, dtype=np.int64)
    r = np.asarray(ref_idx, dtype=np.int64)
    T = len(ref_S)
    assert len(g) == B == len(r), (len(g), B, len(r))
    assert np.all(np.diff(g) > 0), "GPU indices not strictly ascending"
    assert g.min() >= 0 and g.max() < T
    forced = set(range(min(n_sink, T))) | set(range(max(0, T - n_latent), T))
    assert forced <= set(g.tolist())
    diff = set(g.tolist()) ^ set(r.tolist())
    if not diff:
        return 0
    mu = span_means(ref_S, span_w, n_sink)
    admitted = {t // span_w for t in r.tolist() if t not in forced}
    tau = min(mu[j] for j in admitted)
    for t in diff:
        j = t // span_w
        assert abs(mu[j] - tau) <= rtol * tau, "position %d (span %d, mean %.9e) differs; tau %.9e" % (t, j, mu[j], tau)
    return len(diff)


def assert_compact_exact(f, sender_index, K, V, idx):
    o = oracle.default()
    B = f.budgets[sender_index]
    off = f.offsets[sender_index]
    ko, vo = o.compact(K.cpu(), V.cpu(), idx.cpu().numpy().astype(np.int32))
    gk = f.k_out[:, :, off:off + B].cpu().contiguous().view(torch.int16).numpy().view(np.uint16)
    gv = f.v_out[:, :, off:off + B].cpu().contiguous().view(torch.int16).numpy().view(np.uint16)
    assert np.array_equal(gk, ko), "compacted K differs"
    assert np.array_equal(gv, vo), "compacted V differs"


def check_sender(f, i, K, V, Q, o=None, p=2.0, alpha=2.0, pool_w=7, span_w=16, n_sink=1, n_latent=40,
                 scale=None, Kself=None):
    """Full parity of sender i of a finished Filter run against the oracle."""
    o = o or oracle.default()
    ref = oracle_scores(o, K, Q, p=p, alpha=alpha, pool_w=pool_w, scale=scale, Kself=Kself)
    gS = f.scores[i].cpu().numpy()
    err = assert_scores_close(gS, ref["S"])
    B = f.budgets[i]
    gidx = f.idx[i][:B].cpu().numpy()
    ridx = o.select(ref["S"], B, n_sink=n_sink, n_latent=n_latent, span_w=span_w)
    ndiff = assert_selection_matches(gidx, ridx, ref["S"], B, span_w, n_sink, n_latent)
    assert_compact_exact(f, i, K, V, f.idx[i][:B])
    return err, ndiff, ref
