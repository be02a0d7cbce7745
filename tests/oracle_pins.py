"""Pins that tie the CPU oracle to facts outside itself.

Each pin takes an oracle object (the default build, or a build with a planted
mistake) and raises AssertionError when the oracle disagrees with:
  - a library routine the step reduces to (torch's scaled_dot_product_attention
    for the attention weights and the GQA head mapping, scipy's windowed max
    filter for Pool_7, numpy fancy indexing for the gather);
  - a closed form (App. C.1's unpooled-variance identity; hand-solved one-hot
    attention patterns with pooling; identical keys);
  - an invariant (softmax rows sum to one, sum_t of the layer term is |L|, C >= 1);
  - hand-derived selections under App. C.2's rule (tests/golden/select_cases.json);
  - the literal numpy restatement in oracle/brute.py on tiny inputs.
"""
from __future__ import annotations

import json
import math
import os

import numpy as np
import torch

import synth
from oracle import brute

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")


def _bits(x: torch.Tensor) -> np.ndarray:
    return x.contiguous().view(torch.int16).numpy().view(np.uint16)


def _bf16(a) -> torch.Tensor:
    return torch.as_tensor(np.asarray(a, dtype=np.float32)).to(torch.bfloat16)


def _rand_case(nL=2, Hq=4, Hkv=2, d=32, T=53, m=5, seed=1):
    w = synth.custom_workload(synth.Shape(nL, Hq, Hkv, d), [T], m, seed=seed, n_planted_spans=1, n_latent=4)
    return w.senders[0].K, w.senders[0].V, w.queries[0]


def _rel(x, y):
    x, y = np.asarray(x, np.float64), np.asarray(y, np.float64)
    return float(np.max(np.abs(x - y) / np.maximum(np.abs(y), 1e-300)))


# --------------------------------------------------------------------------
# Pool_7 (App. C.1): local maximum over seven positions, centred, clipped
# --------------------------------------------------------------------------

def pin_pool_one_hot(o):
    T = 20
    for p in (0, 1, 3, 10, 16, 19):
        x = np.zeros(T)
        x[p] = 1.0
        y = o.pool(x, 7)
        want = np.array([1.0 if abs(t - p) <= 3 else 0.0 for t in range(T)])
        assert np.array_equal(y, want), ("Pool_7 of a one-hot at %d" % p, y, want)


def pin_pool_library(o):
    from scipy.ndimage import maximum_filter1d
    rng = np.random.default_rng(5)
    for T, w in ((1, 7), (2, 7), (5, 7), (64, 7), (33, 3), (40, 1)):
        x = rng.standard_normal(T)
        # mode="nearest" repeats the edge value, which never exceeds the clipped window's max
        want = maximum_filter1d(x, size=w, mode="nearest")
        assert np.array_equal(o.pool(x, w), want), (T, w)


# --------------------------------------------------------------------------
# attention weights and the GQA mapping vs torch's SDPA
# --------------------------------------------------------------------------

def pin_attention_sdpa(o):
    """a[l][h][r][t] equals SDPA's attention probabilities (V = identity)."""
    for (nL, Hq, Hkv, d, T, m) in ((2, 4, 2, 32, 23, 3), (1, 6, 2, 16, 17, 2), (1, 3, 3, 16, 9, 4)):
        K, _, Q = _rand_case(nL, Hq, Hkv, d, T, m, seed=T)
        a = o.attention(K, Q)
        Kd = K.to(torch.float64)            # [nL][Hkv][T][d]
        Qd = Q.to(torch.float64).permute(0, 2, 1, 3)   # [nL][Hq][m][d]
        eye = torch.eye(T, dtype=torch.float64).expand(nL, Hkv, T, T)
        probs = torch.nn.functional.scaled_dot_product_attention(
            Qd, Kd, eye, scale=1.0 / math.sqrt(d), enable_gqa=True)
        assert np.allclose(a, probs.numpy(), rtol=1e-12, atol=1e-15), (nL, Hq, Hkv)


# --------------------------------------------------------------------------
# closed forms
# --------------------------------------------------------------------------

def _one_hot_case(T=32, t1=10, t2=12, gamma=4.0, kappa=4.0, d=16):
    """One layer, one head, two query tokens.  q_r = gamma e_r; k_t1 = kappa e_0,
    k_t2 = kappa e_1, other keys zero.  Row r has one logit gamma*kappa/sqrt(d) at
    t_r and zeros elsewhere, so a = hi at t_r and lo elsewhere."""
    K = np.zeros((1, 1, T, d), np.float32)
    K[0, 0, t1, 0] = kappa
    K[0, 0, t2, 1] = kappa
    Q = np.zeros((1, 2, 1, d), np.float32)
    Q[0, 0, 0, 0] = gamma
    Q[0, 1, 0, 1] = gamma
    z = gamma * kappa / math.sqrt(d)
    E = math.exp(z)
    hi, lo = E / (E + T - 1), 1.0 / (E + T - 1)
    return _bf16(K), _bf16(Q), hi, lo


def pin_one_hot_closed_form(o):
    T, t1, t2 = 32, 10, 12
    K, Q, hi, lo = _one_hot_case(T, t1, t2)
    for p, alpha in ((2.0, 2.0), (3.0, 1.0), (2.0, 0.0), (1.5, 4.0)):
        r = o.score(K, Q, p=p, alpha=alpha, pool_w=7)
        for t in range(T):
            P1 = hi if abs(t - t1) <= 3 else lo       # Pool_7(b_1)_t
            P2 = hi if abs(t - t2) <= 3 else lo       # Pool_7(b_2)_t
            Nw = (P1 ** p + P2 ** p) / 2.0            # mean_r Pool(b_r)^p
            bb = (hi + lo) / 2.0 if (abs(t - t1) <= 3 or abs(t - t2) <= 3) else lo  # Pool_7(mean_r b)_t
            Dw = bb ** p
            Uw = (hi + lo) / 2.0 if t in (t1, t2) else lo   # layer term before pooling
            Qw = bb                                   # Pool_7(U) has the same support as Pool_7(bbar)
            Cw = (Nw / Dw) ** (1.0 / (p - 1.0))
            Sw = Qw * Cw ** alpha
            for key, want in (("U", Uw), ("Q", Qw), ("N", Nw), ("D", Dw), ("C", Cw), ("S", Sw)):
                got = r[key][t]
                assert abs(got - want) <= 1e-12 * abs(want), (key, t, p, alpha, got, want)


def pin_zero_denominator(o):
    """Logits 1024 apart underflow a to exactly 0 away from t1: both sums vanish there and C = 1."""
    T, t1, d = 32, 5, 16
    K = np.zeros((1, 1, T, d), np.float32)
    K[0, 0, t1, 0] = 64.0
    Q = np.zeros((1, 1, 1, d), np.float32)
    Q[0, 0, 0, 0] = 64.0
    r = o.score(_bf16(K), _bf16(Q))
    far = [t for t in range(T) if abs(t - t1) > 3]
    assert np.all(r["D"][far] == 0.0) and np.all(r["N"][far] == 0.0)
    assert np.all(r["C"][far] == 1.0), r["C"][far]
    assert np.all(r["S"][far] == 0.0)


def pin_variance_identity(o):
    """App. C.1: at p = 2 without pooling, C_t = 1 + sum_s Var_r(b) / sum_s (mean_r b)^2,
    with b from torch's SDPA probabilities averaged over each KV head's query heads."""
    for (nL, Hq, Hkv, d, T, m) in ((2, 4, 2, 32, 40, 6), (1, 8, 2, 16, 25, 3)):
        K, _, Q = _rand_case(nL, Hq, Hkv, d, T, m, seed=7 + T)
        r = o.score(K, Q, p=2.0, alpha=2.0, pool_w=1)
        Qd = Q.to(torch.float64).permute(0, 2, 1, 3)
        eye = torch.eye(T, dtype=torch.float64).expand(nL, Hkv, T, T)
        a = torch.nn.functional.scaled_dot_product_attention(
            Qd, K.to(torch.float64), eye, scale=1.0 / math.sqrt(d), enable_gqa=True).numpy()
        G = Hq // Hkv
        b = a.reshape(nL, Hkv, G, m, T).mean(axis=2)      # [nL][Hkv][m][T]
        var = b.var(axis=2).sum(axis=(0, 1))
        mean2 = (b.mean(axis=2) ** 2).sum(axis=(0, 1))
        want = 1.0 + var / mean2
        assert _rel(r["C"], want) < 1e-12, _rel(r["C"], want)


def pin_identical_keys(o):
    """All keys equal: a = 1/T, Q_t = |L|/T, C = 1, all span means tie, and the
    selection is [0, B - n_latent) plus the latent tail."""
    nL, Hq, Hkv, d, T, m = 3, 4, 2, 16, 200, 5
    K, _, Q = _rand_case(nL, Hq, Hkv, d, T, m, seed=11)
    K = K[:, :, :1, :].expand(nL, Hkv, T, d).contiguous()
    r = o.score(K, Q)
    assert np.allclose(r["Q"], nL / T, rtol=1e-13, atol=0)
    assert np.allclose(r["C"], 1.0, rtol=1e-13, atol=0)
    assert np.all(r["S"] == r["S"][0])
    for B in (41, 60, 77, 150, 200):
        idx = o.select(r["S"], B, n_sink=1, n_latent=40, span_w=16)
        want = sorted(set(range(B - 40)) | set(range(T - 40, T)))
        assert idx.tolist() == want, (B, idx.tolist())


# --------------------------------------------------------------------------
# invariants and special cases
# --------------------------------------------------------------------------

def pin_invariants(o):
    for (nL, Hq, Hkv, d, T, m) in ((2, 4, 2, 32, 61, 5), (3, 8, 4, 16, 100, 7)):
        K, _, Q = _rand_case(nL, Hq, Hkv, d, T, m, seed=T + m)
        a = o.attention(K, Q)
        assert np.allclose(a.sum(axis=-1), 1.0, rtol=0, atol=1e-13)
        r = o.score(K, Q)
        assert abs(r["U"].sum() - nL) < 1e-12 * nL, r["U"].sum()
        assert np.all(r["C"] >= 1.0 - 1e-13), r["C"].min()
        assert np.all(r["Q"] >= r["U"] - 1e-18)          # a max-pool never lowers a value
        for p in (1.5, 3.0, 8.0):
            assert np.all(o.score(K, Q, p=p)["C"] >= 1.0 - 1e-13)


def pin_special_cases(o):
    K, _, Q = _rand_case(2, 4, 2, 32, 47, 6, seed=3)
    # one query token: pooling then averaging over r is the identity, so C = 1 and S = Q
    r1 = o.score(K, Q[:, :1].contiguous())
    assert np.allclose(r1["C"], 1.0, rtol=1e-13, atol=0) and _rel(r1["S"], r1["Q"]) < 1e-13
    # alpha = 0 is mean query attention (App. D.2)
    r0 = o.score(K, Q, alpha=0.0)
    assert np.array_equal(r0["S"], r0["Q"])
    # MHA (G = 1): b = a, so N = sum_l mean_r Pool(a)^p with a from SDPA
    Km, _, Qm = _rand_case(1, 3, 3, 16, 30, 4, seed=9)
    rm = o.score(Km, Qm, pool_w=7)
    from scipy.ndimage import maximum_filter1d
    Qd = Qm.to(torch.float64).permute(0, 2, 1, 3)
    eye = torch.eye(30, dtype=torch.float64).expand(1, 3, 30, 30)
    a = torch.nn.functional.scaled_dot_product_attention(Qd, Km.to(torch.float64), eye,
                                                         scale=0.25).numpy()
    pooled = maximum_filter1d(a, size=7, axis=-1, mode="nearest")
    assert _rel(rm["N"], (pooled ** 2).mean(axis=2).sum(axis=(0, 1))) < 1e-12


def pin_equivariance(o):
    """S does not change when query tokens, heads within a group, KV groups with
    their heads, or layers are permuted."""
    nL, Hq, Hkv, d, T, m = 2, 8, 2, 16, 45, 5
    K, _, Q = _rand_case(nL, Hq, Hkv, d, T, m, seed=21)
    S = o.score(K, Q)["S"]
    G = Hq // Hkv
    variants = []
    variants.append((K, Q[:, [3, 0, 4, 1, 2]]))                               # query tokens
    variants.append((K, Q[:, :, [2, 0, 3, 1, 5, 7, 4, 6]]))                   # heads within each group
    variants.append((K[:, [1, 0]], Q[:, :, list(range(G, 2 * G)) + list(range(G))]))  # KV groups
    variants.append((K[[1, 0]], Q[[1, 0]]))                                    # layers
    for Kp, Qp in variants:
        Sp = o.score(Kp.contiguous(), Qp.contiguous())["S"]
        assert _rel(Sp, S) < 1e-12, _rel(Sp, S)


def pin_brute(o):
    """The C oracle and the literal numpy restatement agree on tiny inputs."""
    for (nL, Hq, Hkv, d, T, m, p, alpha, w) in ((2, 4, 2, 32, 61, 5, 2.0, 2.0, 7), (1, 8, 2, 16, 40, 3, 3.0, 1.0, 7),
                                                (2, 2, 2, 16, 7, 1, 2.0, 2.0, 7), (1, 4, 1, 16, 33, 4, 1.5, 4.0, 3)):
        K, _, Q = _rand_case(nL, Hq, Hkv, d, T, m, seed=T * 3 + m)
        r = o.score(K, Q, p=p, alpha=alpha, pool_w=w)
        b = brute.score(_bits(K), _bits(Q), p=p, alpha=alpha, pool_w=w)
        for k in ("S", "Q", "C", "U", "N", "D"):
            assert _rel(r[k], b[k]) < 1e-12, (k, _rel(r[k], b[k]))
        for B in ((max(41, T // 4) if T >= 41 else T), T):
            assert o.select(r["S"], B).tolist() == brute.select(r["S"], B).tolist()


def pin_p_infinity(o):
    """p = infinity (App. D.2): C = max_{s,r} Pool(b) / max_s Pool(mean_r b), pinned by
    (i) the literal numpy restatement, (ii) the limit of the finite-p oracle, which for any p
    lies within factors (A/B)^(1/(p-1)) (m nS)^(-1/(p-1)) and (A/B)^(1/(p-1)) nS^(1/(p-1)) of
    C_inf (A, B the two maxima), (iii) one group without pooling, where C = max_r b / mean_r b
    with b from torch's SDPA, and (iv) one query token, where C = 1."""
    inf = float("inf")
    for (nL, Hq, Hkv, d, T, m, w) in ((2, 4, 2, 32, 61, 5, 7), (1, 8, 2, 16, 40, 3, 3)):
        K, _, Q = _rand_case(nL, Hq, Hkv, d, T, m, seed=T + 7 * m)
        r = o.score(K, Q, p=inf, alpha=2.0, pool_w=w)
        b = brute.score(_bits(K), _bits(Q), p=inf, alpha=2.0, pool_w=w)
        for k in ("S", "C", "N", "D"):
            assert _rel(r[k], b[k]) < 1e-12, (k, _rel(r[k], b[k]))
    # (ii) the finite-p limit, on a case small enough that b^p stays far from underflow
    nL, Hq, Hkv, d, T, m = 2, 4, 2, 16, 24, 4
    K, _, Q = _rand_case(nL, Hq, Hkv, d, T, m, seed=77)
    ri = o.score(K, Q, p=inf, alpha=1.0)
    A, B = ri["N"], ri["D"]
    nS = nL * Hkv
    for p in (24.0, 48.0):
        rp = o.score(K, Q, p=p, alpha=1.0)
        e = 1.0 / (p - 1.0)
        ratio = rp["C"] / ri["C"]
        lo = (A / B) ** e * (m * nS) ** (-e)
        hi = (A / B) ** e * nS ** e
        assert np.all(ratio >= lo * (1 - 1e-12)) and np.all(ratio <= hi * (1 + 1e-12)), p
    # (iii) one group, no pooling
    K1, _, Q1 = _rand_case(1, 2, 1, 16, 30, 4, seed=5)
    r1 = o.score(K1, Q1, p=inf, alpha=1.0, pool_w=1)
    Qd = Q1.to(torch.float64).permute(0, 2, 1, 3)                     # [1][Hq][m][d]
    Kd = K1.to(torch.float64).expand(1, 2, 30, 16)
    eye = torch.eye(30, dtype=torch.float64).expand(1, 2, 30, 30)
    a = torch.nn.functional.scaled_dot_product_attention(Qd, Kd, eye, scale=0.25).numpy()   # [1][2][4][30]
    bb = a[0].mean(axis=0)                                              # [m][T]: mean over the group's heads
    assert _rel(r1["C"], bb.max(axis=0) / bb.mean(axis=0)) < 1e-12
    # (iv) one query token
    assert np.allclose(o.score(K, Q[:, :1].contiguous(), p=inf)["C"], 1.0, rtol=1e-13, atol=0)


def pin_self_keys(o):
    """The query tokens' own keys in the softmax (the causal prefix of a real forward pass): the
    sender attention equals torch's SDPA over [sender keys, query keys] with query token r
    allowed the query keys 0..r, and the scores equal the numpy restatement."""
    nL, Hq, Hkv, d, T, m = 2, 8, 2, 16, 37, 5
    K, _, Q = _rand_case(nL, Hq, Hkv, d, T, m, seed=41)
    Ks = synth.normal_bf16_shaped((nL, m, Hkv, d), synth.stream_key(41, 99))
    a = o.attention(K, Q, Kself=Ks)
    G = Hq // Hkv
    Kall = torch.cat([K.to(torch.float64), Ks.to(torch.float64).permute(0, 2, 1, 3)], dim=2)   # [nL][Hkv][T+m][d]
    Kall = Kall.repeat_interleave(G, dim=1)                                                   # [nL][Hq][T+m][d]
    Qd = Q.to(torch.float64).permute(0, 2, 1, 3)                                              # [nL][Hq][m][d]
    mask = torch.ones(m, T + m, dtype=torch.bool)
    mask[:, T:] = torch.tril(torch.ones(m, m, dtype=torch.bool))
    eye = torch.eye(T + m, dtype=torch.float64).expand(nL, Hq, T + m, T + m)
    ref = torch.nn.functional.scaled_dot_product_attention(Qd, Kall, eye, attn_mask=mask, scale=d ** -0.5)
    assert _rel(a, ref[..., :T].numpy()) < 1e-12
    assert np.all(a.sum(axis=-1) < 1.0)                  # part of every row's mass is on query keys
    r = o.score(K, Q, Kself=Ks)
    b = brute.score(_bits(K), _bits(Q), Ksbits=_bits(Ks))
    for k in ("S", "Q", "C", "U", "N", "D"):
        assert _rel(r[k], b[k]) < 1e-12, (k, _rel(r[k], b[k]))


# --------------------------------------------------------------------------
# selection (App. C.2)
# --------------------------------------------------------------------------

def _expand(spec, T):
    if spec == "ramp":
        return np.arange(T, dtype=np.float64)
    if isinstance(spec, str):
        out = []
        for part in spec.split(","):
            if ".." in part:
                a, b = part.split("..")
                out.extend(range(int(a), int(b) + 1))
            else:
                out.append(int(part))
        return out
    return spec


def pin_select_golden(o):
    with open(os.path.join(GOLDEN, "select_cases.json")) as f:
        cases = json.load(f)["cases"]
    for c in cases:
        T = c["T"]
        S = np.asarray(_expand(c["S"], T), dtype=np.float64)
        want = _expand(c["expected"], T)
        for arr in (S, S.astype(np.float32)):
            got = o.select(arr, c["B"], n_sink=c["n_sink"], n_latent=c["n_latent"], span_w=c["span_w"])
            assert got.tolist() == list(want), (c["name"], got.tolist(), want)


def pin_select_integrity(o):
    rng = np.random.default_rng(17)
    for T in (41, 42, 100, 257, 1000):
        S = rng.random(T)
        for keep in (0.05, 0.25, 0.5, 1.0):
            B = max(41, math.ceil(keep * T)) if T >= 41 else T
            B = min(B, T)
            idx = o.select(S, B)
            assert len(idx) == B
            assert np.all(np.diff(idx) > 0)
            forced = {0} | set(range(T - 40, T))
            assert forced <= set(idx.tolist())
    # budget below the forced count is rejected
    try:
        o.select(np.ones(100), 40)
    except ValueError:
        pass
    else:
        raise AssertionError("budget below the forced positions accepted")


def pin_compact(o):
    K, V, _ = _rand_case(2, 4, 2, 32, 50, 2, seed=4)
    idx = np.array([0, 3, 4, 17, 49], dtype=np.int32)
    off = 3
    ko, vo = o.compact(K, V, idx, offset=off)
    Kb, Vb = _bits(K), _bits(V)
    assert np.array_equal(ko[:, :, off:], Kb[:, :, idx]) and np.array_equal(vo[:, :, off:], Vb[:, :, idx])
    assert not ko[:, :, :off].any() and not vo[:, :, :off].any()


def _rope_ref(x, pos, base, style):
    """Textbook rotary embedding of x [..., d] at integer positions pos [...] (float64 torch)."""
    d = x.shape[-1]
    theta = base ** (-2.0 * torch.arange(d // 2, dtype=torch.float64) / d)
    ang = pos.to(torch.float64)[..., None] * theta
    c, s = torch.cos(ang), torch.sin(ang)
    if style == 0:                                        # rotate_half: pairs (k, k + d/2)
        x1, x2 = x[..., : d // 2], x[..., d // 2:]
        return torch.cat([x1 * c - x2 * s, x2 * c + x1 * s], dim=-1)
    xe, xo = x[..., 0::2], x[..., 1::2]                   # interleaved pairs (2k, 2k + 1)
    out = torch.empty_like(x)
    out[..., 0::2] = xe * c - xo * s
    out[..., 1::2] = xo * c + xe * s
    return out


def pin_compact_rope(o):
    """K moved from sender positions to receiver positions: equals the textbook rotary embedding
    applied at the new positions to the raw keys (within the two bf16 roundings), is the identity
    when the positions agree, keeps V unchanged."""
    nL, Hkv, T, d, base = 2, 2, 90, 32, 10000.0
    g = torch.Generator().manual_seed(8)
    raw = torch.randn(nL, Hkv, T, d, generator=g, dtype=torch.float64)
    pos = torch.arange(T)
    V = torch.randn(nL, Hkv, T, d, generator=g).to(torch.bfloat16)
    idx = np.array([0, 5, 6, 30, 61, 89], dtype=np.int32)
    for style in (0, 1):
        K = _rope_ref(raw, pos.expand(nL, Hkv, T), base, style).to(torch.bfloat16)
        pos0, off = 1000, 3
        ko, vo = o.compact_rope(K, V, idx, base, style, pos0=pos0, offset=off)
        new_pos = torch.tensor(pos0 + off + np.arange(len(idx)))
        want = _rope_ref(raw[:, :, idx], new_pos.expand(nL, Hkv, len(idx)), base, style)
        got = torch.from_numpy(ko[:, :, off:].view(np.int16)).view(torch.bfloat16).to(torch.float64)
        err = (got - want).abs().max() / want.abs().max()
        assert err < 2e-2, (style, float(err))
        assert np.array_equal(vo[:, :, off:], _bits(V)[:, :, idx])
        # positions that agree: the identity, bit for bit
        ko0, _ = o.compact_rope(K, V, np.arange(5, 12, dtype=np.int32), base, style, pos0=5)
        assert np.array_equal(ko0, _bits(K)[:, :, 5:12])


def pin_gather(o):
    """Message rows (App. C.3) equal numpy fancy indexing, for hidden-state rows and token IDs."""
    rng = np.random.default_rng(4)
    rows = rng.integers(0, 1 << 16, size=(70, 48), dtype=np.uint16)
    ids = rng.integers(0, 150000, size=70, dtype=np.int32)
    idx = np.array([0, 3, 4, 17, 40, 41, 69], dtype=np.int32)
    assert np.array_equal(o.gather(rows, idx, offset=2)[2:], rows[idx])
    assert not o.gather(rows, idx, offset=2)[:2].any()
    assert np.array_equal(o.gather(ids, idx), ids[idx])


def pin_unpage(o):
    """Paged layout (App. F, vLLM block table): a hand-traced table, a single identity page,
    and a second layer / head reading the same table; a page entry outside the pool is refused."""
    # 1 layer, 1 KV head, d = 2, P = 2, 3 pages; element value = 100 * page + 10 * row + k
    pool = np.array([[[[[100 * p + 10 * r + k for k in range(2)]] for r in range(2)] for p in range(3)]],
                    dtype=np.uint16)                       # [1][3][2][1][2]
    got = o.unpage(pool, [2, 0, 1], 5)[0, 0]
    # positions 0..4 -> (page, row) = (2,0) (2,1) (0,0) (0,1) (1,0), traced by hand
    want = np.array([[200, 201], [210, 211], [0, 1], [10, 11], [100, 101]], dtype=np.uint16)
    assert np.array_equal(got, want), got
    # one page holding every position in order: the pool itself, rearranged to [l][g][t][k]
    rng = np.random.default_rng(6)
    one = rng.integers(0, 1 << 16, size=(2, 1, 7, 3, 4), dtype=np.uint16)
    assert np.array_equal(o.unpage(one, [0], 7), one[:, 0].transpose(0, 2, 1, 3))
    # two layers, two heads: layer 1 / head 1 of position 3 comes from page 0, row 1 (P = 2, pages [1, 0])
    big = rng.integers(0, 1 << 16, size=(2, 2, 2, 2, 4), dtype=np.uint16)
    u = o.unpage(big, [1, 0], 4)
    assert np.array_equal(u[1, 1, 3], big[1, 0, 1, 1]) and np.array_equal(u[0, 1, 0], big[0, 1, 0, 1])
    assert np.array_equal(u[1, 0, 2], big[1, 0, 0, 0]) and np.array_equal(u[0, 0, 1], big[0, 1, 1, 0])
    try:
        o.unpage(pool, [2, 3, 1], 5)
    except RuntimeError:
        pass
    else:
        raise AssertionError("a page entry outside the pool was accepted")


ALL_PINS = [
    pin_pool_one_hot, pin_pool_library, pin_attention_sdpa, pin_one_hot_closed_form,
    pin_zero_denominator, pin_variance_identity, pin_identical_keys, pin_invariants,
    pin_special_cases, pin_equivariance, pin_brute, pin_p_infinity, pin_self_keys, pin_select_golden,
    pin_select_integrity,
    pin_compact, pin_compact_rope, pin_gather, pin_unpage,
]
