"""Literal numpy restatement of App. C.1 / C.2 for tiny inputs (T <= a few hundred).

TEST INFRASTRUCTURE.  A second, independently structured oracle: it builds the
full attention tensor a[l][h][r][t] with one einsum over explicitly repeated
KV heads, pools with an explicit window max, and selects with Python sorting.
Used only to cross-check the C oracle on tiny inputs.
"""
from __future__ import annotations

import math

import numpy as np


def bf16_bits_to_f64(bits: np.ndarray) -> np.ndarray:
    return (bits.astype(np.uint32) << 16).view(np.float32).astype(np.float64)


def pool(x: np.ndarray, w: int = 7) -> np.ndarray:
    """Pool_w over the last axis: max of the w positions centred on t, clipped."""
    T = x.shape[-1]
    half = w // 2
    out = np.empty_like(x)
    for t in range(T):
        lo, hi = max(0, t - half), min(T, t + half + 1)
        out[..., t] = x[..., lo:hi].max(axis=-1)
    return out


def attention(Kd: np.ndarray, Qd: np.ndarray, scale: float, Ksd=None) -> np.ndarray:
    """a[l][h][r][t] with query head h reading KV head h // G.  Ksd [nL][m][Hkv][d]: the query
    tokens' own keys, appended to every row's softmax with a causal mask (token r sees 0..r);
    only the sender columns are returned."""
    nL, Hkv, T, d = Kd.shape
    _, m, Hq, _ = Qd.shape
    G = Hq // Hkv
    Krep = np.repeat(Kd, G, axis=1)                      # [nL][Hq][T][d]
    z = np.einsum("lrhd,lhtd->lhrt", Qd, Krep) * scale   # [nL][Hq][m][T]
    if Ksd is not None:
        Ksrep = np.repeat(Ksd, G, axis=2)                # [nL][m][Hq][d]
        zs = np.einsum("lrhd,luhd->lhru", Qd, Ksrep) * scale   # [nL][Hq][m][m]
        causal = np.tril(np.ones((m, m), dtype=bool))
        zs = np.where(causal, zs, -np.inf)
        z = np.concatenate([z, zs], axis=-1)
    z = z - z.max(axis=-1, keepdims=True)
    e = np.exp(z)
    return (e / e.sum(axis=-1, keepdims=True))[..., :T]


def score(Kbits, Qbits, p=2.0, alpha=2.0, pool_w=7, scale=None, Ksbits=None) -> dict:
    Kd, Qd = bf16_bits_to_f64(Kbits), bf16_bits_to_f64(Qbits)
    nL, Hkv, T, d = Kd.shape
    _, m, Hq, _ = Qd.shape
    G = Hq // Hkv
    if scale is None:
        scale = 1.0 / math.sqrt(d)
    a = attention(Kd, Qd, scale, None if Ksbits is None else bf16_bits_to_f64(Ksbits))
    # mean query attention: sum over layers of the (r, h)-average, then Pool
    U = a.mean(axis=(1, 2)).sum(axis=0)                  # [T]
    Qt = pool(U, pool_w)
    # KV-group means b[l][g][r][t]
    b = a.reshape(nL, Hkv, G, m, T).mean(axis=2)
    if math.isinf(p):
        # the p -> infinity limit (App. D.2): largest pooled token attention over the largest
        # pooled token mean, over all groups
        num = pool(b, pool_w).max(axis=(0, 1, 2))
        den = pool(b.mean(axis=2), pool_w).max(axis=(0, 1))
        expo = 1.0
    else:
        num = (pool(b, pool_w) ** p).mean(axis=2).sum(axis=(0, 1))
        den = (pool(b.mean(axis=2), pool_w) ** p).sum(axis=(0, 1))
        expo = 1.0 / (p - 1.0)
    with np.errstate(divide="ignore", invalid="ignore"):
        C = np.where(den > 0, (num / np.where(den > 0, den, 1.0)) ** expo, 1.0)
    S = Qt * C ** alpha
    return {"S": S, "Q": Qt, "C": C, "U": U, "N": num, "D": den, "a": a, "b": b}


def select(S, B, n_sink=1, n_latent=40, span_w=16):
    """Span selection written with Python lists and sorted()."""
    S = [float(x) for x in S]
    T = len(S)
    forced = set(range(min(n_sink, T))) | set(range(max(0, T - n_latent), T))
    if B < len(forced) or B > T:
        raise ValueError("budget below the forced positions or above T")
    Sp = list(S)
    if n_sink > 0:
        Sp[0] = max(S)
    spans = [list(range(j, min(T, j + span_w))) for j in range(0, T, span_w)]
    means = [sum(Sp[t] for t in sp) / len(sp) for sp in spans]
    order = sorted(range(len(spans)), key=lambda j: (-means[j], j))
    chosen = set(forced)
    for j in order:
        if len(chosen) == B:
            break
        u = [t for t in spans[j] if t not in chosen]
        if not u:
            continue
        if len(chosen) + len(u) <= B:
            chosen.update(u)
        else:
            best = max(Sp[t] for t in u)
            c = min(t for t in u if Sp[t] == best)
            need = B - len(chosen)
            chosen.update(sorted(u, key=lambda t: (abs(t - c), t))[:need])
    return np.array(sorted(chosen), dtype=np.int32)
