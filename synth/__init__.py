"""Seeded synthetic workloads for the CacheBack score -> select -> compact path.

This module is shared by the CPU oracle's tests and the CUDA path's tests and
benchmark. It holds none of the method's arithmetic: it only draws inputs.

Every random value comes from one counter-based generator (splitmix64 over the
element index, mapped through a fixed table of standard-normal quantiles), so a
tensor generated on a GPU is bit-identical to the same tensor generated on the
CPU.  That lets the GPU tests draw large workloads on the device and regenerate
any sampled sender on the host for the oracle.

Shapes follow the paper's workloads (Sec. 2 notation: a sender holds T = H + G
positions, one K/V entry per layer per position; App. C.1: m query tokens, the
scored layers, query heads sharing KV heads):

  K, V : bf16 [nL][Hkv][T][d]   post-RoPE keys / values of one sender
  Q    : bf16 [nL][m][Hq][d]    post-RoPE query vectors of the receiver query

Relevance is planted as in the workload recipe: for each (layer, KV head) a
direction u = Q[l][r*][h*] / |.| * sqrt(d) is taken from a random query token r*
and a random query head h* of that group, and planted positions get
K <- beta * u + N(0, 1).  Planted spans are 16-aligned, disjoint, and avoid the
first span and the forced latent tail.
"""
from __future__ import annotations

import dataclasses
import math
from typing import List, Optional, Sequence

import numpy as np
import torch

# ---------------------------------------------------------------------------
# counter-based generator
# ---------------------------------------------------------------------------

_M64 = (1 << 64) - 1


def _s64(x: int) -> int:
    """Two's-complement view of an unsigned 64-bit constant (torch int64)."""
    x &= _M64
    return x - (1 << 64) if x >= (1 << 63) else x


_GAMMA = _s64(0x9E3779B97F4A7C15)
_MUL1 = _s64(0xBF58476D1CE4E5B9)
_MUL2 = _s64(0x94D049BB133111EB)


def _srl(x: torch.Tensor, k: int) -> torch.Tensor:
    """Logical right shift of int64 tensors (torch's >> is arithmetic)."""
    return (x >> k) & ((1 << (64 - k)) - 1)


def _mix64(z: torch.Tensor) -> torch.Tensor:
    """splitmix64 output function (Steele, Lea, Flood 2014), wrapping int64."""
    z = (z ^ _srl(z, 30)) * _MUL1
    z = (z ^ _srl(z, 27)) * _MUL2
    return z ^ _srl(z, 31)


def _mix64_int(x: int) -> int:
    z = x & _M64
    z = ((z ^ (z >> 30)) * 0xBF58476D1CE4E5B9) & _M64
    z = ((z ^ (z >> 27)) * 0x94D049BB133111EB) & _M64
    return z ^ (z >> 31)


def stream_key(seed: int, *ids: int) -> int:
    """64-bit key of one random stream, derived from the seed and stream ids."""
    k = _mix64_int(0x5EED0000 + seed)
    for i in ids:
        k = _mix64_int(k ^ (0x9E3779B97F4A7C15 * (i + 1)))
    return k


_TABLE_CACHE = {}


def _normal_table(device) -> torch.Tensor:
    """65536 bf16 standard-normal quantiles Phi^-1((k + 1/2) / 65536)."""
    dev = torch.device(device)
    t = _TABLE_CACHE.get(str(dev))
    if t is None:
        from statistics import NormalDist
        nd = NormalDist()
        q = np.array([nd.inv_cdf((k + 0.5) / 65536.0) for k in range(65536)], dtype=np.float64)
        t = torch.from_numpy(q.astype(np.float32)).to(torch.bfloat16).to(dev)
        _TABLE_CACHE[str(dev)] = t
    return t


def normal_bf16(n: int, key: int, device="cpu", offset: int = 0) -> torch.Tensor:
    """n bf16 draws of N(0,1) (table-quantised), elements offset..offset+n-1 of stream `key`.

    Four values come from each 64-bit hash (16 bits each).  Identical on every
    device: only wrapping int64 arithmetic and a table gather are used.
    """
    if n == 0:
        return torch.empty(0, dtype=torch.bfloat16, device=device)
    table = _normal_table(device)
    first, last = offset // 4, (offset + n - 1) // 4
    cnt = torch.arange(first, last + 1, dtype=torch.int64, device=device)
    state = cnt * _GAMMA + _s64(key)
    h = _mix64(state)
    idx = torch.stack([_srl(h, 16 * c) & 0xFFFF for c in range(4)], dim=1).reshape(-1)
    vals = table[idx]
    start = offset - 4 * first
    return vals[start:start + n]


def normal_bf16_shaped(shape: Sequence[int], key: int, device="cpu", chunk: int = 1 << 26) -> torch.Tensor:
    n = int(np.prod(shape)) if len(shape) else 1
    out = torch.empty(n, dtype=torch.bfloat16, device=device)
    for off in range(0, n, chunk):
        c = min(chunk, n - off)
        out[off:off + c] = normal_bf16(c, key, device, offset=off)
    return out.view(*shape)


# ---------------------------------------------------------------------------
# workload descriptions
# ---------------------------------------------------------------------------

@dataclasses.dataclass(frozen=True)
class Shape:
    n_layers: int      # |L|, scored (global-attention) layers only
    n_q_heads: int     # Hq
    n_kv_heads: int    # Hkv
    head_dim: int      # d


@dataclasses.dataclass(frozen=True)
class WorkloadSpec:
    name: str
    shape: Shape
    T: tuple           # positions per sender
    m: int             # receiver query tokens
    keeps: tuple       # keep ratios (budget = ceil(keep * T))
    senders_per_task: int
    n_tasks: int
    planting: str      # "spans" (fixed beta) or "zipf"
    planted_frac: float = 0.0     # fraction of positions planted (spans mode)
    n_planted_spans: int = 0      # explicit span count (overrides planted_frac)
    beta: float = 0.5
    zipf_s: float = 1.1
    n_latent: int = 40
    span_width: int = 16
    shared_sender: bool = False   # every (sender, query) pair holds sender state 0 (multi-query serving)

    @property
    def n_senders(self) -> int:
        return self.n_tasks * self.senders_per_task


QWEN3_8B = Shape(36, 32, 8, 128)

SPECS = {
    # 2 layers, 4/2 heads, d=64, T=512, m=16, 3 planted spans of 16, keep 25%
    "tiny": WorkloadSpec("tiny", Shape(2, 4, 2, 64), (512,), 16, (0.25,), 1, 1,
                         "spans", n_planted_spans=3, beta=0.5),
    # Qwen3-8B-shaped single sender, T=8192, m=64, 5% of positions planted, keep 25%
    "qwen8b": WorkloadSpec("qwen8b", QWEN3_8B, (8192,), 64, (0.25,), 1, 1,
                           "spans", planted_frac=0.05, beta=0.5),
    # fan-in: 3 senders x 16384, one shared query of 128 tokens, keep 25% each
    "fanin": WorkloadSpec("fanin", QWEN3_8B, (16384, 16384, 16384), 128, (0.25,), 3, 1,
                          "spans", planted_frac=0.05, beta=0.5),
    # hybrid/long-context: 8 attention layers, T=65536, m=64, Zipf(1.1) over 64 spans, keep 10%
    "hybrid": WorkloadSpec("hybrid", Shape(8, 32, 8, 128), (65536,), 64, (0.10,), 1, 1,
                           "zipf", n_planted_spans=64, beta=1.0, zipf_s=1.1),
    # concurrency sweep: 16 tasks x 3 senders x 8192, per-task query of 64 tokens
    "sweep": WorkloadSpec("sweep", QWEN3_8B, (8192,) * 3, 64, (0.10, 0.25, 0.50), 3, 16,
                          "spans", planted_frac=0.05, beta=0.5),
    # multi-query serving: one Qwen3-8B-shaped sender state (T=8192) scored against 8 receiver
    # queries of 64 tokens in one launch, keep 25% per query
    "multiquery": WorkloadSpec("multiquery", QWEN3_8B, (8192,), 64, (0.25,), 1, 8,
                               "spans", planted_frac=0.05, beta=0.5, shared_sender=True),
}


@dataclasses.dataclass
class Sender:
    K: torch.Tensor            # bf16 [nL][Hkv][T][d]
    V: torch.Tensor            # bf16 [nL][Hkv][T][d]
    task: int                  # index of the query this sender is scored against
    planted_spans: List[int]   # span indices (16-aligned) that carry planted keys
    planted_beta: List[float]

    @property
    def T(self) -> int:
        return self.K.shape[2]


@dataclasses.dataclass
class Workload:
    spec: WorkloadSpec
    seed: int
    queries: List[torch.Tensor]   # bf16 [nL][m][Hq][d], one per task
    senders: List[Sender]

    def budgets(self, keep: float) -> List[int]:
        # ceil(keep*T) in double (App. C.2, B_i = ceil(T_i / r) with keep = 1/r)
        return [min(s.T, max(0, math.ceil(keep * s.T))) for s in self.senders]


def _planted(spec: WorkloadSpec, T: int, rng: np.random.Generator):
    w = spec.span_width
    n_spans_total = T // w
    # candidate spans: not the first span, not touching the forced latent tail
    last_ok = (T - spec.n_latent) // w  # spans [j*w, j*w+w) with j < last_ok end before the tail
    cands = np.arange(1, max(1, last_ok))
    if spec.planting == "zipf" or spec.n_planted_spans:
        k = spec.n_planted_spans
    else:
        k = int(round(spec.planted_frac * T / w))
    k = min(k, len(cands))
    chosen = np.sort(rng.choice(cands, size=k, replace=False)) if k else np.array([], dtype=np.int64)
    if spec.planting == "zipf":
        # heavy-tailed strengths beta_j = beta * rank^-s over a random rank order
        ranks = rng.permutation(k) + 1
        betas = [spec.beta * float(rk) ** (-spec.zipf_s) for rk in ranks]
    else:
        betas = [spec.beta] * k
    del n_spans_total
    return [int(j) for j in chosen], betas


def make_query(spec: WorkloadSpec, seed: int, task: int, device="cpu") -> torch.Tensor:
    s = spec.shape
    key = stream_key(seed, 1, task)
    return normal_bf16_shaped((s.n_layers, spec.m, s.n_q_heads, s.head_dim), key, device)


def make_query_keys(spec: WorkloadSpec, seed: int, task: int, device="cpu") -> torch.Tensor:
    """The receiver query tokens' own post-RoPE keys, bf16 [nL][m][Hkv][d], N(0,1)."""
    s = spec.shape
    key = stream_key(seed, 7, task)          # a stream of its own (K and V use ids 2 and 3)
    return normal_bf16_shaped((s.n_layers, spec.m, s.n_kv_heads, s.head_dim), key, device)


def _directions(spec: WorkloadSpec, Qcpu: torch.Tensor, rng: np.random.Generator) -> torch.Tensor:
    """Per-(layer, KV head) unit-RMS direction taken from one query row (fp32, CPU)."""
    s = spec.shape
    G = s.n_q_heads // s.n_kv_heads
    out = torch.empty(s.n_layers, s.n_kv_heads, s.head_dim, dtype=torch.float32)
    for l in range(s.n_layers):
        for g in range(s.n_kv_heads):
            r = int(rng.integers(spec.m))
            h = g * G + int(rng.integers(G))
            q = Qcpu[l, r, h].to(torch.float32)
            nrm = float(torch.linalg.vector_norm(q.double()))
            out[l, g] = (q.double() / nrm * math.sqrt(s.head_dim)).to(torch.float32)
    return out


def make_sender(spec: WorkloadSpec, seed: int, index: int, Qcpu: Optional[torch.Tensor] = None,
                device="cpu") -> Sender:
    """Sender `index` of the workload, generated directly on `device`."""
    s = spec.shape
    T = spec.T[index % len(spec.T)]
    task = index // spec.senders_per_task
    if Qcpu is None:
        Qcpu = make_query(spec, seed, task, "cpu")
    rng = np.random.default_rng([seed, 7, index])
    spans, betas = _planted(spec, T, rng)
    dirs = _directions(spec, Qcpu, rng)
    shp = (s.n_layers, s.n_kv_heads, T, s.head_dim)
    K = normal_bf16_shaped(shp, stream_key(seed, 2, index), device)
    V = normal_bf16_shaped(shp, stream_key(seed, 3, index), device)
    w = spec.span_width
    if spans:
        for j, beta in zip(spans, betas):
            # beta*u formed on the host in fp32, the add on the device: both IEEE-exact steps
            bu = (dirs * torch.tensor(beta, dtype=torch.float32)).unsqueeze(2).to(device)
            seg = K[:, :, j * w:(j + 1) * w, :]
            K[:, :, j * w:(j + 1) * w, :] = (seg.to(torch.float32) + bu).to(torch.bfloat16)
    return Sender(K=K, V=V, task=task, planted_spans=spans, planted_beta=betas)


def make_workload(name: str, seed: int = 0, device="cpu", senders: Optional[Sequence[int]] = None) -> Workload:
    spec = SPECS[name]
    ids = list(range(spec.n_senders)) if senders is None else list(senders)
    return _assemble(spec, seed, device, ids)


def _assemble(spec: WorkloadSpec, seed: int, device, ids: Sequence[int]) -> Workload:
    tasks = sorted({i // spec.senders_per_task for i in ids})
    qcpu = {t: make_query(spec, seed, t, "cpu") for t in tasks}
    queries = {t: qcpu[t].to(device) for t in tasks}
    out = []
    if spec.shared_sender:
        # one sender state (planted toward task 0's query); pair i scores it against task i's query
        base = make_sender(spec, seed, 0, make_query(spec, seed, 0, "cpu"), device)
        for i in ids:
            out.append(Sender(K=base.K, V=base.V, task=i // spec.senders_per_task,
                              planted_spans=base.planted_spans, planted_beta=base.planted_beta))
    else:
        for i in ids:
            out.append(make_sender(spec, seed, i, qcpu[i // spec.senders_per_task], device))
    # re-map task ids to positions in the returned query list
    order = {t: k for k, t in enumerate(tasks)}
    for snd in out:
        snd.task = order[snd.task]
    return Workload(spec=spec, seed=seed, queries=[queries[t] for t in tasks], senders=out)


def custom_workload(shape: Shape, Ts: Sequence[int], m: int, seed: int = 0, device="cpu",
                    n_planted_spans: int = 2, beta: float = 0.5, n_latent: int = 40,
                    shared_query: bool = True, name: str = "custom") -> Workload:
    """Same recipe at arbitrary sizes (parity cases with ragged T, odd m, ...)."""
    spec = WorkloadSpec(name, shape, tuple(Ts), m, (0.25,), len(Ts) if shared_query else 1,
                        1 if shared_query else len(Ts), "spans",
                        n_planted_spans=n_planted_spans, beta=beta, n_latent=n_latent)
    return make_workload_from_spec(spec, seed, device)


def make_workload_from_spec(spec: WorkloadSpec, seed: int = 0, device="cpu") -> Workload:
    return _assemble(spec, seed, device, list(range(spec.n_senders)))
