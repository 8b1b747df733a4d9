"""Seeded synthetic inputs for the GraceKV compression pass.

This module only draws random numbers and arranges them into the shapes the
compression pass consumes: post-RoPE keys K and values V of shape
[L, G, T, d], observation-window queries Q of shape [L, Hq, W, d], and (for
the skewed stress workload) externally supplied slot boundaries.  It holds
none of the compression method's arithmetic; both the CUDA path and the CPU
oracle consume its tensors verbatim.

Recipe (one per workload, all seeded):

* Segment structure shared by every (layer, KV head): consecutive token
  segments whose lengths are either 8 draws from U{64..256} rescaled to sum
  to T (largest-remainder rounding), or lognormal(ln 200, 0.5) draws clamped
  to [16, 2000] until T is covered (the last one truncated).
* For every (l, g, X in {K, V}) an independent sub-stream: segment means
  follow a stationary AR(1) walk mu_0 ~ N(0, I), mu_s = 0.8 mu_{s-1} +
  0.6 xi_s; each token is x_t = (mu_{s(t)} + eps_t) / sqrt(2), so every
  channel keeps an N(0, 1) marginal; a few outlier channels (drawn without
  replacement) are scaled up.
* Keys are then rotated the way a RoPE model's forward pass rotates them
  (half-split pairs, theta_i = base^(-2i/d), angle t * theta_i), which makes
  them post-RoPE keys; values are not rotated.  This is input synthesis of a
  model's cache, not a step of the compression method.
* Queries are iid N(0, 1).
* The skewed workload additionally plants three 512-token regions whose keys
  point along a per-(l, g) direction c_r, and aims each query at one region
  (query u at region u mod 3), giving cosine about 0.9 between a query and
  the keys of its region.  Its slot boundaries are drawn, not segmented:
  length 1 with p = 0.01, U{4097..8192} with p = 0.01, else U{16..128}.

Decoding inputs (make_decode_cache) stand in for a packed compressed cache
at compression ratio x: L G T / x entries split over the (l, g) by
lognormal(0, 0.35) shares (largest remainder, at least 32 each); within an
(l, g) the last 32 entries are a recent window of single tokens, and every
other entry is a single token with p = 0.3, else a prototype of n = 2^U(1, 7)
tokens with coherence c ~ U(0.35, 1): log m = log clamp(n c, 1, n), key
N(0, c) per channel, value N(0, 1) times U(0.3, 1).  Single tokens carry
N(0, 1) keys and values and log m = 0.  Decode queries are N(0, 1) per
channel, every other query head scaled by 3 (sharper softmax).  Appended
rows are N(0, 1).  These are draws, not the compression's arithmetic.

Every tensor is produced on the requested device with a torch.Generator
seeded from numpy's SeedSequence(seed, spawn_key=(...)), so a slice (a subset
of layers / heads) regenerates independently of the rest.  CPU and CUDA
generators give different (equally valid) draws; a test always feeds the
same tensors to both sides.
"""
from __future__ import annotations

import dataclasses
import math
from typing import Optional, Sequence

import numpy as np
import torch

__all__ = ["Workload", "WORKLOADS", "Inputs", "make_inputs", "segment_lengths",
           "supplied_slots", "DecodeCache", "make_decode_cache", "make_graph_queries"]


@dataclasses.dataclass(frozen=True)
class Workload:
    name: str
    L: int
    G: int
    Hq: int
    d: int
    T: int
    W: int
    dtype: str            # "f32" or "bf16"
    seg_mode: str         # "uniform8" or "lognormal"
    n_outlier: int
    outlier_scale: float
    rope_base: float
    ratios: tuple
    seed: int
    skew: bool = False


WORKLOADS = {
    # 1 layer, 2 KV heads (no GQA), d=128, T=1024, fp32, 8 segments.
    "pr1": Workload("pr1", 1, 2, 2, 128, 1024, 32, "f32", "uniform8", 4, 8.0,
                    1.0e4, (8,), 0),
    # 16 layers, 8 KV heads, 32 query heads, d=64, T=8192, bf16.
    "small": Workload("small", 16, 8, 32, 64, 8192, 64, "bf16", "lognormal", 4,
                      8.0, 1.0e4, (8, 16, 32), 1),
    # Llama-3-8B shape at 32K and 128K context.
    "llama32k": Workload("llama32k", 32, 8, 32, 128, 32768, 64, "bf16",
                         "lognormal", 3, 10.0, 5.0e5, (32,), 2),
    "llama128k": Workload("llama128k", 32, 8, 32, 128, 131072, 64, "bf16",
                          "lognormal", 3, 10.0, 5.0e5, (32, 128), 3),
    # Skewed-importance stress, externally supplied slots.
    "skew": Workload("skew", 32, 8, 32, 128, 65536, 64, "bf16", "lognormal", 3,
                     10.0, 5.0e5, (4, 8, 16, 32, 64, 128), 4, skew=True),
}


@dataclasses.dataclass
class Inputs:
    K: torch.Tensor           # [L', G', T, d] post-RoPE keys
    V: torch.Tensor           # [L', G', T, d]
    Q: torch.Tensor           # [L', Hq', W, d]
    seg_lengths: np.ndarray   # generator segment lengths (shared)
    slots: Optional[np.ndarray] = None   # supplied slot starts (skew only)
    layers: tuple = ()
    heads: tuple = ()


def _stream(seed: int, *key: int, device="cpu") -> torch.Generator:
    ss = np.random.SeedSequence(seed, spawn_key=tuple(int(k) for k in key))
    g = torch.Generator(device=device)
    g.manual_seed(int(ss.generate_state(1, dtype=np.uint64)[0] & ((1 << 63) - 1)))
    return g


def _np_stream(seed: int, *key: int) -> np.random.Generator:
    return np.random.Generator(np.random.PCG64(
        np.random.SeedSequence(seed, spawn_key=tuple(int(k) for k in key))))


def segment_lengths(w: Workload, T: Optional[int] = None) -> np.ndarray:
    """Generator segment lengths (shared by all layers and heads)."""
    T = w.T if T is None else T
    rng = _np_stream(w.seed, 1_000_001)
    if w.seg_mode == "uniform8":
        raw = rng.integers(64, 257, size=8).astype(np.float64)
        exact = raw * T / raw.sum()
        base = np.floor(exact).astype(np.int64)
        rem = T - int(base.sum())
        order = np.argsort(-(exact - base), kind="stable")
        base[order[:rem]] += 1
        return base
    lens = []
    tot = 0
    while tot < T:
        n = int(np.clip(np.rint(rng.lognormal(math.log(200.0), 0.5)), 16, 2000))
        n = min(n, T - tot)
        lens.append(n)
        tot += n
    return np.asarray(lens, dtype=np.int64)


def supplied_slots(w: Workload, N: int) -> np.ndarray:
    """Slot starts (len J+1, last = N) drawn for the skewed workload."""
    rng = _np_stream(w.seed, 1_000_002)
    starts = [0]
    pos = 0
    while pos < N:
        u = rng.random()
        if u < 0.01:
            n = 1
        elif u < 0.02:
            n = int(rng.integers(4097, 8193))
        else:
            n = int(rng.integers(16, 129))
        pos = min(N, pos + n)
        starts.append(pos)
    return np.asarray(starts, dtype=np.int32)


def _rotate_like_rope_model(x: torch.Tensor, base: float) -> torch.Tensor:
    """Forward RoPE a model applies to keys at positions 0..T-1 (input synthesis)."""
    T, d = x.shape[-2], x.shape[-1]
    half = d // 2
    i = torch.arange(half, dtype=torch.float64, device=x.device)
    inv = torch.pow(torch.tensor(base, dtype=torch.float64, device=x.device), -2.0 * i / d)
    ang = torch.arange(T, dtype=torch.float64, device=x.device)[:, None] * inv[None, :]
    c, s = torch.cos(ang), torch.sin(ang)
    x = x.to(torch.float64)
    a, b = x[..., :half], x[..., half:]
    return torch.cat([a * c - b * s, a * s + b * c], dim=-1)


def _stream_tokens(w: Workload, seg_id: torch.Tensor, n_seg: int, l: int, g: int,
                   which: int, T: int, device) -> torch.Tensor:
    gen = _stream(w.seed, l, g, which, device=device)
    d = w.d
    xi = torch.randn(n_seg, d, generator=gen, device=device, dtype=torch.float64).cpu().numpy()
    mu = np.empty_like(xi)
    mu[0] = xi[0]
    for s in range(1, n_seg):
        mu[s] = 0.8 * mu[s - 1] + 0.6 * xi[s]
    mu = torch.from_numpy(mu).to(device)
    eps = torch.randn(T, d, generator=gen, device=device, dtype=torch.float64)
    x = (mu[seg_id] + eps) / math.sqrt(2.0)
    perm = torch.randperm(d, generator=gen, device=device)[: w.n_outlier]
    x[:, perm] *= w.outlier_scale
    return x


def make_inputs(w: Workload, device="cpu", layers: Optional[Sequence[int]] = None,
                heads: Optional[Sequence[int]] = None, T: Optional[int] = None,
                W: Optional[int] = None) -> Inputs:
    """Build the seeded inputs of workload ``w`` (optionally a layer/head slice).

    ``layers`` / ``heads`` select KV heads; query heads of the selected KV
    heads are kept.  ``T`` / ``W`` shrink the sequence / probe count (the
    segment structure is regenerated for the new T with the same seed).
    """
    T = w.T if T is None else int(T)
    W = w.W if W is None else int(W)
    layers = tuple(range(w.L)) if layers is None else tuple(int(x) for x in layers)
    heads = tuple(range(w.G)) if heads is None else tuple(int(x) for x in heads)
    lens = segment_lengths(w, T)
    seg_id = torch.repeat_interleave(torch.arange(len(lens), device=device),
                                     torch.as_tensor(lens, device=device))
    gq = w.Hq // w.G
    tdt = torch.float32 if w.dtype == "f32" else torch.bfloat16
    K = torch.empty(len(layers), len(heads), T, w.d, dtype=tdt, device=device)
    V = torch.empty_like(K)
    Q = torch.empty(len(layers), len(heads) * gq, W, w.d, dtype=tdt, device=device)
    regions = None
    if w.skew:
        rr = _np_stream(w.seed, 1_000_003)
        # three non-overlapping 512-token regions inside [0, T - 32)
        span = T - 32 - 3 * 512
        cuts = np.sort(rr.choice(span + 1, size=3, replace=True))
        regions = [int(cuts[k]) + 512 * k for k in range(3)]
    for li, l in enumerate(layers):
        for gi, g in enumerate(heads):
            kx = _rotate_like_rope_model(
                _stream_tokens(w, seg_id, len(lens), l, g, 0, T, device), w.rope_base)
            V[li, gi] = _stream_tokens(w, seg_id, len(lens), l, g, 1, T, device).to(tdt)
            cdir = None
            if regions is not None:
                gen = _stream(w.seed, l, g, 3, device=device)
                cdir = torch.randn(3, w.d, generator=gen, device=device, dtype=torch.float64)
                cdir /= cdir.norm(dim=-1, keepdim=True)
                for r, off in enumerate(regions):
                    e = torch.randn(512, w.d, generator=gen, device=device, dtype=torch.float64)
                    e /= e.norm(dim=-1, keepdim=True)
                    kx[off:off + 512] = math.sqrt(w.d) * (0.95 * cdir[r] + 0.312 * e)
            K[li, gi] = kx.to(tdt)
            for hh in range(gq):
                h = g * gq + hh
                gen = _stream(w.seed, l, h, 2, device=device)
                q = torch.randn(W, w.d, generator=gen, device=device, dtype=torch.float64)
                if cdir is not None:
                    nu = q / q.norm(dim=-1, keepdim=True)
                    q = math.sqrt(w.d) * (0.95 * cdir[torch.arange(W, device=device) % 3] + 0.312 * nu)
                Q[li, gi * gq + hh] = q.to(tdt)
    slots = None
    if w.skew:
        slots = supplied_slots(w, T - 32)
    return Inputs(K, V, Q, lens, slots, layers, heads)



@dataclasses.dataclass
class DecodeCache:
    q: torch.Tensor           # [L, Hq, d] decode queries (one step)
    K: torch.Tensor           # [E, d] packed keys
    V: torch.Tensor           # [E, d] packed values
    log_m: torch.Tensor       # [E] fp32
    offsets: torch.Tensor     # [L*G + 1] int64
    K_app: torch.Tensor       # [L, G, app_cap, d] appended keys
    V_app: torch.Tensor       # [L, G, app_cap, d]
    n_app: int


def decode_counts(L: int, G: int, E: int, seed: int) -> np.ndarray:
    """Entries per (l, g): lognormal(0, 0.35) shares of E, at least 32 each."""
    rng = _np_stream(seed, 2_000_001)
    w = rng.lognormal(0.0, 0.35, size=L * G)
    spare = E - 32 * L * G
    assert spare >= 0
    exact = w * spare / w.sum()
    base = np.floor(exact).astype(np.int64)
    order = np.argsort(-(exact - base), kind="stable")
    base[order[:spare - int(base.sum())]] += 1
    return base + 32


def make_decode_cache(w: Workload, ratio: int, n_app: int = 0, app_cap: Optional[int] = None,
                      device="cpu", counts: Optional[np.ndarray] = None,
                      seed: Optional[int] = None) -> DecodeCache:
    """Seeded packed cache + appended rows + one step of decode queries."""
    seed = w.seed if seed is None else seed
    L, G, Hq, d = w.L, w.G, w.Hq, w.d
    if counts is None:
        counts = decode_counts(L, G, L * G * w.T // ratio, seed)
    counts = np.asarray(counts, dtype=np.int64)
    E = int(counts.sum())
    off = np.zeros(L * G + 1, dtype=np.int64)
    off[1:] = np.cumsum(counts)
    rng = _np_stream(seed, 2_000_002)
    single = rng.random(E) < 0.3
    n = np.exp2(rng.uniform(1.0, 7.0, size=E))
    coh = rng.uniform(0.35, 1.0, size=E)
    vs = rng.uniform(0.3, 1.0, size=E)
    for lg in range(L * G):                       # recent window: single tokens
        single[max(off[lg + 1] - 32, off[lg]):off[lg + 1]] = True
    logm = np.where(single, 0.0, np.log(np.clip(n * coh, 1.0, n)))
    kscale = np.where(single, 1.0, np.sqrt(coh))
    vscale = np.where(single, 1.0, vs)
    tdt = torch.float32 if w.dtype == "f32" else torch.bfloat16
    gen = _stream(seed, 2_000_003, device=device)
    K = torch.randn(E, d, generator=gen, device=device)
    K *= torch.as_tensor(kscale, dtype=torch.float32, device=device)[:, None]
    V = torch.randn(E, d, generator=gen, device=device)
    V *= torch.as_tensor(vscale, dtype=torch.float32, device=device)[:, None]
    app_cap = max(n_app, 1) if app_cap is None else app_cap
    gen = _stream(seed, 2_000_004, device=device)
    Ka = torch.randn(L, G, app_cap, d, generator=gen, device=device)
    Va = torch.randn(L, G, app_cap, d, generator=gen, device=device)
    gen = _stream(seed, 2_000_005, device=device)
    q = torch.randn(L, Hq, d, generator=gen, device=device)
    q[:, 1::2] *= 3.0
    return DecodeCache(q.to(tdt), K.to(tdt), V.to(tdt),
                       torch.as_tensor(logm, dtype=torch.float32, device=device),
                       torch.as_tensor(off, device=device), Ka.to(tdt), Va.to(tdt), n_app)


def make_graph_queries(w: Workload, graph_layers: Sequence[int], T: Optional[int] = None,
                       device="cpu", heads: Optional[Sequence[int]] = None) -> torch.Tensor:
    """Queries of every position at the graph layers, [n_graph, Hq', T, d]:
    N(0, 1) per channel, rotated like the keys (the position's RoPE angle), so
    that a seed's attention over its past carries the keys' structure."""
    T = w.T if T is None else int(T)
    heads = tuple(range(w.Hq)) if heads is None else tuple(int(h) for h in heads)
    tdt = torch.float32 if w.dtype == "f32" else torch.bfloat16
    out = torch.empty(len(graph_layers), len(heads), T, w.d, dtype=tdt, device=device)
    for gi, l in enumerate(graph_layers):
        for hi, h in enumerate(heads):
            gen = _stream(w.seed, 3_000_001, l, h, device=device)
            q = torch.randn(T, w.d, generator=gen, device=device, dtype=torch.float64)
            out[gi, hi] = _rotate_like_rope_model(q, w.rope_base).to(tdt)
    return out
