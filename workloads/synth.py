"""Seeded synthetic inputs for the TReVS pruning path.

This module only draws random tensors with the shapes and value distributions of
the paper's workloads (LLaVA-1.5 576-token images, LLaVA-NeXT 2,880-token
high-resolution images, 16,384-token multi-image/video inputs and a ragged
serving batch). It holds none of the method's arithmetic: scores, selections
and gathers live in the oracle and in the CUDA library, which both consume the
bytes produced here.

Layouts (rows packed over the requests of a batch, bf16 stored as uint16 bits):
  Z      [sum N, d]        projected visual features      (Sec. 4.1, Z = Projector(X_v))
  T      [sum M, d]        query text embeddings          (Sec. 4.1, t_j)
  s_v    [sum N] float32   [CLS]-attention saliency       (Eq. 3)
  Q      [sum L, Hq, dh]   text queries at layer l*       (Sec. 4.2)
  K, V   [sum K1, Hkv, dh] visual keys / values at l*     (Sec. 4.2)
  hidden [sum K1, d]       visual hidden states at l*     (Sec. 4.2)

Every request b of workload `cfg` draws from numpy PCG64 seeded with
1000 * cfg + b; the stage-2 tensors use an independent child stream so that the
sweep over the stage-1 keep size changes no stage-1 input.
"""
from __future__ import annotations

import dataclasses
import math

import numpy as np


def f32_to_bf16_bits(x: np.ndarray) -> np.ndarray:
    """Round float32 values to bfloat16 (round-to-nearest-even); return uint16 bits."""
    x = np.ascontiguousarray(x, dtype=np.float32)
    b = x.view(np.uint32)
    # finite inputs only: b + 0x7FFF + lsb cannot wrap below 0x7F800000
    return ((b + (np.uint32(0x7FFF) + ((b >> np.uint32(16)) & np.uint32(1)))) >> np.uint32(16)).astype(np.uint16)


@dataclasses.dataclass
class Request:
    n: int          # visual tokens N
    m: int          # query text tokens M (stage 1)
    k1: int         # pre-LLM keep K1
    ratio: float    # textual ratio r
    l: int          # text query rows at layer l* (stage 2)
    k2: int         # final keep K2


@dataclasses.dataclass
class Workload:
    name: str
    d: int                 # projected feature width d' (= LLM hidden width)
    hq: int                # query heads at l*
    hkv: int               # key/value heads at l*
    dh: int                # head width
    n_keep_heads: int      # |H*|
    reqs: list
    Z: np.ndarray
    T: np.ndarray
    s_v: np.ndarray
    Q: np.ndarray
    K: np.ndarray
    V: np.ndarray
    hidden: np.ndarray
    planted: list = dataclasses.field(default_factory=list)
    lse_other: np.ndarray | None = None   # [hq, sum L] float32: full-sequence softmax variant

    @property
    def B(self) -> int:
        return len(self.reqs)

    def offsets(self, field: str) -> np.ndarray:
        v = np.array([getattr(r, field) for r in self.reqs], dtype=np.int64)
        return np.concatenate([[0], np.cumsum(v)])

    def visual_tokens(self) -> int:
        return int(sum(r.n for r in self.reqs))


def _saliency(rng, n, sigma, spikes, tile):
    """[CLS] saliency stand-in: softmax of N(0, sigma^2) logits per ViT tile."""
    logits = rng.standard_normal(n) * sigma
    if spikes:
        pos = rng.choice(n, size=spikes, replace=False)
        logits[pos] += 8.0
    out = np.empty(n, dtype=np.float64)
    for s in range(0, n, tile):
        e = np.exp(logits[s:s + tile] - logits[s:s + tile].max())
        out[s:s + tile] = e / e.sum()
    return out.astype(np.float32)


def _planted_positions(rng, n, count, clusters):
    if count <= 0:
        return np.zeros(0, dtype=np.int64)
    if clusters <= 0:
        return np.sort(rng.choice(n, size=count, replace=False))
    per = [count // clusters + (1 if c < count % clusters else 0) for c in range(clusters)]
    seg = n // clusters
    pos = []
    for c, k in enumerate(per):
        start = c * seg + int(rng.integers(0, max(1, seg - k)))
        pos.extend(range(start, start + k))
    return np.array(sorted(pos), dtype=np.int64)


def _stage1(rng, n, m, d, planted_count, clusters, sal_sigma, spikes, tile):
    """Z ~ N(0,1) with planted query-correlated rows; T correlated with the query."""
    Z = rng.standard_normal((n, d), dtype=np.float32)
    u = rng.standard_normal(d)
    u /= np.linalg.norm(u)
    pos = _planted_positions(rng, n, planted_count, clusters)
    sd = math.sqrt(d)
    if len(pos):
        # cos(z_i, u) ~ 0.75 and cos(t_j, u) ~ 0.8, so cos(z_i, t_j) ~ 0.6
        Z[pos] = (0.75 * sd * u[None, :] + 0.66 * Z[pos]).astype(np.float32)
    T = (0.8 * sd * u[None, :] + 0.6 * rng.standard_normal((m, d))).astype(np.float32)
    s_v = _saliency(rng, n, sal_sigma, spikes, tile)
    return f32_to_bf16_bits(Z), f32_to_bf16_bits(T), s_v, pos


def _stage2(rng, k1, l, hq, hkv, dh, d_model):
    """Text queries with per-head logit scales U(0.5, 4); keys, values, hidden ~ N(0,1)."""
    scale = rng.uniform(0.5, 4.0, size=hq).astype(np.float32)
    Q = rng.standard_normal((l, hq, dh), dtype=np.float32) * scale[None, :, None]
    K = rng.standard_normal((k1, hkv, dh), dtype=np.float32)
    V = rng.standard_normal((k1, hkv, dh), dtype=np.float32)
    H = rng.standard_normal((k1, d_model), dtype=np.float32)
    return (f32_to_bf16_bits(Q), f32_to_bf16_bits(K), f32_to_bf16_bits(V),
            f32_to_bf16_bits(H))


def _assemble(name, cfg, d, hq, hkv, dh, n_keep_heads, reqs, planted_frac, clusters,
              sal_sigma, spikes, tile, planted_count=None):
    Zs, Ts, Ss, Qs, Ks, Vs, Hs, P = [], [], [], [], [], [], [], []
    for b, r in enumerate(reqs):
        rng = np.random.Generator(np.random.PCG64(1000 * cfg + b))
        rng2 = np.random.Generator(np.random.PCG64([1000 * cfg + b, 2]))
        pc = planted_count if planted_count is not None else int(round(planted_frac * r.n))
        Z, T, s_v, pos = _stage1(rng, r.n, r.m, d, pc, clusters, sal_sigma, spikes, tile)
        Q, K, V, H = _stage2(rng2, r.k1, r.l, hq, hkv, dh, d)
        Zs.append(Z); Ts.append(T); Ss.append(s_v); P.append(pos)
        Qs.append(Q); Ks.append(K); Vs.append(V); Hs.append(H)
    cat = lambda xs, shape: (np.concatenate(xs, axis=0) if xs else np.zeros(shape, np.uint16))
    return Workload(
        name=name, d=d, hq=hq, hkv=hkv, dh=dh, n_keep_heads=n_keep_heads, reqs=reqs,
        Z=cat(Zs, (0, d)), T=cat(Ts, (0, d)),
        s_v=np.concatenate(Ss).astype(np.float32) if Ss else np.zeros(0, np.float32),
        Q=cat(Qs, (0, hq, dh)), K=cat(Ks, (0, hkv, dh)), V=cat(Vs, (0, hkv, dh)),
        hidden=cat(Hs, (0, d)), planted=P)


def llava15_single(k1=64, ratio=0.5, k2=32):
    """576 visual tokens, d'=4096, 32 query tokens, 24 planted, 32x128 heads."""
    reqs = [Request(n=576, m=32, k1=k1, ratio=ratio, l=32, k2=k2)]
    return _assemble("llava15_576_single", 0, 4096, 32, 32, 128, 8, reqs, 0.0, 0,
                     2.0, 8, 576, planted_count=24)


def llava15_batch32(k1=64, ratio=0.5, k2=32, batch=32):
    """Config-0 generators over 32 requests, query lengths uniform in 16..64."""
    lens = np.random.Generator(np.random.PCG64(1000 * 1 + 999)).integers(16, 65, size=batch)
    reqs = [Request(n=576, m=int(m), k1=k1, ratio=ratio, l=int(m), k2=k2) for m in lens]
    return _assemble(f"llava15_576_b{batch}_k{k1}_r{ratio:g}_k{k2}", 1, 4096, 32, 32, 128, 8,
                     reqs, 0.0, 0, 2.0, 8, 576, planted_count=24)


def llava_next_batch8(batch=8):
    """2,880 tokens (5 tiles x 576), 5% planted, per-tile saliency, 64 query tokens."""
    reqs = [Request(n=2880, m=64, k1=320, ratio=0.5, l=64, k2=160) for _ in range(batch)]
    return _assemble("llava_next_2880_b8", 2, 4096, 32, 32, 128, 8, reqs, 0.05, 0,
                     2.0, 0, 576)


def long_video_batch2(batch=2):
    """16,384 tokens, d'=3584, GQA 28/4 heads, 2% planted in 16 clusters, 128 query tokens."""
    reqs = [Request(n=16384, m=128, k1=1024, ratio=0.5, l=128, k2=512) for _ in range(batch)]
    return _assemble("long_16384_b2_gqa", 3, 3584, 28, 4, 128, 7, reqs, 0.02, 16,
                     3.0, 0, 16384)


def video_llava_batch(batch=4):
    """Video-LLaVA-shaped: 8 frames x 256 tokens = 2,048 per video, saliency per frame, 3%
    planted in 8 clusters (one object across the frames), M ~ U{16..48}, d' = 4096 with
    32 x 128 heads and the top half kept. K1 = 272 and K2 = 91: with the second prune after
    layer 8 of 32, the LLM keeps (8 * 272 + 24 * 91) / 32 = 136.25 visual tokens per layer,
    the paper's 136 of 2,048 (K1 about 3 K2)."""
    lens = np.random.Generator(np.random.PCG64(1000 * 5 + 999)).integers(16, 49, size=batch)
    reqs = [Request(n=2048, m=int(m), k1=272, ratio=0.5, l=int(m), k2=91) for m in lens]
    return _assemble(f"video_llava_2048_b{batch}", 5, 4096, 32, 32, 128, 16, reqs, 0.03, 8,
                     2.0, 0, 256)


def ragged_serving_batch64(batch=64):
    """64 varlen requests, N in {576,1152,2880}, M log-uniform 8..256, keep 5.6% (min 32)."""
    g = np.random.Generator(np.random.PCG64(1000 * 4 + 999))
    ns = g.choice([576, 1152, 2880], size=batch)
    ms = np.exp(g.uniform(math.log(8), math.log(256), size=batch)).astype(np.int64)
    reqs = []
    for n, m in zip(ns, ms):
        k2 = max(32, int(n) // 18)
        reqs.append(Request(n=int(n), m=int(m), k1=3 * k2, ratio=0.5, l=int(m), k2=k2))
    return _assemble("ragged_varlen_b64", 4, 4096, 32, 32, 128, 8, reqs, 0.05, 0,
                     2.0, 0, 576)


def small_case(seed_cfg=90, n=(300, 77, 129), m=(5, 17, 1), d=200, hq=4, hkv=2, dh=128,
               n_keep_heads=2, k1=(40, 77, 3), ratio=(0.5, 0.25, 1.0), k2=(13, 20, 1),
               planted=0.1):
    """Small ragged batch for parity at sizes the oracle finishes instantly."""
    reqs = [Request(n=a, m=b, k1=c, ratio=r, l=b, k2=e)
            for a, b, c, r, e in zip(n, m, k1, ratio, k2)]
    return _assemble("small_ragged", seed_cfg, d, hq, hkv, dh, n_keep_heads, reqs, planted, 0,
                     2.0, 0, 64)


def cls_inputs(n, heads=16, dh=64, seed=77, spikes=8):
    """Inputs of Eq. 2-3 for requests of n[b] patches, as bf16 bits: the [CLS] query of every
    head, [B, heads, dh], and the patch keys of the penultimate ViT layer, [sum n, heads, dh].
    Queries carry per-head scales U(0.5, 2); in every request `spikes` patches get keys pushed
    along their head's query (the few patches [CLS] attends to). CLIP ViT-L/14 has 16 heads of
    width 64."""
    rng = np.random.Generator(np.random.PCG64(seed))
    B = len(n)
    q = rng.standard_normal((B, heads, dh)) * rng.uniform(0.5, 2.0, size=(B, heads, 1))
    K = rng.standard_normal((int(sum(n)), heads, dh))
    off = 0
    for b, nb in enumerate(n):
        if nb > 0 and spikes > 0:
            idx = rng.choice(nb, size=min(spikes, nb), replace=False)
            u = q[b] / np.linalg.norm(q[b], axis=1, keepdims=True)
            K[off + idx] += 4.0 * u[None, :, :]
        off += nb
    return f32_to_bf16_bits(q.astype(np.float32)), f32_to_bf16_bits(K.astype(np.float32))


def with_full_sequence_softmax(w, seed=7, system_tokens=35):
    """A copy of `w` with lse_other [hq, sum L] (float32): for text row q of a request, the log
    of the summed exp-logits of the keys a causal LLM row also attends to besides the visual
    ones (`system_tokens` system-prompt keys and the text keys up to q). Those logits are drawn
    with the spread of the row's own visual logits, sigma = ||Q_h[q]|| / sqrt(dh), and the first
    system key gets sigma * 4 + 2 more (the usual attention sink)."""
    rng = np.random.Generator(np.random.PCG64(seed))
    Q = w.Q.astype(np.uint32) << np.uint32(16)
    Qf = Q.view(np.float32).astype(np.float64)                     # [sum L, hq, dh]
    sigma = np.sqrt((Qf * Qf).sum(axis=2)) / math.sqrt(w.dh)        # [sum L, hq]
    lse = np.empty((w.hq, Qf.shape[0]), dtype=np.float64)
    l_off = w.offsets("l")
    for b in range(w.B):
        for q in range(w.reqs[b].l):
            row = l_off[b] + q
            n_o = system_tokens + q + 1
            x = rng.standard_normal((w.hq, n_o)) * sigma[row][:, None]
            x[:, 0] += 4.0 * sigma[row] + 2.0
            m = x.max(axis=1)
            lse[:, row] = m + np.log(np.exp(x - m[:, None]).sum(axis=1))
    return dataclasses.replace(w, name=w.name + "_fullseq", lse_other=lse.astype(np.float32))


WORKLOADS = {
    "llava15_576_single": llava15_single,
    "llava15_576_b32": llava15_batch32,
    "llava_next_2880_b8": llava_next_batch8,
    "long_16384_b2_gqa": long_video_batch2,
    "ragged_varlen_b64": ragged_serving_batch64,
    "video_llava_2048_b4": video_llava_batch,
}
