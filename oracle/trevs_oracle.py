"""Plain CPU oracle of the TReVS two-stage visual-token pruning path (fp64).

TEST INFRASTRUCTURE ONLY. Nothing on the product path imports this module: only
the tests, the smoke check and the CPU-baseline leg of the benchmark do. It
shares no code with the CUDA library; the two meet only in the seeded input
bytes produced by `workloads.synth`.

Every function restates one step of the method in the paper's order and
notation, with library primitives (matmul, exp, stable sort) as its only
building blocks and no blocking, fusion or reordering. Inputs arrive as
bfloat16 bit patterns (uint16) or float32 and are widened exactly to float64.

Readings where the paper is silent or leaves a choice open:
  * A zero-norm vector has cosine 0 with everything (Eq. 4 divides by the norm; Eq. 1 alike).
  * Med is the lower median: the ascending element of rank floor((N-1)/2) (Eq. 6).
  * epsilon of Eq. 6 defaults to 1e-6.
  * Textual-ratio selection (Sec. 3.1): K_t = floor(r*K1 + 0.5) textual tokens,
    K_v = K1 - K_t saliency tokens; the saliency top-K_v is taken first, the
    textual top-K_t over the remaining tokens; both rank the raw scores.
  * TopK ties go to the lower token (or head) index; kept sets are returned in
    ascending index order, which preserves the original token order.
  * The text-to-vision softmax of Sec. 4.2 spans the K1 visual keys of each text
    row (each row sums to 1); no causal mask (every visual token precedes the
    text); scale 1/sqrt(d_h); query head h reads key head floor(h*Hkv/Hq).
  * Var_i in Eq. 8 is the population variance (divide by K1), two-pass.
  * H* holds n_keep_heads heads (the paper's default is half of the heads).
  * Context preservation (Sec. 3.1): the K_d diversity tokens are drawn by farthest
    point sampling over C = [N] minus the pivots S_r. The distance of a candidate to
    the selected set is its smallest cosine distance 1 - cos(z_i, z_s) to any token
    selected so far, the pivots included; each step takes the candidate of largest
    distance (ties to the lower index). With no pivots every candidate starts at
    distance +inf, so the first pick is the lowest index of C.
  * K_d = floor(rho*K1 + 0.5) for a diversity share rho (the paper's K_r:K_d = 3:1 is
    rho = 0.25); the pivots are the top K_r = K1 - K_d of the stage-1 rule.
  * Full-sequence variant of the Sec. 4.2 softmax (off by default): given lse_other[h, q],
    the log of the summed exp-logits of row q's non-visual keys (system and text tokens),
    the denominator also counts that mass, as the LLM's own softmax over the whole sequence
    does; rows then sum to less than 1, and Eq. 8-9 take those values as they are.
  * Eq. 1 compares each head's visual-token attention distribution under two questions; a
    head's distribution is its attention averaged over the text rows (a distribution again).
  * [CLS] saliency (Eq. 2-3): the softmax of each head runs over the N patch keys, as Eq. 2
    writes it (K_v holds the patch keys only), with scale 1/sqrt(d_h); s^v is the plain mean
    of the H heads' distributions.

Parity pins: every function here is pinned by tests/test_oracle_pins.py against
closed forms, hand-derived worked examples (tests/golden/), brute force on tiny
inputs and invariants; none is "parity unpinned".
"""
from __future__ import annotations

import math

import numpy as np

# ---------------------------------------------------------------- encodings


def bf16_bits_to_f64(bits: np.ndarray) -> np.ndarray:
    """bfloat16 bit patterns -> float64 (exact: bf16 is the top half of a float32)."""
    u = np.asarray(bits, dtype=np.uint16).astype(np.uint32) << np.uint32(16)
    return u.view(np.float32).astype(np.float64)


# ---------------------------------------------------------------- stage 1 (Sec. 4.1)


def cls_saliency(q_cls: np.ndarray, K_v: np.ndarray, scale: float | None = None) -> np.ndarray:
    """Eq. 2-3: s^v_i = (1/H) sum_h Softmax_i( q^h_[CLS] . k^h_i / sqrt(d_h) ).

    q_cls is [H, d_h] (the [CLS] query of every head), K_v is [N, H, d_h] (the patch keys of
    the penultimate ViT layer). Returns s^v, [N], a distribution over the patches.
    """
    q = np.asarray(q_cls, dtype=np.float64)
    K = np.asarray(K_v, dtype=np.float64)
    N, H, dh = K.shape
    if scale is None:
        scale = 1.0 / math.sqrt(dh)
    A = np.empty((H, N), dtype=np.float64)
    for h in range(H):
        logits = (K[:, h, :] @ q[h]) * scale                  # Eq. 2, before the softmax
        e = np.exp(logits - logits.max())
        A[h] = e / e.sum()
    return A.sum(axis=0) / H                                  # Eq. 3


def rectified_cosine(Z: np.ndarray, T: np.ndarray) -> np.ndarray:
    """Eq. 4: m[j, i] = max(tbar_j . zbar_i, 0) with zbar, tbar the L2-normalised rows.

    Z is [N, d'] visual features, T is [M, d'] text embeddings; returns [M, N].
    A zero-norm row has cosine 0 with every other row.
    """
    Z = np.asarray(Z, dtype=np.float64)
    T = np.asarray(T, dtype=np.float64)
    nz = np.sqrt(np.sum(Z * Z, axis=1))
    nt = np.sqrt(np.sum(T * T, axis=1))
    zbar = np.divide(Z, nz[:, None], out=np.zeros_like(Z), where=nz[:, None] > 0)
    tbar = np.divide(T, nt[:, None], out=np.zeros_like(T), where=nt[:, None] > 0)
    cos = tbar @ zbar.T
    return np.maximum(cos, 0.0)


def textual_relevance(Z: np.ndarray, T: np.ndarray) -> np.ndarray:
    """Eq. 5: s^t_i = sqrt( (1/M) * sum_j m[j, i]^2 ), the RMS over the M text tokens."""
    m = rectified_cosine(Z, T)
    M = m.shape[0]
    if M == 0:
        raise ValueError("textual relevance needs at least one text token")
    return np.sqrt(np.sum(m * m, axis=0) / M)


def lower_median(x: np.ndarray) -> float:
    """Med of Eq. 6: the ascending element of rank floor((N-1)/2)."""
    x = np.sort(np.asarray(x, dtype=np.float64), kind="stable")
    return float(x[(len(x) - 1) // 2])


def mad(x: np.ndarray) -> float:
    """MAD of Eq. 6: the median of |x_i - Med(x)|."""
    x = np.asarray(x, dtype=np.float64)
    return lower_median(np.abs(x - lower_median(x)))


def robust_normalise(s: np.ndarray, tau: float, eps: float) -> np.ndarray:
    """Eq. 6: shat_i = [ (s_i - Med(s)) / (MAD(s) + eps) ]_+ / tau."""
    s = np.asarray(s, dtype=np.float64)
    z = (s - lower_median(s)) / (mad(s) + eps)
    return np.maximum(z, 0.0) / tau


def fused_score(sv_hat: np.ndarray, st_hat: np.ndarray, lam: float) -> np.ndarray:
    """Eq. 7: s_i = max(shat^v_i, shat^t_i) + lambda * sqrt(shat^v_i * shat^t_i)."""
    sv_hat = np.asarray(sv_hat, dtype=np.float64)
    st_hat = np.asarray(st_hat, dtype=np.float64)
    return np.maximum(sv_hat, st_hat) + lam * np.sqrt(sv_hat * st_hat)


def top_k(score: np.ndarray, k: int, allowed: np.ndarray | None = None) -> np.ndarray:
    """TopK of Eq. 7 / Eq. 9: the k best entries by (score descending, index ascending).

    `allowed` (bool mask) restricts the candidates. Returns indices in ascending order.
    """
    score = np.asarray(score, dtype=np.float64)
    idx = np.arange(len(score))
    if allowed is not None:
        idx = idx[np.asarray(allowed, dtype=bool)]
    if k < 0 or k > len(idx):
        raise ValueError(f"top_k: k={k} outside [0, {len(idx)}]")
    order = np.lexsort((idx, -score[idx]))     # primary: -score ascending; then index
    return np.sort(idx[order[:k]])


def textual_count(k1: int, ratio: float) -> int:
    """K_t = floor(r * K1 + 0.5): the textual share of the keep budget (Sec. 3.1)."""
    return int(math.floor(float(np.float32(ratio)) * k1 + 0.5))


def select_ratio(s_v: np.ndarray, s_t: np.ndarray, k1: int, ratio: float) -> np.ndarray:
    """Sec. 3.1 budget split: saliency top-K_v, then textual top-K_t over the rest."""
    k_t = textual_count(k1, ratio)
    k_v = k1 - k_t
    S_v = top_k(s_v, k_v)
    rest = np.ones(len(s_v), dtype=bool)
    rest[S_v] = False
    S_t = top_k(s_t, k_t, allowed=rest)
    return np.sort(np.concatenate([S_v, S_t]))


def select_fused(s_v, s_t, k1, tau_v=1.4, tau_t=1.0, lam=1.0, eps=1e-6):
    """Eq. 6-7 pivot selection S_r = TopK(s, K_r) with K_r = K1 (no diversity tokens)."""
    s = fused_score(robust_normalise(s_v, tau_v, eps), robust_normalise(s_t, tau_t, eps), lam)
    return top_k(s, k1), s


def cosine_distance_to(Z: np.ndarray, j: int) -> np.ndarray:
    """1 - cos(z_i, z_j) for every row i of Z (Sec. 3.1); a zero-norm row has cosine 0."""
    Z = np.asarray(Z, dtype=np.float64)
    nz = np.sqrt(np.sum(Z * Z, axis=1))
    zbar = np.divide(Z, nz[:, None], out=np.zeros_like(Z), where=nz[:, None] > 0)
    return 1.0 - zbar @ zbar[j]


def farthest_point_sampling(Z: np.ndarray, pivots, k_d: int):
    """Sec. 3.1 context preservation: S_d = FPS({z_i | i in C}, K_d), C = [N] minus S_r.

    Z is [N, d'] (float64 values); `pivots` is S_r. Each of the K_d steps takes the
    candidate farthest from everything selected so far: its distance is the minimum of
    1 - cos over the selected tokens (pivots and earlier picks); ties go to the lower
    index. Returns (picks in the order they are taken, the distance of each when taken).
    """
    Z = np.asarray(Z, dtype=np.float64)
    N = len(Z)
    cand = np.ones(N, dtype=bool)
    dist = np.full(N, np.inf)
    for s in np.asarray(pivots, dtype=np.int64):
        cand[s] = False
        dist = np.minimum(dist, cosine_distance_to(Z, int(s)))
    if k_d < 0 or k_d > int(cand.sum()):
        raise ValueError(f"farthest_point_sampling: K_d={k_d} outside [0, {int(cand.sum())}]")
    picks, taken_at = [], []
    for _ in range(k_d):
        idx = np.flatnonzero(cand)
        j = int(idx[np.argmax(dist[idx])])     # first maximum = lowest index among ties
        picks.append(j)
        taken_at.append(dist[j])
        cand[j] = False
        dist = np.minimum(dist, cosine_distance_to(Z, j))
    return np.array(picks, dtype=np.int64), np.array(taken_at, dtype=np.float64)


def diversity_count(k1: int, rho: float) -> int:
    """K_d = floor(rho * K1 + 0.5): the diversity share of the stage-1 budget (Sec. 3.1)."""
    return int(math.floor(float(np.float32(rho)) * k1 + 0.5))


def gather_rows(X: np.ndarray, idx: np.ndarray) -> np.ndarray:
    """Sec. 4.1: the kept rows, in ascending index order, are passed to the LLM."""
    return np.asarray(X)[np.asarray(idx, dtype=np.int64)]


# ---------------------------------------------------------------- stage 2 (Sec. 4.2)


def text_to_vision_attention(Q: np.ndarray, K: np.ndarray, scale: float | None = None,
                             lse_other: np.ndarray | None = None):
    """A^h_{T->V}[q, i] = softmax_i( Q[q, h] . K[i, g(h)] * scale ), g(h) = floor(h*Hkv/Hq).

    Q is [L, Hq, dh] (text rows at layer l*), K is [K1, Hkv, dh] (visual keys).
    Returns A as [Hq, L, K1]; every row is a distribution over the K1 visual keys. With
    lse_other [Hq, L] the denominator of row (h, q) also holds exp(lse_other[h, q]), the mass
    of the row's non-visual keys, and the row sums to less than 1.
    """
    Q = np.asarray(Q, dtype=np.float64)
    K = np.asarray(K, dtype=np.float64)
    L, Hq, dh = Q.shape
    K1, Hkv, _ = K.shape
    if scale is None:
        scale = 1.0 / math.sqrt(dh)
    A = np.empty((Hq, L, K1), dtype=np.float64)
    for h in range(Hq):
        g = (h * Hkv) // Hq
        logits = (Q[:, h, :] @ K[:, g, :].T) * scale          # [L, K1]
        mx = logits.max(axis=1, keepdims=True)
        if lse_other is not None:
            other = np.asarray(lse_other, dtype=np.float64)[h][:, None]
            mx = np.maximum(mx, other)
        e = np.exp(logits - mx)
        den = e.sum(axis=1, keepdims=True)
        if lse_other is not None:
            den = den + np.exp(other - mx)
        A[h] = e / den
    return A


def head_visual_attention(A: np.ndarray) -> np.ndarray:
    """s_h of Eq. 1: head h's attention over the visual tokens, averaged over the text rows.

    A is [Hq, L, K1] (text-to-vision attention); returns [Hq, K1].
    """
    A = np.asarray(A, dtype=np.float64)
    return A.sum(axis=1) / A.shape[1]


def textual_sensitivity(s1: np.ndarray, s2: np.ndarray) -> np.ndarray:
    """Eq. 1: TS_h = 1 - cos(s_h^(1), s_h^(2)) for the distributions of every head under two
    questions; s1 and s2 are [Hq, K1]. Returns [Hq]. A zero vector has cosine 0 (as for Eq. 4)."""
    s1 = np.asarray(s1, dtype=np.float64)
    s2 = np.asarray(s2, dtype=np.float64)
    num = (s1 * s2).sum(axis=1)
    den = np.sqrt((s1 * s1).sum(axis=1)) * np.sqrt((s2 * s2).sum(axis=1))
    return 1.0 - np.divide(num, den, out=np.zeros_like(num), where=den > 0)


def head_variance(A: np.ndarray) -> np.ndarray:
    """Eq. 8: u_h = (1/L) sum_q Var_i A^h[q, i] (population variance, two-pass)."""
    A = np.asarray(A, dtype=np.float64)
    K1 = A.shape[2]
    mean = A.sum(axis=2, keepdims=True) / K1
    var = ((A - mean) ** 2).sum(axis=2) / K1                 # [Hq, L]
    return var.sum(axis=1) / A.shape[1]


def select_heads(u: np.ndarray, n_keep: int) -> np.ndarray:
    """H*: the n_keep heads of largest u_h (ties to the lower head), ascending."""
    return top_k(u, n_keep)


def token_scores(A: np.ndarray, heads: np.ndarray) -> np.ndarray:
    """Eq. 9: p_i = max_q (1/|H*|) sum_{h in H*} A^h[q, i]."""
    A = np.asarray(A, dtype=np.float64)
    heads = np.asarray(heads, dtype=np.int64)
    mean_over_heads = A[heads].sum(axis=0) / len(heads)      # [L, K1]
    return mean_over_heads.max(axis=0)


# ---------------------------------------------------------------- per-request drivers


def pre_llm_request(Z_bits, T_bits, s_v, k1, ratio, mode="ratio", tau_v=1.4, tau_t=1.0,
                    lam=1.0, eps=1e-6, diversity=0.0):
    """Stage 1 for one request: s^t (Eq. 4-5), selection, gather of the kept rows.

    With a diversity share rho > 0 the rule picks the K_r = K1 - K_d pivots S_r and
    farthest point sampling adds K_d = floor(rho*K1 + 0.5) tokens (Sec. 3.1); the kept
    set is S_r and S_d together, in ascending order.
    """
    Z = bf16_bits_to_f64(Z_bits)
    T = bf16_bits_to_f64(T_bits)
    s_v = np.asarray(s_v, dtype=np.float64)
    if len(Z) == 0:   # a request without visual tokens has nothing to score or keep
        empty = np.zeros(0)
        return {"s_t": empty, "s_fused": empty, "kept": np.zeros(0, np.int64),
                "Z_out": np.asarray(Z_bits)[:0]}
    s_t = textual_relevance(Z, T)
    out = {"s_t": s_t}
    k_d = diversity_count(k1, diversity)
    k_r = k1 - k_d
    if mode == "ratio":
        kept = select_ratio(s_v, s_t, k_r, ratio)
    elif mode == "fused":
        kept, s = select_fused(s_v, s_t, k_r, tau_v, tau_t, lam, eps)
        out["s_fused"] = s
    else:
        raise ValueError(mode)
    if k_d > 0:
        picks, taken_at = farthest_point_sampling(Z, kept, k_d)
        out["pivots"], out["fps"], out["fps_dist"] = kept, picks, taken_at
        kept = np.sort(np.concatenate([kept, picks]))
    out["kept"] = kept
    out["Z_out"] = gather_rows(np.asarray(Z_bits), kept)
    return out


def in_llm_request(Q_bits, K_bits, V_bits, hidden_bits, n_keep_heads, k2, scale=None, lse_other=None):
    """Stage 2 for one request: attention, Eq. 8 variance, H*, Eq. 9 scores, top-K2, compaction.
    lse_other [Hq, L] selects the full-sequence softmax variant of Sec. 4.2."""
    Q = bf16_bits_to_f64(Q_bits)
    K = bf16_bits_to_f64(K_bits)
    A = text_to_vision_attention(Q, K, scale, lse_other)
    u = head_variance(A)
    heads = select_heads(u, n_keep_heads)
    p = token_scores(A, heads)
    kept = top_k(p, k2)
    return {
        "u": u, "heads": heads, "p": p, "kept": kept,
        "hidden_out": gather_rows(np.asarray(hidden_bits), kept),
        "K_out": gather_rows(np.asarray(K_bits), kept),
        "V_out": gather_rows(np.asarray(V_bits), kept),
    }


def run_workload(w, mode="ratio", stage1=True, stage2=True, requests=None, **params):
    """Both stages over every request of a `workloads.synth.Workload` (or a subset)."""
    n_off, m_off = w.offsets("n"), w.offsets("m")
    k1_off, l_off = w.offsets("k1"), w.offsets("l")
    out = []
    for b in (range(w.B) if requests is None else requests):
        r = w.reqs[b]
        res = {}
        if stage1:
            res["pre"] = pre_llm_request(
                w.Z[n_off[b]:n_off[b + 1]], w.T[m_off[b]:m_off[b + 1]],
                w.s_v[n_off[b]:n_off[b + 1]], r.k1, r.ratio, mode, **params)
        if stage2:
            lse = getattr(w, "lse_other", None)
            res["in"] = in_llm_request(
                w.Q[l_off[b]:l_off[b + 1]], w.K[k1_off[b]:k1_off[b + 1]],
                w.V[k1_off[b]:k1_off[b + 1]], w.hidden[k1_off[b]:k1_off[b + 1]],
                w.n_keep_heads, r.k2, lse_other=None if lse is None else lse[:, l_off[b]:l_off[b + 1]])
        out.append(res)
    return out
