"""Pins that tie the oracle to facts other than itself.

Each pin checks one oracle function against a closed form, a worked example
derived by hand from the paper's equations (tests/golden/), brute force over
all subsets on tiny inputs, or an invariant the mathematics fixes. Pins call
the oracle through its module attribute so the mutation tests can swap in a
planted mistake and see a pin fail.
"""
from __future__ import annotations

import itertools
import json
import math
import pathlib

import numpy as np

import oracle.trevs_oracle as O

GOLDEN = pathlib.Path(__file__).parent / "golden"
_ENV = {"__builtins__": {}, "sqrt": math.sqrt, "ln2": math.log(2.0), "ln3": math.log(3.0)}


def _val(expr) -> float:
    return float(eval(str(expr), _ENV)) if isinstance(expr, str) else float(expr)


def _vals(xs):
    return np.array([_val(x) if not isinstance(x, list) else _vals(x) for x in xs], dtype=np.float64)


def _golden(name):
    return json.loads((GOLDEN / name).read_text())


def _close(a, b, tol=1e-12):
    a = np.asarray(a, dtype=np.float64)
    b = np.asarray(b, dtype=np.float64)
    assert a.shape == b.shape, (a.shape, b.shape)
    assert np.all(np.abs(a - b) <= tol * (1.0 + np.abs(b))), (a, b)


# ------------------------------------------------------------- Eq. 4-5


def pin_textual_relevance_worked_example():
    g = _golden("textual_relevance_2d.json")
    Z, T = np.array(g["Z"], float), np.array(g["T"], float)
    _close(O.rectified_cosine(Z, T), _vals(g["m"]))
    _close(O.textual_relevance(Z, T), _vals(g["s_t"]))


def pin_textual_relevance_closed_forms():
    rng = np.random.default_rng(7)
    z = rng.standard_normal(33)
    T_par = np.stack([0.5 * z, 3.0 * z, 1.0 * z])           # all parallel -> cos 1
    assert abs(O.textual_relevance(z[None], T_par)[0] - 1.0) < 1e-12
    assert O.textual_relevance(z[None], -T_par)[0] == 0.0     # anti-parallel -> 0
    e = np.eye(5)
    assert np.all(O.textual_relevance(e[:2], e[2:]) == 0.0)   # orthogonal -> 0
    assert np.all(O.textual_relevance(np.zeros((3, 5)), e) == 0.0)   # zero norm -> 0
    # RMS of a constant: identical text tokens give relu(cos) itself
    t = rng.standard_normal(33)
    Z = rng.standard_normal((6, 33))
    cos = (Z @ t) / (np.linalg.norm(Z, axis=1) * np.linalg.norm(t))
    _close(O.textual_relevance(Z, np.stack([t] * 4)), np.maximum(cos, 0.0))


def pin_textual_relevance_invariants():
    rng = np.random.default_rng(11)
    Z = rng.standard_normal((9, 17))
    T = rng.standard_normal((4, 17))
    T[0] = Z[2]                                                # one strong match
    s = O.textual_relevance(Z, T)
    cz = rng.uniform(0.1, 10.0, size=9)[:, None]
    ct = rng.uniform(0.1, 10.0, size=4)[:, None]
    _close(O.textual_relevance(Z * cz, T * ct), s, 1e-12)      # positive row scaling
    perm_t = rng.permutation(4)
    _close(O.textual_relevance(Z, T[perm_t]), s, 1e-12)        # text order irrelevant
    perm_z = rng.permutation(9)
    _close(O.textual_relevance(Z[perm_z], T), s[perm_z], 1e-12)
    # one text token: s^t = relu(cos) of that token
    cos = (Z @ T[1]) / (np.linalg.norm(Z, axis=1) * np.linalg.norm(T[1]))
    _close(O.textual_relevance(Z, T[1:2]), np.maximum(cos, 0.0))
    # the RMS lies between the mean and the max of m over text tokens
    m = np.array([[max(0.0, float(np.dot(T[j], Z[i]) / np.linalg.norm(T[j]) / np.linalg.norm(Z[i])))
                   for i in range(9)] for j in range(4)])
    assert np.all(s >= m.mean(axis=0) - 1e-12) and np.all(s <= m.max(axis=0) + 1e-12)


# ------------------------------------------------------------- Eq. 6-7


def pin_median_mad_worked_example():
    g = _golden("robust_fused_5.json")
    for key in ("a", "b", "c"):
        assert O.lower_median(np.array(g[key], float)) == _val(g[key + "_med"])
        assert O.mad(np.array(g[key], float)) == _val(g[key + "_mad"])


def pin_median_by_counting():
    rng = np.random.default_rng(3)
    for n in range(1, 12):
        for _ in range(20):
            x = rng.integers(0, 4, size=n).astype(float)        # many ties
            med = O.lower_median(x)
            below = int(np.sum(x < med))
            upto = int(np.sum(x <= med))
            assert below <= (n - 1) // 2 < upto
            dev = np.abs(x - med)
            mad = O.mad(x)
            assert int(np.sum(dev < mad)) <= (n - 1) // 2 < int(np.sum(dev <= mad))


def pin_robust_fused_worked_example():
    g = _golden("robust_fused_5.json")
    ah = O.robust_normalise(np.array(g["a"], float), g["tau_a"], 0.0)
    bh = O.robust_normalise(np.array(g["b"], float), g["tau_b"], 0.0)
    _close(ah, _vals(g["a_hat"]))
    _close(bh, _vals(g["b_hat"]))
    s = O.fused_score(ah, bh, g["lambda"])
    _close(s, _vals(g["s"]))
    assert list(O.top_k(s, 2)) == g["top2"]
    # eps enters the denominator: MAD + eps
    _close(O.robust_normalise(np.array(g["a"], float), 1.0, 1.0), [0, 0, 0, 0.5, 3.5])


def pin_fused_score_closed_forms():
    x = np.array([0.0, 2.0, 3.0, 4.0])
    y = np.array([0.0, 0.0, 3.0, 1.0])
    _close(O.fused_score(x, y, 0.0), np.maximum(x, y))           # lambda=0: plain max
    _close(O.fused_score(x, y, 1.0), [0.0, 2.0, 6.0, 6.0])       # equal pair: 2x
    _close(O.fused_score(y, x, 0.5), O.fused_score(x, y, 0.5))   # symmetric


# ------------------------------------------------------------- TopK / Sec. 3.1 split


def _brute_top(score, k, allowed):
    """The unique k-subset whose every member precedes every non-member."""
    cand = [i for i in range(len(score)) if allowed[i]]
    found = []
    for S in itertools.combinations(cand, k):
        Sset = set(S)
        ok = all((score[i] > score[j]) or (score[i] == score[j] and i < j)
                 for i in S for j in cand if j not in Sset)
        if ok:
            found.append(list(S))
    assert len(found) == 1
    return found[0]


def pin_top_k_brute_force():
    rng = np.random.default_rng(5)
    for n in range(1, 9):
        for _ in range(6):
            s = rng.integers(0, 3, size=n).astype(float)
            allowed = rng.random(n) < 0.8
            for k in range(0, int(allowed.sum()) + 1):
                assert list(O.top_k(s, k, allowed)) == _brute_top(s, k, allowed)
    # -0.0 and +0.0 are the same score: tie to the lower index
    assert list(O.top_k(np.array([-0.0, 0.0, -0.0]), 2)) == [0, 1]


def pin_ratio_split_worked_example():
    g = _golden("ratio_split_6.json")
    sv, st = np.array(g["s_v"]), np.array(g["s_t"])
    for r, kt, kept in g["cases"]:
        assert O.textual_count(g["k1"], r) == kt
        assert list(O.select_ratio(sv, st, g["k1"], r)) == kept


def pin_ratio_split_brute_force():
    rng = np.random.default_rng(9)
    for n in range(2, 9):
        for _ in range(5):
            sv = rng.integers(0, 3, size=n).astype(float)
            st = rng.integers(0, 3, size=n).astype(float)
            for k1 in range(1, n + 1):
                for r in (0.0, 0.25, 0.5, 0.75, 1.0):
                    kt = int(math.floor(r * k1 + 0.5))
                    Sv = _brute_top(sv, k1 - kt, [True] * n)
                    rest = [i not in Sv for i in range(n)]
                    St = _brute_top(st, kt, rest)
                    got = list(O.select_ratio(sv, st, k1, r))
                    assert got == sorted(Sv + St)
                    assert len(got) == k1 and len(set(got)) == k1
            # ratio 0 and 1 reduce to the single-signal top-K
            assert list(O.select_ratio(sv, st, 2, 0.0)) == list(O.top_k(sv, 2))
            assert list(O.select_ratio(sv, st, 2, 1.0)) == list(O.top_k(st, 2))


def pin_gather_preserves_order():
    X = np.arange(40).reshape(10, 4)
    idx = np.array([1, 4, 5, 9])
    out = O.gather_rows(X, idx)
    assert out.shape == (4, 4) and np.all(out[:, 0] == idx * 4)


# ------------------------------------------------------------- Sec. 4.2, Eq. 8-9


def _golden_stage2():
    g = _golden("head_variance_2x2.json")
    Q = _vals(g["Q"])[:, :, None]                             # [L=2, Hq=2, dh=1]
    K = np.array(g["K"], float)[:, None, None]                 # [K1=3, Hkv=1, 1]
    return g, Q, K


def pin_stage2_worked_example():
    g, Q, K = _golden_stage2()
    A = O.text_to_vision_attention(Q, K, 1.0)
    _close(A, _vals(g["A"]))
    u = O.head_variance(A)
    _close(u, _vals(g["u"]))
    for nh, key in ((1, "nh1"), (2, "nh2")):
        heads = O.select_heads(u, nh)
        assert list(heads) == g[key]["heads"]
        p = O.token_scores(A, heads)
        _close(p, _vals(g[key]["p"]))
        assert list(O.top_k(p, 1)) == g[key]["top1"]
        assert list(O.top_k(p, 2)) == g[key]["top2"]


def pin_softmax_rows_and_shift():
    rng = np.random.default_rng(13)
    Q = rng.standard_normal((5, 4, 8)) * 3
    K = rng.standard_normal((11, 2, 8))
    A = O.text_to_vision_attention(Q, K)
    assert A.shape == (4, 5, 11)
    assert np.all(np.abs(A.sum(axis=2) - 1.0) < 1e-12)
    # a constant key offset shifts each row's logits equally: A is unchanged
    _close(O.text_to_vision_attention(Q, K + rng.standard_normal((1, 2, 8))), A, 1e-9)
    # default scale is 1/sqrt(dh)
    _close(O.text_to_vision_attention(Q, K), O.text_to_vision_attention(Q, K, 1 / math.sqrt(8)))
    _close(O.text_to_vision_attention(Q / math.sqrt(8), K, 1.0), A, 1e-12)


def pin_uniform_attention():
    Q = np.zeros((3, 6, 4))
    K = np.random.default_rng(1).standard_normal((10, 3, 4))
    A = O.text_to_vision_attention(Q, K)
    assert np.all(A == 0.1)
    u = O.head_variance(A)
    assert np.all(u == 0.0)
    heads = O.select_heads(u, 4)
    assert list(heads) == [0, 1, 2, 3]
    p = O.token_scores(A, heads)
    assert np.allclose(p, 0.1)
    assert list(O.top_k(p, 3)) == [0, 1, 2]


def pin_one_hot_variance():
    K1 = 7
    K = np.eye(K1)[:, None, :] * 1.0                            # key i = e_i
    Q = np.zeros((1, 1, K1))
    Q[0, 0, 3] = 1e4                                            # one key dominates
    A = O.text_to_vision_attention(Q, K, 1.0)
    assert abs(A[0, 0, 3] - 1.0) < 1e-12
    u = O.head_variance(A)
    assert abs(u[0] - (1.0 / K1) * (1.0 - 1.0 / K1)) < 1e-12


def pin_variance_naive_formula():
    rng = np.random.default_rng(17)
    A = O.text_to_vision_attention(rng.standard_normal((6, 5, 16)) * 2,
                                   rng.standard_normal((23, 5, 16)))
    K1 = A.shape[2]
    naive = ((A ** 2).sum(axis=2) / K1 - (A.sum(axis=2) / K1) ** 2).mean(axis=1)
    _close(O.head_variance(A), naive, 1e-9)


def pin_gqa_mapping():
    rng = np.random.default_rng(19)
    Q = rng.standard_normal((4, 8, 16))
    Kg = rng.standard_normal((9, 2, 16))                        # 2 KV heads for 8 query heads
    Kfull = np.repeat(Kg, 4, axis=1)                            # query head h reads kv head h // 4
    _close(O.text_to_vision_attention(Q, Kg), O.text_to_vision_attention(Q, Kfull), 1e-12)
    # with Hkv = Hq the mapping is the identity: permuting heads permutes A
    perm = rng.permutation(8)
    _close(O.text_to_vision_attention(Q[:, perm], Kfull[:, perm]),
           O.text_to_vision_attention(Q, Kfull)[perm], 1e-12)


def pin_token_score_single_head():
    rng = np.random.default_rng(23)
    A = O.text_to_vision_attention(rng.standard_normal((6, 3, 8)), rng.standard_normal((12, 3, 8)))
    _close(O.token_scores(A, np.array([1])), A[1].max(axis=0))
    _close(O.token_scores(A, np.array([0, 2])), ((A[0] + A[2]) / 2).max(axis=0))


def pin_select_heads_brute_force():
    rng = np.random.default_rng(29)
    for _ in range(30):
        u = rng.integers(0, 3, size=6).astype(float)
        for k in range(0, 7):
            assert list(O.select_heads(u, k)) == _brute_top(u, k, [True] * 6)


def pin_bf16_decode():
    bits = np.array([0x3F80, 0xC020, 0x0000, 0x8000, 0x7F7F, 0x0001], dtype=np.uint16)
    got = O.bf16_bits_to_f64(bits)
    want = [1.0, -2.5, 0.0, -0.0, (2 - 2 ** -7) * 2.0 ** 127, 2.0 ** -133]
    assert list(got) == want



# ------------------------------------------------------------- Sec. 3.1, context preservation


def _hypercube16():
    return np.array([[1 - 2 * ((k >> c) & 1) for c in range(4)] for k in range(16)], dtype=np.float64)


def pin_fps_worked_example():
    g = _golden("fps_hypercube_16.json")
    Z = _hypercube16()
    picks, dist = O.farthest_point_sampling(Z, g["pivots"], len(g["order"]))
    assert list(picks) == g["order"]
    assert list(dist) == g["dist"]
    assert list(O.farthest_point_sampling(Z, [], 16)[0]) == g["order_no_pivots"]
    Z0 = np.vstack([Z, np.zeros((1, 4))])
    assert list(O.farthest_point_sampling(Z0, g["pivots"], 16)[0]) == g["order_zero_row"]
    # positive row scales by powers of two change no bit of a cosine
    scale = 2.0 ** np.arange(-3, 13)[:, None]
    assert list(O.farthest_point_sampling(Z * scale, g["pivots"], 15)[0]) == g["order"]
    # fewer picks are a prefix of the sequence
    assert list(O.farthest_point_sampling(Z, g["pivots"], 4)[0]) == g["order"][:4]


def _euclid_fps(Z, pivots, k):
    """FPS by squared Euclidean distance between the unit rows, from scipy's cdist: on the
    unit sphere |a - b|^2 = 2 (1 - cos(a, b)), so the picks are the same."""
    from scipy.spatial.distance import cdist
    U = Z / np.linalg.norm(Z, axis=1, keepdims=True)
    D = cdist(U, U, "sqeuclidean")
    sel = list(pivots)
    picks, dists = [], []
    for _ in range(k):
        best, best_d = None, -1.0
        for i in range(len(Z)):
            if i in sel:
                continue
            di = min((D[i, s] for s in sel), default=np.inf)
            if di > best_d:
                best, best_d = i, di
        sel.append(best)
        picks.append(best)
        dists.append(best_d / 2.0)
    return picks, dists


def pin_fps_euclidean_equivalence():
    rng = np.random.default_rng(21)
    for n in range(2, 13):
        for _ in range(4):
            Z = rng.standard_normal((n, 5))
            kr = int(rng.integers(0, n))
            piv = sorted(rng.choice(n, size=kr, replace=False).tolist())
            k = n - kr
            picks, dist = O.farthest_point_sampling(Z, piv, k)
            want, want_d = _euclid_fps(Z, piv, k)
            assert list(picks) == want
            fin = np.isfinite(want_d)
            assert list(np.isfinite(dist)) == list(fin)
            _close(np.asarray(dist)[fin], np.asarray(want_d)[fin], 1e-9)


def pin_fps_two_approximation():
    """Greedy farthest-point selection covers within twice the best possible radius
    (Gonzalez), for the Euclidean metric on the unit rows; brute force over all subsets."""
    rng = np.random.default_rng(23)
    for n in range(3, 10):
        for _ in range(3):
            Z = rng.standard_normal((n, 3))
            U = Z / np.linalg.norm(Z, axis=1, keepdims=True)
            E = np.sqrt(np.maximum(((U[:, None, :] - U[None, :, :]) ** 2).sum(-1), 0.0))
            piv = [int(rng.integers(0, n))]
            cand = [i for i in range(n) if i not in piv]
            for k in range(1, len(cand)):
                picks, _ = O.farthest_point_sampling(Z, piv, k)
                S = piv + list(picks)
                radius = max(min(E[i, s] for s in S) for i in range(n))
                best = min(max(min(E[i, s] for s in piv + list(c)) for i in range(n))
                           for c in itertools.combinations(cand, k))
                assert radius <= 2.0 * best + 1e-12


def pin_fps_invariants():
    rng = np.random.default_rng(29)
    Z = rng.standard_normal((40, 16))
    piv = [3, 17, 22, 39]
    picks, dist = O.farthest_point_sampling(Z, piv, 36)
    assert sorted(picks) == [i for i in range(40) if i not in piv]   # K_d = |C|: all of C
    assert np.all(np.diff(dist) <= 0)                                # distances never grow
    p2, d2 = O.farthest_point_sampling(Z * rng.uniform(0.1, 10.0, size=(40, 1)), piv, 36)
    assert list(p2) == list(picks)                                   # positive row scales
    _close(d2, dist, 1e-12)
    # an orthonormal basis: every distance is 1, so picks go in index order
    p3, d3 = O.farthest_point_sampling(np.eye(9), [4], 8)
    assert list(p3) == [0, 1, 2, 3, 5, 6, 7, 8] and list(d3) == [1.0] * 8
    # a duplicate of a pivot is at distance 0 and comes last
    Zd = np.vstack([Z[:6], Z[2:3]])
    p4, d4 = O.farthest_point_sampling(Zd, [2], 6)
    assert p4[-1] == 6 and abs(d4[-1]) < 1e-12


def pin_diversity_share():
    assert O.diversity_count(64, 0.25) == 16
    assert O.diversity_count(192, 0.25) == 48
    assert O.diversity_count(10, 0.25) == 3     # 2.5 rounds half up
    assert O.diversity_count(6, 0.25) == 2      # 1.5 + 0.5
    assert O.diversity_count(7, 0.0) == 0
    # a request with rho > 0: the pivots are the rule's top K1 - K_d, FPS adds K_d more
    rng = np.random.default_rng(31)
    N, d, M, K1 = 48, 64, 5, 12
    f32 = lambda x: (np.asarray(x, np.float32).view(np.uint32) >> 16).astype(np.uint16)
    Zb, Tb = f32(rng.standard_normal((N, d))), f32(rng.standard_normal((M, d)))
    sv = rng.random(N)
    for mode in ("fused", "ratio"):
        r = O.pre_llm_request(Zb, Tb, sv, K1, 0.5, mode, diversity=0.25)
        base = O.pre_llm_request(Zb, Tb, sv, K1 - 3, 0.5, mode)
        assert list(r["pivots"]) == list(base["kept"])
        assert len(r["fps"]) == 3 and not set(r["fps"]) & set(base["kept"])
        assert list(r["kept"]) == sorted(list(base["kept"]) + list(r["fps"]))
        assert list(O.pre_llm_request(Zb, Tb, sv, K1, 0.5, mode, diversity=0.0)["kept"]) == \
            list(O.pre_llm_request(Zb, Tb, sv, K1, 0.5, mode)["kept"])



# ------------------------------------------------------------- Eq. 2-3, [CLS] saliency


def pin_cls_saliency_worked_example():
    g = _golden("cls_saliency_3x2.json")
    q = _vals(g["q_cls"])
    K = _vals(g["K_v"])
    _close(O.cls_saliency(q, K), _vals(g["s_v"]), 1e-12)


def pin_cls_saliency_single_head_is_softmax():
    from scipy.special import softmax
    rng = np.random.default_rng(37)
    for N, dh in ((1, 8), (5, 64), (300, 128)):
        q = rng.standard_normal((1, dh))
        K = 3.0 * rng.standard_normal((N, 1, dh))
        _close(O.cls_saliency(q, K), softmax(K[:, 0, :] @ q[0] / math.sqrt(dh)), 1e-12)


def pin_cls_saliency_closed_forms():
    rng = np.random.default_rng(41)
    N, H, dh = 9, 4, 16
    K = rng.standard_normal((N, H, dh))
    _close(O.cls_saliency(np.zeros((H, dh)), K), np.full(N, 1.0 / N))            # q = 0: uniform
    _close(O.cls_saliency(rng.standard_normal((H, dh)), np.repeat(K[:1], N, 0)), np.full(N, 1.0 / N))
    # one key along q: logit x, the others 0 -> e^x / (e^x + N - 1)
    q = np.zeros((1, 4)); q[0, 0] = 2.0
    Kx = np.zeros((N, 1, 4)); Kx[5, 0, 0] = 1.5              # logit 2 * 1.5 / sqrt(4) = 1.5
    want = np.full(N, 1.0 / (math.exp(1.5) + N - 1)); want[5] = math.exp(1.5) / (math.exp(1.5) + N - 1)
    _close(O.cls_saliency(q, Kx), want)


def pin_cls_saliency_invariants():
    rng = np.random.default_rng(43)
    N, H, dh = 50, 6, 32
    q = rng.standard_normal((H, dh))
    K = 2.0 * rng.standard_normal((N, H, dh))
    s = O.cls_saliency(q, K)
    assert abs(s.sum() - 1.0) < 1e-12 and np.all(s > 0)
    perm = rng.permutation(H)
    _close(O.cls_saliency(q[perm], K[:, perm]), s)                           # head order
    _close(O.cls_saliency(q * 4.0, K / 4.0), s)                              # q.k unchanged
    _close(O.cls_saliency(q, K + rng.standard_normal((1, H, dh))), s, 1e-10)  # one shift per head



# ------------------------------------------------------------- Sec. 4.2 full-sequence variant, Eq. 1


def pin_full_sequence_softmax_is_a_restriction():
    """The variant with lse_other = logsumexp of some extra keys' logits equals the plain
    softmax over the visual keys and those extra keys, restricted to the visual columns."""
    from scipy.special import logsumexp, softmax
    rng = np.random.default_rng(47)
    L, Hq, Hkv, dh, K1, E = 5, 4, 2, 16, 11, 7
    Q = rng.standard_normal((L, Hq, dh)) * 2.0
    K = rng.standard_normal((K1, Hkv, dh))
    Kx = rng.standard_normal((E, Hkv, dh))                 # the non-visual keys
    lse = np.empty((Hq, L))
    want = np.empty((Hq, L, K1))
    for h in range(Hq):
        g = (h * Hkv) // Hq
        lv = Q[:, h, :] @ K[:, g, :].T / 4.0
        lx = Q[:, h, :] @ Kx[:, g, :].T / 4.0
        lse[h] = logsumexp(lx, axis=1)
        want[h] = softmax(np.concatenate([lv, lx], axis=1), axis=1)[:, :K1]
    _close(O.text_to_vision_attention(Q, K, lse_other=lse), want, 1e-12)


def pin_full_sequence_softmax_closed_forms():
    rng = np.random.default_rng(53)
    L, H, dh, K1 = 3, 2, 8, 6
    K = rng.standard_normal((K1, H, dh))
    # Q = 0: every logit is 0, so a row is 1 / (K1 + c) with lse_other = ln c
    A = O.text_to_vision_attention(np.zeros((L, H, dh)), K, lse_other=np.full((H, L), math.log(3.0)))
    _close(A, np.full((H, L, K1), 1.0 / (K1 + 3.0)))
    # lse_other = -inf is the plain softmax
    Q = rng.standard_normal((L, H, dh))
    _close(O.text_to_vision_attention(Q, K, lse_other=np.full((H, L), -np.inf)),
           O.text_to_vision_attention(Q, K))


def pin_textual_sensitivity():
    s1 = np.array([[1.0, 0.0], [0.25, 0.75], [0.5, 0.5]])
    s2 = np.array([[0.5, 0.5], [0.25, 0.75], [1.0, 0.0]])
    # head 0: cos = (1/2) / (1 * sqrt(1/2)) = 1/sqrt(2); head 1: identical; head 2: cos = 1/sqrt(2)
    _close(O.textual_sensitivity(s1, s2), [1 - 1 / math.sqrt(2), 0.0, 1 - 1 / math.sqrt(2)])
    _close(O.textual_sensitivity(np.array([[1.0, 0.0, 0.0]]), np.array([[0.0, 0.3, 0.7]])), [1.0])   # disjoint
    rng = np.random.default_rng(59)
    a, b = rng.random((4, 9)), rng.random((4, 9))
    _close(O.textual_sensitivity(a, 3.0 * b), O.textual_sensitivity(a, b))          # scale
    _close(O.textual_sensitivity(a, b), O.textual_sensitivity(b, a))                # symmetric
    # a zero distribution has cosine 0 with anything (the reading of Eq. 4 carried over)
    _close(O.textual_sensitivity(np.zeros((1, 3)), np.array([[0.2, 0.3, 0.5]])), [1.0])


def pin_head_visual_attention():
    A = np.array([[[1.0, 0.0], [0.0, 1.0]], [[0.25, 0.75], [0.75, 0.25]]])
    _close(O.head_visual_attention(A), [[0.5, 0.5], [0.5, 0.5]])
    rng = np.random.default_rng(61)
    A = O.text_to_vision_attention(rng.standard_normal((7, 3, 8)), rng.standard_normal((13, 3, 8)))
    _close(O.head_visual_attention(A).sum(axis=1), np.ones(3))


ALL_PINS = [v for k, v in sorted(globals().items()) if k.startswith("pin_") and callable(v)]
