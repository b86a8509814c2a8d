"""Plant plausible mistakes in the oracle (on the CPU) and check that a pin catches each one.

A mutant replaces one oracle function for the duration of a test; the pin
suite must then fail somewhere. This shows the pins are tight enough that a
dropped term, a wrong sign, a wrong index or a transposed operand in the oracle
would not pass unnoticed.
"""
import math

import numpy as np
import pytest

import oracle.trevs_oracle as O
from tests import oracle_pins

_orig = {name: getattr(O, name) for name in dir(O) if callable(getattr(O, name))}


def _no_relu(Z, T):
    Z = np.asarray(Z, float); T = np.asarray(T, float)
    nz = np.linalg.norm(Z, axis=1); nt = np.linalg.norm(T, axis=1)
    zb = np.divide(Z, nz[:, None], out=np.zeros_like(Z), where=nz[:, None] > 0)
    tb = np.divide(T, nt[:, None], out=np.zeros_like(T), where=nt[:, None] > 0)
    return tb @ zb.T


def _wrong_norm(Z, T):   # normalises the visual rows by the text norms' mean
    Z = np.asarray(Z, float); T = np.asarray(T, float)
    nt = np.linalg.norm(T, axis=1)
    return np.maximum((T / nt[:, None]) @ Z.T / np.mean(nt), 0.0)


def _mean_not_rms(Z, T):
    return _orig["rectified_cosine"](Z, T).mean(axis=0)


def _no_sqrt(Z, T):
    m = _orig["rectified_cosine"](Z, T)
    return np.sum(m * m, axis=0) / m.shape[0]


def _upper_median(x):
    x = np.sort(np.asarray(x, float))
    return float(x[len(x) // 2])


def _mad_by_mean(x):
    x = np.asarray(x, float)
    return float(np.mean(np.abs(x - _orig["lower_median"](x))))


def _no_clamp(s, tau, eps):
    s = np.asarray(s, float)
    return (s - _orig["lower_median"](s)) / (_orig["mad"](s) + eps) / tau


def _tau_times(s, tau, eps):
    s = np.asarray(s, float)
    return np.maximum((s - _orig["lower_median"](s)) / (_orig["mad"](s) + eps), 0.0) * tau


def _eps_outside(s, tau, eps):
    s = np.asarray(s, float)
    return np.maximum((s - _orig["lower_median"](s)) / _orig["mad"](s) + eps, 0.0) / tau


def _fused_no_reward(a, b, lam):
    return np.maximum(np.asarray(a, float), np.asarray(b, float))


def _fused_min(a, b, lam):
    a = np.asarray(a, float); b = np.asarray(b, float)
    return np.minimum(a, b) + lam * np.sqrt(a * b)


def _fused_sum(a, b, lam):
    a = np.asarray(a, float); b = np.asarray(b, float)
    return np.maximum(a, b) + lam * (a * b)


def _topk_high_index(score, k, allowed=None):
    score = np.asarray(score, float)
    idx = np.arange(len(score))
    if allowed is not None:
        idx = idx[np.asarray(allowed, bool)]
    order = np.lexsort((-idx, -score[idx]))
    return np.sort(idx[order[:k]])


def _topk_ascending(score, k, allowed=None):
    return _orig["top_k"](-np.asarray(score, float), k, allowed)


def _count_floor(k1, ratio):
    return int(math.floor(float(np.float32(ratio)) * k1))


def _ratio_text_first(s_v, s_t, k1, ratio):
    kt = O.textual_count(k1, ratio)
    St = O.top_k(s_t, kt)
    rest = np.ones(len(s_t), bool); rest[St] = False
    return np.sort(np.concatenate([St, O.top_k(s_v, k1 - kt, rest)]))


def _ratio_not_disjoint(s_v, s_t, k1, ratio):
    kt = O.textual_count(k1, ratio)
    return np.unique(np.concatenate([O.top_k(s_v, k1 - kt), O.top_k(s_t, kt)]))


def _ratio_swapped(s_v, s_t, k1, ratio):
    return _orig["select_ratio"](s_t, s_v, k1, ratio)


def _softmax_over_queries(Q, K, scale=None):
    Q = np.asarray(Q, float); K = np.asarray(K, float)
    L, Hq, dh = Q.shape; K1, Hkv, _ = K.shape
    scale = 1 / math.sqrt(dh) if scale is None else scale
    A = np.empty((Hq, L, K1))
    for h in range(Hq):
        lg = Q[:, h] @ K[:, (h * Hkv) // Hq].T * scale
        e = np.exp(lg - lg.max(axis=0, keepdims=True))
        A[h] = e / e.sum(axis=0, keepdims=True)
    return A


def _gqa_modulo(Q, K, scale=None):
    Q = np.asarray(Q, float); K = np.asarray(K, float)
    L, Hq, dh = Q.shape; K1, Hkv, _ = K.shape
    scale = 1 / math.sqrt(dh) if scale is None else scale
    A = np.empty((Hq, L, K1))
    for h in range(Hq):
        lg = Q[:, h] @ K[:, h % Hkv].T * scale
        e = np.exp(lg - lg.max(axis=1, keepdims=True))
        A[h] = e / e.sum(axis=1, keepdims=True)
    return A


def _no_scale(Q, K, scale=None):
    return _orig["text_to_vision_attention"](Q, K, 1.0)


def _var_unbiased(A):
    A = np.asarray(A, float); K1 = A.shape[2]
    return (((A - A.mean(axis=2, keepdims=True)) ** 2).sum(axis=2) / (K1 - 1)).mean(axis=1)


def _var_over_queries(A):
    A = np.asarray(A, float)
    return A.var(axis=1).mean(axis=1)


def _std_not_var(A):
    A = np.asarray(A, float)
    return A.std(axis=2).mean(axis=1)


def _heads_lowest(u, n):
    return _orig["top_k"](-np.asarray(u, float), n)


def _mean_of_max(A, heads):
    A = np.asarray(A, float)
    return A[np.asarray(heads)].max(axis=1).mean(axis=0)


def _sum_not_mean(A, heads):
    A = np.asarray(A, float)
    return A[np.asarray(heads)].sum(axis=0).max(axis=0)


def _all_heads(A, heads):
    return np.asarray(A, float).mean(axis=0).max(axis=0)


def _gather_reversed(X, idx):
    return np.asarray(X)[np.asarray(idx)[::-1]]


def _decode_truncating(bits):
    return (np.asarray(bits, np.uint16).astype(np.int64) / 16384.0)



def _fps_generic(Z, pivots, k_d, *, use_pivots=True, setdist=np.minimum, pick="far_low", normalise=True):
    Z = np.asarray(Z, dtype=np.float64)
    N = len(Z)
    nz = np.sqrt((Z * Z).sum(1))
    U = np.divide(Z, nz[:, None], out=np.zeros_like(Z), where=nz[:, None] > 0) if normalise else Z
    cand = np.ones(N, dtype=bool)
    first = setdist is np.minimum
    dist = np.full(N, np.inf if first else -np.inf)
    for s in pivots:
        cand[s] = False
        if use_pivots:
            dist = setdist(dist, 1.0 - U @ U[s])
    picks, at = [], []
    for _ in range(k_d):
        idx = np.flatnonzero(cand)
        v = dist[idx]
        if pick == "far_low":
            j = idx[np.argmax(v)]
        elif pick == "far_high":
            j = idx[len(v) - 1 - np.argmax(v[::-1])]
        else:
            j = idx[np.argmin(v)]
        picks.append(int(j))
        at.append(dist[j])
        cand[j] = False
        dist = setdist(dist, 1.0 - U @ U[j])
    return np.array(picks, dtype=np.int64), np.array(at)


def _fps_ignores_pivots(Z, pivots, k_d):
    return _fps_generic(Z, pivots, k_d, use_pivots=False)


def _fps_max_not_min(Z, pivots, k_d):
    return _fps_generic(Z, pivots, k_d, setdist=np.maximum)


def _fps_tie_high(Z, pivots, k_d):
    return _fps_generic(Z, pivots, k_d, pick="far_high")


def _fps_nearest(Z, pivots, k_d):
    return _fps_generic(Z, pivots, k_d, pick="near")


def _fps_unnormalised(Z, pivots, k_d):
    return _fps_generic(Z, pivots, k_d, normalise=False)


def _diversity_floor(k1, rho):
    return int(np.floor(np.float32(rho) * k1))



def _cls_generic(q_cls, K_v, scale=None, *, scaled=True, reduce="mean", axis="tokens"):
    q = np.asarray(q_cls, dtype=np.float64)
    K = np.asarray(K_v, dtype=np.float64)
    N, H, dh = K.shape
    L = np.einsum("nhd,hd->hn", K, q) * (1.0 / np.sqrt(dh) if scaled else 1.0)
    if axis == "tokens":
        e = np.exp(L - L.max(axis=1, keepdims=True))
        A = e / e.sum(axis=1, keepdims=True)
    else:
        e = np.exp(L - L.max(axis=0, keepdims=True))
        A = e / e.sum(axis=0, keepdims=True)
    return A.sum(0) / H if reduce == "mean" else (A.sum(0) if reduce == "sum" else A.max(0))


def _cls_no_scale(q, K, scale=None):
    return _cls_generic(q, K, scaled=False)


def _cls_sum_heads(q, K, scale=None):
    return _cls_generic(q, K, reduce="sum")


def _cls_max_heads(q, K, scale=None):
    return _cls_generic(q, K, reduce="max")


def _cls_softmax_over_heads(q, K, scale=None):
    return _cls_generic(q, K, axis="heads")



_plain_attention = O.text_to_vision_attention


def _lse_ignored(Q, K, scale=None, lse_other=None):
    return _plain_attention(Q, K, scale)


def _ts_cos(s1, s2):
    s1, s2 = np.asarray(s1, float), np.asarray(s2, float)
    return (s1 * s2).sum(1) / (np.linalg.norm(s1, axis=1) * np.linalg.norm(s2, axis=1))


def _ts_unnormalised(s1, s2):
    return 1.0 - (np.asarray(s1, float) * np.asarray(s2, float)).sum(1)


def _head_attention_max(A):
    return np.asarray(A, float).max(axis=1)


MUTANTS = {
    "cos_no_relu": ("rectified_cosine", _no_relu),
    "cos_wrong_norm": ("rectified_cosine", _wrong_norm),
    "st_mean_not_rms": ("textual_relevance", _mean_not_rms),
    "st_no_sqrt": ("textual_relevance", _no_sqrt),
    "upper_median": ("lower_median", _upper_median),
    "mad_by_mean": ("mad", _mad_by_mean),
    "norm_no_clamp": ("robust_normalise", _no_clamp),
    "norm_tau_times": ("robust_normalise", _tau_times),
    "norm_eps_outside": ("robust_normalise", _eps_outside),
    "fused_no_reward": ("fused_score", _fused_no_reward),
    "fused_min": ("fused_score", _fused_min),
    "fused_product_no_sqrt": ("fused_score", _fused_sum),
    "topk_tie_high_index": ("top_k", _topk_high_index),
    "topk_ascending": ("top_k", _topk_ascending),
    "count_floor": ("textual_count", _count_floor),
    "ratio_text_first": ("select_ratio", _ratio_text_first),
    "ratio_not_disjoint": ("select_ratio", _ratio_not_disjoint),
    "ratio_swapped_signals": ("select_ratio", _ratio_swapped),
    "softmax_over_queries": ("text_to_vision_attention", _softmax_over_queries),
    "gqa_modulo": ("text_to_vision_attention", _gqa_modulo),
    "no_softmax_scale": ("text_to_vision_attention", _no_scale),
    "var_unbiased": ("head_variance", _var_unbiased),
    "var_over_queries": ("head_variance", _var_over_queries),
    "std_not_var": ("head_variance", _std_not_var),
    "heads_lowest_variance": ("select_heads", _heads_lowest),
    "p_mean_of_max": ("token_scores", _mean_of_max),
    "p_sum_not_mean": ("token_scores", _sum_not_mean),
    "p_all_heads": ("token_scores", _all_heads),
    "gather_reversed": ("gather_rows", _gather_reversed),
    "bf16_decode_wrong": ("bf16_bits_to_f64", _decode_truncating),
    "fps_ignores_pivots": ("farthest_point_sampling", _fps_ignores_pivots),
    "fps_max_not_min": ("farthest_point_sampling", _fps_max_not_min),
    "fps_tie_high_index": ("farthest_point_sampling", _fps_tie_high),
    "fps_nearest": ("farthest_point_sampling", _fps_nearest),
    "fps_unnormalised": ("farthest_point_sampling", _fps_unnormalised),
    "diversity_floor": ("diversity_count", _diversity_floor),
    "cls_no_scale": ("cls_saliency", _cls_no_scale),
    "cls_sum_heads": ("cls_saliency", _cls_sum_heads),
    "cls_max_heads": ("cls_saliency", _cls_max_heads),
    "cls_softmax_over_heads": ("cls_saliency", _cls_softmax_over_heads),
    "lse_other_ignored": ("text_to_vision_attention", _lse_ignored),
    "ts_cos_not_distance": ("textual_sensitivity", _ts_cos),
    "ts_unnormalised": ("textual_sensitivity", _ts_unnormalised),
    "head_attention_max": ("head_visual_attention", _head_attention_max),
}


@pytest.mark.parametrize("name", sorted(MUTANTS))
def test_some_pin_catches_mutant(name, monkeypatch):
    attr, fn = MUTANTS[name]
    monkeypatch.setattr(O, attr, fn)
    caught = []
    for pin in oracle_pins.ALL_PINS:
        try:
            pin()
        except Exception:           # an assertion or a shape error both count as caught
            caught.append(pin.__name__)
    assert caught, f"mutant {name} of {attr} passed every pin"
