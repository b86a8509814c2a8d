"""Runs a synthetic workload through the C ABI on the GPU and compares it with the oracle.

Comparison rules (tolerances follow from fp32 accumulation of bf16 products):
  * float scores (s^t, fused s, u_h, p_i): |gpu - oracle| <= RTOL * |oracle| + ATOL;
  * kept index sets: identical, unless the oracle's K-th and (K+1)-th scores differ by
    less than NEAR_TIE relative. Such near-ties are counted, and the GPU set must then
    equal the oracle's outside the tie band: every candidate whose oracle score lies above
    the K-th score by more than NEAR_TIE relative is kept, none below it by more than
    NEAR_TIE is, and the set holds exactly K distinct valid indices;
  * at a near tie on the head variances the GPU's H* must pass the same band rule, and the
    token scores and the stage-2 kept set are then checked against the oracle's Eq. 9 over
    the GPU's own H*;
  * gathered / compacted rows: bit-exact copies of the rows the GPU kept.
"""
from __future__ import annotations

import dataclasses

import numpy as np

import oracle.trevs_oracle as O
from workloads.device import DeviceRun, build_batches, collect, dev_bf16, dev_f32, host_u16, run_gpu  # noqa: F401

RTOL = 1e-3
ATOL_ST = 1e-6     # s^t is a mean of squares of cosines: fp32 cosine error ~1e-7 absolute
ATOL_FUSED = 1e-4  # fused scores near 0 are (s - Med) / MAD with fp32 Med and MAD
ATOL_P = 1e-7      # attention probabilities
NEAR_TIE = 1e-4
FPS_TOL = 5e-5     # farthest point sampling: fp32 cosines of bf16 rows err near 1e-6


# ------------------------------------------------------------------ comparisons


def assert_close(gpu, ref, rtol, atol, what):
    gpu = np.asarray(gpu, np.float64)
    ref = np.asarray(ref, np.float64)
    assert gpu.shape == ref.shape, (what, gpu.shape, ref.shape)
    err = np.abs(gpu - ref)
    bad = err > atol + rtol * np.abs(ref)
    if bad.any():
        i = int(np.argmax(err - (atol + rtol * np.abs(ref))))
        raise AssertionError(f"{what}: {int(bad.sum())} of {gpu.size} outside tolerance; worst at {i}: "
                             f"gpu {gpu.flat[i]!r} oracle {ref.flat[i]!r}")


def boundary_gap(scores, k, allowed=None):
    """Relative gap between the oracle's k-th and (k+1)-th scores (inf if no (k+1)-th)."""
    s = np.asarray(scores, np.float64)
    if allowed is not None:
        s = s[np.asarray(allowed, bool)]
    if k <= 0 or k >= len(s):
        return np.inf
    top = np.sort(s)[::-1]
    a, b = top[k - 1], top[k]
    den = max(abs(a), abs(b))
    return 0.0 if den == 0 else abs(a - b) / den


def _rel(a, b):
    den = np.maximum(np.abs(a), np.abs(b))
    return np.divide(np.abs(a - b), den, out=np.zeros_like(den, dtype=np.float64), where=den > 0)


def check_band(kept, scores, k, allowed=None, what="", below=True):
    """The band rule at a near tie: `kept` (indices) holds every candidate whose oracle score
    exceeds the oracle's k-th score by more than NEAR_TIE relative and (with `below`) no
    candidate that falls short of it by more than NEAR_TIE; only candidates inside the band
    may differ from the oracle's set. Returns the number of candidates inside the band."""
    s = np.asarray(scores, np.float64)
    cand = np.ones(len(s), bool) if allowed is None else np.asarray(allowed, bool).copy()
    kept = np.asarray(kept, np.int64)
    mask = np.zeros(len(s), bool)
    mask[kept] = True
    assert not (mask & ~cand).any(), f"{what}: kept an index that is not a candidate"
    if k <= 0:
        assert not (mask & cand).any(), f"{what}: kept a candidate with k = 0"
        return 0
    tau = np.sort(s[cand])[::-1][k - 1]
    far = _rel(s, tau) > NEAR_TIE
    above = cand & far & (s > tau)
    under = cand & far & (s < tau)
    missing = np.flatnonzero(above & ~mask)
    assert missing.size == 0, (f"{what}: {missing.size} candidates above the tie band dropped, "
                               f"first {int(missing[0])} at {s[missing[0]]!r} (k-th {tau!r})")
    if below:
        extra = np.flatnonzero(under & mask)
        assert extra.size == 0, (f"{what}: {extra.size} candidates below the tie band kept, "
                                 f"first {int(extra[0])} at {s[extra[0]]!r} (k-th {tau!r})")
    return int((cand & ~far).sum())


@dataclasses.dataclass
class Tally:
    requests: int = 0
    stage1_near_ties: int = 0
    stage2_near_ties: int = 0
    stage1_exact: int = 0
    stage2_exact: int = 0


def check_workload(w, g: DeviceRun, ref, mode="ratio", tally: Tally | None = None, params=None):
    """Element-wise comparison of one GPU run with the oracle, request by request."""
    tally = tally or Tally()
    params = params or {}
    n_off, k1_off, k2_off, l_off = w.offsets("n"), w.offsets("k1"), w.offsets("k2"), w.offsets("l")
    for b, r in enumerate(w.reqs):
        tally.requests += 1
        res = ref[b]
        # ---- stage 1
        if "pre" in res:
            pre = res["pre"]
            st = g.s_t[n_off[b]:n_off[b + 1]]
            assert_close(st, pre["s_t"], RTOL, ATOL_ST, f"req {b} s_t")
            kept = g.kept1[k1_off[b]:k1_off[b + 1]]
            assert len(kept) == r.k1
            assert np.all(np.diff(kept) > 0), f"req {b}: stage-1 indices not strictly ascending"
            assert kept.size == 0 or (kept[0] >= 0 and kept[-1] < r.n)
            if mode == "ratio":
                kt = O.textual_count(r.k1, r.ratio)
                sv = w.s_v[n_off[b]:n_off[b + 1]].astype(np.float64)
                Sv = O.top_k(sv, r.k1 - kt)
                rest = np.ones(r.n, bool)
                rest[Sv] = False
                # saliency decisions compare the same fp32 inputs on both sides: exact;
                # only the computed textual scores carry a near-tie band
                near = boundary_gap(pre["s_t"], kt, rest) < NEAR_TIE
                if near:
                    kept_set = set(kept.tolist())
                    assert set(Sv.tolist()) <= kept_set, f"req {b}: saliency side S_v not kept"
                    St = np.array(sorted(kept_set - set(Sv.tolist())), np.int64)
                    assert len(St) == kt
                    check_band(St, pre["s_t"], kt, rest, f"req {b} stage-1 textual side")
            else:
                assert_close(g.s_fused[n_off[b]:n_off[b + 1]], pre["s_fused"], RTOL, ATOL_FUSED, f"req {b} fused")
                near = boundary_gap(pre["s_fused"], r.k1) < NEAR_TIE
                if near:
                    check_band(kept, pre["s_fused"], r.k1, None, f"req {b} stage-1 fused")
            if near:
                tally.stage1_near_ties += 1
            else:
                np.testing.assert_array_equal(kept, pre["kept"], err_msg=f"req {b} stage-1 kept set")
                tally.stage1_exact += 1
            # gathered rows are exact copies of the rows the GPU kept
            Zb = w.Z[n_off[b]:n_off[b + 1]]
            np.testing.assert_array_equal(g.Z_out[k1_off[b]:k1_off[b + 1]], Zb[kept], err_msg=f"req {b} Z_out")
        # ---- stage 2
        if "in" in res:
            inn = res["in"]
            assert_close(g.u[b], inn["u"], RTOL, 1e-9, f"req {b} u")
            heads = g.heads[b]
            head_near = boundary_gap(inn["u"], w.n_keep_heads) < NEAR_TIE
            kept2 = g.kept2[k2_off[b]:k2_off[b + 1]]
            assert len(kept2) == r.k2
            assert np.all(np.diff(kept2) > 0), f"req {b}: stage-2 indices not strictly ascending"
            assert kept2.size == 0 or (kept2[0] >= 0 and kept2[-1] < r.k1)
            p_ref = inn["p"]
            if head_near:
                # H* may differ inside the band; Eq. 9 is then checked over the GPU's own H*
                assert len(heads) == w.n_keep_heads and np.all(np.diff(heads) > 0), f"req {b}: bad H*"
                check_band(heads, inn["u"], w.n_keep_heads, None, f"req {b} H*")
                lse = None if w.lse_other is None else w.lse_other[:, l_off[b]:l_off[b + 1]]
                A = O.text_to_vision_attention(O.bf16_bits_to_f64(w.Q[l_off[b]:l_off[b + 1]]),
                                               O.bf16_bits_to_f64(w.K[k1_off[b]:k1_off[b + 1]]), lse_other=lse)
                p_ref = O.token_scores(A, heads)
            else:
                np.testing.assert_array_equal(heads, inn["heads"], err_msg=f"req {b} heads")
            assert_close(g.p[k1_off[b]:k1_off[b + 1]], p_ref, RTOL, ATOL_P, f"req {b} p")
            p_near = boundary_gap(p_ref, r.k2) < NEAR_TIE
            if p_near:
                check_band(kept2, p_ref, r.k2, None, f"req {b} stage-2 kept set")
            else:
                np.testing.assert_array_equal(kept2, O.top_k(p_ref, r.k2), err_msg=f"req {b} stage-2 kept set")
            if head_near or p_near:
                tally.stage2_near_ties += 1
            else:
                tally.stage2_exact += 1
            Hb = w.hidden[k1_off[b]:k1_off[b + 1]]
            Kb = w.K[k1_off[b]:k1_off[b + 1]]
            Vb = w.V[k1_off[b]:k1_off[b + 1]]
            np.testing.assert_array_equal(g.hidden_out[k2_off[b]:k2_off[b + 1]], Hb[kept2], err_msg=f"req {b} hidden")
            np.testing.assert_array_equal(g.K_out[k2_off[b]:k2_off[b + 1]], Kb[kept2], err_msg=f"req {b} K_out")
            np.testing.assert_array_equal(g.V_out[k2_off[b]:k2_off[b + 1]], Vb[kept2], err_msg=f"req {b} V_out")
    return tally


# ------------------------------------------------------------------ diversity draws (Sec. 3.1)


def unit_rows(Z_bits):
    Z = O.bf16_bits_to_f64(Z_bits)
    nz = np.sqrt((Z * Z).sum(1))
    return np.divide(Z, nz[:, None], out=np.zeros_like(Z), where=nz[:, None] > 0)


def check_draw_set(Z_bits, pivots, draws):
    """`draws` (a set) is what K_d farthest-point steps from `pivots` can yield: replayed
    greedily, every step's farthest member of the set is within FPS_TOL of the farthest row."""
    U = unit_rows(Z_bits)
    cand = np.ones(len(U), dtype=bool)
    cur = np.full(len(U), np.inf)
    for s in pivots:
        cand[s] = False
        cur = np.minimum(cur, 1.0 - U @ U[s])
    left = set(int(x) for x in draws)
    while left:
        g = max(left, key=lambda i: (cur[i], -i))
        best = cur[cand].max()
        assert cur[g] >= best - FPS_TOL, f"draw {g} at {cur[g]!r}, the farthest is at {best!r}"
        left.remove(g)
        cand[g] = False
        cur = np.minimum(cur, 1.0 - U @ U[g])


def check_method_stage1(w, g, mode, rho):
    """Stage 1 with diversity draws against the oracle, request by request. Returns
    (exact, near): near counts requests that left the oracle's set at a near tie, either of
    the rule at K_r (then every candidate above the rule's tie band must still be kept) or of
    the draws (then the pivots must match and the draws form a valid farthest-point set)."""
    n_off, m_off, k1_off = w.offsets("n"), w.offsets("m"), w.offsets("k1")
    exact = near = 0
    for b, r in enumerate(w.reqs):
        Zb = w.Z[n_off[b]:n_off[b + 1]]
        ref = O.pre_llm_request(Zb, w.T[m_off[b]:m_off[b + 1]], w.s_v[n_off[b]:n_off[b + 1]], r.k1, r.ratio,
                                mode, diversity=rho)
        kept = g.kept1[k1_off[b]:k1_off[b + 1]]
        assert len(kept) == r.k1
        if r.k1 == 0:
            continue
        assert np.all(np.diff(kept) > 0) and kept[0] >= 0 and kept[-1] < r.n, f"req {b}: bad kept set"
        np.testing.assert_array_equal(g.Z_out[k1_off[b]:k1_off[b + 1]], Zb[kept])
        if list(kept) == list(ref["kept"]):
            exact += 1
            continue
        kd = O.diversity_count(r.k1, rho)
        kr = r.k1 - kd
        piv = list(ref.get("pivots", ref["kept"]))
        if not set(piv) <= set(kept.tolist()):
            sv = w.s_v[n_off[b]:n_off[b + 1]].astype(np.float64)
            if mode == "fused":
                gap = boundary_gap(ref["s_fused"], kr)
            else:
                kt = O.textual_count(kr, r.ratio)
                Sv = O.top_k(sv, kr - kt)
                rest = np.ones(r.n, bool)
                rest[Sv] = False
                gap = min(boundary_gap(sv, kr - kt), boundary_gap(ref["s_t"], kt, rest))
            assert gap < NEAR_TIE, f"req {b}: pivots differ without a near tie (gap {gap})"
            # the pivots are a subset of the kept set: every candidate above the tie band of
            # the rule is kept (below the band a token may still be a draw)
            if mode == "fused":
                check_band(kept, ref["s_fused"], kr, None, f"req {b} pivots (fused)", below=False)
            else:
                Sv_set = set(Sv.tolist())
                check_band(sorted(Sv_set & set(kept.tolist())), sv, kr - kt, None,
                           f"req {b} pivots (saliency side)", below=False)
                check_band(sorted(set(kept.tolist()) - Sv_set), ref["s_t"], kt, rest,
                           f"req {b} pivots (textual side)", below=False)
        else:
            check_draw_set(Zb, piv, sorted(set(kept.tolist()) - set(piv)))
        near += 1
    return exact, near
