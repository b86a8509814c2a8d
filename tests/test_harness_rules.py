"""The GPU parity checker itself, on the CPU: it accepts the oracle's own results, accepts a
different choice inside a near-tie band, and rejects a kept set that drops a candidate above
the band or keeps one below it. The "GPU" results here are the oracle's, with one planted
mistake per case."""
import dataclasses

import numpy as np
import pytest

import oracle.trevs_oracle as O
from tests import gpu_harness as H
from workloads import synth


def _fake_run(w, ref):
    """A DeviceRun holding the oracle's results in the GPU layouts."""
    cat = lambda key, stage, dtype=None: np.concatenate(
        [np.asarray(r[stage][key], dtype) for r in ref]) if ref else np.zeros(0)
    return H.DeviceRun(
        s_t=cat("s_t", "pre", np.float32), s_fused=None,
        kept1=cat("kept", "pre", np.int32), Z_out=np.concatenate([r["pre"]["Z_out"] for r in ref]),
        u=np.stack([np.asarray(r["in"]["u"], np.float32) for r in ref]),
        heads=np.stack([np.asarray(r["in"]["heads"], np.int32) for r in ref]),
        p=cat("p", "in", np.float32), kept2=cat("kept", "in", np.int32),
        hidden_out=np.concatenate([r["in"]["hidden_out"] for r in ref]),
        K_out=np.concatenate([r["in"]["K_out"] for r in ref]),
        V_out=np.concatenate([r["in"]["V_out"] for r in ref]))


@pytest.fixture(scope="module")
def case():
    w = synth.small_case(seed_cfg=97)
    return w, O.run_workload(w)


def test_oracle_results_pass(case):
    w, ref = case
    t = H.check_workload(w, _fake_run(w, ref), ref)
    assert t.stage1_exact + t.stage1_near_ties == w.B


def test_dropped_stage1_token_fails(case):
    w, ref = case
    g = _fake_run(w, ref)
    # request 0: replace its best textual token by the worst token outside the kept set
    kt = O.textual_count(w.reqs[0].k1, w.reqs[0].ratio)
    assert kt > 0
    s_t = ref[0]["pre"]["s_t"]
    kept = list(ref[0]["pre"]["kept"])
    sv = w.s_v[:w.reqs[0].n].astype(np.float64)
    Sv = set(O.top_k(sv, w.reqs[0].k1 - kt).tolist())
    best = max((i for i in kept if i not in Sv), key=lambda i: s_t[i])
    worst = min((i for i in range(w.reqs[0].n) if i not in kept), key=lambda i: s_t[i])
    kept[kept.index(best)] = worst
    g.kept1[:w.reqs[0].k1] = np.sort(kept)
    g.Z_out[:w.reqs[0].k1] = w.Z[:w.reqs[0].n][np.sort(kept)]
    with pytest.raises(AssertionError):
        H.check_workload(w, g, ref)


def test_dropped_stage2_token_fails(case):
    w, ref = case
    g = _fake_run(w, ref)
    b = 0
    k1, k2 = w.reqs[b].k1, w.reqs[b].k2
    p = ref[b]["in"]["p"]
    kept = list(ref[b]["in"]["kept"])
    out = [i for i in range(k1) if i not in kept]
    kept[int(np.argmax(p[kept]))] = min(out, key=lambda i: p[i])
    g.kept2[:k2] = np.sort(kept)
    with pytest.raises(AssertionError):
        H.check_workload(w, g, ref)


def test_band_rule():
    s = np.array([9.0, 5.0, 4.0, 4.0 * (1 + 5e-5), 4.0 * (1 - 5e-5), 1.0])
    # k = 3: 9 and 5 are above the band; 4(1+5e-5), 4 and 4(1-5e-5) are inside; 1 is below
    assert H.check_band([0, 1, 3], s, 3) == 3
    H.check_band([0, 1, 2], s, 3)      # another choice inside the band
    H.check_band([0, 1, 4], s, 3)
    with pytest.raises(AssertionError):
        H.check_band([0, 2, 3], s, 3)  # drops 5, which is above the band
    with pytest.raises(AssertionError):
        H.check_band([0, 1, 5], s, 3)  # keeps 1, which is below the band
    H.check_band([0, 1, 5], s, 3, below=False)
    allowed = np.array([True, False, True, True, True, True])
    with pytest.raises(AssertionError):
        H.check_band([1, 2, 3], s, 3, allowed)   # keeps a token that is not a candidate


def test_head_near_tie_checks_p_over_gpu_heads():
    # two heads with exactly equal u: either may be kept; p must then follow the GPU's H*
    w = synth.small_case(seed_cfg=98, n=(90,), m=(6,), k1=(40,), ratio=(0.5,), k2=(10,), hq=4, hkv=2,
                         n_keep_heads=1)
    Q = w.Q.copy()
    # heads 0 and 1 share KV head 0: the same (sharpened, x4 exactly) queries give both the
    # same attention and the largest variance
    q0 = O.bf16_bits_to_f64(Q[:, 0, :]) * 4.0
    Q[:, 0, :] = Q[:, 1, :] = synth.f32_to_bf16_bits(q0.astype(np.float32))
    w = dataclasses.replace(w, Q=Q)
    ref = O.run_workload(w)
    u = ref[0]["in"]["u"]
    assert u[0] == u[1] and ref[0]["in"]["heads"][0] == 0, u
    g = _fake_run(w, ref)
    g.heads[0, 0] = 1 - ref[0]["in"]["heads"][0]   # the other head of the tie
    H.check_workload(w, g, ref)                    # identical attention: same p, same set
    g.p[:] = g.p * 1.01                            # p off by 1%: rejected
    with pytest.raises(AssertionError):
        H.check_workload(w, g, ref)
