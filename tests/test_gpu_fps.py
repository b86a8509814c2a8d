"""Farthest point sampling (Sec. 3.1 context preservation) on the GPU against the oracle.

The pivots are inputs shared by both sides, so a near-tie in the stage-1 rule cannot hide
an FPS error. The GPU's draw sequence is checked in fp64 along its own prefix: every draw
must be a farthest candidate within TOL, its reported distance must match, and the
sequence must equal the oracle's until the first step whose two best candidates are
within TOL of each other (a near tie, counted). TOL covers the fp32 cosines of bf16 rows:
rounding of a d' = 4096 dot product and of the two norms stays near 1e-6.
"""
import numpy as np
import pytest

import oracle.trevs_oracle as O
from workloads import synth

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")
if not torch.cuda.is_available():   # pragma: no cover - CPU container
    pytest.skip("needs a CUDA GPU", allow_module_level=True)

from paper_2609_37581_gb300 import trevs as T  # noqa: E402
from tests import gpu_harness as H  # noqa: E402

TOL = H.FPS_TOL
_unit_rows = H.unit_rows
check_method_stage1 = H.check_method_stage1


def check_draws(Z_bits, pivots, picks, dist, k_d):
    """Returns 1 if the sequence left the oracle's at a near tie, else 0 (then identical)."""
    U = _unit_rows(Z_bits)
    N = len(U)
    cand = np.ones(N, dtype=bool)
    cur = np.full(N, np.inf)
    for s in pivots:
        if 0 <= s < N:
            cand[s] = False
            cur = np.minimum(cur, 1.0 - U @ U[s])
    ref, _ = O.farthest_point_sampling(O.bf16_bits_to_f64(Z_bits), [s for s in pivots if 0 <= s < N], k_d)
    assert len(picks) == k_d
    diverged = False
    for t, g in enumerate(picks):
        assert 0 <= g < N and cand[g], f"draw {t}: {g} is not a remaining candidate"
        best = cur[cand].max()
        assert cur[g] >= best - TOL, f"draw {t}: {g} at {cur[g]!r}, the farthest is at {best!r}"
        if np.isfinite(cur[g]):
            assert abs(dist[t] - cur[g]) <= TOL, f"draw {t}: distance {dist[t]!r}, fp64 {cur[g]!r}"
        else:
            assert np.isinf(dist[t])
        if not diverged and g != ref[t]:
            top = np.sort(cur[cand])[::-1]
            near = len(top) > 1 and np.all(np.isfinite(top[:2])) and top[0] - top[1] <= TOL
            assert near, f"draw {t}: {g} instead of {ref[t]} without a near tie"
            diverged = True
        cand[g] = False
        cur = np.minimum(cur, 1.0 - U @ U[g])
    return int(diverged)


def run_fps(Z_bits, pivots, k_d, pool=0):
    N, d = Z_bits.shape
    Z = H.dev_bf16(Z_bits)
    piv = torch.tensor(np.asarray(pivots, np.int32), device="cuda") if len(pivots) else None
    picks = torch.full((max(k_d, 1),), -7, dtype=torch.int32, device="cuda")
    dist = torch.full((max(k_d, 1),), -7.0, dtype=torch.float32, device="cuda")
    ws = T.workspace(T.trevs_pre_llm_fps_workspace_size(N, len(pivots), d))
    T.trevs_pre_llm_fps(Z, piv, k_d, picks, dist, pool=pool, ws=ws)
    T.workspace_status(ws)
    return picks.cpu().numpy()[:k_d], dist.cpu().numpy()[:k_d]


def _llava_request():
    """A LLaVA-1.5-shaped request and its Eq. 6-7 pivots for K1 = 64 at K_r:K_d = 3:1."""
    w = synth.llava15_single()
    r = O.pre_llm_request(w.Z, w.T, w.s_v, 64, 0.5, "fused", diversity=0.25)
    return w.Z, list(r["pivots"]), len(r["fps"])


def _clusters(seed, n, d, k, noise=0.3, zero_rows=()):
    rng = np.random.default_rng(seed)
    centers = rng.standard_normal((k, d))
    Z = centers[rng.integers(0, k, size=n)] + noise * rng.standard_normal((n, d))
    Z[list(zero_rows)] = 0.0
    return synth.f32_to_bf16_bits(Z.astype(np.float32))


@pytest.mark.parametrize("pool", [0, 1, 17, 128])
def test_fps_llava_request(pool):
    Z, piv, k_d = _llava_request()
    assert (len(piv), k_d) == (48, 16)
    picks, dist = run_fps(Z, piv, k_d, pool)
    check_draws(Z, piv, picks, dist, k_d)


def _hypercube_rows(copies, repeat, seed):
    """Vertices of {+1, -1}^8, each coordinate repeated `repeat` times, `copies` of each
    vertex, rows shuffled. With repeat a power of four the row norm is a power of two, so
    every cosine (1 - hamming / 4) is exact in fp32 as well: the draws, ties included,
    have exactly one correct answer."""
    v = np.array([[1 - 2 * ((k >> c) & 1) for c in range(8)] for k in range(256)], np.float32)
    Zf = np.repeat(np.tile(v, (copies, 1)), repeat, axis=1)
    Zf = Zf[np.random.default_rng(seed).permutation(len(Zf))]
    return synth.f32_to_bf16_bits(Zf)


@pytest.mark.parametrize("pool", [0, 3, 128])
def test_fps_exact_distances(pool):
    Z = _hypercube_rows(3, 128, 29)      # 768 rows, d' = 1024
    piv = [0, 1, 2, 3, 4]
    picks, dist = run_fps(Z, piv, 300, pool)
    ref, ref_d = O.farthest_point_sampling(O.bf16_bits_to_f64(Z), piv, 300)
    np.testing.assert_array_equal(picks, ref)
    np.testing.assert_array_equal(dist, ref_d.astype(np.float32))


def test_fps_no_pivots():
    Z = _clusters(7, 333, 200, 6)        # d' = 200: a ragged last 64-column chunk
    picks, dist = run_fps(Z, [], 25)
    assert picks[0] == 0 and np.isinf(dist[0])
    check_draws(Z, [], picks, dist, 25)


@pytest.mark.parametrize("n,d,k_r", [(129, 64, 9), (300, 200, 37), (1, 8, 0)])
def test_fps_every_candidate(n, d, k_r):
    Z = _clusters(n, n, d, 5)
    rng = np.random.default_rng(n)
    piv = sorted(rng.choice(n, size=k_r, replace=False).tolist())
    picks, dist = run_fps(Z, piv, n - k_r)
    assert sorted(picks) == [i for i in range(n) if i not in piv]
    check_draws(Z, piv, picks, dist, n - k_r)


def test_fps_zero_rows_tie_to_lower_index():
    # rows in the positive orthant have cosines > 0 with each other (distance < 1); zero
    # rows sit at distance exactly 1 from everything, so they come first, in index order
    rng = np.random.default_rng(11)
    Zf = np.abs(rng.standard_normal((200, 96))).astype(np.float32)
    zeros = [3, 50, 51, 120, 199]
    Zf[zeros] = 0.0
    Z = synth.f32_to_bf16_bits(Zf)
    piv = [0, 10, 20]
    picks, dist = run_fps(Z, piv, 12)
    assert list(picks[:5]) == zeros and np.all(dist[:5] == 1.0)
    check_draws(Z, piv, picks, dist, 12)


@pytest.mark.parametrize("k_r", [257, 600])
def test_fps_pivots_beyond_one_pass(k_r):
    # more than 256 pivots: the distances take one pass of the contraction per 256 pivot
    # columns, each later pass keeping the max cosine
    Z = _clusters(31 + k_r, 3000, 256, 60, noise=0.5)
    rng = np.random.default_rng(k_r)
    piv = rng.choice(3000, size=k_r, replace=False).tolist()
    picks, dist = run_fps(Z, piv, 50)
    check_draws(Z, piv, picks, dist, 50)


def test_fps_exact_distances_beyond_one_pass():
    # 300 pivots over the exact-cosine hypercube rows: every draw and distance has one answer
    Z = _hypercube_rows(3, 128, 37)
    piv = list(range(0, 600, 2))
    picks, dist = run_fps(Z, piv, 100)
    ref, ref_d = O.farthest_point_sampling(O.bf16_bits_to_f64(Z), piv, 100)
    np.testing.assert_array_equal(picks, ref)
    np.testing.assert_array_equal(dist, ref_d.astype(np.float32))


def test_fps_large_request_and_many_pivots():
    # above 4096 rows the pool is chosen with the keys in memory
    Z = _clusters(13, 5000, 512, 40, noise=0.5)
    rng = np.random.default_rng(17)
    piv = rng.choice(5000, size=256, replace=False).tolist()
    picks, dist = run_fps(Z, piv, 64)
    check_draws(Z, piv, picks, dist, 64)


def test_fps_llava_next_shape():
    # K1 = 320 at 3:1 on a 2,880-token request: 240 pivots, 80 draws
    rng = np.random.default_rng(19)
    Z = synth.f32_to_bf16_bits(rng.standard_normal((2880, 4096)).astype(np.float32))
    piv = sorted(rng.choice(2880, size=240, replace=False).tolist())
    picks, dist = run_fps(Z, piv, 80)
    check_draws(Z, piv, picks, dist, 80)


def test_fps_pivot_outside_range_is_a_zero_row():
    Z = _clusters(23, 400, 128, 8)
    picks, dist = run_fps(Z, [5, 400, -3, 77], 20)
    # the documented reading, restated for the oracle: one zero pivot row appended
    Zz = np.vstack([Z, np.zeros((1, Z.shape[1]), np.uint16)])
    check_draws(Zz, [5, 77, 400], picks, dist, 20)


# ------------------------------------------------------------------ the batched Method path


@pytest.mark.parametrize("mode", ["fused", "ratio"])
@pytest.mark.parametrize("rho", [0.25, 0.5, 1.0])
def test_method_path_small_ragged(mode, rho):
    w = synth.small_case()
    m = T.SELECT_FUSED if mode == "fused" else T.SELECT_RATIO
    g, ws = H.run_gpu(w, m, params=T.default_params(m, diversity=rho), stages="pre")
    T.workspace_status(ws)
    exact, near = check_method_stage1(w, g, mode, rho)
    assert exact + near == sum(1 for r in w.reqs if r.k1 > 0)


def test_method_path_llava_batch32_both_stages():
    # the paper's Method settings (fused score, K_r:K_d = 3:1) on the 32 x 576 batch, both
    # stages through trevs_prune_varlen (the draws run beside stage 2)
    w = synth.llava15_batch32()
    g, ws = H.run_gpu(w, T.SELECT_FUSED, params=T.default_params(T.SELECT_FUSED, diversity=0.25), reps=2)
    T.workspace_status(ws)
    exact, near = check_method_stage1(w, g, "fused", 0.25)
    # six of these requests have a draw whose two best candidates are within 2e-6 in fp64,
    # about the size of an fp32 cosine's rounding: those may leave the oracle's sequence
    assert exact + near == w.B and exact >= w.B - 8, (exact, near)
    ref = O.run_workload(w, "fused", stage1=False)
    H.check_workload(w, g, ref, "fused")


@pytest.mark.parametrize("mode", ["fused", "ratio"])
def test_method_path_k1_1024(mode):
    # the Method settings at K1 = 1024 (768 pivots and 256 draws, K_r:K_d = 3:1) on requests
    # shaped like the long-video batch but narrower (d' = 256, so that the oracle stays quick)
    w = synth.small_case(seed_cfg=170, n=(6000, 4096), m=(128, 60), d=256, k1=(1024, 700),
                         ratio=(0.5, 0.5), k2=(0, 0), planted=0.02)
    m = T.SELECT_FUSED if mode == "fused" else T.SELECT_RATIO
    g, ws = H.run_gpu(w, m, params=T.default_params(m, diversity=0.25), stages="pre")
    T.workspace_status(ws)
    exact, near = check_method_stage1(w, g, mode, 0.25)
    assert exact + near == w.B
