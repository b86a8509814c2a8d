"""GPU path (through the C ABI) against the oracle, element by element, on seeded inputs."""
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


def _run_and_check(w, mode="ratio", **params):
    m = T.SELECT_FUSED if mode == "fused" else T.SELECT_RATIO
    g, ws = H.run_gpu(w, m, T.default_params(m, **params))
    ref = O.run_workload(w, mode=mode, **params)
    tally = H.check_workload(w, g, ref, mode)
    # tickets must be back at zero after a completed call
    assert int(ws[:1024].view(torch.int32).abs().sum()) == 0
    return tally, g


def test_small_ragged_ratio():
    w = synth.small_case()
    tally, _ = _run_and_check(w)
    assert tally.stage1_exact + tally.stage1_near_ties == w.B


def test_small_ragged_fused():
    w = synth.small_case(seed_cfg=91)
    _run_and_check(w, "fused")


def test_small_ragged_fused_nondefault_params():
    w = synth.small_case(seed_cfg=92)
    _run_and_check(w, "fused", tau_v=2.0, tau_t=0.5, lam=0.25, eps=1e-3)


def test_edge_sizes_stage1():
    # K1 = N, K1 = 0, N = 0, M = 1, M = 256 (maximum), N not a multiple of the 64-row tile,
    # d not a multiple of the 64-column chunk, textual ratio 0 and 1
    w = synth.small_case(seed_cfg=93, n=(65, 64, 0, 5, 130), m=(1, 3, 0, 256, 2), d=72,
                         k1=(65, 0, 0, 1, 33), ratio=(0.5, 0.5, 0.5, 1.0, 0.0), k2=(0, 0, 0, 0, 0))
    for mode in ("ratio", "fused"):
        m = T.SELECT_FUSED if mode == "fused" else T.SELECT_RATIO
        g, _ = H.run_gpu(w, m, stages="pre")
        H.check_workload(w, g, O.run_workload(w, mode=mode, stage2=False), mode)


def test_edge_sizes_stage2():
    # K2 = K1, K2 = 0, K1 = 1, L = 1, one KV head for eight query heads, |H*| = Hq
    for nkh in (3, 8):
        w = synth.small_case(seed_cfg=95, n=(70, 9, 40), m=(1, 3, 17), d=64, hq=8, hkv=1, n_keep_heads=nkh,
                             k1=(65, 1, 33), ratio=(0.5, 0.5, 0.5), k2=(65, 1, 0))
        g, _ = H.run_gpu(w, stages="in")
        H.check_workload(w, g, O.run_workload(w, stage1=False))


def test_stage2_max_k1():
    w = synth.small_case(seed_cfg=96, n=(2048, 3000), m=(4, 256), d=64, hq=4, hkv=2, n_keep_heads=2,
                         k1=(2048, 1500), ratio=(0.5, 0.5), k2=(700, 1))
    g, _ = H.run_gpu(w)
    H.check_workload(w, g, O.run_workload(w))


def test_deterministic_repeat():
    w = synth.small_case(seed_cfg=94)
    g1, _ = H.run_gpu(w)
    g2, _ = H.run_gpu(w, reps=3)
    for f in ("s_t", "kept1", "Z_out", "u", "heads", "p", "kept2", "hidden_out", "K_out", "V_out"):
        np.testing.assert_array_equal(getattr(g1, f), getattr(g2, f), err_msg=f)


@pytest.mark.parametrize("make", [synth.llava15_single, synth.llava_next_batch8, synth.long_video_batch2,
                                  synth.ragged_serving_batch64, synth.video_llava_batch,
                                  lambda: synth.with_full_sequence_softmax(synth.video_llava_batch()),
                                  lambda: synth.with_full_sequence_softmax(synth.llava15_single())],
                         ids=["llava15_576", "llava_next_2880_b8", "long_16384_gqa", "ragged_b64",
                              "video_llava_2048_b4", "video_llava_2048_b4_fullseq", "llava15_576_fullseq"])
def test_full_size_workloads(make):
    w = make()
    tally, _ = _run_and_check(w)
    print(f"\n{w.name}: {tally}")
    # near ties are checked by the band rule; their number stays small on these inputs
    bound = max(1, w.B // 8)
    assert tally.stage1_near_ties <= bound and tally.stage2_near_ties <= bound, (
        f"{w.name}: {tally.stage1_near_ties} stage-1 and {tally.stage2_near_ties} stage-2 near ties "
        f"of {w.B} requests (bound {bound})")


@pytest.mark.parametrize("k1", [192, 128, 64])
@pytest.mark.parametrize("k2", [64, 32])
def test_llava15_batch32_sweep(k1, k2):
    import copy
    base = synth.llava15_batch32(k1=k1, ratio=0.5, k2=k2)   # the ratio changes no input
    for ratio in (0.0, 0.25, 0.5, 0.75, 1.0):
        w = copy.copy(base)
        w.reqs = [synth.Request(r.n, r.m, r.k1, ratio, r.l, r.k2) for r in base.reqs]
        tally, _ = _run_and_check(w)
        assert tally.stage1_near_ties <= 2 and tally.stage2_near_ties <= 2, f"ratio {ratio}: {tally}"


def test_fused_full_size():
    w = synth.llava_next_batch8()
    _run_and_check(w, "fused")


@pytest.mark.parametrize("k1,l", [(40, 9), (128, 64), (300, 33), (1024, 128)])
def test_full_sequence_softmax_stage2(k1, l):
    """The Sec. 4.2 variant whose rows also count the non-visual keys' mass, on both stage-2
    paths (small: L <= 64 and K1 <= 128), against the oracle's variant."""
    w = synth.small_case(seed_cfg=120 + l, n=(k1 + 3, k1), m=(l, max(1, l // 3)), d=64, hq=8, hkv=2,
                         n_keep_heads=3, k1=(k1, k1), ratio=(0.5, 0.5), k2=(k1 // 3, k1 // 2))
    w = synth.with_full_sequence_softmax(w, seed=k1)
    g, _ = H.run_gpu(w, stages="in")
    tally = H.check_workload(w, g, O.run_workload(w, stage1=False))
    assert tally.stage2_near_ties <= 1, tally


@pytest.mark.parametrize("d,m", [(200, (5, 17, 128, 64)), (512, (128, 100, 1, 33)), (576, (64, 64, 64, 64)),
                                 (512, (128, 200, 113, 256))])
def test_tiles_split_between_scoring_ctas(d, m):
    """Several 128-row tiles per scoring CTA, tiles split between CTAs, odd tile counts, text
    lengths from 1 to 128 and a partial last slice of d'."""
    w = synth.small_case(seed_cfg=150 + d, n=(1000, 512, 1536, 264), m=m, d=d, k1=(100, 64, 200, 8),
                         ratio=(0.5, 0.25, 0.75, 1.0), k2=(0, 0, 0, 0))
    for mode in ("ratio", "fused"):
        mm = T.SELECT_FUSED if mode == "fused" else T.SELECT_RATIO
        g, _ = H.run_gpu(w, mm, stages="pre")
        H.check_workload(w, g, O.run_workload(w, mode=mode, stage2=False), mode)


@pytest.mark.parametrize("make,reserve", [(synth.llava15_batch32, 0), (synth.llava15_batch32, 60),
                                          (synth.llava_next_batch8, 0), (synth.llava_next_batch8, 8),
                                          (synth.llava_next_batch8, 500)],
                         ids=["b32_after", "b32_r60", "next_after", "next_r8", "next_clamped"])
def test_overlap_reserve_settings(make, reserve):
    # The reserve moves stage 2 behind (0) or beside the scoring grid and changes how the
    # tiles split between scoring CTAs; the results stay those of the oracle.
    w = make()
    T.load().trevs_set_overlap_reserve(reserve)
    try:
        _run_and_check(w)
    finally:
        T.load().trevs_set_overlap_reserve(-1)
