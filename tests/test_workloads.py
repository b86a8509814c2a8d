"""Seeded workload generators: shapes, budgets and the structure the configs ask for."""
import numpy as np

import oracle.trevs_oracle as O
from workloads import synth


def test_video_llava_shape_and_budget():
    w = synth.video_llava_batch()
    assert w.B == 4 and w.d == 4096 and (w.hq, w.hkv, w.dh, w.n_keep_heads) == (32, 32, 128, 16)
    assert all(r.n == 2048 and r.k1 == 272 and r.k2 == 91 and 16 <= r.m <= 48 for r in w.reqs)
    assert w.Z.shape == (4 * 2048, 4096) and w.Z.dtype == np.uint16
    # the paper's budget: 136 visual tokens per LLM layer on average, 32 layers, second prune
    # after layer 8 (K1 = 3 K2 up to rounding)
    r = w.reqs[0]
    assert abs((8 * r.k1 + 24 * r.k2) / 32 - 136) < 0.5
    # saliency per frame: each 256-token frame is a distribution
    frames = w.s_v.reshape(-1, 256).astype(np.float64).sum(axis=1)
    assert np.allclose(frames, 1.0, atol=1e-5)
    # the generator is seeded: a second call gives the same bytes
    assert np.array_equal(synth.video_llava_batch().Z[:2048], w.Z[:2048])


def test_video_llava_oracle_runs_one_request():
    w = synth.video_llava_batch(batch=1)
    res = O.run_workload(w, "fused", diversity=0.25)[0]
    assert len(res["pre"]["kept"]) == 272 and len(res["pre"]["fps"]) == 68
    assert len(res["in"]["kept"]) == 91 and len(res["in"]["heads"]) == 16


def test_cls_inputs_shapes_and_spikes():
    n = [576, 0, 10]
    q, K = synth.cls_inputs(n, heads=16, dh=64, seed=1, spikes=8)
    assert q.shape == (3, 16, 64) and K.shape == (586, 16, 64)
    s = O.cls_saliency(O.bf16_bits_to_f64(q[0]), O.bf16_bits_to_f64(K[:576]))
    # the planted patches take a large share of the [CLS] attention
    assert np.sort(s)[-8:].sum() > 0.2
