"""[CLS] saliency (Eq. 2-3) on the GPU against the oracle.

Each request's s^v is compared element by element with the fp64 oracle on the same bf16
inputs: relative 1e-4 (fp32 dot products of d_h <= 128 bf16 products, fp32 exp and sums
over at most 16,384 patches) with an absolute floor of 1e-9 for the smallest shares.
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


def _check(q_bits, K_bits, n, s_v, scale=None):
    off = 0
    for b, nb in enumerate(n):
        if nb == 0:
            continue
        ref = O.cls_saliency(O.bf16_bits_to_f64(q_bits[b]), O.bf16_bits_to_f64(K_bits[off:off + nb]), scale)
        H.assert_close(s_v[off:off + nb], ref, 1e-4, 1e-9, f"request {b} s_v")
        assert abs(float(np.sum(s_v[off:off + nb], dtype=np.float64)) - 1.0) < 1e-4
        off += nb


def _run(q_bits, K_bits, n, heads, scale=0.0, K_dev=None, reps=2):
    q = H.dev_bf16(q_bits)
    K = K_dev if K_dev is not None else H.dev_bf16(K_bits)
    s_v = torch.full((max(sum(n), 1),), -1.0, dtype=torch.float32, device="cuda")
    ws = T.workspace(T.trevs_cls_saliency_workspace_size(n, heads))
    for _ in range(reps):   # the second call checks that the tickets reset themselves
        T.trevs_cls_saliency_varlen(q, K, n, s_v, scale=scale, ws=ws)
    torch.cuda.synchronize()
    return s_v.cpu().numpy()[:sum(n)]


@pytest.mark.parametrize("n,heads,dh", [([576] * 4, 16, 64), ([1, 577, 1000, 0, 33], 8, 128),
                                        ([16384, 5], 4, 32), ([2880] * 2, 16, 64)])
def test_cls_saliency_matches_oracle(n, heads, dh):
    q_bits, K_bits = synth.cls_inputs(n, heads, dh, seed=sum(n) + heads)
    _check(q_bits, K_bits, n, _run(q_bits, K_bits, n, heads))


def test_cls_saliency_head_major_keys_and_scale():
    n, heads, dh = [300, 200], 6, 64
    q_bits, K_bits = synth.cls_inputs(n, heads, dh, seed=5)
    # a head-major cache [heads, sum n, dh], passed as a strided [sum n, heads, dh] view
    Kh = H.dev_bf16(np.ascontiguousarray(K_bits.transpose(1, 0, 2)))
    s_v = _run(q_bits, K_bits, n, heads, scale=0.25, K_dev=Kh.permute(1, 0, 2))
    _check(q_bits, K_bits, n, s_v, scale=0.25)


def test_cls_saliency_feeds_stage1():
    # the saliency of the bench's request shape, then stage 1 on it: the same kept set as the
    # oracle's stage 1 on the oracle's saliency (ratio split, no near tie at these sizes)
    n, heads, dh = [576], 16, 64
    q_bits, K_bits = synth.cls_inputs(n, heads, dh, seed=11)
    s_v = _run(q_bits, K_bits, n, heads)
    ref = O.cls_saliency(O.bf16_bits_to_f64(q_bits[0]), O.bf16_bits_to_f64(K_bits))
    assert H.boundary_gap(ref, 32) > 1e-3
    np.testing.assert_array_equal(O.top_k(s_v.astype(np.float64), 32), O.top_k(ref, 32))
