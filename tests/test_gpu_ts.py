"""Eq. 1 textual sensitivity on the GPU (through the C ABI) against the oracle."""
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

# TS_h = 1 - cos is formed in fp32 from sums of fp32 probabilities: about 1e-6 absolute
TS_ATOL = 1e-5


def _attention(w, b):
    l_off, k1_off = w.offsets("l"), w.offsets("k1")
    return O.text_to_vision_attention(O.bf16_bits_to_f64(w.Q[l_off[b]:l_off[b + 1]]),
                                      O.bf16_bits_to_f64(w.K[k1_off[b]:k1_off[b + 1]]))


@pytest.mark.parametrize("k1,l1,l2", [(1, 1, 1), (64, 32, 20), (129, 7, 64), (1024, 128, 96)])
def test_textual_sensitivity(k1, l1, l2):
    # two questions about the same image: the same visual keys K, two query sets
    w = synth.small_case(seed_cfg=140 + k1, n=(k1, k1), m=(l1, l2), d=64, hq=8, hkv=2, n_keep_heads=2,
                         k1=(k1, k1), ratio=(0.5, 0.5), k2=(0, 0))
    w.K[k1:] = w.K[:k1]
    A1, A2 = _attention(w, 0), _attention(w, 1)
    want = O.textual_sensitivity(O.head_visual_attention(A1), O.head_visual_attention(A2))
    a1, a2 = H.dev_f32(A1), H.dev_f32(A2)
    ts = torch.full((w.hq,), -1.0, dtype=torch.float32, device="cuda")
    s1 = torch.zeros((w.hq, k1), dtype=torch.float32, device="cuda")
    s2 = torch.zeros((w.hq, k1), dtype=torch.float32, device="cuda")
    ws = T.workspace(T.load().trevs_textual_sensitivity_workspace_size(w.hq, k1))
    for _ in range(2):   # twice: the tickets must be back at zero after a call
        T.trevs_textual_sensitivity(a1, a2, ts, s1, s2, ws=ws)
        torch.cuda.synchronize()
        H.assert_close(ts.cpu().numpy(), want, 1e-3, TS_ATOL, "TS_h")
        H.assert_close(s1.cpu().numpy(), O.head_visual_attention(A1), H.RTOL, H.ATOL_P, "s_h^(1)")
        H.assert_close(s2.cpu().numpy(), O.head_visual_attention(A2), H.RTOL, H.ATOL_P, "s_h^(2)")


def test_textual_sensitivity_closed_forms():
    # the same attention under both questions: TS = 0; disjoint supports: TS = 1
    Hq, L, K1 = 3, 4, 300
    rng = np.random.default_rng(7)
    A = rng.random((Hq, L, K1))
    A /= A.sum(axis=2, keepdims=True)
    B = np.zeros((Hq, L, K1))
    B[:, :, :150] = 1.0 / 150
    C = np.zeros((Hq, 2, K1))
    C[:, :, 150:] = 1.0 / 150
    ts = torch.zeros(Hq, dtype=torch.float32, device="cuda")
    T.trevs_textual_sensitivity(H.dev_f32(A), H.dev_f32(A), ts)
    assert np.all(np.abs(ts.cpu().numpy()) < TS_ATOL)
    T.trevs_textual_sensitivity(H.dev_f32(B), H.dev_f32(C), ts)
    np.testing.assert_array_equal(ts.cpu().numpy(), np.ones(Hq, np.float32))
