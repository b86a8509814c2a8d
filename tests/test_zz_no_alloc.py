"""The allocation-free stage-2 selection against the workspace form, through the C ABI.

trevs_in_llm_select_noalloc keeps its scratch in a fixed device array of the library. It must
give what trevs_in_llm_select gives on the same inputs, call after call, whatever an earlier
call left in that array. The file name sorts last so that the tests also run after the rest
of the suite has used the library on the same device.
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


def _both(u, attn, Hq, L, K1, nk, K2):
    """Runs the workspace form and the allocation-free form; returns (heads, p, kept) of each."""
    out = []
    for form in ("workspace", "noalloc"):
        kept = torch.full((K2,), -1, dtype=torch.int32, device="cuda")
        heads = torch.full((nk,), -1, dtype=torch.int32, device="cuda")
        p = torch.full((K1,), 7.0, dtype=torch.float32, device="cuda")   # not zero: the call clears it
        if form == "workspace":
            ws = T.workspace(T.load().trevs_in_llm_workspace_size(Hq, L, K1))
            T.trevs_in_llm_select(u, attn, Hq, L, K1, nk, K2, kept, heads_out=heads, p_out=p, ws=ws)
        else:
            T.trevs_in_llm_select_noalloc(u, attn, Hq, L, K1, nk, K2, kept, heads_out=heads, p_out=p)
            assert T.last_launch_count() == 3
        out.append((heads.cpu().numpy(), p.cpu().numpy(), kept.cpu().numpy()))
    return out


def _same(a, b):
    for x, y, what in zip(a, b, ("heads", "p", "kept")):
        # the same kernel on the same inputs: identical results (tolerance zero)
        np.testing.assert_array_equal(x, y, err_msg=what)


def test_noalloc_matches_workspace_form_on_model_attention():
    w = synth.llava15_single()
    r = w.reqs[0]
    Q, K = H.dev_bf16(w.Q), H.dev_bf16(w.K)
    qs, ks = (128, w.hq * 128), (128, w.hkv * 128)
    u = torch.zeros(w.hq, dtype=torch.float32, device="cuda")
    attn = torch.zeros((w.hq, r.l, r.k1), dtype=torch.float32, device="cuda")
    ws = T.workspace(T.load().trevs_in_llm_workspace_size(w.hq, r.l, r.k1))
    T.trevs_in_llm_head_scores(Q, K, w.hq, w.hkv, r.l, r.k1, u, attn, qs, ks, ws=ws)
    ref = O.in_llm_request(w.Q, w.K, w.V, w.hidden, w.n_keep_heads, r.k2)
    for _ in range(2):                                   # two calls in a row
        a, b = _both(u, attn, w.hq, r.l, r.k1, w.n_keep_heads, r.k2)
        _same(a, b)
        np.testing.assert_array_equal(b[0], ref["heads"])
        H.assert_close(b[1], ref["p"], H.RTOL, H.ATOL_P, "p")
        if H.boundary_gap(ref["p"], r.k2) >= H.NEAR_TIE:
            np.testing.assert_array_equal(b[2], ref["kept"])


@pytest.mark.parametrize("Hq,L,K1,nk,K2", [(32, 40, 2048, 8, 512),    # the largest K1 the array holds
                                            (6, 21, 130, 3, 40),       # smaller after larger
                                            (28, 64, 1000, 7, 333),
                                            (4, 1, 1, 1, 1)])
def test_noalloc_two_calls_in_a_row(Hq, L, K1, nk, K2):
    rng = np.random.default_rng(Hq * 1000 + K1)
    A = rng.integers(0, 5, size=(Hq, L, K1)).astype(np.float32) / 16     # sums exact in fp32
    u = rng.integers(0, 9, size=Hq).astype(np.float32) / 8                # ties between heads
    du, dA = H.dev_f32(u), H.dev_f32(A)
    want_h = O.select_heads(u.astype(np.float64), nk)
    want_p = O.token_scores(A.astype(np.float64), want_h)
    for _ in range(2):
        a, b = _both(du, dA, Hq, L, K1, nk, K2)
        _same(a, b)
        np.testing.assert_array_equal(b[0], want_h)
        H.assert_close(b[1], want_p, 1e-6, 1e-7, "p")
        np.testing.assert_array_equal(b[2], O.top_k(want_p, K2))


def test_noalloc_without_optional_outputs_and_device_memory_steady():
    rng = np.random.default_rng(11)
    Hq, L, K1, nk, K2 = 16, 32, 576, 4, 64
    A = rng.random((Hq, L, K1)).astype(np.float32)
    u = rng.random(Hq).astype(np.float32)
    du, dA = H.dev_f32(u), H.dev_f32(A)
    kept = torch.full((K2,), -1, dtype=torch.int32, device="cuda")
    T.trevs_in_llm_select_noalloc(du, dA, Hq, L, K1, nk, K2, kept)      # p kept in the library's array
    torch.cuda.synchronize()
    free0 = torch.cuda.mem_get_info()[0]
    for _ in range(3):
        k2 = torch.full((K2,), -1, dtype=torch.int32, device="cuda")
        T.trevs_in_llm_select_noalloc(du, dA, Hq, L, K1, nk, K2, k2)
        torch.cuda.synchronize()
        np.testing.assert_array_equal(k2.cpu().numpy(), kept.cpu().numpy())
    assert torch.cuda.mem_get_info()[0] >= free0
    want_p = O.token_scores(A.astype(np.float64), O.select_heads(u.astype(np.float64), nk))
    if H.boundary_gap(want_p, K2) >= H.NEAR_TIE:
        np.testing.assert_array_equal(kept.cpu().numpy(), O.top_k(want_p, K2))


def test_noalloc_rejects_k1_beyond_the_array():
    dummy = torch.zeros(4, dtype=torch.float32, device="cuda")
    st = T.load().trevs_in_llm_select_noalloc(T._ptr(dummy), T._ptr(dummy), 4, 8, T.MAX_STAGE2_TOKENS + 1, 1, 8,
                                              None, None, T._ptr(dummy), None)
    assert st == T.TREVS_ERR_UNSUPPORTED
    assert "K1" in T.load().trevs_last_error_string().decode()
