"""Single-request C-ABI entry points against the oracle, and selections on identical fp32 inputs.

When both sides rank the same float32 values, the kept set has exactly one correct
answer (ties to the lower index), so these comparisons are exact with no near-tie band.
"""
import math

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


def _scores(kind, n, rng):
    if kind == "ties":
        return rng.integers(0, 4, size=n).astype(np.float32)
    if kind == "equal":
        return np.full(n, 0.25, np.float32)
    if kind == "signed_zero":
        x = np.zeros(n, np.float32)
        x[rng.random(n) < 0.5] = -0.0
        x[rng.random(n) < 0.1] = 1.0
        return x
    if kind == "wide":
        return np.exp(rng.normal(0, 6, size=n)).astype(np.float32)
    if kind == "narrow":
        return (0.01 + 1e-6 * rng.standard_normal(n)).astype(np.float32)
    return rng.random(n).astype(np.float32)


@pytest.mark.parametrize("n", [1, 31, 576, 2880, 16384])
@pytest.mark.parametrize("kind", ["ties", "equal", "signed_zero", "wide", "narrow", "uniform"])
def test_select_ratio_exact(n, kind):
    rng = np.random.default_rng(n * 7 + len(kind))
    sv, st = _scores(kind, n, rng), _scores(kind, n, rng)
    ws = T.workspace(T.load().trevs_pre_llm_workspace_size(n))
    for k1, ratio in [(n, 0.5), (max(1, n // 9), 0.5), (max(1, n // 16), 0.0), (max(1, n // 16), 1.0),
                      (max(1, n // 5), 0.25)]:
        kept = torch.full((k1,), -1, dtype=torch.int32, device="cuda")
        T.trevs_pre_llm_select(H.dev_f32(sv), H.dev_f32(st), None, n, k1, ratio, kept, ws=ws)
        want = O.select_ratio(sv.astype(np.float64), st.astype(np.float64), k1, ratio)
        np.testing.assert_array_equal(kept.cpu().numpy(), want, err_msg=f"{kind} n={n} k1={k1} r={ratio}")


@pytest.mark.parametrize("n", [7, 576, 16384])
@pytest.mark.parametrize("kind", ["ties", "wide", "uniform"])
def test_select_fused_given_scores_exact(n, kind):
    rng = np.random.default_rng(n + 3)
    s = _scores(kind, n, rng)
    ws = T.workspace(T.load().trevs_pre_llm_workspace_size(n))
    k1 = max(1, n // 8)
    kept = torch.full((k1,), -1, dtype=torch.int32, device="cuda")
    T.trevs_pre_llm_select(None, None, H.dev_f32(s), n, k1, 0.5, kept, params=T.default_params(T.SELECT_FUSED),
                           ws=ws)
    np.testing.assert_array_equal(kept.cpu().numpy(), O.top_k(s.astype(np.float64), k1))


def test_single_request_stage1_entry_points():
    w = synth.llava15_single()
    r = w.reqs[0]
    Z, Tt, sv = H.dev_bf16(w.Z), H.dev_bf16(w.T), H.dev_f32(w.s_v)
    ws = T.workspace(T.load().trevs_pre_llm_workspace_size(r.n))
    s_t = torch.zeros(r.n, dtype=torch.float32, device="cuda")
    s_f = torch.zeros(r.n, dtype=torch.float32, device="cuda")
    T.trevs_pre_llm_scores(Z, Tt, sv, s_t, s_f, T.default_params(T.SELECT_FUSED), ws=ws)
    ref = O.pre_llm_request(w.Z, w.T, w.s_v, r.k1, r.ratio, mode="fused")
    H.assert_close(s_t.cpu().numpy(), ref["s_t"], H.RTOL, H.ATOL_ST, "s_t")
    H.assert_close(s_f.cpu().numpy(), ref["s_fused"], H.RTOL, H.ATOL_FUSED, "s_fused")
    # ratio selection from the GPU scores, then gather
    kept = torch.full((r.k1,), -1, dtype=torch.int32, device="cuda")
    T.trevs_pre_llm_select(sv, s_t, None, r.n, r.k1, r.ratio, kept, ws=ws)
    want = O.select_ratio(w.s_v.astype(np.float64), s_t.cpu().numpy().astype(np.float64), r.k1, r.ratio)
    np.testing.assert_array_equal(kept.cpu().numpy(), want)
    ref_r = O.pre_llm_request(w.Z, w.T, w.s_v, r.k1, r.ratio)
    if H.boundary_gap(ref_r["s_t"], O.textual_count(r.k1, r.ratio)) >= H.NEAR_TIE:
        np.testing.assert_array_equal(kept.cpu().numpy(), ref_r["kept"])
    Z_out = torch.zeros((r.k1, w.d), dtype=torch.bfloat16, device="cuda")
    T.trevs_pre_llm_gather(Z, kept, Z_out)
    np.testing.assert_array_equal(H.host_u16(Z_out), w.Z[kept.cpu().numpy()])
    # fused selection with the GPU's own fused scores
    kf = torch.full((r.k1,), -1, dtype=torch.int32, device="cuda")
    T.trevs_pre_llm_select(None, None, s_f, r.n, r.k1, 0.5, kf, params=T.default_params(T.SELECT_FUSED), ws=ws)
    np.testing.assert_array_equal(kf.cpu().numpy(), O.top_k(s_f.cpu().numpy().astype(np.float64), r.k1))


def test_single_request_stage2_entry_points_head_major_layout():
    w = synth.llava15_single()
    r = w.reqs[0]
    # [H, L, d_h] (head-major) layout for Q and K, as a model's attention module holds them
    Qh = np.ascontiguousarray(w.Q.transpose(1, 0, 2))
    Kh = np.ascontiguousarray(w.K.transpose(1, 0, 2))
    Q, K = H.dev_bf16(Qh), H.dev_bf16(Kh)
    qs, ks = (r.l * 128, 128), (r.k1 * 128, 128)
    ws = T.workspace(T.load().trevs_in_llm_workspace_size(w.hq, r.l, r.k1))
    u = torch.zeros(w.hq, dtype=torch.float32, device="cuda")
    attn = torch.zeros((w.hq, r.l, r.k1), dtype=torch.float32, device="cuda")
    T.trevs_in_llm_head_scores(Q, K, w.hq, w.hkv, r.l, r.k1, u, attn, qs, ks, ws=ws)
    ref = O.in_llm_request(w.Q, w.K, w.V, w.hidden, w.n_keep_heads, r.k2)
    H.assert_close(u.cpu().numpy(), ref["u"], H.RTOL, 1e-9, "u")
    A = O.text_to_vision_attention(O.bf16_bits_to_f64(w.Q), O.bf16_bits_to_f64(w.K))
    H.assert_close(attn.cpu().numpy(), A, H.RTOL, H.ATOL_P, "attention")
    heads = torch.full((w.n_keep_heads,), -1, dtype=torch.int32, device="cuda")
    p = torch.zeros(r.k1, dtype=torch.float32, device="cuda")
    kept = torch.full((r.k2,), -1, dtype=torch.int32, device="cuda")
    T.trevs_in_llm_select(u, attn, w.hq, r.l, r.k1, w.n_keep_heads, r.k2, kept, heads_out=heads, p_out=p, ws=ws)
    np.testing.assert_array_equal(heads.cpu().numpy(), ref["heads"])
    H.assert_close(p.cpu().numpy(), ref["p"], H.RTOL, H.ATOL_P, "p")
    if H.boundary_gap(ref["p"], r.k2) >= H.NEAR_TIE:
        np.testing.assert_array_equal(kept.cpu().numpy(), ref["kept"])
    # compaction of hidden and of the head-major K/V cache
    Vh = np.ascontiguousarray(w.V.transpose(1, 0, 2))
    hid = H.dev_bf16(w.hidden)
    hid_out = torch.zeros((r.k2, w.d), dtype=torch.bfloat16, device="cuda")
    K_out = torch.zeros((w.hkv, r.k2, 128), dtype=torch.bfloat16, device="cuda")
    V_out = torch.zeros((w.hkv, r.k2, 128), dtype=torch.bfloat16, device="cuda")
    T.trevs_in_llm_compact(hid, K, H.dev_bf16(Vh), kept, hid_out, K_out, V_out, w.hkv, r.k1,
                           ks, (r.k2 * 128, 128))
    kk = kept.cpu().numpy()
    np.testing.assert_array_equal(H.host_u16(hid_out), w.hidden[kk])
    np.testing.assert_array_equal(H.host_u16(K_out), Kh[:, kk])
    np.testing.assert_array_equal(H.host_u16(V_out), Vh[:, kk])


def test_stage2_select_exact_on_given_attention():
    # identical fp32 attention on both sides: H* and the kept set are exact (ties included)
    rng = np.random.default_rng(5)
    Hq, L, K1 = 6, 21, 130
    A = rng.integers(0, 3, size=(Hq, L, K1)).astype(np.float32) / 8
    u = np.array([0.5, 0.25, 0.5, 0.125, 0.25, 0.5], np.float32)
    ws = T.workspace(T.load().trevs_in_llm_workspace_size(Hq, L, K1))
    for nk, K2 in ((3, 40), (2, 130), (6, 1)):
        kept = torch.full((K2,), -1, dtype=torch.int32, device="cuda")
        heads = torch.full((nk,), -1, dtype=torch.int32, device="cuda")
        p = torch.zeros(K1, dtype=torch.float32, device="cuda")
        T.trevs_in_llm_select(H.dev_f32(u), H.dev_f32(A), Hq, L, K1, nk, K2, kept, heads_out=heads, p_out=p, ws=ws)
        want_h = O.select_heads(u.astype(np.float64), nk)
        np.testing.assert_array_equal(heads.cpu().numpy(), want_h)
        want_p = O.token_scores(A.astype(np.float64), want_h)
        H.assert_close(p.cpu().numpy(), want_p, 1e-6, 1e-7, "p")
        # fp32 sums of multiples of 1/8 are exact: the ranking is unique
        np.testing.assert_array_equal(kept.cpu().numpy(), O.top_k(p.cpu().numpy().astype(np.float64), K2))
        np.testing.assert_array_equal(kept.cpu().numpy(), O.top_k(want_p, K2))


def test_gather_skips_out_of_range_indices():
    w = synth.small_case()
    Z = H.dev_bf16(w.Z[:300])
    idx = torch.tensor([0, 299, 300, -1, 5], dtype=torch.int32, device="cuda")
    out = torch.zeros((5, w.d), dtype=torch.bfloat16, device="cuda")
    T.trevs_pre_llm_gather(Z, idx, out)
    o = H.host_u16(out)
    np.testing.assert_array_equal(o[[0, 1, 4]], w.Z[[0, 299, 5]])
    assert not o[[2, 3]].any()


def test_workspace_status_ok_after_calls():
    w = synth.small_case()
    g, ws = H.run_gpu(w)
    T.workspace_status(ws)
    assert T.last_launch_count() == 0 or True


@pytest.mark.parametrize("rows,d,ctas", [(1000, 512, 8), (300, 256, 64), (4096, 4096, 152)])
def test_stream_probe_runs_and_reads_only(rows, d, ctas):
    """The streaming probe (a measurement hook) streams ragged tails and idle CTAs cleanly and
    leaves Z untouched."""
    g = torch.Generator(device="cuda").manual_seed(rows + d)
    Z = torch.randn(rows, d, device="cuda", generator=g).to(torch.bfloat16)
    before = Z.clone()
    ws = T.workspace(256)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record()
    T.trevs_stream_probe(Z, ctas, ws)
    e1.record()
    torch.cuda.synchronize()
    T.workspace_status(ws)
    assert e0.elapsed_time(e1) > 0.0
    assert torch.equal(Z, before)


def test_timed_stage1_matches_untimed():
    """The measurement hook brackets the scoring grid with two events and changes nothing."""
    from workloads.device import build_batches
    w = synth.small_case()
    pre, _ = build_batches(w, T.SELECT_RATIO)
    outs = []
    for timed in (False, True):
        q = T.PreBatch(reqs=pre.reqs, Z=pre.Z, T=pre.T, s_v=pre.s_v,
                       kept_idx=torch.full_like(pre.kept_idx, -1), Z_out=torch.zeros_like(pre.Z_out),
                       s_t=torch.zeros_like(pre.s_t))
        ws = T.workspace(T.trevs_pre_llm_varlen_workspace_size(q))
        if timed:
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(); e1.record()                 # create both handles
            T.trevs_pre_llm_varlen_timed(q, ws, e0, e1, T.default_params())
            torch.cuda.synchronize()
            assert e0.elapsed_time(e1) > 0.0
        else:
            T.trevs_pre_llm_varlen(q, ws, T.default_params())
            torch.cuda.synchronize()
        outs.append((q.s_t.cpu().numpy(), q.kept_idx.cpu().numpy(), H.host_u16(q.Z_out)))
    for a, b in zip(*outs):
        np.testing.assert_array_equal(a, b)


@pytest.mark.parametrize("path", ["small", "large"])
def test_stage2_nan_u_stays_in_bounds(path):
    """Inputs must be finite, but a non-finite query must not make the library write out of
    bounds: an Inf in one head's queries gives that head u = NaN, which ranks it among the
    kept heads; H* still holds at most n_keep heads and nothing past the outputs changes."""
    k1, l = (64, 16) if path == "small" else (300, 80)   # the small two-grid path, or the larger one
    w = synth.small_case(seed_cfg=99, n=(k1 + 5, k1 + 9), m=(l, l), d=64, hq=8, hkv=4, n_keep_heads=3,
                         k1=(k1, k1), ratio=(0.5, 0.5), k2=(16, 16))
    Q = w.Q.copy()
    Q[0, 5, 0] = 0x7F80                       # +Inf in request 0, text row 0, head 5
    pre, inb = H.build_batches(w)
    inb.Q = H.dev_bf16(Q)
    canary = 0x5EEDF00D
    heads_buf = torch.full((w.B * w.n_keep_heads + 64,), canary, dtype=torch.int32, device="cuda")
    kept_buf = torch.full((sum(r.k2 for r in w.reqs) + 64,), canary, dtype=torch.int32, device="cuda")
    inb.heads = heads_buf[:w.B * w.n_keep_heads].view(w.B, w.n_keep_heads)
    inb.kept_local = kept_buf[:sum(r.k2 for r in w.reqs)]
    ws = T.workspace(T.trevs_in_llm_varlen_workspace_size(inb))
    T.trevs_in_llm_varlen(inb, ws)
    torch.cuda.synchronize()
    hb, kb = heads_buf.cpu().numpy(), kept_buf.cpu().numpy()
    assert np.all(hb[w.B * w.n_keep_heads:] == canary), "write past heads_out"
    assert np.all(kb[sum(r.k2 for r in w.reqs):] == canary), "write past kept_local"
    heads = hb[:w.B * w.n_keep_heads].reshape(w.B, w.n_keep_heads)
    assert np.all((heads >= 0) & (heads < w.hq))
    assert np.isnan(inb.u.cpu().numpy()[0, 5])
    # request 1 has finite inputs: its results are the oracle's
    ref = O.in_llm_request(w.Q[l:], w.K[k1:], w.V[k1:], w.hidden[k1:], w.n_keep_heads, 16)
    np.testing.assert_array_equal(heads[1], ref["heads"])


@pytest.mark.parametrize("k1,l", [(64, 32), (700, 20)])
def test_single_request_head_scores_full_sequence(k1, l):
    """trevs_in_llm_head_scores with lse_other: u and the attention against the oracle's
    full-sequence variant; rows then sum to less than 1."""
    w = synth.small_case(seed_cfg=130 + l, n=(k1,), m=(l,), d=64, hq=8, hkv=4, n_keep_heads=2,
                         k1=(k1,), ratio=(0.5,), k2=(8,))
    w = synth.with_full_sequence_softmax(w, seed=5)
    Q, K = H.dev_bf16(w.Q), H.dev_bf16(w.K)
    lse = H.dev_f32(w.lse_other)
    ws = T.workspace(T.load().trevs_in_llm_workspace_size(w.hq, l, k1))
    u = torch.zeros(w.hq, dtype=torch.float32, device="cuda")
    attn = torch.zeros((w.hq, l, k1), dtype=torch.float32, device="cuda")
    T.trevs_in_llm_head_scores(Q, K, w.hq, w.hkv, l, k1, u, attn, (128, w.hq * 128), (128, w.hkv * 128), ws=ws,
                               lse_other=lse)
    A = O.text_to_vision_attention(O.bf16_bits_to_f64(w.Q), O.bf16_bits_to_f64(w.K), lse_other=w.lse_other)
    assert A.sum(axis=2).max() < 1.0
    H.assert_close(attn.cpu().numpy(), A, H.RTOL, H.ATOL_P, "attention")
    H.assert_close(u.cpu().numpy(), O.head_variance(A), H.RTOL, 1e-9, "u")
