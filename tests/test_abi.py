"""The C ABI loads, exports every symbol include/trevs.h declares, and validates on the host.

These tests need no GPU: every call here fails validation before any CUDA call, or is
a size query.
"""
import ctypes
import pathlib
import re

import pytest

from paper_2609_37581_gb300 import trevs as t

ROOT = pathlib.Path(__file__).resolve().parent.parent
HEADER = ROOT / "include" / "trevs.h"
FAKE = ctypes.c_void_p(0x10000)        # aligned, never dereferenced: validation fails first


def declared():
    text = HEADER.read_text()
    return sorted(set(re.findall(r"TREVS_API\s+[\w\s\*]+?\b(trevs_\w+)\s*\(", text)))


@pytest.fixture(scope="module")
def lib():
    return t.load()


def test_header_declares_entry_points():
    names = declared()
    for must in ("trevs_pre_llm_scores", "trevs_pre_llm_select", "trevs_pre_llm_gather",
                 "trevs_in_llm_head_scores", "trevs_in_llm_select", "trevs_in_llm_compact",
                 "trevs_prune_varlen"):
        assert must in names


def test_every_declared_symbol_is_exported(lib):
    for name in declared():
        assert hasattr(lib, name), name
        assert name in t.EXPORTED, name


def test_version_and_defaults(lib):
    assert t.version().count(".") == 2
    p = t.default_params()
    assert (round(p.tau_v, 6), p.tau_t, p.lambda_, p.select_mode) == (1.4, 1.0, 1.0, t.SELECT_RATIO)
    assert p.diversity == 0.0
    assert abs(p.eps - 1e-6) < 1e-12


def _err(lib):
    return lib.trevs_last_error_string().decode()


def test_select_validation(lib):
    assert lib.trevs_pre_llm_select(FAKE, FAKE, None, 10, 11, 0.5, None, FAKE, FAKE, 1 << 20, None) == 1
    assert "K1" in _err(lib)
    assert lib.trevs_pre_llm_select(FAKE, FAKE, None, 10, 5, 1.5, None, FAKE, FAKE, 1 << 20, None) == 1
    assert lib.trevs_pre_llm_select(FAKE, None, None, 10, 5, 0.5, None, FAKE, FAKE, 1 << 20, None) == 1
    # K1 = 0 is a valid no-op
    assert lib.trevs_pre_llm_select(None, None, None, 10, 0, 0.5, None, None, None, 0, None) == 0
    # bad mode
    p = t.default_params(mode=7)
    assert lib.trevs_pre_llm_select(FAKE, FAKE, None, 10, 5, 0.5, ctypes.byref(p), FAKE, FAKE, 1 << 20, None) == 1


def test_workspace_validation(lib):
    need = lib.trevs_pre_llm_workspace_size(1000)
    assert need > 0 and need % 256 == 0
    assert lib.trevs_pre_llm_select(FAKE, FAKE, None, 1000, 5, 0.5, None, FAKE, FAKE, need - 1, None) == 2
    assert lib.trevs_pre_llm_select(FAKE, FAKE, None, 1000, 5, 0.5, None, FAKE, None, need, None) == 2
    assert lib.trevs_pre_llm_select(FAKE, FAKE, None, 1000, 5, 0.5, None, FAKE,
                                    ctypes.c_void_p(0x10010), need, None) == 2
    assert lib.trevs_in_llm_workspace_size(32, 64, 320) > lib.trevs_in_llm_workspace_size(32, 32, 64)


def test_scores_validation(lib):
    args = lambda N, d, M, zs=4096: (FAKE, zs, N, d, FAKE, 4096, M, FAKE, None, FAKE, None, FAKE, 1 << 24, None)
    assert lib.trevs_pre_llm_scores(*args(576, 4096, 257)) == t.TREVS_ERR_UNSUPPORTED
    assert lib.trevs_pre_llm_scores(*args(576, 4100, 32, 4100)) == t.TREVS_ERR_INVALID_ARGUMENT
    assert lib.trevs_pre_llm_scores(*args(576, 4096, 0)) == t.TREVS_ERR_INVALID_ARGUMENT
    assert lib.trevs_pre_llm_scores(*args(576, 4096, 32, 4000)) == t.TREVS_ERR_INVALID_ARGUMENT
    misaligned = (ctypes.c_void_p(0x10002), 4096, 576, 4096, FAKE, 4096, 32, FAKE, None, FAKE, None, FAKE,
                  1 << 24, None)
    assert lib.trevs_pre_llm_scores(*misaligned) == t.TREVS_ERR_INVALID_ARGUMENT
    assert lib.trevs_pre_llm_scores(None, 0, 0, 4096, None, 0, 0, None, None, None, None, None, 0, None) == 0


def test_fps_validation(lib):
    need = lib.trevs_pre_llm_fps_workspace_size(576, 48, 4096)
    assert need > 0 and need % 256 == 0
    assert lib.trevs_pre_llm_fps_workspace_size(576, 48, 4096) > lib.trevs_pre_llm_fps_workspace_size(100, 48, 4096)
    assert lib.trevs_pre_llm_fps_workspace_size(-1, 0, 4096) == 0

    def fps(N=576, d=4096, K_r=48, K_d=16, pool=0, zs=4096, Z=FAKE, piv=FAKE, picks=FAKE, ws=FAKE, nb=need):
        return lib.trevs_pre_llm_fps(Z, zs, N, d, piv, K_r, K_d, pool, picks, None, ws, nb, None)
    assert fps(K_r=500, K_d=100) == t.TREVS_ERR_INVALID_ARGUMENT          # K_r + K_d > N
    assert "exceeds" in _err(lib)
    assert fps(K_d=-1) == t.TREVS_ERR_INVALID_ARGUMENT
    assert fps(pool=-2) == t.TREVS_ERR_INVALID_ARGUMENT
    # more than 256 pivots run in passes; they need a larger workspace, nothing else
    assert fps(K_r=257, N=1000) == t.TREVS_ERR_WORKSPACE
    assert lib.trevs_pre_llm_fps_workspace_size(1000, 257, 4096) > need
    assert fps(d=4100, zs=4100) == t.TREVS_ERR_INVALID_ARGUMENT
    assert fps(zs=4000) == t.TREVS_ERR_INVALID_ARGUMENT
    assert fps(Z=ctypes.c_void_p(0x10002)) == t.TREVS_ERR_INVALID_ARGUMENT
    assert fps(piv=None) == t.TREVS_ERR_INVALID_ARGUMENT
    assert fps(picks=None) == t.TREVS_ERR_INVALID_ARGUMENT
    assert fps(nb=need - 1) == t.TREVS_ERR_WORKSPACE
    assert fps(ws=ctypes.c_void_p(0x10010)) == t.TREVS_ERR_WORKSPACE
    # K_d = 0 is a valid no-op, and so is an empty request
    assert fps(K_d=0, Z=None, piv=None, picks=None, ws=None, nb=0) == 0
    assert fps(N=0, K_r=0, K_d=0, Z=None, piv=None, picks=None, ws=None, nb=0) == 0
    assert t.last_launch_count() == 0


def test_cls_saliency_validation(lib):
    arr = lambda xs: (ctypes.c_int32 * len(xs))(*xs)
    n = arr([576, 0, 1000])
    need = lib.trevs_cls_saliency_workspace_size(3, n, 16)
    assert need > 4 * 16 * 1576 and need % 256 == 0
    assert lib.trevs_cls_saliency_workspace_size(0, n, 16) == 0

    def cls(B=3, nn=n, H=16, dh=64, q=FAKE, K=FAKE, s=FAKE, ws=FAKE, nb=need, strides=(1024, 64, 1024, 64),
            scale=0.0):
        return lib.trevs_cls_saliency_varlen(q, strides[0], strides[1], K, strides[2], strides[3], B, nn, H, dh,
                                             scale, s, ws, nb, None)
    assert cls(dh=72) == t.TREVS_ERR_UNSUPPORTED
    assert cls(H=129) == t.TREVS_ERR_UNSUPPORTED
    assert cls(nn=arr([576, 16385, 1])) == t.TREVS_ERR_UNSUPPORTED
    assert cls(nn=arr([576, -1, 1])) == t.TREVS_ERR_INVALID_ARGUMENT
    assert cls(H=0) == t.TREVS_ERR_INVALID_ARGUMENT
    assert cls(K=ctypes.c_void_p(0x10008)) == t.TREVS_ERR_INVALID_ARGUMENT
    assert cls(strides=(1024, 64, 1020, 64)) == t.TREVS_ERR_INVALID_ARGUMENT
    assert cls(s=None) == t.TREVS_ERR_INVALID_ARGUMENT
    assert cls(scale=float("inf")) == t.TREVS_ERR_INVALID_ARGUMENT
    assert cls(nb=need - 1) == t.TREVS_ERR_WORKSPACE
    assert cls(B=0, nn=None, q=None, K=None, s=None, ws=None, nb=0) == 0
    assert cls(B=2, nn=arr([0, 0]), q=None, K=None, s=None, ws=None, nb=0) == 0
    assert t.last_launch_count() == 0


def test_stage2_validation(lib):
    def hs(Hq, Hkv, L, K1, dh):
        return lib.trevs_in_llm_head_scores(FAKE, 4096, 128, FAKE, 8192, 128, Hq, Hkv, L, K1, dh, 0.0,
                                            None, FAKE, FAKE, FAKE, 1 << 24, None)
    assert hs(32, 5, 32, 64, 128) == t.TREVS_ERR_INVALID_ARGUMENT      # Hq % Hkv
    assert hs(32, 32, 32, 64, 64) == t.TREVS_ERR_UNSUPPORTED           # d_h
    assert hs(32, 32, 32, 4096, 128) == t.TREVS_ERR_UNSUPPORTED        # K1 beyond the limit
    assert hs(32, 32, 0, 64, 128) == t.TREVS_ERR_INVALID_ARGUMENT      # no text rows
    assert hs(256, 32, 32, 64, 128) == t.TREVS_ERR_UNSUPPORTED         # Hq
    sel = lambda nk, K2: lib.trevs_in_llm_select(FAKE, FAKE, 32, 32, 64, nk, K2, None, None, FAKE, FAKE, 1 << 24,
                                                 None)
    assert sel(0, 32) == t.TREVS_ERR_INVALID_ARGUMENT
    assert sel(33, 32) == t.TREVS_ERR_INVALID_ARGUMENT
    assert sel(8, 65) == t.TREVS_ERR_INVALID_ARGUMENT
    na = lambda K1, nk, K2: lib.trevs_in_llm_select_noalloc(FAKE, FAKE, 32, 32, K1, nk, K2, None, None, FAKE, None)
    assert na(t.MAX_STAGE2_TOKENS + 1, 8, 8) == t.TREVS_ERR_UNSUPPORTED    # beyond the fixed scratch
    assert "K1" in _err(lib)
    assert na(64, 0, 8) == t.TREVS_ERR_INVALID_ARGUMENT
    assert na(64, 8, 65) == t.TREVS_ERR_INVALID_ARGUMENT
    assert lib.trevs_in_llm_select_noalloc(FAKE, None, 32, 32, 64, 8, 8, None, None, FAKE,
                                           None) == t.TREVS_ERR_INVALID_ARGUMENT
    assert lib.trevs_in_llm_compact(FAKE, 4096, 4096, None, None, 0, 0, 1, 128, 64, FAKE, 65, FAKE, 4096,
                                    None, None, 0, 0, None) == t.TREVS_ERR_INVALID_ARGUMENT
    assert lib.trevs_in_llm_compact(FAKE, 4096, 4096, FAKE, None, 0, 0, 1, 128, 64, FAKE, 32, FAKE, 4096,
                                    None, None, 0, 0, None) == t.TREVS_ERR_INVALID_ARGUMENT


def _pre_batch(reqs, d=4096):
    arr = (t.PreRequest * len(reqs))(*[t.PreRequest(*r) for r in reqs])
    b = t.PreBatchC(len(reqs), d, ctypes.cast(arr, ctypes.POINTER(t.PreRequest)), FAKE, d, FAKE, d, FAKE,
                    None, None, FAKE, None, 0)
    b._keep = arr
    return b


def test_varlen_validation(lib):
    ok = _pre_batch([(576, 32, 64, 0.5), (0, 0, 0, 0.5), (1152, 8, 96, 0.25)])
    need = lib.trevs_pre_llm_varlen_workspace_size(ctypes.byref(ok))
    assert need >= 13 * (576 + 1152)
    bad = [
        _pre_batch([(576, 32, 577, 0.5)]),          # k1 > n
        _pre_batch([(576, 0, 64, 0.5)]),            # no text
        _pre_batch([(576, 32, 64, -0.1)]),          # ratio
        _pre_batch([(576, 32, 64, 0.5)], d=100),    # d % 8
        _pre_batch([(-1, 32, 0, 0.5)]),
    ]
    for b in bad:
        assert lib.trevs_pre_llm_varlen(ctypes.byref(b), None, FAKE, 1 << 30, None) == t.TREVS_ERR_INVALID_ARGUMENT
    assert lib.trevs_pre_llm_varlen(ctypes.byref(_pre_batch([(576, 300, 64, 0.5)])), None, FAKE, 1 << 30,
                                    None) == t.TREVS_ERR_UNSUPPORTED
    assert lib.trevs_pre_llm_varlen(ctypes.byref(ok), None, FAKE, need - 256, None) == t.TREVS_ERR_WORKSPACE
    empty = t.PreBatchC()
    assert lib.trevs_pre_llm_varlen(ctypes.byref(empty), None, None, 0, None) == 0


def test_varlen_diversity_validation(lib):
    ok = _pre_batch([(576, 32, 64, 0.5), (2880, 64, 320, 0.5)])
    need = lib.trevs_pre_llm_varlen_workspace_size(ctypes.byref(ok))
    for rho in (-0.1, 1.5, float("nan")):
        p = t.default_params(t.SELECT_FUSED, diversity=rho)
        assert lib.trevs_pre_llm_varlen(ctypes.byref(ok), ctypes.byref(p), FAKE, need, None) == \
            t.TREVS_ERR_INVALID_ARGUMENT
        assert "diversity" in _err(lib)
    # K1 = 1024 at rho = 0.25 leaves 768 pivots (three passes of the contraction): validation
    # passes up to the workspace, for any share
    big = _pre_batch([(16384, 128, 1024, 0.5)], d=3584)
    nb = lib.trevs_pre_llm_varlen_workspace_size(ctypes.byref(big))
    for rho in (0.25, 0.75):
        p = t.default_params(t.SELECT_FUSED, diversity=rho)
        assert lib.trevs_pre_llm_varlen(ctypes.byref(big), ctypes.byref(p), FAKE, nb - 256, None) == \
            t.TREVS_ERR_WORKSPACE


def test_varlen_timed_validation(lib):
    ok = _pre_batch([(576, 32, 64, 0.5), (1152, 8, 96, 0.25)])
    need = lib.trevs_pre_llm_varlen_workspace_size(ctypes.byref(ok))
    f = lib.trevs_pre_llm_varlen_timed
    assert f(ctypes.byref(ok), None, FAKE, need, None, None, FAKE) == t.TREVS_ERR_INVALID_ARGUMENT
    assert f(ctypes.byref(ok), None, FAKE, need, None, FAKE, None) == t.TREVS_ERR_INVALID_ARGUMENT
    assert f(ctypes.byref(_pre_batch([(576, 32, 577, 0.5)])), None, FAKE, 1 << 30, None, FAKE,
             FAKE) == t.TREVS_ERR_INVALID_ARGUMENT
    assert f(ctypes.byref(t.PreBatchC()), None, None, 0, None, FAKE, FAKE) == t.TREVS_ERR_INVALID_ARGUMENT
    big = _pre_batch([(8, 1, 1, 0.5)] * 257)     # more requests than one launch chunk
    assert f(ctypes.byref(big), None, FAKE, 1 << 30, None, FAKE, FAKE) == t.TREVS_ERR_UNSUPPORTED
    assert f(ctypes.byref(ok), None, FAKE, need - 256, None, FAKE, FAKE) == t.TREVS_ERR_WORKSPACE


def test_stream_probe_validation(lib):
    f = lib.trevs_stream_probe
    bad = t.TREVS_ERR_INVALID_ARGUMENT
    assert f(None, 4096, 1024, 4096, 128, FAKE, 64, None) == bad                    # no Z
    assert f(ctypes.c_void_p(0x10008), 4096, 1024, 4096, 128, FAKE, 64, None) == bad   # unaligned Z
    assert f(FAKE, 4096, 0, 4096, 128, FAKE, 64, None) == bad                      # no rows
    assert f(FAKE, 4160, 1024, 4160, 128, FAKE, 64, None) == bad                   # d not a multiple of 256
    assert f(FAKE, 4095, 1024, 4096, 128, FAKE, 64, None) == bad                   # stride < d
    assert f(FAKE, 4096, 1024, 4096, 0, FAKE, 64, None) == bad                     # no CTAs
    assert f(FAKE, 4096, 1024, 4096, 128, None, 64, None) == bad                   # no status word
    assert f(FAKE, 4096, 1024, 4096, 128, FAKE, 4, None) == bad


def _in_batch(reqs, Hq=32, Hkv=32, nk=8):
    arr = (t.InRequest * len(reqs))(*[t.InRequest(*r) for r in reqs])
    b = t.InBatchC()
    b.B, b.Hq, b.Hkv, b.d_h, b.d_model, b.n_keep_heads = len(reqs), Hq, Hkv, 128, 4096, nk
    b.reqs = ctypes.cast(arr, ctypes.POINTER(t.InRequest))
    b.Q, b.q_head_stride, b.q_tok_stride = FAKE, 128, Hq * 128
    b.K, b.kv_head_stride, b.kv_tok_stride = FAKE, 128, Hkv * 128
    b.kept_local = FAKE
    b._keep = arr
    return b


def test_in_varlen_validation(lib):
    ok = _in_batch([(64, 32, 32), (192, 16, 64)])
    need = lib.trevs_in_llm_varlen_workspace_size(ctypes.byref(ok))
    assert need > 0
    for b in (_in_batch([(64, 32, 65)]), _in_batch([(0, 32, 0)]), _in_batch([(64, 0, 8)]),
              _in_batch([(64, 32, 8)], Hkv=3), _in_batch([(64, 32, 8)], nk=0), _in_batch([(64, 32, 8)], nk=33)):
        assert lib.trevs_in_llm_varlen(ctypes.byref(b), FAKE, 1 << 30, None) == t.TREVS_ERR_INVALID_ARGUMENT
    big = _in_batch([(4096, 32, 8)])
    assert lib.trevs_in_llm_varlen(ctypes.byref(big), FAKE, 1 << 30, None) == t.TREVS_ERR_UNSUPPORTED
    half = _in_batch([(64, 32, 8)])
    half.hidden = FAKE                               # hidden without hidden_out
    assert lib.trevs_in_llm_varlen(ctypes.byref(half), FAKE, 1 << 30, None) == t.TREVS_ERR_INVALID_ARGUMENT
    pre = _pre_batch([(576, 32, 64, 0.5)])
    tot = lib.trevs_prune_varlen_workspace_size(ctypes.byref(pre), ctypes.byref(ok))
    assert tot >= lib.trevs_pre_llm_varlen_workspace_size(ctypes.byref(pre)) + need
    assert lib.trevs_prune_varlen(ctypes.byref(pre), None, ctypes.byref(ok), FAKE, tot - 256,
                                  None) == t.TREVS_ERR_WORKSPACE


def test_textual_sensitivity_validation(lib):
    ts = lib.trevs_textual_sensitivity
    need = lib.trevs_textual_sensitivity_workspace_size(28, 1024)
    assert need > 0 and lib.trevs_textual_sensitivity_workspace_size(0, 5) == 0
    assert ts(FAKE, 4, FAKE, 4, 0, 10, FAKE, None, None, FAKE, need, None) == t.TREVS_ERR_INVALID_ARGUMENT
    assert ts(FAKE, 0, FAKE, 4, 2, 10, FAKE, None, None, FAKE, need, None) == t.TREVS_ERR_INVALID_ARGUMENT
    assert ts(None, 4, FAKE, 4, 2, 10, FAKE, None, None, FAKE, need, None) == t.TREVS_ERR_INVALID_ARGUMENT
    assert ts(FAKE, 4, FAKE, 4, 28, 1024, FAKE, None, None, FAKE, need - 1, None) == t.TREVS_ERR_WORKSPACE
    assert ts(FAKE, 4, FAKE, 4, 28, 1024, FAKE, None, None, None, need, None) == t.TREVS_ERR_WORKSPACE


def test_failure_hooks_validate_on_the_host(lib):
    assert lib.trevs_workspace_set_wait_limit(None, 1 << 20, 5, None) == t.TREVS_ERR_WORKSPACE
    assert lib.trevs_workspace_set_wait_limit(FAKE, 4, 5, None) == t.TREVS_ERR_WORKSPACE
    lib.trevs_test_fail_launch(0)   # disarmed: nothing to check without a GPU
    lib.trevs_set_overlap_reserve(7)   # host-side setting only
    lib.trevs_set_overlap_reserve(-1)
