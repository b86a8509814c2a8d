"""Thin Python binding of libtrevs (the C ABI in include/trevs.h).

Argument marshalling only: every step of the pruning path runs in the CUDA
library. PyTorch supplies device memory and the current stream. The binding
refuses to work without the compiled library; there is no fallback.
"""
from __future__ import annotations

import ctypes
import dataclasses
import os
import pathlib

_PKG = pathlib.Path(__file__).resolve().parent
LIB_PATH = _PKG / "libtrevs.so"

TREVS_OK = 0
TREVS_ERR_INVALID_ARGUMENT = 1
TREVS_ERR_WORKSPACE = 2
TREVS_ERR_CUDA = 3
TREVS_ERR_UNSUPPORTED = 4
TREVS_ERR_TIMEOUT = 5
SELECT_RATIO = 0
SELECT_FUSED = 1
MAX_TEXT_TOKENS = 256
HEAD_DIM = 128
MAX_STAGE2_TOKENS = 2048
MAX_HEADS = 128

_c_i32, _c_i64, _c_f32, _c_sz, _vp = ctypes.c_int32, ctypes.c_int64, ctypes.c_float, ctypes.c_size_t, ctypes.c_void_p


class TrevsError(RuntimeError):
    def __init__(self, status: int, message: str):
        super().__init__(f"trevs status {status}: {message}")
        self.status = status


class PreParams(ctypes.Structure):
    _fields_ = [("tau_v", _c_f32), ("tau_t", _c_f32), ("lambda_", _c_f32), ("eps", _c_f32),
                ("select_mode", _c_i32), ("diversity", _c_f32)]


class PreRequest(ctypes.Structure):
    _fields_ = [("n", _c_i32), ("m", _c_i32), ("k1", _c_i32), ("ratio", _c_f32)]


class PreBatchC(ctypes.Structure):
    _fields_ = [("B", _c_i32), ("d", _c_i32), ("reqs", ctypes.POINTER(PreRequest)),
                ("Z", _vp), ("z_row_stride", _c_i64), ("T", _vp), ("t_row_stride", _c_i64),
                ("s_v", _vp), ("s_t", _vp), ("s_fused", _vp), ("kept_idx", _vp),
                ("Z_out", _vp), ("z_out_row_stride", _c_i64)]


class InRequest(ctypes.Structure):
    _fields_ = [("k1", _c_i32), ("l", _c_i32), ("k2", _c_i32)]


class InBatchC(ctypes.Structure):
    _fields_ = [("B", _c_i32), ("Hq", _c_i32), ("Hkv", _c_i32), ("d_h", _c_i32), ("d_model", _c_i32),
                ("n_keep_heads", _c_i32), ("softmax_scale", _c_f32), ("reqs", ctypes.POINTER(InRequest)),
                ("Q", _vp), ("q_head_stride", _c_i64), ("q_tok_stride", _c_i64),
                ("K", _vp), ("V", _vp), ("kv_head_stride", _c_i64), ("kv_tok_stride", _c_i64),
                ("hidden", _vp), ("hidden_row_stride", _c_i64),
                ("u", _vp), ("heads", _vp), ("p", _vp), ("kept_local", _vp),
                ("hidden_out", _vp), ("hidden_out_row_stride", _c_i64),
                ("K_out", _vp), ("V_out", _vp), ("out_head_stride", _c_i64), ("out_tok_stride", _c_i64),
                ("lse_other", _vp), ("lse_head_stride", _c_i64), ("lse_row_stride", _c_i64)]


_SIGS = {
    "trevs_pre_params_default": (None, [ctypes.POINTER(PreParams)]),
    "trevs_version": (ctypes.c_char_p, []),
    "trevs_last_error_string": (ctypes.c_char_p, []),
    "trevs_last_launch_count": (_c_i32, []),
    "trevs_workspace_init": (_c_i32, [_vp, _c_sz, _vp]),
    "trevs_workspace_status": (_c_i32, [_vp, _c_sz, _vp]),
    "trevs_workspace_set_wait_limit": (_c_i32, [_vp, _c_sz, ctypes.c_uint32, _vp]),
    "trevs_test_fail_launch": (None, [_c_i32]),
    "trevs_set_overlap_reserve": (None, [_c_i32]),
    "trevs_pre_llm_workspace_size": (_c_sz, [_c_i32]),
    "trevs_pre_llm_scores": (_c_i32, [_vp, _c_i64, _c_i32, _c_i32, _vp, _c_i64, _c_i32, _vp,
                                      ctypes.POINTER(PreParams), _vp, _vp, _vp, _c_sz, _vp]),
    "trevs_pre_llm_select": (_c_i32, [_vp, _vp, _vp, _c_i32, _c_i32, _c_f32, ctypes.POINTER(PreParams),
                                      _vp, _vp, _c_sz, _vp]),
    "trevs_pre_llm_gather": (_c_i32, [_vp, _c_i64, _c_i32, _c_i32, _vp, _c_i32, _vp, _c_i64, _vp]),
    "trevs_cls_saliency_workspace_size": (_c_sz, [_c_i32, ctypes.POINTER(_c_i32), _c_i32]),
    "trevs_cls_saliency_varlen": (_c_i32, [_vp, _c_i64, _c_i64, _vp, _c_i64, _c_i64, _c_i32,
                                           ctypes.POINTER(_c_i32), _c_i32, _c_i32, _c_f32, _vp, _vp, _c_sz, _vp]),
    "trevs_pre_llm_fps_workspace_size": (_c_sz, [_c_i32, _c_i32, _c_i32]),
    "trevs_pre_llm_fps": (_c_i32, [_vp, _c_i64, _c_i32, _c_i32, _vp, _c_i32, _c_i32, _c_i32, _vp, _vp,
                                   _vp, _c_sz, _vp]),
    "trevs_in_llm_workspace_size": (_c_sz, [_c_i32, _c_i32, _c_i32]),
    "trevs_in_llm_head_scores": (_c_i32, [_vp, _c_i64, _c_i64, _vp, _c_i64, _c_i64, _c_i32, _c_i32,
                                          _c_i32, _c_i32, _c_i32, _c_f32, _vp, _vp, _vp, _vp, _c_sz, _vp]),
    "trevs_in_llm_select": (_c_i32, [_vp, _vp, _c_i32, _c_i32, _c_i32, _c_i32, _c_i32, _vp, _vp, _vp,
                                     _vp, _c_sz, _vp]),
    "trevs_textual_sensitivity_workspace_size": (_c_sz, [_c_i32, _c_i32]),
    "trevs_textual_sensitivity": (_c_i32, [_vp, _c_i32, _vp, _c_i32, _c_i32, _c_i32, _vp, _vp, _vp, _vp, _c_sz,
                                           _vp]),
    "trevs_in_llm_select_noalloc": (_c_i32, [_vp, _vp, _c_i32, _c_i32, _c_i32, _c_i32, _c_i32, _vp, _vp, _vp,
                                             _vp]),
    "trevs_in_llm_compact": (_c_i32, [_vp, _c_i64, _c_i32, _vp, _vp, _c_i64, _c_i64, _c_i32, _c_i32,
                                      _c_i32, _vp, _c_i32, _vp, _c_i64, _vp, _vp, _c_i64, _c_i64, _vp]),
    "trevs_pre_llm_varlen_workspace_size": (_c_sz, [ctypes.POINTER(PreBatchC)]),
    "trevs_in_llm_varlen_workspace_size": (_c_sz, [ctypes.POINTER(InBatchC)]),
    "trevs_prune_varlen_workspace_size": (_c_sz, [ctypes.POINTER(PreBatchC), ctypes.POINTER(InBatchC)]),
    "trevs_pre_llm_varlen": (_c_i32, [ctypes.POINTER(PreBatchC), ctypes.POINTER(PreParams), _vp, _c_sz, _vp]),
    "trevs_pre_llm_varlen_timed": (_c_i32, [ctypes.POINTER(PreBatchC), ctypes.POINTER(PreParams), _vp, _c_sz, _vp,
                                            _vp, _vp]),
    "trevs_in_llm_varlen": (_c_i32, [ctypes.POINTER(InBatchC), _vp, _c_sz, _vp]),
    "trevs_stream_probe": (_c_i32, [_vp, _c_i64, _c_i64, _c_i32, _c_i32, _vp, _c_sz, _vp]),
    "trevs_prune_varlen": (_c_i32, [ctypes.POINTER(PreBatchC), ctypes.POINTER(PreParams),
                                    ctypes.POINTER(InBatchC), _vp, _c_sz, _vp]),
}

EXPORTED = tuple(_SIGS)
_lib = None


def load(path: str | os.PathLike | None = None) -> ctypes.CDLL:
    """Loads libtrevs.so (built by __graft_entry__.build()); raises if it is missing."""
    global _lib
    if _lib is not None and path is None:
        return _lib
    p = pathlib.Path(path) if path else LIB_PATH
    if not p.exists():
        raise RuntimeError(f"libtrevs not built: {p} is missing (run __graft_entry__.build())")
    lib = ctypes.CDLL(str(p))
    for name, (res, args) in _SIGS.items():
        fn = getattr(lib, name)
        fn.restype = res
        fn.argtypes = args
    if path is None:
        _lib = lib
    return lib


def check(status: int) -> None:
    if status != TREVS_OK:
        raise TrevsError(status, load().trevs_last_error_string().decode())


def last_launch_count() -> int:
    """Kernels (and memsets) the last library call on this thread enqueued."""
    return int(load().trevs_last_launch_count())


def version() -> str:
    return load().trevs_version().decode()


def default_params(mode: int = SELECT_RATIO, **kw) -> PreParams:
    p = PreParams()
    load().trevs_pre_params_default(ctypes.byref(p))
    p.select_mode = mode
    for k, v in kw.items():
        setattr(p, "lambda_" if k in ("lambda", "lam") else k, v)
    return p


# ------------------------------------------------------------------ torch marshalling

def _torch():
    import torch
    return torch


def _ptr(t):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _stream(stream):
    torch = _torch()
    if stream is None:
        stream = torch.cuda.current_stream()
    return ctypes.c_void_p(stream.cuda_stream)


def workspace(nbytes: int, device="cuda"):
    """A zero-filled, 256-byte aligned byte buffer for the library's scratch memory."""
    torch = _torch()
    return torch.zeros(max(int(nbytes), 256), dtype=torch.uint8, device=device)


def _ws_args(ws):
    return (None, 0) if ws is None else (_ptr(ws), ws.numel() * ws.element_size())


def workspace_status(ws, stream=None):
    """Raises TrevsError(TREVS_ERR_TIMEOUT) if a device-side wait of an earlier call gave up."""
    w, nb = _ws_args(ws)
    check(load().trevs_workspace_status(w, nb, _stream(stream)))


def trevs_stream_probe(Z, ctas, ws, stream=None):
    """One pass of the streaming probe over the rows of Z [rows, d] on `ctas` CTAs."""
    w, nb = _ws_args(ws)
    check(load().trevs_stream_probe(_ptr(Z), Z.stride(0), Z.shape[0], Z.shape[1], int(ctas), w, nb,
                                    _stream(stream)))


# single-request entry points --------------------------------------------------------

def trevs_pre_llm_scores(Z, T, s_v=None, s_t_out=None, s_fused_out=None, params=None, ws=None, stream=None):
    N, d = Z.shape
    M = T.shape[0]
    w, nb = _ws_args(ws)
    check(load().trevs_pre_llm_scores(_ptr(Z), Z.stride(0), N, d, _ptr(T), T.stride(0), M, _ptr(s_v),
                                      ctypes.byref(params) if params is not None else None,
                                      _ptr(s_t_out), _ptr(s_fused_out), w, nb, _stream(stream)))


def trevs_pre_llm_select(s_v, s_t, s_fused, N, K1, ratio, kept_idx, params=None, ws=None, stream=None):
    w, nb = _ws_args(ws)
    check(load().trevs_pre_llm_select(_ptr(s_v), _ptr(s_t), _ptr(s_fused), N, K1, ratio,
                                      ctypes.byref(params) if params is not None else None,
                                      _ptr(kept_idx), w, nb, _stream(stream)))


def trevs_pre_llm_gather(Z, kept_idx, Z_out, stream=None):
    N, d = Z.shape
    check(load().trevs_pre_llm_gather(_ptr(Z), Z.stride(0), N, d, _ptr(kept_idx), kept_idx.numel(),
                                      _ptr(Z_out), Z_out.stride(0), _stream(stream)))


def _i32_array(xs):
    xs = [int(x) for x in xs]
    return (_c_i32 * max(len(xs), 1))(*xs)


def trevs_cls_saliency_workspace_size(n, H):
    arr = _i32_array(n)
    return int(load().trevs_cls_saliency_workspace_size(len(n), arr, H))


def trevs_cls_saliency_varlen(q_cls, K_v, n, s_v, scale=0.0, ws=None, stream=None):
    """Eq. 2-3 for a batch: q_cls [B, H, d_h] and K_v [sum n, H, d_h] (bf16, any strides with
    a unit innermost stride), n the patch count of each request; writes s_v [sum n]."""
    B, H, dh = q_cls.shape
    arr = _i32_array(n)
    w, nb = _ws_args(ws)
    check(load().trevs_cls_saliency_varlen(_ptr(q_cls), q_cls.stride(0), q_cls.stride(1), _ptr(K_v),
                                           K_v.stride(0), K_v.stride(1), B, arr, H, dh, scale, _ptr(s_v),
                                           w, nb, _stream(stream)))


def trevs_pre_llm_fps_workspace_size(N, K_r, d):
    return int(load().trevs_pre_llm_fps_workspace_size(N, K_r, d))


def trevs_pre_llm_fps(Z, pivots, K_d, picks, pick_dist=None, pool=0, ws=None, stream=None):
    """Sec. 3.1 context preservation: K_d draws of farthest point sampling over the rows of Z
    that are not in `pivots` (int32, may be None for none), in draw order into `picks`."""
    N, d = Z.shape
    K_r = 0 if pivots is None else pivots.numel()
    w, nb = _ws_args(ws)
    check(load().trevs_pre_llm_fps(_ptr(Z), Z.stride(0), N, d, _ptr(pivots), K_r, K_d, pool, _ptr(picks),
                                   _ptr(pick_dist), w, nb, _stream(stream)))


def trevs_in_llm_head_scores(Q, K, Hq, Hkv, L, K1, u_out, attn_out, q_strides, k_strides,
                             scale=0.0, ws=None, stream=None, lse_other=None):
    """lse_other: optional [Hq, L] float32 (contiguous), the full-sequence softmax variant."""
    w, nb = _ws_args(ws)
    check(load().trevs_in_llm_head_scores(_ptr(Q), q_strides[0], q_strides[1], _ptr(K), k_strides[0],
                                          k_strides[1], Hq, Hkv, L, K1, HEAD_DIM, scale, _ptr(lse_other),
                                          _ptr(u_out), _ptr(attn_out), w, nb, _stream(stream)))


def trevs_in_llm_select(u, attn, Hq, L, K1, n_keep, K2, kept_local, heads_out=None, p_out=None, ws=None,
                        stream=None):
    w, nb = _ws_args(ws)
    check(load().trevs_in_llm_select(_ptr(u), _ptr(attn), Hq, L, K1, n_keep, K2, _ptr(heads_out), _ptr(p_out),
                                     _ptr(kept_local), w, nb, _stream(stream)))


def trevs_textual_sensitivity(attn1, attn2, ts_out, s1_out=None, s2_out=None, ws=None, stream=None):
    """Eq. 1 for attention tensors [Hq, L1, K1] and [Hq, L2, K1] (float32, contiguous)."""
    Hq, L1, K1 = attn1.shape
    L2 = attn2.shape[1]
    if ws is None:
        ws = workspace(load().trevs_textual_sensitivity_workspace_size(Hq, K1))
    w, nb = _ws_args(ws)
    check(load().trevs_textual_sensitivity(_ptr(attn1), L1, _ptr(attn2), L2, Hq, K1, _ptr(ts_out), _ptr(s1_out),
                                           _ptr(s2_out), w, nb, _stream(stream)))


def trevs_in_llm_select_noalloc(u, attn, Hq, L, K1, n_keep, K2, kept_local, heads_out=None, p_out=None,
                                stream=None):
    """trevs_in_llm_select without a workspace: the library's fixed device scratch is used."""
    check(load().trevs_in_llm_select_noalloc(_ptr(u), _ptr(attn), Hq, L, K1, n_keep, K2, _ptr(heads_out),
                                             _ptr(p_out), _ptr(kept_local), _stream(stream)))


def trevs_in_llm_compact(hidden, Kc, Vc, kept_local, hidden_out, K_out, V_out, Hkv, K1,
                         kv_strides, out_strides, stream=None):
    K2 = kept_local.numel()
    d_model = hidden.shape[1] if hidden is not None else 0
    check(load().trevs_in_llm_compact(
        _ptr(hidden), hidden.stride(0) if hidden is not None else 0, d_model, _ptr(Kc), _ptr(Vc),
        kv_strides[0], kv_strides[1], Hkv, HEAD_DIM, K1, _ptr(kept_local), K2, _ptr(hidden_out),
        hidden_out.stride(0) if hidden_out is not None else 0, _ptr(K_out), _ptr(V_out),
        out_strides[0], out_strides[1], _stream(stream)))


# batched entry points ----------------------------------------------------------------

@dataclasses.dataclass
class PreBatch:
    """Stage-1 batch: packed device tensors plus host-side per-request sizes."""
    reqs: list                 # [(n, m, k1, ratio)]
    Z: object                  # [sum n, d] bf16
    T: object                  # [sum m, d] bf16
    s_v: object                # [sum n] f32
    kept_idx: object           # [sum k1] i32
    Z_out: object = None       # [sum k1, d] bf16
    s_t: object = None         # [sum n] f32
    s_fused: object = None     # [sum n] f32

    def c(self):
        arr = (PreRequest * max(1, len(self.reqs)))(*[PreRequest(int(n), int(m), int(k), float(r))
                                                       for n, m, k, r in self.reqs])
        self._keep = arr
        return PreBatchC(len(self.reqs), int(self.Z.shape[1]), ctypes.cast(arr, ctypes.POINTER(PreRequest)),
                         _ptr(self.Z), self.Z.stride(0), _ptr(self.T), self.T.stride(0), _ptr(self.s_v),
                         _ptr(self.s_t), _ptr(self.s_fused), _ptr(self.kept_idx), _ptr(self.Z_out),
                         self.Z_out.stride(0) if self.Z_out is not None else 0)


@dataclasses.dataclass
class InBatch:
    """Stage-2 batch. Q is [sum l, Hq, dh]; K, V are [sum k1, Hkv, dh]; hidden [sum k1, d_model]."""
    reqs: list                 # [(k1, l, k2)]
    Hq: int
    Hkv: int
    n_keep_heads: int
    Q: object
    K: object
    kept_local: object         # [sum k2] i32
    V: object = None
    hidden: object = None
    hidden_out: object = None
    K_out: object = None       # [sum k2, Hkv, dh]
    V_out: object = None
    u: object = None           # [B, Hq] f32
    heads: object = None       # [B, n_keep] i32
    p: object = None           # [sum k1] f32
    softmax_scale: float = 0.0
    lse_other: object = None   # [Hq, sum l] f32: full-sequence softmax variant (Sec. 4.2)

    def c(self):
        arr = (InRequest * max(1, len(self.reqs)))(*[InRequest(int(a), int(b), int(c)) for a, b, c in self.reqs])
        self._keep = arr
        ko = self.K_out if self.K_out is not None else self.V_out
        return InBatchC(
            len(self.reqs), self.Hq, self.Hkv, HEAD_DIM,
            int(self.hidden.shape[1]) if self.hidden is not None else 0, self.n_keep_heads,
            self.softmax_scale, ctypes.cast(arr, ctypes.POINTER(InRequest)),
            _ptr(self.Q), self.Q.stride(1), self.Q.stride(0),
            _ptr(self.K), _ptr(self.V), self.K.stride(1), self.K.stride(0),
            _ptr(self.hidden), self.hidden.stride(0) if self.hidden is not None else 0,
            _ptr(self.u), _ptr(self.heads), _ptr(self.p), _ptr(self.kept_local),
            _ptr(self.hidden_out), self.hidden_out.stride(0) if self.hidden_out is not None else 0,
            _ptr(self.K_out), _ptr(self.V_out),
            ko.stride(1) if ko is not None else 0, ko.stride(0) if ko is not None else 0,
            _ptr(self.lse_other), self.lse_other.stride(0) if self.lse_other is not None else 0,
            self.lse_other.stride(1) if self.lse_other is not None else 0)


def trevs_pre_llm_varlen_workspace_size(pre: PreBatch) -> int:
    return load().trevs_pre_llm_varlen_workspace_size(ctypes.byref(pre.c()))


def trevs_in_llm_varlen_workspace_size(inb: InBatch) -> int:
    return load().trevs_in_llm_varlen_workspace_size(ctypes.byref(inb.c()))


def trevs_prune_varlen_workspace_size(pre: PreBatch, inb: InBatch) -> int:
    return load().trevs_prune_varlen_workspace_size(ctypes.byref(pre.c()), ctypes.byref(inb.c()))


def trevs_pre_llm_varlen(pre: PreBatch, ws, params=None, stream=None):
    w, nb = _ws_args(ws)
    check(load().trevs_pre_llm_varlen(ctypes.byref(pre.c()),
                                      ctypes.byref(params) if params is not None else None, w, nb, _stream(stream)))


def trevs_pre_llm_varlen_timed(pre: PreBatch, ws, ev_begin, ev_end, params=None, stream=None):
    """trevs_pre_llm_varlen with the scoring grid bracketed by two timing events (torch.cuda.Event
    objects that have been recorded once, or raw cudaEvent_t handles)."""
    w, nb = _ws_args(ws)
    h = lambda e: getattr(e, "cuda_event", e)
    check(load().trevs_pre_llm_varlen_timed(ctypes.byref(pre.c()),
                                            ctypes.byref(params) if params is not None else None, w, nb,
                                            _stream(stream), h(ev_begin), h(ev_end)))


def trevs_in_llm_varlen(inb: InBatch, ws, stream=None):
    w, nb = _ws_args(ws)
    check(load().trevs_in_llm_varlen(ctypes.byref(inb.c()), w, nb, _stream(stream)))


def trevs_prune_varlen(pre: PreBatch, inb: InBatch, ws, params=None, stream=None):
    w, nb = _ws_args(ws)
    check(load().trevs_prune_varlen(ctypes.byref(pre.c()), ctypes.byref(params) if params is not None else None,
                                    ctypes.byref(inb.c()), w, nb, _stream(stream)))


class PreparedCall:
    """A trevs_prune_varlen call with its argument structs built once (for repeated launches)."""

    def __init__(self, pre: PreBatch, inb: InBatch, ws, params=None):
        self.lib = load()
        self.pre_c = pre.c()
        self.pre_keep = pre._keep
        self.in_c = inb.c()
        self.in_keep = inb._keep
        self.params = params
        self.ws = ws
        self.w, self.nb = _ws_args(ws)

    def __call__(self, stream=None):
        check(self.lib.trevs_prune_varlen(ctypes.byref(self.pre_c),
                                          ctypes.byref(self.params) if self.params is not None else None,
                                          ctypes.byref(self.in_c), self.w, self.nb, _stream(stream)))
