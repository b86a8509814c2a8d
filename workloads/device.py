"""Places a synthetic workload on the GPU as C-ABI batch descriptors and runs it.

Device placement and marshalling only: no score, selection or gather arithmetic.
"""
from __future__ import annotations

import dataclasses

import numpy as np

from paper_2609_37581_gb300 import trevs as T


def _torch():
    import torch
    return torch


def dev_bf16(a):
    torch = _torch()
    return torch.from_numpy(np.ascontiguousarray(a).view(np.int16)).cuda().view(torch.bfloat16)


def dev_f32(a):
    torch = _torch()
    return torch.from_numpy(np.ascontiguousarray(a, dtype=np.float32)).cuda()


def host_u16(t):
    return t.view(_torch().int16).cpu().numpy().view(np.uint16)


@dataclasses.dataclass
class DeviceRun:
    s_t: np.ndarray
    s_fused: np.ndarray | None
    kept1: np.ndarray
    Z_out: np.ndarray
    u: np.ndarray
    heads: np.ndarray
    p: np.ndarray
    kept2: np.ndarray
    hidden_out: np.ndarray
    K_out: np.ndarray
    V_out: np.ndarray


def build_batches(w, mode=T.SELECT_RATIO, dev=None):
    """Device tensors and C-ABI batch descriptors for workload `w`."""
    torch = _torch()
    dev = dev or {}
    sum_n, sum_k1 = w.Z.shape[0], sum(r.k1 for r in w.reqs)
    sum_k2 = sum(r.k2 for r in w.reqs)
    Z = dev.get("Z", dev_bf16(w.Z))
    Tt = dev.get("T", dev_bf16(w.T))
    s_v = dev.get("s_v", dev_f32(w.s_v))
    pre = T.PreBatch(
        reqs=[(r.n, r.m, r.k1, r.ratio) for r in w.reqs], Z=Z, T=Tt, s_v=s_v,
        kept_idx=torch.full((max(sum_k1, 1),), -1, dtype=torch.int32, device="cuda"),
        Z_out=torch.zeros((max(sum_k1, 1), w.d), dtype=torch.bfloat16, device="cuda"),
        s_t=torch.zeros(max(sum_n, 1), dtype=torch.float32, device="cuda"),
        s_fused=(torch.zeros(max(sum_n, 1), dtype=torch.float32, device="cuda")
                 if mode == T.SELECT_FUSED else None))
    Q = dev.get("Q", dev_bf16(w.Q))
    K = dev.get("K", dev_bf16(w.K))
    V = dev.get("V", dev_bf16(w.V))
    H = dev.get("hidden", dev_bf16(w.hidden))
    inb = T.InBatch(
        reqs=[(r.k1, r.l, r.k2) for r in w.reqs], Hq=w.hq, Hkv=w.hkv, n_keep_heads=w.n_keep_heads,
        Q=Q, K=K, V=V, hidden=H,
        kept_local=torch.full((max(sum_k2, 1),), -1, dtype=torch.int32, device="cuda"),
        hidden_out=torch.zeros((max(sum_k2, 1), w.d), dtype=torch.bfloat16, device="cuda"),
        K_out=torch.zeros((max(sum_k2, 1), w.hkv, w.dh), dtype=torch.bfloat16, device="cuda"),
        V_out=torch.zeros((max(sum_k2, 1), w.hkv, w.dh), dtype=torch.bfloat16, device="cuda"),
        u=torch.zeros((w.B, w.hq), dtype=torch.float32, device="cuda"),
        heads=torch.full((w.B, w.n_keep_heads), -1, dtype=torch.int32, device="cuda"),
        p=torch.zeros(max(sum_k1, 1), dtype=torch.float32, device="cuda"),
        lse_other=None if w.lse_other is None else dev.get("lse_other", dev_f32(w.lse_other)))
    return pre, inb


def run_gpu(w, mode=T.SELECT_RATIO, params=None, reps=1, stages="both"):
    """Runs trevs_prune_varlen (stages="both"), trevs_pre_llm_varlen ("pre") or
    trevs_in_llm_varlen ("in") on workload `w`."""
    torch = _torch()
    pre, inb = build_batches(w, mode)
    if params is None:
        params = T.default_params(mode)
    if stages == "both":
        ws = T.workspace(T.trevs_prune_varlen_workspace_size(pre, inb))
        call = lambda: T.trevs_prune_varlen(pre, inb, ws, params)
    elif stages == "pre":
        ws = T.workspace(T.trevs_pre_llm_varlen_workspace_size(pre))
        call = lambda: T.trevs_pre_llm_varlen(pre, ws, params)
    else:
        ws = T.workspace(T.trevs_in_llm_varlen_workspace_size(inb))
        call = lambda: T.trevs_in_llm_varlen(inb, ws)
    for _ in range(reps):
        call()
    torch.cuda.synchronize()
    return collect(w, pre, inb), ws


def collect(w, pre, inb):
    sum_n, sum_k1 = w.Z.shape[0], sum(r.k1 for r in w.reqs)
    sum_k2 = sum(r.k2 for r in w.reqs)
    return DeviceRun(
        s_t=pre.s_t.cpu().numpy()[:sum_n],
        s_fused=None if pre.s_fused is None else pre.s_fused.cpu().numpy()[:sum_n],
        kept1=pre.kept_idx.cpu().numpy()[:sum_k1], Z_out=host_u16(pre.Z_out)[:sum_k1],
        u=inb.u.cpu().numpy(), heads=inb.heads.cpu().numpy(), p=inb.p.cpu().numpy()[:sum_k1],
        kept2=inb.kept_local.cpu().numpy()[:sum_k2], hidden_out=host_u16(inb.hidden_out)[:sum_k2],
        K_out=host_u16(inb.K_out)[:sum_k2], V_out=host_u16(inb.V_out)[:sum_k2])


