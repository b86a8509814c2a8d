"""Failure paths on the GPU, none of which faults, traps or hangs the device: bounded device-side
waits that give up (a short wait limit set through the workspace header), and launches that fail
on the host (a test hook), including one that fails after the call has forked onto its second
stream inside a stream capture."""
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


def test_bounded_wait_gives_up_then_recovers():
    lib = T.load()
    w = synth.llava15_batch32()
    pre, _ = H.build_batches(w)
    ws = T.workspace(T.trevs_pre_llm_varlen_workspace_size(pre))
    # every wait of the scoring grid now gives up after 1 us: long before its first tile is in
    T.check(lib.trevs_workspace_set_wait_limit(T._ptr(ws), ws.numel(), 1, T._stream(None)))
    T.trevs_pre_llm_varlen(pre, ws, T.default_params(T.SELECT_RATIO))
    torch.cuda.synchronize()
    with pytest.raises(T.TrevsError) as e:
        T.workspace_status(ws)
    assert e.value.status == T.TREVS_ERR_TIMEOUT
    # the device is usable and a re-initialised workspace (limit cleared) gives the right answer
    T.check(lib.trevs_workspace_init(T._ptr(ws), ws.numel(), T._stream(None)))
    T.trevs_pre_llm_varlen(pre, ws, T.default_params(T.SELECT_RATIO))
    torch.cuda.synchronize()
    T.workspace_status(ws)
    g = H.collect(w, pre, H.build_batches(w)[1])
    ref = O.run_workload(w, stage2=False, requests=range(4))
    w4 = synth.llava15_batch32()
    w4.reqs = w4.reqs[:4]
    n4 = sum(r.n for r in w4.reqs)
    k4 = sum(r.k1 for r in w4.reqs)
    g4 = H.DeviceRun(s_t=g.s_t[:n4], s_fused=None, kept1=g.kept1[:k4], Z_out=g.Z_out[:k4], u=g.u, heads=g.heads,
                     p=g.p, kept2=g.kept2, hidden_out=g.hidden_out, K_out=g.K_out, V_out=g.V_out)
    H.check_workload(w4, g4, ref)


@pytest.mark.parametrize("fail_at", [1, 2, 3, 4, 5, 6, 7])
def test_injected_launch_failure_then_recovery(fail_at):
    lib = T.load()
    w = synth.small_case(seed_cfg=160)
    pre, inb = H.build_batches(w)
    ws = T.workspace(T.trevs_prune_varlen_workspace_size(pre, inb))
    params = T.default_params(T.SELECT_RATIO)
    T.trevs_prune_varlen(pre, inb, ws, params)
    launches = T.last_launch_count()
    torch.cuda.synchronize()
    lib.trevs_test_fail_launch(fail_at)
    if fail_at <= launches:
        with pytest.raises(T.TrevsError) as e:
            T.trevs_prune_varlen(pre, inb, ws, params)
        assert e.value.status == T.TREVS_ERR_CUDA
        assert "launch" in str(e.value)
    else:
        T.trevs_prune_varlen(pre, inb, ws, params)
    lib.trevs_test_fail_launch(0)
    torch.cuda.synchronize()
    # a failed call leaves tickets it never reached behind: re-initialise, then all is well
    T.check(lib.trevs_workspace_init(T._ptr(ws), ws.numel(), T._stream(None)))
    T.trevs_prune_varlen(pre, inb, ws, params)
    torch.cuda.synchronize()
    T.workspace_status(ws)
    H.check_workload(w, H.collect(w, pre, inb), O.run_workload(w))


def test_injected_failure_inside_a_capture_leaves_the_capture_whole():
    """A call that fails after forking onto its second stream still joins it, so the caller's
    stream capture ends cleanly."""
    lib = T.load()
    w = synth.llava15_batch32()
    pre, inb = H.build_batches(w)
    ws = T.workspace(T.trevs_prune_varlen_workspace_size(pre, inb))
    params = T.default_params(T.SELECT_RATIO)
    T.trevs_prune_varlen(pre, inb, ws, params)   # warm-up outside the capture
    torch.cuda.synchronize()
    stream = torch.cuda.Stream()
    for fail_at in (4, 6):   # the stage-1 tail, after the fork
        g = torch.cuda.CUDAGraph()
        failed = False
        with torch.cuda.graph(g, stream=stream):
            lib.trevs_test_fail_launch(fail_at)
            try:
                T.trevs_prune_varlen(pre, inb, ws, params, stream)
            except T.TrevsError as e:
                failed = e.status == T.TREVS_ERR_CUDA
        lib.trevs_test_fail_launch(0)
        assert failed
        del g
    torch.cuda.synchronize()
