"""Failure reporting of the bounded device-side waits, on the GPU, without a fault: a wait that is
never satisfied gives up after its limit and sets the workspace status word, the block's other
waits follow it out through the shared abort flag, and the context stays usable."""
import pytest
import torch

from paper_2609_13846_gb300 import dtp, synth

pytestmark = pytest.mark.gpu
DEV = "cuda:0"


def test_unsatisfied_wait_gives_up_and_reports():
    limit = 20 * 10 ** 6   # 20 ms
    r = dtp.selftest_bounded_wait(limit, complete=False, device=DEV)
    assert r["status"] == dtp.DTP_ERR_NOT_CONVERGED
    waited, follower = r["elapsed_ns"]
    assert limit <= waited < limit + 200 * 10 ** 6
    # the second wait has the library's own 2 s limit but leaves on the abort flag
    assert 0 < follower < 10 ** 9


def test_satisfied_wait_reports_ok():
    r = dtp.selftest_bounded_wait(10 ** 9, complete=True, device=DEV)
    assert r["status"] == dtp.DTP_OK
    assert r["elapsed_ns"][0] < 10 ** 9


def test_context_usable_after_a_wait_gave_up():
    dtp.selftest_bounded_wait(10 ** 6, complete=False, device=DEV)
    L = synth.make_layer(256, 2, 200, 300, seed=5, dtype="bf16")
    g = {k: v.to(DEV) for k, v in L.items()}
    ws = dtp.affinity_workspace(300, 256, 2, 200, dtp.DTP_BF16, DEV)
    A = dtp.affinity_accumulate(g["X"], g["C"], g["W_gate"], g["W_up"], workspace=ws)
    assert dtp.workspace_status(ws) == dtp.DTP_OK
    assert torch.isfinite(A).all() and (A >= 0).all() and A.sum() > 0
