"""The allocation-free affinity entry point (dtp_affinity_accumulate_noalloc).

It serves callers that cannot allocate device memory or hand the library a
workspace (e.g. a plugin whose host owns every device allocation); its scratch
is a fixed array inside the library.  It must give the same A as
dtp_affinity_accumulate with a caller workspace, on consecutive calls that
reuse the shared array with different shapes.
"""
import numpy as np
import pytest
import torch

from paper_2609_13846_gb300 import dtp, synth

pytestmark = pytest.mark.gpu
DEV = "cuda:0"
BF16_TOL = 5e-3  # the relative Frobenius tolerance of the bf16 affinity tests


def _rel_fro(a, b):
    a, b = a.double().cpu().numpy(), b.double().cpu().numpy()
    return float(np.linalg.norm(a - b) / np.linalg.norm(b))


def test_noalloc_matches_workspace_entry_point_on_two_calls():
    for d, G, N, T, seed in ((1024, 8, 384, 1000, 11), (328, 3, 300, 333, 12)):
        L = synth.make_layer(d, G, N, T, seed, dtype="bf16", device=DEV)
        A_ref = dtp.affinity_accumulate(L["X"], L["C"], L["W_gate"], L["W_up"])
        A_new = torch.zeros((G, N), dtype=torch.float32, device=DEV)
        dtp.affinity_accumulate_noalloc(L["X"], L["C"], L["W_gate"], L["W_up"], A_new)
        torch.cuda.synchronize()
        assert torch.isfinite(A_new).all()
        assert _rel_fro(A_new, A_ref) <= BF16_TOL


def test_noalloc_rejects_calls_beyond_its_scratch():
    # 129 chunks, rounded up to 130: 130 * ceil(N/128) * H_kv = 130 * 16 * 16 > 32768, the documented limit
    G, N, T, d = 16, 2048, 129 * 128, 8
    X = torch.zeros((T, d), dtype=torch.bfloat16, device=DEV)
    C = torch.zeros((G, T, d), dtype=torch.bfloat16, device=DEV)
    W = torch.zeros((N, d), dtype=torch.bfloat16, device=DEV)
    A = torch.zeros((G, N), dtype=torch.float32, device=DEV)
    with pytest.raises(dtp.DTPError) as e:
        dtp.affinity_accumulate_noalloc(X, C, W, W, A)
    assert e.value.status == dtp.DTP_ERR_WORKSPACE
    # exactly at the limit (128 * 16 * 16 = 32768) the call is accepted
    T = 128 * 128
    dtp.affinity_accumulate_noalloc(X[:T].contiguous(), C[:, :T].contiguous(), W, W, A)
    torch.cuda.synchronize()
    assert torch.all(A == 0)
