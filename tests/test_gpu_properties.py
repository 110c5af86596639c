"""Properties of the first-order affinity (Sec. 3 "Affinity scores") that hold at any size,
checked on the full Qwen3-0.6B-shaped layer (T = 16384) in the launch configuration the
benchmark uses, where the oracle can only sample columns.

* Each row of A depends only on its own head's writes C_h, through the same arithmetic
  wherever the head sits, so permuting the heads permutes the rows of A bit for bit, and a
  zeroed head gives a zero row while the other rows stay bit for bit the same.
* Scaling C by 2 scales every projection, hence Delta, by 2 and Delta^2 by 4; binary scaling
  commutes with every rounding step (no overflow or underflow at these magnitudes), so
  A(2C) = 4 A(C) exactly.
* Permuting the neurons (rows of W_gate and W_up together) permutes the columns of A, and
  permuting the tokens (rows of X and C together) leaves A unchanged, both up to the order of
  floating-point sums (checked to 1e-5 relative).
"""
import pytest
import torch

from paper_2609_13846_gb300 import dtp, synth

pytestmark = pytest.mark.gpu
DEV = "cuda:0"


@pytest.fixture(scope="module")
def layer():
    w = synth.WORKLOADS["qwen3_0.6b_layer"]
    L = synth.make_workload_layer(w, device=DEV)
    sms = torch.cuda.get_device_properties(0).multi_processor_count
    return w, L, sms - 1


def _A(L, max_ctas, X=None, C=None, Wg=None, Wu=None):
    A = dtp.affinity_accumulate(L["X"] if X is None else X, L["C"] if C is None else C,
                                L["W_gate"] if Wg is None else Wg, L["W_up"] if Wu is None else Wu,
                                max_ctas=max_ctas)
    torch.cuda.synchronize()
    return A


def test_head_permutation_permutes_rows_bitwise(layer):
    w, L, mc = layer
    A = _A(L, mc)
    perm = torch.randperm(w.G, generator=torch.Generator().manual_seed(1)).to(DEV)
    Ap = _A(L, mc, C=L["C"][perm].contiguous())
    assert torch.equal(Ap, A[perm])


def test_zeroed_head_gives_zero_row(layer):
    w, L, mc = layer
    A = _A(L, mc)
    C = L["C"].clone()
    C[3].zero_()
    Az = _A(L, mc, C=C)
    assert torch.all(Az[3] == 0)
    keep = [g for g in range(w.G) if g != 3]
    assert torch.equal(Az[keep], A[keep])


def test_doubling_C_multiplies_A_by_four_exactly(layer):
    w, L, mc = layer
    A = _A(L, mc)
    A2 = _A(L, mc, C=L["C"] * 2)
    assert torch.equal(A2, A * 4)


def test_neuron_permutation_permutes_columns(layer):
    w, L, mc = layer
    A = _A(L, mc)
    perm = torch.randperm(w.N, generator=torch.Generator().manual_seed(2)).to(DEV)
    Ap = _A(L, mc, Wg=L["W_gate"][perm].contiguous(), Wu=L["W_up"][perm].contiguous())
    ref = A[:, perm]
    assert torch.allclose(Ap, ref, rtol=1e-5, atol=0)


def test_token_permutation_leaves_A_unchanged(layer):
    w, L, mc = layer
    A = _A(L, mc)
    perm = torch.randperm(w.T, generator=torch.Generator().manual_seed(3)).to(DEV)
    Ap = _A(L, mc, X=L["X"][perm].contiguous(), C=L["C"][:, perm].contiguous())
    rel = (torch.linalg.norm(Ap - A) / torch.linalg.norm(A)).item()
    assert rel <= 1e-5, rel


@pytest.mark.parametrize("D", [2, 4])
def test_exact_optimum_invariant_under_permutations(layer, D):
    """The best layout's score (integer fixed point, order-independent) is the same when the heads
    or the neurons of A are permuted: both only relabel the balanced layouts.  The returned layout
    maps back onto one of the same score."""
    w, L, mc = layer
    A = _A(L, mc)
    base = dtp.search_global(A, D)
    ph = torch.randperm(w.G, generator=torch.Generator().manual_seed(4)).to(DEV)
    pn = torch.randperm(w.N, generator=torch.Generator().manual_seed(5)).to(DEV)
    rh = dtp.search_global(A[ph].contiguous(), D)
    rn = dtp.search_global(A[:, pn].contiguous(), D)
    torch.cuda.synchronize()
    assert int(rh["score_q"]) == int(base["score_q"])
    assert int(rn["score_q"]) == int(base["score_q"])
    # the layouts found on the permuted inputs, mapped back, score the same on the original A
    # (co-located q = floor(A 2^(40 - e)), e the binary exponent of max A, summed exactly)
    e = int(torch.frexp(A.max().double()).exponent)
    q = torch.floor(A.double() * 2.0 ** (40 - e)).long()

    def score(h, nu):
        return int((q * (h.long()[:, None] == nu.long()[None, :])).sum())

    h_back = torch.empty_like(rh["h"])
    h_back[ph] = rh["h"]
    nu_back = torch.empty_like(rn["nu"])
    nu_back[pn] = rn["nu"]
    assert score(base["h"], base["nu"]) == int(base["score_q"])
    assert score(h_back, rh["nu"]) == int(base["score_q"])
    assert score(rn["h"], nu_back) == int(base["score_q"])
