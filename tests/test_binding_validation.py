"""Host-side argument checks of the Python binding: bad tensors are rejected with a clear error
before any CUDA call (no GPU needed)."""
import numpy as np
import pytest
import torch

from paper_2609_13846_gb300 import ablation, dtp


def _bf16(*shape):
    return torch.zeros(shape, dtype=torch.bfloat16)


def test_affinity_rejects_host_tensors():
    with pytest.raises(ValueError, match="CUDA"):
        dtp.affinity_accumulate(_bf16(16, 64), _bf16(2, 16, 64), _bf16(128, 64), _bf16(128, 64))
    with pytest.raises(ValueError, match="CUDA"):
        dtp.affinity_accumulate_grouped(_bf16(16, 64), _bf16(4, 16, 64), _bf16(128, 64), _bf16(128, 64), 2)
    with pytest.raises(ValueError, match="CUDA"):
        dtp.affinity_accumulate_down(_bf16(16, 64), _bf16(2, 16, 64), _bf16(128, 64), _bf16(128, 64),
                                     torch.ones(16))
    with pytest.raises(ValueError, match="CUDA"):
        dtp.affinity_accumulate_noalloc(_bf16(16, 64), _bf16(2, 16, 64), _bf16(128, 64), _bf16(128, 64),
                                        torch.zeros(2, 128))


def test_head_writes_rejects_bad_inputs():
    with pytest.raises(ValueError, match="bf16 CUDA"):
        dtp.head_writes(torch.zeros(8, 64), _bf16(32, 64), torch.zeros(32), torch.ones(8), 16)


def test_search_rejects_host_or_misshaped_matrices():
    with pytest.raises(ValueError):
        dtp.search_layout_batched(torch.zeros(2, 8, 64), 2, 10)
    with pytest.raises(ValueError):
        dtp.search_chain(torch.zeros(3, 8, 64), torch.zeros(1, 8, 64), 2, 10)
    with pytest.raises(ValueError):
        dtp.search_global(torch.zeros(8, 64), 2)


def test_layout_helpers_reject_bad_types():
    with pytest.raises(ValueError, match="int32"):
        dtp.layout_order(torch.zeros(4, dtype=torch.int64), 2)
    with pytest.raises(ValueError):
        dtp.permute_cols(torch.zeros(4, 8), torch.zeros(8, dtype=torch.int64))


def test_ablation_names_and_masks():
    for L in (1, 16, 28):
        mh, mn, mini = ablation.ablation_masks(L, "optimised")
        assert mh is None and mn is None and not mini
        mh, mn, mini = ablation.ablation_masks(L, "heads_only")
        assert mh.all() and not mn.any() and not mini
        mh, mn, mini = ablation.ablation_masks(L, "neurons_only")
        assert not mh.any() and mn.all()
        assert ablation.ablation_masks(L, "anti")[2]
    mh, mn, _ = ablation.ablation_masks(28, "layers8")
    assert np.flatnonzero(mh).tolist() == [0, 3, 7, 10, 14, 17, 21, 24] and np.array_equal(mh, mn)
    with pytest.raises(ValueError):
        ablation.ablation_masks(4, "sideways")
    with pytest.raises(ValueError):
        ablation.random_layout(2, 6, 64, 4, 1)


def test_affinity_opts_struct_layout():
    o = dtp.AffinityOpts(max_ctas=151)
    assert o.max_ctas == 151 and all(x == 0 for x in o.reserved)
    import ctypes
    assert ctypes.sizeof(dtp.AffinityOpts) == 32          # eight ints, as dtp_affinity_opts in dtp.h


def test_add_and_down_edge_reject_host_tensors():
    with pytest.raises(ValueError, match="CUDA"):
        dtp.affinity_add_accumulate(_bf16(2, 16, 64), _bf16(128, 64), _bf16(128, 64))
    with pytest.raises(ValueError, match="CUDA"):
        dtp.affinity_add_accumulate_grouped(_bf16(4, 16, 64), _bf16(128, 64), _bf16(128, 64), 2)
    with pytest.raises(ValueError, match="CUDA"):
        dtp.down_weight_sqnorm(_bf16(2, 24, 64), _bf16(64), _bf16(64, 128))
    with pytest.raises(ValueError, match="CUDA"):
        dtp.down_finalize(torch.zeros(128), torch.zeros(2, 128), 16)
