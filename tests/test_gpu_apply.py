"""GPU parity of the producer of C and of the layout application (Sec. 3) against the oracle.

Producer: C = gamma . (a_h W_o^(h)T) / r from bf16 attention outputs and o_proj,
rounded once to bf16: relative Frobenius error <= 5e-3 against the fp64 oracle
on the same bf16 inputs.  Layout application: index work, so the order and the
permuted weights are bit-exact against the oracle's.
"""
import numpy as np
import pytest
import torch

import oracle
from oracle import dense_block
from paper_2609_13846_gb300 import ablation, dtp, synth

pytestmark = pytest.mark.gpu
DEV = "cuda:0"
BF16_TOL = 5e-3


def _rel(a, b):
    a = np.asarray(a, np.float64)
    b = np.asarray(b, np.float64)
    return float(np.linalg.norm(a - b) / np.linalg.norm(b))


def _producer_inputs(T, d, Hq, hd, seed):
    g = torch.Generator().manual_seed(seed)
    attn = torch.randn((T, Hq * hd), generator=g).to(torch.bfloat16)
    Wo = (torch.randn((d, Hq * hd), generator=g) * 0.02).to(torch.bfloat16)
    gamma = 1.0 + 0.1 * torch.randn(d, generator=g)
    rms = 0.5 + torch.rand(T, generator=g)
    return attn, Wo, gamma, rms


@pytest.mark.parametrize("T,d,Hq,hd,q", [
    (300, 256, 16, 64, 1),
    (257, 1024, 16, 128, 2),     # Qwen3-0.6B: 16 query heads of 128, 2 per KV group
    (257, 1024, 16, 128, 1),
    (129, 1536, 16, 96, 2),      # Danube3-500M: head_dim 96 (K blocks of 64 + 32)
    (129, 1536, 16, 96, 1),
    (64, 328, 6, 48, 3),         # ragged d (a partial 64-column box), K = 48 and 144
    (1, 64, 2, 16, 1)])
def test_head_writes_match_oracle(T, d, Hq, hd, q):
    attn, Wo, gamma, rms = _producer_inputs(T, d, Hq, hd, seed=T + d + q)
    C = dtp.head_writes(attn.to(DEV), Wo.to(DEV), gamma.to(DEV), rms.to(DEV), hd, q, check=True)
    torch.cuda.synchronize()
    assert C.shape == (Hq // q, T, d) and C.dtype == torch.bfloat16
    ref = oracle.head_writes(attn.double().numpy(), Wo.double().numpy(), gamma.double().numpy(),
                             rms.double().numpy(), hd, q)
    assert _rel(C.float().cpu().numpy(), ref) <= BF16_TOL


def test_head_writes_silent_head_and_row_sums():
    T, d, Hq, hd = 200, 512, 8, 64
    attn, Wo, gamma, rms = _producer_inputs(T, d, Hq, hd, seed=3)
    attn[:, 3 * hd:4 * hd] = 0
    a, w, gm, r = attn.to(DEV), Wo.to(DEV), gamma.to(DEV), rms.to(DEV)
    per = dtp.head_writes(a, w, gm, r, hd, 1, check=True)
    grp = dtp.head_writes(a, w, gm, r, hd, 2, check=True)
    torch.cuda.synchronize()
    assert not per[3].any()
    summed = per.float().reshape(4, 2, T, d).sum(1)
    assert _rel(grp.float().cpu().numpy(), summed.cpu().numpy()) <= BF16_TOL


def test_producer_feeds_the_per_query_head_affinity():
    """attention outputs -> C per query head -> first-order score summed per KV group, against the
    oracle's C and score in fp64."""
    T, d, Hq, hd, q, N = 256, 512, 8, 64, 2, 384
    attn, Wo, gamma, rms = _producer_inputs(T, d, Hq, hd, seed=4)
    L = synth.make_layer(d, 1, N, T, seed=5, dtype="bf16")
    g = {k: v.to(DEV) for k, v in L.items()}
    C = dtp.head_writes(attn.to(DEV), Wo.to(DEV), gamma.to(DEV), rms.to(DEV), hd, 1, check=True)
    A = dtp.affinity_accumulate_grouped(g["X"], C, g["W_gate"], g["W_up"], q)
    torch.cuda.synchronize()
    C_ref = oracle.head_writes(attn.double().numpy(), Wo.double().numpy(), gamma.double().numpy(),
                               rms.double().numpy(), hd, 1)
    A_ref = oracle.affinity_fo_qheads(L["X"].double().numpy(), C_ref, L["W_gate"].double().numpy(),
                                      L["W_up"].double().numpy(), q)
    assert _rel(A.cpu().numpy(), A_ref) <= 2 * BF16_TOL     # C rounded to bf16, then A's own error
    A_same = oracle.affinity_fo_qheads(L["X"].double().numpy(), C.double().cpu().numpy(),
                                       L["W_gate"].double().numpy(), L["W_up"].double().numpy(), q)
    assert _rel(A.cpu().numpy(), A_same) <= BF16_TOL


@pytest.mark.parametrize("layers,n,D", [(3, 8, 4), (28, 3072, 4), (2, 14336, 8), (5, 96, 3), (1, 2, 2)])
def test_layout_order_bit_exact(layers, n, D):
    rng = np.random.default_rng(n + D)
    lab = np.stack([rng.permutation(np.repeat(np.arange(D), n // D)) for _ in range(layers)]).astype(np.int32)
    out = dtp.layout_order(torch.as_tensor(lab, device=DEV), D).cpu().numpy()
    for i in range(layers):
        np.testing.assert_array_equal(out[i], oracle.layout_order(lab[i], D))


def test_layout_order_unbalanced_and_invalid():
    lab = np.array([[0, 0, 1, 0, 2, 2, 0]], np.int32)
    out = dtp.layout_order(torch.as_tensor(lab, device=DEV), 3, balanced=False).cpu().numpy()
    np.testing.assert_array_equal(out[0], oracle.layout_order(lab[0], 3))
    with pytest.raises(dtp.DTPError):
        dtp.layout_order(torch.as_tensor(np.array([[0, 0, 1, 1, 2, 0]], np.int32), device=DEV), 3)
    with pytest.raises(dtp.DTPError):
        dtp.layout_order(torch.as_tensor(np.array([[0, 3, 1, 1]], np.int32), device=DEV), 2)


def _qwen_like_layer(d, Hq, G, hd, N, seed):
    W = dense_block.random_layer(d, Hq, G, hd, N, seed)
    return {k: torch.as_tensor(v, dtype=torch.float32).to(torch.bfloat16) for k, v in W.items()}


@pytest.mark.parametrize("d,Hq,G,hd,N,D", [(1024, 16, 8, 128, 3072, 4), (1536, 16, 8, 96, 4096, 4),
                                           (64, 8, 4, 16, 48, 2), (40, 6, 3, 8, 30, 3)])
def test_apply_layout_bit_exact(d, Hq, G, hd, N, D):
    W = _qwen_like_layer(d, Hq, G, hd, N, seed=N)
    h, nu = ablation.random_layout(1, G, N, D, 1000)
    gW = {k: v.to(DEV).contiguous() for k, v in W.items()}
    out, ho, no = dtp.apply_layout(gW, torch.as_tensor(h[0], device=DEV), torch.as_tensor(nu[0], device=DEV), D, hd)
    ref, rho, rno = dense_block.apply_layout({k: v.float().numpy() for k, v in W.items()}, h[0], nu[0], D, G, hd)
    np.testing.assert_array_equal(ho.cpu().numpy(), rho)
    np.testing.assert_array_equal(no.cpu().numpy(), rno)
    for k in ("q", "k", "v", "o", "gate", "up", "down"):
        assert torch.equal(out[k].cpu().float(), torch.as_tensor(ref[k], dtype=torch.float32)), k


def test_apply_layout_batched_over_layers_and_dense_function():
    """Four layers stacked [L, ...]: each layer gathered with its own permutation; the permuted
    small block computes the same dense function in fp64."""
    Lyr, d, Hq, G, hd, N, D = 4, 64, 8, 4, 16, 64, 2
    Ws = [_qwen_like_layer(d, Hq, G, hd, N, seed=10 + i) for i in range(Lyr)]
    stacked = {k: torch.stack([w[k] for w in Ws]).to(DEV).contiguous() for k in Ws[0]}
    h, nu = ablation.random_layout(Lyr, G, N, D, 1003)
    out, _, _ = dtp.apply_layout(stacked, torch.as_tensor(h, device=DEV), torch.as_tensor(nu, device=DEV), D, hd)
    x = np.random.default_rng(0).standard_normal((12, d))
    for i in range(Lyr):
        Wi = {k: Ws[i][k].double().numpy() for k in Ws[i]}
        Wp = {k: out[k][i].double().cpu().numpy() for k in out}
        np.testing.assert_allclose(dense_block.block(x, Wp, G, hd), dense_block.block(x, Wi, G, hd),
                                   rtol=1e-10, atol=1e-10)
        ref, _, _ = dense_block.apply_layout(Wi, h[i], nu[i], D, G, hd)
        for k in ("q", "o", "down"):
            np.testing.assert_array_equal(Wp[k], ref[k])


def test_permute_rejects_out_of_range_entries():
    src = torch.randn(8, 16, device=DEV).to(torch.bfloat16)
    bad = torch.tensor([0, 1, 9, 3], dtype=torch.int32, device=DEV)
    with pytest.raises(dtp.DTPError) as e:
        dtp.permute_rows(src, bad, 2)
    assert e.value.status == dtp.DTP_ERR_ARG
    with pytest.raises(dtp.DTPError):
        dtp.permute_cols(src, torch.tensor([0, -1], dtype=torch.int32, device=DEV), 8)


@pytest.mark.parametrize("dtype,rows,cols,block", [
    (torch.float32, 64, 96, 1), (torch.float32, 40, 30, 3), (torch.bfloat16, 33, 3072, 1),
    (torch.bfloat16, 16, 24, 8), (torch.uint8, 10, 48, 3), (torch.uint8, 7, 21, 7), (torch.float64, 9, 12, 2),
    (torch.float64, 8, 14, 1), (torch.uint8, 12, 64, 1), (torch.bfloat16, 5, 14336, 1), (torch.float32, 3, 4100, 2)])
def test_gathers_match_indexing(dtype, rows, cols, block):
    """Every width path of the gathers (16-byte words, packed elements, plain elements) against
    plain indexing, on two stacked layers with different permutations."""
    rng = np.random.default_rng(rows + cols)
    src = torch.randint(0, 250, (2, rows, cols)).to(dtype)
    pc = np.stack([rng.permutation(cols // block) for _ in range(2)]).astype(np.int32)
    rb = 1 if rows % 2 else 2
    pr = np.stack([rng.permutation(rows // rb) for _ in range(2)]).astype(np.int32)
    got_c = dtp.permute_cols(src.to(DEV), torch.as_tensor(pc, device=DEV), block).cpu()
    got_r = dtp.permute_rows(src.to(DEV), torch.as_tensor(pr, device=DEV), rb).cpu()
    for i in range(2):
        ci = np.concatenate([np.arange(b * block, (b + 1) * block) for b in pc[i]])
        ri = np.concatenate([np.arange(b * rb, (b + 1) * rb) for b in pr[i]])
        assert torch.equal(got_c[i], src[i][:, ci])
        assert torch.equal(got_r[i], src[i][ri])


def test_staged_column_gather_rejects_out_of_range_entries():
    """One-column blocks of a bf16 matrix (the packed path with vector permutation reads); a bad entry is reported."""
    src = torch.randn(4, 32, device=DEV).to(torch.bfloat16)
    perm = torch.arange(32, dtype=torch.int32, device=DEV)
    assert torch.equal(dtp.permute_cols(src, perm, 1), src)
    perm[5] = 32
    with pytest.raises(dtp.DTPError) as e:
        dtp.permute_cols(src, perm, 1)
    assert e.value.status == dtp.DTP_ERR_ARG


@pytest.mark.parametrize("layers,rows,cols", [(28, 1024, 3072), (1, 4096, 14336), (16, 1536, 4096)])
def test_down_column_gather_at_model_size(layers, rows, cols):
    """The down_proj column gather (one column per neuron, rows staged in shared memory) at the
    Qwen3-0.6B (28 layers), Llama-3.1-8B and Danube3-500M shapes: bit-exact against indexing."""
    g = torch.Generator(device=DEV).manual_seed(cols)
    src = torch.randn((layers, rows, cols), device=DEV, generator=g).to(torch.bfloat16)
    perm = torch.stack([torch.randperm(cols, device=DEV, generator=g) for _ in range(layers)]).to(torch.int32)
    got = dtp.permute_cols(src, perm, 1)
    ref = torch.gather(src, 2, perm.long().unsqueeze(1).expand(layers, rows, cols))
    assert torch.equal(got, ref)



@pytest.mark.parametrize("dtype,rows,cols", [(torch.bfloat16, 40, 3072), (torch.float32, 9, 100)])
def test_column_gather_with_padded_permutation_rows(dtype, rows, cols):
    """Through the C ABI with perm_layer_stride larger than the permutation (layers' entries padded
    apart, as a C caller may lay them out): each layer uses its own entries only."""
    layers, pad = 3, 5
    g = torch.Generator().manual_seed(cols)
    src = torch.randint(0, 250, (layers, rows, cols), generator=g).to(dtype).to(DEV)
    perms = [torch.randperm(cols, generator=g) for _ in range(layers)]
    padded = torch.full((layers, cols + pad), -7, dtype=torch.int32)   # padding would be out of range
    for i, p in enumerate(perms):
        padded[i, :cols] = p.to(torch.int32)
    padded = padded.to(DEV)
    dst = torch.empty_like(src)
    ws = torch.zeros(256, dtype=torch.uint8, device=DEV)
    st = dtp.lib().dtp_permute_cols(dtp._ptr(src), dtp._ptr(dst), layers, rows, cols, src.element_size(), 1,
                                    dtp._ptr(padded), cols + pad, dtp._ptr(ws), ws.numel(), dtp._stream(None))
    assert st == dtp.DTP_OK
    assert dtp.workspace_status(ws) == dtp.DTP_OK
    for i, p in enumerate(perms):
        assert torch.equal(dst[i].cpu(), src[i].cpu()[:, p])


def test_row_gather_with_padded_permutation_rows():
    """dtp_permute_rows through the C ABI with perm_layer_stride larger than the permutation."""
    layers, rows, cols, block, pad = 3, 48, 64, 2, 3
    g = torch.Generator().manual_seed(7)
    src = torch.randint(0, 250, (layers, rows, cols), generator=g).to(torch.bfloat16).to(DEV)
    nb = rows // block
    perms = [torch.randperm(nb, generator=g) for _ in range(layers)]
    padded = torch.full((layers, nb + pad), -3, dtype=torch.int32)
    for i, p in enumerate(perms):
        padded[i, :nb] = p.to(torch.int32)
    padded = padded.to(DEV)
    dst = torch.empty_like(src)
    ws = torch.zeros(256, dtype=torch.uint8, device=DEV)
    st = dtp.lib().dtp_permute_rows(dtp._ptr(src), dtp._ptr(dst), layers, rows, cols * src.element_size(), block,
                                    dtp._ptr(padded), nb + pad, dtp._ptr(ws), ws.numel(), dtp._stream(None))
    assert st == dtp.DTP_OK
    assert dtp.workspace_status(ws) == dtp.DTP_OK
    for i, p in enumerate(perms):
        idx = torch.cat([torch.arange(b * block, (b + 1) * block) for b in p.tolist()])
        assert torch.equal(dst[i].cpu(), src[i].cpu()[idx])
