"""Minimal driver for profiling one kernel of the hot path under ncu.

Draws one seeded layer on the device and runs the chosen entry point a few
times, with nothing else in between, so that an ncu capture with
``-k regex:<kernel> -s 1 -c 1`` sees a warm launch after one warm-up.

    python -m paper_2609_13846_gb300.profile_case --what affinity --workload qwen3_0.6b_layer --launches 2
    python -m paper_2609_13846_gb300.profile_case --what search --workload qwen3_0.6b_model --D 4 --layers 28
    python -m paper_2609_13846_gb300.profile_case --what producer --workload qwen3_0.6b_layer --qrow 1
    python -m paper_2609_13846_gb300.profile_case --what gather --workload qwen3_0.6b_model --layers 28
    python -m paper_2609_13846_gb300.profile_case --what add --workload qwen3_0.6b_layer
"""
from __future__ import annotations

import argparse

import torch

from . import dtp, synth


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--what", choices=["affinity", "search", "producer", "gather", "add"], default="affinity")
    ap.add_argument("--qrow", type=int, default=1, help="producer: query heads per output row")
    ap.add_argument("--workload", default="qwen3_0.6b_layer")
    ap.add_argument("--T", type=int, default=None, help="token count (default: the workload's)")
    ap.add_argument("--launches", type=int, default=2)
    ap.add_argument("--D", type=int, default=None)
    ap.add_argument("--layers", type=int, default=1)
    args = ap.parse_args()
    w = synth.WORKLOADS[args.workload]
    dev = torch.device("cuda:0")
    if args.what == "affinity":
        L = synth.make_workload_layer(w, T=args.T, device=dev)
        T = L["X"].shape[0]
        A = torch.zeros((w.G, w.N), dtype=torch.float32, device=dev)
        ws = dtp.affinity_workspace(T, w.d, w.G, w.N, dtp.DTP_BF16 if w.dtype == "bf16" else dtp.DTP_F32, dev)
        torch.cuda.synchronize()
        for _ in range(args.launches):
            dtp.affinity_accumulate(L["X"], L["C"], L["W_gate"], L["W_up"], A=A, workspace=ws)
        torch.cuda.synchronize()
        print(f"affinity {args.workload} T={T}: {args.launches} launches, A sum {float(A.sum()):.6e}")
    elif args.what == "add":
        L = synth.make_workload_layer(w, T=args.T, device=dev)
        T = L["X"].shape[0]
        A = torch.zeros((w.G, w.N), dtype=torch.float32, device=dev)
        torch.cuda.synchronize()
        for _ in range(args.launches):
            dtp.affinity_add_accumulate(L["C"], L["W_gate"], L["W_up"], A_add=A)
        torch.cuda.synchronize()
        print(f"add {args.workload} T={T}: {args.launches} launches, A sum {float(A.sum()):.6e}")
    elif args.what == "producer":
        T = args.T or w.T
        P = synth.make_attention_inputs(T, w.d, w.G * w.q_per_group, w.head_dim, w.seed, device=dev)
        C = torch.empty(((w.G * w.q_per_group) // args.qrow, T, w.d), dtype=torch.bfloat16, device=dev)
        torch.cuda.synchronize()
        for _ in range(args.launches):
            dtp.head_writes(P["attn"], P["W_o"], P["gamma"], P["rms"], w.head_dim, args.qrow, out=C)
        torch.cuda.synchronize()
        print(f"producer {args.workload} T={T} rows={C.shape[0]}: {args.launches} launches")
    elif args.what == "gather":
        Wt = synth.make_dense_weights(args.layers, w.d, w.G * w.q_per_group, w.G, w.head_dim, w.N, w.seed,
                                      device=dev)
        D = args.D or w.D[-1]
        nu = torch.stack([torch.randperm(w.N, device=dev) % D for _ in range(args.layers)]).to(torch.int32)
        no = dtp.layout_order(nu, D)
        torch.cuda.synchronize()
        for _ in range(args.launches):
            dtp.permute_cols(Wt["down"], no, 1, check=False)
            dtp.permute_rows(Wt["gate"], no, 1, check=False)
        torch.cuda.synchronize()
        print(f"gather {args.workload} layers={args.layers}: {args.launches} launches each")
    else:
        As = torch.stack([synth.make_affinity_matrix(w.G, w.N, seed=w.seed + i, device="cpu")
                          for i in range(args.layers)]).to(dev).contiguous()
        D = args.D or w.D[0]
        for _ in range(args.launches):
            r = dtp.search_layout_batched(As, D, w.iters)
        print(f"search {args.workload} layers={args.layers} D={D}: mean score {float(r['score'].mean()):.6f}")


if __name__ == "__main__":
    main()
