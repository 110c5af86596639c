"""GB300-native hot path of affinity-aware sharding for Delayed Tensor Parallelism.

Implements, for sm_103a, the two data-parallel parts of "Affinity-Aware
Sharding for Delayed Tensor Parallelism" (arXiv 2609.13846), Sec. 3:

* the first-order head->neuron affinity A[kv_head, neuron] of one layer
  (a tcgen05/TMEM bf16 GEMM with a fused SwiGLU first-order epilogue and an
  on-chip token reduction; an fp32 CUDA-core mode for tight checks), and
* the coordinate-ascent layout optimiser (exact balanced neuron assignment,
  exhaustive labelled head-partition search, exact integer objective).

Both live in the C-ABI library ``libdtp.so`` (declared in ``include/dtp.h``);
:mod:`paper_2609_13846_gb300.dtp` is the thin ctypes binding.  Import of the
binding is lazy so that :mod:`paper_2609_13846_gb300.synth` (seeded inputs)
can be used without the compiled library.
"""

__all__ = ["dtp", "synth"]
