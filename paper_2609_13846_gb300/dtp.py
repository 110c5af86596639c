"""ctypes binding of libdtp.so (include/dtp.h), argument marshalling only.

Every computation runs in the library's CUDA kernels; this module checks
tensor shapes, dtypes and devices, allocates caller-side outputs and
workspaces with PyTorch, and passes raw device pointers plus the current CUDA
stream.  It raises if the library was not built: there is no CPU fallback.
"""
from __future__ import annotations

import ctypes
import os

import torch

_PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_PKG, "libdtp.so")

DTP_OK = 0
DTP_ERR_ARG = -1
DTP_ERR_CUDA = -2
DTP_ERR_NOT_CONVERGED = -3
DTP_ERR_UNSUPPORTED = -4
DTP_ERR_WORKSPACE = -5
DTP_BF16 = 0
DTP_F32 = 1
DTP_AFFINITY_DEFER_REDUCE = 1

_lib = None

_vp = ctypes.c_void_p
_i64 = ctypes.c_int64
_i32 = ctypes.c_int
_sz = ctypes.c_size_t


class AffinityOpts(ctypes.Structure):
    """dtp_affinity_opts: max_ctas caps the persistent grid (0 = one CTA per SM; rounded down to an
    even count when the kernel runs as CTA pairs)."""
    _fields_ = [("max_ctas", ctypes.c_int), ("flags", ctypes.c_int), ("reserved", ctypes.c_int * 6)]


class DTPError(RuntimeError):
    """A libdtp call returned a non-zero dtp_status."""

    def __init__(self, fn: str, status: int):
        self.status = status
        super().__init__(f"{fn}: {status_string(status)} ({status})")


def lib():
    """Load libdtp.so (built by ``paper_2609_13846_gb300.build``)."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(LIB_PATH):
        raise RuntimeError(f"{LIB_PATH} is missing: build it with `python -m paper_2609_13846_gb300.build`")
    L = ctypes.CDLL(LIB_PATH)
    L.dtp_version.restype = _i32
    L.dtp_status_string.argtypes = [_i32]
    L.dtp_status_string.restype = ctypes.c_char_p
    L.dtp_affinity_workspace_size.argtypes = [_i64, _i32, _i32, _i32, _i32, ctypes.POINTER(_sz)]
    L.dtp_affinity_accumulate.argtypes = [_vp, _vp, _vp, _vp, _i64, _i32, _i32, _i32, _i32, _vp, _vp, _sz, _vp]
    L.dtp_affinity_finalize.argtypes = [_vp, _i32, _i32, _i64, _vp, _vp]
    L.dtp_down_sqnorm.argtypes = [_vp, _i32, _i32, _i32, _vp, _vp]
    L.dtp_affinity_accumulate_noalloc.argtypes = [_vp, _vp, _vp, _vp, _i64, _i32, _i32, _i32, _vp, _vp]
    L.dtp_affinity_noalloc_status.argtypes = [_vp]
    L.dtp_affinity_accumulate_ex.argtypes = [_vp, _vp, _vp, _vp, _vp, _i64, _i32, _i32, _i32, _i32, _vp, _vp, _vp,
                                             _sz, _vp]
    L.dtp_affinity_grouped_workspace_size.argtypes = [_i64, _i32, _i32, _i32, _i32, _i32, ctypes.POINTER(_sz)]
    L.dtp_affinity_accumulate_grouped.argtypes = [_vp, _vp, _vp, _vp, _vp, _i64, _i32, _i32, _i32, _i32, _i32, _vp,
                                                  _vp, _vp, _sz, _vp]
    L.dtp_affinity_add_grouped_workspace_size.argtypes = [_i64, _i32, _i32, _i32, _i32, ctypes.POINTER(_sz)]
    L.dtp_affinity_add_accumulate_grouped.argtypes = [_vp, _vp, _vp, _i64, _i32, _i32, _i32, _i32, _vp, _vp, _sz,
                                                      _vp]
    L.dtp_affinity_accumulate_opts.argtypes = [_vp, _vp, _vp, _vp, _vp, _i64, _i32, _i32, _i32, _i32, _vp, _vp,
                                               ctypes.POINTER(AffinityOpts), _vp, _sz, _vp]
    L.dtp_affinity_reduce.argtypes = [_vp, _sz, _i64, _i32, _i32, _i32, _vp, _vp, _i32, _i32, _vp]
    L.dtp_affinity_add_workspace_size.argtypes = [_i64, _i32, _i32, _i32, ctypes.POINTER(_sz)]
    L.dtp_affinity_add_accumulate.argtypes = [_vp, _vp, _vp, _i64, _i32, _i32, _i32, _vp, _vp, _sz, _vp]
    L.dtp_down_weight_workspace_size.argtypes = [_i32, _i32, _i32, _i32, ctypes.POINTER(_sz)]
    L.dtp_down_weight_sqnorm.argtypes = [_vp, _vp, _vp, _i32, _i32, _i32, _i32, _i32, _vp, _vp, _sz, _vp]
    L.dtp_down_finalize.argtypes = [_vp, _vp, _i32, _i32, _i64, _vp, _vp]
    L.dtp_search_chain_workspace_size.argtypes = [_i32, _i32, _i32, _i32, ctypes.POINTER(_sz)]
    L.dtp_search_chain.argtypes = [_vp, _vp, _i32, _i32, _i32, _i32, _i32, _vp, _vp, _vp, _vp, _vp, _vp, _sz, _vp]
    L.dtp_search_chain_ex.argtypes = [_vp, _vp, _i32, _i32, _i32, _i32, _i32, _vp, _vp, _i32, _vp, _vp, _vp, _vp,
                                      _vp, _vp, _sz, _vp]
    L.dtp_chain_score.argtypes = [_vp, _vp, _i32, _i32, _i32, _i32, _vp, _vp, _vp, _vp, _vp, _vp, _sz, _vp]
    L.dtp_head_writes_workspace_size.argtypes = [ctypes.POINTER(_sz)]
    L.dtp_head_writes.argtypes = [_vp, _vp, _vp, _vp, _i64, _i32, _i32, _i32, _i32, _vp, _vp, _sz, _vp]
    L.dtp_layout_order.argtypes = [_vp, _i32, _i32, _i32, _i32, _vp, _vp, _sz, _vp]
    L.dtp_permute_rows.argtypes = [_vp, _vp, _i32, _i64, _i64, _i32, _vp, _i64, _vp, _sz, _vp]
    L.dtp_permute_cols.argtypes = [_vp, _vp, _i32, _i64, _i64, _i32, _i32, _vp, _i64, _vp, _sz, _vp]
    L.dtp_search_global_workspace_size.argtypes = [_i32, _i32, _i32, _i32, ctypes.POINTER(_sz)]
    L.dtp_search_global.argtypes = [_vp, _i32, _i32, _i32, _i32, _vp, _vp, _vp, _vp, _vp, _sz, _vp]
    L.dtp_apply_layout.argtypes = [_vp, _vp, _i32, _i32, _i32, _i32, _i32, _i32, _i32, _i32,
                                   ctypes.POINTER(_vp), ctypes.POINTER(_vp), _vp, _vp, _vp, _sz, _vp]
    L.dtp_affinity_top_share.argtypes = [_vp, _i32, _i32, _i32, _vp, _vp]
    L.dtp_workspace_status.argtypes = [_vp, _sz, _vp]
    L.dtp_selftest_bounded_wait.argtypes = [ctypes.c_uint64, _i32, _vp, _sz, ctypes.POINTER(ctypes.c_uint64), _vp]
    L.dtp_search_workspace_size.argtypes = [_i32, _i32, _i32, _i32, ctypes.POINTER(_sz)]
    L.dtp_search_layout.argtypes = [_vp, _i32, _i32, _i32, _i32, _vp, _vp, _vp, _vp, _vp, _vp, _sz, _vp]
    L.dtp_search_layout_batched.argtypes = [_vp, _i32, _i32, _i32, _i32, _i32, _vp, _vp, _vp, _vp, _vp, _vp, _sz,
                                            _vp]
    for fn in ("dtp_search_chain_workspace_size", "dtp_search_chain", "dtp_search_chain_ex", "dtp_chain_score",
               "dtp_affinity_grouped_workspace_size", "dtp_affinity_accumulate_grouped",
               "dtp_head_writes_workspace_size", "dtp_head_writes", "dtp_layout_order", "dtp_permute_rows",
               "dtp_affinity_accumulate_opts", "dtp_search_global_workspace_size", "dtp_search_global",
               "dtp_affinity_reduce", "dtp_apply_layout", "dtp_affinity_top_share",
               "dtp_permute_cols",
               "dtp_affinity_add_grouped_workspace_size", "dtp_affinity_add_accumulate_grouped",
               "dtp_affinity_accumulate_ex", "dtp_affinity_add_workspace_size", "dtp_affinity_add_accumulate",
               "dtp_down_weight_workspace_size", "dtp_down_weight_sqnorm", "dtp_down_finalize",
               "dtp_affinity_workspace_size", "dtp_affinity_accumulate", "dtp_affinity_accumulate_noalloc",
               "dtp_affinity_noalloc_status", "dtp_affinity_finalize",
               "dtp_down_sqnorm", "dtp_workspace_status", "dtp_search_workspace_size", "dtp_search_layout",
               "dtp_search_layout_batched", "dtp_selftest_bounded_wait"):
        getattr(L, fn).restype = _i32
    _lib = L
    return L


def status_string(status: int) -> str:
    return lib().dtp_status_string(int(status)).decode()


def _check(fn: str, status: int):
    if status != DTP_OK:
        raise DTPError(fn, status)


def _stream(stream=None) -> int:
    s = torch.cuda.current_stream() if stream is None else stream
    return int(s.cuda_stream)


def _keep(t: torch.Tensor, stream) -> torch.Tensor:
    """Mark a temporary as in use on ``stream`` so the caching allocator does not hand it out early."""
    if stream is not None:
        t.record_stream(stream)
    return t


def _device_mask(m, L: int, dev, stream) -> torch.Tensor | None:
    if m is None:
        return None
    t = torch.as_tensor(m).reshape(-1)
    if t.numel() != L:
        raise ValueError(f"layer mask must have {L} entries, got {t.numel()}")
    return _keep((t != 0).to(torch.uint8).to(dev).contiguous(), stream)


def _ptr(t: torch.Tensor | None):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _dtype_code(t: torch.Tensor) -> int:
    if t.dtype == torch.bfloat16:
        return DTP_BF16
    if t.dtype == torch.float32:
        return DTP_F32
    raise TypeError(f"unsupported dtype {t.dtype}; use bfloat16 or float32")


def affinity_workspace_size(T: int, d: int, H_kv: int, N: int, dtype: int) -> int:
    n = _sz(0)
    _check("dtp_affinity_workspace_size", lib().dtp_affinity_workspace_size(T, d, H_kv, N, dtype, ctypes.byref(n)))
    return n.value


def affinity_workspace(T: int, d: int, H_kv: int, N: int, dtype: int, device) -> torch.Tensor:
    """A device workspace tensor sized for these arguments."""
    return torch.empty(affinity_workspace_size(T, d, H_kv, N, dtype), dtype=torch.uint8, device=device)


def _cuda_contig(device, **tensors):
    """Every tensor contiguous and on ``device`` (a CUDA device), else ValueError."""
    for name, t in tensors.items():
        if not t.is_cuda or not t.is_contiguous() or t.device != device:
            raise ValueError(f"{name} must be a contiguous CUDA tensor on the inputs' device")


def _add_shapes(C, W_gate, W_up):
    """C [H,T,d], W_gate/W_up [N,d], all bf16 CUDA tensors on one device; returns (H, T, d, N)."""
    if not C.is_cuda:
        raise ValueError("C must be a contiguous CUDA tensor")
    _cuda_contig(C.device, C=C, W_gate=W_gate, W_up=W_up)
    if not (C.dtype == W_gate.dtype == W_up.dtype == torch.bfloat16):
        raise TypeError("C, W_gate and W_up must be bf16")
    if C.dim() != 3 or W_gate.dim() != 2:
        raise ValueError("shapes must be C [H,T,d], W_gate [N,d], W_up [N,d]")
    H, T, d = C.shape
    N = W_gate.shape[0]
    if W_gate.shape != (N, d) or W_up.shape != (N, d):
        raise ValueError("shapes must be C [H,T,d], W_gate [N,d], W_up [N,d]")
    return H, T, d, N


def _check_f32_out(name, t, shape, device):
    if t.shape != shape or t.dtype != torch.float32 or not t.is_contiguous() or t.device != device:
        raise ValueError(f"{name} must be a contiguous fp32 {list(shape)} tensor on the inputs' device")


def _affinity_shapes(X, C, W_gate, W_up):
    """Check the affinity inputs (contiguous CUDA tensors of one dtype on one device, X [T,d],
    C [H,T,d], W_gate/W_up [N,d]) and return (T, d, H, N)."""
    for name, t in (("X", X), ("C", C), ("W_gate", W_gate), ("W_up", W_up)):
        if not t.is_cuda or not t.is_contiguous():
            raise ValueError(f"{name} must be a contiguous CUDA tensor")
        if t.device != X.device:
            raise ValueError(f"{name} must be on X's device")
    if not (X.dtype == C.dtype == W_gate.dtype == W_up.dtype):
        raise TypeError("X, C, W_gate and W_up must share one dtype")
    if X.dim() != 2 or C.dim() != 3:
        raise ValueError("shapes must be X [T,d], C [H,T,d], W_gate [N,d], W_up [N,d]")
    T, d = X.shape
    H = C.shape[0]
    N = W_gate.shape[0]
    if C.shape != (H, T, d) or W_gate.shape != (N, d) or W_up.shape != (N, d):
        raise ValueError("shapes must be X [T,d], C [H,T,d], W_gate [N,d], W_up [N,d]")
    return T, d, H, N


def affinity_accumulate(X: torch.Tensor, C: torch.Tensor, W_gate: torch.Tensor, W_up: torch.Tensor,
                        A: torch.Tensor | None = None, workspace: torch.Tensor | None = None,
                        stream=None, max_ctas: int = 0, defer_reduce: bool = False) -> torch.Tensor:
    """A[h,k] += sum_t Delta_{t,h,k}^2 (Sec. 3); returns A [H_kv, N] fp32 on X's device.

    X [T,d], C [H_kv,T,d], W_gate/W_up [N,d]: contiguous CUDA tensors, all bf16
    or all fp32.  ``A`` is accumulated into (a zero tensor is made if None).
    max_ctas > 0 caps the bf16 kernel's persistent grid (SMs left to other streams; rounded down
    to an even count, at least 2, when the kernel runs as CTA pairs); with defer_reduce only the
    main kernel runs and affinity_reduce(workspace, ...) finishes A later.
    """
    T, d, H, N = _affinity_shapes(X, C, W_gate, W_up)
    code = _dtype_code(X)
    if A is None:
        A = torch.zeros((H, N), dtype=torch.float32, device=X.device)
    if A.shape != (H, N) or A.dtype != torch.float32 or not A.is_contiguous() or A.device != X.device:
        raise ValueError("A must be a contiguous fp32 [H_kv, N] tensor on X's device")
    if workspace is None:
        workspace = affinity_workspace(T, d, H, N, code, X.device)
    if max_ctas or defer_reduce:
        opts = AffinityOpts(max_ctas=int(max_ctas), flags=DTP_AFFINITY_DEFER_REDUCE if defer_reduce else 0)
        st = lib().dtp_affinity_accumulate_opts(_ptr(X), _ptr(C), _ptr(W_gate), _ptr(W_up), None, T, d, H, N, code,
                                                _ptr(A), None, ctypes.byref(opts), _ptr(workspace), workspace.numel(),
                                                _stream(stream))
        _check("dtp_affinity_accumulate_opts", st)
        return A
    st = lib().dtp_affinity_accumulate(_ptr(X), _ptr(C), _ptr(W_gate), _ptr(W_up), T, d, H, N, code, _ptr(A),
                                       _ptr(workspace), workspace.numel(), _stream(stream))
    _check("dtp_affinity_accumulate", st)
    return A


def top_group_share(A: torch.Tensor, stream=None) -> torch.Tensor:
    """Mean over neurons of the largest KV group's share of the neuron's affinity (Sec. 5), per layer.
    A [L, H_kv, N] (or [H_kv, N]) fp32 CUDA; returns float64 [L] (or a scalar)."""
    x = A.unsqueeze(0) if A.dim() == 2 else A
    if x.dtype != torch.float32 or not x.is_cuda or not x.is_contiguous():
        raise ValueError("A must be a contiguous fp32 CUDA tensor")
    out = _keep(torch.empty(x.shape[0], dtype=torch.float64, device=x.device), stream)
    _check("dtp_affinity_top_share", lib().dtp_affinity_top_share(_ptr(x), x.shape[0], x.shape[1], x.shape[2],
                                                                  _ptr(out), _stream(stream)))
    return out if A.dim() == 3 else out[0]


def affinity_reduce(workspace: torch.Tensor, T: int, d: int, H_kv: int, N: int, A: torch.Tensor,
                    act2: torch.Tensor | None = None, stream=None, max_blocks: int = 0,
                    overwrite: bool = False) -> torch.Tensor:
    """Add (or, with overwrite, store) the unit partials a deferred affinity pass left in
    ``workspace`` into A (and act2); max_blocks > 0 runs it as that many 1024-thread blocks."""
    if A.shape != (H_kv, N) or A.dtype != torch.float32 or not A.is_cuda or not A.is_contiguous():
        raise ValueError("A must be a contiguous fp32 CUDA tensor [H_kv, N]")
    st = lib().dtp_affinity_reduce(_ptr(workspace), workspace.numel(), T, d, H_kv, N, _ptr(A), _ptr(act2),
                                   int(max_blocks), int(bool(overwrite)), _stream(stream))
    _check("dtp_affinity_reduce", st)
    return A


def affinity_accumulate_down(X: torch.Tensor, C: torch.Tensor, W_gate: torch.Tensor, W_up: torch.Tensor,
                             rms_next: torch.Tensor, A: torch.Tensor | None = None, act2: torch.Tensor | None = None,
                             workspace: torch.Tensor | None = None, stream=None):
    """The affinity pass plus the down-edge activation term (Sec. 3).

    A[h,k] += sum_t Delta^2 as in affinity_accumulate, and act2[k] += sum_t
    (silu(g_k) u_k)^2 / rms_next[t]^2 with rms_next [T] fp32 the rms of the
    residual entering the next layer's pre-norm.  Returns (A, act2).
    """
    T, d, H, N = _affinity_shapes(X, C, W_gate, W_up)
    code = _dtype_code(X)
    if A is None:
        A = torch.zeros((H, N), dtype=torch.float32, device=X.device)
    if act2 is None:
        act2 = torch.zeros(N, dtype=torch.float32, device=X.device)
    _check_f32_out("A", A, (H, N), X.device)
    _check_f32_out("act2", act2, (N,), X.device)
    _check_f32_out("rms_next", rms_next, (T,), X.device)
    if workspace is None:
        workspace = affinity_workspace(T, d, H, N, code, X.device)
    st = lib().dtp_affinity_accumulate_ex(_ptr(X), _ptr(C), _ptr(W_gate), _ptr(W_up), _ptr(rms_next), T, d, H, N,
                                          code, _ptr(A), _ptr(act2), _ptr(workspace), workspace.numel(),
                                          _stream(stream))
    _check("dtp_affinity_accumulate_ex", st)
    return A, act2


def affinity_grouped_workspace_size(T: int, d: int, H_q: int, q_per_group: int, N: int, dtype: int) -> int:
    n = _sz(0)
    _check("dtp_affinity_grouped_workspace_size",
           lib().dtp_affinity_grouped_workspace_size(T, d, H_q, q_per_group, N, dtype, ctypes.byref(n)))
    return n.value


def affinity_accumulate_grouped(X: torch.Tensor, C_q: torch.Tensor, W_gate: torch.Tensor, W_up: torch.Tensor,
                                q_per_group: int, A: torch.Tensor | None = None, rms_next: torch.Tensor | None = None,
                                act2: torch.Tensor | None = None, workspace: torch.Tensor | None = None,
                                stream=None):
    """First-order score per query head, summed over each KV group's query heads (Sec. 3).

    C_q [H_q, T, d] holds each query head's write; A [H_q / q_per_group, N] fp32
    is accumulated into.  With rms_next [T] the down-edge activation term is
    added to act2 [N] as in affinity_accumulate_down.  Returns A, or (A, act2)
    when rms_next is given.
    """
    T, d, Hq, N = _affinity_shapes(X, C_q, W_gate, W_up)
    if q_per_group < 1 or Hq % q_per_group:
        raise ValueError("q_per_group must divide H_q")
    code = _dtype_code(X)
    if A is None:
        A = torch.zeros((Hq // q_per_group, N), dtype=torch.float32, device=X.device)
    _check_f32_out("A", A, (Hq // q_per_group, N), X.device)
    if rms_next is not None:
        _check_f32_out("rms_next", rms_next, (T,), X.device)
        if act2 is None:
            act2 = torch.zeros(N, dtype=torch.float32, device=X.device)
        _check_f32_out("act2", act2, (N,), X.device)
    if workspace is None:
        workspace = _keep(torch.empty(affinity_grouped_workspace_size(T, d, Hq, q_per_group, N, code),
                                      dtype=torch.uint8, device=X.device), stream)
    st = lib().dtp_affinity_accumulate_grouped(_ptr(X), _ptr(C_q), _ptr(W_gate), _ptr(W_up), _ptr(rms_next), T, d,
                                               Hq, q_per_group, N, code, _ptr(A),
                                               _ptr(act2) if rms_next is not None else None, _ptr(workspace),
                                               workspace.numel(), _stream(stream))
    _check("dtp_affinity_accumulate_grouped", st)
    return (A, act2) if rms_next is not None else A


def affinity_add_accumulate_grouped(C_q: torch.Tensor, W_gate: torch.Tensor, W_up: torch.Tensor, q_per_group: int,
                                    A_add: torch.Tensor | None = None, workspace: torch.Tensor | None = None,
                                    stream=None) -> torch.Tensor:
    """ADD score per query head, summed over each KV group's query heads (Sec. 3); bf16 inputs."""
    Hq, T, d, N = _add_shapes(C_q, W_gate, W_up)
    if q_per_group < 1 or Hq % q_per_group:
        raise ValueError("q_per_group must divide H_q")
    if A_add is None:
        A_add = torch.zeros((Hq // q_per_group, N), dtype=torch.float32, device=C_q.device)
    _check_f32_out("A_add", A_add, (Hq // q_per_group, N), C_q.device)
    if workspace is None:
        n = _sz(0)
        _check("dtp_affinity_add_grouped_workspace_size",
               lib().dtp_affinity_add_grouped_workspace_size(T, d, Hq, q_per_group, N, ctypes.byref(n)))
        workspace = _keep(torch.empty(n.value, dtype=torch.uint8, device=C_q.device), stream)
    st = lib().dtp_affinity_add_accumulate_grouped(_ptr(C_q), _ptr(W_gate), _ptr(W_up), T, d, Hq, q_per_group, N,
                                                   _ptr(A_add), _ptr(workspace), workspace.numel(), _stream(stream))
    _check("dtp_affinity_add_accumulate_grouped", st)
    return A_add


def affinity_add_accumulate(C: torch.Tensor, W_gate: torch.Tensor, W_up: torch.Tensor,
                            A_add: torch.Tensor | None = None, workspace: torch.Tensor | None = None,
                            stream=None) -> torch.Tensor:
    """ADD score before the mean (Sec. 3): A_add[h,k] += sum_t (p_h.w^g_k)^2 + (p_h.w^u_k)^2; bf16 inputs."""
    H, T, d, N = _add_shapes(C, W_gate, W_up)
    if A_add is None:
        A_add = torch.zeros((H, N), dtype=torch.float32, device=C.device)
    _check_f32_out("A_add", A_add, (H, N), C.device)
    if workspace is None:
        n = _sz(0)
        _check("dtp_affinity_add_workspace_size", lib().dtp_affinity_add_workspace_size(T, d, H, N, ctypes.byref(n)))
        workspace = torch.empty(n.value, dtype=torch.uint8, device=C.device)
    st = lib().dtp_affinity_add_accumulate(_ptr(C), _ptr(W_gate), _ptr(W_up), T, d, H, N, _ptr(A_add),
                                           _ptr(workspace), workspace.numel(), _stream(stream))
    _check("dtp_affinity_add_accumulate", st)
    return A_add


def down_weight_sqnorm(Wqkv_next: torch.Tensor, gamma_next: torch.Tensor, W_down: torch.Tensor,
                       workspace: torch.Tensor | None = None, stream=None) -> torch.Tensor:
    """||b_gk||^2 = ||W^qkv_g (gamma' . w^d_k)||^2 (Sec. 3, down edge) -> fp32 [H_kv, N].

    Wqkv_next [H_kv, R, d]: the next layer's q/k/v rows of each KV group;
    gamma_next [d]: its pre-norm gain; W_down [d, N].  All bf16.
    """
    if not W_down.is_cuda:
        raise ValueError("W_down must be a contiguous CUDA tensor")
    _cuda_contig(W_down.device, Wqkv_next=Wqkv_next, gamma_next=gamma_next, W_down=W_down)
    if not (Wqkv_next.dtype == gamma_next.dtype == W_down.dtype):
        raise TypeError("Wqkv_next, gamma_next and W_down must share one dtype")
    if Wqkv_next.dim() != 3 or W_down.dim() != 2:
        raise ValueError("shapes must be Wqkv_next [H_kv,R,d], gamma_next [d], W_down [d,N]")
    H, R, d = Wqkv_next.shape
    N = W_down.shape[1]
    if gamma_next.shape != (d,) or W_down.shape != (d, N):
        raise ValueError("shapes must be Wqkv_next [H_kv,R,d], gamma_next [d], W_down [d,N]")
    bn = torch.empty((H, N), dtype=torch.float32, device=W_down.device)
    if workspace is None:
        n = _sz(0)
        _check("dtp_down_weight_workspace_size", lib().dtp_down_weight_workspace_size(H, R, d, N, ctypes.byref(n)))
        workspace = torch.empty(n.value, dtype=torch.uint8, device=W_down.device)
    st = lib().dtp_down_weight_sqnorm(_ptr(Wqkv_next), _ptr(gamma_next), _ptr(W_down), H, R, d, N,
                                      _dtype_code(W_down), _ptr(bn), _ptr(workspace), workspace.numel(),
                                      _stream(stream))
    _check("dtp_down_weight_sqnorm", st)
    return bn


def down_finalize(act2: torch.Tensor, bn: torch.Tensor, T_total: int, stream=None) -> torch.Tensor:
    """S_down[g,k] = act2[k] / T_total * bn[g,k] (Sec. 3), stored [H_kv, N]."""
    if not bn.is_cuda or bn.dim() != 2:
        raise ValueError("bn must be a CUDA fp32 [H_kv, N] tensor")
    H, N = bn.shape
    _check_f32_out("bn", bn, (H, N), bn.device)
    _check_f32_out("act2", act2, (N,), bn.device)
    S = torch.empty((H, N), dtype=torch.float32, device=bn.device)
    _check("dtp_down_finalize", lib().dtp_down_finalize(_ptr(act2), _ptr(bn), H, N, int(T_total), _ptr(S),
                                                        _stream(stream)))
    return S


def affinity_accumulate_noalloc(X: torch.Tensor, C: torch.Tensor, W_gate: torch.Tensor, W_up: torch.Tensor,
                                A: torch.Tensor, stream=None) -> torch.Tensor:
    """bf16 affinity pass that allocates nothing: scratch is the library's fixed device array.

    For callers that cannot allocate device memory; the caller passes the
    inputs and the fp32 output A [H_kv, N], which is accumulated into.  Calls
    that overlap on the GPU share the scratch and race.  A device-side failure
    is reported by ``affinity_noalloc_status``, not by this call.
    """
    T, d, H, N = _affinity_shapes(X, C, W_gate, W_up)
    if X.dtype != torch.bfloat16:
        raise TypeError("the allocation-free path takes bf16 inputs")
    _check_f32_out("A", A, (H, N), X.device)
    st = lib().dtp_affinity_accumulate_noalloc(_ptr(X), _ptr(C), _ptr(W_gate), _ptr(W_up), T, d, H, N, _ptr(A),
                                               _stream(stream))
    _check("dtp_affinity_accumulate_noalloc", st)
    return A


def affinity_noalloc_status(stream=None) -> int:
    """Synchronise ``stream`` and read the status word of the last allocation-free affinity call
    on the current device (DTP_OK or DTP_ERR_NOT_CONVERGED)."""
    return int(lib().dtp_affinity_noalloc_status(_stream(stream)))


def workspace_status(workspace: torch.Tensor, stream=None) -> int:
    """Synchronise and read the workspace status word (DTP_OK or DTP_ERR_NOT_CONVERGED)."""
    return int(lib().dtp_workspace_status(_ptr(workspace), workspace.numel(), _stream(stream)))


def selftest_bounded_wait(limit_ns: int, complete: bool, device="cuda:0", stream=None) -> dict:
    """Run the bounded-wait self-test: a device wait with limit_ns that is (complete) or is not
    satisfied.  Returns the workspace status and the two waits' durations in ns."""
    ws = torch.zeros(256, dtype=torch.uint8, device=device)
    el = (ctypes.c_uint64 * 2)()
    _check("dtp_selftest_bounded_wait",
           lib().dtp_selftest_bounded_wait(int(limit_ns), 1 if complete else 0, _ptr(ws), ws.numel(), el,
                                           _stream(stream)))
    return {"status": workspace_status(ws, stream), "elapsed_ns": (int(el[0]), int(el[1]))}


def affinity_finalize(A: torch.Tensor, T_total: int, wd_sqnorm: torch.Tensor | None = None, stream=None):
    """In place: A *= wd_sqnorm[k] / T_total (Sec. 3 E_t mean and ||w^d_k||^2)."""
    H, N = A.shape
    if wd_sqnorm is not None and (wd_sqnorm.shape != (N,) or wd_sqnorm.dtype != torch.float32):
        raise ValueError("wd_sqnorm must be fp32 [N]")
    _check("dtp_affinity_finalize",
           lib().dtp_affinity_finalize(_ptr(A), H, N, int(T_total), _ptr(wd_sqnorm), _stream(stream)))
    return A


def down_sqnorm(W_down: torch.Tensor, stream=None) -> torch.Tensor:
    """||w^d_k||^2 for W_down [d, N] (nn.Linear [out=d, in=N]) -> fp32 [N]."""
    d, N = W_down.shape
    out = torch.empty(N, dtype=torch.float32, device=W_down.device)
    _check("dtp_down_sqnorm",
           lib().dtp_down_sqnorm(_ptr(W_down), d, N, _dtype_code(W_down), _ptr(out), _stream(stream)))
    return out


def search_workspace_size(layers: int, H_kv: int, N: int, D: int) -> int:
    n = _sz(0)
    _check("dtp_search_workspace_size", lib().dtp_search_workspace_size(layers, H_kv, N, D, ctypes.byref(n)))
    return n.value


def search_layout_batched(A: torch.Tensor, D: int, iters: int, workspace: torch.Tensor | None = None,
                          stream=None, check: bool = True) -> dict:
    """Coordinate ascent on each layer of A [L, H_kv, N] (Sec. 3 'Optimiser').

    Returns dict of device tensors: h [L,H_kv] int32, nu [L,N] int32,
    score_q [L] int64, score [L] float64, iters_done [L] int32.  The call is
    asynchronous; with ``check`` (default) it synchronises and raises
    DTPError if the device reported a bad entry of A or a loop limit.
    """
    if A.dim() == 2:
        A = A.unsqueeze(0)
    if A.dtype != torch.float32 or not A.is_cuda or not A.is_contiguous():
        raise ValueError("A must be a contiguous fp32 CUDA tensor [L, H_kv, N]")
    Lyr, H, N = A.shape
    dev = A.device
    out = dict(h=torch.empty((Lyr, H), dtype=torch.int32, device=dev),
               nu=torch.empty((Lyr, N), dtype=torch.int32, device=dev),
               score_q=torch.empty(Lyr, dtype=torch.int64, device=dev),
               score=torch.empty(Lyr, dtype=torch.float64, device=dev),
               iters_done=torch.empty(Lyr, dtype=torch.int32, device=dev))
    if workspace is None:
        workspace = _keep(torch.empty(search_workspace_size(Lyr, H, N, D), dtype=torch.uint8, device=dev), stream)
    for t in out.values():
        _keep(t, stream)
    st = lib().dtp_search_layout_batched(_ptr(A), Lyr, H, N, D, iters, _ptr(out["h"]), _ptr(out["nu"]),
                                         _ptr(out["score_q"]), _ptr(out["score"]), _ptr(out["iters_done"]),
                                         _ptr(workspace), workspace.numel(), _stream(stream))
    _check("dtp_search_layout_batched", st)
    if check:
        _check("dtp_search_layout_batched (device status)", workspace_status(workspace, stream))
    return out


def search_layout(A: torch.Tensor, D: int, iters: int, workspace: torch.Tensor | None = None, stream=None,
                  check: bool = True) -> dict:
    """Coordinate ascent on one layer's A [H_kv, N]; tensors as in search_layout_batched, unbatched."""
    r = search_layout_batched(A.unsqueeze(0) if A.dim() == 2 else A, D, iters, workspace, stream, check)
    return {k: v[0] for k, v in r.items()}


def search_global(A: torch.Tensor, D: int, workspace: torch.Tensor | None = None, stream=None,
                  check: bool = True) -> dict:
    """The exact maximum of each layer's up-edge J over every balanced layout (best exact neuron
    step over the unlabelled head partitions).  A [L, H_kv, N] (or [H_kv, N]) fp32 CUDA.  Returns
    h (canonical labels), nu, score_q, score; unbatched input gives unbatched outputs."""
    x = A.unsqueeze(0) if A.dim() == 2 else A
    if x.dtype != torch.float32 or not x.is_cuda or not x.is_contiguous():
        raise ValueError("A must be a contiguous fp32 CUDA tensor [L, H_kv, N]")
    Lyr, H, N = x.shape
    dev = x.device
    out = dict(h=torch.empty((Lyr, H), dtype=torch.int32, device=dev),
               nu=torch.empty((Lyr, N), dtype=torch.int32, device=dev),
               score_q=torch.empty(Lyr, dtype=torch.int64, device=dev),
               score=torch.empty(Lyr, dtype=torch.float64, device=dev))
    for t in out.values():
        _keep(t, stream)
    if workspace is None:
        n = _sz(0)
        _check("dtp_search_global_workspace_size", lib().dtp_search_global_workspace_size(Lyr, H, N, D, ctypes.byref(n)))
        workspace = _keep(torch.empty(n.value, dtype=torch.uint8, device=dev), stream)
    st = lib().dtp_search_global(_ptr(x), Lyr, H, N, D, _ptr(out["h"]), _ptr(out["nu"]), _ptr(out["score_q"]),
                                 _ptr(out["score"]), _ptr(workspace), workspace.numel(), _stream(stream))
    _check("dtp_search_global", st)
    if check:
        _check("dtp_search_global (device status)", workspace_status(workspace, stream))
    return out if A.dim() == 3 else {k: v[0] for k, v in out.items()}


def _chain_inputs(S_up: torch.Tensor, S_down: torch.Tensor | None):
    if S_up.dtype != torch.float32 or not S_up.is_cuda or not S_up.is_contiguous():
        raise ValueError("S_up must be a contiguous fp32 CUDA tensor [L, H_kv, N]")
    Lyr, H, N = S_up.shape
    if Lyr > 1 and (S_down is None or S_down.shape != (Lyr - 1, H, N) or not S_down.is_contiguous()
                    or S_down.dtype != torch.float32 or S_down.device != S_up.device):
        raise ValueError("S_down must be a contiguous fp32 tensor [L-1, H_kv, N] on S_up's device")
    return Lyr, H, N


def search_chain_workspace_size(layers: int, H_kv: int, N: int, D: int) -> int:
    """Bytes of workspace for search_chain and chain_score."""
    n = _sz(0)
    _check("dtp_search_chain_workspace_size",
           lib().dtp_search_chain_workspace_size(layers, H_kv, N, D, ctypes.byref(n)))
    return n.value


def _chain_workspace(Lyr, H, N, D, dev, stream):
    return _keep(torch.empty(search_chain_workspace_size(Lyr, H, N, D), dtype=torch.uint8, device=dev), stream)


def search_chain(S_up: torch.Tensor, S_down: torch.Tensor | None, D: int, iters: int,
                 workspace: torch.Tensor | None = None, stream=None, check: bool = True,
                 move_heads=None, move_neurons=None, minimize: bool = False) -> dict:
    """Coordinate ascent on the whole-model objective (Sec. 3, Eq. objective, up and down edges).

    S_up [L, H_kv, N], S_down [L-1, H_kv, N] (None when L == 1), fp32 CUDA.
    move_heads / move_neurons: per-layer 0/1 (None = every layer moves) and
    minimize: the ablation layouts of Sec. 3 'Optimiser' (Table 4).
    Returns device tensors: h [L,H_kv] int32, nu [L,N] int32, J_q int64 (units
    of 2^-43), J float64, iters_done int32.  Asynchronous unless ``check``.
    """
    Lyr, H, N = _chain_inputs(S_up, S_down)
    dev = S_up.device
    out = dict(h=torch.empty((Lyr, H), dtype=torch.int32, device=dev),
               nu=torch.empty((Lyr, N), dtype=torch.int32, device=dev),
               J_q=torch.empty((), dtype=torch.int64, device=dev),
               J=torch.empty((), dtype=torch.float64, device=dev),
               iters_done=torch.empty((), dtype=torch.int32, device=dev))
    for t in out.values():
        _keep(t, stream)
    mh = _device_mask(move_heads, Lyr, dev, stream)
    mn = _device_mask(move_neurons, Lyr, dev, stream)
    if workspace is None:
        workspace = _chain_workspace(Lyr, H, N, D, dev, stream)
    st = lib().dtp_search_chain_ex(_ptr(S_up), _ptr(S_down) if Lyr > 1 else None, Lyr, H, N, D, iters, _ptr(mh),
                                   _ptr(mn), int(bool(minimize)), _ptr(out["h"]), _ptr(out["nu"]), _ptr(out["J_q"]),
                                   _ptr(out["J"]), _ptr(out["iters_done"]), _ptr(workspace), workspace.numel(),
                                   _stream(stream))
    _check("dtp_search_chain_ex", st)
    if check:
        _check("dtp_search_chain_ex (device status)", workspace_status(workspace, stream))
    return out


def chain_score(S_up: torch.Tensor, S_down: torch.Tensor | None, h: torch.Tensor, nu: torch.Tensor, D: int,
                workspace: torch.Tensor | None = None, stream=None, check: bool = True) -> dict:
    """J of a given layout (Eq. objective) and its per-edge terms.

    h [L, H_kv], nu [L, N] int32 CUDA, entries in [0, D).  Returns device
    tensors: edge_q [2L-1] int64 (up_0, down_0, up_1, ...; units of 2^-43 of
    each edge), J_q int64, J float64.
    """
    Lyr, H, N = _chain_inputs(S_up, S_down)
    dev = S_up.device
    for name, t, shape in (("h", h, (Lyr, H)), ("nu", nu, (Lyr, N))):
        if t.dtype != torch.int32 or t.device != dev or not t.is_contiguous() or tuple(t.shape) != shape:
            raise ValueError(f"{name} must be a contiguous int32 tensor {shape} on S_up's device")
    out = dict(edge_q=torch.empty(2 * Lyr - 1, dtype=torch.int64, device=dev),
               J_q=torch.empty((), dtype=torch.int64, device=dev),
               J=torch.empty((), dtype=torch.float64, device=dev))
    if workspace is None:
        workspace = _chain_workspace(Lyr, H, N, D, dev, stream)
    st = lib().dtp_chain_score(_ptr(S_up), _ptr(S_down) if Lyr > 1 else None, Lyr, H, N, D, _ptr(h), _ptr(nu),
                               _ptr(out["edge_q"]), _ptr(out["J_q"]), _ptr(out["J"]), _ptr(workspace),
                               workspace.numel(), _stream(stream))
    _check("dtp_chain_score", st)
    if check:
        _check("dtp_chain_score (device status)", workspace_status(workspace, stream))
    return out


# ------------------------------------------------------------ producer / apply --

def _status_workspace(dev, stream) -> torch.Tensor:
    n = _sz(0)
    _check("dtp_head_writes_workspace_size", lib().dtp_head_writes_workspace_size(ctypes.byref(n)))
    return _keep(torch.empty(n.value, dtype=torch.uint8, device=dev), stream)


def head_writes(attn: torch.Tensor, W_o: torch.Tensor, gamma: torch.Tensor, rms: torch.Tensor, head_dim: int,
                q_per_row: int = 1, out: torch.Tensor | None = None, workspace: torch.Tensor | None = None,
                stream=None, check: bool = False) -> torch.Tensor:
    """C[j,t,:] = gamma * (sum of a_{h,t} W_o^(h)T over the heads of row j) / rms[t] (Sec. 3), bf16.

    attn [T, H_q*head_dim] and W_o [d, H_q*head_dim] bf16 CUDA; gamma [d] and
    rms [T] fp32.  Returns C [H_q/q_per_row, T, d] bf16.
    """
    for name, t in (("attn", attn), ("W_o", W_o)):
        if t.dtype != torch.bfloat16 or not t.is_cuda or not t.is_contiguous():
            raise ValueError(f"{name} must be a contiguous bf16 CUDA tensor")
    T, K = attn.shape
    d = W_o.shape[0]
    if W_o.shape != (d, K) or K % head_dim:
        raise ValueError("W_o must be [d, H_q*head_dim] with attn [T, H_q*head_dim]")
    Hq = K // head_dim
    if q_per_row < 1 or Hq % q_per_row:
        raise ValueError("q_per_row must divide H_q")
    if gamma.shape != (d,) or gamma.dtype != torch.float32 or rms.shape != (T,) or rms.dtype != torch.float32:
        raise ValueError("gamma must be fp32 [d] and rms fp32 [T]")
    if out is None:
        out = torch.empty((Hq // q_per_row, T, d), dtype=torch.bfloat16, device=attn.device)
    if workspace is None:
        workspace = _status_workspace(attn.device, stream)
    st = lib().dtp_head_writes(_ptr(attn), _ptr(W_o), _ptr(gamma.contiguous()), _ptr(rms.contiguous()), T, d, Hq,
                               head_dim, q_per_row, _ptr(out), _ptr(workspace), workspace.numel(), _stream(stream))
    _check("dtp_head_writes", st)
    if check:
        _check("dtp_head_writes (device status)", workspace_status(workspace, stream))
    return out


def layout_order(labels: torch.Tensor, D: int, balanced: bool = True, stream=None, check: bool = True) -> torch.Tensor:
    """order[i][p]: layer i's items listed device by device (each device's in increasing index).

    labels [layers, n] (or [n]) int32 CUDA: head_part or neuron_dev.
    """
    lab = labels.unsqueeze(0) if labels.dim() == 1 else labels
    if lab.dtype != torch.int32 or not lab.is_cuda or not lab.is_contiguous():
        raise ValueError("labels must be a contiguous int32 CUDA tensor")
    Lyr, n = lab.shape
    order = torch.empty_like(lab)
    ws = _status_workspace(lab.device, stream)
    st = lib().dtp_layout_order(_ptr(lab), Lyr, n, D, int(balanced), _ptr(order), _ptr(ws), ws.numel(),
                                _stream(stream))
    _check("dtp_layout_order", st)
    if check:
        _check("dtp_layout_order (device status)", workspace_status(ws, stream))
    return order if labels.dim() == 2 else order[0]


def permute_rows(src: torch.Tensor, perm: torch.Tensor, block_rows: int = 1, out: torch.Tensor | None = None,
                 stream=None, check: bool = True) -> torch.Tensor:
    """dst[i][b*B + r] = src[i][perm[i][b]*B + r] for src [layers, rows, ...] (or [rows, ...]), perm [layers, rows/B]."""
    x = src.unsqueeze(0) if perm.dim() == 1 else src
    pm = perm.unsqueeze(0) if perm.dim() == 1 else perm
    if not x.is_contiguous() or not pm.is_contiguous() or pm.dtype != torch.int32:
        raise ValueError("src and perm must be contiguous, perm int32")
    Lyr, rows = x.shape[0], x.shape[1]
    row_bytes = x[0, 0].numel() * x.element_size()
    dst = torch.empty_like(x) if out is None else (out.unsqueeze(0) if perm.dim() == 1 else out)
    ws = _status_workspace(x.device, stream)
    st = lib().dtp_permute_rows(_ptr(x), _ptr(dst), Lyr, rows, row_bytes, block_rows, _ptr(pm), pm.shape[1],
                                _ptr(ws), ws.numel(), _stream(stream))
    _check("dtp_permute_rows", st)
    if check:
        _check("dtp_permute_rows (device status)", workspace_status(ws, stream))
    return dst[0] if perm.dim() == 1 else dst


def permute_cols(src: torch.Tensor, perm: torch.Tensor, block_cols: int = 1, out: torch.Tensor | None = None,
                 stream=None, check: bool = True) -> torch.Tensor:
    """dst[i][r][b*B + c] = src[i][r][perm[i][b]*B + c] for src [layers, rows, cols] (or [rows, cols])."""
    x = src.unsqueeze(0) if perm.dim() == 1 else src
    pm = perm.unsqueeze(0) if perm.dim() == 1 else perm
    if x.dim() != 3 or not x.is_contiguous() or not pm.is_contiguous() or pm.dtype != torch.int32:
        raise ValueError("src must be contiguous [layers, rows, cols] and perm contiguous int32")
    Lyr, rows, cols = x.shape
    dst = torch.empty_like(x) if out is None else (out.unsqueeze(0) if perm.dim() == 1 else out)
    ws = _status_workspace(x.device, stream)
    st = lib().dtp_permute_cols(_ptr(x), _ptr(dst), Lyr, rows, cols, x.element_size(), block_cols, _ptr(pm),
                                pm.shape[1], _ptr(ws), ws.numel(), _stream(stream))
    _check("dtp_permute_cols", st)
    if check:
        _check("dtp_permute_cols (device status)", workspace_status(ws, stream))
    return dst[0] if perm.dim() == 1 else dst


def apply_layout(W: dict, h: torch.Tensor, nu: torch.Tensor, D: int, head_dim: int, stream=None,
                 check: bool = True) -> tuple[dict, torch.Tensor, torch.Tensor]:
    """Permute dense weights for a layout so that device l's KV groups and neurons are the l-th
    contiguous shard (Sec. 3).

    W holds q [.., Hq*hd, d], k and v [.., G*hd, d], o [.., d, Hq*hd], gate and
    up [.., N, d], down [.., d, N], with an optional leading layers axis that
    h [layers, G] and nu [layers, N] then share.  Other entries are copied by
    reference.  Returns (permuted weights, head order, neuron order).
    """
    names = ("q", "k", "v", "o", "gate", "up", "down")
    mats = [W[n] for n in names]
    stacked = h.dim() == 2
    if all(m.is_cuda and m.is_contiguous() and m.dtype == mats[0].dtype and m.dim() == (3 if stacked else 2)
           for m in mats) and h.dtype == torch.int32 and nu.dtype == torch.int32:
        # one native call: both orders and the seven gathers
        Lyr = h.shape[0] if stacked else 1
        G, N, d = h.shape[-1], nu.shape[-1], mats[0].shape[-1]
        qpg = mats[0].shape[-2] // (G * head_dim)
        outs = [torch.empty_like(m) for m in mats]
        hc, nc = _keep(h.contiguous(), stream), _keep(nu.contiguous(), stream)
        ho, no = torch.empty_like(hc), torch.empty_like(nc)
        ws = _status_workspace(h.device, stream)
        src = (_vp * 7)(*[m.data_ptr() for m in mats])
        dst = (_vp * 7)(*[o.data_ptr() for o in outs])
        st = lib().dtp_apply_layout(_ptr(hc), _ptr(nc), Lyr, G, N, D, qpg, head_dim, d,
                                    mats[0].element_size(), src, dst, _ptr(ho), _ptr(no), _ptr(ws), ws.numel(),
                                    _stream(stream))
        _check("dtp_apply_layout", st)
        if check:
            _check("dtp_apply_layout (device status)", workspace_status(ws, stream))
        out = dict(W)
        out.update(zip(names, outs))
        return out, ho, no
    ho = layout_order(h, D, stream=stream, check=check)
    no = layout_order(nu, D, stream=stream, check=check)
    G = h.shape[-1]
    hq = W["q"].shape[-2] // head_dim
    blk = (hq // G) * head_dim
    out = dict(W)
    out["q"] = permute_rows(W["q"], ho, blk, stream=stream, check=check)
    out["k"] = permute_rows(W["k"], ho, head_dim, stream=stream, check=check)
    out["v"] = permute_rows(W["v"], ho, head_dim, stream=stream, check=check)
    out["o"] = permute_cols(W["o"], ho, blk, stream=stream, check=check)
    out["gate"] = permute_rows(W["gate"], no, 1, stream=stream, check=check)
    out["up"] = permute_rows(W["up"], no, 1, stream=stream, check=check)
    out["down"] = permute_cols(W["down"], no, 1, stream=stream, check=check)
    return out, ho, no
