"""GB300-native hot path of Online Speculative Decoding (Liu et al., ICML 2024).

Thin ctypes binding over ``libosd.so`` (the C ABI in ``include/osd.h``): it
turns torch tensors into device pointers, sizes and the current CUDA stream,
allocates outputs with torch, and raises ``OsdError`` on a non-OK status.
Every step of verify and distill runs in the library's CUDA kernels; there is
no CPU path.  If the library has not been built, calls raise immediately.

    osd_verify(draft_logits [B,k,V], target_logits [B,k+1,V], draft_tokens [B,k],
               uniforms [B,k+1], temperature)           # Appendix A.1, Algorithm 1
    osd_distill(draft_logits [..,V], target_logits [..,V], mask, loss_kind, beta)
                                                       # Eq. 2-3, Section 4.1
"""
from __future__ import annotations

import contextlib
import ctypes
import os
from typing import NamedTuple, Optional

import torch

from ._build import LIB_PATH, build as build_library  # noqa: F401

OSD_OK, OSD_ERR_INVALID_ARG, OSD_ERR_UNSUPPORTED, OSD_ERR_CUDA, OSD_ERR_TIMEOUT = range(5)
OSD_F32, OSD_BF16 = 0, 1
LOSS_KINDS = {"fkl": 0, "rkl": 1, "jsd": 2, "tvd": 3, "ce": 4}
VERIFY_MAX_K = 64
VERIFY_MAX_V = 1 << 21

# every symbol include/osd.h declares
EXPORTS = ("osd_status_string", "osd_abi_version", "osd_verify_workspace_size",
           "osd_verify", "osd_verify_noalloc", "osd_distill", "osd_distill_accepted",
           "osd_mixed_sample", "osd_verify_tree_workspace_size", "osd_verify_tree", "osd_check_bounded_wait")


class OsdError(RuntimeError):
    def __init__(self, status: int, what: str):
        self.status = status
        super().__init__(f"{what}: {osd_status_string(status)}")


_lib = None
ABI_MAJOR = 2  # osd_distill gained its temperature argument in 2.0


def load_library():
    """Load libosd.so (raises if it has not been built)."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(LIB_PATH):
        raise RuntimeError(f"{LIB_PATH} is missing: build it with paper_2310_07177_gb300.build_library()")
    lib = ctypes.CDLL(LIB_PATH)
    vp, i32, i64, f32, sz = ctypes.c_void_p, ctypes.c_int, ctypes.c_int64, ctypes.c_float, ctypes.c_size_t
    lib.osd_status_string.restype = ctypes.c_char_p
    lib.osd_status_string.argtypes = [i32]
    lib.osd_abi_version.restype = i32
    lib.osd_abi_version.argtypes = []
    if lib.osd_abi_version() >> 16 != ABI_MAJOR:
        raise RuntimeError(f"{LIB_PATH} has ABI {lib.osd_abi_version() >> 16}.x, this binding needs "
                           f"{ABI_MAJOR}.x: rebuild it with paper_2310_07177_gb300.build_library()")
    lib.osd_verify_workspace_size.restype = i32
    lib.osd_verify_workspace_size.argtypes = [i32, i32, i32, ctypes.POINTER(sz)]
    lib.osd_verify.restype = i32
    lib.osd_verify.argtypes = [vp, vp, i32, i32, i32, i32, vp, vp, f32, vp, vp, vp, vp, vp, vp, sz, vp]
    lib.osd_verify_noalloc.restype = i32
    lib.osd_verify_noalloc.argtypes = [vp, vp, i32, i32, i32, i32, vp, vp, f32, vp, vp, vp, vp, vp, vp]
    lib.osd_distill.restype = i32
    lib.osd_distill.argtypes = [vp, vp, i32, i32, i32, i32, i64, i64, i64, i64, vp, i32, f32, f32, vp, vp, vp, vp]
    lib.osd_distill_accepted.restype = i32
    lib.osd_distill_accepted.argtypes = [vp, vp, i32, i32, i32, i32, vp, i32, f32, f32, vp, vp, vp, vp, vp, vp]
    lib.osd_verify_tree_workspace_size.restype = i32
    lib.osd_verify_tree_workspace_size.argtypes = [i32, i32, i32, ctypes.POINTER(sz)]
    lib.osd_verify_tree.restype = i32
    lib.osd_verify_tree.argtypes = [vp, vp, i32, i32, i32, i32, ctypes.POINTER(ctypes.c_int32), vp, vp, f32,
                                    vp, vp, vp, vp, vp, vp, vp, sz, vp]
    lib.osd_check_bounded_wait.restype = i32
    lib.osd_check_bounded_wait.argtypes = [ctypes.c_uint32, vp, vp, vp]
    lib.osd_mixed_sample.restype = i32
    lib.osd_mixed_sample.argtypes = [vp, vp, i32, i32, i32, i64, i64, vp, f32, f32, vp, vp, vp, vp]
    _lib = lib
    return lib


def osd_status_string(status: int) -> str:
    return load_library().osd_status_string(int(status)).decode()


def osd_abi_version() -> int:
    return load_library().osd_abi_version()


def osd_verify_workspace_size(B: int, k: int, V: int) -> int:
    n = ctypes.c_size_t(0)
    st = load_library().osd_verify_workspace_size(B, k, V, ctypes.byref(n))
    if st != OSD_OK:
        raise OsdError(st, "osd_verify_workspace_size")
    return n.value


def _dtype_code(t: torch.Tensor) -> int:
    if t.dtype == torch.float32:
        return OSD_F32
    if t.dtype == torch.bfloat16:
        return OSD_BF16
    raise TypeError(f"logits must be float32 or bfloat16, got {t.dtype}")


def _ptr(t: Optional[torch.Tensor]):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _stream(device, stream):
    s = stream if stream is not None else torch.cuda.current_stream(device)
    return ctypes.c_void_p(s.cuda_stream)


def _on(dev):
    """Make ``dev`` the current device for a library call: the C functions work
    on the current device (its workspace, its streams), which need not be the
    device the tensors live on."""
    if dev is None or dev.index is None or torch.cuda.current_device() == dev.index:
        return contextlib.nullcontext()
    return torch.cuda.device(dev)


def _need_cuda(*ts):
    dev = None
    for t in ts:
        if t is None:
            continue
        if not t.is_cuda:
            raise ValueError("osd kernels take CUDA tensors only")
        if dev is None:
            dev = t.device
        elif t.device != dev:
            raise ValueError("all tensors must live on the same CUDA device")
    return dev


class VerifyResult(NamedTuple):
    accepted: torch.Tensor       # [B] int32
    out_tokens: torch.Tensor     # [B, k+1] int32
    mismatch_mask: torch.Tensor  # [B, k] uint8
    diag_margin: Optional[torch.Tensor]   # [B, k] float32
    diag_cdf_gap: Optional[torch.Tensor]  # [B] float32


def osd_verify(draft_logits: torch.Tensor, target_logits: torch.Tensor, draft_tokens: torch.Tensor,
               uniforms: Optional[torch.Tensor], temperature: float, *, diagnostics: bool = True,
               workspace: Optional[torch.Tensor] = None, out: Optional[VerifyResult] = None,
               stream: Optional[torch.cuda.Stream] = None) -> VerifyResult:
    """Speculative-sampling verification (Appendix A.1); see include/osd.h.

    ``draft_logits`` [B,k,V] and ``target_logits`` [B,k+1,V] must be contiguous
    and of the same dtype; at temperature 0 ``draft_logits`` and ``uniforms``
    may be None.  ``workspace`` (uint8, >= osd_verify_workspace_size bytes) and
    ``out`` may be preallocated to avoid allocations on the hot path.
    """
    lib = load_library()
    B, k1, V = target_logits.shape
    k = k1 - 1
    dev = _need_cuda(draft_logits, target_logits, draft_tokens, uniforms)
    if not target_logits.is_contiguous() or (draft_logits is not None and not draft_logits.is_contiguous()):
        raise ValueError("verify logits must be contiguous")
    dt = _dtype_code(target_logits)
    if draft_logits is not None:
        if draft_logits.dtype != target_logits.dtype or tuple(draft_logits.shape) != (B, k, V):
            raise ValueError("draft_logits must be [B, k, V] with the target's dtype")
    if draft_tokens.dtype != torch.int32 or tuple(draft_tokens.shape) != (B, k) or not draft_tokens.is_contiguous():
        raise ValueError("draft_tokens must be contiguous int32 [B, k]")
    if uniforms is not None and (uniforms.dtype != torch.float32 or tuple(uniforms.shape) != (B, k + 1)
                                 or not uniforms.is_contiguous()):
        raise ValueError("uniforms must be contiguous float32 [B, k+1]")
    need = osd_verify_workspace_size(B, k, V)
    if workspace is None:
        workspace = torch.empty(need, dtype=torch.uint8, device=dev)
    if out is None:
        out = VerifyResult(
            torch.empty(B, dtype=torch.int32, device=dev),
            torch.empty(B, k + 1, dtype=torch.int32, device=dev),
            torch.empty(B, k, dtype=torch.uint8, device=dev),
            torch.empty(B, k, dtype=torch.float32, device=dev) if diagnostics else None,
            torch.empty(B, dtype=torch.float32, device=dev) if diagnostics else None)
    with _on(dev):
        st = lib.osd_verify(_ptr(draft_logits), _ptr(target_logits), dt, B, k, V, _ptr(draft_tokens),
                            _ptr(uniforms), float(temperature), _ptr(out.accepted), _ptr(out.out_tokens),
                            _ptr(out.mismatch_mask), _ptr(out.diag_margin), _ptr(out.diag_cdf_gap),
                            _ptr(workspace), workspace.numel() * workspace.element_size(), _stream(dev, stream))
    if st != OSD_OK:
        raise OsdError(st, "osd_verify")
    return out


def osd_verify_noalloc(draft_logits: torch.Tensor, target_logits: torch.Tensor, draft_tokens: torch.Tensor,
                       uniforms: Optional[torch.Tensor], temperature: float, out: VerifyResult, *,
                       stream: Optional[torch.cuda.Stream] = None) -> VerifyResult:
    """osd_verify on the library's own static workspace, for callers that must not
    allocate device memory while serving (see include/osd.h).  Outputs are
    caller-provided in ``out``; calls that overlap on the GPU must be serialised."""
    lib = load_library()
    B, k1, V = target_logits.shape
    dev = _need_cuda(draft_logits, target_logits, draft_tokens, uniforms, *out)
    with _on(dev):
        st = lib.osd_verify_noalloc(_ptr(draft_logits), _ptr(target_logits), _dtype_code(target_logits), B, k1 - 1, V,
                                    _ptr(draft_tokens), _ptr(uniforms), float(temperature), _ptr(out.accepted),
                                    _ptr(out.out_tokens), _ptr(out.mismatch_mask), _ptr(out.diag_margin),
                                    _ptr(out.diag_cdf_gap), _stream(dev, stream))
    if st != OSD_OK:
        raise OsdError(st, "osd_verify_noalloc")
    return out


def _rows_view(t: torch.Tensor):
    """(G, P, V, stride_g, stride_p) of a [N,V] or [G,P,V] view with contiguous rows."""
    if t.stride(-1) != 1:
        raise ValueError("the vocabulary dimension must be contiguous")
    if t.dim() == 2:
        return t.shape[0], 1, t.shape[1], t.stride(0), 0
    if t.dim() == 3:
        return t.shape[0], t.shape[1], t.shape[2], t.stride(0), t.stride(1)
    raise ValueError("distill logits must be [N, V] or [G, P, V]")


def osd_distill(draft_logits: torch.Tensor, target_logits: torch.Tensor, mask: Optional[torch.Tensor] = None,
                loss_kind: str = "fkl", beta: float = 0.5, *, temperature: float = 1.0,
                loss: Optional[torch.Tensor] = None,
                dlogits: Optional[torch.Tensor] = None, status: Optional[torch.Tensor] = None,
                stream: Optional[torch.cuda.Stream] = None):
    """Per-position distillation loss and d loss / d draft_logits (Eq. 2-3) at
    softmax temperature ``temperature`` (Section 4.1); ``loss_kind`` is one of
    fkl, rkl, jsd, tvd, ce (label fine-tuning to the target argmax).

    Logits are [N,V] or [G,P,V] views whose rows are contiguous (e.g.
    ``target[:, :k, :]`` of a [B,k+1,V] tensor).  Returns ``(loss, dlogits)``:
    fp32 [..] and fp32 [.., V] contiguous.  Rows with mask 0 get loss 0 and are
    not written in ``dlogits`` (pass a prefilled ``dlogits`` to keep them).
    """
    lib = load_library()
    dev = _need_cuda(draft_logits, target_logits, mask, loss, dlogits, status)
    G, P, V, dsg, dsp = _rows_view(draft_logits)
    G2, P2, V2, tsg, tsp = _rows_view(target_logits)
    if (G, P, V) != (G2, P2, V2) or draft_logits.dtype != target_logits.dtype:
        raise ValueError("draft and target logits must have the same shape and dtype")
    lead = tuple(draft_logits.shape[:-1])
    if mask is not None and (mask.dtype != torch.uint8 or tuple(mask.shape) != lead or not mask.is_contiguous()):
        raise ValueError("mask must be contiguous uint8 with the logits' leading shape")
    if loss is None:
        loss = torch.empty(lead, dtype=torch.float32, device=dev)
    if dlogits is None:
        dlogits = torch.empty(*lead, V, dtype=torch.float32, device=dev)
    if (loss.dtype != torch.float32 or not loss.is_contiguous() or tuple(loss.shape) != lead
            or dlogits.dtype != torch.float32 or not dlogits.is_contiguous()
            or tuple(dlogits.shape) != lead + (V,)):
        raise ValueError("loss / dlogits must be contiguous float32 of the logits' shape")
    kind = LOSS_KINDS[loss_kind] if isinstance(loss_kind, str) else int(loss_kind)
    with _on(dev):
        st = lib.osd_distill(_ptr(draft_logits), _ptr(target_logits), _dtype_code(draft_logits), G, P, V,
                             dsg, dsp, tsg, tsp, _ptr(mask), kind, float(beta), float(temperature), _ptr(loss),
                             _ptr(dlogits),
                             _ptr(status), _stream(dev, stream))
    if st != OSD_OK:
        raise OsdError(st, "osd_distill")
    return loss, dlogits


class DistillAcceptedResult(NamedTuple):
    """Outputs of osd_distill_accepted: slot r < count holds sequence seq_of_row[r]."""
    loss: torch.Tensor        # [B] fp32 (0 beyond count)
    dlogits: torch.Tensor     # [B, V] fp32 (rows beyond count untouched)
    seq_of_row: torch.Tensor  # [B] int32
    count: torch.Tensor       # [1] int32 on the device


def osd_distill_accepted(draft_logits: torch.Tensor, target_logits: torch.Tensor, accepted: torch.Tensor,
                         loss_kind: str = "rkl", beta: float = 0.5, *, temperature: float = 1.0,
                         out: Optional[DistillAcceptedResult] = None, status: Optional[torch.Tensor] = None,
                         stream: Optional[torch.cuda.Stream] = None) -> DistillAcceptedResult:
    """Distil the rows verification rejected (Algorithm 1's buffer R, Eq. 2-3).

    ``draft_logits`` [B,k,V] and ``target_logits`` [B,k+1,V] are the contiguous
    tensors osd_verify read; ``accepted`` [B] int32 is its output.  Sequence b
    contributes row (b, accepted[b]) when that is < k; results are compacted on
    the device, active sequences first (see ``DistillAcceptedResult``).
    """
    lib = load_library()
    dev = _need_cuda(draft_logits, target_logits, accepted, status, *(out or ()))
    if draft_logits.dim() != 3 or target_logits.dim() != 3:
        raise ValueError("draft_logits must be [B,k,V] and target_logits [B,k+1,V]")
    B, k, V = draft_logits.shape
    if (tuple(target_logits.shape) != (B, k + 1, V) or draft_logits.dtype != target_logits.dtype
            or not draft_logits.is_contiguous() or not target_logits.is_contiguous()):
        raise ValueError("draft_logits [B,k,V] and target_logits [B,k+1,V] must be contiguous, same dtype")
    if accepted.dtype != torch.int32 or tuple(accepted.shape) != (B,) or not accepted.is_contiguous():
        raise ValueError("accepted must be contiguous int32 [B]")
    if out is None:
        out = DistillAcceptedResult(torch.empty(B, dtype=torch.float32, device=dev),
                                    torch.empty(B, V, dtype=torch.float32, device=dev),
                                    torch.empty(B, dtype=torch.int32, device=dev),
                                    torch.empty(1, dtype=torch.int32, device=dev))
    kind = LOSS_KINDS[loss_kind] if isinstance(loss_kind, str) else int(loss_kind)
    with _on(dev):
        st = lib.osd_distill_accepted(_ptr(draft_logits), _ptr(target_logits), _dtype_code(draft_logits), B, k, V,
                                      _ptr(accepted), kind, float(beta), float(temperature), _ptr(out.loss),
                                      _ptr(out.dlogits), _ptr(out.seq_of_row), _ptr(out.count), _ptr(status),
                                      _stream(dev, stream))
    if st != OSD_OK:
        raise OsdError(st, "osd_distill_accepted")
    return out


def _rows_2d(t: torch.Tensor):
    """(N, V, row stride) of a 2-D view whose rows are contiguous (stride 0 repeats a row)."""
    if t.dim() != 2 or (t.shape[1] > 1 and t.stride(1) != 1):
        raise ValueError("logits must be a 2-D [N, V] view with contiguous rows")
    return t.shape[0], t.shape[1], t.stride(0)


def osd_mixed_sample(draft_logits: torch.Tensor, target_logits: torch.Tensor, uniforms: torch.Tensor,
                     beta: float, *, temperature: float = 1.0, tokens: Optional[torch.Tensor] = None,
                     cdf_gap: Optional[torch.Tensor] = None, status: Optional[torch.Tensor] = None,
                     stream: Optional[torch.cuda.Stream] = None):
    """One token per row from beta p + (1 - beta) q (Section 4.1, mixed sampling).

    ``draft_logits`` and ``target_logits`` are [N, V] views with contiguous rows
    (``expand`` of one row is fine); ``uniforms`` [N] fp32 in [0, 1).  Returns
    ``(tokens [N] int32, cdf_gap [N] fp32 or None)``.
    """
    lib = load_library()
    dev = _need_cuda(draft_logits, target_logits, uniforms, tokens, cdf_gap, status)
    N, V, ds = _rows_2d(draft_logits)
    N2, V2, tsd = _rows_2d(target_logits)
    if (N, V) != (N2, V2) or draft_logits.dtype != target_logits.dtype:
        raise ValueError("draft and target logits must have the same shape and dtype")
    if uniforms.dtype != torch.float32 or tuple(uniforms.shape) != (N,) or not uniforms.is_contiguous():
        raise ValueError("uniforms must be contiguous float32 [N]")
    if tokens is None:
        tokens = torch.empty(N, dtype=torch.int32, device=dev)
    with _on(dev):
        st = lib.osd_mixed_sample(_ptr(draft_logits), _ptr(target_logits), _dtype_code(draft_logits), N, V, ds, tsd,
                                  _ptr(uniforms), float(beta), float(temperature), _ptr(tokens), _ptr(cdf_gap),
                                  _ptr(status), _stream(dev, stream))
    if st != OSD_OK:
        raise OsdError(st, "osd_mixed_sample")
    return tokens, cdf_gap


def osd_verify_tree_workspace_size(B: int, n_nodes: int, V: int) -> int:
    n = ctypes.c_size_t(0)
    st = load_library().osd_verify_tree_workspace_size(int(B), int(n_nodes), int(V), ctypes.byref(n))
    if st != OSD_OK:
        raise OsdError(st, "osd_verify_tree_workspace_size")
    return n.value


class TreeResult(NamedTuple):
    accepted: torch.Tensor      # [B] int32
    path: torch.Tensor          # [B, n_nodes] int32
    out_tokens: torch.Tensor    # [B, n_nodes] int32
    last_node: torch.Tensor     # [B] int32
    diag_margin: Optional[torch.Tensor]   # [B, n_nodes] fp32
    diag_cdf_gap: Optional[torch.Tensor]  # [B] fp32


def osd_verify_tree(draft_logits: Optional[torch.Tensor], target_logits: torch.Tensor, parent, tokens: torch.Tensor,
                    uniforms: Optional[torch.Tensor], temperature: float, *, diagnostics: bool = True,
                    workspace: Optional[torch.Tensor] = None, out: Optional[TreeResult] = None,
                    stream: Optional[torch.cuda.Stream] = None) -> TreeResult:
    """Multi-candidate verification over a token tree (see include/osd.h).

    ``draft_logits`` and ``target_logits`` are contiguous [B, n_nodes, V];
    ``parent`` is the static tree (a host sequence of n_nodes ints, parent[0] =
    -1); ``tokens`` [B, n_nodes] int32; ``uniforms`` [B, n_nodes] fp32.  At
    temperature 0 the draft logits and uniforms may be None.
    """
    lib = load_library()
    B, n, V = target_logits.shape
    dev = _need_cuda(draft_logits, target_logits, tokens, uniforms, workspace, *(out or ()))
    par = (ctypes.c_int32 * n)(*[int(x) for x in (parent.tolist() if hasattr(parent, "tolist") else parent)])
    if len(par) != n:
        raise ValueError("parent must have n_nodes entries")
    if not target_logits.is_contiguous() or (draft_logits is not None and (
            tuple(draft_logits.shape) != (B, n, V) or not draft_logits.is_contiguous()
            or draft_logits.dtype != target_logits.dtype)):
        raise ValueError("draft/target logits must be contiguous [B, n_nodes, V] of one dtype")
    if tokens.dtype != torch.int32 or tuple(tokens.shape) != (B, n) or not tokens.is_contiguous():
        raise ValueError("tokens must be contiguous int32 [B, n_nodes]")
    if uniforms is not None and (uniforms.dtype != torch.float32 or tuple(uniforms.shape) != (B, n)
                                 or not uniforms.is_contiguous()):
        raise ValueError("uniforms must be contiguous float32 [B, n_nodes]")
    if workspace is None:
        workspace = torch.empty(max(osd_verify_tree_workspace_size(B, n, V), 16), dtype=torch.uint8, device=dev)
    if out is None:
        i32 = torch.int32
        out = TreeResult(torch.empty(B, dtype=i32, device=dev), torch.empty(B, n, dtype=i32, device=dev),
                         torch.empty(B, n, dtype=i32, device=dev), torch.empty(B, dtype=i32, device=dev),
                         torch.empty(B, n, dtype=torch.float32, device=dev) if diagnostics else None,
                         torch.empty(B, dtype=torch.float32, device=dev) if diagnostics else None)
    with _on(dev):
        st = lib.osd_verify_tree(_ptr(draft_logits), _ptr(target_logits), _dtype_code(target_logits), B, n, V, par,
                                 _ptr(tokens), _ptr(uniforms), float(temperature), _ptr(out.accepted), _ptr(out.path),
                                 _ptr(out.out_tokens), _ptr(out.last_node), _ptr(out.diag_margin),
                                 _ptr(out.diag_cdf_gap), _ptr(workspace), workspace.numel() * workspace.element_size(),
                                 _stream(dev, stream))
    if st != OSD_OK:
        raise OsdError(st, "osd_verify_tree")
    return out


def osd_check_bounded_wait(limit_us: int, *, device=None, stream: Optional[torch.cuda.Stream] = None):
    """Run the shared bounded-wait failure path against a barrier nothing
    completes; returns (status, waited_ns) read back from the device (status is
    OSD_ERR_TIMEOUT when the path works)."""
    lib = load_library()
    dev = torch.device("cuda") if device is None else torch.device(device)
    st = torch.full((1,), -1, dtype=torch.int32, device=dev)
    waited = torch.zeros(1, dtype=torch.int64, device=dev)
    with _on(dev):
        rc = lib.osd_check_bounded_wait(int(limit_us), _ptr(st), _ptr(waited), _stream(dev, stream))
    if rc != OSD_OK:
        raise OsdError(rc, "osd_check_bounded_wait")
    return int(st.item()), int(waited.item())
