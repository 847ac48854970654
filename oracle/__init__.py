"""CPU oracle for the OSD verify and distill operations (test infrastructure).

TEST INFRASTRUCTURE ONLY: tests/, ``__graft_entry__.smoke()`` and the
``cpu_baseline`` leg of ``bench.py`` (plus ``--impl reference``) may import
this package.  The product path (``paper_2310_07177_gb300``) never does.

The arithmetic lives in ``osd_oracle.c`` (plain C, double precision); this
module only compiles it with gcc and marshals numpy arrays through ctypes.
Inputs of any float dtype are converted to float64, which is exact for bf16
and fp32 logits.  ``torch`` tensors are accepted and converted on the CPU.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "osd_oracle.c")
LIB_PATH = os.path.join(_HERE, "libosd_oracle.so")

LOSS_KINDS = {"fkl": 0, "rkl": 1, "jsd": 2, "tvd": 3, "ce": 4}

_lib = None
_lock = threading.Lock()


GCC_FLAGS = ["-O2", "-std=c99", "-fPIC", "-shared", "-ffp-contract=off", "-fno-fast-math"]


def compile_source(src: str, out: str) -> str:
    """gcc one oracle source file into a shared library (IEEE double, no FMA
    contraction, so x86 and aarch64 round identically)."""
    tmp = out + f".tmp{os.getpid()}"
    subprocess.run(["gcc", *GCC_FLAGS, "-o", tmp, src, "-lm"], check=True)
    os.replace(tmp, out)
    return out


def build(force: bool = False) -> str:
    """Compile osd_oracle.c into libosd_oracle.so unless it is up to date."""
    if (not force and os.path.exists(LIB_PATH)
            and os.path.getmtime(LIB_PATH) >= os.path.getmtime(_SRC)):
        return LIB_PATH
    return compile_source(_SRC, LIB_PATH)


def _load():
    global _lib
    with _lock:
        if _lib is not None:
            return _lib
        # OSD_ORACLE_LIB lets tests/test_oracle_mutants.py load a copy of the
        # oracle compiled with a planted mistake, to show the pins catch it.
        path = os.environ.get("OSD_ORACLE_LIB")
        if not path:
            path = build()
        lib = ctypes.CDLL(path)
        dp = ctypes.POINTER(ctypes.c_double)
        i32p = ctypes.POINTER(ctypes.c_int32)
        u8p = ctypes.POINTER(ctypes.c_uint8)
        L = ctypes.c_long
        lib.osd_oracle_verify.restype = ctypes.c_int
        lib.osd_oracle_verify.argtypes = [dp, dp, L, L, L, i32p, dp, ctypes.c_double,
                                          i32p, i32p, u8p, dp, dp, dp]
        lib.osd_oracle_distill.restype = ctypes.c_int
        lib.osd_oracle_distill.argtypes = [dp, dp, L, L, u8p, ctypes.c_int,
                                           ctypes.c_double, ctypes.c_double, dp, dp]
        lib.osd_oracle_log_softmax.restype = None
        lib.osd_oracle_log_softmax.argtypes = [dp, L, ctypes.c_double, dp]
        lib.osd_oracle_verify_tree.restype = ctypes.c_int
        lib.osd_oracle_verify_tree.argtypes = [dp, dp, L, L, L, i32p, i32p, dp, ctypes.c_double,
                                               i32p, i32p, i32p, i32p, dp, dp]
        lib.osd_oracle_mixed_sample.restype = ctypes.c_int
        lib.osd_oracle_mixed_sample.argtypes = [dp, dp, L, L, L, L, dp, ctypes.c_double, ctypes.c_double,
                                                i32p, dp]
        _lib = lib
        return lib


def _np(x, dtype):
    if hasattr(x, "detach"):  # torch tensor
        x = x.detach().to("cpu")
        if dtype is np.float64:
            x = x.double()
        x = x.numpy()
    return np.ascontiguousarray(np.asarray(x, dtype=dtype))


def _ptr(a, ctype):
    return a.ctypes.data_as(ctypes.POINTER(ctype))


def log_softmax(x, temperature: float = 1.0) -> np.ndarray:
    """Row-wise log softmax(x / T) in double precision."""
    lib = _load()
    x = _np(x, np.float64)
    out = np.empty_like(x)
    V = x.shape[-1]
    xf = x.reshape(-1, V)
    of = out.reshape(-1, V)
    for r in range(xf.shape[0]):
        lib.osd_oracle_log_softmax(_ptr(xf[r], ctypes.c_double), V,
                                   float(temperature), _ptr(of[r], ctypes.c_double))
    return out


def verify(draft_logits, target_logits, draft_tokens, uniforms, temperature):
    """Speculative-sampling verification (Appendix A.1), double precision.

    draft_logits [B, k, V], target_logits [B, k+1, V], draft_tokens [B, k],
    uniforms [B, k+1], temperature a float (pass the exact fp32 value the GPU
    sees, e.g. ``float(np.float32(0.7))``).  Returns a dict with accepted [B],
    out_tokens [B, k+1], mismatch_mask [B, k], margin [B, k], cdf_gap [B],
    ratio [B, k].
    """
    lib = _load()
    z = _np(draft_logits, np.float64)
    t = _np(target_logits, np.float64)
    y = _np(draft_tokens, np.int32)
    u = _np(uniforms, np.float64)
    B, k, V = z.shape
    assert t.shape == (B, k + 1, V) and y.shape == (B, k) and u.shape == (B, k + 1)
    acc = np.empty(B, np.int32)
    out = np.empty((B, k + 1), np.int32)
    mask = np.empty((B, k), np.uint8)
    margin = np.empty((B, k), np.float64)
    gap = np.empty(B, np.float64)
    ratio = np.empty((B, k), np.float64)
    rc = lib.osd_oracle_verify(_ptr(z, ctypes.c_double), _ptr(t, ctypes.c_double), B, k, V,
                               _ptr(y, ctypes.c_int32), _ptr(u, ctypes.c_double),
                               float(temperature), _ptr(acc, ctypes.c_int32),
                               _ptr(out, ctypes.c_int32), _ptr(mask, ctypes.c_uint8),
                               _ptr(margin, ctypes.c_double), _ptr(gap, ctypes.c_double),
                               _ptr(ratio, ctypes.c_double))
    if rc != 0:
        raise ValueError("osd_oracle_verify rejected its arguments")
    return {"accepted": acc, "out_tokens": out, "mismatch_mask": mask,
            "margin": margin, "cdf_gap": gap, "ratio": ratio}


def distill(draft_logits, target_logits, mask=None, loss_kind="fkl", beta=0.5,
            dlogits_init=None, temperature=1.0):
    """Per-position distillation loss and d loss / d draft_logits (Eq. 2-3),
    both softmaxes at ``temperature`` (Section 4.1); ``loss_kind`` "ce" is the
    label fine-tuning cross-entropy to the target argmax.

    draft_logits, target_logits [N, V] (any leading shape is flattened to
    rows); mask [N] of 0/1 or None.  Returns (loss [N], dlogits [N, V]) in
    float64.  Rows with mask 0 get loss 0 and keep ``dlogits_init`` (NaN by
    default) in their gradient row.
    """
    lib = _load()
    z = _np(draft_logits, np.float64)
    t = _np(target_logits, np.float64)
    V = z.shape[-1]
    lead = z.shape[:-1]
    z = z.reshape(-1, V)
    t = t.reshape(-1, V)
    N = z.shape[0]
    assert t.shape == (N, V)
    m = None if mask is None else _np(mask, np.uint8).reshape(-1)
    loss = np.empty(N, np.float64)
    if dlogits_init is None:
        g = np.full((N, V), np.nan, np.float64)
    else:
        g = _np(dlogits_init, np.float64).reshape(N, V).copy()
    kind = LOSS_KINDS[loss_kind] if isinstance(loss_kind, str) else int(loss_kind)
    rc = lib.osd_oracle_distill(_ptr(z, ctypes.c_double), _ptr(t, ctypes.c_double), N, V,
                                None if m is None else _ptr(m, ctypes.c_uint8),
                                kind, float(beta), float(temperature), _ptr(loss, ctypes.c_double),
                                _ptr(g, ctypes.c_double))
    if rc != 0:
        raise ValueError("osd_oracle_distill rejected its arguments")
    return loss.reshape(lead), g.reshape(*lead, V)


def distill_rejected(draft_logits, target_logits, accepted, loss_kind="rkl", beta=0.5, temperature=1.0):
    """Distillation on the positions verification rejected (Algorithm 1).

    Each serving step of Algorithm 1 stores, for every sequence whose draft
    proposal was cut short, the first rejected position and the target's
    distribution there in the buffer R; the loss of Eq. 2 is then taken over R.
    Sequence b has a = accepted[b] accepted tokens: it contributes draft row
    (b, a) of draft_logits [B, k, V] and target row (b, a) of target_logits
    [B, k+1, V] when 0 <= a < k, and nothing when a == k (every token
    accepted) or a == -1 (a bad draft token).

    Returns (loss [B], dlogits [B, V], seq_of_row [B], count) in the order of a
    stable partition: the count active sequences first in increasing b, then
    the inactive ones; loss is 0 and dlogits NaN in the inactive slots.
    """
    z = _np(draft_logits, np.float64)
    t = _np(target_logits, np.float64)
    acc = _np(accepted, np.int64).reshape(-1)
    B, k, V = z.shape
    assert t.shape == (B, k + 1, V) and acc.shape == (B,)
    active = [b for b in range(B) if 0 <= acc[b] < k]
    inactive = [b for b in range(B) if not 0 <= acc[b] < k]
    loss = np.zeros(B, np.float64)
    g = np.full((B, V), np.nan, np.float64)
    if active:
        rows_z = np.stack([z[b, acc[b]] for b in active])
        rows_t = np.stack([t[b, acc[b]] for b in active])
        l, gr = distill(rows_z, rows_t, None, loss_kind, beta, temperature=temperature)
        loss[:len(active)] = l
        g[:len(active)] = gr
    seq = np.array(active + inactive, np.int64)
    return loss, g, seq, len(active)


def mixed_sample(draft_logits, target_logits, uniforms, beta, temperature=1.0):
    """One token per row from beta p + (1 - beta) q (Section 4.1, mixed
    sampling), p = softmax(target / T), q = softmax(draft / T), by inverse CDF
    in ascending vocabulary order with uniforms [N].  Rows are [N, V] (any
    leading shape is flattened).  Returns (tokens [N] int32, cdf_gap [N])."""
    lib = _load()
    z = _np(draft_logits, np.float64)
    t = _np(target_logits, np.float64)
    V = z.shape[-1]
    z = z.reshape(-1, V)
    t = t.reshape(-1, V)
    N = z.shape[0]
    assert t.shape == (N, V)
    u = _np(uniforms, np.float64).reshape(-1)
    assert u.shape == (N,)
    tok = np.empty(N, np.int32)
    gap = np.empty(N, np.float64)
    rc = lib.osd_oracle_mixed_sample(_ptr(z, ctypes.c_double), _ptr(t, ctypes.c_double), N, V, V, V,
                                     _ptr(u, ctypes.c_double), float(beta), float(temperature),
                                     _ptr(tok, ctypes.c_int32), _ptr(gap, ctypes.c_double))
    if rc != 0:
        raise ValueError("osd_oracle_mixed_sample rejected its arguments")
    return tok, gap


def verify_tree(draft_logits, target_logits, parent, tokens, uniforms, temperature):
    """Multi-candidate verification over a token tree (the tree-style decoding
    of the paper's Medusa study), double precision.

    draft_logits, target_logits [B, n_nodes, V]; parent [n_nodes] (parent[0] =
    -1, parent[i] < i); tokens [B, n_nodes] (node 0 unused); uniforms
    [B, n_nodes] (u[:, 0] drives the extra draw, u[:, i] tests node i).
    Returns a dict with accepted [B], path [B, n_nodes], out_tokens
    [B, n_nodes], last_node [B], margin [B, n_nodes], cdf_gap [B].
    """
    lib = _load()
    z = _np(draft_logits, np.float64)
    t = _np(target_logits, np.float64)
    par = _np(parent, np.int32).reshape(-1)
    y = _np(tokens, np.int32)
    u = _np(uniforms, np.float64)
    B, n, V = t.shape
    assert z.shape == (B, n, V) and par.shape == (n,) and y.shape == (B, n) and u.shape == (B, n)
    acc = np.empty(B, np.int32)
    path = np.empty((B, n), np.int32)
    out = np.empty((B, n), np.int32)
    last = np.empty(B, np.int32)
    margin = np.empty((B, n), np.float64)
    gap = np.empty(B, np.float64)
    rc = lib.osd_oracle_verify_tree(_ptr(z, ctypes.c_double), _ptr(t, ctypes.c_double), B, n, V,
                                    _ptr(par, ctypes.c_int32), _ptr(y, ctypes.c_int32), _ptr(u, ctypes.c_double),
                                    float(temperature), _ptr(acc, ctypes.c_int32), _ptr(path, ctypes.c_int32),
                                    _ptr(out, ctypes.c_int32), _ptr(last, ctypes.c_int32),
                                    _ptr(margin, ctypes.c_double), _ptr(gap, ctypes.c_double))
    if rc != 0:
        raise ValueError("osd_oracle_verify_tree rejected its arguments")
    return {"accepted": acc, "path": path, "out_tokens": out, "last_node": last, "margin": margin,
            "cdf_gap": gap}
