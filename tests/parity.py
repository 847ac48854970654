"""Comparison rules between the CUDA path and the oracle.

Decisions (accepted counts, output tokens, mismatch masks) must be bit-exact,
except in sequences where the oracle's accept margin |u - r| or its CDF
boundary gap is below 1e-6: there fp32 and fp64 may legitimately disagree, so
those sequences are counted and only checked for validity.  Losses must agree
to |l - l_ref| <= 1e-4 |l_ref| + 1e-6 and gradients, row by row, to
max|g - g_ref| <= 1e-4 max|g_ref| + 1e-7 (an elementwise relative error is
meaningless for entries of 1e-9; the 1e-7 floor is fp32 resolution of
probabilities, reached when p and q nearly coincide and every entry is ~0).
TVD's gradient is compared as ``grad_rows`` describes: entries where fp32
cannot order q and p are left out, and rows where their sign choice could
matter must match the subgradient of the GPU's own choice there.
"""
from __future__ import annotations

from typing import NamedTuple, Optional

import numpy as np

TIE = 1e-6
LOSS_RTOL, LOSS_ATOL = 1e-4, 1e-6
GRAD_RTOL = 1e-4
GRAD_ATOL = 1e-7


def near_tie_rows(ref: dict, tie: float = TIE) -> np.ndarray:
    margin = np.where(np.isnan(ref["margin"]), np.inf, ref["margin"])
    gap = np.where(np.isnan(ref["cdf_gap"]), np.inf, ref["cdf_gap"])
    return (margin.min(axis=1) < tie) | (gap < tie)


def check_verify(gpu, ref: dict, k: int, V: int, tie: float = TIE) -> dict:
    """Assert decision parity; returns counts for the report."""
    acc = gpu.accepted.cpu().numpy()
    out = gpu.out_tokens.cpu().numpy()
    mask = gpu.mismatch_mask.cpu().numpy()
    B = acc.shape[0]
    flagged = near_tie_rows(ref, tie)
    ok = ~flagged
    bad_acc = np.nonzero(ok & (acc != ref["accepted"]))[0]
    assert bad_acc.size == 0, (f"accepted differs at {bad_acc[:8]}: gpu {acc[bad_acc[:8]]} "
                               f"oracle {ref['accepted'][bad_acc[:8]]} margins {ref['margin'][bad_acc[:8]]}")
    bad_out = np.nonzero(ok & np.any(out != ref["out_tokens"], axis=1))[0]
    assert bad_out.size == 0, (f"out_tokens differ at {bad_out[:8]}: gpu {out[bad_out[:4]]} oracle "
                               f"{ref['out_tokens'][bad_out[:4]]} gaps {ref['cdf_gap'][bad_out[:4]]}")
    bad_mask = np.nonzero(ok & np.any(mask != ref["mismatch_mask"], axis=1))[0]
    assert bad_mask.size == 0, f"mismatch_mask differs at {bad_mask[:8]}"
    # every sequence, flagged or not, must be a valid outcome
    for b in range(B):
        a = acc[b]
        if ref["accepted"][b] < 0:
            assert a == -1 and np.all(out[b] == -1) and np.all(mask[b] == 0)
            continue
        assert 0 <= a <= k
        assert np.all(out[b, a + 1:] == -1) and 0 <= out[b, a] < V
        assert mask[b].sum() == (1 if a < k else 0)
    differ = flagged & ((acc != ref["accepted"]) | np.any(out != ref["out_tokens"], axis=1))
    return {"sequences": B, "near_tie": int(flagged.sum()), "near_tie_differ": int(differ.sum())}


def check_margins(gpu, ref: dict, tol: float = 2e-6) -> float:
    """|margin_gpu - margin_oracle| over positions both sides decided; returns the max."""
    if gpu.diag_margin is None:
        return 0.0
    mg = gpu.diag_margin.cpu().numpy().astype(np.float64)
    mr = ref["margin"]
    both = np.isfinite(mg) & np.isfinite(mr)
    if not both.any():
        return 0.0
    err = np.abs(mg[both] - mr[both]) / np.maximum(1.0, np.abs(ref["ratio"][both]))
    worst = float(err.max())
    assert worst <= tol, f"accept ratio error {worst:.3g} exceeds {tol}"
    return worst


TVD_TIE = 1e-5  # |ln q - ln p| below this: fp32 cannot tell which of q and p is larger


class TvdTies(NamedTuple):
    """What the TVD comparison needs from the oracle besides its gradient:
    amb [rows, V] marks entries whose sign(q - p) fp32 cannot decide; q and
    d = ln q - ln p are the oracle's (float64); tau the temperature."""
    amb: np.ndarray
    q: np.ndarray
    d: np.ndarray
    tau: float


def tvd_ties(z, t, tau: float = 1.0) -> TvdTies:
    import oracle
    V = z.shape[-1]
    lq = oracle.log_softmax(np.asarray(z, np.float64).reshape(-1, V), tau)
    lp = oracle.log_softmax(np.asarray(t, np.float64).reshape(-1, V), tau)
    d = lq - lp
    return TvdTies(np.abs(d) < TVD_TIE, np.exp(lq), d, float(tau))


def tvd_subgradient(q: np.ndarray, s: np.ndarray, tau: float) -> np.ndarray:
    """d/dz of 1/2 sum|p - q| for the sign choice s_j in {-1, 0, 1} of
    sign(q_j - p_j): q_k (s_k / 2 - sum_j q_j s_j / 2) / tau (reading 9)."""
    return q * (0.5 * s - 0.5 * np.sum(q * s, axis=1, keepdims=True)) / tau


def grad_rows(gg: np.ndarray, gr: np.ndarray, tvd: Optional[TvdTies] = None) -> dict:
    """Row-by-row gradient comparison (float64 [rows, V]).

    TVD is not differentiable where q_j = p_j: any value in [-1/2, 1/2] of the
    sign there gives a valid subgradient (reading 9).  Entries whose order fp32
    cannot decide (|ln q - ln p| < 1e-5) are left out of the comparison, and
    their sign also enters every other entry through sum_j q_j s_j / 2: a flip
    moves entry k by up to q_k (sum of q over those entries) / tau.  Rows where
    that can exceed half the tolerance are near-tie rows: there the GPU's
    gradient must equal the exact subgradient for the signs it chose at those
    entries (read off its own gradient), with the oracle's q and its signs
    everywhere else.  Returns ok, rel [rows] and the near_tie, near_tie_differ
    masks."""
    rows = gg.shape[0]
    near = np.zeros(rows, bool)
    differ = np.zeros(rows, bool)
    g, r = gg, gr
    if tvd is not None:
        g = np.where(tvd.amb, 0.0, gg)
        r = np.where(tvd.amb, 0.0, gr)
    scale = np.max(np.abs(r), axis=1)
    lim = GRAD_RTOL * scale + GRAD_ATOL
    err = np.max(np.abs(g - r), axis=1)
    ok = err <= lim
    rel = err / np.maximum(scale, GRAD_ATOL / GRAD_RTOL)
    if tvd is not None:
        qmax = np.max(np.where(tvd.amb, 0.0, tvd.q), axis=1)
        shift = qmax * np.sum(np.where(tvd.amb, tvd.q, 0.0), axis=1) / tvd.tau
        near = shift > 0.5 * lim
        for i in np.nonzero(near & ~ok)[0]:
            s = np.where(tvd.amb[i], np.sign(gg[i]), np.sign(tvd.d[i]))[None, :]
            alt = tvd_subgradient(tvd.q[i][None, :], s, tvd.tau)[0]
            e2 = np.max(np.abs(gg[i] - alt))
            if e2 <= lim[i]:
                ok[i] = True
                differ[i] = True
                rel[i] = e2 / max(scale[i], GRAD_ATOL / GRAD_RTOL)
    return {"ok": ok, "rel": rel, "near_tie": near, "near_tie_differ": differ}


def check_distill(loss_g, grad_g, loss_r, grad_r, active: np.ndarray, skip_elems=None) -> dict:
    """Loss / gradient parity on active rows; inactive rows keep their sentinel."""
    lg = np.asarray(loss_g, np.float64)
    gg = np.asarray(grad_g, np.float64)
    lr = np.asarray(loss_r, np.float64)
    gr = np.asarray(grad_r, np.float64)
    act = np.asarray(active, bool)
    assert np.all(lg[~act] == 0.0), "inactive rows must get loss 0"
    assert np.all(np.isnan(gg[~act])), "inactive gradient rows must stay untouched"
    la, lra = lg[act], lr[act]
    same_inf = np.isinf(la) & (la == lra)
    err = np.abs(la - lra)
    lim = LOSS_RTOL * np.abs(lra) + LOSS_ATOL
    bad = ~same_inf & ~(err <= lim)
    assert not bad.any(), f"loss mismatch: gpu {la[bad][:5]} oracle {lra[bad][:5]}"
    # rows with an infinite loss (q puts mass where p has none, for RKL) have no
    # defined gradient on either side: only the loss is compared there
    fin = np.isfinite(lra)
    ga, gra = gg[act][fin], gr[act][fin]
    tvd = None
    if skip_elems is not None:  # a TvdTies for the same rows as the logits
        sel = np.nonzero(act)[0][fin]
        tvd = TvdTies(skip_elems.amb[sel], skip_elems.q[sel], skip_elems.d[sel], skip_elems.tau)
    assert np.all(np.isfinite(ga)), "non-finite gradients"
    res = grad_rows(ga, gra, tvd)
    worst = float(res["rel"].max()) if res["rel"].size else 0.0
    assert np.all(res["ok"]), f"gradient mismatch: worst row-relative error {worst:.3g}"
    lrel = err[~same_inf] / np.maximum(np.abs(lra[~same_inf]), 1e-30)
    return {"rows": int(act.sum()), "infinite_loss_rows": int((~fin).sum()), "grad_rel_max": worst,
            "loss_rel_max": float(lrel.max()) if lrel.size else 0.0,
            "near_tie": int(res["near_tie"].sum()), "near_tie_differ": int(res["near_tie_differ"].sum())}
