"""Whole-workload parity: every row of a full-size GPU result against the oracle.

The benchmark's workloads hold up to 65536 rows of 32000 logits (16.8 GB of
inputs and gradients together), more than the oracle should see at once.  The
rows are therefore brought to the host in chunks; each chunk is split into
small row blocks that a thread pool hands to the oracle (its C calls release
the GIL, so the blocks run on every host core), and every block is compared
with the GPU's rows under the rules of ``tests/parity.py`` (TVD near-tie rows
included).  Nothing is sampled: the report counts every row.
"""
from __future__ import annotations

import concurrent.futures as cf
import os

import numpy as np
import torch

import oracle
from tests.parity import LOSS_ATOL, LOSS_RTOL, TIE, grad_rows, near_tie_rows, tvd_ties


def _threads() -> int:
    return max(1, min(32, os.cpu_count() or 1))


def _block_distill(z, t, lg, gg, kind, beta, tau):
    """Oracle and comparison for one block of active rows (float32 numpy in)."""
    lr, gr = oracle.distill(z, t, None, kind, beta, temperature=tau)
    lg = lg.astype(np.float64)
    same_inf = np.isinf(lg) & (lg == lr)
    lerr = np.abs(lg - lr)
    loss_bad = ~same_inf & ~(lerr <= LOSS_RTOL * np.abs(lr) + LOSS_ATOL)
    fin = np.isfinite(lr)
    ties = tvd_ties(z[fin], t[fin], tau) if kind == "tvd" else None
    res = grad_rows(gg[fin].astype(np.float64), gr[fin], ties)
    lrel = np.where(~same_inf, lerr / np.maximum(np.abs(lr), 1e-30), 0.0)
    return {"rows": z.shape[0], "loss_bad": int(loss_bad.sum()), "grad_bad": int((~res["ok"]).sum()),
            "inf_rows": int((~fin).sum()),
            "grad_rel_max": float(np.nanmax(res["rel"])) if res["rel"].size else 0.0,
            "loss_rel_max": float(np.nanmax(lrel)) if lrel.size else 0.0,
            "tvd_skipped": int(ties.amb.sum()) if ties is not None else 0,
            "near_tie": int(res["near_tie"].sum()), "near_tie_differ": int(res["near_tie_differ"].sum())}


def distill_parity(z: torch.Tensor, t: torch.Tensor, active, loss_g: torch.Tensor, grad_g: torch.Tensor,
                   kind: str, beta: float, tau: float = 1.0, chunk: int = 4096, block: int = 64) -> dict:
    """Compare every row of (loss_g, grad_g) with the oracle.

    z, t: [N, V] logits (device or host, rows contiguous); active: bool [N]
    (numpy) or None for all rows; loss_g [N], grad_g [N, V]: the GPU results,
    inactive rows of grad_g expected to hold the NaN sentinel.  Asserts parity
    and returns the counts of the whole comparison."""
    N, V = z.shape
    act_all = np.ones(N, bool) if active is None else np.asarray(active, bool)
    tot = {"rows": 0, "loss_bad": 0, "grad_bad": 0, "inf_rows": 0, "grad_rel_max": 0.0, "loss_rel_max": 0.0,
           "tvd_skipped": 0, "near_tie": 0, "near_tie_differ": 0, "inactive_rows": 0}
    with cf.ThreadPoolExecutor(max_workers=_threads()) as ex:
        for c0 in range(0, N, chunk):
            c1 = min(N, c0 + chunk)
            act = act_all[c0:c1]
            lg = loss_g[c0:c1].cpu().numpy()
            idle = np.nonzero(~act)[0]
            if idle.size:
                assert np.all(lg[idle] == 0.0), "inactive rows must get loss 0"
                gi = grad_g[c0:c1][torch.as_tensor(idle, device=grad_g.device)]
                assert bool(torch.isnan(gi).all()), "inactive gradient rows must stay untouched"
                tot["inactive_rows"] += int(idle.size)
            rows = np.nonzero(act)[0]
            if rows.size == 0:
                continue
            ridx = torch.as_tensor(rows + c0, device=z.device)
            zc = z[ridx].float().cpu().numpy()
            tc = t[ridx].float().cpu().numpy()
            gc = grad_g[torch.as_tensor(rows + c0, device=grad_g.device)].cpu().numpy()
            lc = lg[rows]
            futs = [ex.submit(_block_distill, zc[b:b + block], tc[b:b + block], lc[b:b + block],
                              gc[b:b + block], kind, beta, tau)
                    for b in range(0, rows.size, block)]
            for f in futs:
                r = f.result()
                for key in ("rows", "loss_bad", "grad_bad", "inf_rows", "tvd_skipped", "near_tie", "near_tie_differ"):
                    tot[key] += r[key]
                tot["grad_rel_max"] = max(tot["grad_rel_max"], r["grad_rel_max"])
                tot["loss_rel_max"] = max(tot["loss_rel_max"], r["loss_rel_max"])
    assert tot["rows"] == int(act_all.sum())
    assert tot["loss_bad"] == 0, f"loss mismatch on {tot['loss_bad']} of {tot['rows']} rows: {tot}"
    assert tot["grad_bad"] == 0, f"gradient mismatch on {tot['grad_bad']} of {tot['rows']} rows: {tot}"
    return tot


def verify_oracle(draft, target, tokens, uniforms, T: float, block: int = 8) -> dict:
    """The oracle's verification of every sequence, blocks of sequences on the
    host cores; returns the same dict as ``oracle.verify``."""
    z, t, y, u = draft.cpu(), target.cpu(), tokens.cpu(), uniforms.cpu()
    B = y.shape[0]

    def one(b0):
        b1 = min(B, b0 + block)
        return oracle.verify(z[b0:b1], t[b0:b1], y[b0:b1], u[b0:b1], T)

    with cf.ThreadPoolExecutor(max_workers=_threads()) as ex:
        parts = list(ex.map(one, range(0, B, block)))
    return {key: np.concatenate([p[key] for p in parts]) for key in parts[0]}


def tie_report(ref: dict, tie: float = TIE) -> int:
    return int(near_tie_rows(ref, tie).sum())
