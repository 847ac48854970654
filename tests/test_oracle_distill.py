"""Pins for the distill oracle (Eq. 2-3, Section 4.1) against facts fixed
outside the oracle: hand-derived closed forms, scipy's entropy and
Jensen-Shannon routines, invariants of the divergences, and central finite
differences of the oracle's own loss for the gradient formulas."""
import math
import os

import numpy as np
import pytest
from scipy.spatial.distance import cityblock, jensenshannon
from scipy.special import log_softmax, rel_entr, softmax
from scipy.stats import entropy

import oracle

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "distill_v2_worked.txt")
KINDS = ["fkl", "rkl", "jsd", "tvd", "ce"]


def _golden():
    vals = {}
    for line in open(GOLDEN):
        if line.startswith("#") or not line.strip():
            continue
        name, expr, val = line.split()
        v = float(val)
        # the stored value must be its own closed form
        assert abs(eval(expr, {"ln": math.log, "min": min}) - v) < 1e-15
        vals[name] = v
    return vals


def test_worked_example_v2():
    """Eq. 3 on p = (1/2, 1/2), q = (3/4, 1/4): tests/golden/distill_v2_worked.txt."""
    g = _golden()
    z = np.array([[math.log(3.0), 0.0]])
    t = np.array([[0.0, 0.0]])
    for kind, beta, lname, gname in [("fkl", 0.5, "loss_fkl", "grad_fkl"),
                                     ("rkl", 0.5, "loss_rkl", "grad_rkl"),
                                     ("jsd", 0.5, "loss_jsd_0.5", "grad_jsd_0.5"),
                                     ("jsd", 0.1, "loss_jsd_0.1", None),
                                     ("jsd", 0.9, "loss_jsd_0.9", None),
                                     ("tvd", 0.5, "loss_tvd", "grad_tvd"),
                                     ("ce", 0.5, "loss_ce", "grad_ce")]:
        loss, grad = oracle.distill(z, t, loss_kind=kind, beta=beta)
        assert abs(loss[0] - g[lname]) < 1e-14, (kind, beta, loss[0], g[lname])
        if gname:
            assert abs(grad[0, 0] - g[gname]) < 1e-14, (kind, grad[0])
            assert abs(grad[0, 1] + g[gname]) < 1e-14, (kind, grad[0])


def _rows(rng, n, V, scale=2.0):
    z = rng.normal(0, scale, (n, V))
    t = z + rng.normal(0, 1.0, (n, V))
    return z, t


@pytest.mark.parametrize("V", [3, 50, 1000])
def test_kl_matches_scipy_entropy(V):
    """FKL = KL(p||q), RKL = KL(q||p) (Eq. 3) against scipy.stats.entropy."""
    rng = np.random.default_rng(11 + V)
    z, t = _rows(rng, 6, V)
    fkl, _ = oracle.distill(z, t, loss_kind="fkl")
    rkl, _ = oracle.distill(z, t, loss_kind="rkl")
    for n in range(6):
        p, q = softmax(t[n]), softmax(z[n])
        assert fkl[n] == pytest.approx(entropy(p, q), rel=1e-11, abs=1e-14)
        assert rkl[n] == pytest.approx(entropy(q, p), rel=1e-11, abs=1e-14)


@pytest.mark.parametrize("beta", [0.5, 0.2, 0.85])
def test_jsd_matches_scipy(beta):
    """JSD[beta] of Eq. 3; at beta = 1/2 it is scipy's Jensen-Shannon distance squared."""
    rng = np.random.default_rng(5)
    z, t = _rows(rng, 5, 200)
    loss, _ = oracle.distill(z, t, loss_kind="jsd", beta=beta)
    for n in range(5):
        p, q = softmax(t[n]), softmax(z[n])
        m = beta * p + (1 - beta) * q
        want = beta * entropy(p, m) + (1 - beta) * entropy(q, m)
        assert loss[n] == pytest.approx(want, rel=1e-11, abs=1e-14)
        if beta == 0.5:
            assert loss[n] == pytest.approx(jensenshannon(p, q) ** 2, rel=1e-9)


def test_tvd_matches_scipy_cityblock():
    rng = np.random.default_rng(6)
    z, t = _rows(rng, 5, 300)
    loss, _ = oracle.distill(z, t, loss_kind="tvd")
    for n in range(5):
        assert loss[n] == pytest.approx(0.5 * cityblock(softmax(t[n]), softmax(z[n])), rel=1e-12)


def _fd_grad(z, t, kind, beta, tau=1.0, h=1e-6):
    g = np.empty_like(z)
    for j in range(z.shape[-1]):
        zp, zm = z.copy(), z.copy()
        zp[0, j] += h
        zm[0, j] -= h
        lp, _ = oracle.distill(zp, t, loss_kind=kind, beta=beta, temperature=tau)
        lm, _ = oracle.distill(zm, t, loss_kind=kind, beta=beta, temperature=tau)
        g[0, j] = (lp[0] - lm[0]) / (2 * h)
    return g


@pytest.mark.parametrize("kind", KINDS)
@pytest.mark.parametrize("V", [2, 7, 64])
@pytest.mark.parametrize("tau", [1.0, 0.5, 2.0])
def test_gradient_matches_central_differences(kind, V, tau):
    """The analytic gradient w.r.t. the raw draft logits (Algorithm 1, update
    step; temperature of Section 4.1) against central finite differences of
    the oracle's loss."""
    rng = np.random.default_rng(100 + V + 7 * KINDS.index(kind) + int(10 * tau))
    for beta in ([0.5, 0.3] if kind == "jsd" else [0.5]):
        z, t = _rows(rng, 1, V, scale=1.5)
        while kind == "tvd" and np.min(np.abs(softmax(t[0] / tau) - softmax(z[0] / tau))) < 1e-5:
            z, t = _rows(rng, 1, V, scale=1.5)  # FD is only valid off the kinks of |p - q|
        _, g = oracle.distill(z, t, loss_kind=kind, beta=beta, temperature=tau)
        fd = _fd_grad(z, t, kind, beta, tau)
        np.testing.assert_allclose(g, fd, atol=4e-8, rtol=1e-6)


def test_ce_matches_scipy_log_softmax():
    """FT (Table 1): cross-entropy of q to the target's argmax label."""
    rng = np.random.default_rng(21)
    z, t = _rows(rng, 6, 300)
    t[2, 7] = t[2, 9] = t[2].max() + 1.0  # tie: the lowest index is the label
    for tau in (1.0, 0.7):
        loss, _ = oracle.distill(z, t, loss_kind="ce", temperature=tau)
        for n in range(6):
            y = int(np.argmax(t[n]))
            assert loss[n] == pytest.approx(-log_softmax(z[n] / tau)[y], rel=1e-12)
    assert int(np.argmax(t[2])) == 7


@pytest.mark.parametrize("kind", ["fkl", "rkl", "jsd", "tvd"])
def test_temperature_against_library(kind):
    """Section 4.1: temperature divides both rows' logits before the softmax."""
    rng = np.random.default_rng(22)
    z, t = _rows(rng, 4, 120)
    tau = 0.6
    loss, _ = oracle.distill(z, t, loss_kind=kind, beta=0.5, temperature=tau)
    for n in range(4):
        p, q = softmax(t[n] / tau), softmax(z[n] / tau)
        m = 0.5 * (p + q)
        want = {"fkl": entropy(p, q), "rkl": entropy(q, p),
                "jsd": 0.5 * entropy(p, m) + 0.5 * entropy(q, m),
                "tvd": 0.5 * cityblock(p, q)}[kind]
        assert loss[n] == pytest.approx(want, rel=1e-10, abs=1e-14)


@pytest.mark.parametrize("kind", KINDS)
def test_gradient_sums_to_zero(kind):
    """Softmax is invariant to adding a constant to z, so sum_k dl/dz_k = 0."""
    rng = np.random.default_rng(3)
    z, t = _rows(rng, 4, 500)
    _, g = oracle.distill(z, t, loss_kind=kind, beta=0.4)
    assert np.max(np.abs(g.sum(axis=1))) < 1e-12


@pytest.mark.parametrize("kind", ["fkl", "rkl", "jsd", "tvd"])
def test_identical_inputs_give_zero(kind):
    rng = np.random.default_rng(4)
    z = rng.normal(0, 3, (3, 400))
    loss, g = oracle.distill(z, z.copy(), loss_kind=kind, beta=0.5)
    assert np.all(np.abs(loss) < 1e-13)
    assert np.all(np.abs(g) < 1e-15)


@pytest.mark.parametrize("kind", KINDS)
def test_shift_invariance(kind):
    rng = np.random.default_rng(8)
    z, t = _rows(rng, 2, 100)
    l0, g0 = oracle.distill(z, t, loss_kind=kind, beta=0.3)
    l1, g1 = oracle.distill(z + 7.25, t - 3.5, loss_kind=kind, beta=0.3)
    np.testing.assert_allclose(l1, l0, rtol=1e-11, atol=1e-13)
    np.testing.assert_allclose(g1, g0, rtol=1e-9, atol=1e-13)


def test_jsd_endpoints_and_symmetry():
    """m = q at beta = 0 and m = p at beta = 1, so both endpoints give 0;
    JSD[1/2] is symmetric in p and q (loss only)."""
    rng = np.random.default_rng(9)
    z, t = _rows(rng, 3, 80)
    for beta in (0.0, 1.0):
        loss, g = oracle.distill(z, t, loss_kind="jsd", beta=beta)
        assert np.all(np.abs(loss) < 1e-14) and np.all(np.abs(g) < 1e-15)
    a, _ = oracle.distill(z, t, loss_kind="jsd", beta=0.5)
    b, _ = oracle.distill(t, z, loss_kind="jsd", beta=0.5)
    np.testing.assert_allclose(a, b, rtol=1e-12)


def test_bounds():
    rng = np.random.default_rng(10)
    z, t = _rows(rng, 20, 64, scale=4.0)
    fkl, _ = oracle.distill(z, t, loss_kind="fkl")
    jsd, _ = oracle.distill(z, t, loss_kind="jsd", beta=0.5)
    tvd, _ = oracle.distill(z, t, loss_kind="tvd")
    assert np.all(fkl >= 0)
    assert np.all((jsd >= 0) & (jsd <= math.log(2)))
    assert np.all((tvd >= 0) & (tvd <= 1))


def test_mask_leaves_inactive_rows_untouched():
    rng = np.random.default_rng(12)
    z, t = _rows(rng, 6, 33)
    mask = np.array([1, 0, 1, 0, 0, 1], np.uint8)
    loss, g = oracle.distill(z, t, mask=mask, loss_kind="rkl")
    assert np.all(loss[mask == 0] == 0)
    assert np.all(np.isnan(g[mask == 0]))
    assert np.all(np.isfinite(g[mask == 1]))
    full, gfull = oracle.distill(z, t, loss_kind="rkl")
    np.testing.assert_array_equal(loss[mask == 1], full[mask == 1])
    np.testing.assert_array_equal(g[mask == 1], gfull[mask == 1])


def test_minus_inf_entries():
    """-inf logits are probability 0: they contribute nothing (0 log 0 = 0)."""
    z = np.array([[0.0, 1.0, -np.inf, 0.5]])
    t = np.array([[0.2, -np.inf, -np.inf, 0.1]])
    fkl, gf = oracle.distill(z, t, loss_kind="fkl")
    p = softmax(np.array([0.2, 0.1]))
    q = softmax(np.array([0.0, 1.0, 0.5]))
    # rel_entr does not renormalise q, which keeps mass on vocabulary entry 1
    assert fkl[0] == pytest.approx(rel_entr(p, q[[0, 2]]).sum(), rel=1e-12)
    assert gf[0, 2] == 0.0
    rkl, _ = oracle.distill(z, t, loss_kind="rkl")
    assert rkl[0] == np.inf  # q puts mass where p has none
