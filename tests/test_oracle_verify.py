"""Pins for the verify oracle (speculative sampling, Appendix A.1 and
Algorithm 1) against facts fixed outside the oracle:

* the output tokens follow the target distribution exactly (Section 3, the
  property proved by Leviathan et al.), checked by chi-square tests over 10^6
  seeded sequences on tiny vocabularies, at T = 1 and T != 1;
* the acceptance probability of one position is sum_x min(p, q) (closed form
  of the accept rule), and with the same (p, q) at every position the mean
  generated length is (1 - alpha^(k+1)) / (1 - alpha) (Eq. 1);
* the residual of a rejection is norm(max(0, p - q)) (Appendix A.1), checked
  statistically and on hand-built cases;
* T = 0 reduces to argmax-prefix matching (numpy argmax, first maximum);
* hand-built cases for the strict accept test, the uniform layout, the
  inverse-CDF convention and the bad-token sentinel.
"""
import math

import numpy as np
import pytest
from scipy.special import softmax
from scipy.stats import chisquare

import oracle


def _sample_rows(rng, probs, n):
    """n iid draws from each categorical row of probs [k, V] -> [n, k]."""
    k = probs.shape[0]
    out = np.empty((n, k), np.int32)
    for i in range(k):
        c = np.cumsum(probs[i])
        c[-1] = 1.0
        out[:, i] = np.searchsorted(c, rng.random(n), side="right")
    return out


def _run_mc(z1, t1, T, n, seed):
    """Verify n sequences that share per-position logits z1 [k, V], t1 [k+1, V]."""
    rng = np.random.default_rng(seed)
    k, V = z1.shape
    q = softmax(z1 / T, axis=1)
    y = _sample_rows(rng, q, n)
    u = rng.random((n, k + 1))
    z = np.broadcast_to(z1, (n, k, V))
    t = np.broadcast_to(t1, (n, k + 1, V))
    return oracle.verify(z, t, y, u, T), y


def _chi2_ok(tokens, probs, V):
    obs = np.bincount(tokens, minlength=V)
    exp = probs * len(tokens)
    keep = exp > 0
    assert np.all(obs[~keep] == 0)
    return chisquare(obs[keep], exp[keep]).pvalue


@pytest.mark.parametrize("T,V,k", [(1.0, 5, 3), (0.6, 4, 2), (1.7, 8, 1)])
def test_output_distribution_equals_target(T, V, k):
    """Every emitted token is distributed as p at its position."""
    rng = np.random.default_rng(1000 + V)
    z1 = rng.normal(0, 1.5, (k, V))
    t1 = rng.normal(0, 1.5, (k + 1, V))
    n = 1_000_000
    res, _ = _run_mc(z1, t1, T, n, seed=2000 + V)
    a = res["accepted"]
    out = res["out_tokens"]
    assert a.min() >= 0 and a.max() <= k
    p = softmax(t1 / T, axis=1)
    q = softmax(z1 / T, axis=1)
    for i in range(k + 1):
        emitted = a >= i          # position i is emitted iff the first i were accepted
        pv = _chi2_ok(out[emitted, i], p[i], V)
        assert pv > 1e-3, (i, pv)
    # acceptance at each position: P(a >= i+1 | a >= i) = sum min(p_i, q_i)
    for i in range(k):
        reach = np.sum(a >= i)
        acc = np.sum(a >= i + 1)
        alpha = np.minimum(p[i], q[i]).sum()
        sd = math.sqrt(alpha * (1 - alpha) / reach)
        assert abs(acc / reach - alpha) < 5 * sd, (i, acc / reach, alpha)


def test_expected_length_eq1():
    """Eq. 1: with the same (p, q) at every position, E[a + 1] = (1 - a^(k+1)) / (1 - a)."""
    rng = np.random.default_rng(77)
    V, k = 6, 4
    zrow = rng.normal(0, 1.0, V)
    trow = rng.normal(0, 1.0, V)
    z1 = np.tile(zrow, (k, 1))
    t1 = np.tile(trow, (k + 1, 1))
    res, _ = _run_mc(z1, t1, 1.0, 1_000_000, seed=78)
    alpha = np.minimum(softmax(trow), softmax(zrow)).sum()
    want = (1 - alpha ** (k + 1)) / (1 - alpha)
    L = res["accepted"] + 1.0
    assert abs(L.mean() - want) < 5 * L.std() / math.sqrt(len(L)), (L.mean(), want)


def test_residual_distribution_after_rejection():
    """Appendix A.1: after a rejection the extra token ~ norm(max(0, p - q))."""
    rng = np.random.default_rng(31)
    V, k = 6, 1
    z1 = rng.normal(0, 1.5, (k, V))
    t1 = rng.normal(0, 1.5, (k + 1, V))
    res, _ = _run_mc(z1, t1, 1.0, 1_000_000, seed=32)
    rej = res["accepted"] == 0
    w = np.maximum(softmax(t1[0]) - softmax(z1[0]), 0)
    pv = _chi2_ok(res["out_tokens"][rej, 0], w / w.sum(), V)
    assert pv > 1e-3
    assert np.all(res["mismatch_mask"][rej, 0] == 1)
    assert np.all(res["mismatch_mask"][~rej] == 0)


def _one(z, t, y, u, T=1.0):
    return oracle.verify(np.asarray(z, float)[None], np.asarray(t, float)[None],
                         np.asarray(y, np.int32)[None], np.asarray(u, float)[None], T)


def test_identical_distributions_accept_everything():
    """p == q gives r = 1 exactly, so every u < 1 accepts and a = k."""
    rng = np.random.default_rng(40)
    B, k, V = 64, 5, 50
    z = rng.normal(0, 2, (B, k + 1, V))
    y = rng.integers(0, V, (B, k)).astype(np.int32)
    u = rng.random((B, k + 1))
    res = oracle.verify(z[:, :k], z, y, u, 1.0)
    assert np.all(res["accepted"] == k)
    np.testing.assert_array_equal(res["out_tokens"][:, :k], y)
    assert np.all(res["mismatch_mask"] == 0)
    np.testing.assert_allclose(res["ratio"], 1.0, rtol=0, atol=1e-15)


def test_strict_accept_at_u_equal_r():
    """Reading of the accept test: strict u < r.  With p == q (r = 1) and
    u = 1 the proposal is rejected; the residual is empty (W = 0), so the
    extra token falls back to argmax p."""
    z = [[0.3, 1.2, -0.5]]
    t = [[0.3, 1.2, -0.5], [0.0, 0.0, 2.0]]
    res = _one(z, t, [0], [1.0, 0.4])
    assert res["accepted"][0] == 0
    assert res["out_tokens"][0].tolist() == [1, -1]
    res = _one(z, t, [0], [1.0 - 1e-12, 0.4])
    assert res["accepted"][0] == 1


def test_residual_hand_built():
    """p = (.4, .35, .1, .15), q = (.1, .25, .5, .15), draft token 2:
    r = 0.1 / 0.5 = 0.2 and w = max(0, p - q) = (.3, .1, 0, 0), W = 0.4."""
    p = np.array([0.4, 0.35, 0.1, 0.15])
    q = np.array([0.1, 0.25, 0.5, 0.15])
    z = [np.log(q)]
    t = [np.log(p), np.zeros(4)]
    res = _one(z, t, [2], [0.5, 0.7])          # tau = 0.28 < C_0 = 0.3
    assert res["accepted"][0] == 0 and res["out_tokens"][0].tolist() == [0, -1]
    assert res["ratio"][0, 0] == pytest.approx(0.2, rel=1e-12)
    assert res["margin"][0, 0] == pytest.approx(0.3, rel=1e-12)
    assert res["cdf_gap"][0] == pytest.approx(0.02 / 0.4, rel=1e-9)
    res = _one(z, t, [2], [0.5, 0.8])          # tau = 0.32 -> j* = 1
    assert res["out_tokens"][0].tolist() == [1, -1]
    res = _one(z, t, [2], [0.1, 0.8])          # u < r: accept, bonus from p_1
    assert res["accepted"][0] == 1 and res["out_tokens"][0, 0] == 2


def test_uniform_layout():
    """u[b, i] tests position i and u[b, k] drives the extra sample.
    Both positions have r = 0.5: u = (0.3, 0.9, .) accepts once."""
    p = np.array([0.2, 0.8])
    q = np.array([0.4, 0.6])
    z = [np.log(q), np.log(q)]
    t = [np.log(p), np.log(p), np.log([0.5, 0.5])]
    res = _one(z, t, [0, 0], [0.3, 0.9, 0.1])
    assert res["accepted"][0] == 1
    assert res["mismatch_mask"][0].tolist() == [0, 1]
    # residual at position 1 is all on token 1
    assert res["out_tokens"][0].tolist() == [0, 1, -1]


def test_inverse_cdf_convention():
    """Bonus sample (a = k) from p = (.1, .2, .3, .4): j* = min{j : C_j > u W},
    ascending index; zero-weight entries are never chosen."""
    p = np.log([0.1, 0.2, 0.3, 0.4])
    z = [p]
    t = [p, p]
    for u, want in [(0.0, 0), (0.0999999, 0), (0.1000001, 1), (0.25, 1), (0.6000001, 3), (0.999999, 3)]:
        res = _one(z, t, [3], [0.5, u])
        assert res["accepted"][0] == 1 and res["out_tokens"][0, 1] == want, (u, res)
    res = _one(z, t, [3], [0.5, 0.25])
    assert res["cdf_gap"][0] == pytest.approx(0.05, rel=1e-9)
    q0 = np.array([-np.inf, np.log(0.2), np.log(0.3), np.log(0.5)])
    res = _one([q0], [q0, q0], [1], [0.5, 0.0])
    assert res["out_tokens"][0].tolist() == [1, 1]


def test_greedy_is_argmax_prefix():
    """T = 0: accept while y_i == argmax t_i (first maximum), then emit
    argmax t_a; uniforms are ignored."""
    rng = np.random.default_rng(50)
    B, k, V = 400, 4, 7
    t = rng.integers(-3, 3, (B, k + 1, V)).astype(float)   # many ties
    am = np.argmax(t, axis=2)
    y = am[:, :k].copy()
    flip = rng.random((B, k)) < 0.3
    y[flip] = rng.integers(0, V, flip.sum())
    z = rng.normal(size=(B, k, V))
    res = oracle.verify(z, t, y.astype(np.int32), rng.random((B, k + 1)), 0.0)
    for b in range(B):
        a = 0
        while a < k and y[b, a] == am[b, a]:
            a += 1
        assert res["accepted"][b] == a
        assert res["out_tokens"][b, :a].tolist() == y[b, :a].tolist()
        assert res["out_tokens"][b, a] == am[b, a]
        assert np.all(res["out_tokens"][b, a + 1:] == -1)
        assert res["mismatch_mask"][b].tolist() == [int(i == a) for i in range(k)]


def test_bad_tokens_mark_the_sequence():
    rng = np.random.default_rng(60)
    B, k, V = 4, 3, 10
    z = rng.normal(size=(B, k, V))
    t = rng.normal(size=(B, k + 1, V))
    y = rng.integers(0, V, (B, k)).astype(np.int32)
    y[1, 2] = V
    y[3, 0] = -1
    for T in (1.0, 0.0):
        res = oracle.verify(z, t, y, rng.random((B, k + 1)), T)
        for b in (1, 3):
            assert res["accepted"][b] == -1
            assert np.all(res["out_tokens"][b] == -1)
            assert np.all(res["mismatch_mask"][b] == 0)
        assert res["accepted"][0] >= 0 and res["accepted"][2] >= 0


def test_draft_zero_probability_token():
    """q(y) = 0 and p(y) > 0: r = +inf, always accepted."""
    z = [[-np.inf, 0.0, 1.0]]
    t = [[0.5, 0.0, 0.0], [0.0, 0.0, 0.0]]
    res = _one(z, t, [0], [0.999, 0.3])
    assert res["accepted"][0] == 1 and res["ratio"][0, 0] == np.inf
