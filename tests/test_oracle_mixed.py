"""Pins for the mixed-sampling oracle (Section 4.1: y ~ beta p + (1 - beta) q)
against facts fixed outside it:

* the sampled tokens follow the mixture beta softmax(t/T) + (1 - beta)
  softmax(z/T), computed with scipy, by chi-square over 2e5 draws, at
  beta in {0, 0.3, 1} and T in {1, 0.6};
* at beta = 1 the draw is the verify oracle's bonus token (the inverse-CDF
  draw from p when every proposal is accepted), token for token;
* hand-built cases fix the inverse-CDF convention: ascending index, strict
  C_j > u W, zero-weight entries never chosen, the reported CDF gap.
"""
import numpy as np
import pytest
from scipy.special import softmax
from scipy.stats import chisquare

import oracle

pytestmark = pytest.mark.filterwarnings("ignore::RuntimeWarning")


def _rows(V, seed):
    rng = np.random.default_rng(seed)
    return rng.normal(0, 1.2, V), rng.normal(0, 1.2, V)


@pytest.mark.parametrize("beta", [0.0, 0.3, 1.0])
@pytest.mark.parametrize("T", [1.0, 0.6])
def test_draws_follow_the_mixture(beta, T):
    V, n = 6, 200_000
    z1, t1 = _rows(V, 4)
    z = np.broadcast_to(z1, (n, V))
    t = np.broadcast_to(t1, (n, V))
    u = np.random.default_rng(int(beta * 10) + int(T * 100)).random(n)
    tok, gap = oracle.mixed_sample(z, t, u, beta, T)
    mix = beta * softmax(t1 / T) + (1 - beta) * softmax(z1 / T)
    counts = np.bincount(tok, minlength=V)
    assert counts.sum() == n
    _, pval = chisquare(counts, mix * n)
    assert pval > 1e-4, (counts, mix * n)
    assert np.all(gap >= 0) and np.all(gap <= 1)


def test_beta_one_is_the_verify_bonus_draw():
    B, k, V = 300, 2, 9
    rng = np.random.default_rng(8)
    t = rng.normal(0, 1.5, (B, k + 1, V))
    z = t[:, :k].copy()  # draft = target: every proposal is accepted (r = 1 > u)
    tokens = rng.integers(0, V, (B, k)).astype(np.int32)
    u = rng.random((B, k + 1))
    ref = oracle.verify(z, t, tokens, u, 0.8)
    assert np.all(ref["accepted"] == k)
    tok, _ = oracle.mixed_sample(rng.normal(size=(B, V)), t[:, k], u[:, k], 1.0, 0.8)
    assert np.array_equal(tok, ref["out_tokens"][:, k])


def test_inverse_cdf_convention():
    # p = q = (1/2, 1/2) exactly: W = 1, C = (1/2, 1); u W on the edge picks the next index
    z = np.zeros((3, 2))
    tok, gap = oracle.mixed_sample(z, z, np.array([0.5, 0.4999, 0.0]), 0.5)
    assert tok.tolist() == [1, 0, 0]
    assert gap[0] == 0.0 and abs(gap[1] - 0.0001) < 1e-12
    # zero-weight entries are never drawn, even at u = 0
    z = np.array([[-np.inf, 0.0, 0.0, -np.inf]])
    tok, _ = oracle.mixed_sample(z, z, np.array([0.0]), 0.3)
    assert tok[0] == 1
    tok, _ = oracle.mixed_sample(z, z, np.array([0.999999]), 0.3)
    assert tok[0] == 2
    # the mixture's weights, written out: p = (3/4, 1/4), q = (1/4, 3/4), beta = 1/4
    t = np.log(np.array([[0.75, 0.25]]))
    z = np.log(np.array([[0.25, 0.75]]))
    w0 = 0.25 * 0.75 + 0.75 * 0.25  # 0.375
    for u, want in ((w0 - 1e-9, 0), (w0 + 1e-9, 1)):
        tok, _ = oracle.mixed_sample(z, t, np.array([u]), 0.25)
        assert tok[0] == want, (u, tok)


def test_bad_arguments():
    z = np.zeros((1, 3))
    with pytest.raises(ValueError):
        oracle.mixed_sample(z, z, np.array([0.5]), 1.5)
    with pytest.raises(ValueError):
        oracle.mixed_sample(z, z, np.array([0.5]), 0.5, 0.0)
