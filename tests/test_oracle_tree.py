"""Pins for the token-tree (multi-candidate) verification oracle against facts
fixed outside it:

* a chain tree (one child per node) is ordinary speculative sampling: the
  result equals the verify oracle's token for token, with the uniforms mapped
  (node i's test is the verify test of position i - 1, the root's uniform is
  the extra draw);
* the emitted token at the root follows the target distribution p exactly when
  the root's candidates are independent draws from q (the property that
  multi-candidate speculative sampling keeps), by chi-square over 2e5 trees,
  with two and with four candidates, duplicates allowed, at T = 1 and T = 0.6;
* the second emitted token follows p at the accepted child (chi-square, every
  child's target row distinct);
* p == q at the root: its first child is always accepted;
* T = 0: the first child equal to argmax p is taken (numpy argmax), else the
  extra token is argmax p;
* bad tokens and malformed trees are rejected.
"""
import numpy as np
import pytest
from scipy.special import softmax
from scipy.stats import chisquare

import oracle

pytestmark = pytest.mark.filterwarnings("ignore::RuntimeWarning")


def _chain(k):
    return np.array([-1] + list(range(k)), np.int32)


def test_chain_tree_is_speculative_sampling():
    B, k, V, T = 400, 4, 9, 0.8
    rng = np.random.default_rng(3)
    z = rng.normal(0, 1.5, (B, k, V))
    t = z[:, :, :] * 0.7 + rng.normal(0, 1.0, (B, k, V))
    t = np.concatenate([t, rng.normal(0, 1.5, (B, 1, V))], axis=1)  # [B, k+1, V]
    y = np.empty((B, k), np.int32)
    for b in range(B):
        for i in range(k):
            y[b, i] = rng.choice(V, p=softmax(z[b, i] / T))
    u = rng.random((B, k + 1))
    ref = oracle.verify(z, t, y, u, T)
    # the same step as a chain tree of k + 1 nodes
    zt = np.concatenate([z, np.zeros((B, 1, V))], axis=1)
    yt = np.concatenate([np.zeros((B, 1), np.int32), y], axis=1)
    ut = np.concatenate([u[:, k:], u[:, :k]], axis=1)
    res = oracle.verify_tree(zt, t, _chain(k), yt, ut, T)
    assert np.array_equal(res["accepted"], ref["accepted"])
    assert np.array_equal(res["out_tokens"], ref["out_tokens"])
    # the ratio is exp(lp - lq) there and exp(lp) / exp(lq) here: equal up to rounding
    np.testing.assert_allclose(res["margin"][:, 1:], ref["margin"], rtol=1e-12, atol=1e-14)
    np.testing.assert_allclose(res["cdf_gap"], ref["cdf_gap"], rtol=1e-9, atol=1e-14)
    a = ref["accepted"]
    assert np.all(res["last_node"] == a)
    for b in range(B):
        assert res["path"][b, :a[b]].tolist() == list(range(1, a[b] + 1))


def _star(m):
    return np.array([-1] + [0] * m, np.int32)


@pytest.mark.parametrize("m,T", [(2, 1.0), (4, 1.0), (4, 0.6)])
def test_root_token_follows_the_target(m, T):
    V, n = 5, 200_000
    rng = np.random.default_rng(m * 10 + int(T * 10))
    z1 = rng.normal(0, 1.2, V)
    t1 = rng.normal(0, 1.2, V)
    q = softmax(z1 / T)
    p = softmax(t1 / T)
    nodes = m + 1
    z = np.broadcast_to(z1, (n, nodes, V))
    t = np.broadcast_to(t1, (n, nodes, V))
    y = np.zeros((n, nodes), np.int32)
    y[:, 1:] = rng.choice(V, size=(n, m), p=q)  # independent candidates, duplicates allowed
    u = rng.random((n, nodes))
    res = oracle.verify_tree(z, t, _star(m), y, u, T)
    first = res["out_tokens"][:, 0]
    counts = np.bincount(first, minlength=V)
    _, pval = chisquare(counts, p * n)
    assert pval > 1e-4, (counts, p * n)
    # more candidates accept more often than one would: 1 - P(all rejected)
    assert np.mean(res["accepted"] == 1) > np.minimum(p, q).sum() - 0.01


def test_second_token_follows_the_target_at_the_accepted_child():
    V, n, m, T = 4, 200_000, 3, 1.0
    rng = np.random.default_rng(17)
    nodes = m + 1
    z1 = rng.normal(0, 1.0, V)
    q = softmax(z1)
    trows = rng.normal(0, 1.5, (nodes, V))  # a different p after every child
    z = np.broadcast_to(z1, (n, nodes, V))
    t = np.broadcast_to(trows, (n, nodes, V))
    y = np.zeros((n, nodes), np.int32)
    y[:, 1:] = rng.choice(V, size=(n, m), p=q)
    u = rng.random((n, nodes))
    res = oracle.verify_tree(z, t, _star(m), y, u, T)
    took = res["accepted"] == 1
    for c in range(1, nodes):
        sel = took & (res["last_node"] == c)
        counts = np.bincount(res["out_tokens"][sel, 1], minlength=V)
        exp = softmax(trows[c]) * sel.sum()
        _, pval = chisquare(counts, exp)
        assert pval > 1e-4, (c, counts, exp)


def test_equal_distributions_accept_the_first_child():
    B, V = 50, 7
    rng = np.random.default_rng(2)
    z = rng.normal(size=(B, 4, V))
    par = np.array([-1, 0, 0, 1], np.int32)
    y = rng.integers(0, V, (B, 4)).astype(np.int32)
    res = oracle.verify_tree(z, z, par, y, rng.random((B, 4)) * 0.999, 1.0)
    assert np.all(res["path"][:, 0] == 1)
    assert np.all(res["accepted"] == 2) and np.all(res["path"][:, 1] == 3)


def test_greedy_takes_the_first_child_equal_to_the_argmax():
    V = 6
    par = np.array([-1, 0, 0, 0, 2], np.int32)
    t = np.zeros((1, 5, V))
    t[0, 0] = [0, 1, 3, 2, 3, 0]    # argmax 2 (first of the two maxima)
    t[0, 2] = [5, 0, 0, 0, 0, 0]    # argmax 0
    t[0, 4] = [0, 0, 0, 0, 0, 9]    # argmax 5
    y = np.array([[0, 4, 2, 2, 1]], np.int32)
    res = oracle.verify_tree(np.zeros_like(t), t, par, y, np.zeros((1, 5)), 0.0)
    assert res["path"][0].tolist() == [2, -1, -1, -1, -1]  # node 2 (token 2) wins over node 3
    assert res["out_tokens"][0].tolist() == [2, 0, -1, -1, -1]  # node 4 (token 1) != argmax 0
    assert res["accepted"][0] == 1 and res["last_node"][0] == 2
    assert np.all(np.isnan(res["margin"])) and np.isnan(res["cdf_gap"][0])


def test_bad_tokens_and_malformed_trees():
    V = 4
    par = np.array([-1, 0, 1], np.int32)
    z = np.zeros((2, 3, V))
    y = np.array([[0, 1, 2], [0, 1, V]], np.int32)
    res = oracle.verify_tree(z, z, par, y, np.full((2, 3), 0.5), 1.0)
    assert res["accepted"].tolist()[1] == -1 and np.all(res["out_tokens"][1] == -1)
    assert res["accepted"][0] == 2
    for bad_par in ([0, 0, 1], [-1, 1, 0], [-1, 0, 2]):
        with pytest.raises(ValueError):
            oracle.verify_tree(z, z, np.array(bad_par, np.int32), y[:1].repeat(2, 0), np.full((2, 3), 0.5), 1.0)
