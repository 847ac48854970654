"""The comparison rules of tests/parity.py, on the CPU: TVD's near-tie rows
accept exactly the subgradients of the signs chosen at entries fp32 cannot
order (reading 9), and nothing else."""
import numpy as np

import oracle
from tests.parity import grad_rows, tvd_subgradient, tvd_ties


def _tied_rows(seed=0, V=50):
    # q and p agree on entries 0..4 up to a relative 3e-7: fp64 orders them, fp32 cannot
    rng = np.random.default_rng(seed)
    q = rng.random((3, V))
    q /= q.sum(1, keepdims=True)
    p = q.copy()
    r = rng.random((3, V - 5))
    p[:, 5:] = r / r.sum(1, keepdims=True) * (1 - q[:, :5].sum(1, keepdims=True))
    p[:, 0] *= 1 + 3e-7
    q[:, 1] *= 1 - 2e-7
    return np.log(q), np.log(p)


def test_tvd_other_sign_choice_is_a_near_tie_not_an_error():
    z, t = _tied_rows()
    _, gr = oracle.distill(z, t, None, "tvd", 0.5)
    ties = tvd_ties(z, t, 1.0)
    assert (ties.amb.sum(1) == 5).all()
    flipped = np.where(ties.amb, -np.sign(ties.d) + (ties.d == 0), np.sign(ties.d))
    alt = tvd_subgradient(ties.q, flipped, 1.0)
    res = grad_rows(alt, gr, ties)
    assert res["ok"].all() and res["near_tie"].all() and res["near_tie_differ"].all()
    same = grad_rows(gr.copy(), gr, ties)
    assert same["ok"].all() and not same["near_tie_differ"].any()


def test_tvd_near_tie_rows_still_catch_errors():
    z, t = _tied_rows(1)
    _, gr = oracle.distill(z, t, None, "tvd", 0.5)
    ties = tvd_ties(z, t, 1.0)
    alt = tvd_subgradient(ties.q, np.where(ties.amb, 1.0, np.sign(ties.d)), 1.0)
    bad = alt.copy()
    bad[0, 20] += 1e-2 * np.abs(gr[0]).max()   # off a tie: must fail
    assert list(grad_rows(bad, gr, ties)["ok"]) == [False, True, True]
    worse = gr.copy()
    worse[1] *= 1.01                            # a wrong scale on a near-tie row: must fail
    assert list(grad_rows(worse, gr, ties)["ok"]) == [True, False, True]


def test_tvd_subgradient_matches_the_oracle_away_from_ties():
    rng = np.random.default_rng(3)
    z, t = rng.normal(0, 2, (4, 40)), rng.normal(0, 2, (4, 40))
    for tau in (1.0, 0.7):
        _, gr = oracle.distill(z, t, None, "tvd", 0.5, temperature=tau)
        ties = tvd_ties(z, t, tau)
        assert not ties.amb.any()
        np.testing.assert_allclose(tvd_subgradient(ties.q, np.sign(ties.d), tau), gr, rtol=1e-9, atol=1e-15)
