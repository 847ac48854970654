"""Pins for oracle.distill_rejected, the distillation of the positions that
verification rejected (Algorithm 1), against facts fixed outside it:

* the positions it keeps are exactly the ones the verify oracle's mismatch
  mask marks (the mask is pinned by the verify tests: the first rejected
  position of a sequence, none when every proposal was accepted);
* hand-built accepted counts give the stable partition written out by hand;
* each kept row's loss and gradient are those of the per-position distill
  oracle (pinned by closed forms and finite differences) on that row.
"""
import numpy as np
import pytest

import oracle
from paper_2310_07177_gb300 import workloads as W

pytestmark = pytest.mark.filterwarnings("ignore::RuntimeWarning")


def _case(B, k, V, seed):
    rng = np.random.default_rng(seed)
    z = rng.normal(0, 2, (B, k + 1, V))
    t = z + rng.normal(0, 1.5, (B, k + 1, V))
    draft = np.ascontiguousarray(z[:, :k])
    tokens = np.empty((B, k), np.int32)
    for b in range(B):
        for i in range(k):
            p = np.exp(draft[b, i] - draft[b, i].max())
            tokens[b, i] = rng.choice(V, p=p / p.sum())
    u = rng.random((B, k + 1)).astype(np.float32)
    return draft, t, tokens, u


def test_kept_rows_are_the_mismatch_mask():
    B, k, V = 96, 4, 12
    draft, t, tokens, u = _case(B, k, V, 5)
    res = oracle.verify(draft, t, tokens, u, 1.0)
    acc, mask = res["accepted"], res["mismatch_mask"]
    loss, g, seq, count = oracle.distill_rejected(draft, t, acc, "rkl")
    marked = [b for b in range(B) if mask[b].any()]
    assert list(seq[:count]) == marked
    assert 0 < count < B  # the case exercises both kinds of sequences
    for r, b in enumerate(seq[:count]):
        assert mask[b, acc[b]] == 1 and mask[b].sum() == 1
    # every other sequence accepted all k proposals (no bad tokens here)
    assert all(acc[b] == k for b in seq[count:])


def test_hand_built_partition():
    k, V = 3, 5
    acc = np.array([k, -1, 0, k - 1, 2, k], np.int32)
    B = len(acc)
    rng = np.random.default_rng(1)
    z = rng.normal(size=(B, k, V))
    t = rng.normal(size=(B, k + 1, V))
    loss, g, seq, count = oracle.distill_rejected(z, t, acc, "fkl")
    assert count == 3
    assert list(seq) == [2, 3, 4, 0, 1, 5]
    assert np.all(loss[3:] == 0) and np.all(np.isnan(g[3:]))


@pytest.mark.parametrize("kind", ["fkl", "rkl", "jsd", "tvd", "ce"])
def test_rows_match_the_per_position_oracle(kind):
    B, k, V = 40, 5, 33
    rng = np.random.default_rng(11)
    z = rng.normal(0, 2, (B, k, V))
    t = rng.normal(0, 2, (B, k + 1, V))
    acc = W.accepted_inputs(B, k, seed=3).numpy()
    loss, g, seq, count = oracle.distill_rejected(z, t, acc, kind, 0.3, temperature=0.8)
    for r in range(count):
        b = seq[r]
        l1, g1 = oracle.distill(z[b, acc[b]][None], t[b, acc[b]][None], None, kind, 0.3, temperature=0.8)
        assert loss[r] == l1[0] and np.array_equal(g[r], g1[0])


def test_accepted_generator_covers_every_case():
    a = W.accepted_inputs(4000, 6, seed=9).numpy()
    assert a.min() == -1 and a.max() == 6 and set(np.unique(a)) == set(range(-1, 7))
