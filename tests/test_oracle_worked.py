"""The oracle against the hand-worked fixtures of tests/golden/ (V = 4 cases
whose probabilities are small-integer ratios): speculative-sampling
verification (Appendix A.1), mixed sampling (Section 4.1) and token-tree
verification, every decision and token fixed by hand arithmetic."""
import numpy as np
import pytest

import oracle
from tests import worked as W

VERIFY = W.verify_cases()
MIXED = W.mixed_cases()
TREE = W.tree_cases()


def test_fixtures_cover_every_outcome():
    assert {c[4] for c in VERIFY} == {0, 1, 2} and {c[1] for c in VERIFY} == {0.0, 0.5, 1.0}
    assert {c[4] for c in MIXED} == {0, 1, 2, 3}
    assert {c[7] for c in TREE} == {0, 1, 2} and {c[4] for c in TREE} == {0.0, 1.0}


@pytest.mark.parametrize("case", VERIFY, ids=[c[0] for c in VERIFY])
def test_verify_worked(case):
    name, T, tokens, u, acc, out = case
    z = W.logits(W.VERIFY_DRAFT_W)[None]
    t = W.logits(W.VERIFY_TARGET_W)[None]
    ref = oracle.verify(z, t, np.array([tokens], np.int32), np.array([u], np.float32), T)
    assert int(ref["accepted"][0]) == acc, name
    assert ref["out_tokens"][0].tolist() == out, name
    mask = [1 if (acc < 2 and i == acc) else 0 for i in range(2)]
    assert ref["mismatch_mask"][0].tolist() == mask, name
    if T > 0:  # no test or draw sits near its boundary
        m = ref["margin"][0]
        assert np.nanmin(m) > 5e-3 and ref["cdf_gap"][0] > 4e-3, (name, m, ref["cdf_gap"])


@pytest.mark.parametrize("case", MIXED, ids=[c[0] for c in MIXED])
def test_mixed_worked(case):
    name, T, beta, u, tok = case
    tokens, gap = oracle.mixed_sample(W.logits(W.MIXED_DRAFT_W)[None], W.logits(W.MIXED_TARGET_W)[None],
                                      np.array([u], np.float32), beta, T)
    assert int(tokens[0]) == tok, name
    assert gap[0] > 4e-3, (name, gap)


@pytest.mark.parametrize("case", TREE, ids=[c[0] for c in TREE])
def test_tree_worked(case):
    name, parent, dw, tw, T, tokens, u, acc, path, out, last = case
    ref = oracle.verify_tree(W.logits(dw)[None], W.logits(tw)[None], np.array(parent, np.int32),
                             np.array([tokens], np.int32), np.array([u], np.float32), T)
    assert int(ref["accepted"][0]) == acc, name
    assert ref["path"][0].tolist() == path, name
    assert ref["out_tokens"][0].tolist() == out, name
    assert int(ref["last_node"][0]) == last, name
    if T > 0:
        m = ref["margin"][0]
        assert np.nanmin(m) > 5e-3, (name, m)
