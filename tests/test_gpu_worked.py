"""The CUDA path, through the C ABI, against the hand-worked fixtures of
tests/golden/: every verify, mixed-sampling and token-tree case gives the
hand-derived decisions and tokens exactly (fp32 logits ln(w) of small integer
weights; each case's uniforms sit well clear of its ratios and CDF steps)."""
import numpy as np
import pytest
import torch

from tests import worked as W

pytestmark = pytest.mark.gpu
VERIFY = W.verify_cases()
MIXED = W.mixed_cases()
TREE = W.tree_cases()


@pytest.fixture(scope="module")
def osd():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA GPU")
    import paper_2310_07177_gb300 as pkg
    pkg.build_library()
    pkg.load_library()
    return pkg


def _dev(a, dtype=None):
    t = torch.as_tensor(np.ascontiguousarray(a))
    return (t if dtype is None else t.to(dtype)).cuda()


def test_verify_worked_batched(osd):
    # all cases of one temperature as one batch, so that the sequences of a launch differ
    for T in sorted({c[1] for c in VERIFY}):
        cases = [c for c in VERIFY if c[1] == T]
        B = len(cases)
        z = np.broadcast_to(W.logits(W.VERIFY_DRAFT_W), (B, 2, 4))
        t = np.broadcast_to(W.logits(W.VERIFY_TARGET_W), (B, 3, 4))
        y = np.array([c[2] for c in cases], np.int32)
        u = np.array([c[3] for c in cases], np.float32)
        res = osd.osd_verify(_dev(z) if T > 0 else None, _dev(t), _dev(y), _dev(u) if T > 0 else None, T)
        torch.cuda.synchronize()
        for b, (name, _, _, _, acc, out) in enumerate(cases):
            assert int(res.accepted[b]) == acc, name
            assert res.out_tokens[b].tolist() == out, name
            assert res.mismatch_mask[b].tolist() == [1 if (acc < 2 and i == acc) else 0 for i in range(2)], name


def test_mixed_worked_batched(osd):
    for (T, beta) in sorted({(c[1], c[2]) for c in MIXED}):
        cases = [c for c in MIXED if (c[1], c[2]) == (T, beta)]
        N = len(cases)
        z = np.broadcast_to(W.logits(W.MIXED_DRAFT_W), (N, 4))
        t = np.broadcast_to(W.logits(W.MIXED_TARGET_W), (N, 4))
        u = np.array([c[3] for c in cases], np.float32)
        tok, _ = osd.osd_mixed_sample(_dev(z), _dev(t), _dev(u), beta, temperature=T)
        torch.cuda.synchronize()
        assert tok.tolist() == [c[4] for c in cases], (T, beta)


@pytest.mark.parametrize("case", TREE, ids=[c[0] for c in TREE])
def test_tree_worked(osd, case):
    name, parent, dw, tw, T, tokens, u, acc, path, out, last = case
    res = osd.osd_verify_tree(_dev(W.logits(dw)[None]) if T > 0 else None, _dev(W.logits(tw)[None]), parent,
                              _dev(np.array([tokens], np.int32)), _dev(np.array([u], np.float32)) if T > 0 else None,
                              T)
    torch.cuda.synchronize()
    assert int(res.accepted[0]) == acc and res.path[0].tolist() == path, name
    assert res.out_tokens[0].tolist() == out and int(res.last_node[0]) == last, name
