"""GPU parity of osd_verify_tree (multi-candidate verification over a token
tree) against the oracle: chain, star and Medusa-style trees, both dtypes,
aligned and unaligned vocabularies, T > 0 and greedy; decisions bit-exact
outside near-ties; the GPU's own root tokens pass a chi-square test against
the target distribution."""
import numpy as np
import pytest
import torch
from scipy.special import softmax
from scipy.stats import chisquare

import oracle
from paper_2310_07177_gb300 import workloads as W

pytestmark = pytest.mark.gpu
TIE = 1e-6

TREES = {
    "chain5": [-1, 0, 1, 2, 3, 4],
    "star4": [-1, 0, 0, 0, 0],
    "medusa27": W.MEDUSA_TREE,
}


@pytest.fixture(scope="module")
def osd():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA GPU")
    import paper_2310_07177_gb300 as pkg
    pkg.build_library()
    pkg.load_library()
    return pkg


def _near_tie(ref):
    """Sequences whose oracle decisions sit within 1e-6 of a flip."""
    m = np.nan_to_num(ref["margin"], nan=np.inf).min(axis=1)
    g = np.nan_to_num(ref["cdf_gap"], nan=np.inf)
    return (m < TIE) | (g < TIE)


def _check(osd, inp, T):
    dev = torch.device("cuda")
    T32 = float(np.float32(T))
    z = inp["draft"].to(dev) if T > 0 else None
    u = inp["uniforms"].to(dev) if T > 0 else None
    res = osd.osd_verify_tree(z, inp["target"].to(dev), inp["parent"], inp["tokens"].to(dev), u, T)
    torch.cuda.synchronize()
    ref = oracle.verify_tree(inp["draft"], inp["target"], np.array(inp["parent"], np.int32), inp["tokens"],
                             inp["uniforms"], T32)
    flag = _near_tie(ref) if T > 0 else np.zeros(len(ref["accepted"]), bool)
    ok = ~flag
    for key in ("accepted", "path", "out_tokens", "last_node"):
        got = getattr(res, key).cpu().numpy()
        bad = np.nonzero(ok & np.any((got != ref[key]).reshape(len(got), -1), axis=1))[0]
        assert bad.size == 0, f"{key} differs at {bad[:6]}: gpu {got[bad[:3]]} oracle {ref[key][bad[:3]]}"
    if T > 0:
        gm = res.diag_margin.cpu().numpy()
        rm = ref["margin"]
        both = ok[:, None] & ~np.isnan(rm)
        assert np.all(~np.isnan(gm[both]))
        assert np.max(np.abs(gm[both] - rm[both]), initial=0.0) < 5e-6
        # every flagged sequence still produced a valid outcome
        acc = res.accepted.cpu().numpy()
        out = res.out_tokens.cpu().numpy()
        V = inp["target"].shape[-1]
        for b in np.nonzero(flag)[0]:
            assert 0 <= acc[b] < len(inp["parent"]) and 0 <= out[b, acc[b]] < V
    return int(flag.sum())


CASES = [  # (tree, B, V, dtype, T)
    ("chain5", 16, 7, torch.float32, 1.0),
    ("star4", 32, 100, torch.bfloat16, 1.0),
    ("medusa27", 8, 4097, torch.float32, 0.7),
    ("medusa27", 12, 32000, torch.bfloat16, 1.0),
    ("star4", 6, 33001, torch.bfloat16, 1.3),
    ("chain5", 4, 65539, torch.float32, 1.0),
    ("medusa27", 3, 128256, torch.bfloat16, 1.0),
    ("medusa27", 16, 32000, torch.bfloat16, 0.0),
    ("star4", 24, 101, torch.float32, 0.0),
]


@pytest.mark.parametrize("tree,B,V,dtype,T", CASES)
def test_matches_oracle(osd, tree, B, V, dtype, T):
    # a target close to the draft, so that walks go deep and test many children
    inp = W.tree_inputs(B, TREES[tree], V, dtype, T, seed=B * 1000 + V, target_noise=0.8)
    _check(osd, inp, T)


def test_workload_full_size(osd):
    """The benchmark's tree workload exactly as it launches it: B=32 sequences over the
    27-node tree, V=32000 bf16, T=1, every sequence checked against the oracle."""
    inp = W.tree_inputs(32, W.MEDUSA_TREE, 32000, torch.bfloat16, 1.0, seed=2310071778, target_noise=0.8)
    ties = _check(osd, inp, 1.0)
    print(f"tree workload: {ties} of 32 sequences near a tie")


@pytest.mark.parametrize("extreme", ["zero", "below_one"])
def test_extreme_uniforms(osd, extreme):
    """Every uniform at 0, or at the largest float below 1: the tree's draws at the ends
    of the CDF, against the oracle."""
    inp = W.tree_inputs(16, W.MEDUSA_TREE, 5000, torch.bfloat16, 1.0, seed=77, target_noise=0.8)
    val = 0.0 if extreme == "zero" else float(np.nextafter(np.float32(1.0), np.float32(0.0)))
    inp["uniforms"] = torch.full_like(inp["uniforms"], val)
    _check(osd, inp, 1.0)


def test_acceptance_reaches_every_depth(osd):
    """On draft == target logits every first child passes: the walk follows
    first children to a leaf."""
    par = W.MEDUSA_TREE
    inp = W.tree_inputs(8, par, 2000, torch.bfloat16, 1.0, seed=4, target_noise=0.0, target_scale=1.0)
    res = osd.osd_verify_tree(inp["draft"].cuda(), inp["target"].cuda(), par, inp["tokens"].cuda(),
                              inp["uniforms"].cuda() * 0.999, 1.0)
    torch.cuda.synchronize()
    node, depth = 0, 0
    firsts = []
    while True:
        kids = [i for i in range(len(par)) if par[i] == node]
        if not kids:
            break
        node = kids[0]
        firsts.append(node)
    got = res.path.cpu().numpy()
    for b in range(8):
        assert got[b, :len(firsts)].tolist() == firsts
    assert torch.all(res.accepted == len(firsts))


def test_gpu_root_token_follows_the_target(osd):
    V, n, m, T = 8, 200_000, 4, 1.0
    par = [-1] + [0] * m
    g = torch.Generator().manual_seed(12)
    z1 = torch.randn(V, generator=g) * 1.2
    t1 = torch.randn(V, generator=g) * 1.2
    q = softmax(z1.double().numpy())
    rng = np.random.default_rng(5)
    tok = np.zeros((n, m + 1), np.int32)
    tok[:, 1:] = rng.choice(V, size=(n, m), p=q)
    dev = torch.device("cuda")
    z = z1.to(dev).expand(n, m + 1, V).contiguous()
    t = t1.to(dev).expand(n, m + 1, V).contiguous()
    u = torch.from_numpy(rng.random((n, m + 1)).astype(np.float32)).to(dev)
    res = osd.osd_verify_tree(z, t, par, torch.from_numpy(tok).to(dev), u, T, diagnostics=False)
    first = res.out_tokens[:, 0].cpu().numpy()
    counts = np.bincount(first, minlength=V)
    p = softmax(t1.double().numpy())
    _, pval = chisquare(counts, p * n)
    assert pval > 1e-4, (counts, p * n)


def test_empty_batch_and_root_only_tree(osd):
    dev = torch.device("cuda")
    e = torch.empty(0, 3, 16, device=dev)
    res = osd.osd_verify_tree(e, e, [-1, 0, 0], torch.empty(0, 3, dtype=torch.int32, device=dev),
                              torch.empty(0, 3, device=dev), 1.0)
    assert res.accepted.numel() == 0 and res.out_tokens.numel() == 0
    # a tree of the root alone: nothing to test, the extra token is drawn from p at the root
    inp = W.tree_inputs(24, [-1], 700, torch.float32, 1.0, seed=5)
    ties = _check(osd, inp, 1.0)
    assert ties < 24


def test_bad_tokens(osd):
    par = [-1, 0, 0, 1]
    inp = W.tree_inputs(3, par, 50, torch.float32, 1.0, seed=1)
    inp["tokens"][1, 2] = 50
    inp["tokens"][2, 3] = -1
    res = osd.osd_verify_tree(inp["draft"].cuda(), inp["target"].cuda(), par, inp["tokens"].cuda(),
                              inp["uniforms"].cuda(), 1.0)
    torch.cuda.synchronize()
    acc = res.accepted.cpu().numpy()
    assert acc[0] >= 0 and acc[1] == -1 and acc[2] == -1
    assert torch.all(res.out_tokens[1:] == -1) and torch.all(res.path[1:] == -1)
    assert torch.all(res.last_node[1:] == -1)


def test_invalid_arguments_are_rejected(osd):
    dev = torch.device("cuda")
    t = torch.zeros(2, 3, 16, device=dev)
    y = torch.zeros(2, 3, dtype=torch.int32, device=dev)
    u = torch.zeros(2, 3, device=dev)
    with pytest.raises(osd.OsdError) as ei:
        osd.osd_verify_tree(t, t, [-1, 1, 0], y, u, 1.0)
    assert ei.value.status == osd.OSD_ERR_INVALID_ARG
    with pytest.raises(osd.OsdError) as ei:
        osd.osd_verify_tree(t, t, [-1, 0, 0], y, u, -0.5)
    assert ei.value.status == osd.OSD_ERR_INVALID_ARG
    with pytest.raises(ValueError):
        osd.osd_verify_tree(t, t, [-1, 0, 0], y.long(), u, 1.0)
