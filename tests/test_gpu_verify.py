"""GPU parity of osd_verify (C ABI through the Python binding) against the
oracle, plus a chi-square test of the GPU path's output distribution."""
import math

import numpy as np
import pytest
import torch
from scipy.special import softmax
from scipy.stats import chisquare

import oracle
from paper_2310_07177_gb300 import workloads as W
from tests.parity import check_margins, check_verify

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def osd():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA GPU")
    import paper_2310_07177_gb300 as pkg
    pkg.build_library()
    pkg.load_library()
    return pkg


def _t32(T):
    return float(np.float32(T))


def _run(osd, inp, T, greedy_tokens=False):
    dev = torch.device("cuda")
    z = inp["draft"].to(dev)
    t = inp["target"].to(dev)
    y = (inp["greedy_tokens"] if greedy_tokens else inp["tokens"]).to(dev)
    u = inp["uniforms"].to(dev)
    res = osd.osd_verify(z, t, y, u, T)
    torch.cuda.synchronize()
    ref = oracle.verify(inp["draft"], inp["target"], y.cpu(), inp["uniforms"], _t32(T))
    return res, ref


CASES = [  # (B, k, V, dtype, T)
    (3, 1, 1, torch.float32, 1.0),
    (5, 2, 7, torch.bfloat16, 1.0),
    (4, 3, 100, torch.float32, 0.7),
    (6, 4, 4097, torch.bfloat16, 1.0),
    (2, 5, 8193, torch.float32, 1.3),
    (4, 4, 33001, torch.bfloat16, 0.7),
    (3, 6, 32000, torch.bfloat16, 1.0),
    (8, 2, 65539, torch.float32, 1.0),
    (512, 4, 16, torch.bfloat16, 1.0),       # many sequences over a tiny vocabulary
    (1024, 8, 64, torch.float32, 0.7),
    (16, 64, 300, torch.bfloat16, 1.0),      # the largest k
    (160, 2, 20000, torch.bfloat16, 1.0),    # past 128 sequences: 4 finalize CTAs per sequence
    (130, 3, 40961, torch.float32, 0.7),     # the same, element-wise path
    (2, 3, 1 << 21, torch.bfloat16, 1.0),    # the largest vocabulary
    # past 128 sequences the finalize takes clusters of at most 4 CTAs
    (129, 1, 4096, torch.float32, 1.0),
    (200, 3, 8264, torch.bfloat16, 1.0),
    (300, 2, 16384, torch.float32, 0.7),     # exactly one slice
    (150, 4, 49160, torch.bfloat16, 1.3),    # a ragged last slice
    (140, 2, 16392, torch.bfloat16, 0.7),    # a last slice of one 8-entry vector
    # a single sequence: one cluster (the one-launch path where the rows are 16-byte aligned)
    (1, 1, 1, torch.float32, 1.0),
    (1, 5, 7, torch.bfloat16, 0.7),
    (1, 5, 32000, torch.bfloat16, 1.0),
    (1, 8, 128256, torch.bfloat16, 0.7),
    (1, 3, 32000, torch.float32, 1.3),
]


@pytest.mark.parametrize("B,k,V,dtype,T", CASES)
def test_verify_matches_oracle(osd, B, k, V, dtype, T):
    spec = W.VerifySpec(B, k, V, dtype, 2.0, 0.8, 1.2, T)
    inp = W.verify_inputs(spec, seed=1234 + V + k)
    res, ref = _run(osd, inp, T)
    rep = check_verify(res, ref, k, V)
    check_margins(res, ref)
    print(f"B={B} k={k} V={V} {dtype} T={T}: {rep}")


GREEDY_CASES = [
    (16, 3, 1, torch.float32), (32, 4, 1001, torch.bfloat16), (9, 2, 40000, torch.float32),
    (12, 5, 32000, torch.bfloat16), (38, 7, 32768, torch.bfloat16), (7, 3, 4096, torch.bfloat16),
    (5, 1, 40, torch.float32), (20, 5, 16000, torch.float32), (39, 7, 32768, torch.bfloat16),
    (4, 8, 32000, torch.bfloat16), (1, 5, 32000, torch.bfloat16), (1, 1, 1, torch.float32),
]


@pytest.mark.parametrize("B,k,V,dtype", GREEDY_CASES)
def test_greedy_matches_oracle(osd, B, k, V, dtype):
    spec = W.VerifySpec(B, k, V, dtype, 2.0, 1.0, 0.3, 0.0)
    inp = W.verify_inputs(spec, seed=99 + V)
    # round logits to a coarse grid so argmax ties occur
    for key in ("draft", "target"):
        inp[key] = (inp[key].float() * 2).round().div(2).to(dtype)
    inp["greedy_tokens"] = torch.argmax(inp["draft"].float(), -1).to(torch.int32)
    res, ref = _run(osd, inp, 0.0, greedy_tokens=True)
    np.testing.assert_array_equal(res.accepted.cpu().numpy(), ref["accepted"])
    np.testing.assert_array_equal(res.out_tokens.cpu().numpy(), ref["out_tokens"])
    np.testing.assert_array_equal(res.mismatch_mask.cpu().numpy(), ref["mismatch_mask"])
    assert torch.isnan(res.diag_margin).all() and torch.isnan(res.diag_cdf_gap).all()
    # greedy needs neither draft logits nor uniforms
    dev = torch.device("cuda")
    res2 = osd.osd_verify(None, inp["target"].to(dev), inp["greedy_tokens"].to(dev), None, 0.0)
    assert torch.equal(res2.out_tokens, res.out_tokens)
    # draft tokens outside [0, V) mark their sequence bad; the others are unaffected
    if B >= 3:
        bad = inp["greedy_tokens"].clone()
        bad[1, 0] = V
        bad[2, k - 1] = -1
        res3 = osd.osd_verify(None, inp["target"].to(dev), bad.to(dev), None, 0.0)
        torch.cuda.synchronize()
        ref3 = oracle.verify(inp["draft"], inp["target"], bad, inp["uniforms"], 0.0)
        np.testing.assert_array_equal(res3.accepted.cpu().numpy(), ref3["accepted"])
        np.testing.assert_array_equal(res3.out_tokens.cpu().numpy(), ref3["out_tokens"])
        np.testing.assert_array_equal(res3.mismatch_mask.cpu().numpy(), ref3["mismatch_mask"])
        assert res3.accepted[1].item() == -1 and res3.accepted[2].item() == -1


@pytest.mark.parametrize("B,V", [(16, 5000), (160, 8192)])
def test_identical_logits_accept_all(osd, B, V):
    spec = W.VerifySpec(B, 5, V, torch.bfloat16, 2.0, 1.0, 0.0, 1.0)
    inp = W.verify_inputs(spec, seed=5)
    inp["target"] = torch.cat([inp["draft"], inp["target"][:, -1:]], dim=1).contiguous()
    res, ref = _run(osd, inp, 1.0)
    assert (res.accepted.cpu() == 5).all()
    check_verify(res, ref, 5, V)


def test_extreme_and_neg_inf_logits(osd):
    B, k, V = 6, 3, 2000
    g = torch.Generator().manual_seed(7)
    z = torch.randn(B, k, V, generator=g) * 3
    t = torch.randn(B, k + 1, V, generator=g) * 3
    z[0, 0, :] = -1e4
    z[0, 0, 5] = 1e4
    t[1, :, 100:] = float("-inf")
    z[2, 1, :50] = float("-inf")
    t[3, 0, :] = torch.linspace(-1e4, 1e4, V)
    y = torch.randint(0, 100, (B, k), generator=g).to(torch.int32)
    y[0, 0] = 5
    inp = {"draft": z, "target": t, "tokens": y, "uniforms": torch.rand(B, k + 1, generator=g)}
    res, ref = _run(osd, inp, 1.0)
    check_verify(res, ref, k, V)


def test_bad_tokens_and_empty_batch(osd):
    spec = W.VerifySpec(5, 3, 300, torch.float32, 2.0, 1.0, 1.0, 1.0)
    inp = W.verify_inputs(spec, seed=8)
    inp["tokens"][1, 2] = 300
    inp["tokens"][3, 0] = -5
    res, ref = _run(osd, inp, 1.0)
    check_verify(res, ref, 3, 300)
    assert res.accepted[1].item() == -1 and res.accepted[3].item() == -1
    dev = torch.device("cuda")
    e = osd.osd_verify(torch.empty(0, 3, 10, device=dev), torch.empty(0, 4, 10, device=dev),
                       torch.empty(0, 3, dtype=torch.int32, device=dev),
                       torch.empty(0, 4, device=dev), 1.0)
    assert e.accepted.numel() == 0


def test_invalid_arguments_are_rejected(osd):
    import ctypes
    lib = osd.load_library()
    n = ctypes.c_size_t(0)
    assert lib.osd_verify_workspace_size(4, 0, 100, ctypes.byref(n)) == osd.OSD_ERR_INVALID_ARG
    assert lib.osd_verify_workspace_size(4, 65, 100, ctypes.byref(n)) == osd.OSD_ERR_UNSUPPORTED
    assert lib.osd_verify_workspace_size(4, 2, (1 << 21) + 1, ctypes.byref(n)) == osd.OSD_ERR_UNSUPPORTED
    dev = torch.device("cuda")
    z = torch.zeros(2, 2, 16, device=dev)
    t = torch.zeros(2, 3, 16, device=dev)
    y = torch.zeros(2, 2, dtype=torch.int32, device=dev)
    u = torch.zeros(2, 3, device=dev)
    for T in (-1.0, float("nan"), float("inf")):
        with pytest.raises(osd.OsdError) as ei:
            osd.osd_verify(z, t, y, u, T)
        assert ei.value.status == osd.OSD_ERR_INVALID_ARG
    small = torch.empty(8, dtype=torch.uint8, device=dev)
    with pytest.raises(osd.OsdError):
        osd.osd_verify(z, t, y, u, 1.0, workspace=small)


def _mc(osd, z1, t1, T, n, seed):
    k, V = z1.shape
    rng = np.random.default_rng(seed)
    q = softmax(z1 / T, axis=1)
    y = np.empty((n, k), np.int32)
    for i in range(k):
        c = np.cumsum(q[i]); c[-1] = 1.0
        y[:, i] = np.searchsorted(c, rng.random(n), side="right")
    dev = torch.device("cuda")
    zt = torch.tensor(z1, dtype=torch.float32, device=dev).expand(n, k, V).contiguous()
    tt = torch.tensor(t1, dtype=torch.float32, device=dev).expand(n, k + 1, V).contiguous()
    u = torch.tensor(rng.random((n, k + 1)), dtype=torch.float32, device=dev)
    res = osd.osd_verify(zt, tt, torch.tensor(y, device=dev), u, T, diagnostics=False)
    return res.accepted.cpu().numpy(), res.out_tokens.cpu().numpy()


@pytest.mark.parametrize("T,V,k", [(1.0, 5, 3), (0.6, 8, 2)])
def test_gpu_output_distribution_equals_target(osd, T, V, k):
    """Section 3: the emitted tokens follow p exactly; chi-square over 10^6 sequences."""
    rng = np.random.default_rng(4000 + V)
    z1 = rng.normal(0, 1.5, (k, V))
    t1 = rng.normal(0, 1.5, (k + 1, V))
    a, out = _mc(osd, z1, t1, T, 1_000_000, seed=4100 + V)
    p = softmax(t1 / T, axis=1)
    q = softmax(z1 / T, axis=1)
    for i in range(k + 1):
        tok = out[a >= i, i]
        obs = np.bincount(tok, minlength=V)
        pv = chisquare(obs, p[i] * tok.size).pvalue
        assert pv > 1e-3, (i, pv)
    for i in range(k):
        reach, acc = np.sum(a >= i), np.sum(a >= i + 1)
        alpha = np.minimum(p[i], q[i]).sum()
        assert abs(acc / reach - alpha) < 5 * math.sqrt(alpha * (1 - alpha) / reach)


def test_gpu_output_distribution_large_batch(osd):
    """Section 3 at a large batch: 2 x 10^5 sequences at V = 4096, k = 1; the
    first emitted token follows p_0.  The vocabulary is binned into 8 hot
    entries and 16 ranges of the rest."""
    rng = np.random.default_rng(4321)
    V, k, n = 4096, 1, 200_000
    z1 = rng.normal(0, 1.0, (k, V))
    t1 = rng.normal(0, 1.0, (k + 1, V))
    hot = rng.choice(V, 8, replace=False)
    t1[0, hot] += 5.0
    z1[0, hot[:4]] += 5.5      # the draft favours half of them, the residual the other half
    a, out = _mc(osd, z1, t1, 1.0, n, seed=4322)
    p0 = softmax(t1[0])
    bins = np.full(V, -1)
    bins[hot] = np.arange(8)
    rest = np.setdiff1d(np.arange(V), hot)
    bins[rest] = 8 + np.arange(rest.size) * 16 // rest.size
    obs = np.bincount(bins[out[:, 0]], minlength=24)
    exp = np.bincount(bins, weights=p0, minlength=24) * n
    assert chisquare(obs, exp).pvalue > 1e-3
    # the acceptance rate at position 0 is sum min(p, q)
    q0 = softmax(z1[0])
    alpha = np.minimum(p0, q0).sum()
    acc = (a >= 1).mean()
    assert abs(acc - alpha) < 5 * math.sqrt(alpha * (1 - alpha) / n), (acc, alpha)


@pytest.mark.parametrize("B,V,dtype", [(64, 1000, torch.float32), (64, 32000, torch.bfloat16),
                                       (64, 4099, torch.bfloat16), (160, 32000, torch.bfloat16),
                                       (136, 20000, torch.float32)])
def test_extreme_uniforms(osd, B, V, dtype):
    """The extra-token draw at u = 0 (the first positive weight) and at the largest float
    below 1 (tau next to W), and accept tests at both ends, against the oracle."""
    spec = W.VerifySpec(B, 3, V, dtype, 2.0, 0.8, 1.2, 1.0)
    inp = W.verify_inputs(spec, seed=500 + V)
    u = inp["uniforms"]
    below_one = float(np.nextafter(np.float32(1.0), np.float32(0.0)))
    u[0::2, :] = 0.0
    u[1::2, -1] = below_one
    u[1::4, :-1] = below_one
    res, ref = _run(osd, inp, 1.0)
    check_verify(res, ref, spec.k, V)
    check_margins(res, ref)


def test_gpu_expected_length_eq1(osd):
    """Eq. 1 on the GPU's own decisions: the same (p, q) at every position gives
    E[a + 1] = (1 - alpha^(k+1)) / (1 - alpha), alpha = sum min(p, q)."""
    rng = np.random.default_rng(88)
    V, k = 6, 4
    zrow = rng.normal(0, 1.0, V)
    trow = rng.normal(0, 1.0, V)
    a, _ = _mc(osd, np.tile(zrow, (k, 1)), np.tile(trow, (k + 1, 1)), 1.0, 1_000_000, seed=89)
    alpha = np.minimum(softmax(trow), softmax(zrow)).sum()
    want = (1 - alpha ** (k + 1)) / (1 - alpha)
    L = a + 1.0
    assert abs(L.mean() - want) < 5 * L.std() / math.sqrt(len(L)), (L.mean(), want)


# ----------------------------------------------------------------- full-size workloads
@pytest.mark.parametrize("cfg", [1, 2])
def test_workload_small_configs_full(osd, cfg):
    spec = W.VERIFY[cfg]
    inp = W.verify_inputs(spec, seed=W.seed_for(cfg))
    res, ref = _run(osd, inp, spec.temperature)
    rep = check_verify(res, ref, spec.k, spec.V)
    check_margins(res, ref)
    print(f"config {cfg}: {rep}, alpha={np.mean(ref['accepted']) / spec.k:.3f}")
    if cfg == 2:  # greedy pass on the same logits with argmax proposals
        res0, ref0 = _run(osd, inp, 0.0, greedy_tokens=True)
        np.testing.assert_array_equal(res0.out_tokens.cpu().numpy(), ref0["out_tokens"])
        np.testing.assert_array_equal(res0.accepted.cpu().numpy(), ref0["accepted"])


def test_unaligned_largest_vocabulary_past_128_sequences(osd):
    """The element-wise finalize (rows off the 16-byte path) at B > 128 and a
    vocabulary near the limit: its spans need more than four CTAs a sequence."""
    V = (1 << 21) - 1  # odd: bf16 rows are not 16-byte multiples
    spec = W.VerifySpec(130, 1, V, torch.bfloat16, 2.0, 1.0, 1.0, 1.0)
    inp = W.verify_inputs(spec, seed=2121, device="cuda")
    res = osd.osd_verify(inp["draft"], inp["target"], inp["tokens"], inp["uniforms"], 1.0)
    torch.cuda.synchronize()
    idx = torch.arange(0, 130, 26)
    ref = oracle.verify(inp["draft"][idx].cpu(), inp["target"][idx].cpu(), inp["tokens"][idx].cpu(),
                        inp["uniforms"][idx].cpu(), 1.0)

    class Sub:
        pass
    sub = Sub()
    for f in ("accepted", "out_tokens", "mismatch_mask", "diag_margin", "diag_cdf_gap"):
        setattr(sub, f, getattr(res, f)[idx.to(res.accepted.device)])
    check_verify(sub, ref, spec.k, V)
    acc = res.accepted.cpu()
    assert ((acc >= 0) & (acc <= 1)).all()
    out = res.out_tokens.cpu()
    assert ((out[torch.arange(130), acc.long()] >= 0) & (out[torch.arange(130), acc.long()] < V)).all()
