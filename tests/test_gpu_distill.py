"""GPU parity of osd_distill (C ABI through the Python binding) against the
oracle, for every loss kind, both dtypes, strided views, masks, ragged and
unaligned vocabularies, and the full-size buffer-flush workloads."""
import numpy as np
import pytest
import torch

import oracle
from paper_2310_07177_gb300 import workloads as W
from tests.parity import check_distill, tvd_ties

pytestmark = pytest.mark.gpu
KINDS = ["fkl", "rkl", "jsd", "tvd", "ce"]


@pytest.fixture(scope="module")
def osd():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA GPU")
    import paper_2310_07177_gb300 as pkg
    pkg.build_library()
    pkg.load_library()
    return pkg


def _tvd_ambiguous(z, t, tau=1.0):
    """The TVD near-tie data of these rows (entries where fp32 cannot order q and p)."""
    V = z.shape[-1]
    return tvd_ties(z.reshape(-1, V).double().numpy(), t.reshape(-1, V).double().numpy(), tau)


def _run(osd, z, t, mask, kind, beta, dev="cuda", tau=1.0):
    zd, td = z.to(dev), t.to(dev)
    md = None if mask is None else mask.to(dev)
    V = z.shape[-1]
    lead = tuple(z.shape[:-1])
    dl = torch.full(lead + (V,), float("nan"), dtype=torch.float32, device=dev)
    loss, g = osd.osd_distill(zd, td, md, kind, beta, dlogits=dl, temperature=tau)
    torch.cuda.synchronize()
    return loss.cpu().numpy().reshape(-1), g.cpu().numpy().reshape(-1, V)


def _oracle(z, t, mask, kind, beta, tau=1.0):
    V = z.shape[-1]
    zc = z.reshape(-1, V)
    tc = t.reshape(-1, V)
    m = None if mask is None else mask.reshape(-1)
    return oracle.distill(zc, tc, m, kind, beta, temperature=float(np.float32(tau)))


SHAPES = [  # (N, V, dtype)
    (3, 1, torch.float32),
    (5, 7, torch.bfloat16),
    (6, 100, torch.float32),
    (4, 8200, torch.bfloat16),
    (3, 32000, torch.bfloat16),
    (2, 32000, torch.float32),
    (3, 33001, torch.bfloat16),
    (2, 32128, torch.float32),
    (2, 128256, torch.bfloat16),   # spans of 16032: 256-thread CTAs for every kind but TVD
    (2, 100000, torch.bfloat16),   # the wide path with 12544-entry spans
    (2, 100003, torch.bfloat16),   # the same length off the 16-byte path: 128-thread CTAs
    (2, 393216, torch.bfloat16),   # the largest vocabulary per dtype: 192 KB of staging per CTA
    (2, 196608, torch.float32),
]


@pytest.mark.parametrize("kind", KINDS)
@pytest.mark.parametrize("N,V,dtype", SHAPES)
def test_distill_matches_oracle(osd, kind, N, V, dtype):
    spec = W.DistillSpec(N, V, dtype, 2.0, "draft+noise", 1.5, 1.0)
    inp = W.distill_inputs(spec, seed=77 + V + N)
    z, t = inp["draft"], inp["target"]
    mask = torch.ones(N, dtype=torch.uint8)
    if N >= 3:
        mask[1] = 0
    beta = 0.3 if kind == "jsd" else 0.5
    for tau in (1.0, 0.7) if V in (100, 33001, 128256) else (1.0,):
        lg, gg = _run(osd, z, t, mask, kind, beta, tau=tau)
        lr, gr = _oracle(z, t, mask, kind, beta, tau=tau)
        skip = _tvd_ambiguous(z, t, tau) if kind == "tvd" else None
        rep = check_distill(lg, gg, lr, gr, mask.numpy() == 1, skip)
        print(f"{kind} N={N} V={V} {dtype} tau={tau}: {rep}")


@pytest.mark.parametrize("kind", KINDS)
def test_strided_target_view(osd, kind):
    """Distill the [B,k] draft rows against target[:, :k] of a [B,k+1,V] tensor (no copy)."""
    spec = W.VerifySpec(3, 4, 5000, torch.bfloat16, 2.0, 1.0, 1.0, 1.0)
    inp = W.verify_inputs(spec, seed=3)
    z, t = inp["draft"], inp["target"]
    dev = torch.device("cuda")
    td = t.to(dev)
    view = td[:, :4, :]
    assert not view.is_contiguous()
    mask = torch.tensor([[1, 0, 1, 1], [0, 0, 1, 0], [1, 1, 1, 1]], dtype=torch.uint8)
    dl = torch.full((3, 4, 5000), float("nan"), device=dev)
    loss, g = osd.osd_distill(z.to(dev), view, mask.to(dev), kind, 0.5, dlogits=dl)
    torch.cuda.synchronize()
    lr, gr = _oracle(z, t[:, :4].contiguous(), mask, kind, 0.5)
    skip = _tvd_ambiguous(z, t[:, :4].contiguous()) if kind == "tvd" else None
    check_distill(loss.cpu().numpy().reshape(-1), g.cpu().numpy().reshape(-1, 5000), lr, gr,
                  mask.numpy().reshape(-1) == 1, skip)


def test_ce_label_ties_take_the_lowest_index(osd):
    """FT (Table 1): the label is the first target maximum, also across CTAs of a cluster."""
    z = torch.randn(3, 40000, generator=torch.Generator().manual_seed(4)).to(torch.bfloat16)
    t = torch.randn(3, 40000, generator=torch.Generator().manual_seed(5)).to(torch.bfloat16)
    t[0, 30000] = t[0, 9000] = t[0, 35000] = 20.0   # tie spanning several CTAs of the row
    t[1, 5] = t[1, 6] = 20.0                        # tie inside one chunk
    t[2, 39999] = 20.0                              # label in the last entry
    lg, gg = _run(osd, z, t, None, "ce", 0.5)
    lr, gr = _oracle(z, t, None, "ce", 0.5)
    check_distill(lg, gg, lr, gr, np.ones(3, bool))
    assert np.argmin(gg[0]) == 9000 and np.argmin(gg[1]) == 5 and np.argmin(gg[2]) == 39999


def test_unaligned_rows(osd):
    """Rows starting off a 16-byte boundary take the element-wise path."""
    base = torch.randn(4 * 1001 + 3, generator=torch.Generator().manual_seed(1)) * 2
    z = base[3:].view(4, 1001)
    t = (z + 0.5 * torch.randn(4, 1001, generator=torch.Generator().manual_seed(2)))
    dev = torch.device("cuda")
    zd = base.to(dev)[3:].view(4, 1001)
    for kind in KINDS:
        dl = torch.full((4, 1001), float("nan"), device=dev)
        loss, g = osd.osd_distill(zd, t.to(dev), None, kind, 0.5, dlogits=dl)
        torch.cuda.synchronize()
        lr, gr = _oracle(z, t, None, kind, 0.5)
        skip = _tvd_ambiguous(z, t) if kind == "tvd" else None
        check_distill(loss.cpu().numpy(), g.cpu().numpy(), lr, gr, np.ones(4, bool), skip)


def test_identical_rows_and_jsd_endpoints(osd):
    dev = torch.device("cuda")
    z = (torch.randn(4, 3000) * 3).to(torch.bfloat16).to(dev)
    for kind in ("fkl", "rkl", "jsd", "tvd"):
        loss, g = osd.osd_distill(z, z, None, kind, 0.5)
        assert loss.abs().max().item() < 1e-6
        assert g.abs().max().item() < 1e-7
    t = (torch.randn(4, 3000) * 3).to(torch.bfloat16).to(dev)
    for beta in (0.0, 1.0):
        loss, g = osd.osd_distill(z, t, None, "jsd", beta)
        assert loss.abs().max().item() == 0.0 and g.abs().max().item() == 0.0


@pytest.mark.parametrize("dtype", [torch.float32, torch.bfloat16])
def test_identical_rows_peaked_and_two_mode(osd, dtype):
    # identical rows where a few entries hold most of the mass: every kind's loss and
    # gradient stay at the parity floor (the oracle gives exactly 0 here)
    g0 = torch.Generator().manual_seed(21)
    z = torch.randn(6, 32000, generator=g0)
    z[0, 7] = 25.0                       # one entry holds almost all the mass
    z[1, 3], z[1, 31000] = 20.0, 20.0    # two equal modes
    z[2, 11], z[2, 12] = 14.0, 13.3      # two unequal modes
    z[3] *= 6.0                          # broad, large logits
    z[4, :16000] = float("-inf")         # half the vocabulary impossible
    z[5] = z[5] * 0.01                   # nearly uniform
    zd = z.to(dtype).cuda()
    for kind in ("fkl", "rkl", "jsd", "tvd", "ce"):
        for beta in ((0.1, 0.5, 0.9) if kind == "jsd" else (0.5,)):
            loss, g = osd.osd_distill(zd, zd, None, kind, beta)
            torch.cuda.synchronize()
            if kind == "ce":  # CE is -log q(argmax t), not a distance: only its gradient's form is checked
                continue
            assert loss.abs().max().item() < 1e-6, (kind, beta, loss)
            assert g.abs().max().item() < 1e-7, (kind, beta, g.abs().max(dim=1).values)


@pytest.mark.parametrize("dtype", [torch.float32, torch.bfloat16])
@pytest.mark.parametrize("beta", [0.01, 0.05, 0.95, 0.99])
def test_jsd_beta_near_the_ends(osd, beta, dtype):
    # m = beta p + (1 - beta) q is then dominated by one side; log2(p/m) and log2(q/m)
    # still come out against the oracle within the parity bar
    spec = W.DistillSpec(4, 32000, dtype, 2.0, "draft+noise", 1.5, 1.0)
    inp = W.distill_inputs(spec, seed=1234 + int(beta * 100))
    z, t = inp["draft"], inp["target"]
    for tau in (1.0, 0.7):
        lg, gg = _run(osd, z, t, None, "jsd", beta, tau=tau)
        lr, gr = _oracle(z, t, None, "jsd", beta, tau=tau)
        check_distill(lg, gg, lr, gr, np.ones(4, bool))


def test_extreme_and_neg_inf_logits(osd):
    g0 = torch.Generator().manual_seed(9)
    z = torch.randn(5, 3000, generator=g0) * 3
    t = torch.randn(5, 3000, generator=g0) * 3
    z[0] *= 30
    t[1, 500:] = float("-inf")
    z[2, :100] = float("-inf")
    t[2, :100] = float("-inf")
    t[3, 7] = 60.0
    for kind in KINDS:
        lg, gg = _run(osd, z, t, None, kind, 0.4, tau=1.3)
        lr, gr = _oracle(z, t, None, kind, 0.4, tau=1.3)
        skip = _tvd_ambiguous(z, t, 1.3) if kind == "tvd" else None
        check_distill(lg, gg, lr, gr, np.ones(5, bool), skip)


@pytest.mark.parametrize("dtype", [torch.bfloat16, torch.float32])
@pytest.mark.parametrize("tau", [1.0, 0.7])
def test_logits_far_above_the_first_chunks(osd, dtype, tau):
    """TVD and JSD sum against a reference taken from each thread's first chunk; a
    logit far above it later in the row (or a row whose first chunks are all -inf)
    must give the same result as the true maxima."""
    g0 = torch.Generator().manual_seed(31)
    N, V = 6, 32000
    z = torch.randn(N, V, generator=g0) * 2
    t = torch.randn(N, V, generator=g0) * 2
    z[0, V - 1] = 80.0                       # a late spike in the draft row
    t[1, 31000] = 50.0                       # ... in the target row only
    z[2, :4096] = float("-inf")              # every first chunk of the span is -inf
    t[2, :4096] = float("-inf")
    t[3] = z[3]                              # identical rows with a late spike in both
    z[3, 20000] = t[3, 20000] = 70.0
    z[4, 9000:9100] = 45.0                   # a late plateau
    z, t = z.to(dtype), t.to(dtype)
    for kind in KINDS:
        lg, gg = _run(osd, z, t, None, kind, 0.3, tau=tau)
        lr, gr = _oracle(z, t, None, kind, 0.3, tau=tau)
        skip = _tvd_ambiguous(z, t, tau) if kind == "tvd" else None
        check_distill(lg, gg, lr, gr, np.ones(N, bool), skip)


def test_invalid_arguments_are_rejected(osd):
    dev = torch.device("cuda")
    z = torch.zeros(2, 16, device=dev)
    with pytest.raises(osd.OsdError) as ei:
        osd.osd_distill(z, z, None, "jsd", 1.5)
    assert ei.value.status == osd.OSD_ERR_INVALID_ARG
    with pytest.raises(osd.OsdError) as ei:
        osd.osd_distill(z, z, None, 7, 0.5)
    assert ei.value.status == osd.OSD_ERR_INVALID_ARG
    with pytest.raises(osd.OsdError) as ei:
        osd.osd_distill(z, z, None, "fkl", 0.5, temperature=0.0)
    assert ei.value.status == osd.OSD_ERR_INVALID_ARG
    big = torch.zeros(1, 500000, dtype=torch.bfloat16, device=dev)
    with pytest.raises(osd.OsdError) as ei:
        osd.osd_distill(big, big, None, "fkl", 0.5)
    assert ei.value.status == osd.OSD_ERR_UNSUPPORTED
    st = torch.full((1,), 123, dtype=torch.int32, device=dev)
    e = torch.zeros(0, 16, device=dev)
    osd.osd_distill(e, e, None, "fkl", 0.5, status=st)
    assert st.item() == 0


# ----------------------------------------------------------------- full-size workloads
def test_workload_tiny_config_full(osd):
    """Forward-KL of the 16 draft rows against target rows 0..k-1 (strided view)."""
    spec = W.VERIFY[1]
    inp = W.verify_inputs(spec, seed=W.seed_for(1))
    z, t = inp["draft"], inp["target"]
    dev = torch.device("cuda")
    td = t.to(dev)
    status = torch.full((1,), -1, dtype=torch.int32, device=dev)
    dl = torch.full((4, 4, spec.V), float("nan"), device=dev)
    loss, g = osd.osd_distill(z.to(dev), td[:, :4], None, "fkl", 0.5, dlogits=dl, status=status)
    torch.cuda.synchronize()
    assert status.item() == 0
    lr, gr = _oracle(z, t[:, :4].contiguous(), None, "fkl", 0.5)
    check_distill(loss.cpu().numpy().reshape(-1), g.cpu().numpy().reshape(-1, spec.V), lr, gr,
                  np.ones(16, bool))


@pytest.mark.parametrize("kind", KINDS)
def test_many_rows_long_spans_sampled(osd, kind):
    """More rows than SMs at V = 100000 bf16: full-length spans of 12544 entries, which every
    kind but TVD runs on 256-thread CTAs; 8 sampled rows against the oracle."""
    N, V = 200, 100000
    spec = W.DistillSpec(N, V, torch.bfloat16, 2.0, "draft+noise", 1.5, 1.0)
    inp = W.distill_inputs(spec, seed=4242, device="cuda")
    z, t = inp["draft"], inp["target"]
    dl = torch.full((N, V), float("nan"), device="cuda")
    beta = 0.3 if kind == "jsd" else 0.5
    loss, g = osd.osd_distill(z, t, None, kind, beta, dlogits=dl, temperature=0.9)
    torch.cuda.synchronize()
    idx = torch.tensor(sorted(np.random.default_rng(7).choice(N, 8, replace=False)), device="cuda")
    zs, ts = z[idx].cpu(), t[idx].cpu()
    lr, gr = _oracle(zs, ts, None, kind, beta, tau=0.9)
    skip = _tvd_ambiguous(zs, ts, 0.9) if kind == "tvd" else None
    check_distill(loss[idx].cpu().numpy(), g[idx].cpu().numpy(), lr, gr, np.ones(8, bool), skip)
    assert not torch.isnan(g).any()


@pytest.mark.parametrize("kind", ["tvd", "jsd"])
@pytest.mark.parametrize("V", [8196, 32004, 100, 12])
def test_single_row_ragged_tail(osd, kind, V):
    """One bf16 row with V = 4 (mod 8): the row is on the 16-byte path, and its last span ends
    in a tail of 4 entries shorter than a 16-byte chunk (the TMEM-staged kernel keeps those in
    registers; TVD keeps q sign(q - p) there for its gradient)."""
    g0 = torch.Generator().manual_seed(V)
    z = (torch.randn(1, V, generator=g0) * 2).to(torch.bfloat16)
    t = (z.float() + torch.randn(1, V, generator=g0)).to(torch.bfloat16)
    t[0, V - 1] = 9.0   # mass in the tail itself
    z[0, V - 2] = 7.0
    for tau in (1.0, 0.8):
        lg, gg = _run(osd, z, t, None, kind, 0.4, tau=tau)
        lr, gr = _oracle(z, t, None, kind, 0.4, tau=tau)
        skip = _tvd_ambiguous(z, t, tau) if kind == "tvd" else None
        check_distill(lg, gg, lr, gr, np.ones(1, bool), skip)


MASK_PATTERNS = ["random40", "none", "all", "last_only", "first_and_last"]


@pytest.mark.parametrize("kind", ["rkl", "jsd", "tvd"])
@pytest.mark.parametrize("pattern", MASK_PATTERNS)
def test_masked_rows_every_pattern(osd, kind, pattern):
    """Masked launches on the TMEM-staged runs of rows: every active row must match
    the oracle and every masked-out row keep loss 0 and its untouched gradient,
    for 1003 rows (runs of 8, pairs and single rows, the last run ragged) with
    40 %, none, all, only the last, or only the first and last rows active."""
    N, V = 1003, 4000
    spec = W.DistillSpec(N, V, torch.bfloat16, 2.0, "draft+noise", 1.5, 1.0)
    inp = W.distill_inputs(spec, seed=501)
    z, t = inp["draft"], inp["target"]
    mask = torch.zeros(N, dtype=torch.uint8)
    if pattern == "random40":
        g = torch.Generator().manual_seed(502)
        mask[torch.randperm(N, generator=g)[: round(0.4 * N)]] = 1
    elif pattern == "all":
        mask[:] = 1
    elif pattern == "last_only":
        mask[-1] = 1
    elif pattern == "first_and_last":
        mask[0] = 1
        mask[-1] = 1
    lg, gg = _run(osd, z, t, mask, kind, 0.5)
    lr, gr = _oracle(z, t, mask, kind, 0.5)
    skip = _tvd_ambiguous(z, t) if kind == "tvd" else None
    rep = check_distill(lg, gg, lr, gr, mask.numpy() == 1, skip)
    print(f"{kind} {pattern}: {rep}")


@pytest.mark.parametrize("kind", ["rkl", "jsd", "tvd"])
def test_masked_rows_unaligned_mask_and_few_rows(osd, kind):
    """A mask view that starts off a 16-byte boundary, and launches with fewer
    rows than resident clusters (each row a run of its own), masked or not."""
    dev = torch.device("cuda")
    for N, off in ((300, 1), (5, 0), (5, 3)):
        spec = W.DistillSpec(N, 4000, torch.bfloat16, 2.0, "draft+noise", 1.5, 1.0)
        inp = W.distill_inputs(spec, seed=600 + N + off)
        z, t = inp["draft"], inp["target"]
        g = torch.Generator().manual_seed(601 + N)
        mask = (torch.rand(N, generator=g) < 0.5).to(torch.uint8)
        mask[0] = 1
        big = torch.zeros(N + 16, dtype=torch.uint8, device=dev)
        big[off:off + N] = mask.to(dev)
        md = big[off:off + N]
        dl = torch.full((N, 4000), float("nan"), dtype=torch.float32, device=dev)
        loss, gg = osd.osd_distill(z.to(dev), t.to(dev), md, kind, 0.5, dlogits=dl)
        torch.cuda.synchronize()
        lr, gr = _oracle(z, t, mask, kind, 0.5)
        skip = _tvd_ambiguous(z, t) if kind == "tvd" else None
        check_distill(loss.cpu().numpy(), gg.cpu().numpy(), lr, gr, mask.numpy() == 1, skip)


def test_concurrent_flushes_on_two_streams(osd):
    """Two buffer flushes on the TMEM-staged runs in flight at once on two streams
    (RKL beside TVD, FKL beside JSD): their clusters share the SMs and tensor memory,
    and every CTA's shared-memory request keeps the resident CTAs within the SM's 512
    columns, so each flush gives exactly the results it gives alone."""
    dev = torch.device("cuda")
    spec = W.DistillSpec(1024, 32000, torch.bfloat16, 2.0, "draft+noise", 2.0, 1.0)
    a = W.distill_inputs(spec, seed=701, device=dev)
    b = W.distill_inputs(spec, seed=702, device=dev)
    for ka, kb in (("rkl", "tvd"), ("fkl", "jsd")):
        ref_a = osd.osd_distill(a["draft"], a["target"], None, ka, 0.5)
        ref_b = osd.osd_distill(b["draft"], b["target"], None, kb, 0.5)
        torch.cuda.synchronize()
        s1, s2 = torch.cuda.Stream(), torch.cuda.Stream()
        s1.wait_stream(torch.cuda.current_stream())
        s2.wait_stream(torch.cuda.current_stream())
        with torch.cuda.stream(s1):
            out_a = osd.osd_distill(a["draft"], a["target"], None, ka, 0.5, stream=s1)
        with torch.cuda.stream(s2):
            out_b = osd.osd_distill(b["draft"], b["target"], None, kb, 0.5, stream=s2)
        torch.cuda.synchronize()
        for ref, out in ((ref_a, out_a), (ref_b, out_b)):
            assert torch.equal(ref[0], out[0]) and torch.equal(ref[1], out[1])
