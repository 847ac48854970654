"""Every row of the full-size workloads against the oracle, launched exactly as
the benchmark launches them (Appendix A.1 for verification, Eq. 2-3 for the
distillation loss and gradient):

  - the 16384 x 32128 buffer flush, JSD beta = 1/2 under its 40 % mask: all
    6554 active rows, and all 9830 inactive rows left untouched;
  - the 65536 x 32000 flush, reverse KL and TVD: all 65536 rows of each;
  - the 128k-vocabulary verify, B = 256, k = 8, V = 128256, T = 0.7: all 256
    sequences, with the near-tie count and how many of those differ;
  - its forward-KL distillation of the rejected rows, both through the mask on
    the [B, k] draft rows against target[:, :k] and through
    osd_distill_accepted: every rejected row.

Each test prints the counts of its whole comparison."""
import numpy as np
import pytest
import torch

from paper_2310_07177_gb300 import workloads as W
from tests.fullsize import distill_parity, verify_oracle
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


def _flush(osd, workload, kind, beta):
    spec = W.DISTILL[workload]
    inp = W.distill_inputs(spec, seed=W.seed_for(workload), device="cuda")
    z, t, mask = inp["draft"], inp["target"], inp["mask"]
    dl = torch.full((spec.N, spec.V), float("nan"), device="cuda")
    status = torch.full((1,), -1, dtype=torch.int32, device="cuda")
    loss, g = osd.osd_distill(z, t, mask, kind, beta, dlogits=dl, status=status)
    torch.cuda.synchronize()
    assert status.item() == 0
    active = None if mask is None else mask.cpu().numpy() == 1
    rep = distill_parity(z, t, active, loss, g, kind, beta)
    print(f"flush {spec.N} x {spec.V} {kind}: {rep}")
    return spec, rep


def test_masked_flush_jsd_every_row(osd):
    spec, rep = _flush(osd, 3, "jsd", 0.5)
    n_on = int(round(spec.active_frac * spec.N))
    assert rep["rows"] == n_on == 6554
    assert rep["inactive_rows"] == spec.N - n_on == 9830


@pytest.mark.parametrize("kind", ["rkl", "tvd"])
def test_flush_65536_rows_every_row(osd, kind):
    spec, rep = _flush(osd, 4, kind, 0.5)
    assert rep["rows"] == spec.N == 65536 and rep["inactive_rows"] == 0


@pytest.fixture(scope="module")
def large_vocab(osd):
    spec = W.VERIFY[5]
    inp = W.verify_inputs(spec, seed=W.seed_for(5), device="cuda")
    res = osd.osd_verify(inp["draft"], inp["target"], inp["tokens"], inp["uniforms"], spec.temperature)
    torch.cuda.synchronize()
    ref = verify_oracle(inp["draft"], inp["target"], inp["tokens"], inp["uniforms"],
                        float(np.float32(spec.temperature)))
    return spec, inp, res, ref


def test_large_vocab_verify_every_sequence(large_vocab):
    spec, inp, res, ref = large_vocab
    rep = check_verify(res, ref, spec.k, spec.V)
    worst = check_margins(res, ref)
    assert rep["sequences"] == spec.B == 256
    acc = res.accepted.cpu().numpy()
    print(f"verify B=256 k=8 V=128256: {rep}, accept-ratio error max {worst:.3g}, "
          f"mean accepted {acc.mean():.3f}, rejecting sequences {int((acc < spec.k).sum())}")


def test_large_vocab_fkl_chain_every_rejected_row(osd, large_vocab):
    """osd_verify's mismatch mask drives forward-KL distillation of the [B, k]
    draft rows against the target[:, :k] view on the same stream."""
    spec, inp, res, ref = large_vocab
    B, k, V = spec.B, spec.k, spec.V
    dl = torch.full((B, k, V), float("nan"), device="cuda")
    loss, g = osd.osd_distill(inp["draft"], inp["target"][:, :k], res.mismatch_mask, "fkl", 0.5, dlogits=dl)
    torch.cuda.synchronize()
    active = res.mismatch_mask.cpu().numpy().reshape(-1) == 1
    assert active.sum() == int((res.accepted.cpu() < k).sum())
    rep = distill_parity(inp["draft"].reshape(-1, V), inp["target"][:, :k].reshape(-1, V), active,
                         loss.reshape(-1), g.reshape(-1, V), "fkl", 0.5)
    assert rep["rows"] + rep["inactive_rows"] == B * k
    print(f"verify B=256 k=8 V=128256 -> FKL chain: {rep}")


def test_large_vocab_distill_accepted_every_row(osd, large_vocab):
    """The same rows chosen on the device from the accepted counts and compacted."""
    spec, inp, res, ref = large_vocab
    B, k, V = spec.B, spec.k, spec.V
    rej = osd.DistillAcceptedResult(torch.empty(B, device="cuda"),
                                    torch.full((B, V), float("nan"), device="cuda"),
                                    torch.empty(B, dtype=torch.int32, device="cuda"),
                                    torch.empty(1, dtype=torch.int32, device="cuda"))
    osd.osd_distill_accepted(inp["draft"], inp["target"], res.accepted, "fkl", 0.5, out=rej)
    torch.cuda.synchronize()
    acc = res.accepted.cpu().numpy()
    act = [b for b in range(B) if 0 <= acc[b] < k]
    n = len(act)
    assert int(rej.count.item()) == n
    seq = rej.seq_of_row.cpu().numpy()
    assert list(seq[:n]) == act and list(seq[n:]) == [b for b in range(B) if not 0 <= acc[b] < k]
    bi = torch.as_tensor(act, device="cuda", dtype=torch.long)
    ai = torch.as_tensor(acc[act], device="cuda", dtype=torch.long)
    rep = distill_parity(inp["draft"][bi, ai], inp["target"][bi, ai], None, rej.loss[:n], rej.dlogits[:n],
                         "fkl", 0.5)
    assert (rej.loss[n:] == 0).all() and torch.isnan(rej.dlogits[n:]).all()
    print(f"V=128256 osd_distill_accepted: {rep}, slots beyond the count {B - n}")
