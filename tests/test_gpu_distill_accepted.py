"""GPU parity of osd_distill_accepted (distillation of the rows verification
rejected, chosen and compacted on the device) against oracle.distill_rejected,
alone, chained after osd_verify on the same stream, and inside a CUDA graph."""
import numpy as np
import pytest
import torch

import oracle
from paper_2310_07177_gb300 import workloads as W
from tests.parity import check_distill, tvd_ties, check_verify

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


def _fresh_out(osd, B, V, dev="cuda"):
    return osd.DistillAcceptedResult(torch.full((B,), float("nan"), device=dev),
                                     torch.full((B, V), float("nan"), device=dev),
                                     torch.full((B,), -7, dtype=torch.int32, device=dev),
                                     torch.full((1,), -7, dtype=torch.int32, device=dev))


def _logits(B, k, V, dtype, seed):
    g = torch.Generator().manual_seed(seed)
    z = (torch.randn(B, k, V, generator=g) * 2).to(dtype)
    t = (torch.randn(B, k + 1, V, generator=g) * 2).to(dtype)
    return z, t


def _compare(res, ref, V, tvd_skip=None):
    loss_r, g_r, seq_r, count_r = ref
    count = int(res.count.item())
    assert count == count_r
    assert np.array_equal(res.seq_of_row.cpu().numpy(), seq_r)
    loss = res.loss.cpu().numpy()
    g = res.dlogits.cpu().numpy()
    assert np.all(loss[count:] == 0.0), "inactive slots must get loss 0"
    assert np.all(np.isnan(g[count:])), "inactive gradient rows must stay untouched"
    if count:
        check_distill(loss[:count], g[:count], loss_r[:count], g_r[:count], np.ones(count, bool), tvd_skip)
    return count


CASES = [  # (B, k, V, dtype)
    (1, 1, 1, torch.float32),
    (7, 3, 100, torch.float32),
    (16, 5, 32000, torch.bfloat16),
    (9, 4, 33001, torch.bfloat16),
    (64, 8, 4097, torch.float32),
    (5, 2, 128256, torch.bfloat16),
]


@pytest.mark.parametrize("B,k,V,dtype", CASES)
@pytest.mark.parametrize("kind", KINDS)
def test_matches_oracle(osd, B, k, V, dtype, kind):
    z, t = _logits(B, k, V, dtype, seed=B * 131 + V)
    acc = W.accepted_inputs(B, k, seed=B + k)
    tau = 0.8 if kind in ("rkl", "tvd") else 1.0
    out = _fresh_out(osd, B, V)
    res = osd.osd_distill_accepted(z.cuda(), t.cuda(), acc.cuda(), kind, 0.3, temperature=tau, out=out)
    torch.cuda.synchronize()
    ref = oracle.distill_rejected(z, t, acc, kind, 0.3, temperature=float(np.float32(tau)))
    skip = None
    if kind == "tvd":  # entries whose sign(q - p) fp32 cannot decide, for the compacted rows
        _, _, seq, count = ref
        a = acc.numpy()
        if count:
            rows_z = np.stack([z[b, a[b]].double().numpy() for b in seq[:count]])
            rows_t = np.stack([t[b, a[b]].double().numpy() for b in seq[:count]])
            skip = tvd_ties(rows_z, rows_t, float(np.float32(tau)))
    _compare(res, ref, V, skip)


def test_every_sequence_inactive_and_empty_batch(osd):
    B, k, V = 6, 3, 500
    z, t = _logits(B, k, V, torch.bfloat16, seed=2)
    for fill in (k, -1):
        acc = torch.full((B,), fill, dtype=torch.int32)
        out = _fresh_out(osd, B, V)
        osd.osd_distill_accepted(z.cuda(), t.cuda(), acc.cuda(), "rkl", out=out)
        torch.cuda.synchronize()
        assert out.count.item() == 0
        assert out.seq_of_row.cpu().tolist() == list(range(B))
        assert torch.all(out.loss == 0) and torch.all(torch.isnan(out.dlogits))
    e = torch.zeros(0, k, V, dtype=torch.bfloat16, device="cuda")
    et = torch.zeros(0, k + 1, V, dtype=torch.bfloat16, device="cuda")
    out = _fresh_out(osd, 0, V)
    osd.osd_distill_accepted(e, et, torch.zeros(0, dtype=torch.int32, device="cuda"), "fkl", out=out)
    torch.cuda.synchronize()
    assert out.count.item() == 0


def _serving_inputs():
    spec = W.VERIFY[2]
    return spec, W.verify_inputs(spec, seed=W.seed_for(2) + 17, device="cuda")


def test_chained_after_verify(osd):
    """verify then distill on its accepted counts, same stream, no host sync in between."""
    spec, inp = _serving_inputs()
    res = osd.osd_verify(inp["draft"], inp["target"], inp["tokens"], inp["uniforms"], spec.temperature)
    out = osd.osd_distill_accepted(inp["draft"], inp["target"], res.accepted, "rkl")
    torch.cuda.synchronize()
    T = float(np.float32(spec.temperature))
    ref_v = oracle.verify(inp["draft"].cpu(), inp["target"].cpu(), inp["tokens"].cpu(), inp["uniforms"].cpu(), T)
    rep = check_verify(res, ref_v, spec.k, spec.V)
    assert rep["near_tie_differ"] == 0, "this seed must not hit a near tie"
    ref = oracle.distill_rejected(inp["draft"].cpu(), inp["target"].cpu(), ref_v["accepted"], "rkl")
    # the binding allocated the outputs with torch.empty: compare the active slots
    loss_r, g_r, seq_r, count_r = ref
    assert int(out.count.item()) == count_r > 0
    assert np.array_equal(out.seq_of_row.cpu().numpy(), seq_r)
    check_distill(out.loss.cpu().numpy()[:count_r], out.dlogits.cpu().numpy()[:count_r], loss_r[:count_r],
                  g_r[:count_r], np.ones(count_r, bool))
    assert np.all(out.loss.cpu().numpy()[count_r:] == 0)


def test_graph_replay_matches_eager(osd):
    """verify + distill_accepted captured in one CUDA graph give the eager results bit for bit."""
    spec, inp = _serving_inputs()
    B, k, V = spec.B, spec.k, spec.V
    static = {key: inp[key].clone() for key in ("draft", "target", "tokens", "uniforms")}
    ws = torch.empty(osd.osd_verify_workspace_size(B, k, V), dtype=torch.uint8, device="cuda")
    out = _fresh_out(osd, B, V)

    def step():
        r = osd.osd_verify(static["draft"], static["target"], static["tokens"], static["uniforms"],
                           spec.temperature, workspace=ws)
        osd.osd_distill_accepted(static["draft"], static["target"], r.accepted, "tvd", out=out)
        return r

    side = torch.cuda.Stream()
    side.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(side):
        step()  # warm-up outside capture
    torch.cuda.current_stream().wait_stream(side)
    torch.cuda.synchronize()
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph):
        gres = step()
    # new inputs into the captured buffers, then replay
    inp2 = W.verify_inputs(spec, seed=W.seed_for(2) + 99, device="cuda")
    for key in static:
        static[key].copy_(inp2[key])
    out.dlogits.fill_(float("nan"))
    graph.replay()
    torch.cuda.synchronize()
    got = (gres.accepted.clone(), out.loss.clone(), out.dlogits.clone(), out.seq_of_row.clone(), out.count.clone())
    eager_v = osd.osd_verify(inp2["draft"], inp2["target"], inp2["tokens"], inp2["uniforms"], spec.temperature)
    eager = osd.osd_distill_accepted(inp2["draft"], inp2["target"], eager_v.accepted, "tvd",
                                     out=_fresh_out(osd, B, V))
    torch.cuda.synchronize()
    assert torch.equal(got[0], eager_v.accepted)
    n = int(eager.count.item())
    assert int(got[4].item()) == n and torch.equal(got[3], eager.seq_of_row)
    assert torch.equal(got[1], eager.loss)
    assert torch.equal(got[2][:n], eager.dlogits[:n])


def test_invalid_arguments_are_rejected(osd):
    z = torch.zeros(2, 3, 16, device="cuda")
    t = torch.zeros(2, 4, 16, device="cuda")
    with pytest.raises(ValueError):
        osd.osd_distill_accepted(z, t[:, :3], torch.zeros(2, dtype=torch.int32, device="cuda"))
    with pytest.raises(ValueError):
        osd.osd_distill_accepted(z, t, torch.zeros(2, dtype=torch.int64, device="cuda"))
    with pytest.raises(osd.OsdError) as ei:
        osd.osd_distill_accepted(z, t, torch.zeros(2, dtype=torch.int32, device="cuda"), "jsd", 2.0)
    assert ei.value.status == osd.OSD_ERR_INVALID_ARG
