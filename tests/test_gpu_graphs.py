"""CUDA-graph capture of the entry points a serving loop replays every step:
greedy verification, mixed-token sampling and token-tree verification captured
in one graph, replayed on new inputs, give the eager results bit for bit.
(verify at T > 0 with the fused distillation is covered in
test_gpu_distill_accepted.py.)"""
import pytest
import torch

from paper_2310_07177_gb300 import workloads as W

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def osd():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA GPU")
    import paper_2310_07177_gb300 as pkg
    pkg.build_library()
    pkg.load_library()
    return pkg


def _inputs(seed):
    dev = torch.device("cuda")
    spec = W.VERIFY[2]
    v = W.verify_inputs(spec, seed=seed, device=dev)
    tree = W.tree_inputs(8, W.MEDUSA_TREE, 4096, torch.bfloat16, 1.0, seed=seed, device=dev, target_noise=0.8)
    g = torch.Generator(device=dev).manual_seed(seed)
    u = torch.rand(spec.B, generator=g, device=dev)
    return spec, v, tree, u


def test_graph_replay_matches_eager(osd):
    spec, v, tree, u = _inputs(W.seed_for(2))
    par = W.MEDUSA_TREE
    B, k, V = spec.B, spec.k, spec.V
    static = {"target": v["target"].clone(), "greedy": v["greedy_tokens"].clone(), "u": u.clone(),
              "z0": v["draft"][:, 0].contiguous(), "t0": v["target"][:, 0].contiguous(),
              "tz": tree["draft"].clone(), "tt": tree["target"].clone(), "ty": tree["tokens"].clone(),
              "tu": tree["uniforms"].clone()}
    ws = torch.empty(osd.osd_verify_workspace_size(B, k, V), dtype=torch.uint8, device="cuda")
    tws = torch.empty(osd.osd_verify_tree_workspace_size(8, len(par), 4096), dtype=torch.uint8, device="cuda")
    tok = torch.empty(B, dtype=torch.int32, device="cuda")

    def step():
        r0 = osd.osd_verify(None, static["target"], static["greedy"], None, 0.0, workspace=ws)
        osd.osd_mixed_sample(static["z0"], static["t0"], static["u"], 0.4, temperature=0.8, tokens=tok)
        rt = osd.osd_verify_tree(static["tz"], static["tt"], par, static["ty"], static["tu"], 1.0, workspace=tws)
        return r0, rt

    side = torch.cuda.Stream()
    side.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(side):
        step()  # warm-up outside capture
    torch.cuda.current_stream().wait_stream(side)
    torch.cuda.synchronize()
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph):
        g0, gt = step()

    # new inputs into the captured buffers, then replay
    spec2, v2, tree2, u2 = _inputs(W.seed_for(2) + 7)
    static["target"].copy_(v2["target"])
    static["greedy"].copy_(v2["greedy_tokens"])
    static["u"].copy_(u2)
    static["z0"].copy_(v2["draft"][:, 0])
    static["t0"].copy_(v2["target"][:, 0])
    for a, b in (("tz", "draft"), ("tt", "target"), ("ty", "tokens"), ("tu", "uniforms")):
        static[a].copy_(tree2[b])
    graph.replay()
    torch.cuda.synchronize()

    e0 = osd.osd_verify(None, v2["target"], v2["greedy_tokens"], None, 0.0)
    etok, _ = osd.osd_mixed_sample(v2["draft"][:, 0].contiguous(), v2["target"][:, 0].contiguous(), u2, 0.4,
                                   temperature=0.8)
    et = osd.osd_verify_tree(tree2["draft"], tree2["target"], par, tree2["tokens"], tree2["uniforms"], 1.0)
    torch.cuda.synchronize()
    assert torch.equal(g0.accepted, e0.accepted) and torch.equal(g0.out_tokens, e0.out_tokens)
    assert torch.equal(g0.mismatch_mask, e0.mismatch_mask)
    assert torch.equal(tok, etok)
    for f in ("accepted", "path", "out_tokens", "last_node"):
        assert torch.equal(getattr(gt, f), getattr(et, f)), f
