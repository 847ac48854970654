"""osd_verify_noalloc: verification for callers that must not allocate device
memory while serving (an engine that reserved all free memory for its KV cache,
a plugin without an allocator, a loop that cannot afford cudaMalloc's device
synchronisation).  It runs on the library's own static workspace; its results
must equal osd_verify's on the same inputs, call after call.

This file is collected last on purpose, and it needs nothing from the other
tests: it passes alone in a fresh process and after the rest of the suite."""
import ctypes

import numpy as np
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


def _outputs(B, k, dev):
    import paper_2310_07177_gb300 as pkg
    return pkg.VerifyResult(torch.full((B,), -7, dtype=torch.int32, device=dev),
                            torch.full((B, k + 1), -7, dtype=torch.int32, device=dev),
                            torch.full((B, k), 7, dtype=torch.uint8, device=dev),
                            torch.full((B, k), -7.0, device=dev), torch.full((B,), -7.0, device=dev))


def _same(a, b):
    assert torch.equal(a.accepted, b.accepted)
    assert torch.equal(a.out_tokens, b.out_tokens)
    assert torch.equal(a.mismatch_mask, b.mismatch_mask)
    # diagnostics come from identical kernels on identical inputs: equal, NaN where NaN
    for x, y in ((a.diag_margin, b.diag_margin), (a.diag_cdf_gap, b.diag_cdf_gap)):
        xs, ys = x.cpu().numpy(), y.cpu().numpy()
        np.testing.assert_array_equal(np.isnan(xs), np.isnan(ys))
        np.testing.assert_allclose(xs[~np.isnan(xs)], ys[~np.isnan(ys)], rtol=0, atol=0)


def test_noalloc_matches_verify_on_consecutive_calls(osd):
    dev = torch.device("cuda")
    cases = [(W.VERIFY[2], W.seed_for(2), 1.0), (W.VerifySpec(48, 4, 50257, torch.bfloat16, 3.0, 0.5, 2.0, 0.7),
                                                   11, 0.7),
             (W.VERIFY[2], W.seed_for(2) + 1, 0.0)]
    for spec, seed, T in cases:  # consecutive calls reuse the same static workspace
        inp = W.verify_inputs(spec, seed=seed, device=dev)
        y = inp["greedy_tokens"] if T == 0.0 else inp["tokens"]
        ref = osd.osd_verify(inp["draft"], inp["target"], y, inp["uniforms"], T)
        out = _outputs(spec.B, spec.k, dev)
        got = osd.osd_verify_noalloc(inp["draft"], inp["target"], y, inp["uniforms"], T, out)
        torch.cuda.synchronize()
        _same(got, ref)


def test_noalloc_rejects_sizes_beyond_its_scratch(osd):
    lib = osd.load_library()
    n = ctypes.c_size_t(0)
    assert lib.osd_verify_workspace_size(4096, 16, 128256, ctypes.byref(n)) == osd.OSD_OK
    assert n.value > 4 << 20
    dev = torch.device("cuda")
    fake = ctypes.c_void_p(16)  # never dereferenced: the size check fails first
    st = lib.osd_verify_noalloc(fake, fake, osd.OSD_BF16, 4096, 16, 128256, fake, fake, 1.0,
                                fake, fake, fake, None, None, None)
    assert st == osd.OSD_ERR_UNSUPPORTED
    # the largest workload still fits
    assert lib.osd_verify_workspace_size(256, 8, 128256, ctypes.byref(n)) == osd.OSD_OK
    assert n.value <= 4 << 20
