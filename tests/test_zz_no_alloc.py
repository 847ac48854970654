"""osd_verify_noalloc: verification for callers that must not allocate device
memory while serving (an engine that reserved all free memory for its KV cache,
a plugin without an allocator, a loop that cannot afford cudaMalloc's device
synchronisation).  It runs on the library's own static workspace; its results
must equal osd_verify's on the same inputs, call after call, and match the
oracle like osd_verify's do; and a call must leave the device's free memory
and torch's allocations where they were.

This file is collected last on purpose, and it needs nothing from the other
tests: it passes alone in a fresh process and after the rest of the suite."""
import ctypes
import gc

import numpy as np
import pytest
import torch

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


CASES = [(W.VERIFY[2], W.seed_for(2), 1.0),
         (W.VerifySpec(48, 4, 50257, torch.bfloat16, 3.0, 0.5, 2.0, 0.7), 11, 0.7),
         (W.VERIFY[2], W.seed_for(2) + 1, 0.0)]


def test_noalloc_allocates_nothing(osd):
    """Neither the first call in this process (which looks up the array's
    address; this test runs before the file's others) nor the calls after it
    change torch's allocations or the device's free memory."""
    dev = torch.device("cuda")
    spec = W.VERIFY[2]
    inp = W.verify_inputs(spec, seed=W.seed_for(2) + 7, device=dev)
    # the kernels' module is loaded (with the array in it) by a plain osd_verify call first
    osd.osd_verify(inp["draft"], inp["target"], inp["tokens"], inp["uniforms"], 1.0)
    outs = [_outputs(spec.B, spec.k, dev) for _ in range(3)]
    # earlier tests' tensors held in reference cycles would otherwise be freed by the
    # cyclic collector in the middle of the measurement
    gc.collect()
    gc.disable()
    try:
        torch.cuda.synchronize()
        alloc0 = torch.cuda.memory_allocated(dev)
        reserved0 = torch.cuda.memory_reserved(dev)
        free0, _ = torch.cuda.mem_get_info(dev)
        for out in outs:
            osd.osd_verify_noalloc(inp["draft"], inp["target"], inp["tokens"], inp["uniforms"], 1.0, out)
            torch.cuda.synchronize()
            assert torch.cuda.memory_allocated(dev) == alloc0
            assert torch.cuda.memory_reserved(dev) == reserved0
            free1, _ = torch.cuda.mem_get_info(dev)
            assert free1 == free0, f"device free memory moved by {free0 - free1} bytes"
    finally:
        gc.enable()
    _same(outs[1], outs[0])
    _same(outs[2], outs[0])


def test_noalloc_matches_verify_and_oracle_on_consecutive_calls(osd):
    dev = torch.device("cuda")
    for spec, seed, T in CASES:  # consecutive calls reuse the same static workspace
        inp = W.verify_inputs(spec, seed=seed, device=dev)
        y = inp["greedy_tokens"] if T == 0.0 else inp["tokens"]
        ref = osd.osd_verify(inp["draft"], inp["target"], y, inp["uniforms"], T)
        out = _outputs(spec.B, spec.k, dev)
        got = osd.osd_verify_noalloc(inp["draft"], inp["target"], y, inp["uniforms"], T, out)
        torch.cuda.synchronize()
        _same(got, ref)
        # and against the oracle, under the same rules as osd_verify
        oref = oracle.verify(inp["draft"].cpu(), inp["target"].cpu(), y.cpu(), inp["uniforms"].cpu(),
                             float(np.float32(T)))
        rep = check_verify(got, oref, spec.k, spec.V)
        if T > 0:
            check_margins(got, oref)
        print(f"noalloc B={spec.B} k={spec.k} V={spec.V} T={T}: {rep}")


def test_noalloc_rejects_sizes_beyond_its_scratch(osd):
    lib = osd.load_library()
    n = ctypes.c_size_t(0)
    assert lib.osd_verify_workspace_size(4096, 16, 128256, ctypes.byref(n)) == osd.OSD_OK
    assert n.value > 4 << 20
    fake = ctypes.c_void_p(16)  # never dereferenced: the size check fails first
    st = lib.osd_verify_noalloc(fake, fake, osd.OSD_BF16, 4096, 16, 128256, fake, fake, 1.0,
                                fake, fake, fake, None, None, None)
    assert st == osd.OSD_ERR_UNSUPPORTED
    # the largest workload still fits, as do 512-row batches whose slices are longer
    for B, k, V in ((256, 8, 128256), (512, 8, 128256), (64, 4, 1 << 21)):
        assert lib.osd_verify_workspace_size(B, k, V, ctypes.byref(n)) == osd.OSD_OK
        assert n.value <= 4 << 20, (B, k, V, n.value)
