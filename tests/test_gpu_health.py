"""The shared failure path: a bounded device-side wait that runs out reports
OSD_ERR_TIMEOUT through its status word and leaves the context usable.  The
wait is on an mbarrier that nothing completes (no fault, no trap, no copy in
flight)."""
import numpy as np
import pytest
import torch

import oracle
from tests.parity import check_distill

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def osd():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA GPU")
    import paper_2310_07177_gb300 as pkg
    pkg.build_library()
    pkg.load_library()
    return pkg


def test_bounded_wait_runs_out_and_reports(osd):
    status, waited = osd.osd_check_bounded_wait(20_000)  # 20 ms
    assert status == osd.OSD_ERR_TIMEOUT
    assert 20_000_000 <= waited < 1_000_000_000
    # the context is still usable: a distill call right after gives the oracle's results
    g = torch.Generator().manual_seed(3)
    z = torch.randn(4, 3000, generator=g)
    t = torch.randn(4, 3000, generator=g)
    st = torch.full((1,), 77, dtype=torch.int32, device="cuda")
    loss, grad = osd.osd_distill(z.cuda(), t.cuda(), None, "rkl", 0.5, status=st)
    torch.cuda.synchronize()
    assert st.item() == osd.OSD_OK
    lr, gr = oracle.distill(z, t, None, "rkl", 0.5)
    check_distill(loss.cpu().numpy(), grad.cpu().numpy(), lr, gr, np.ones(4, bool))


def test_invalid_limits_are_rejected(osd):
    with pytest.raises(osd.OsdError):
        osd.osd_check_bounded_wait(0)
    with pytest.raises(osd.OsdError):
        osd.osd_check_bounded_wait(20_000_000)
