"""The C-ABI library builds, loads and exports every function include/osd.h
declares; host-side argument checks answer without touching a GPU."""
import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "osd.h")


def _declared():
    src = open(HEADER).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(osd_[a-z_0-9]+)\s*\(", src)))


@pytest.fixture(scope="module")
def lib():
    import paper_2310_07177_gb300 as osd
    osd.build_library()
    return osd.load_library()


def test_every_declared_symbol_is_exported(lib):
    import paper_2310_07177_gb300 as osd
    names = _declared()
    assert set(names) == set(osd.EXPORTS), names
    for name in names:
        assert hasattr(lib, name), f"{name} missing from libosd.so"


def test_status_strings_and_version(lib):
    import paper_2310_07177_gb300 as osd
    assert osd.osd_abi_version() >> 16 == osd.ABI_MAJOR == 2
    for code in range(5):
        assert osd.osd_status_string(code).startswith("OSD_")
    assert osd.osd_status_string(99) == "OSD_ERR_UNKNOWN"


def test_workspace_size_host_checks(lib):
    import paper_2310_07177_gb300 as osd
    n = ctypes.c_size_t(0)
    assert lib.osd_verify_workspace_size(256, 8, 128256, ctypes.byref(n)) == osd.OSD_OK
    assert n.value >= 256 * 17 * 16 and n.value % 256 == 0  # >= one 16-byte statistic per row
    assert lib.osd_verify_workspace_size(-1, 8, 100, ctypes.byref(n)) == osd.OSD_ERR_INVALID_ARG
    assert lib.osd_verify_workspace_size(4, 8, 0, ctypes.byref(n)) == osd.OSD_ERR_INVALID_ARG
    assert lib.osd_verify_workspace_size(4, 65, 100, ctypes.byref(n)) == osd.OSD_ERR_UNSUPPORTED
    assert lib.osd_verify_workspace_size(4, 8, 100, None) == osd.OSD_ERR_INVALID_ARG


def test_argument_errors_return_before_any_launch(lib):
    """Invalid arguments are rejected on the host (no device pointer is touched)."""
    import paper_2310_07177_gb300 as osd
    fake = ctypes.c_void_p(0x1000)  # never dereferenced: every call below fails validation first
    # bad dtype, bad temperature
    assert lib.osd_verify(fake, fake, 7, 2, 2, 16, fake, fake, 1.0, fake, fake, fake, None, None,
                          fake, 1 << 20, None) == osd.OSD_ERR_INVALID_ARG
    assert lib.osd_verify(fake, fake, 0, 2, 2, 16, fake, fake, -1.0, fake, fake, fake, None, None,
                          fake, 1 << 20, None) == osd.OSD_ERR_INVALID_ARG
    # workspace too small
    assert lib.osd_verify(fake, fake, 0, 2, 2, 16, fake, fake, 1.0, fake, fake, fake, None, None,
                          fake, 8, None) == osd.OSD_ERR_INVALID_ARG
    # empty batch is a no-op
    assert lib.osd_verify(None, None, 0, 0, 2, 16, None, None, 1.0, None, None, None, None, None,
                          None, 0, None) == osd.OSD_OK
    # distill: bad beta, bad kind, bad temperature, vocabulary beyond the limit, negative stride
    assert lib.osd_distill(fake, fake, 1, 2, 1, 16, 16, 0, 16, 0, None, 2, 1.5, 1.0, fake, fake, None,
                           None) == osd.OSD_ERR_INVALID_ARG
    assert lib.osd_distill(fake, fake, 1, 2, 1, 16, 16, 0, 16, 0, None, 9, 0.5, 1.0, fake, fake, None,
                           None) == osd.OSD_ERR_INVALID_ARG
    for tau in (0.0, -1.0, float("nan"), float("inf")):
        assert lib.osd_distill(fake, fake, 1, 2, 1, 16, 16, 0, 16, 0, None, 0, 0.5, tau, fake, fake, None,
                               None) == osd.OSD_ERR_INVALID_ARG
    assert lib.osd_distill(fake, fake, 1, 1, 1, 500000, 0, 0, 0, 0, None, 0, 0.5, 1.0, fake, fake, None,
                           None) == osd.OSD_ERR_UNSUPPORTED
    assert lib.osd_distill(fake, fake, 1, 2, 1, 16, -16, 0, 16, 0, None, 0, 0.5, 1.0, fake, fake, None,
                           None) == osd.OSD_ERR_INVALID_ARG
    assert lib.osd_distill(None, None, 1, 0, 4, 16, 16, 0, 16, 0, None, 0, 0.5, 1.0, None, None, None,
                           None) == osd.OSD_OK
    # distill_accepted: k < 1, negative B, missing accepted, bad kind / temperature; B = 0 with no count
    fa = lib.osd_distill_accepted
    assert fa(fake, fake, 1, 2, 0, 16, fake, 0, 0.5, 1.0, fake, fake, None, None, None,
              None) == osd.OSD_ERR_INVALID_ARG
    assert fa(fake, fake, 1, -1, 2, 16, fake, 0, 0.5, 1.0, fake, fake, None, None, None,
              None) == osd.OSD_ERR_INVALID_ARG
    assert fa(fake, fake, 1, 2, 2, 16, None, 0, 0.5, 1.0, fake, fake, None, None, None,
              None) == osd.OSD_ERR_INVALID_ARG
    assert fa(fake, fake, 1, 2, 2, 16, fake, 9, 0.5, 1.0, fake, fake, None, None, None,
              None) == osd.OSD_ERR_INVALID_ARG
    assert fa(fake, fake, 1, 2, 2, 16, fake, 0, 0.5, 0.0, fake, fake, None, None, None,
              None) == osd.OSD_ERR_INVALID_ARG
    assert fa(fake, fake, 1, 2, 2, 500000, fake, 0, 0.5, 1.0, fake, fake, None, None, None,
              None) == osd.OSD_ERR_UNSUPPORTED
    assert fa(None, None, 1, 0, 2, 16, None, 0, 0.5, 1.0, None, None, None, None, None,
              None) == osd.OSD_OK
    # tree verification: malformed trees, too many nodes, workspace too small, empty batch
    ft = lib.osd_verify_tree
    P = ctypes.c_int32 * 3
    good, loop, root_kid = P(-1, 0, 1), P(-1, 1, 0), P(0, 0, 1)
    for par in (loop, root_kid):
        assert ft(fake, fake, 1, 2, 3, 16, par, fake, fake, 1.0, fake, fake, fake, fake, None, None, fake,
                  1 << 20, None) == osd.OSD_ERR_INVALID_ARG
    assert ft(fake, fake, 1, 2, 3, 16, good, fake, fake, -1.0, fake, fake, fake, fake, None, None, fake,
              1 << 20, None) == osd.OSD_ERR_INVALID_ARG
    assert ft(fake, fake, 1, 2, 3, 16, good, fake, fake, 1.0, fake, fake, fake, fake, None, None, fake,
              8, None) == osd.OSD_ERR_INVALID_ARG
    P65 = ctypes.c_int32 * 65
    big = P65(-1, *range(64))
    assert ft(fake, fake, 1, 2, 65, 16, big, fake, fake, 1.0, fake, fake, fake, fake, None, None, fake,
              1 << 20, None) == osd.OSD_ERR_UNSUPPORTED
    assert ft(None, None, 1, 0, 3, 16, good, None, None, 1.0, None, None, None, None, None, None, None,
              0, None) == osd.OSD_OK
    n = ctypes.c_size_t(0)
    assert lib.osd_verify_tree_workspace_size(32, 27, 32000, ctypes.byref(n)) == osd.OSD_OK
    assert n.value >= 2 * 32 * 27 * 16 and n.value % 256 == 0
    # the bounded-wait check: null status, zero or huge limit
    assert lib.osd_check_bounded_wait(1000, None, None, None) == osd.OSD_ERR_INVALID_ARG
    assert lib.osd_check_bounded_wait(0, fake, None, None) == osd.OSD_ERR_INVALID_ARG
    assert lib.osd_check_bounded_wait(20_000_000, fake, None, None) == osd.OSD_ERR_INVALID_ARG
    # mixed sampling: beta outside [0, 1], bad temperature, null uniforms, V beyond the limit
    fm = lib.osd_mixed_sample
    assert fm(fake, fake, 1, 2, 16, 16, 16, fake, 1.5, 1.0, fake, None, None, None) == osd.OSD_ERR_INVALID_ARG
    assert fm(fake, fake, 1, 2, 16, 16, 16, fake, 0.5, 0.0, fake, None, None, None) == osd.OSD_ERR_INVALID_ARG
    assert fm(fake, fake, 1, 2, 16, 16, 16, None, 0.5, 1.0, fake, None, None, None) == osd.OSD_ERR_INVALID_ARG
    assert fm(fake, fake, 1, 2, 16, -16, 16, fake, 0.5, 1.0, fake, None, None, None) == osd.OSD_ERR_INVALID_ARG
    assert fm(fake, fake, 1, 2, (1 << 21) + 1, 0, 0, fake, 0.5, 1.0, fake, None, None, None) == osd.OSD_ERR_UNSUPPORTED
    assert fm(None, None, 1, 0, 16, 16, 16, None, 0.5, 1.0, None, None, None, None) == osd.OSD_OK


def test_product_path_fails_loudly_without_library(tmp_path, monkeypatch):
    import paper_2310_07177_gb300 as osd
    monkeypatch.setattr(osd, "LIB_PATH", str(tmp_path / "missing.so"))
    monkeypatch.setattr(osd, "_lib", None)
    with pytest.raises(RuntimeError, match="missing"):
        osd.load_library()
