"""Shared pytest setup: the `gpu` marker and access to the oracle and the CUDA library."""
import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (GB300, sm_103a)")
    config.addinivalue_line("markers", "expect_index_checks: makes the checked build's index "
                                       "checks fire on purpose")


def pytest_collection_modifyitems(config, items):
    have_gpu = False
    try:
        import torch
        have_gpu = torch.cuda.is_available()
    except Exception:
        pass
    if have_gpu:
        return
    skip = pytest.mark.skip(reason="no CUDA device")
    for item in items:
        if "gpu" in item.keywords:
            item.add_marker(skip)


@pytest.fixture(scope="session")
def oracle_mod():
    import oracle
    oracle.lib()
    return oracle


@pytest.fixture(scope="session")
def grpo():
    import paper_2609_36932_gb300 as g
    g.lib()
    return g


@pytest.fixture(autouse=True)
def _checked_build_report(request):
    """With FASTRL_GRPO_CHECKED=1 (the checked build, see tests/test_gpu_checked_build.py), every
    GPU test must leave the device index checks silent."""
    yield
    if os.environ.get("FASTRL_GRPO_CHECKED") != "1" or "gpu" not in request.keywords:
        return
    if request.node.get_closest_marker("expect_index_checks") is not None:
        return
    import paper_2609_36932_gb300 as g
    assert b"checked" in g.lib().grpo_version()
    mask, site = g.grpo_debug_checks(reset=True)
    assert mask == 0, "index check failed in file bit mask 0x%x, first at file %d line %d" % (
        mask, site // 100000, site % 100000)
