"""Failure detection without faulting the GPU: host-made failures (NaN
inputs, out-of-range ids) and a device wait that is made to run out must be
reported through the status word while the context stays usable."""
import numpy as np
import pytest
import torch

from paper_2607_20357_gb300 import svl, synth
from tests.gpu_common import Case

pytestmark = pytest.mark.gpu

if not torch.cuda.is_available():
    pytest.skip("needs a CUDA GPU", allow_module_level=True)

TINY = synth.WORKLOADS["tiny"]


@pytest.fixture()
def case():
    c = Case(TINY.dims, TINY, seed=0)
    yield c
    c.close()


def test_bounded_wait_reports_timeout_and_context_survives(case):
    assert svl.svl_get_device_status(case.model.handle) == 0
    svl.svl_selftest_wait_timeout(case.model.handle, 200000)
    torch.cuda.synchronize()
    assert svl.svl_get_device_status(case.model.handle) & svl.SVL_DEV_TIMEOUT
    # the status word was cleared by the read; a normal run still works
    out = case.run()
    assert int(out["k"][0]) == 32


def test_nan_feature_sets_nonfinite(case):
    case.b["vis"][3, 7] = float("nan")
    out = case.model.run(case.b, stages=("select",))
    torch.cuda.synchronize()
    assert svl.svl_get_device_status(case.model.handle) & svl.SVL_DEV_NONFINITE
    assert int(out["k"][0]) == 32


def test_out_of_range_text_id_sets_bad_index(case):
    case.b["text_ids"][0] = TINY.dims.vocab + 5
    out = case.model.run(case.b, stages=("select", "pack"))
    torch.cuda.synchronize()
    assert svl.svl_get_device_status(case.model.handle) & svl.SVL_DEV_BAD_INDEX
    k = int(out["k"][0])
    assert torch.count_nonzero(out["X"][k]).item() == 0  # the bad row is zero-filled
