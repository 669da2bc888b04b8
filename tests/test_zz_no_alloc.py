"""svl_score_select_noalloc: the token controller for callers that cannot
allocate device memory for a workspace (stream capture, a host framework that
owns all device memory, real-time paths). It must give the same results as
svl_score_select with a workspace, call after call, although every call
reuses the library's one fixed scratch array.

This file is collected last on purpose: if it fails, every other test of a
run that stops at the first failure has already run.
"""
import numpy as np
import pytest
import torch

from paper_2607_20357_gb300 import svl, synth
from tests.gpu_common import to_device

pytestmark = pytest.mark.gpu

if not torch.cuda.is_available():
    pytest.skip("needs a CUDA GPU", allow_module_level=True)

LLAVA = synth.WORKLOADS["llava"]


def _outputs(B, nv, dev, fill):
    i32 = dict(dtype=torch.int32, device=dev)
    return {"scores": torch.full((max(nv, 1),), float(fill), dtype=torch.float32, device=dev),
            "k": torch.full((B,), fill, **i32), "kept_idx": torch.full((max(nv, 1),), fill, **i32),
            "kept_off": torch.full((B + 1,), fill, **i32), "flags": torch.full((B,), fill, **i32)}


def _call(model, batch, out, workspace=None):
    B, nv = batch["B"], batch["vis"].shape[0]
    text_len = (batch["text_off"][1:] - batch["text_off"][:-1]).contiguous()
    args = (model.handle, B, nv, batch["vis"], batch["vis_off"], text_len, batch["budget"], batch["keep_count"],
            batch["layer_gate"], batch["group_gate"], out["scores"], out["k"], out["kept_idx"], out["kept_off"],
            out["flags"])
    if workspace is None:
        svl.svl_score_select_noalloc(*args)
    else:
        svl.svl_score_select(*args, workspace[0], workspace[1])


@pytest.fixture(scope="module")
def model():
    dims = synth.reduced(LLAVA.dims, n_layers=1)
    w = to_device(synth.make_weights(dims, 21))
    m = svl.GatedPrefill(dims, w, max_seq=1024)
    yield m
    m.close()


def test_noalloc_matches_workspace_entry_on_consecutive_calls(model):
    dev = torch.device("cuda")
    batches = [
        synth.make_batch(LLAVA, 31, budget=0.5, device=dev, dims=model.dims),
        synth.make_batch(LLAVA, 32, device=dev, dims=model.dims, n_vis_list=[576, 0, 33, 576, 300],
                         s_text_list=[64, 8, 1, 200, 17], keep_list=[-1, -1, 5, 100, -1],
                         budget_list=[0.3, 1.0, 1.0, 0.9, 0.05]),
    ]
    for batch in batches:
        B, nv, nt = batch["B"], batch["vis"].shape[0], batch["text_ids"].shape[0]
        ref = _outputs(B, nv, dev, -3)
        got = _outputs(B, nv, dev, -7)
        _call(model, batch, ref, workspace=model.workspace(B, nv, nt))
        _call(model, batch, got)
        torch.cuda.synchronize()
        assert svl.svl_get_device_status(model.handle) == 0
        total = int(ref["kept_off"][-1])
        np.testing.assert_allclose(got["scores"][:nv].cpu().numpy(), ref["scores"][:nv].cpu().numpy(),
                                   rtol=1e-4, atol=1e-5)
        for key in ("k", "kept_off", "flags"):
            np.testing.assert_array_equal(got[key].cpu().numpy(), ref[key].cpu().numpy())
        np.testing.assert_array_equal(got["kept_idx"][:total].cpu().numpy(), ref["kept_idx"][:total].cpu().numpy())


def test_noalloc_rejects_sizes_beyond_its_array(model):
    dev = torch.device("cuda")
    batch = synth.make_batch(LLAVA, 33, budget=0.5, batch=2, device=dev, dims=model.dims)
    out = _outputs(257, 70000, dev, 0)
    big = dict(batch, B=257)
    with pytest.raises(svl.SvlError) as e:
        _call(model, big, out)
    assert e.value.code == 2  # SVL_ERR_SHAPE
    text_len = (batch["text_off"][1:] - batch["text_off"][:-1]).contiguous()
    with pytest.raises(svl.SvlError) as e:
        svl.svl_score_select_noalloc(model.handle, 2, 65537, batch["vis"], batch["vis_off"], text_len,
                                     batch["budget"], None, batch["layer_gate"], batch["group_gate"],
                                     out["scores"], out["k"], out["kept_idx"], out["kept_off"], out["flags"])
    assert e.value.code == 2
