"""The per-kernel timing calls (svl_profile_start / svl_profile_stop /
svl_profile_launches) behind the bench's per-kernel figures: within a window
every kernel launch of a profiled tag gets one record, the records add up to
the library's own launch counter, each tag's total is the sum of its
launches, and a tag mask records only the masked-in kernels."""
import pytest
import torch

from paper_2607_20357_gb300 import svl, synth

pytestmark = pytest.mark.gpu

if not torch.cuda.is_available():
    pytest.skip("needs a CUDA GPU", allow_module_level=True)

TINY = synth.WORKLOADS["tiny"]
DECODER_TAGS = ("qkv_gemm", "attention", "o_gemm", "gateup_gemm", "down_gemm")


def test_profile_window_records_every_launch():
    dims = TINY.dims
    w = synth.make_weights(dims, 4, device="cuda")
    model = svl.GatedPrefill(dims, w, max_seq=1024)
    b = synth.make_batch(TINY, 4, batch=3, device="cuda")
    model.run(b)  # the first launches configure the kernels
    torch.cuda.synchronize()

    n0 = svl.svl_launch_count()
    svl.svl_profile_start(model.handle)
    model.run(b)
    per_tag = svl.svl_profile_stop(model.handle)
    n1 = svl.svl_launch_count()
    launches = svl.svl_profile_launches(model.handle)
    assert svl.svl_get_device_status(model.handle) == 0

    assert sum(c for c, _ in per_tag.values()) == n1 - n0 == len(launches) > 0
    for tag in ("budget_embed", "score", "select", "pack", "schedule", "lm_head") + DECODER_TAGS:
        assert tag in per_tag, (tag, sorted(per_tag))
    for tag in DECODER_TAGS:  # one launch per layer, whatever the gates
        assert per_tag[tag][0] == dims.n_layers, (tag, per_tag[tag])
    for tag, (count, total) in per_tag.items():
        times = [ms for name, ms in launches if name == tag]
        assert len(times) == count
        assert all(ms > 0 for ms in times), (tag, times)
        assert abs(sum(times) - total) <= 1e-3 * max(total, 1e-3), (tag, sum(times), total)

    # a mask: only the attention launches are recorded, and profiling is off
    # again after the stop
    svl.svl_profile_start(model.handle, tags=["attention"])
    model.run(b)
    per_tag = svl.svl_profile_stop(model.handle)
    assert set(per_tag) == {"attention"} and per_tag["attention"][0] == dims.n_layers
    assert [name for name, _ in svl.svl_profile_launches(model.handle)] == ["attention"] * dims.n_layers
    model.run(b)
    torch.cuda.synchronize()
    assert len(svl.svl_profile_launches(model.handle)) == dims.n_layers  # still the last window's
    model.close()
