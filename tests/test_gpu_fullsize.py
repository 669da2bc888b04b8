"""Parity at the workloads' full sizes, in the launch configuration the
benchmark times (whole batch through the three C entry points), checked on
samples the oracle recomputes one by one.

Hidden states and logits must be within 2e-2 (max-abs and L2 relative) of
the fp32-storage oracle, or within 1.5x the distance between the
bf16-emulated oracle and the fp32-storage oracle where bf16 storage alone
already exceeds 2e-2 (32 layers: about 3.2e-2).

The LLaVA-1.5-7B batch runs with all 32 layers; the Qwen2-VL-7B, video and
mixed-serving batches keep their full batch, sequence and width shapes with
the decoder cut to 2 layers (LLaVA-1.5-13B: 3 layers, one of them a prefix
layer) so the float64 oracle stays within seconds per sample.
"""
import numpy as np
import pytest
import torch

from oracle import smartvl_oracle as O
from paper_2607_20357_gb300 import svl, synth
from tests.gpu_common import bar_for, check_selection, l2_err, numpy_weights_lazy, rel_err, to_device

pytestmark = pytest.mark.gpu

if not torch.cuda.is_available():
    pytest.skip("needs a CUDA GPU", allow_module_level=True)


def _run_full(wl, dims, seed, samples, budget=None, modify=None):
    dev = torch.device("cuda")
    w = synth.make_weights(dims, seed, device=dev)
    batch = synth.make_batch(wl, seed, budget=budget, device=dev, dims=dims)
    if modify:
        modify(batch)
    S_max = int((batch["vis_off"][1:] - batch["vis_off"][:-1] + batch["text_off"][1:] - batch["text_off"][:-1]).max())
    model = svl.GatedPrefill(dims, w, max_seq=S_max + 8)
    out = model.run(batch)
    torch.cuda.synchronize()
    assert svl.svl_get_device_status(model.handle) == 0
    out = {k: v.cpu() for k, v in out.items()}
    w_np = numpy_weights_lazy(w)
    b_np = O.to_numpy_batch(batch)
    errs = []
    for b in samples:
        r = O.forward_batch(dims, w_np, b_np, mode="fp32", samples=[b])[0]
        r16 = O.forward_batch(dims, w_np, b_np, mode="bf16", samples=[b])[0]
        assert int(out["k"][b]) == r["k"]
        assert int(out["flags"][b]) == r["flags"]
        v0, v1 = b_np["vis_off"][b], b_np["vis_off"][b + 1]
        kept = out["kept_idx"][out["kept_off"][b]:out["kept_off"][b + 1]].numpy()
        np.testing.assert_allclose(out["scores"][v0:v1].double().numpy(), r["z"], rtol=1e-4, atol=1e-5)
        if not check_selection(out["scores"][v0:v1].numpy(), kept, r):
            # a tie-band swap: the oracle on the GPU's (valid) kept set
            t0, t1 = b_np["text_off"][b], b_np["text_off"][b + 1]
            args = (dims, w_np, b_np["vis"][v0:v1], b_np["text_ids"][t0:t1], b_np["budget"][b],
                    b_np["layer_gate"][b], b_np["group_gate"][b], int(b_np["keep_count"][b]))
            r = O.forward_sample(*args, mode="fp32", kept=kept)
            r16 = O.forward_sample(*args, mode="bf16", kept=kept)
            print(f"sample {b}: GPU selection differs inside the tie band; compared on the GPU's kept set")
        cu = out["cu_seqlens"].numpy()
        got = {"hidden": out["X"][cu[b]:cu[b + 1]].double().numpy(), "logits": out["logits"][b].double().numpy()}
        for key in ("hidden", "logits"):
            for err in (rel_err, l2_err):
                e, bar = err(got[key], r[key]), bar_for(r, r16, key, err)
                errs.append((b, key, err.__name__, round(e, 5), round(bar, 5)))
                assert e < bar, errs[-1]
    model.close()
    assert errs
    return errs


def test_llava_full_depth_budget_half():
    wl = synth.WORKLOADS["llava"]
    print(_run_full(wl, wl.dims, 1000, samples=[0, 15], budget=0.5))


def test_qwen_full_shapes_two_layers():
    wl = synth.WORKLOADS["qwen"]
    dims = synth.reduced(wl.dims, n_layers=2)
    print(_run_full(wl, dims, 3000, samples=[0, 5]))


def test_video_full_shapes_two_layers():
    wl = synth.WORKLOADS["video"]
    dims = synth.reduced(wl.dims, n_layers=2)
    print(_run_full(wl, dims, 4000, samples=[0, 1], budget=0.25))


def test_mixed_full_batch_two_layers():
    wl = synth.WORKLOADS["mixed"]
    dims = synth.reduced(wl.dims, n_layers=2)
    print(_run_full(wl, dims, 5000, samples=[0, 31, 63]))


def test_llava13b_full_shapes_three_layers_with_prefix():
    """LLaVA-1.5-13B widths (d 5120, 40 heads, FFN 13824) on the full batch,
    the decoder cut to 3 layers of which 1 is a prefix layer (the model has a
    20-layer prefix over 40 layers), with budget-scaled head gates on the
    others."""
    wl = synth.WORKLOADS["llava13b"]
    dims = synth.reduced(wl.dims, n_layers=3, n_prefix=1)

    def gate(batch):
        g = torch.Generator().manual_seed(13)
        batch["group_gate"].copy_((torch.rand(batch["group_gate"].shape, generator=g) < 0.7).to(torch.uint8))

    print(_run_full(wl, dims, 1300, samples=[0, 9], budget=0.5, modify=gate))


class _LazyFp8:
    """Per-layer e4m3 weight codes of the oracle, made when a layer is
    reached (one layer in host memory at a time)."""

    def __init__(self, layers):
        self.layers = layers

    def __getitem__(self, i):
        return O.fp8_layer_weights(self.layers[i])


def test_llava_full_depth_e4m3_budget_half():
    """The e4m3 model (SVL_GEMM_E4M3) at the benchmark's LLaVA-1.5-7B shape --
    the whole batch of 16 through all 32 layers at b = 0.5 -- against the
    oracle's plain e4m3 definition on sample 0: hidden states and logits
    within 2e-2 or 1.5x the definition's own storage sensitivity (its fp8
    forward against fp8_s32), max-abs and L2.

    At this depth the e4m3 codes' rounding (3 mantissa bits) compounds
    through 32 layers of random weights: the definition's two storage
    variants (bf16 or fp32 intermediates) already differ by about 30 %, and
    the GPU lands inside that (about 27-30 % from the fp8 forward). The tight
    e4m3 checks are the per-stage and 2-4 layer tests; this one covers the
    benchmark's launch configuration end to end."""
    wl = synth.WORKLOADS["llava"]
    dims = wl.dims
    dev = torch.device("cuda")
    w = synth.make_weights(dims, 1001, device=dev)
    batch = synth.make_batch(wl, 1001, budget=0.5, device=dev, dims=dims)
    model = svl.GatedPrefill(dims, w, max_seq=700, gemm_format=svl.SVL_GEMM_E4M3)
    out = model.run(batch)
    torch.cuda.synchronize()
    assert svl.svl_get_device_status(model.handle) == 0
    out = {k: v.cpu() for k, v in out.items()}
    model.close()
    w_np = numpy_weights_lazy(w)
    b_np = O.to_numpy_batch(batch)
    b = 0
    v0, v1 = b_np["vis_off"][b], b_np["vis_off"][b + 1]
    t0, t1 = b_np["text_off"][b], b_np["text_off"][b + 1]
    kept = out["kept_idx"][out["kept_off"][b]:out["kept_off"][b + 1]].numpy()
    args = (dims, w_np, b_np["vis"][v0:v1], b_np["text_ids"][t0:t1], b_np["budget"][b], b_np["layer_gate"][b],
            b_np["group_gate"][b], int(b_np["keep_count"][b]))
    qws = _LazyFp8(w_np["layers"])
    r8 = O.forward_sample(*args, mode="fp8", qws=qws)
    assert int(out["k"][b]) == r8["k"]
    np.testing.assert_allclose(out["scores"][v0:v1].double().numpy(), r8["z"], rtol=1e-4, atol=1e-5)
    if not check_selection(out["scores"][v0:v1].numpy(), kept, r8):
        print("sample 0: GPU selection differs inside the tie band; compared on the GPU's kept set")
        r8 = O.forward_sample(*args, mode="fp8", qws=qws, kept=kept)
    r8s = O.forward_sample(*args, mode="fp8_s32", qws=qws, kept=kept)
    cu = out["cu_seqlens"].numpy()
    got = {"hidden": out["X"][cu[b]:cu[b + 1]].double().numpy(), "logits": out["logits"][b].double().numpy()}
    errs = []
    for key in ("hidden", "logits"):
        for err in (rel_err, l2_err):
            e, bar = err(got[key], r8[key]), max(2e-2, 1.5 * err(r8s[key], r8[key]))
            errs.append((key, err.__name__, round(e, 5), round(bar, 5)))
            assert e < bar, errs[-1]
    print(errs)
