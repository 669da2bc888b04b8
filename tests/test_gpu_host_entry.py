"""GPU parity of the host-buffer entry point (svl_prefill_from_host): pinned
host inputs in, last-row logits and k out, through the C ABI, with the
host-to-device and device-to-host copies inside the call.

Bars:
- k is bit-exact against the oracle (integer budget arithmetic) and against
  the device-resident path (svl_score_select, svl_pack and svl_gated_prefill
  on device inputs, the same kernels).
- Logits are within 1e-3 (relative) of the device-resident path, and within
  the end-to-end bar of the oracle (2e-2, or 1.5x the bf16-storage drift).
- Two calls enqueued back to back on one stream and one workspace, with
  different batches and no host wait in between, each give the result of the
  same call made alone.
"""
import pytest
import torch

from oracle import smartvl_oracle as O
from paper_2607_20357_gb300 import svl, synth
from tests.gpu_common import Case, bar_for, check_selection, rel_err

pytestmark = pytest.mark.gpu

if not torch.cuda.is_available():
    pytest.skip("needs a CUDA GPU", allow_module_level=True)

TINY = synth.WORKLOADS["tiny"]
LLAVA = synth.WORKLOADS["llava"]


def _pinned(batch, dims):
    h = {k: (v.detach().cpu().pin_memory() if isinstance(v, torch.Tensor) else v) for k, v in batch.items()}
    h["logits"] = torch.zeros(batch["B"], dims.vocab, dtype=torch.float32).pin_memory()
    h["k"] = torch.full((batch["B"],), -1, dtype=torch.int32).pin_memory()
    return h


def _sizes(h):
    return h["B"], int(h["vis"].shape[0]), int(h["text_ids"].shape[0])


def _workspace(model, h):
    need = svl.svl_host_workspace_size(model.handle, *_sizes(h))
    return torch.empty(need, dtype=torch.uint8, device="cuda"), need


def _call(model, h, ws, need, stream):
    B, nv, nt = _sizes(h)
    svl.svl_prefill_from_host(model.handle, B, nv, nt, h["vis"], h["vis_off"], h["text_ids"], h["text_off"],
                              h["budget"], h["keep_count"], h["layer_gate"], h["group_gate"], h["logits"], h["k"],
                              ws, need, stream)


def _check_oracle(case, out, logits, k):
    """k bit-exact; logits within the end-to-end bar, on the GPU's kept set
    where the selection differs inside the tie band."""
    ref = case.oracle("fp32")
    ref16 = case.oracle("bf16")
    bn = case.b_np
    kept_off = out["kept_off"].numpy()
    for b in range(bn["B"]):
        r, r16 = ref[b], ref16[b]
        assert int(k[b]) == r["k"], (b, int(k[b]), r["k"])
        v0, v1 = bn["vis_off"][b], bn["vis_off"][b + 1]
        kept = out["kept_idx"][kept_off[b]:kept_off[b + 1]].numpy()
        if not check_selection(out["scores"][v0:v1].numpy(), kept, r):
            t0, t1 = bn["text_off"][b], bn["text_off"][b + 1]
            args = (case.dims, case.w_np, bn["vis"][v0:v1], bn["text_ids"][t0:t1], bn["budget"][b],
                    bn["layer_gate"][b], bn["group_gate"][b], int(bn["keep_count"][b]))
            r = O.forward_sample(*args, mode="fp32", kept=kept)
            r16 = O.forward_sample(*args, mode="bf16", kept=kept)
        e = rel_err(logits[b].double().numpy(), r["logits"])
        assert e < bar_for(r, r16, "logits"), (b, e)


def test_host_entry_matches_device_path_and_oracle():
    case = Case(TINY.dims, TINY, seed=11, batch=3)
    out = case.run()  # device-resident path (also the source of the kept sets)
    h = _pinned(case.b, case.dims)
    ws, need = _workspace(case.model, h)
    stream = torch.cuda.current_stream()
    _call(case.model, h, ws, need, stream)
    torch.cuda.synchronize()
    assert svl.svl_get_device_status(case.model.handle) == 0
    assert torch.equal(h["k"], out["k"].to(torch.int32)), (h["k"], out["k"])
    e = rel_err(h["logits"].double().numpy(), out["logits"].double().numpy())
    assert e < 1e-3, e
    _check_oracle(case, out, h["logits"], h["k"])
    case.close()


def test_host_entry_back_to_back_calls():
    """Two batches (different features, budgets 0.3 and 0.9) enqueued one
    after the other on the same stream and workspace before the host waits;
    each must equal the same call made alone."""
    dims = TINY.dims
    case = Case(dims, TINY, seed=21, batch=3)
    # different features and budgets, the same sizes (64 visual + 16 text tokens per sample)
    batches = [synth.make_batch(TINY, 21 + i, budget=bud, batch=3) for i, bud in enumerate((0.3, 0.9))]
    hosts = [_pinned(b, dims) for b in batches]
    assert _sizes(hosts[0]) == _sizes(hosts[1])
    ws, need = _workspace(case.model, hosts[0])
    stream = torch.cuda.current_stream()
    alone = []
    for h in hosts:
        _call(case.model, h, ws, need, stream)
        torch.cuda.synchronize()
        alone.append((h["k"].clone(), h["logits"].clone()))
        h["k"].fill_(-1)
        h["logits"].zero_()
    for h in hosts:
        _call(case.model, h, ws, need, stream)
    torch.cuda.synchronize()
    assert svl.svl_get_device_status(case.model.handle) == 0
    for h, (k, logits) in zip(hosts, alone):
        assert torch.equal(h["k"], k)
        assert torch.equal(h["logits"], logits)
    # the two batches hold different features, so their results differ
    assert not torch.equal(alone[0][1], alone[1][1])
    case.close()


def test_host_entry_llava_shapes_two_layers():
    """LLaVA-7B widths and the benchmark batch (16 x (576 + 64) tokens), two
    decoder layers: the host entry point against the device-resident path
    (whose parity with the oracle the full-size tests establish)."""
    wl = synth.dataclasses.replace(LLAVA, dims=synth.reduced(LLAVA.dims, n_layers=2))
    dims = wl.dims
    w = synth.make_weights(dims, 3, device="cuda")
    model = svl.GatedPrefill(dims, w, max_seq=wl.n_vis[1] + wl.s_text[1] + 64)
    for bud in (0.25, 1.0):
        b = synth.make_batch(wl, 3, budget=bud, device="cuda")
        out = model.run(b)
        torch.cuda.synchronize()
        h = _pinned(b, dims)
        ws, need = _workspace(model, h)
        _call(model, h, ws, need, torch.cuda.current_stream())
        torch.cuda.synchronize()
        assert svl.svl_get_device_status(model.handle) == 0
        assert torch.equal(h["k"], out["k"].cpu().to(torch.int32))
        e = rel_err(h["logits"].double().numpy(), out["logits"].cpu().double().numpy())
        assert e < 1e-3, (bud, e)
    model.close()
