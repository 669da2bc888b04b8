"""GPU parity of gated decode with a KV cache (svl_gated_prefill_kv,
svl_decode_step) against the oracle's cache-free definition: after feeding
tokens t_1..t_n, the logits are those of the prefill forward over the prompt
extended by t_1..t_n under the same gates (oracle ``decode_reference``). The
fed tokens are fixed in advance (teacher forcing), so a near-tie in a greedy
choice cannot make the two sides diverge; the greedy next token is checked
against the GPU's own logits."""
import numpy as np
import pytest
import torch

from oracle import smartvl_oracle as O
from paper_2607_20357_gb300 import svl, synth
from tests.gpu_common import Case, bar_for, check_selection, rel_err

pytestmark = pytest.mark.gpu

if not torch.cuda.is_available():
    pytest.skip("needs a CUDA GPU", allow_module_level=True)

TINY = synth.WORKLOADS["tiny"]


def _decode(dims, wl, seed, n_vis, s_text, budgets, steps, max_len):
    case = Case(dims, wl, seed=seed, batch=None, max_seq=max(max_len, 256))
    b = synth.make_batch(wl, seed, n_vis_list=n_vis, s_text_list=s_text, keep_list=[-1] * len(n_vis),
                         budget_list=budgets, dims=dims)
    g = torch.Generator().manual_seed(seed)
    B, L, G = len(n_vis), dims.n_layers, dims.n_groups
    b["group_gate"] = (torch.rand(B, L, G, generator=g) < 0.7).to(torch.uint8)
    b["layer_gate"] = torch.ones(B, L, dtype=torch.uint8)
    b["layer_gate"][0, L - 1] = 0  # sample 0 skips the last layer
    case.b_np = O.to_numpy_batch(b)
    case.b = {k: (v.cuda() if isinstance(v, torch.Tensor) else v) for k, v in b.items()}
    m = case.model
    out = m.run(case.b, stages=("select", "pack"))
    nv, nt = int(case.b["vis"].shape[0]), int(case.b["text_ids"].shape[0])
    ws, wsb = m.workspace(B, nv, nt, "cuda", ("prefill",))
    kv = torch.empty(svl.svl_kv_cache_size(m.handle, B, max_len), dtype=torch.uint8, device="cuda")
    cache_len = torch.zeros(B, dtype=torch.int32, device="cuda")
    svl.svl_gated_prefill_kv(m.handle, B, nv + nt, out["X"], out["cu_seqlens"], out["pos"], case.b["layer_gate"],
                             case.b["group_gate"], svl.SVL_LOGITS_LAST, out["logits"], kv, max_len, cache_len, ws, wsb)
    prompt_logits = out["logits"].clone()
    prompt_len = cache_len.clone()
    dws = torch.empty(svl.svl_decode_workspace_size(m.handle, B), dtype=torch.uint8, device="cuda")
    fed = torch.randint(0, dims.vocab, (steps, B), generator=g, dtype=torch.int32)
    logits = torch.empty(B, dims.vocab, dtype=torch.float32, device="cuda")
    nxt = torch.empty(B, dtype=torch.int32, device="cuda")
    step_logits, step_next = [], []
    for t in range(steps):
        svl.svl_decode_step(m.handle, B, fed[t].cuda(), kv, max_len, cache_len, case.b["layer_gate"],
                            case.b["group_gate"], logits, nxt, dws, dws.numel())
        step_logits.append(logits.cpu().clone())
        step_next.append(nxt.cpu().clone())
    torch.cuda.synchronize()
    assert svl.svl_get_device_status(m.handle) == 0
    res = dict(out={k: v.cpu() for k, v in out.items()}, prompt_logits=prompt_logits.cpu(),
               prompt_len=prompt_len.cpu(), cache_len=cache_len.cpu(), fed=fed, logits=step_logits, next=step_next)
    return case, res


@pytest.mark.parametrize("prefix", [0, 1])
def test_decode_steps_match_extended_prefill(prefix):
    dims = synth.reduced(TINY.dims, n_layers=4, n_prefix=prefix)
    n_vis, s_text, budgets = [64, 40, 64], [16, 9, 30], [0.8, 1.0, 0.5]
    steps = 5
    case, r = _decode(dims, TINY, 61 + prefix, n_vis, s_text, budgets, steps, max_len=160)
    out = r["out"]
    cu = out["cu_seqlens"].numpy()
    np.testing.assert_array_equal(r["prompt_len"].numpy(), np.diff(cu))
    np.testing.assert_array_equal(r["cache_len"].numpy(), np.diff(cu) + steps)
    compared = 0
    for i in range(len(n_vis)):
        v0, v1 = case.b_np["vis_off"][i], case.b_np["vis_off"][i + 1]
        t0, t1 = case.b_np["text_off"][i], case.b_np["text_off"][i + 1]
        args = (dims, case.w_np, case.b_np["vis"][v0:v1], case.b_np["text_ids"][t0:t1], budgets[i],
                case.b_np["layer_gate"][i], case.b_np["group_gate"][i], r["fed"][:, i].numpy())
        f32, s32 = O.decode_reference(*args, mode="fp32")
        f16, s16 = O.decode_reference(*args, mode="bf16")
        kept = out["kept_idx"][out["kept_off"][i]:out["kept_off"][i + 1]].numpy()
        if not check_selection(out["scores"][v0:v1].numpy(), kept, f32):
            # a tie-band swap: the oracle on the GPU's (valid) kept set
            f32, s32 = O.decode_reference(*args, mode="fp32", kept=kept)
            f16, s16 = O.decode_reference(*args, mode="bf16", kept=kept)
        assert rel_err(r["prompt_logits"][i].double().numpy(), f32["logits"]) < bar_for(f32, f16, "logits")
        for t in range(steps):
            got = r["logits"][t][i].double().numpy()
            e, bar = rel_err(got, s32[t]["logits"]), bar_for(s32[t], s16[t], "logits")
            assert e < bar, (i, t, e, bar)
            assert int(r["next"][t][i]) == int(np.argmax(r["logits"][t][i].numpy()))
        compared += 1
    assert compared >= 2
    case.close()


def test_decode_llava_width_two_layers():
    """LLaVA-7B widths (d 4096, 32 heads of 128), 2 layers, 2 samples, 3 steps."""
    wl = synth.WORKLOADS["llava"]
    dims = synth.reduced(wl.dims, n_layers=2)
    case, r = _decode(dims, wl, 71, [576, 576], [64, 64], [0.5, 0.25], 3, max_len=700)
    out = r["out"]
    for i in range(2):
        v0, v1 = case.b_np["vis_off"][i], case.b_np["vis_off"][i + 1]
        t0, t1 = case.b_np["text_off"][i], case.b_np["text_off"][i + 1]
        args = (dims, case.w_np, case.b_np["vis"][v0:v1], case.b_np["text_ids"][t0:t1], [0.5, 0.25][i],
                case.b_np["layer_gate"][i], case.b_np["group_gate"][i], r["fed"][:, i].numpy())
        f32, s32 = O.decode_reference(*args, mode="fp32")
        f16, s16 = O.decode_reference(*args, mode="bf16")
        kept = out["kept_idx"][out["kept_off"][i]:out["kept_off"][i + 1]].numpy()
        if not check_selection(out["scores"][v0:v1].numpy(), kept, f32):
            # a tie-band swap: the oracle on the GPU's (valid) kept set
            f32, s32 = O.decode_reference(*args, mode="fp32", kept=kept)
            f16, s16 = O.decode_reference(*args, mode="bf16", kept=kept)
        for t in range(3):
            got = r["logits"][t][i].double().numpy()
            assert rel_err(got, s32[t]["logits"]) < bar_for(s32[t], s16[t], "logits"), (i, t)
    case.close()


def test_decode_past_full_cache_saturates():
    """Stepping a batch past max_len: a sample whose cache is full takes no
    step -- its length stays at max_len, its next token is -1 -- and the
    status word reports SVL_DEV_BAD_INDEX, while the other samples keep
    decoding as before (their logits equal those of a run that never hit
    the limit)."""
    dims = synth.reduced(TINY.dims, n_layers=2)
    n_vis, s_text = [40, 20], [10, 6]
    wl = TINY
    case = Case(dims, wl, seed=75, batch=None, max_seq=256)
    b = synth.make_batch(wl, 75, n_vis_list=n_vis, s_text_list=s_text, keep_list=[-1, -1], budget_list=[1.0, 1.0],
                         dims=dims)
    B = 2
    b["group_gate"] = torch.ones(B, dims.n_layers, dims.n_groups, dtype=torch.uint8)
    b["layer_gate"] = torch.ones(B, dims.n_layers, dtype=torch.uint8)
    bd = {k: (v.cuda() if isinstance(v, torch.Tensor) else v) for k, v in b.items()}
    m = case.model
    fed = torch.randint(0, dims.vocab, (5, B), generator=torch.Generator().manual_seed(76), dtype=torch.int32)

    def run(max_len):
        out = m.run(bd, stages=("select", "pack"))
        nv, nt = int(bd["vis"].shape[0]), int(bd["text_ids"].shape[0])
        ws, wsb = m.workspace(B, nv, nt, "cuda", ("prefill",))
        kv = torch.zeros(svl.svl_kv_cache_size(m.handle, B, max_len), dtype=torch.uint8, device="cuda")
        cache_len = torch.zeros(B, dtype=torch.int32, device="cuda")
        svl.svl_gated_prefill_kv(m.handle, B, nv + nt, out["X"], out["cu_seqlens"], out["pos"], bd["layer_gate"],
                                 bd["group_gate"], svl.SVL_LOGITS_LAST, out["logits"], kv, max_len, cache_len, ws, wsb)
        dws = torch.empty(svl.svl_decode_workspace_size(m.handle, B), dtype=torch.uint8, device="cuda")
        logits = torch.empty(B, dims.vocab, dtype=torch.float32, device="cuda")
        nxt = torch.empty(B, dtype=torch.int32, device="cuda")
        lens, nexts, lg = [], [], []
        for t in range(fed.shape[0]):
            svl.svl_decode_step(m.handle, B, fed[t].cuda(), kv, max_len, cache_len, bd["layer_gate"],
                                bd["group_gate"], logits, nxt, dws, dws.numel())
            lens.append(cache_len.cpu().clone())
            nexts.append(nxt.cpu().clone())
            lg.append(logits.cpu().clone())
        torch.cuda.synchronize()
        return np.diff(out["cu_seqlens"].cpu().numpy()), lens, nexts, lg

    prompt, lens_ok, _, lg_ok = run(128)  # never full
    assert svl.svl_get_device_status(m.handle) == 0
    full = int(prompt.max())
    assert prompt[0] == full > prompt[1]
    max_len = full + 2  # sample 0 fills after two steps
    _, lens, nexts, lg = run(max_len)
    status = svl.svl_get_device_status(m.handle)
    assert status & svl.SVL_DEV_BAD_INDEX, status
    for t in range(fed.shape[0]):
        assert int(lens[t][0]) == min(full + t + 1, max_len)
        assert int(lens[t][1]) == prompt[1] + t + 1
        if full + t >= max_len:
            assert int(nexts[t][0]) == -1
        else:
            assert int(nexts[t][0]) >= 0
        # the sample that still has room decodes exactly as without the limit
        np.testing.assert_array_equal(lg[t][1].numpy(), lg_ok[t][1].numpy())
    case.close()
