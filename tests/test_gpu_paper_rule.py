"""GPU parity of the paper's own inference rule (svl_score_select_paper):
sigma(z) > 0.5 tokens, gates from the compute controller's logits, and the
budget projection with its head-group fallback (Sec. 3.1, Sec. 3.3).

k, the flags and the projected gates are integers decided from float32
logits, so the oracle's rule is applied to the GPU's own logits (the same
precision) and must agree bit for bit; the logits themselves match the
oracle's float64 ones to 1e-4, and the kept sets agree outside the 1e-4 tie
band. The prefill driven by the projected gates matches the oracle's forward
under the same gates."""
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


def _case(seed, n_vis, s_text, keep, budgets, dims):
    wl = synth.Workload("rule", dims, batch=len(n_vis), n_vis=(0, 0), s_text=(1, 1), budgets=(1.0,),
                        gates="bern_heads", features="normal")
    case = Case(dims, wl, seed=seed, batch=None, max_seq=4096)
    b = synth.make_batch(wl, seed, n_vis_list=n_vis, s_text_list=s_text, keep_list=keep, budget_list=budgets)
    g = torch.Generator().manual_seed(seed + 1)
    b["gate_logits"] = torch.randn(len(n_vis), dims.n_layers, dims.n_groups, generator=g)
    case.b_np = O.to_numpy_batch(b)
    case.b = {k: (v.cuda() if isinstance(v, torch.Tensor) else v) for k, v in b.items()}
    return case


def test_paper_rule_select_and_gates():
    dims = synth.reduced(TINY.dims, n_layers=4, n_prefix=1)
    n_vis = [64, 64, 64, 64, 200, 0, 32, 64]
    s_text = [16, 16, 16, 200, 300, 8, 4, 16]
    keep = [-1, -1, -1, -1, -1, -1, 5, -1]
    budgets = [1.0, 0.5, 0.2, 0.05, 0.01, 0.3, 0.5, 0.9]
    case = _case(21, n_vis, s_text, keep, budgets, dims)
    out = case.model.run(case.b, stages=("select",), rule="paper")
    torch.cuda.synchronize()
    assert svl.svl_get_device_status(case.model.handle) == 0
    out = {k: v.cpu() for k, v in out.items()}
    kept_off = out["kept_off"].numpy()
    seen = 0
    for i in range(len(n_vis)):
        v0, v1 = case.b_np["vis_off"][i], case.b_np["vis_off"][i + 1]
        logits = case.b_np["gate_logits"][i]
        z, k_ref, fl_ref, kept_ref, gates_ref = O.paper_rule_sample(dims, case.w_np, case.b_np["vis"][v0:v1],
                                                                    budgets[i], s_text[i], logits, keep[i])
        z_gpu = out["scores"][v0:v1].double().numpy()
        if v1 > v0:
            np.testing.assert_allclose(z_gpu, z, rtol=1e-4, atol=1e-5)
        # the same decision on the GPU's own float32 logits
        k_own, fl_own, gates_own = O.paper_rule_counts(dims, budgets[i], v1 - v0, s_text[i], z_gpu, logits, keep[i])
        assert int(out["k"][i]) == k_own, (i, int(out["k"][i]), k_own)
        assert int(out["flags"][i]) == fl_own, (i, int(out["flags"][i]), fl_own)
        np.testing.assert_array_equal(out["group_gate"][i].numpy(), gates_own)
        np.testing.assert_array_equal(out["layer_gate"][i].numpy(), gates_own.any(axis=1).astype(np.uint8))
        assert (k_own, fl_own) == (k_ref, fl_ref) and (gates_own == gates_ref).all()
        gk = out["kept_idx"][kept_off[i]:kept_off[i + 1]].numpy()
        if v1 > v0:
            check_selection(out["scores"][v0:v1].numpy(), gk, {"k": k_ref, "kept": kept_ref, "z": z})
        seen |= fl_ref
    # the cases above reach the group fallback and the over-budget flag
    assert seen & O.GROUPS_DROPPED and seen & O.OVER_BUDGET
    case.close()


def test_paper_rule_end_to_end_prefill():
    """The projected gates drive svl_gated_prefill: hidden states and logits
    match the oracle's forward under the same tokens and gates."""
    dims = synth.reduced(TINY.dims, n_layers=4, n_prefix=1)
    n_vis = [64, 48, 64]
    s_text = [16, 24, 120]
    budgets = [0.9, 0.4, 0.08]
    case = _case(33, n_vis, s_text, [-1, -1, -1], budgets, dims)
    out = case.model.run(case.b, rule="paper")
    torch.cuda.synchronize()
    assert svl.svl_get_device_status(case.model.handle) == 0
    out = {k: v.cpu() for k, v in out.items()}
    cu = out["cu_seqlens"].numpy()
    kept_off = out["kept_off"].numpy()
    for i in range(len(n_vis)):
        v0, v1 = case.b_np["vis_off"][i], case.b_np["vis_off"][i + 1]
        t0, t1 = case.b_np["text_off"][i], case.b_np["text_off"][i + 1]
        z, k, fl, kept, gates = O.paper_rule_sample(dims, case.w_np, case.b_np["vis"][v0:v1], budgets[i],
                                                    t1 - t0, case.b_np["gate_logits"][i])
        gk = out["kept_idx"][kept_off[i]:kept_off[i + 1]].numpy()
        # on a tie-band swap the oracle runs on the GPU's (valid) kept set
        same = check_selection(out["scores"][v0:v1].numpy(), gk, {"k": k, "kept": kept, "z": z})
        lg = np.ones(dims.n_layers, dtype=np.uint8)
        refs = {}
        for mode in ("fp32", "bf16"):
            # keep_count = k keeps the same top-k set; the projected gates drive the layers
            refs[mode] = O.forward_sample(dims, case.w_np, case.b_np["vis"][v0:v1], case.b_np["text_ids"][t0:t1],
                                          budgets[i], lg, gates, keep_count=k, mode=mode,
                                          kept=None if same else gk)
            np.testing.assert_array_equal(refs[mode]["kept"], kept if same else gk)
        hid = out["X"][cu[i]:cu[i + 1]].double().numpy()
        assert rel_err(hid, refs["fp32"]["hidden"]) < bar_for(refs["fp32"], refs["bf16"], "hidden")
        assert rel_err(out["logits"][i].double().numpy(), refs["fp32"]["logits"]) < \
            bar_for(refs["fp32"], refs["bf16"], "logits")
    case.close()
