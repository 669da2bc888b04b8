"""GPU parity of the LLM-side compute controller (Sec. 3.2, Eq. 7):
svl_score_select_paper without gate logits (tokens with z > 0, kappa),
svl_pack_controlled (budget token appended) and svl_controlled_prefill
(prefix layers, gate head, gates on the device, remaining layers).

The gate decisions are taken from float32 logits computed on a bf16 residual
stream, so they are checked in the GPU's own precision: the gates must be
exactly (GPU logit > 0) followed by the oracle's projection applied to the GPU
logits, and the GPU logits must match the oracle's within the bar the bf16
storage itself sets. The forward under those gates must match the oracle's
forward replaying the same gates."""
import numpy as np
import pytest
import torch

from oracle import smartvl_oracle as O
from paper_2607_20357_gb300 import svl, synth
from tests.gpu_common import Case, bar_for, check_selection, l2_err, rel_err

pytestmark = pytest.mark.gpu

if not torch.cuda.is_available():
    pytest.skip("needs a CUDA GPU", allow_module_level=True)

TINY = synth.WORKLOADS["tiny"]


def _case(dims, seed, n_vis, s_text, budgets):
    wl = synth.Workload("ctl", dims, batch=len(n_vis), n_vis=(0, 0), s_text=(1, 1), budgets=(1.0,),
                        gates="bern_heads", features="normal")
    case = Case(dims, wl, seed=seed, batch=None, max_seq=4096)
    b = synth.make_batch(wl, seed, n_vis_list=n_vis, s_text_list=s_text, keep_list=[-1] * len(n_vis),
                         budget_list=budgets)
    case.b_np = O.to_numpy_batch(b)
    case.b = {k: (v.cuda() if isinstance(v, torch.Tensor) else v) for k, v in b.items()}
    return case


@pytest.mark.parametrize("prefix", [1, 0])
def test_controller_gates_and_forward(prefix):
    dims = synth.reduced(TINY.dims, n_layers=4, n_prefix=prefix)
    n_vis = [64, 40, 64, 64, 0]
    s_text = [16, 24, 16, 120, 12]
    budgets = [1.0, 0.7, 0.35, 0.2, 0.5]
    case = _case(dims, 41 + prefix, n_vis, s_text, budgets)
    out = case.model.run(case.b, rule="controller")
    torch.cuda.synchronize()
    assert svl.svl_get_device_status(case.model.handle) == 0
    out = {k: v.cpu() for k, v in out.items()}
    cu = out["cu_seqlens"].numpy()
    kept_off = out["kept_off"].numpy()
    L, G, P = dims.n_layers, dims.n_groups, dims.n_prefix
    seen, compared = 0, 0
    for i in range(len(n_vis)):
        v0, v1 = case.b_np["vis_off"][i], case.b_np["vis_off"][i + 1]
        t0, t1 = case.b_np["text_off"][i], case.b_np["text_off"][i + 1]
        x, ids = case.b_np["vis"][v0:v1], case.b_np["text_ids"][t0:t1]
        ref = O.forward_controlled(dims, case.w_np, x, ids, budgets[i], mode="fp32")
        z_gpu = out["scores"][v0:v1].double().numpy()
        if v1 > v0:
            np.testing.assert_allclose(z_gpu, ref["z"], rtol=1e-4, atol=1e-5)
        # tokens: sigma(z) > 0.5 on the GPU's own logits; kappa
        k = int(out["k"][i])
        assert k == int(np.sum(z_gpu > 0))
        assert abs(float(out["kappa"][i]) - O.survival_rate(z_gpu)) < 1e-6
        assert abs(float(out["kappa"][i]) - ref["kappa"]) < 1e-5
        assert cu[i + 1] - cu[i] == k + (t1 - t0) + 1  # + the budget token
        np.testing.assert_array_equal(out["pos"][cu[i]:cu[i + 1]].numpy(), np.arange(cu[i + 1] - cu[i]))
        # gates: the GPU's logits decide, in its own precision
        lg_gpu = out["gate_logits"][i].double().numpy()[:L - P]
        raw = np.ones((L, G), dtype=np.int64)
        raw[P:] = (lg_gpu > 0).astype(np.int64)
        full = np.zeros((L, G))
        full[P:] = lg_gpu
        want, fl = O.project_gates(dims, budgets[i], v1 - v0, t1 - t0, k, raw, full) if budgets[i] < 1.0 else (raw, 0)
        np.testing.assert_array_equal(out["group_gate"][i].numpy(), want)
        np.testing.assert_array_equal(out["layer_gate"][i].numpy(), want.any(axis=1).astype(np.uint8))
        assert int(out["flags"][i]) == fl
        seen |= fl
        # the GPU's gate logits against the oracle's (bar set by bf16 storage)
        ref16 = O.forward_controlled(dims, case.w_np, x, ids, budgets[i], mode="bf16")
        bar = max(2e-2, 1.5 * rel_err(ref16["gate_logits"], ref["gate_logits"]))
        assert rel_err(lg_gpu, ref["gate_logits"]) < bar, (i, rel_err(lg_gpu, ref["gate_logits"]), bar)
        # the forward under the GPU's gates
        gk = out["kept_idx"][kept_off[i]:kept_off[i + 1]].numpy()
        # on a tie-band swap the oracle runs on the GPU's (valid) kept set
        same = v1 == v0 or check_selection(out["scores"][v0:v1].numpy(), gk,
                                           {"k": k, "kept": O.select_kept(ref["z"], k), "z": ref["z"]})
        kov = None if same else gk
        r32 = O.forward_controlled(dims, case.w_np, x, ids, budgets[i], mode="fp32", keep_count=k, gates_override=want,
                                   kept=kov)
        r16 = O.forward_controlled(dims, case.w_np, x, ids, budgets[i], mode="bf16", keep_count=k, gates_override=want,
                                   kept=kov)
        hid = out["X"][cu[i]:cu[i + 1]].double().numpy()
        assert rel_err(hid, r32["hidden"]) < bar_for(r32, r16, "hidden"), i
        assert l2_err(hid, r32["hidden"]) < bar_for(r32, r16, "hidden", l2_err), i
        assert rel_err(out["logits"][i].double().numpy(), r32["logits"]) < bar_for(r32, r16, "logits"), i
        compared += 1
    assert compared >= 3
    assert seen & O.GROUPS_DROPPED  # the budgets above reach the projection
    case.close()
