"""GPU parity of the e4m3 (FP8) gated projections against the oracle's
``fp8`` mode: per-row e4m3 quantisation bit for bit (svl_quantize_rows_e4m3),
then the prefill and decode with SVL_GEMM_E4M3 models.

The quantised codes and scales are integer and float decisions taken in
float32 on both sides from the same bf16 inputs, so they must agree exactly.
The e4m3 GEMM on its own (svl_gemm_e4m3) must equal the exact product of
the decoded codes times both scales to float32 accumulation error.

The forward compares with the oracle's plain fp8 definition: e4m3 of
RMSNorm(X) * gain (QKV, gate/up), of the attention output (O) and of the
SwiGLU output (down) against e4m3 of W as given, per row. An activation is
quantised from values the GPU computes in float32 with bf16 storage and
the oracle in float64: where the two differ by a bf16 step, a value can sit
on opposite sides of an e4m3 rounding boundary and jump by a whole e4m3 step
(6-12 %). The end-to-end bar is therefore 1.5x the distance between the
oracle's fp8 forward with bf16 storage and with fp32 storage (the same
definition under storage-level perturbation), at least 2e-2. The layers'
update of the residual stream (final hidden minus the packed input rows)
must lie within 1.5x that storage sensitivity measured on the update itself
(at these small widths bf16 storage alone moves the update by 5-7 %), and
closer to the fp8 definition's update than to the bf16 one's, which shows the
e4m3 arithmetic is what ran. Per-stage checks at LLaVA-7B width
(tests/test_gpu_stages.py) carry the element-wise claim."""
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
E4M3 = svl.SVL_GEMM_E4M3


def _codes_to_values(codes: torch.Tensor) -> np.ndarray:
    return codes.view(torch.float8_e4m3fn).to(torch.float64).numpy()


@pytest.mark.parametrize("rows,cols,ld_src", [(300, 4096, 4096), (37, 72, 80), (5, 8, 8)])
def test_quantize_rows_bit_exact(rows, cols, ld_src):
    g = torch.Generator().manual_seed(rows + cols)
    mag = 10.0 ** (torch.rand(rows, 1, generator=g) * 8 - 4)
    x = (torch.randn(rows, ld_src, generator=g) * mag).to(torch.bfloat16)
    x[0] = 0  # all-zero row
    if rows > 3:
        x[1, : cols // 2] = 0
        x[2] = (torch.randn(ld_src, generator=g) * 1e-3).to(torch.bfloat16)
        x[2, 3] = 3.0  # a large outlier: most of the row lands in e4m3's subnormal range
    xd = x.cuda()
    ld_dst = ((cols + 15) // 16) * 16
    dst = torch.full((rows, ld_dst), 0xAB, dtype=torch.uint8, device="cuda")
    scale = torch.empty(rows, dtype=torch.float32, device="cuda")
    svl.svl_quantize_rows_e4m3(xd, rows, cols, ld_src, dst, ld_dst, scale)
    torch.cuda.synchronize()
    codes, sc = O.quantize_rows_e4m3(x[:, :cols].to(torch.float64).numpy())
    got = _codes_to_values(dst[:, :cols].cpu())
    np.testing.assert_array_equal(got, codes)
    np.testing.assert_array_equal(scale.cpu().numpy(), sc.astype(np.float32))
    # nothing written past `cols`
    assert (dst[:, cols:].cpu() == 0xAB).all()


def test_quantize_rows_rejects_misaligned():
    x = torch.zeros(4, 16, dtype=torch.bfloat16, device="cuda")
    d = torch.zeros(4, 16, dtype=torch.uint8, device="cuda")
    s = torch.zeros(4, dtype=torch.float32, device="cuda")
    with pytest.raises(svl.SvlError):
        svl.svl_quantize_rows_e4m3(x, 4, 12, 16, d, 16, s)  # cols not a multiple of 8
    with pytest.raises(svl.SvlError):
        svl.svl_quantize_rows_e4m3(x, 4, 16, 16, d, 8, s)   # ld_dst < cols


def fp8_bar(ref8, ref8_s32, key):
    return max(2e-2, 1.5 * rel_err(ref8[key], ref8_s32[key]))


@pytest.mark.parametrize("M,N,K", [(300, 4096, 4096), (128, 256, 128), (1, 32, 11264)])
def test_gemm_e4m3_exact_products(M, N, K):
    case = Case(synth.reduced(TINY.dims, n_layers=1), TINY, seed=5, max_seq=256)
    g = torch.Generator().manual_seed(M + N + K)
    a = (torch.randn(M, K, generator=g) * 3).to(torch.bfloat16).cuda()
    b = (torch.randn(N, K, generator=g) * 0.02).to(torch.bfloat16).cuda()
    aq = torch.empty(M, K, dtype=torch.uint8, device="cuda")
    bq = torch.empty(N, K, dtype=torch.uint8, device="cuda")
    asc = torch.empty(M, device="cuda")
    bsc = torch.empty(N, device="cuda")
    svl.svl_quantize_rows_e4m3(a, M, K, K, aq, K, asc)
    svl.svl_quantize_rows_e4m3(b, N, K, K, bq, K, bsc)
    C = torch.empty(M, N, device="cuda")
    svl.svl_gemm_e4m3(case.model.handle, aq, asc, bq, bsc, M, N, K, C)
    torch.cuda.synchronize()
    A, Bm = _codes_to_values(aq.cpu()), _codes_to_values(bq.cpu())
    raw = A @ Bm.T
    ref = raw * asc.cpu().double().numpy()[:, None] * bsc.cpu().double().numpy()[None, :]
    # float32 accumulation of K exact products: |error| <= K 2^-24 sum |terms| (loosely)
    bound = K * 2.0 ** -24 * (np.abs(A) @ np.abs(Bm).T) * asc.cpu().double().numpy()[:, None] * \
        bsc.cpu().double().numpy()[None, :] + 1e-30
    assert (np.abs(C.cpu().double().numpy() - ref) <= bound).all()
    case.close()


def _compare(case, out, n_samples, min_compared):
    """GPU e4m3 forward against the oracle's fp8, bf16 and fp32 forwards."""
    refs = {m: case.oracle(mode=m, samples=range(n_samples)) for m in ("fp8", "fp8_s32", "bf16", "fp32")}
    cu = out["cu_seqlens"].numpy()
    compared = 0
    for i in range(n_samples):
        v0, v1 = case.b_np["vis_off"][i], case.b_np["vis_off"][i + 1]
        kept = out["kept_idx"][out["kept_off"][i]:out["kept_off"][i + 1]].numpy()
        ref = {m: refs[m][i] for m in refs}
        if not check_selection(out["scores"][v0:v1].numpy(), kept, ref["fp32"]):
            # a tie-band swap: the oracle's forwards on the GPU's (valid) kept set
            bn = case.b_np
            t0, t1 = bn["text_off"][i], bn["text_off"][i + 1]
            args = (case.dims, case.w_np, bn["vis"][v0:v1], bn["text_ids"][t0:t1], bn["budget"][i],
                    bn["layer_gate"][i], bn["group_gate"][i], int(bn["keep_count"][i]))
            ref = {m: O.forward_sample(*args, mode=m, kept=kept) for m in refs}
            print(f"sample {i}: GPU selection differs inside the tie band; compared on the GPU's kept set")
        hid = out["X"][cu[i]:cu[i + 1]].double().numpy()
        lg = out["logits"][i].double().numpy()
        for key, got in (("hidden", hid), ("logits", lg)):
            bar = fp8_bar(ref["fp8"], ref["fp8_s32"], key)
            e8 = rel_err(got, ref["fp8"][key])
            assert e8 < bar, (i, key, e8, bar)
        # the layers' update: closer to the fp8 definition than to the bf16 one
        t0, t1 = case.b_np["text_off"][i], case.b_np["text_off"][i + 1]
        x0, _ = O.pack_sample(case.dims, case.w_np, case.b_np["vis"][v0:v1], kept,
                              case.b_np["text_ids"][t0:t1], O.round_bf16)
        d_got = hid - x0
        e8 = l2_err(d_got, ref["fp8"]["hidden"] - x0)
        e16 = l2_err(d_got, ref["bf16"]["hidden"] - x0)
        assert e8 < e16, (i, e8, e16)
        # and within 1.5x the definition's own storage sensitivity on the update
        sens = l2_err(ref["fp8_s32"]["hidden"] - x0, ref["fp8"]["hidden"] - x0)
        assert e8 < 1.5 * sens, (i, e8, sens)
        compared += 1
    assert compared >= min_compared
    return refs


@pytest.mark.parametrize("prefix,random_gains", [(0, False), (1, False), (0, True)])
def test_fp8_prefill_tiny_gated(prefix, random_gains):
    dims = synth.reduced(TINY.dims, n_layers=4, n_prefix=prefix)
    wl = synth.Workload("fp8", dims, batch=6, n_vis=(40, 64), s_text=(5, 40), budgets=(1.0,),
                        gates="bern_heads", features="normal", keep_count=24)
    case = Case(dims, wl, seed=81 + prefix, batch=6, max_seq=512, gemm_format=E4M3, random_gains=random_gains)
    out = case.run()
    _compare(case, out, 6, 4)
    case.close()


def test_fp8_prefill_llava_width_two_layers():
    """LLaVA-7B widths: d 4096, FFN 11,008 (2,752 channels per group, padded
    to 2,816 in the e4m3 down weights), 2 layers, group gates on."""
    wl = synth.WORKLOADS["llava"]
    dims = synth.reduced(wl.dims, n_layers=2)
    case = Case(dims, wl, seed=91, batch=2, budget=0.25, gemm_format=E4M3)
    g = torch.Generator().manual_seed(92)
    gg = (torch.rand(2, 2, dims.n_groups, generator=g) < 0.6).to(torch.uint8)
    gg[:, :, 0] = 1
    case.b["group_gate"] = gg.cuda()
    case.b_np["group_gate"] = gg.numpy()
    out = case.run()
    _compare(case, out, 2, 1)
    case.close()


def test_fp8_decode_matches_extended_prefill():
    dims = synth.reduced(TINY.dims, n_layers=3, n_prefix=1)
    n_vis, s_text, budgets = [64, 40], [16, 9], [0.8, 1.0]
    steps, max_len = 4, 128
    wl = TINY
    case = Case(dims, wl, seed=97, batch=None, max_seq=256, gemm_format=E4M3)
    b = synth.make_batch(wl, 97, n_vis_list=n_vis, s_text_list=s_text, keep_list=[-1] * 2, budget_list=budgets,
                         dims=dims)
    g = torch.Generator().manual_seed(98)
    B, L, G = 2, dims.n_layers, dims.n_groups
    b["group_gate"] = (torch.rand(B, L, G, generator=g) < 0.7).to(torch.uint8)
    b["layer_gate"] = torch.ones(B, L, dtype=torch.uint8)
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
    dws = torch.empty(svl.svl_decode_workspace_size(m.handle, B), dtype=torch.uint8, device="cuda")
    fed = torch.randint(0, dims.vocab, (steps, B), generator=g, dtype=torch.int32)
    logits = torch.empty(B, dims.vocab, dtype=torch.float32, device="cuda")
    nxt = torch.empty(B, dtype=torch.int32, device="cuda")
    got = []
    for t in range(steps):
        svl.svl_decode_step(m.handle, B, fed[t].cuda(), kv, max_len, cache_len, case.b["layer_gate"],
                            case.b["group_gate"], logits, nxt, dws, dws.numel())
        got.append(logits.cpu().clone())
    torch.cuda.synchronize()
    assert svl.svl_get_device_status(m.handle) == 0
    outc = {k: v.cpu() for k, v in out.items()}
    compared = 0
    for i in range(B):
        v0, v1 = case.b_np["vis_off"][i], case.b_np["vis_off"][i + 1]
        t0, t1 = case.b_np["text_off"][i], case.b_np["text_off"][i + 1]
        args = (dims, case.w_np, case.b_np["vis"][v0:v1], case.b_np["text_ids"][t0:t1], budgets[i],
                case.b_np["layer_gate"][i], case.b_np["group_gate"][i], fed[:, i].numpy())
        r8, s8 = O.decode_reference(*args, mode="fp8")
        r8s, s8s = O.decode_reference(*args, mode="fp8_s32")
        r32, s32 = O.decode_reference(*args, mode="fp32")
        kept = outc["kept_idx"][outc["kept_off"][i]:outc["kept_off"][i + 1]].numpy()
        if not check_selection(outc["scores"][v0:v1].numpy(), kept, r32):
            # a tie-band swap: the oracle on the GPU's (valid) kept set
            r8, s8 = O.decode_reference(*args, mode="fp8", kept=kept)
            r8s, s8s = O.decode_reference(*args, mode="fp8_s32", kept=kept)
        for t in range(steps):
            e8 = rel_err(got[t][i].double().numpy(), s8[t]["logits"])
            assert e8 < fp8_bar(s8[t], s8s[t], "logits"), (i, t, e8)
        compared += 1
    assert compared >= 1
    case.close()


def test_fp8_prefill_qwen_gqa_two_layers():
    """Qwen2-VL-7B widths with e4m3 projections: GQA 28/4 (one KV head per
    group), d 3584, FFN 18,944 (4,736 channels per group, no padding), no
    projector, 2 layers, one group gated off in one sample's second layer."""
    wl = synth.WORKLOADS["qwen"]
    dims = synth.reduced(wl.dims, n_layers=2)
    case = Case(dims, wl, seed=7, batch=2, gemm_format=E4M3)
    b = synth.make_batch(wl, 7, n_vis_list=[256, 300], s_text_list=[128, 128], keep_list=[-1, -1],
                         budget_list=[0.6, 0.9], dims=dims)
    b["group_gate"][1, 1, 2] = 0
    case.b_np = O.to_numpy_batch(b)
    case.b = {k: (v.cuda() if isinstance(v, torch.Tensor) else v) for k, v in b.items()}
    out = case.run()
    _compare(case, out, 2, 1)
    case.close()
