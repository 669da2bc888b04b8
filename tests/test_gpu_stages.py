"""Per-stage GPU parity of one decoder layer at LLaVA-1.5-7B widths (and
Qwen2-VL-7B's GQA widths) against the oracle's bf16-emulated stages (Sec. 3.2
attention and MLP blocks).

Each stage runs alone through svl_layer_stage -- the same kernels and launch
configuration the prefill uses -- on inputs the GPU stored, and the oracle
recomputes the stage in float64 from those same bf16 values and rounds its
output to bf16. The bar:

* QKV + RoPE, O projection + residual, gate/up + SwiGLU, down projection +
  residual: every element within one bf16 ulp of the oracle, plus the
  float32 accumulation error of the GPU's sum, bounded by
  2^-15 * sum_k |x_k w_k| (twice the recursive-summation bound of the
  K/16 + 16 fp32 additions a K-deep tensor-core product makes). For a typical
  element that term is under half an ulp, so two roundings of nearly the same
  value differ by one ulp at most; it matters only for outputs near zero,
  where the products cancel. The number of differing elements is reported,
  and with unit gains and bf16 operands the L2 relative error must be within
  1e-3.
* Attention: the kernel rounds the unnormalised probabilities to bf16 before
  the P.V product (relative error at most 2^-8 each) and divides by the
  float32 sum of the unrounded ones, so per element
  |O_gpu - O| <= 2^-8 * sum_j p_j |v_j| / sum_j p_j + one bf16 ulp (+ float32
  accumulation); checked against the exact definition and against the
  variant that rounds P to bf16 at the true row maximum (2^-7 there).
* Gated-off work is never issued: the columns of gated-off heads in Q, K and
  the attention output and the gated-off FFN channels are filled with NaN
  before the stage; producers must leave them NaN and consumers must not read
  them (the residual rows stay finite).

The e4m3 model is checked against the plain e4m3 definition of the oracle
(e4m3(RMSNorm(X) * gain) x e4m3(W), random gains). The kernel quantises
X * gain and applies 1/rms after the product: the codes equal the plain ones
except at exact e4m3 ties that float32 rounding splits (about 0.1 % with bf16
inputs); the bar adds, per element, the exact effect of those one-step code
differences, computed here from both sets of codes.
"""
import numpy as np
import pytest
import torch

from oracle import smartvl_oracle as O
from paper_2607_20357_gb300 import svl, synth
from tests.gpu_common import l2_err

pytestmark = pytest.mark.gpu

if not torch.cuda.is_available():
    pytest.skip("needs a CUDA GPU", allow_module_level=True)

LENGTHS = [300, 131, 64]  # ragged: several 128-row tiles, partial tails, a one-tile sample


def ulp_bf16(x):
    a = np.maximum(np.abs(np.asarray(x, dtype=np.float64)), 2.0 ** -126)
    return 2.0 ** (np.floor(np.log2(a)) - 7)


def check_close(name, got, ref, extra=0.0, l2_bar=1e-3):
    """Every element within one bf16 ulp (plus `extra`) of the oracle."""
    got = np.asarray(got, dtype=np.float64)
    ref = np.asarray(ref, dtype=np.float64)
    assert np.isfinite(got).all(), f"{name}: non-finite output"
    err = np.abs(got - ref)
    tol = ulp_bf16(np.maximum(np.abs(got), np.abs(ref))) + extra + 2.0 ** -18 * np.abs(ref)
    flips = int((got != ref).sum())
    l2 = l2_err(got, ref)
    worst = float((err / tol).max()) if err.size else 0.0
    print(f"{name}: {flips}/{got.size} elements differ ({100.0 * flips / max(got.size, 1):.3f} %), "
          f"L2 rel {l2:.2e}, max err / tol {worst:.3f}")
    assert (err <= tol).all(), f"{name}: {int((err > tol).sum())} elements beyond the bar (max ratio {worst})"
    if l2_bar is not None:
        assert l2 <= l2_bar, (name, l2)
    return flips, l2


class Layer:
    """One decoder layer of a workload's widths (LLaVA-7B by default) on the
    GPU and the oracle's view."""

    def __init__(self, seed, gemm_format=svl.SVL_GEMM_BF16, random_gains=False, workload="llava", lengths=None,
                 gg=None):
        wl = synth.WORKLOADS[workload]
        self.dims = dims = synth.reduced(wl.dims, n_layers=1, vocab=512)
        w = synth.make_weights(dims, seed)
        if random_gains:
            g = torch.Generator().manual_seed(seed + 1)
            for lw in w["layers"]:
                for key in ("attn_norm", "ffn_norm"):
                    lw[key] = (0.5 + torch.rand(dims.d_model, generator=g)).to(torch.bfloat16)
        self.lw = {k: v.to(torch.float64).numpy() for k, v in w["layers"][0].items()}
        wd = {k: (v.cuda() if isinstance(v, torch.Tensor) else v) for k, v in w.items() if k != "layers"}
        wd["layers"] = [{k: v.cuda() for k, v in l.items()} for l in w["layers"]]
        self.w = wd
        self.model = svl.GatedPrefill(dims, wd, max_seq=1024, gemm_format=gemm_format)
        lengths = LENGTHS if lengths is None else lengths
        self.B = B = len(lengths)
        self.cu = np.concatenate([[0], np.cumsum(lengths)]).astype(np.int64)
        self.T = int(self.cu[-1])
        self.t_cap = self.T + 5  # rows past the packed batch must stay untouched
        self.t_pad = (self.t_cap + 7) // 8 * 8
        gen = torch.Generator().manual_seed(seed + 2)
        X = torch.zeros(self.t_cap, dims.d_model)
        X[:self.T] = torch.randn(self.T, dims.d_model, generator=gen) * (0.5 + torch.rand(self.T, 1, generator=gen))
        self.X = X.to(torch.bfloat16).cuda()
        self.pos = torch.cat([torch.arange(n) for n in lengths] + [torch.zeros(5, dtype=torch.int64)]).to(
            torch.int32).cuda()
        self.cu_d = torch.tensor(self.cu, dtype=torch.int32).cuda()
        G = dims.n_groups
        if gg is None:
            gg = np.ones((B, 1, G), np.uint8)
            gg[1, 0, 2] = 0              # one group off in sample 1
            gg[2, 0, 0] = gg[2, 0, 3] = 0  # two groups off in sample 2
        self.gg = gg
        self.group_gate = torch.tensor(gg).cuda()
        self.layer_gate = torch.ones(B, 1, dtype=torch.uint8).cuda()
        need = svl.svl_workspace_size_for(self.model.handle, ("prefill",), B, self.t_cap, 0)
        self.ws = torch.empty(need, dtype=torch.uint8, device="cuda")
        self.qw = O.fp8_layer_weights(self.lw) if gemm_format == svl.SVL_GEMM_E4M3 else None

    def stage(self, stage, X, **bufs):
        svl.svl_layer_stage(self.model.handle, stage, 0, self.B, self.t_cap, X, self.cu_d, self.pos,
                            self.layer_gate, self.group_gate, workspace=self.ws, workspace_bytes=self.ws.numel(),
                            **bufs)
        torch.cuda.synchronize()
        assert svl.svl_get_device_status(self.model.handle) == 0

    def rows(self, b):
        return slice(int(self.cu[b]), int(self.cu[b + 1]))

    def head_cols(self, b, n_heads):
        """Column mask of the heads (of n_heads) whose group is on for sample b."""
        dh, G = self.dims.d_head, self.dims.n_groups
        on = np.repeat(self.gg[b, 0].astype(bool), n_heads // G)
        return np.repeat(on, dh)

    def chan_cols(self, b):
        return np.repeat(self.gg[b, 0].astype(bool), self.dims.d_ffn // self.dims.n_groups)

    def close(self):
        self.model.close()


def np64(t):
    return t.detach().to("cpu", torch.float64).numpy()


def _codes(x):
    return O.quantize_rows_e4m3(x)


ACC = 2.0 ** -15  # float32 accumulation, relative to sum |x_k w_k|


def _acc_floor(a, w):
    """Accumulation error bound of a @ w^T on the GPU: ACC * |a| @ |w|^T."""
    return ACC * (np.abs(a) @ np.abs(w).T)


def _norm_step_bound(L, Xb, gain, w_codes):
    """Per-element effect of the one-step code differences between the plain
    codes of RMSNorm(X) * gain and the kernel's codes of X * gain, on
    xn W^T: |codes_plain - codes_kernel| . |W codes|^T times both scales."""
    d = L.dims
    pc, ps = _codes(O.rmsnorm(Xb, gain, d.rms_eps))
    fc, _ = _codes((Xb.astype(np.float32) * gain.astype(np.float32)).astype(np.float64))
    wc, wsc = w_codes
    return (np.abs(pc - fc) @ np.abs(wc).T) * ps[:, None] * wsc[None, :], float((pc != fc).mean())


def _rope_pair_sum(e, heads, dh):
    """An error bound e [S, heads*dh] carried through RoPE: each rotated
    component mixes the pair (i, i + dh/2), so it is bounded by the sum of the
    pair's bounds."""
    e = e.reshape(e.shape[0], heads, dh)
    half = dh // 2
    s = e[..., :half] + e[..., half:]
    return np.concatenate([s, s], axis=-1).reshape(e.shape[0], heads * dh)


def check_attention(L, qg, kg, vg, aog):
    """Attention of every sample against the oracle on the GPU's own Q, K, V:
    the exact definition and the bf16-P variant, per element; gated-off heads
    stay NaN."""
    d = L.dims
    A, Akv, dh = d.n_heads, d.n_kv_heads, d.d_head
    store = O.round_bf16
    for b in range(L.B):
        r = L.rows(b)
        S = r.stop - r.start
        cq = L.head_cols(b, A)
        if not cq.any():  # every group of the sample off: nothing is computed or stored
            assert np.isnan(aog[r]).all()
            continue
        groups = L.gg[b, 0]
        qb, kb, vb = qg[r].reshape(S, A, dh), kg[r].reshape(S, Akv, dh), vg[r].reshape(S, Akv, dh)
        exact = O.attention_heads(qb, kb, vb, groups, d, lambda a: a)
        var = O.attention_heads(qb, kb, vb, groups, d, lambda a: a, p_bf16=True)
        # W = sum_j p_j |v_j| / sum_j p_j per (query, head, dim): the weighted mean of |v|
        W = O.attention_heads(qb, kb, np.abs(vb), groups, d, lambda a: a)
        got = aog[r][:, cq]
        check_close(f"attn s{b} vs exact", got, store(exact)[:, cq], (2.0 ** -8 * (1 + 1e-3) + ACC) * W[:, cq],
                    l2_bar=4e-3)
        check_close(f"attn s{b} vs bf16-P variant", got, store(var)[:, cq], (2.0 ** -7 * (1 + 1e-3) + ACC) * W[:, cq],
                    l2_bar=4e-3)
        assert np.isnan(aog[r][:, ~cq]).all()


def run_layer_checks(L):
    d = L.dims
    A, Akv, dh, G = d.n_heads, d.n_kv_heads, d.d_head, d.n_groups
    hq, dkv = A * dh, Akv * dh
    store = O.round_bf16
    qw = L.qw
    X_np = np64(L.X)
    nan = float("nan")
    fold = not np.all(L.lw["attn_norm"] == 1.0) and qw is None  # bf16 path folds the gains into bf16 weights

    # ---- QKV + RoPE
    q = torch.full((L.t_cap, hq), nan, dtype=torch.bfloat16, device="cuda")
    k = torch.full((L.t_cap, dkv), nan, dtype=torch.bfloat16, device="cuda")
    vt = torch.zeros(dkv, L.t_pad, dtype=torch.bfloat16, device="cuda")
    L.stage(svl.SVL_LAYER_QKV, L.X, q=q, k=k, vt=vt)
    qg, kg, vg = np64(q), np64(k), np64(vt).T
    for b in range(L.B):
        r = L.rows(b)
        pos = np.arange(r.stop - r.start)
        qr, kr, vr = O.attention_projections(X_np[r], pos, L.lw, d, store, qw)
        qr, kr, vr = qr.reshape(-1, hq), kr.reshape(-1, dkv), vr.reshape(-1, dkv)
        cq, ck = L.head_cols(b, A), L.head_cols(b, Akv)
        extra = {}
        xn = O.rmsnorm(X_np[r], L.lw["attn_norm"], d.rms_eps)
        for key, wn, heads, cols, rope in (("q", "wq", A, cq, True), ("k", "wk", Akv, ck, True),
                                           ("v", "wv", Akv, ck, False)):
            e = _acc_floor(xn, L.lw[wn]) * (1.15 if qw is not None else 1.0)
            if qw is not None:
                step, frac = _norm_step_bound(L, X_np[r], L.lw["attn_norm"], qw[wn])
                print(f"qkv s{b} {key}: {100 * frac:.3f} % of the activation codes differ (e4m3 ties)")
                e = e + step
            elif fold:
                # bf16(W * gain): relative error 2^-8 per weight
                e = e + 2.0 ** -8 * (np.abs(xn) @ np.abs(L.lw[wn]).T)
            extra[key] = (_rope_pair_sum(e, heads, dh) if rope else e)[:, cols]
        l2_bar = 1e-3 if (qw is None and not fold) else None
        check_close(f"qkv s{b} q", qg[r][:, cq], qr[:, cq], extra["q"], l2_bar)
        check_close(f"qkv s{b} k", kg[r][:, ck], kr[:, ck], extra["k"], l2_bar)
        check_close(f"qkv s{b} v", vg[r][:, ck], vr[:, ck], extra["v"], l2_bar)
        # gated-off heads: never written
        assert np.isnan(qg[r][:, ~cq]).all() and np.isnan(kg[r][:, ~ck]).all()
        assert (vg[r][:, ~ck] == 0).all()
    assert np.isnan(qg[L.T:]).all()  # rows past the packed batch untouched

    # ---- attention (on the GPU's own Q, K, V)
    ao = torch.full((L.t_cap, hq), nan, dtype=torch.bfloat16, device="cuda")
    L.stage(svl.SVL_LAYER_ATTN, L.X, q=q, k=k, vt=vt, ao=ao)
    aog = np64(ao)
    check_attention(L, qg, kg, vg, aog)

    # ---- O projection + residual (gated-off heads of ao hold NaN: never read)
    Xo = L.X.clone()
    L.stage(svl.SVL_LAYER_OPROJ, Xo, ao=ao)
    Xo_np = np64(Xo)
    for b in range(L.B):
        r = L.rows(b)
        o = np.where(L.head_cols(b, A)[None, :], aog[r], 0.0)
        ref = O.attention_residual(X_np[r], o, L.lw, store, qw)
        check_close(f"oproj s{b}", Xo_np[r], ref, _acc_floor(o, L.lw["wo"]) * (1.15 if qw is not None else 1.0),
                    1e-3 if qw is None else None)
    assert (Xo_np[L.T:] == X_np[L.T:]).all()

    # ---- gate/up + SwiGLU (on the GPU's residual rows)
    h = torch.full((L.t_cap, d.d_ffn), nan, dtype=torch.bfloat16, device="cuda")
    L.stage(svl.SVL_LAYER_GATEUP, Xo, h=h)
    hg = np64(h)
    for b in range(L.B):
        r = L.rows(b)
        ref = O.mlp_hidden(Xo_np[r], L.lw, L.gg[b, 0], d, store, qw)
        cc = L.chan_cols(b)
        xn = O.rmsnorm(Xo_np[r], L.lw["ffn_norm"], d.rms_eps)
        f8 = 1.15 if qw is not None else 1.0
        eg, eu = _acc_floor(xn, L.lw["wg"]) * f8, _acc_floor(xn, L.lw["wu"]) * f8
        if qw is not None:
            eg = eg + _norm_step_bound(L, Xo_np[r], L.lw["ffn_norm"], qw["wg"])[0]
            eu = eu + _norm_step_bound(L, Xo_np[r], L.lw["ffn_norm"], qw["wu"])[0]
            gv, uv = O.linear_e4m3(xn, qw["wg"]), O.linear_e4m3(xn, qw["wu"])
        else:
            if fold:
                eg = eg + 2.0 ** -8 * (np.abs(xn) @ np.abs(L.lw["wg"]).T)
                eu = eu + 2.0 ** -8 * (np.abs(xn) @ np.abs(L.lw["wu"]).T)
            gv, uv = xn @ L.lw["wg"].T, xn @ L.lw["wu"].T
        # d(SiLU(g) u) <= 1.1 |u| dg + |SiLU(g)| du + 1.1 dg du  (|SiLU'| <= 1.1)
        extra = (1.1 * np.abs(uv) * eg + np.abs(O.silu(gv)) * eu + 1.1 * eg * eu)[:, cc]
        check_close(f"gateup s{b}", hg[r][:, cc], ref[:, cc], extra, 1e-3 if (qw is None and not fold) else None)
        assert np.isnan(hg[r][:, ~cc]).all()

    # ---- down projection + residual (gated-off channels of h hold NaN: never read)
    Xd = Xo.clone()
    L.stage(svl.SVL_LAYER_DOWN, Xd, h=h)
    Xd_np = np64(Xd)
    for b in range(L.B):
        r = L.rows(b)
        u = np.where(L.chan_cols(b)[None, :], hg[r], 0.0)
        ref = O.mlp_residual(Xo_np[r], u, L.lw, store, qw)
        check_close(f"down s{b}", Xd_np[r], ref, _acc_floor(u, L.lw["wd"]) * (1.15 if qw is not None else 1.0),
                    1e-3 if qw is None else None)
    assert (Xd_np[L.T:] == X_np[L.T:]).all()


def test_stages_bf16_llava_width():
    L = Layer(seed=301)
    run_layer_checks(L)
    L.close()


def test_stages_bf16_qwen_width_gqa():
    """Qwen2-VL-7B widths: d 3584, GQA 28 query / 4 KV heads (one KV head per
    group, 7 query heads sharing it), FFN 18,944 (4,736 channels per group),
    RoPE theta 1e6, RMSNorm eps 1e-6; groups off as in the LLaVA case, so a
    gated-off group removes one KV head and its seven query heads."""
    L = Layer(seed=311, workload="qwen")
    run_layer_checks(L)
    L.close()


def test_stages_bf16_llava_width_cta_pairs(monkeypatch):
    """The QKV and gate/up stages on CTA pairs (256-row tiles, tcgen05
    cta_group::2; chosen with SVL_PAIR_GEMM=1 at model creation) against the
    same bars."""
    monkeypatch.setenv("SVL_PAIR_GEMM", "1")
    L = Layer(seed=307)
    run_layer_checks(L)
    L.close()


def test_stages_bf16_llava_width_random_gains():
    """Non-unit RMSNorm gains: the bf16 path folds them into bf16 copies of
    W_qkv and W_g,u (relative error 2^-8 per weight), which the bar of the
    QKV and gate/up stages adds per element."""
    L = Layer(seed=303, random_gains=True)
    run_layer_checks(L)
    L.close()


def test_stages_e4m3_llava_width_random_gains():
    """e4m3 projections with random gains against the plain e4m3 definition."""
    L = Layer(seed=305, gemm_format=svl.SVL_GEMM_E4M3, random_gains=True)
    run_layer_checks(L)
    L.close()


def test_quantize_with_gain_bit_exact():
    """svl_quantize_rows_e4m3 with a gain vector: codes and scales of
    x * gain (exact float32 products) bit for bit against the oracle's
    quantiser on the same products."""
    g = torch.Generator().manual_seed(17)
    rows, cols = 200, 4096
    x = (torch.randn(rows, cols, generator=g) * 10.0 ** (torch.rand(rows, 1, generator=g) * 4 - 2)).to(torch.bfloat16)
    gain = (0.5 + torch.rand(cols, generator=g)).to(torch.bfloat16)
    dst = torch.empty(rows, cols, dtype=torch.uint8, device="cuda")
    scale = torch.empty(rows, dtype=torch.float32, device="cuda")
    svl.svl_quantize_rows_e4m3(x.cuda(), rows, cols, cols, dst, cols, scale, gain=gain.cuda())
    torch.cuda.synchronize()
    prod = (x.to(torch.float32) * gain.to(torch.float32)).to(torch.float64).numpy()
    codes, sc = O.quantize_rows_e4m3(prod)
    got = dst.cpu().view(torch.float8_e4m3fn).to(torch.float64).numpy()
    np.testing.assert_array_equal(got, codes)
    np.testing.assert_array_equal(scale.cpu().numpy(), sc.astype(np.float32))


def test_attention_many_ragged_samples():
    """Attention at LLaVA-7B widths over 16 ragged samples: single-row
    samples, sample starts off the 8-row alignment of the key tiles, lengths
    around the 128-query unit and the 256-query item (units whose later half
    is empty), one sample with every group off and random groups elsewhere.
    The kernel takes its units from a counter; every unit's output is checked
    against the oracle, and rows of gated-off heads stay NaN."""
    lengths = [1, 7, 8, 9, 127, 128, 129, 255, 256, 257, 3, 200, 64, 1, 300, 17]
    rng = np.random.default_rng(7)
    gg = (rng.random((len(lengths), 1, 4)) < 0.6).astype(np.uint8)
    gg[:, 0, 1] = 1        # at least one group on ...
    gg[5, 0, :] = 0        # ... except in sample 5
    L = Layer(seed=401, lengths=lengths, gg=gg)
    d = L.dims
    hq, dkv = d.n_heads * d.d_head, d.n_kv_heads * d.d_head
    nan = float("nan")
    q = torch.full((L.t_cap, hq), nan, dtype=torch.bfloat16, device="cuda")
    k = torch.full((L.t_cap, dkv), nan, dtype=torch.bfloat16, device="cuda")
    vt = torch.zeros(dkv, L.t_pad, dtype=torch.bfloat16, device="cuda")
    L.stage(svl.SVL_LAYER_QKV, L.X, q=q, k=k, vt=vt)
    ao = torch.full((L.t_cap, hq), nan, dtype=torch.bfloat16, device="cuda")
    L.stage(svl.SVL_LAYER_ATTN, L.X, q=q, k=k, vt=vt, ao=ao)
    check_attention(L, np64(q), np64(k), np64(vt).T, np64(ao))
    assert np.isnan(np64(ao)[L.T:]).all()  # rows past the packed batch untouched
    L.close()

