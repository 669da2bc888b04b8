"""Seeded synthetic inputs and weights for the budget-conditioned gated prefill.

This module only draws numbers. It holds none of the method's arithmetic: no
scoring, no budget accounting, no selection, no decoder math. Both the CUDA
path (through the tests and the benchmark) and the CPU oracle receive the very
same tensors from here.

Workload shapes follow the paper's evaluation models (LLaVA-1.5-7B decoder,
CLIP ViT-L/14-336 visual tokens, Sec. 4.1; 13B scaling, Sec. 4.4) and the
model dims that the Qwen2-VL-7B and video workloads use. The paper's
benchmark datasets (VQAv2, GQA, ...) are not available, so features are
synthetic with a structure that makes token scores spread: low rank plus a few
salient clusters, temporally correlated for video.

Weights follow PyTorch ``nn.Linear`` layout (``[out_features, in_features]``)
and are drawn N(0, 0.02); RMSNorm gains are 1.
"""
from __future__ import annotations

import dataclasses
import math
from typing import Optional

import torch


@dataclasses.dataclass(frozen=True)
class ModelDims:
    n_layers: int
    d_model: int
    n_heads: int
    n_kv_heads: int
    d_ffn: int
    vocab: int
    n_groups: int
    n_prefix: int
    c_vis: int
    h_ctrl: int
    proj_hidden: int      # 0: identity projector (c_vis == d_model)
    rms_eps: float
    rope_theta: float

    @property
    def d_head(self) -> int:
        return self.d_model // self.n_heads

    @property
    def d_kv(self) -> int:
        return self.n_kv_heads * self.d_head


@dataclasses.dataclass(frozen=True)
class Workload:
    name: str
    dims: ModelDims
    batch: int
    n_vis: tuple          # (lo, hi) inclusive visual tokens per sample
    s_text: tuple         # (lo, hi) inclusive text tokens per sample
    budgets: tuple        # explicit per-batch budget list, or ("uniform", lo, hi)
    gates: str            # "all_on", "bern_heads", "budget_scaled"
    features: str         # "normal", "lowrank_clusters", "video"
    keep_count: Optional[int] = None
    head_gate_p: float = 0.75


LLAVA7B = dict(n_layers=32, d_model=4096, n_heads=32, n_kv_heads=32, d_ffn=11008,
               vocab=32000, n_groups=4, n_prefix=0, c_vis=1024, h_ctrl=64,
               proj_hidden=4096, rms_eps=1e-5, rope_theta=1e4)

LLAVA13B = dict(n_layers=40, d_model=5120, n_heads=40, n_kv_heads=40, d_ffn=13824,
                vocab=32000, n_groups=4, n_prefix=20, c_vis=1024, h_ctrl=64,
                proj_hidden=5120, rms_eps=1e-5, rope_theta=1e4)

WORKLOADS = {
    # 64 visual tokens of dim 256, 16 text ids, MLP 256->64->1 scorer, keep 32,
    # 2-layer d=256 decoder, 4 heads, head gates Bernoulli(0.75).
    "tiny": Workload(
        "tiny",
        ModelDims(n_layers=2, d_model=256, n_heads=4, n_kv_heads=4, d_ffn=1024, vocab=1000,
                  n_groups=4, n_prefix=0, c_vis=256, h_ctrl=64, proj_hidden=0,
                  rms_eps=1e-5, rope_theta=1e4),
        batch=1, n_vis=(64, 64), s_text=(16, 16), budgets=(1.0,), gates="bern_heads",
        features="normal", keep_count=32, head_gate_p=0.75),
    # LLaVA-1.5-7B: 576 CLIP tokens (dim 1024) through a 1024->4096->4096 MLP projector.
    "llava": Workload(
        "llava", ModelDims(**LLAVA7B),
        batch=16, n_vis=(576, 576), s_text=(64, 64), budgets=(0.25, 0.5, 0.75, 1.0),
        gates="all_on", features="lowrank_clusters"),
    # Qwen2-VL-7B shapes: dynamic resolution, GQA 28/4, identity projector.
    "qwen": Workload(
        "qwen",
        ModelDims(n_layers=28, d_model=3584, n_heads=28, n_kv_heads=4, d_ffn=18944,
                  vocab=152064, n_groups=4, n_prefix=0, c_vis=3584, h_ctrl=64,
                  proj_hidden=0, rms_eps=1e-6, rope_theta=1e6),
        batch=8, n_vis=(256, 2048), s_text=(128, 128), budgets=("uniform", 0.2, 1.0),
        gates="all_on", features="lowrank_clusters"),
    # 8 frames x 576 tokens, AR(1) across frames with rho = 0.9.
    "video": Workload(
        "video", ModelDims(**LLAVA7B),
        batch=2, n_vis=(4608, 4608), s_text=(64, 64), budgets=(0.1, 0.25, 0.5),
        gates="all_on", features="video"),
    # LLaVA-1.5-13B (Sec. 4.4: 40 language layers, a fixed 20-layer prefix):
    # the LLaVA batch on the larger backbone.
    "llava13b": Workload(
        "llava13b", ModelDims(**LLAVA13B),
        batch=16, n_vis=(576, 576), s_text=(64, 64), budgets=(0.25, 0.5, 0.75, 1.0),
        gates="all_on", features="lowrank_clusters"),
    # Serving mix: 64 samples, text 16..256, budgets U[0.1,1], budget-scaled gates.
    "mixed": Workload(
        "mixed", ModelDims(**LLAVA7B),
        batch=64, n_vis=(576, 576), s_text=(16, 256), budgets=("uniform", 0.1, 1.0),
        gates="budget_scaled", features="lowrank_clusters"),
}


def reduced(dims: ModelDims, **over) -> ModelDims:
    """Same model with some dims replaced (e.g. fewer layers for a parity case)."""
    return dataclasses.replace(dims, **over)


def _gen(seed: int, device) -> torch.Generator:
    g = torch.Generator(device=device)
    g.manual_seed(int(seed))
    return g


def _normal(shape, std, g, device, dtype=torch.bfloat16):
    t = torch.randn(*shape, generator=g, device=device, dtype=torch.float32)
    if std != 1.0:
        t.mul_(std)
    return t.to(dtype)


def _tensor_seed(seed: int, layer: int, slot: int) -> int:
    """Independent stream per tensor, so any subset of layers is reproducible."""
    return (int(seed) * 1_000_003 + (layer + 1) * 64 + slot) % (1 << 62)


def make_weights(dims: ModelDims, seed: int, device="cpu", std: float = 0.02, layers=None) -> dict:
    """All model weights, bf16, ``nn.Linear`` layout, drawn N(0, std).

    The token embedding table is drawn N(0, 1) so that text rows enter the
    residual stream at a scale comparable to projected visual rows. Each
    tensor has its own seeded stream (``layers`` limits which decoder layers
    are drawn; the others are omitted from the list).

    Keys: ctrl_w1 [H, C_v], ctrl_w2 [H] and ctrl_c2 (float) for the token
    scorer; bud_w1, bud_w2 [H, H] for the budget MLP; proj_w1 [P_h, C_v],
    proj_w2 [D, P_h] when a projector exists; embed [V, D]; per layer
    wq [A*dh, D], wk/wv [A_kv*dh, D], wo [D, A*dh], wg/wu [D_int, D],
    wd [D, D_int], attn_norm/ffn_norm [D]; final_norm [D]; lm_head [V, D];
    compute controller llm_bud_w1, kap_w1 [H, H], llm_bud_w2, kap_w2 [D, H],
    gate_w [(L-P)*G, D] (bf16) and gate_c [(L-P)*G] (float32).
    """
    D, H = dims.d_model, dims.h_ctrl

    def draw(shape, sd, layer, slot):
        return _normal(shape, sd, _gen(_tensor_seed(seed, layer, slot), device), device)

    w = {
        "ctrl_w1": draw((H, dims.c_vis), std, -1, 0),
        "ctrl_w2": draw((H,), std, -1, 1),
        "ctrl_c2": 0.0,
        "bud_w1": draw((H, H), std, -1, 2),
        "bud_w2": draw((H, H), std, -1, 3),
    }
    if dims.proj_hidden:
        w["proj_w1"] = draw((dims.proj_hidden, dims.c_vis), std, -1, 4)
        w["proj_w2"] = draw((D, dims.proj_hidden), std, -1, 5)
    w["embed"] = draw((dims.vocab, D), 1.0, -1, 6)
    out_layers = []
    for l in (range(dims.n_layers) if layers is None else layers):
        out_layers.append({
            "wq": draw((dims.n_heads * dims.d_head, D), std, l, 0),
            "wk": draw((dims.d_kv, D), std, l, 1),
            "wv": draw((dims.d_kv, D), std, l, 2),
            "wo": draw((D, dims.n_heads * dims.d_head), std, l, 3),
            "wg": draw((dims.d_ffn, D), std, l, 4),
            "wu": draw((dims.d_ffn, D), std, l, 5),
            "wd": draw((D, dims.d_ffn), std, l, 6),
            "attn_norm": torch.ones(D, dtype=torch.bfloat16, device=device),
            "ffn_norm": torch.ones(D, dtype=torch.bfloat16, device=device),
        })
    w["layers"] = out_layers
    w["final_norm"] = torch.ones(D, dtype=torch.bfloat16, device=device)
    w["lm_head"] = draw((dims.vocab, D), std, -1, 7)
    # LLM-side compute controller (Sec. 3.2): budget-token MLP H -> H -> D,
    # token-count MLP H -> H -> D, linear gate head over (L - P) x G groups.
    # Scales give the budget token a residual-stream-sized embedding and gate
    # logits of order one; the gate biases are drawn around +0.3 (the paper
    # initialises them positively).
    n_gate = max(dims.n_layers - dims.n_prefix, 0) * dims.n_groups
    cs = 1.0 / math.sqrt(H)
    w["llm_bud_w1"] = draw((H, H), cs, -1, 8)
    w["llm_bud_w2"] = draw((D, H), cs, -1, 9)
    w["kap_w1"] = draw((H, H), cs, -1, 10)
    w["kap_w2"] = draw((D, H), cs, -1, 11)
    w["gate_w"] = draw((max(n_gate, 1), D), 1.0 / math.sqrt(D), -1, 12)
    gc = _gen(_tensor_seed(seed, -1, 13), device)
    w["gate_c"] = (0.3 + torch.randn(max(n_gate, 1), generator=gc, dtype=torch.float32, device=device))
    return w


def _lowrank_cluster_tokens(n: int, c: int, g, device, rank: int = 32, n_clusters: int = 8):
    """Low-rank (rank 32) tokens + isotropic noise + salient clusters on 3x3 blocks."""
    u = torch.randn(n, rank, generator=g, device=device)
    v = torch.randn(c, rank, generator=g, device=device) / math.sqrt(rank)
    x = u @ v.T + 0.1 * torch.randn(n, c, generator=g, device=device)
    typical = x.norm(dim=1).mean()
    side = max(3, int(round(math.sqrt(n))))
    rows = max(3, n // side)
    for _ in range(n_clusters):
        centre = torch.randn(c, generator=g, device=device) * math.sqrt(4.0 / c) * typical
        r0 = int(torch.randint(0, rows - 2, (1,), generator=g, device=device).item())
        c0 = int(torch.randint(0, side - 2, (1,), generator=g, device=device).item())
        for dr in range(3):
            for dc in range(3):
                i = (r0 + dr) * side + (c0 + dc)
                if i < n:
                    x[i] += centre + 0.1 * torch.randn(c, generator=g, device=device)
    return x


def _features(kind: str, n: int, c: int, g, device):
    if kind == "normal":
        return torch.randn(n, c, generator=g, device=device)
    if kind == "lowrank_clusters":
        return _lowrank_cluster_tokens(n, c, g, device)
    if kind == "video":
        per = 576
        frames = [_lowrank_cluster_tokens(per, c, g, device)]
        for _ in range(n // per - 1):
            eps = _lowrank_cluster_tokens(per, c, g, device)
            frames.append(0.9 * frames[-1] + math.sqrt(1 - 0.81) * eps)
        return torch.cat(frames, 0)[:n]
    raise ValueError(kind)


def make_batch(wl: Workload, seed: int, budget: Optional[float] = None, batch: Optional[int] = None,
               device="cpu", dims: Optional[ModelDims] = None, n_vis_list=None, s_text_list=None,
               keep_list=None, budget_list=None) -> dict:
    """One seeded batch: features, offsets, text ids, budgets, gates.

    ``budget`` overrides the workload's budget spec with one value for the
    whole batch; ``n_vis_list`` / ``s_text_list`` / ``keep_list`` /
    ``budget_list`` fix those per sample (edge cases). Returned tensors live on ``device``; offsets and gates are
    int32/uint8, features bf16, budgets float32.
    """
    dims = dims or wl.dims
    B = batch or (len(n_vis_list) if n_vis_list is not None else wl.batch)
    g = _gen(seed, "cpu")
    n_vis = torch.randint(wl.n_vis[0], wl.n_vis[1] + 1, (B,), generator=g)
    s_text = torch.randint(wl.s_text[0], wl.s_text[1] + 1, (B,), generator=g)
    if n_vis_list is not None:
        n_vis = torch.tensor(n_vis_list, dtype=torch.int64)
    if s_text_list is not None:
        s_text = torch.tensor(s_text_list, dtype=torch.int64)
    if budget_list is not None:
        budgets = torch.tensor(budget_list, dtype=torch.float32)
    elif budget is not None:
        budgets = torch.full((B,), float(budget))
    elif wl.budgets[0] == "uniform":
        lo, hi = wl.budgets[1], wl.budgets[2]
        budgets = lo + (hi - lo) * torch.rand(B, generator=g)
    else:
        budgets = torch.full((B,), float(wl.budgets[-1]))
    budgets = budgets.to(torch.float32)

    L, G = dims.n_layers, dims.n_groups
    if wl.gates == "all_on":
        layer_gate = torch.ones(B, L, dtype=torch.uint8)
        group_gate = torch.ones(B, L, G, dtype=torch.uint8)
    elif wl.gates == "bern_heads":
        layer_gate = torch.ones(B, L, dtype=torch.uint8)
        group_gate = (torch.rand(B, L, G, generator=g) < wl.head_gate_p).to(torch.uint8)
    elif wl.gates == "budget_scaled":
        p_head = budgets.double().sqrt()[:, None, None]
        p_layer = (1.0 - 0.3 * (1.0 - budgets.double()))[:, None]
        group_gate = (torch.rand(B, L, G, generator=g, dtype=torch.float64) < p_head).to(torch.uint8)
        layer_gate = (torch.rand(B, L, generator=g, dtype=torch.float64) < p_layer).to(torch.uint8)
    else:
        raise ValueError(wl.gates)

    feats = []
    fg = _gen(seed * 7919 + 1, device)
    for b in range(B):
        feats.append(_features(wl.features, int(n_vis[b]), dims.c_vis, fg, device).to(torch.bfloat16))
    vis = torch.cat(feats, 0) if feats else torch.zeros(0, dims.c_vis, dtype=torch.bfloat16, device=device)
    vis_off = torch.zeros(B + 1, dtype=torch.int32)
    vis_off[1:] = torch.cumsum(n_vis, 0).to(torch.int32)
    text_off = torch.zeros(B + 1, dtype=torch.int32)
    text_off[1:] = torch.cumsum(s_text, 0).to(torch.int32)
    text_ids = torch.randint(0, dims.vocab, (int(text_off[-1]),), generator=g, dtype=torch.int64).to(torch.int32)
    keep = torch.full((B,), -1 if wl.keep_count is None else wl.keep_count, dtype=torch.int32)
    if keep_list is not None:
        keep = torch.tensor(keep_list, dtype=torch.int32)
    return {
        "B": B,
        "vis": vis,
        "vis_off": vis_off.to(device),
        "text_ids": text_ids.to(device),
        "text_off": text_off.to(device),
        "budget": budgets.to(device),
        "keep_count": keep.to(device),
        "layer_gate": layer_gate.to(device),
        "group_gate": group_gate.to(device),
    }
