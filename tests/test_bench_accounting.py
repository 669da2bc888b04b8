"""The benchmark's FLOP accounting (the numerator of every TFLOP/s and
roofline figure it prints) against the oracle's executed-FLOPs count, on the
host: the per-kind GEMM and attention FLOPs must add up to the oracle's total
minus the scorer, projector and LM-head terms, for random gates and lengths."""
import numpy as np
import pytest

import bench
from oracle import smartvl_oracle as O
from paper_2607_20357_gb300 import synth


@pytest.mark.parametrize("name", ["tiny", "llava", "qwen", "llava13b"])
def test_per_kind_flops_add_up_to_the_oracle_count(name):
    dims = synth.WORKLOADS[name].dims
    rng = np.random.default_rng(3)
    B, L, G = 5, dims.n_layers, dims.n_groups
    k = rng.integers(0, 600, size=B)
    s_text = rng.integers(1, 200, size=B)
    n_vis = k + rng.integers(0, 100, size=B)
    lg = (rng.random((B, L)) < 0.8).astype(np.uint8)
    gg = (rng.random((B, L, G)) < 0.7).astype(np.uint8)
    kinds = bench.per_kind_flops(dims, k, s_text, lg, gg)
    want = 0
    for b in range(B):
        on = O.effective_groups(lg[b], gg[b], dims.n_prefix).sum(axis=1)
        total = O.executed_flops(dims, n_vis[b], k[b], s_text[b], on)
        other = 2 * int(n_vis[b]) * dims.c_vis * dims.h_ctrl + 2 * dims.d_model * dims.vocab
        if dims.proj_hidden:
            other += 2 * int(k[b]) * (dims.c_vis * dims.proj_hidden + dims.proj_hidden * dims.d_model)
        want += total - other
    assert sum(kinds.values()) == pytest.approx(want, rel=1e-12)


def test_attention_term_is_causal():
    dims = synth.WORKLOADS["llava"].dims
    L, G = dims.n_layers, dims.n_groups
    kinds = bench.per_kind_flops(dims, np.array([576]), np.array([64]), np.ones((1, L), np.uint8),
                                 np.ones((1, L, G), np.uint8))
    S = 640
    # QK^T and PV over the causal triangle: 2 x 2 x d x S(S+1)/2 per head, A heads of d = D / A
    assert kinds["attention"] == L * 2 * dims.d_model * S * (S + 1)
    assert kinds["gateup_gemm"] == L * 4 * dims.d_model * dims.d_ffn * S
