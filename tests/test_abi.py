"""The C-ABI library loads and exports every entry point include/svl.h
declares; host-only entry points behave (no GPU needed)."""
import ctypes
import os
import re

import numpy as np
import pytest
import torch

from oracle import smartvl_oracle as O
from paper_2607_20357_gb300 import svl, synth

HEADER = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))), "include", "svl.h")


def declared_symbols():
    text = open(HEADER).read()
    return sorted(set(re.findall(r"^\s*(?:const\s+)?[\w\s\*]+?\b(svl_\w+)\s*\(", text, re.M)))


def test_header_declares_the_entry_points():
    syms = declared_symbols()
    for name in ("svl_score_select", "svl_pack", "svl_gated_prefill", "svl_model_create", "svl_flops"):
        assert name in syms
    assert set(syms) == set(svl.SYMBOLS)


def test_library_exports_every_declared_symbol(svl_lib):
    for name in declared_symbols():
        assert hasattr(svl_lib, name), name


def test_status_strings(svl_lib):
    for code in range(8):
        assert svl_lib.svl_status_string(code)
    assert svl_lib.svl_status_string(0) == b"ok"


def test_model_create_rejects_bad_args_without_gpu(svl_lib):
    h = ctypes.c_void_p()
    assert svl_lib.svl_model_create(None, None, ctypes.byref(h)) == 1
    d = svl.model_desc(synth.WORKLOADS["tiny"].dims, 256)
    d.n_groups = 3  # 4 heads are not divisible into 3 groups
    w = svl.Weights()
    assert svl_lib.svl_model_create(ctypes.byref(d), ctypes.byref(w), ctypes.byref(h)) in (1, 3)


@pytest.mark.parametrize("name", ["tiny", "llava", "qwen", "mixed"])
def test_host_flops_match_oracle(svl_lib, name):
    dims = synth.WORKLOADS[name].dims
    desc = svl.model_desc(dims, 8192)
    rng = np.random.default_rng(0)
    for _ in range(10):
        s_text, k, n_vis = int(rng.integers(1, 300)), int(rng.integers(0, 600)), 700
        lg = torch.tensor(rng.random(dims.n_layers) < 0.8, dtype=torch.uint8)
        gg = torch.tensor(rng.random((dims.n_layers, dims.n_groups)) < 0.7, dtype=torch.uint8)
        eq8, ex = svl.svl_flops(desc, s_text, k, n_vis, lg, gg)
        n_on = O.effective_groups(lg.numpy(), gg.numpy(), dims.n_prefix).sum(1)
        assert eq8 == pytest.approx(O.prefill_cost_xG(dims, s_text + k, n_on) / dims.n_groups, rel=1e-15)
        assert ex == pytest.approx(O.executed_flops(dims, n_vis, k, s_text, n_on), rel=1e-12)


def _declared_param_counts():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    out = {}
    for m in re.finditer(r"\b(svl_\w+)\s*\(([^;{]*?)\)\s*;", text, re.S):
        args = m.group(2).strip()
        out[m.group(1)] = 0 if args in ("", "void") else len(args.split(","))
    return out


def test_binding_argument_counts_match_header(svl_lib):
    counts = _declared_param_counts()
    for name in svl.SYMBOLS:
        fn = getattr(svl_lib, name)
        assert len(fn.argtypes) == counts[name], (name, len(fn.argtypes), counts[name])


def test_e4m3_entry_points_reject_bad_args_without_gpu(svl_lib):
    """Host-side checks return SVL_ERR_INVALID_ARG (1) before anything is
    launched: the pointers below are never dereferenced."""
    buf = ctypes.create_string_buffer(4096 + 16)
    base = (ctypes.addressof(buf) + 15) & ~15
    src, dst, sc = ctypes.c_void_p(base), ctypes.c_void_p(base + 1024), ctypes.c_void_p(base + 2048)
    q = svl_lib.svl_quantize_rows_e4m3
    assert q(None, None, 4, 16, 16, dst, 16, sc, None) == 1        # null source
    assert q(src, None, 4, 12, 16, dst, 16, sc, None) == 1         # cols not a multiple of 8
    assert q(src, None, 4, 16, 12, dst, 16, sc, None) == 1         # ld_src < cols
    assert q(src, None, 4, 16, 16, dst, 8, sc, None) == 1          # ld_dst < cols
    assert q(src, None, -1, 16, 16, dst, 16, sc, None) == 1        # negative rows
    assert q(ctypes.c_void_p(base + 2), None, 4, 16, 16, dst, 16, sc, None) == 1  # misaligned source
    assert q(src, ctypes.c_void_p(base + 3074), 4, 16, 16, dst, 16, sc, None) == 1  # misaligned gain
    g = svl_lib.svl_gemm_e4m3
    assert g(None, src, sc, dst, sc, 128, 32, 128, sc, None) == 1  # no model
    d = svl.model_desc(synth.WORKLOADS["tiny"].dims, 256, gemm_format=7)  # unknown operand format
    w = svl.Weights()
    h = ctypes.c_void_p()
    assert svl_lib.svl_model_create(ctypes.byref(d), ctypes.byref(w), ctypes.byref(h)) == 1


def test_ksplit_plan_launch_rule(svl_lib):
    """The K-split launch rule on the host: no split unless the persistent
    grid is resident at once, and otherwise the documented share count."""
    plan = svl.svl_ksplit_plan
    sms = 152
    # LLaVA-7B O projection at b = 0.5: 41 row tiles x 16 column tiles = 656
    # tiles, last wave 656 - 4 * 152 = 48 tiles -> 152 // 48 = 3 shares
    assert plan(656, 1024, sms, 1, 256) == 3
    assert plan(656, 1024, sms, 0, 256) == 1          # grid not resident at once: never split
    assert plan(656, 1024, sms, 1, 0) == 1            # no partial-tile workspace
    assert plan(4 * sms, 1024, sms, 1, 256) == 1      # full last wave
    assert plan(3 * sms + 77, 1024, sms, 1, 256) == 1  # last wave more than half full
    assert plan(3 * sms + 76, 1024, sms, 1, 256) == 2  # exactly half full
    assert plan(16, 1024, sms, 1, 256) == 8            # decode-sized: at most 8 shares
    assert plan(16, 1024, sms, 1, 64) == 4             # limited by the partial tiles (64 // 16)
    assert plan(16, 40, sms, 1, 256) == 2              # limited by the list capacity (1 + 24 // 16)
    assert plan(1, 1024, sms, 1, 256) == 8
    assert plan(0, 1024, sms, 1, 256) == 1
    # brute force over small grids against the stated rule
    for n in (4, 7, 16):
        for tiles in range(0, 5 * n):
            for units in (0, 3, 8, 40):
                for cap in (tiles, tiles + 5, tiles + 100):
                    r = tiles % n if tiles else 0
                    want = 1
                    if r and 2 * r <= n:
                        sp = min(n // r, 8, units // r, 1 + (cap - tiles) // r)
                        want = sp if sp >= 2 else 1
                    assert plan(tiles, cap, n, 1, units) == want, (n, tiles, units, cap)
                    assert plan(tiles, cap, n, 0, units) == 1
