"""Writes budget_k_llava.json: visual tokens kept per budget for one
LLaVA-1.5-7B sample (576 visual + 64 text tokens, every group on), from the
oracle's budget projection (Sec. 3.3 "Inference", Eq. 8). Run from the repo
root: python tests/golden/make_budget_k.py"""
import json
import os
import sys

sys.path.insert(0, os.path.dirname(os.path.dirname(os.path.dirname(os.path.abspath(__file__)))))
from collections import namedtuple  # noqa: E402

from oracle import smartvl_oracle as O  # noqa: E402

# LLaVA-1.5-7B decoder widths (32 layers, d 4096, MHA, SwiGLU 11008, vocab
# 32000, 4 head groups), written out here so that only the oracle computes
Dims = namedtuple("Dims", "n_layers d_model d_kv d_ffn vocab n_groups")
dims = Dims(n_layers=32, d_model=4096, d_kv=4096, d_ffn=11008, vocab=32000, n_groups=4)
ks = {}
for b in ("0.1", "0.25", "0.5", "0.75", "1.0"):
    ks[b] = O.budget_keep_count(dims, float(b), 576, 64, [dims.n_groups] * dims.n_layers)[0]
out = {"workload": "llava", "n_vis": 576, "s_text": 64,
       "cite": "Sec. 3.3 Inference (budget projection drops lowest-confidence tokens first); Eq. 8; Eq. 2",
       "k_by_budget": ks}
with open(os.path.join(os.path.dirname(os.path.abspath(__file__)), "budget_k_llava.json"), "w") as fh:
    json.dump(out, fh, indent=1)
print(out)
