"""Helpers shared by the GPU parity tests: device copies of generated
inputs, oracle runs on the same inputs, and error measures."""
import numpy as np
import torch

from oracle import smartvl_oracle as O
from paper_2607_20357_gb300 import svl, synth

TIE_BAND = 1e-4


def to_device(obj, device="cuda"):
    if isinstance(obj, torch.Tensor):
        return obj.to(device)
    if isinstance(obj, dict):
        return {k: to_device(v, device) for k, v in obj.items()}
    if isinstance(obj, list):
        return [to_device(v, device) for v in obj]
    return obj


def rel_err(got, ref) -> float:
    """max |got - ref| / max |ref| (norm-wise relative error of a tensor)."""
    got = np.asarray(got, dtype=np.float64)
    ref = np.asarray(ref, dtype=np.float64)
    return float(np.abs(got - ref).max() / max(np.abs(ref).max(), 1e-30))


def l2_err(got, ref) -> float:
    got = np.asarray(got, dtype=np.float64)
    ref = np.asarray(ref, dtype=np.float64)
    return float(np.linalg.norm(got - ref) / max(np.linalg.norm(ref), 1e-30))


BAR = 2e-2          # bf16 GPU vs fp32-storage oracle
DRIFT_FACTOR = 1.5  # allowance over the bf16-emulated oracle's own distance


def bar_for(ref32, ref16, key, err=rel_err):
    """Tolerance for tensor `key`: 2e-2, or 1.5x the distance between the
    bf16-emulated and the fp32-storage oracle when bf16 storage alone already
    exceeds 2e-2 (deep stacks: the drift grows as sqrt(layers))."""
    return max(BAR, DRIFT_FACTOR * err(ref16[key], ref32[key]))


def check_selection(gpu_scores, gpu_kept, ref, z_tol=1e-4):
    """Kept sets agree except for tokens whose oracle logits lie within the
    tie band of the k-th largest logit. Returns True when identical."""
    k = ref["k"]
    ours, theirs = set(gpu_kept.tolist()), set(ref["kept"].tolist())
    assert len(ours) == k == len(gpu_kept)
    assert np.all(np.diff(gpu_kept) > 0), "kept indices not strictly ascending"
    if ours == theirs:
        return True
    z = ref["z"]
    kth = np.sort(z)[::-1][k - 1]
    for i in ours ^ theirs:
        assert abs(z[i] - kth) < TIE_BAND, f"token {i}: logit {z[i]} vs k-th {kth}"
    return False


def gpu_topk_valid(scores, kept, k):
    """The kept set is the k largest of the GPU's own logits, ties to lower index."""
    n = len(scores)
    order = sorted(range(n), key=lambda i: (-float(scores[i]), i))
    assert sorted(order[:k]) == sorted(kept.tolist())


class LazyLayers:
    """Decoder layer weights converted to float64 numpy only when the oracle
    reaches that layer (keeps host memory to one layer at a time)."""

    def __init__(self, layers):
        self.layers = layers

    def __len__(self):
        return len(self.layers)

    def __getitem__(self, i):
        return {k: v.detach().to("cpu", torch.float64).numpy() for k, v in self.layers[i].items()}


def numpy_weights_lazy(w):
    out = O.to_numpy_weights(dict(w, layers=[]))
    out["layers"] = LazyLayers(w["layers"])
    return out


class Case:
    """Seeded model + batch on the GPU and the oracle's view of both."""

    def __init__(self, dims, wl, seed, batch=None, budget=None, max_seq=8192, std=0.02, gemm_format=svl.SVL_GEMM_BF16,
                 random_gains=False):
        self.dims = dims
        w = synth.make_weights(dims, seed, std=std)
        if random_gains:
            # RMSNorm gains drawn from U[0.5, 1.5] instead of 1
            g = torch.Generator().manual_seed(seed + 7919)
            for lw in w["layers"]:
                for key in ("attn_norm", "ffn_norm"):
                    lw[key] = (0.5 + torch.rand(dims.d_model, generator=g)).to(torch.bfloat16)
            w["final_norm"] = (0.5 + torch.rand(dims.d_model, generator=g)).to(torch.bfloat16)
        b = synth.make_batch(wl, seed, budget=budget, batch=batch, dims=dims)
        self.w_np = O.to_numpy_weights(w)
        self.b_np = O.to_numpy_batch(b)
        self.w = to_device(w)
        self.b = to_device(b)
        self.model = svl.GatedPrefill(dims, self.w, max_seq=max_seq, gemm_format=gemm_format)

    def run(self, logits_mode=svl.SVL_LOGITS_LAST):
        out = self.model.run(self.b, logits_mode=logits_mode)
        torch.cuda.synchronize()
        status = svl.svl_get_device_status(self.model.handle)
        assert status == 0, f"device status {status:#x}"
        return {k: v.cpu() for k, v in out.items()}

    def oracle(self, mode="fp32", samples=None, n_layers=None):
        return O.forward_batch(self.dims, self.w_np, self.b_np, mode=mode, samples=samples, n_layers=n_layers)

    def close(self):
        self.model.close()
