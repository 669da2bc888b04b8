"""CPU oracle for SmartVL's budget-conditioned gated prefill (TEST INFRASTRUCTURE).

This module is test infrastructure. Only the test suite, the smoke check and
the benchmark's CPU-baseline leg may import it; the product path never does.
It shares no code with the CUDA library: every step is written here again,
plainly, from the paper ("Look Less, Think Faster: Joint Token-Compute
Adaptation for Multimodal LLMs", arXiv 2607.20357).

Arithmetic is float64 throughout. A storage mode rounds the tensors that the
GPU stores in memory: ``"fp64"`` (no rounding), ``"fp32"`` or ``"bf16"``
(round-to-nearest-even emulation of bfloat16 storage). Token logits are never
rounded, and neither are the RMS-normalised rows that feed a projection: they
are an intermediate of the projection, not a stored tensor. ``"fp8"`` is bf16
storage with the four gated projections of every decoder layer (QKV, O,
gate/up, down) computed from e4m3 operands, stated plainly: the projection's
input -- RMSNorm(X) * gain for QKV and gate/up, the attention output for O, the
SwiGLU output for down -- and the weight W as given (no gain folded in) are
quantised row by row: each activation row and each weight row (output
channel) is scaled so that its largest magnitude maps to 448, the largest
finite e4m3 value, and rounded to e4m3; the product of the codes is scaled
back by both scales after the sum. ``"fp8_s32"`` is the same with fp32
storage: how far it lands from ``"fp8"`` measures how strongly e4m3's
rounding boundaries amplify storage-level differences (a value moved across
a boundary jumps by a whole e4m3 step). ``"fp8_s64"`` stores nothing rounded
(the e4m3 definition on its own, for pinning it against library routines).

What each function follows:

* ``sinusoidal_encoding`` / ``budget_embedding`` -- Eq. 5 (PE and MLP of the
  scalar budget, Sec. 3.1), reused on the LLM side (Sec. 3.2).
* ``token_logits`` -- Sec. 3.1, per-token logits z; the scorer is a per-token
  MLP conditioned additively on the budget embedding (reading R1).
* ``prefill_cost_xG`` -- Eq. 8 with integer arithmetic (scaled by G so that
  alpha_l = (sum_j M_lj)/G is exact); 8D^2 generalised to 4D^2 + 4 D D_kv.
* ``budget_keep_count`` -- Sec. 3.3 "Inference": the budget projection drops
  the lowest-confidence visual tokens first, i.e. the largest token count that
  keeps Eq. 8 within b * C_full (Eq. 2).
* ``select_kept`` -- Sec. 3.1 inference rule: discard the lowest-confidence
  tokens, keep the rest as a contiguous sequence in image order.
* ``pack_sample`` -- Sec. 3 problem statement S = S_text + S_vis; kept visual
  tokens (through the LLaVA MLP projector) followed by the text tokens, with
  positions 0..S-1 (Sec. 3.1: RoPE on the compressed contiguous sequence).
* ``decoder_layer`` -- Sec. 3.2 gating: group j of layer l switches its
  attention heads and its slice of FFN channels together; alpha_l = 0 skips
  the layer through its residual connection. Gated-off parts contribute zero
  (masked-dense definition). Its stages, each usable on its own:
  ``attention_projections`` (RMSNorm, Q/K/V, RoPE), ``attention_heads``
  (causal attention of the active heads), ``attention_residual`` (O
  projection + residual), ``mlp_hidden`` (RMSNorm, gate/up, SwiGLU on the
  active channels), ``mlp_residual`` (down projection + residual).
* ``forward_sample`` / ``forward_batch`` -- the whole path, sample by sample.
* ``survival_rate`` / ``controller_gate_logits`` / ``forward_controlled`` --
  Sec. 3.2 LLM-side compute controller: the budget token (Eq. 5 encoding,
  its own MLP to D) appended after the text, P prefix layers at full
  capacity, kappa = sum sigma(z_i) / N, the fused state h + MLP_kappa(PE(kappa))
  (Eq. 7), a linear gate head thresholded at 0, the remaining layers gated.
* ``decode_reference`` -- gated decode, which the paper leaves open (Sec. 5),
  written without a cache: after feeding tokens t_1..t_n, the logits are
  those of the forward over [kept visual][text][t_1..t_n] under the prompt's
  gates, the kept visual tokens fixed by the prompt's own selection.
* ``round_e4m3`` / ``quantize_rows_e4m3`` / ``linear_e4m3`` -- FP8 weights
  for the gated GEMMs, which the paper calls orthogonal to its method
  (Sec. 5); e4m3 is the OCP 8-bit float with 4 exponent bits (bias 7) and 3
  mantissa bits, no infinities, largest finite value 448.
* ``paper_rule_sample`` -- Sec. 3.1 and Sec. 3.3 "Inference", the paper's own
  rule: tokens with sigma(z) > 0.5 survive, gates are the compute
  controller's logits thresholded at 0, and for b < 1 the budget projection
  first drops the lowest-confidence tokens, then (only when no visual token
  fits) head groups, lowest gate logit first.

Pins (checked by ``tests/test_oracle_pins.py``, all CPU): brute-force subset
selection, closed-form budget inversion, an operation counter against Eq. 8,
an independent dense transformer written with library routines, zeroed-weight
and removed-layer equivalences, shortened-sequence equivalence, batch
independence, and the paper's "full 8.5T" LLaVA-1.5-7B figure (Sec. 1).
The accuracy of the learned policy itself is parity unpinned: the paper's
trained weights are not available, so no printed end-to-end value exists.
"""
from __future__ import annotations

import numpy as np
from scipy.special import erf

OVER_BUDGET = 1  # sample flag: even zero visual tokens exceed the budget
GROUPS_DROPPED = 2  # sample flag (paper rule): the projection turned head groups off


# ----------------------------------------------------------------------------
# storage rounding
# ----------------------------------------------------------------------------
def round_bf16(a) -> np.ndarray:
    """Round to the nearest bfloat16 (ties to even), returned as float64.

    The value is first rounded to float32 (as a float32 accumulator would
    hold it), then the low 16 bits are rounded away.
    """
    f = np.ascontiguousarray(np.asarray(a, dtype=np.float32))
    u = f.view(np.uint32).astype(np.uint64)
    nan = np.isnan(f)
    lsb = (u >> np.uint64(16)) & np.uint64(1)
    u = (u + np.uint64(0x7FFF) + lsb) & np.uint64(0xFFFF0000)
    out = u.astype(np.uint32).view(np.float32).astype(np.float64)
    out[nan] = np.nan
    return out


def make_store(mode: str):
    if mode == "fp64":
        return lambda a: np.asarray(a, dtype=np.float64)
    if mode == "fp32":
        return lambda a: np.asarray(a, dtype=np.float32).astype(np.float64)
    if mode in ("bf16", "fp8"):
        return round_bf16
    if mode == "fp8_s32":
        return lambda a: np.asarray(a, dtype=np.float32).astype(np.float64)
    if mode == "fp8_s64":
        return lambda a: np.asarray(a, dtype=np.float64)
    raise ValueError(mode)


# ----------------------------------------------------------------------------
# e4m3 (FP8) operands of the gated projections
# ----------------------------------------------------------------------------
E4M3_MAX = 448.0  # largest finite e4m3 value: exponent field 15, mantissa 110


def round_e4m3(a) -> np.ndarray:
    """Round float32 values to the nearest e4m3 value (ties to the even
    mantissa), saturating to +-448; returned as float64. NaN stays NaN.

    e4m3 has 3 mantissa bits, so in the binade [2^e, 2^(e+1)) the spacing
    is 2^(e-3); below the smallest normal 2^-6 the spacing stays 2^-9
    (subnormals).
    """
    f = np.asarray(a, dtype=np.float32).astype(np.float64)
    m = np.abs(f)
    _, ex = np.frexp(m)                       # m = fr * 2^ex, fr in [0.5, 1)
    e = np.maximum(ex.astype(np.int64) - 1, -6)
    q = np.ldexp(1.0, e - 3)                  # spacing in m's binade
    r = np.rint(m / q) * q                    # exact quotient; rint rounds half to even
    r = np.minimum(r, E4M3_MAX)
    out = np.copysign(r, f)
    out[np.isnan(f)] = np.nan
    return out


def quantize_rows_e4m3(a):
    """Per-row e4m3 quantisation of a 2-D array (rows = activation rows or
    weight output channels). In float32 arithmetic: amax = max |a| of the
    row, inv = 448 / amax, scale = amax / 448 (0 and 0 for an all-zero row);
    the codes are round_e4m3(a * inv). Returns (code values, scales), both
    float64; the row's value is codes * scale."""
    a32 = np.asarray(a, dtype=np.float32)
    amax = np.max(np.abs(a32), axis=1)
    nz = amax > 0
    safe = np.where(nz, amax, np.float32(1))
    inv = np.where(nz, np.float32(E4M3_MAX) / safe, np.float32(0)).astype(np.float32)
    scale = np.where(nz, safe / np.float32(E4M3_MAX), np.float32(0)).astype(np.float32)
    codes = round_e4m3((a32 * inv[:, None]).astype(np.float32))
    return codes, scale.astype(np.float64)


def linear_e4m3(x, wq):
    """x W^T with both operands in e4m3: x's rows are quantised here, the
    weight arrives quantised (codes, per-row scales); the sum of code
    products is scaled by the activation row's and the output channel's
    scale afterwards."""
    xv, xs = quantize_rows_e4m3(x)
    wv, ws = wq
    return (xv @ wv.T) * xs[:, None] * ws[None, :]


def fp8_layer_weights(lw):
    """e4m3 weights of one layer's gated projections: every output channel
    (row of W, as given) quantised on its own. The RMSNorm gains stay on the
    activation side (they scale the normalised rows before those are
    quantised)."""
    return {name: quantize_rows_e4m3(lw[name]) for name in ("wq", "wk", "wv", "wo", "wg", "wu", "wd")}


# ----------------------------------------------------------------------------
# Eq. 5: budget encoding, token controller logits (Sec. 3.1)
# ----------------------------------------------------------------------------
def sinusoidal_encoding(b: float, dim: int) -> np.ndarray:
    """PE(b): dim/2 frequencies 10000^(-2i/dim) of the argument 1000*b;
    sines in the first half, cosines in the second (reading R2)."""
    i = np.arange(dim // 2, dtype=np.float64)
    omega = 10000.0 ** (-2.0 * i / dim)
    arg = 1000.0 * float(b) * omega
    return np.concatenate([np.sin(arg), np.cos(arg)])


def silu(x):
    return x / (1.0 + np.exp(-x))


def gelu(x):
    return 0.5 * x * (1.0 + erf(x / np.sqrt(2.0)))


def budget_embedding(b: float, w1: np.ndarray, w2: np.ndarray) -> np.ndarray:
    """e_b = W2 SiLU(W1 PE(b)) (Eq. 5 without the ViT position term)."""
    pe = sinusoidal_encoding(b, w1.shape[1])
    return w2 @ silu(w1 @ pe)


def token_logits(x: np.ndarray, e_b: np.ndarray, w1: np.ndarray, w2: np.ndarray, c2: float) -> np.ndarray:
    """z_i = w2 . SiLU(W1 x_i + e_b) + c2 for every visual token row x_i."""
    hidden = x @ w1.T + e_b[None, :]
    return silu(hidden) @ w2 + c2


# ----------------------------------------------------------------------------
# Eq. 8: prefill FLOPs, exact in integers (times G)
# ----------------------------------------------------------------------------
def effective_groups(layer_gate, group_gate, n_prefix: int) -> np.ndarray:
    """e_{l,j}: 1 if group j of layer l runs. Prefix layers always run
    (Sec. 3.2); otherwise the layer bit and the group bit must both be on."""
    lg = np.asarray(layer_gate).astype(np.int64)
    gg = np.asarray(group_gate).astype(np.int64)
    e = (lg[:, None] != 0) & (gg != 0)
    e[:n_prefix, :] = True
    return e.astype(np.int64)


def prefill_cost_xG(dims, S: int, groups_on) -> int:
    """G * C(S) of Eq. 8 for one sample.

    groups_on[l] = sum_j M_lj, so alpha_l * G = groups_on[l].  The MHA term
    8 D^2 is written 4 D^2 + 4 D D_kv (Q, O plus K, V projections).
    """
    D, Dkv, Di, V, G = dims.d_model, dims.d_kv, dims.d_ffn, dims.vocab, dims.n_groups
    S = int(S)  # Python integers: exact, no fixed-width overflow
    per_layer = (4 * D * D + 4 * D * Dkv + 6 * D * Di) * S + 4 * D * S * S
    total = 0
    for n_on in groups_on:
        total += int(n_on) * per_layer
    return total + G * 2 * D * V * S


def budget_keep_count(dims, budget: float, n_vis: int, s_text: int, groups_on, keep_count: int = -1):
    """Number of visual tokens to keep and the sample flags (Sec. 3.3).

    With keep_count >= 0 the count is min(keep_count, N). Otherwise it is the
    largest k in [0, N] with C(S_text + k) <= b * C_full, where C_full is
    Eq. 8 at S = N + S_text with every group on. The comparison is done in
    float64 on the exact integers G*C; the budget is the float32 value given.
    """
    n_vis, s_text = int(n_vis), int(s_text)
    if keep_count >= 0:
        return min(int(keep_count), n_vis), 0
    L, G = dims.n_layers, dims.n_groups
    c_full = prefill_cost_xG(dims, n_vis + s_text, [G] * L)
    limit = float(np.float32(budget)) * float(c_full)
    for k in range(n_vis, -1, -1):
        if float(prefill_cost_xG(dims, s_text + k, groups_on)) <= limit:
            return k, 0
    return 0, OVER_BUDGET


def paper_rule_counts(dims, budget: float, n_vis: int, s_text: int, z, gate_logits, keep_count: int = -1):
    """The paper's inference rule for one sample (Sec. 3.1, Sec. 3.3).

    Token mask: sigma(z_i) > 0.5, i.e. z_i > 0 (no Gumbel noise at inference).
    Gates: group j of layer l runs if l < P (prefix layers) or its compute
    controller logit is > 0 (sigma > 0.5). Budget projection against
    b * C_full (Eq. 2 with Eq. 8): first discard the lowest-confidence visual
    tokens, k = min(#{z > 0}, the largest k within the budget for these
    gates); when even k = 0 exceeds the budget, turn active groups of layers
    l >= P off in increasing order of their logit (equal logits: lower
    (l, j) first) until the cost fits, the fewest groups that make it fit
    (k stays 0: tokens went first). If the prefix layers alone exceed it, every
    other group is off and the sample is flagged OVER_BUDGET.

    Returns (k, flags, gates[L, G] as 0/1 ints).
    """
    L, G, P = dims.n_layers, dims.n_groups, dims.n_prefix
    logits = np.asarray(gate_logits, dtype=np.float64).reshape(L, G)
    gates = np.zeros((L, G), dtype=np.int64)
    for l in range(L):
        for j in range(G):
            gates[l, j] = 1 if (l < P or logits[l, j] > 0) else 0
    n_pos = int(np.sum(np.asarray(z, dtype=np.float64) > 0))
    if keep_count >= 0:
        return min(int(keep_count), int(n_vis)), 0, gates
    k, flags = budget_keep_count(dims, budget, n_vis, s_text, gates.sum(axis=1))
    if flags == 0:
        return min(k, n_pos), 0, gates
    # no visual token fits: head groups go, lowest logit first
    c_full = prefill_cost_xG(dims, int(n_vis) + int(s_text), [G] * L)
    limit = float(np.float32(budget)) * float(c_full)
    order = sorted(((logits[l, j], l * G + j) for l in range(P, L) for j in range(G) if gates[l, j]))
    for _, idx in order:
        gates[idx // G, idx % G] = 0
        if float(prefill_cost_xG(dims, int(s_text), gates.sum(axis=1))) <= limit:
            return 0, GROUPS_DROPPED, gates
    return 0, OVER_BUDGET | (GROUPS_DROPPED if order else 0), gates


def paper_rule_sample(dims, weights, x, budget, s_text, gate_logits, keep_count=-1):
    """Token controller under the paper's rule: logits, k, flags, kept indices
    and the projected gates [L, G]."""
    e_b = budget_embedding(float(np.float32(budget)), weights["bud_w1"], weights["bud_w2"])
    z = token_logits(x, e_b, weights["ctrl_w1"], weights["ctrl_w2"], weights["ctrl_c2"])
    k, flags, gates = paper_rule_counts(dims, budget, x.shape[0], s_text, z, gate_logits, keep_count)
    return z, k, flags, select_kept(z, k), gates


def project_gates(dims, budget: float, n_vis: int, s_text: int, k: int, gates, logits):
    """Budget projection on head groups alone, for a token count already
    committed (the compute controller decides after the prefix layers have
    run on the kept tokens, Sec. 3.2): while Eq. 8 at S = S_text + k exceeds
    b * C_full, the active group of layers l >= P with the lowest logit goes
    (equal logits: lower l * G + j first). Returns (gates, flags)."""
    L, G, P = dims.n_layers, dims.n_groups, dims.n_prefix
    gates = np.array(gates, dtype=np.int64).reshape(L, G)
    logits = np.asarray(logits, dtype=np.float64).reshape(L, G)
    limit = float(np.float32(budget)) * float(prefill_cost_xG(dims, int(n_vis) + int(s_text), [G] * L))
    S = int(s_text) + int(k)
    if float(prefill_cost_xG(dims, S, gates.sum(axis=1))) <= limit:
        return gates, 0
    order = sorted(((logits[l, j], l * G + j) for l in range(P, L) for j in range(G) if gates[l, j]))
    for _, idx in order:
        gates[idx // G, idx % G] = 0
        if float(prefill_cost_xG(dims, S, gates.sum(axis=1))) <= limit:
            return gates, GROUPS_DROPPED
    return gates, OVER_BUDGET | (GROUPS_DROPPED if order else 0)


def survival_rate(z) -> float:
    """kappa = sum_i sigma(z_i) / N, the soft fraction of surviving visual
    tokens that conditions the compute controller (Sec. 3.2); 0 for N = 0."""
    z = np.asarray(z, dtype=np.float64)
    return float(np.sum(1.0 / (1.0 + np.exp(-z))) / len(z)) if len(z) else 0.0


def controller_gate_logits(dims, weights, h_prefix, kappa: float) -> np.ndarray:
    """Eq. 7 and the gate head: h~ = h_b^(P) + MLP_kappa(PE(kappa)), then
    W_h h~ + c_h reshaped to [L - P, G] (rows = layers P .. L-1)."""
    h = np.asarray(h_prefix, dtype=np.float64) + budget_embedding(kappa, weights["kap_w1"], weights["kap_w2"])
    n = (dims.n_layers - dims.n_prefix) * dims.n_groups
    out = weights["gate_w"][:n] @ h + weights["gate_c"][:n]
    return out.reshape(dims.n_layers - dims.n_prefix, dims.n_groups)


def forward_controlled(dims, weights, x, text_ids, budget, mode="fp32", keep_count=-1, gates_override=None,
                       project=True, kept=None):
    """The inference path with the compute controller in the loop (Sec. 3.2,
    Sec. 3.3): tokens with z > 0 survive (keep_count >= 0 overrides), the
    sequence is [kept visual][text][budget token] with positions 0..S, the
    prefix layers run at full capacity, the gate head reads the budget
    token's state, the remaining layers run under its gates (thresholded at
    0, then projected onto the budget for b < 1 unless ``project`` is False),
    and the logits come from the last row -- the budget token, which the
    answer follows. ``gates_override`` ([L, G]) replaces the controller's
    decision (to replay another implementation's gates); ``kept`` replaces
    the top-k selection as in forward_sample.
    """
    store = make_store(mode)
    L, G, P = dims.n_layers, dims.n_groups, dims.n_prefix
    e_b = budget_embedding(float(np.float32(budget)), weights["bud_w1"], weights["bud_w2"])
    z = token_logits(x, e_b, weights["ctrl_w1"], weights["ctrl_w2"], weights["ctrl_c2"])
    kappa = survival_rate(z)
    k = min(int(keep_count), x.shape[0]) if keep_count >= 0 else int(np.sum(z > 0))
    kept = select_kept(z, k) if kept is None else np.asarray(kept, dtype=np.int64)
    X, pos = pack_sample(dims, weights, x, kept, text_ids, store)
    tok = store(budget_embedding(float(np.float32(budget)), weights["llm_bud_w1"], weights["llm_bud_w2"]))
    X = np.concatenate([X, tok[None, :]], axis=0)
    pos = np.concatenate([pos, [len(pos)]])
    on = np.ones(G, dtype=np.int64)
    qws = [fp8_layer_weights(lw) if mode in ("fp8", "fp8_s32", "fp8_s64") else None for lw in weights["layers"]]
    for l in range(P):
        X = decoder_layer(X, pos, weights["layers"][l], on, dims, store, qws[l])
    gate_logits = controller_gate_logits(dims, weights, X[-1], kappa)
    full_logits = np.zeros((L, G))
    full_logits[P:] = gate_logits
    gates = np.ones((L, G), dtype=np.int64)
    gates[P:] = (gate_logits > 0).astype(np.int64)
    flags = 0
    if gates_override is not None:
        gates = np.array(gates_override, dtype=np.int64).reshape(L, G)
    elif project and float(np.float32(budget)) < 1.0:
        gates, flags = project_gates(dims, budget, x.shape[0], len(text_ids), k, gates, full_logits)
    for l in range(P, L):
        if gates[l].any():
            X = decoder_layer(X, pos, weights["layers"][l], gates[l], dims, store, qws[l])
    y = store(rmsnorm(X[-1], weights["final_norm"], dims.rms_eps))
    logits = make_store("fp64" if mode == "fp64" else "fp32")(weights["lm_head"] @ y)
    return {"z": z, "kappa": kappa, "k": k, "kept": kept, "gate_logits": gate_logits, "gates": gates,
            "flags": flags, "hidden": X, "logits": logits}


def select_kept(z: np.ndarray, k: int) -> np.ndarray:
    """Indices of the k highest logits (equal logits: lower index first),
    returned in ascending index order."""
    n = len(z)
    order = np.lexsort((np.arange(n), -np.asarray(z, dtype=np.float64)))
    return np.sort(order[:k])


# ----------------------------------------------------------------------------
# decoder pieces
# ----------------------------------------------------------------------------
def rmsnorm(x: np.ndarray, gain: np.ndarray, eps: float) -> np.ndarray:
    ms = np.mean(x * x, axis=-1, keepdims=True)
    return x / np.sqrt(ms + eps) * gain


def rope(x: np.ndarray, pos: np.ndarray, theta: float) -> np.ndarray:
    """Rotary embedding, rotate-half convention: dim i pairs with i + d/2,
    angle pos * theta^(-2i/d). x is [S, heads, d]."""
    d = x.shape[-1]
    half = d // 2
    inv = theta ** (-2.0 * np.arange(half, dtype=np.float64) / d)
    ang = pos.astype(np.float64)[:, None] * inv[None, :]
    cos = np.cos(ang)[:, None, :]
    sin = np.sin(ang)[:, None, :]
    x1, x2 = x[..., :half], x[..., half:]
    return np.concatenate([x1 * cos - x2 * sin, x2 * cos + x1 * sin], axis=-1)


def causal_attention(q: np.ndarray, k: np.ndarray, v: np.ndarray, p_bf16: bool = False) -> np.ndarray:
    """softmax(q k^T / sqrt(d) + causal mask) v for one head; q,k,v are [S, d].

    ``p_bf16`` is a variant, not the definition: the unnormalised
    probabilities exp(s - rowmax) are rounded to bfloat16 before the product
    with v and the row sum is taken of the unrounded values -- the precision
    at which a kernel that feeds the probabilities to a bf16 tensor-core
    product computes this.
    """
    S, d = q.shape
    s = (q @ k.T) / np.sqrt(d)
    s = np.where(np.tril(np.ones((S, S), dtype=bool)), s, -np.inf)
    s = s - s.max(axis=1, keepdims=True)
    p = np.exp(s)
    if p_bf16:
        return (round_bf16(p) @ v) / p.sum(axis=1, keepdims=True)
    p = p / p.sum(axis=1, keepdims=True)
    return p @ v


def attention_projections(X, pos, lw, dims, store, qw=None):
    """Q, K, V of one sample's rows (Sec. 3.2, attention block): the
    RMS-normalised rows times the norm gain, times W_q, W_k, W_v; RoPE on Q
    and K at positions ``pos``. Every head is computed (the gated-off ones
    are ignored downstream). With ``qw`` the three products take e4m3
    operands: the normalised, gain-scaled rows and the weights, each
    quantised per row. Returns q [S, A, d_h], k and v [S, A_kv, d_h]."""
    A, Akv, dh = dims.n_heads, dims.n_kv_heads, dims.d_head
    S = X.shape[0]
    xn = rmsnorm(X, lw["attn_norm"], dims.rms_eps)
    if qw is None:
        q, k, v = xn @ lw["wq"].T, xn @ lw["wk"].T, xn @ lw["wv"].T
    else:
        q, k, v = (linear_e4m3(xn, qw[n]) for n in ("wq", "wk", "wv"))
    q = store(rope(q.reshape(S, A, dh), pos, dims.rope_theta))
    k = store(rope(k.reshape(S, Akv, dh), pos, dims.rope_theta))
    return q, k, store(v.reshape(S, Akv, dh))


def attention_heads(q, k, v, groups, dims, store, p_bf16=False):
    """Causal attention of the heads whose group is on; gated-off heads give
    zero (Sec. 3.2). GQA: query head h reads KV head h // (A / A_kv).
    Returns the attention output [S, A * d_h]."""
    A, Akv, dh, G = dims.n_heads, dims.n_kv_heads, dims.d_head, dims.n_groups
    S = q.shape[0]
    hpg = A // G
    o = np.zeros((S, A, dh))
    for h in range(A):
        if groups[h // hpg]:
            kv = h // (A // Akv)
            o[:, h, :] = causal_attention(q[:, h, :], k[:, kv, :], v[:, kv, :], p_bf16)
    return store(o.reshape(S, A * dh))


def attention_residual(X, o, lw, store, qw=None):
    """X + o W_O^T (e4m3 operands with ``qw``: o quantised per row)."""
    return store(X + (o @ lw["wo"].T if qw is None else linear_e4m3(o, qw["wo"])))


def mlp_hidden(X, lw, groups, dims, store, qw=None):
    """SwiGLU of the RMS-normalised, gain-scaled rows: SiLU(xn W_g^T) * (xn
    W_u^T), with the FFN channels of gated-off groups set to zero (channel c
    belongs to group c // (D_int / G), reading R3). With ``qw`` both products
    take e4m3 operands (xn and the weights quantised per row)."""
    G = dims.n_groups
    xn = rmsnorm(X, lw["ffn_norm"], dims.rms_eps)
    if qw is None:
        u = silu(xn @ lw["wg"].T) * (xn @ lw["wu"].T)
    else:
        u = silu(linear_e4m3(xn, qw["wg"])) * linear_e4m3(xn, qw["wu"])
    cpg = dims.d_ffn // G
    for j in range(G):
        if not groups[j]:
            u[:, j * cpg:(j + 1) * cpg] = 0.0
    return store(u)


def mlp_residual(X, u, lw, store, qw=None):
    """X + u W_down^T (e4m3 operands with ``qw``: u quantised per row)."""
    return store(X + (u @ lw["wd"].T if qw is None else linear_e4m3(u, qw["wd"])))


def decoder_layer(X, pos, lw, groups, dims, store, qw=None):
    """One gated decoder layer on one sample's rows X [S, D] (Sec. 3.2).

    ``groups`` is e_{l,:} (length G). Head h belongs to group h // (A/G);
    FFN channel c to group c // (D_int/G) (reading R3). Off groups give zero
    attention output and zero FFN channels; no rescaling by 1/alpha. With
    every group off the layer is the identity (residual bypass). With ``qw``
    (``fp8_layer_weights``) the four projections take e4m3 operands.
    """
    if not np.any(groups):
        return X
    q, k, v = attention_projections(X, pos, lw, dims, store, qw)
    X = attention_residual(X, attention_heads(q, k, v, groups, dims, store), lw, store, qw)
    return mlp_residual(X, mlp_hidden(X, lw, groups, dims, store, qw), lw, store, qw)


def project_visual(x, weights, dims, store):
    """LLaVA MLP projector W2 GELU(W1 x) (identity when no projector)."""
    if not dims.proj_hidden:
        return x
    h = store(gelu(x @ weights["proj_w1"].T))
    return store(h @ weights["proj_w2"].T)


# ----------------------------------------------------------------------------
# the whole path
# ----------------------------------------------------------------------------
def score_select_sample(dims, weights, x, budget, s_text, layer_gate, group_gate, keep_count=-1):
    """Token controller for one sample: logits, k and ascending kept indices."""
    e_b = budget_embedding(float(np.float32(budget)), weights["bud_w1"], weights["bud_w2"])
    z = token_logits(x, e_b, weights["ctrl_w1"], weights["ctrl_w2"], weights["ctrl_c2"])
    groups_on = effective_groups(layer_gate, group_gate, dims.n_prefix).sum(axis=1)
    k, flags = budget_keep_count(dims, budget, x.shape[0], s_text, groups_on, keep_count)
    return z, k, flags, select_kept(z, k)


def pack_sample(dims, weights, x, kept, text_ids, store):
    """[projected kept visual rows (image order)] ++ [text embedding rows]."""
    vis = project_visual(x[kept], weights, dims, store)
    txt = weights["embed"][np.asarray(text_ids, dtype=np.int64)]
    X = np.concatenate([vis, txt], axis=0)
    return store(X), np.arange(X.shape[0])


def forward_sample(dims, weights, x, text_ids, budget, layer_gate, group_gate,
                   keep_count=-1, mode="fp32", n_layers=None, qws=None, kept=None):
    """Token controller + pack + gated decoder + final norm + last-row logits.

    ``n_layers`` (default: all) runs only the first layers -- used to bound
    the oracle's time; the final norm and LM head then apply after them.
    ``qws`` passes the per-layer e4m3 weights of the fp8 modes when the
    caller has them already (they depend on the weights only). ``kept``
    (ascending token indices) replaces the top-k selection downstream: the
    pack and the decoder then run on that set, e.g. another valid top-k when
    logits tie.
    """
    store = make_store(mode)
    z, k, flags, sel = score_select_sample(dims, weights, x, budget, len(text_ids),
                                           layer_gate, group_gate, keep_count)
    kept = sel if kept is None else np.asarray(kept, dtype=np.int64)
    X, pos = pack_sample(dims, weights, x, kept, text_ids, store)
    e = effective_groups(layer_gate, group_gate, dims.n_prefix)
    nl = dims.n_layers if n_layers is None else n_layers
    for l in range(nl):
        lw = weights["layers"][l]
        qw = None
        if mode in ("fp8", "fp8_s32", "fp8_s64"):
            qw = qws[l] if qws is not None else fp8_layer_weights(lw)
        X = decoder_layer(X, pos, lw, e[l], dims, store, qw)
    y = store(rmsnorm(X[-1], weights["final_norm"], dims.rms_eps))
    logits = make_store("fp64" if mode == "fp64" else "fp32")(weights["lm_head"] @ y)
    return {"z": z, "k": k, "flags": flags, "kept": kept, "hidden": X, "logits": logits}


def decode_reference(dims, weights, x, text_ids, budget, layer_gate, group_gate, fed, keep_count=-1, mode="fp32",
                     kept=None):
    """Prompt forward, then one forward per fed token over the extended
    sequence (the definition a KV cache must reproduce). Returns the prompt's
    result and the list of per-step results (``logits`` of the new position,
    ``hidden`` of all rows). ``kept`` as in forward_sample."""
    first = forward_sample(dims, weights, x, text_ids, budget, layer_gate, group_gate, keep_count, mode, kept=kept)
    steps = []
    for n in range(1, len(fed) + 1):
        ids = np.concatenate([np.asarray(text_ids), np.asarray(fed[:n])])
        steps.append(forward_sample(dims, weights, x, ids, budget, layer_gate, group_gate, first["k"], mode,
                                    kept=first["kept"]))
    return first, steps


def forward_batch(dims, weights, batch, mode="fp32", n_layers=None, samples=None):
    """Run ``forward_sample`` on each sample of a numpy batch dict
    (keys as produced by the input generator, converted to numpy)."""
    out = []
    B = batch["B"]
    qws = None
    if mode in ("fp8", "fp8_s32", "fp8_s64"):
        nl = dims.n_layers if n_layers is None else n_layers
        qws = [fp8_layer_weights(weights["layers"][l]) for l in range(nl)]
    for b in (range(B) if samples is None else samples):
        v0, v1 = batch["vis_off"][b], batch["vis_off"][b + 1]
        t0, t1 = batch["text_off"][b], batch["text_off"][b + 1]
        out.append(forward_sample(
            dims, weights, batch["vis"][v0:v1], batch["text_ids"][t0:t1], batch["budget"][b],
            batch["layer_gate"][b], batch["group_gate"][b], int(batch["keep_count"][b]),
            mode=mode, n_layers=n_layers, qws=qws))
    return out


def executed_flops(dims, n_vis, k, s_text, groups_on, all_logits=False) -> int:
    """Algorithmic FLOPs that the gated path must execute for one sample:
    scorer, projector on kept tokens, active projections and FFN, causal
    attention (2 D S (S+1) alpha) and the LM head."""
    D, Dkv, Di, V, G = dims.d_model, dims.d_kv, dims.d_ffn, dims.vocab, dims.n_groups
    n_vis, k, s_text = int(n_vis), int(k), int(s_text)
    S = k + s_text
    f = 2 * n_vis * dims.c_vis * dims.h_ctrl
    if dims.proj_hidden:
        f += 2 * k * (dims.c_vis * dims.proj_hidden + dims.proj_hidden * D)
    lin = (4 * D * D + 4 * D * Dkv + 6 * D * Di) * S
    att = 2 * D * S * (S + 1)
    fl = 0
    for n_on in groups_on:
        fl += int(n_on) * (lin + att)
    assert fl % G == 0
    f += fl // G
    f += 2 * D * V * (S if all_logits else 1)
    return f


def to_numpy_weights(w) -> dict:
    """Convert a weight dict of torch tensors into float64 numpy arrays."""
    import torch

    def cv(t):
        if isinstance(t, torch.Tensor):
            return t.detach().to("cpu", torch.float64).numpy()
        return t

    out = {k: cv(v) for k, v in w.items() if k != "layers"}
    out["layers"] = [{k: cv(v) for k, v in lw.items()} for lw in w["layers"]]
    return out


def to_numpy_batch(batch) -> dict:
    import torch
    out = {}
    for k, v in batch.items():
        if isinstance(v, torch.Tensor):
            v = v.detach().cpu()
            out[k] = v.to(torch.float64).numpy() if v.dtype == torch.bfloat16 else v.numpy()
        else:
            out[k] = v
    return out
