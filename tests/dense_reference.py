"""An independent dense transformer forward built from PyTorch library routines.

Used only to pin the oracle: RMSNorm via ``F.rms_norm``, attention via
``F.scaled_dot_product_attention(is_causal=True)``, rotary embedding via
complex multiplication (pair (x_i, x_{i+d/2}) as x_i + i x_{i+d/2}, rotated by
exp(i * pos * theta^(-2i/d))), SwiGLU via ``F.silu``. Everything in float64,
no gating, no storage rounding.

``dense_forward_fp8`` is the same forward with the four projections of each
layer on e4m3 operands, built from PyTorch's own float8_e4m3fn conversion:
each input row (RMSNorm(X) * gain, the attention output, the SwiGLU output)
and each weight row is scaled in float32 so that its largest magnitude maps
to 448, converted to float8_e4m3fn (round to nearest even, saturated), and
the float64 product of the decoded codes is scaled back by both scales.
"""
import torch
import torch.nn.functional as F


def _t(a):
    return torch.as_tensor(a, dtype=torch.float64)


def rope_complex(x, pos, theta):
    # x [S, H, d]
    d = x.shape[-1]
    half = d // 2
    inv = theta ** (-2.0 * torch.arange(half, dtype=torch.float64) / d)
    ang = pos.to(torch.float64)[:, None] * inv[None, :]
    rot = torch.polar(torch.ones_like(ang), ang)[:, None, :]
    z = torch.complex(x[..., :half], x[..., half:]) * rot
    return torch.cat([z.real, z.imag], dim=-1)


def e4m3_rows(a):
    """(decoded codes, scales) of the rows of a float64 tensor: float32
    scale amax / 448, codes float8_e4m3fn(a * 448 / amax)."""
    a32 = _t(a).to(torch.float32)
    amax = a32.abs().amax(dim=1)
    nz = amax > 0
    full = torch.full_like(amax, 448.0)
    # tensor / tensor: an IEEE division (a Python scalar over a tensor goes
    # through a reciprocal and is not correctly rounded)
    inv = torch.where(nz, full / torch.where(nz, amax, torch.ones_like(amax)), torch.zeros_like(amax))
    scale = torch.where(nz, amax / full, torch.zeros_like(amax))
    q = (a32 * inv[:, None]).clamp(-448.0, 448.0).to(torch.float8_e4m3fn)
    return q.to(torch.float64), scale.to(torch.float64)


def linear_fp8(x, w):
    """x W^T with both operands quantised per row (e4m3_rows)."""
    xc, xs = e4m3_rows(x)
    wc, ws = e4m3_rows(w)
    return F.linear(xc, wc) * xs[:, None] * ws[None, :]


def dense_layer(X, pos, lw, dims, linear=None):
    linear = linear or (lambda x, w: F.linear(x, _t(w)))
    A, Akv, dh = dims.n_heads, dims.n_kv_heads, dims.d_head
    S = X.shape[0]
    xn = F.rms_norm(X, (X.shape[-1],), weight=_t(lw["attn_norm"]), eps=dims.rms_eps)
    q = linear(xn, lw["wq"]).view(S, A, dh)
    k = linear(xn, lw["wk"]).view(S, Akv, dh)
    v = linear(xn, lw["wv"]).view(S, Akv, dh)
    q = rope_complex(q, pos, dims.rope_theta)
    k = rope_complex(k, pos, dims.rope_theta)
    rep = A // Akv
    k = k.repeat_interleave(rep, dim=1)
    v = v.repeat_interleave(rep, dim=1)
    o = F.scaled_dot_product_attention(q.transpose(0, 1), k.transpose(0, 1), v.transpose(0, 1),
                                       is_causal=True)
    o = o.transpose(0, 1).reshape(S, A * dh)
    X = X + linear(o, lw["wo"])
    xn = F.rms_norm(X, (X.shape[-1],), weight=_t(lw["ffn_norm"]), eps=dims.rms_eps)
    u = F.silu(linear(xn, lw["wg"])) * linear(xn, lw["wu"])
    return X + linear(u, lw["wd"])


def dense_forward(X, layers, final_norm, lm_head, dims, linear=None):
    """X: [S, D] packed input rows; positions 0..S-1. Returns (hidden, last logits)."""
    X = _t(X)
    pos = torch.arange(X.shape[0])
    for lw in layers:
        X = dense_layer(X, pos, lw, dims, linear)
    y = F.rms_norm(X[-1:], (X.shape[-1],), weight=_t(final_norm), eps=dims.rms_eps)
    return X.numpy(), (y @ _t(lm_head).T)[0].numpy()


def dense_forward_fp8(X, layers, final_norm, lm_head, dims):
    """dense_forward with e4m3 operands in the four projections of every layer."""
    return dense_forward(X, layers, final_norm, lm_head, dims, linear=linear_fp8)


def project_visual(x, w1, w2):
    """LLaVA projector from library layers: Linear, exact (erf) GELU, Linear."""
    return F.linear(F.gelu(F.linear(_t(x), _t(w1)), approximate="none"), _t(w2)).numpy()
