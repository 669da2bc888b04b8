"""An independent dense transformer forward built from PyTorch library routines.

Used only to pin the oracle: RMSNorm via ``F.rms_norm``, attention via
``F.scaled_dot_product_attention(is_causal=True)``, rotary embedding via
complex multiplication (pair (x_i, x_{i+d/2}) as x_i + i x_{i+d/2}, rotated by
exp(i * pos * theta^(-2i/d))), SwiGLU via ``F.silu``. Everything in float64,
no gating, no storage rounding.
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


def dense_layer(X, pos, lw, dims):
    A, Akv, dh = dims.n_heads, dims.n_kv_heads, dims.d_head
    S = X.shape[0]
    xn = F.rms_norm(X, (X.shape[-1],), weight=_t(lw["attn_norm"]), eps=dims.rms_eps)
    q = F.linear(xn, _t(lw["wq"])).view(S, A, dh)
    k = F.linear(xn, _t(lw["wk"])).view(S, Akv, dh)
    v = F.linear(xn, _t(lw["wv"])).view(S, Akv, dh)
    q = rope_complex(q, pos, dims.rope_theta)
    k = rope_complex(k, pos, dims.rope_theta)
    rep = A // Akv
    k = k.repeat_interleave(rep, dim=1)
    v = v.repeat_interleave(rep, dim=1)
    o = F.scaled_dot_product_attention(q.transpose(0, 1), k.transpose(0, 1), v.transpose(0, 1),
                                       is_causal=True)
    o = o.transpose(0, 1).reshape(S, A * dh)
    X = X + F.linear(o, _t(lw["wo"]))
    xn = F.rms_norm(X, (X.shape[-1],), weight=_t(lw["ffn_norm"]), eps=dims.rms_eps)
    u = F.silu(F.linear(xn, _t(lw["wg"]))) * F.linear(xn, _t(lw["wu"]))
    return X + F.linear(u, _t(lw["wd"]))


def dense_forward(X, layers, final_norm, lm_head, dims):
    """X: [S, D] packed input rows; positions 0..S-1. Returns (hidden, last logits)."""
    X = _t(X)
    pos = torch.arange(X.shape[0])
    for lw in layers:
        X = dense_layer(X, pos, lw, dims)
    y = F.rms_norm(X[-1:], (X.shape[-1],), weight=_t(final_norm), eps=dims.rms_eps)
    return X.numpy(), (y @ _t(lm_head).T)[0].numpy()
