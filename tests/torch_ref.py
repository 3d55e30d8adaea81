"""A second statement of the Llama block built from torch library routines.

Used only to pin the oracle: attention through
`torch.nn.functional.scaled_dot_product_attention`, RMSNorm through
`torch.nn.functional.rms_norm`, SiLU through `torch.nn.functional.silu`, and
RoPE as multiplication of complex numbers (pair (i, i + D/2) read as
x_i + j x_{i+D/2} and multiplied by exp(j * pos * w_i), the RoFormer
definition).  Everything in float64 on the CPU.
"""
from __future__ import annotations

import torch
import torch.nn.functional as F


def t64(a) -> torch.Tensor:
    if isinstance(a, torch.Tensor):
        return a.detach().to("cpu", torch.float64)
    return torch.as_tensor(a, dtype=torch.float64)


def rope_complex(x: torch.Tensor, pos: torch.Tensor, inv_freq: torch.Tensor) -> torch.Tensor:
    """x: [n, heads, D]; rotate by pos*w via complex multiplication."""
    half = x.shape[-1] // 2
    z = torch.complex(x[..., :half], x[..., half:])
    ang = pos.to(torch.float64)[:, None] * inv_freq[None, :]
    rot = torch.polar(torch.ones_like(ang), ang)[:, None, :]
    z = z * rot
    return torch.cat([z.real, z.imag], dim=-1)


def layer_full(s, lw: dict, x: torch.Tensor, inv_freq: torch.Tensor, pos: torch.Tensor,
               attn_mask: torch.Tensor | None = None, scale: float | None = None):
    """Full layer over all n rows; attn_mask [n, n] boolean (True = may attend) or causal.
    The q/k/v projection takes lw["b_qkv"] as its bias when present; `scale` is the
    softmax's logit factor (None: the library's default 1/sqrt(D))."""
    n = x.shape[0]
    D, Hq, Hkv = s.head_dim, s.n_q_heads, s.n_kv_heads
    n1 = F.rms_norm(x, (x.shape[-1],), weight=t64(lw["attn_norm"]), eps=s.rms_eps)
    b = lw.get("b_qkv")
    qkv = F.linear(n1, t64(lw["w_qkv"]), None if b is None else t64(b))
    q = qkv[:, : Hq * D].reshape(n, Hq, D)
    k = qkv[:, Hq * D: (Hq + Hkv) * D].reshape(n, Hkv, D)
    v = qkv[:, (Hq + Hkv) * D:].reshape(n, Hkv, D)
    q = rope_complex(q, pos, inv_freq)
    k = rope_complex(k, pos, inv_freq)
    grp = Hq // Hkv
    kk = k.repeat_interleave(grp, dim=1)
    vv = v.repeat_interleave(grp, dim=1)
    qh, kh, vh = (t.transpose(0, 1)[None] for t in (q, kk, vv))
    if attn_mask is None:
        o = F.scaled_dot_product_attention(qh, kh, vh, is_causal=True, scale=scale)
    else:
        o = F.scaled_dot_product_attention(qh, kh, vh, attn_mask=attn_mask[None, None], scale=scale)
    o = o[0].transpose(0, 1).reshape(n, Hq * D)
    h = x + F.linear(o, t64(lw["w_o"]))
    n2 = F.rms_norm(h, (h.shape[-1],), weight=t64(lw["mlp_norm"]), eps=s.rms_eps)
    y = h + F.linear(F.silu(F.linear(n2, t64(lw["w_gate"]))) * F.linear(n2, t64(lw["w_up"])),
                     t64(lw["w_down"]))
    return y, k, v
