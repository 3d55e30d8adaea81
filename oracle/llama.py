"""One Llama-3.1 decoder layer in float64 numpy (oracle; test infrastructure only).

The paper runs Llama3.1-8B-Instruct (Sec. 4) in bf16; its decoder block is the
standard pre-norm Llama block:

    h = x + W_o * Attn(RoPE(W_q n1), RoPE(W_k n1), W_v n1),   n1 = RMSNorm(x; g1)
    y = h + W_d (silu(W_g n2) * (W_u n2)),                    n2 = RMSNorm(h; g2)

Attention is grouped-query: query head j reads kv head floor(j / (Hq/Hkv)),
scores are scaled by 1/sqrt(D), and a row attends exactly the cache rows in its
own key range [lo, hi] (causal: hi = the row's own cache index).  The layer here
works on an arbitrary subset of rows so that the same function serves the full
prefill (all rows), the per-chunk isolated prefill (block-diagonal ranges) and
the selective recompute of Sec. 3.2 (selected rows over the whole blended cache).

RoPE is the rotate-half form used by Llama: dimension i is paired with i + D/2
and the pair is rotated by angle pos * w_i, w_i = theta^(-2i/D), with one of two
frequency scalings: Llama 3.1's (factor, low/high frequency factors, original
context), or YaRN's, which the paper's second model (Qwen2.5-7B-Instruct, Sec. 4)
uses.  YaRN also divides the attention logits by a temperature.  The q/k/v
projections may carry an additive bias (the layer dict's optional "b_qkv").

Precision.  Arithmetic is float64.  Sec. 4 of the paper states that the model's
computations run in bfloat16 (only the position adjustment in float32).  With
`Shape.act_bf16` set, the oracle stores in bf16 exactly the activations such a
model holds in bf16 - the RMSNorm outputs that feed a linear layer, q/k/v after
RoPE (k and v are the KV cache), the attention output, the SwiGLU product and
the re-aligned cached keys - and keeps everything else (accumulation, softmax,
the residual stream) in float64.  Without it every tensor stays float64.

`Shape.accum32` makes the linear layers accumulate in float32 instead.  It is
not the reference: it is a second correct implementation whose distance from the
float64 one measures how far two faithful implementations of the same bf16 model
drift apart through accumulation rounding alone (the floor any fp32-accumulating
kernel is judged against).
"""
from __future__ import annotations

import math
from dataclasses import dataclass

import numpy as np

F64 = np.float64

# frequency scaling of the rotary embedding
ROPE_PLAIN, ROPE_LLAMA3, ROPE_YARN = 0, 1, 2


@dataclass(frozen=True)
class Shape:
    hidden: int
    n_q_heads: int
    n_kv_heads: int
    head_dim: int
    mlp_dim: int
    rms_eps: float
    rope_theta: float
    rope_scaling: int = ROPE_PLAIN
    rs_factor: float = 8.0
    rs_low: float = 1.0
    rs_high: float = 4.0
    rs_orig_ctx: int = 8192
    act_bf16: bool = False
    accum32: bool = False

    @staticmethod
    def of(s, act_bf16: bool = False, accum32: bool = False) -> "Shape":
        """Copy the fields from any object that has them (e.g. a ModelShape)."""
        return Shape(s.hidden, s.n_q_heads, s.n_kv_heads, s.head_dim, s.mlp_dim,
                     float(s.rms_eps), float(s.rope_theta), int(s.rope_scaling),
                     float(s.rs_factor), float(s.rs_low), float(s.rs_high), int(s.rs_orig_ctx), act_bf16,
                     accum32)


def as64(a) -> np.ndarray:
    """Any float array (numpy or torch, incl. bf16) -> float64 numpy."""
    if hasattr(a, "detach"):
        a = a.detach().to("cpu")
        if str(a.dtype) == "torch.bfloat16":
            a = a.float()
        a = a.numpy()
    return np.asarray(a, dtype=F64)


def bf16_round(x) -> np.ndarray:
    """Round to the nearest bfloat16 (ties to even) through torch's conversion, as float64."""
    import torch
    t = torch.from_numpy(np.ascontiguousarray(x, dtype=np.float32))
    return t.to(torch.bfloat16).to(torch.float64).numpy()


def act(s: "Shape", x: np.ndarray) -> np.ndarray:
    """An activation the model stores: bf16 when s.act_bf16, else unchanged."""
    return bf16_round(x) if s.act_bf16 else x


# ----------------------------------------------------------------------------- RoPE

def rope_inv_freq(s: Shape) -> np.ndarray:
    """w_i = theta^(-2i/D), i < D/2, then the shape's frequency scaling.

    Llama 3.1 scaling (from the public Llama 3.1 model definition): with wavelength
    lam = 2*pi/w, frequencies whose wavelength is shorter than orig/high are
    kept; those longer than orig/low are divided by `factor`; in between the
    two are blended with s = (orig/lam - low)/(high - low):
        w' = (1 - s) * w / factor + s * w.
    YaRN scaling: `yarn_inv_freq`.
    """
    if s.rope_scaling == ROPE_YARN:
        return yarn_inv_freq(s)
    D = s.head_dim
    i = np.arange(D // 2, dtype=F64)
    w = s.rope_theta ** (-(2.0 * i) / D)
    if s.rope_scaling == ROPE_PLAIN:
        return w
    assert s.rope_scaling == ROPE_LLAMA3, s.rope_scaling
    out = np.empty_like(w)
    lo_wavelen = s.rs_orig_ctx / s.rs_low     # longest wavelength still blended
    hi_wavelen = s.rs_orig_ctx / s.rs_high    # shortest wavelength blended
    for j in range(w.size):
        lam = 2.0 * math.pi / w[j]
        if lam < hi_wavelen:
            out[j] = w[j]
        elif lam > lo_wavelen:
            out[j] = w[j] / s.rs_factor
        else:
            sm = (s.rs_orig_ctx / lam - s.rs_low) / (s.rs_high - s.rs_low)
            out[j] = (1.0 - sm) * w[j] / s.rs_factor + sm * w[j]
    return out


def yarn_inv_freq(s: Shape) -> np.ndarray:
    """YaRN's "NTK-by-parts" interpolation (Peng et al., YaRN, Sec. 3.2), in that
    paper's notation, with s.rs_factor = s, s.rs_low = alpha, s.rs_high = beta and
    s.rs_orig_ctx = L (the context length the model was trained at):

        theta_d  = b^(-2d/|D|)               frequency of rotation pair d
        lambda_d = 2 pi / theta_d            its wavelength in tokens
        r(d)     = L / lambda_d              turns it makes over the original context
        gamma(r) = 0 if r < alpha, 1 if r > beta, (r - alpha)/(beta - alpha) otherwise
        h(theta_d) = (1 - gamma(r(d))) theta_d / s + gamma(r(d)) theta_d

    Pairs that turn fewer than alpha times over L are interpolated by s (position
    interpolation), pairs that turn more than beta times are left alone, and the
    ramp is linear in r between them."""
    D = s.head_dim
    L, scale, alpha, beta = float(s.rs_orig_ctx), float(s.rs_factor), float(s.rs_low), float(s.rs_high)
    out = np.empty(D // 2, dtype=F64)
    for d in range(D // 2):
        theta = s.rope_theta ** (-2.0 * d / D)
        lam = 2.0 * math.pi / theta
        r = L / lam
        if r < alpha:
            gamma = 0.0
        elif r > beta:
            gamma = 1.0
        else:
            gamma = (r - alpha) / (beta - alpha)
        out[d] = (1.0 - gamma) * theta / scale + gamma * theta
    return out


def logit_scale(s: Shape) -> float:
    """Factor applied to q.k before the softmax: 1/sqrt(D).  YaRN (Sec. 3.4 of its
    paper) also divides the logits by a temperature t with sqrt(1/t) = 0.1 ln(s) + 1,
    i.e. multiplies them by (0.1 ln(s) + 1)^2."""
    base = 1.0 / math.sqrt(s.head_dim)
    if s.rope_scaling == ROPE_YARN:
        m = 0.1 * math.log(s.rs_factor) + 1.0
        return base * m * m
    return base


def rope_cos_sin(s: Shape, pos) -> tuple[np.ndarray, np.ndarray]:
    """cos/sin of pos * w_i, float64, shape [len(pos), D/2]."""
    pos = np.asarray(pos, dtype=F64).reshape(-1, 1)
    ang = pos * rope_inv_freq(s).reshape(1, -1)
    return np.cos(ang), np.sin(ang)


def apply_rope(x: np.ndarray, cos: np.ndarray, sin: np.ndarray) -> np.ndarray:
    """Rotate-half RoPE.  x: [n, heads, D]; cos/sin: [n, D/2].

    For pair (x_a, x_b) = (x[i], x[i + D/2]):  x_a' = x_a c - x_b s,  x_b' = x_b c + x_a s.
    """
    half = x.shape[-1] // 2
    a, b = x[..., :half], x[..., half:]
    c, s_ = cos[:, None, :], sin[:, None, :]
    return np.concatenate([a * c - b * s_, b * c + a * s_], axis=-1)


# ----------------------------------------------------------------------------- block pieces

def rmsnorm(x: np.ndarray, g: np.ndarray, eps: float) -> np.ndarray:
    """x / sqrt(mean(x^2) + eps) * g over the last axis."""
    x = as64(x)
    ms = np.mean(x * x, axis=-1, keepdims=True)
    return x / np.sqrt(ms + eps) * as64(g)


def linear(x: np.ndarray, w: np.ndarray, accum32: bool = False) -> np.ndarray:
    """y = x W^T with W stored [out_features, in_features] (float32 products and sums
    when accum32)."""
    if accum32:
        return (np.asarray(x, np.float32) @ np.asarray(as64(w), np.float32).T).astype(F64)
    return as64(x) @ as64(w).T


def silu(x: np.ndarray) -> np.ndarray:
    return x / (1.0 + np.exp(-x))


def attention_rows(s: Shape, q: np.ndarray, k_cache: np.ndarray, v_cache: np.ndarray,
                   row_hi, row_lo=None, block: int = 256) -> np.ndarray:
    """Causal GQA attention of selected rows over a KV cache.

    q:        [m, Hq, D]  (already rotated)
    k_cache:  [n_cache, Hkv, D], v_cache: [n_cache, Hkv, D]
    row_hi:   [m] last cache row each query row may read (its own cache index)
    row_lo:   [m] first cache row it may read (None: 0)
    returns   [m, Hq, D]

    out[r, j] = sum_t softmax_t(c * q[r,j] . k[t, g]) v[t, g] over lo_r <= t <= hi_r,
    g = j // (Hq / Hkv), c = logit_scale(s) (1/sqrt(D) without YaRN); softmax taken
    with max subtraction.
    """
    m, Hq, D = q.shape
    Hkv = k_cache.shape[1]
    grp = Hq // Hkv
    row_hi = np.asarray(row_hi, dtype=np.int64)
    row_lo = np.zeros(m, dtype=np.int64) if row_lo is None else np.asarray(row_lo, dtype=np.int64)
    out = np.zeros((m, Hq, D), dtype=F64)
    scale = logit_scale(s)
    for r0 in range(0, m, block):
        r1 = min(m, r0 + block)
        lo, hi = row_lo[r0:r1], row_hi[r0:r1]
        t_end = int(hi.max()) + 1
        t_beg = int(lo.min())
        t = np.arange(t_beg, t_end)
        allowed = (t[None, :] >= lo[:, None]) & (t[None, :] <= hi[:, None])
        for j in range(Hq):
            g = j // grp
            kk = as64(k_cache[t_beg:t_end, g, :])
            vv = as64(v_cache[t_beg:t_end, g, :])
            sc = (q[r0:r1, j, :] @ kk.T) * scale
            sc = np.where(allowed, sc, -np.inf)
            sc = sc - sc.max(axis=1, keepdims=True)
            p = np.exp(sc)
            p /= p.sum(axis=1, keepdims=True)
            out[r0:r1, j, :] = p @ vv
    return out


def qkv_rows(s: Shape, lw: dict, x: np.ndarray, rope_pos) -> tuple[np.ndarray, np.ndarray, np.ndarray]:
    """RMSNorm -> QKV projection (+ bias) -> RoPE at `rope_pos`.  Returns q [m,Hq,D], k, v [m,Hkv,D]."""
    D, Hq, Hkv = s.head_dim, s.n_q_heads, s.n_kv_heads
    n1 = act(s, rmsnorm(x, lw["attn_norm"], s.rms_eps))
    qkv = linear(n1, lw["w_qkv"], s.accum32)
    if lw.get("b_qkv") is not None:
        qkv = qkv + as64(lw["b_qkv"])
    m = x.shape[0]
    q = qkv[:, : Hq * D].reshape(m, Hq, D)
    k = qkv[:, Hq * D: (Hq + Hkv) * D].reshape(m, Hkv, D)
    v = qkv[:, (Hq + Hkv) * D:].reshape(m, Hkv, D)
    c, sn = rope_cos_sin(s, rope_pos)
    return act(s, apply_rope(q, c, sn)), act(s, apply_rope(k, c, sn)), act(s, v)


def k_rows(s: Shape, lw: dict, x: np.ndarray, rope_pos) -> np.ndarray:
    """Only the key projection (RMSNorm -> W_k (+ bias) -> RoPE), [m, Hkv, D]."""
    D, Hq, Hkv = s.head_dim, s.n_q_heads, s.n_kv_heads
    n1 = act(s, rmsnorm(x, lw["attn_norm"], s.rms_eps))
    wk = as64(lw["w_qkv"])[Hq * D: (Hq + Hkv) * D]
    k = linear(n1, wk, s.accum32)
    if lw.get("b_qkv") is not None:
        k = k + as64(lw["b_qkv"])[Hq * D: (Hq + Hkv) * D]
    k = k.reshape(x.shape[0], Hkv, D)
    c, sn = rope_cos_sin(s, rope_pos)
    return act(s, apply_rope(k, c, sn))


def attn_out_mlp(s: Shape, lw: dict, x: np.ndarray, attn: np.ndarray) -> np.ndarray:
    """x + O-proj(attn), then + SwiGLU MLP of its RMSNorm.  attn: [m, Hq*D]."""
    h = as64(x) + linear(attn, lw["w_o"], s.accum32)
    n2 = act(s, rmsnorm(h, lw["mlp_norm"], s.rms_eps))
    a = act(s, silu(linear(n2, lw["w_gate"], s.accum32)) * linear(n2, lw["w_up"], s.accum32))
    return h + linear(a, lw["w_down"], s.accum32)


def layer_rows(s: Shape, lw: dict, x: np.ndarray, row_idx, rope_pos, k_cache: np.ndarray,
               v_cache: np.ndarray, row_lo=None) -> np.ndarray:
    """One decoder layer applied to rows `row_idx` of a sequence held in a KV cache.

    The rows' fresh K/V are written into the cache (in place) BEFORE any
    attention of this layer, then each row attends cache rows [lo, row_idx].
    Returns the rows' layer output (float64 [m, H]).
    """
    row_idx = np.asarray(row_idx, dtype=np.int64)
    q, k, v = qkv_rows(s, lw, x, rope_pos)
    k_cache[row_idx] = k
    v_cache[row_idx] = v
    a = act(s, attention_rows(s, q, k_cache, v_cache, row_idx, row_lo))
    return attn_out_mlp(s, lw, x, a.reshape(a.shape[0], -1))
