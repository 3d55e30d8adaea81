"""How far two faithful implementations of the Llama-3.1-8B-shaped bf16 layer can drift
apart (CPU, oracle only).

The model stores some activations in bf16 (Sec. 4: the model computes in bf16): the
RMSNorm outputs that feed a linear layer, q/k/v, the attention output and the SwiGLU
product.  A bf16 rounding is a step function, so a perturbation of one part in 10^7
before it (float32 instead of float64 accumulation, an RMSNorm evaluated in float32,
softmax weights held in fp16) now and then moves a value to the neighbouring bf16
number; one such flip in an RMSNorm output reaches all 14,336 gate/up sums and flips a
few per cent of the SwiGLU roundings, which the down projection adds up into a change of
a few 1e-3 on every element of the layer output.  This test measures that drift on
layer 0 of the 8B-shaped model (random N(0, 0.02) weights, 3,904-token context, 64
sampled rows): each single fp32-level change moves the layer output by more than 1e-3
mean-abs against the float64 oracle, i.e. the same order as the stated per-layer bar of
2e-3, so the absolute form of that bar cannot separate a correct fp32 kernel from the
oracle on early layers.  (Measured here: ~2.5e-3 to 3.7e-3.)
"""
import numpy as np
import pytest

from oracle import blend, llama
from oracle.llama import Shape
from paper_2609_09768_gb300 import synth

pytestmark = pytest.mark.slow


def _layer0(shape, w, x0, smp, s, rms32=False, p16=False):
    lw = {k: llama.as64(v) for k, v in w["layers"][0].items()}
    N = x0.shape[0]
    D, Hq, Hkv = s.head_dim, s.n_q_heads, s.n_kv_heads

    def norm(x, g):
        if not rms32:
            return llama.rmsnorm(x, g, s.rms_eps)
        x32 = x.astype(np.float32)
        ms = np.mean(x32 * x32, axis=-1, keepdims=True, dtype=np.float32)
        return (x32 * (np.float32(1) / np.sqrt(ms + np.float32(s.rms_eps))) * g.astype(np.float32)).astype(np.float64)

    n1 = llama.act(s, norm(x0, lw["attn_norm"]))
    qkv = llama.linear(n1, lw["w_qkv"], s.accum32)
    q = qkv[:, : Hq * D].reshape(N, Hq, D)
    k = qkv[:, Hq * D: (Hq + Hkv) * D].reshape(N, Hkv, D)
    v = qkv[:, (Hq + Hkv) * D:].reshape(N, Hkv, D)
    c, sn = llama.rope_cos_sin(s, np.arange(N))
    q, k, v = llama.act(s, llama.apply_rope(q, c, sn)), llama.act(s, llama.apply_rope(k, c, sn)), llama.act(s, v)
    if p16:
        # softmax weights held in fp16 (scaled into its normal range), sums in float64
        out = np.zeros((len(smp), Hq, D))
        for i, r in enumerate(smp):
            for h in range(Hq):
                g = h // (Hq // Hkv)
                sc = (q[r, h] @ k[: r + 1, g].T) * llama.logit_scale(s)
                p = (np.exp(sc - sc.max()) * 128.0).astype(np.float16).astype(np.float64)
                out[i, h] = (p @ v[: r + 1, g]) / p.sum()
    else:
        out = llama.attention_rows(s, q[smp], k, v, smp)
    a = llama.act(s, out).reshape(len(smp), -1)
    return llama.attn_out_mlp(s, lw, x0[smp], a)


def test_fp32_level_changes_move_an_8b_layer_output_by_the_order_of_the_bar():
    wl = synth.WORKLOADS["l8b_1layer"]
    shape = wl.shape
    w = synth.make_model(shape, 0)
    x0 = blend.embed_rows(w["embed"], wl.tokens().numpy())
    smp = np.sort(np.random.default_rng(7).choice(wl.n_total, 64, replace=False))
    base = _layer0(shape, w, x0, smp, Shape.of(shape, act_bf16=True))
    drift = {
        "float32 accumulation": _layer0(shape, w, x0, smp, Shape.of(shape, act_bf16=True, accum32=True)),
        "float32 RMSNorm": _layer0(shape, w, x0, smp, Shape.of(shape, act_bf16=True), rms32=True),
        "fp16 softmax weights": _layer0(shape, w, x0, smp, Shape.of(shape, act_bf16=True), p16=True),
    }
    rms = float(np.sqrt(np.mean(base ** 2)))
    for name, y in drift.items():
        d = np.abs(y - base)
        print(f"layer-0 output drift, {name}: mean {d.mean():.3e} max {d.max():.3e} (output rms {rms:.3f})")
        assert d.mean() > 1e-3, (name, d.mean())
        # ... while staying far inside the same bar taken relative to the output's RMS
        assert d.mean() < 2e-3 * rms and d.max() < 2e-2 * rms, (name, d.mean(), d.max())
