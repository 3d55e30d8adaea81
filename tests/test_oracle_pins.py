"""Pins for the CPU oracle (no GPU): closed forms, library routines, the paper's
invariants and brute force on tiny inputs.  Each pin is chosen so that a
plausible slip in the oracle (a sign, a dropped term, a wrong head index, a
transposed operand) breaks at least one of them; `test_planted_mistakes`
checks that claim by planting such slips in the oracle and re-running pins."""
import json
import math
import os

import numpy as np
import torch

from oracle import blend, llama
from oracle.llama import Shape
from tests import torch_ref
from paper_2609_09768_gb300 import synth

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")

MINI = synth.ModelShape(hidden=64, n_q_heads=4, n_kv_heads=2, head_dim=16, mlp_dim=96,
                        n_layers=2, vocab=97, rms_eps=1e-5, rope_theta=10000.0)
# seven q heads per kv head, YaRN (factor 4 over an original context of 16 tokens), q/k/v bias
MINI_YARN = synth.ModelShape(hidden=64, n_q_heads=7, n_kv_heads=1, head_dim=16, mlp_dim=96,
                             n_layers=2, vocab=97, rms_eps=1e-6, rope_theta=10000.0, rope_scaling=2,
                             rs_factor=4.0, rs_low=1.0, rs_high=32.0, rs_orig_ctx=16, qkv_bias=True)
MINI_L3 = synth.ModelShape(hidden=64, n_q_heads=4, n_kv_heads=2, head_dim=16, mlp_dim=96,
                           n_layers=2, vocab=97, rms_eps=1e-5, rope_theta=500000.0, rope_scaling=1,
                           rs_factor=8.0, rs_low=1.0, rs_high=4.0, rs_orig_ctx=64)


def model(shape, seed=0, n_layers=None):
    shp = shape if n_layers is None else shape.with_layers(n_layers)
    m = synth.make_model(shp, seed)
    m["layers_np"] = [{k: llama.as64(v) for k, v in lw.items()} for lw in m["layers"]]
    return m


def rel(a, b):
    a, b = np.asarray(a, dtype=np.float64), np.asarray(b, dtype=np.float64)
    return float(np.max(np.abs(a - b)) / max(1e-300, np.max(np.abs(b))))


# ------------------------------------------------------------------------------------ RoPE

def test_rope_direction_closed_form():
    """RoFormer's R_m = [[cos m, -sin m],[sin m, cos m]] on a single pair (D=2, w=1)."""
    s = Shape(2, 1, 1, 2, 4, 1e-5, 10000.0)
    for m_ in (0, 1, 3, 1000):
        c, sn = llama.rope_cos_sin(s, [m_])
        y = llama.apply_rope(np.array([[[1.0, 0.0]]]), c, sn)[0, 0]
        assert np.allclose(y, [math.cos(m_), math.sin(m_)], atol=1e-15)
        y = llama.apply_rope(np.array([[[0.0, 1.0]]]), c, sn)[0, 0]
        assert np.allclose(y, [-math.sin(m_), math.cos(m_)], atol=1e-15)


def test_rope_composition_and_norm():
    """R(a) R(b) = R(a + b) (what re-alignment relies on) and rotations keep norms."""
    s = Shape.of(MINI_L3)
    rng = np.random.default_rng(0)
    x = rng.standard_normal((5, 3, s.head_dim))
    a, b = np.array([0, 7, 100, 511, 3]), np.array([5, 9, 0, 1024, 77])
    ca, sa = llama.rope_cos_sin(s, a)
    cb, sb = llama.rope_cos_sin(s, b)
    cab, sab = llama.rope_cos_sin(s, a + b)
    two = llama.apply_rope(llama.apply_rope(x, cb, sb), ca, sa)
    one = llama.apply_rope(x, cab, sab)
    assert rel(two, one) < 1e-12
    assert np.allclose(np.linalg.norm(one, axis=-1), np.linalg.norm(x, axis=-1), rtol=1e-13)


def test_rope_relative_position():
    """<R(m)q, R(n)k> depends only on m - n."""
    s = Shape.of(MINI)
    rng = np.random.default_rng(1)
    q, k = rng.standard_normal((2, 1, 1, s.head_dim))
    def dot(m_, n_):
        cm, sm = llama.rope_cos_sin(s, [m_]); cn, sn = llama.rope_cos_sin(s, [n_])
        return float(np.sum(llama.apply_rope(q, cm, sm) * llama.apply_rope(k, cn, sn)))
    assert abs(dot(10, 3) - dot(107, 100)) < 1e-12
    assert abs(dot(10, 3) - dot(3, 10)) > 1e-6   # not symmetric: direction matters


def test_rope_matches_complex_multiplication():
    s = Shape.of(MINI_L3)
    rng = np.random.default_rng(2)
    x = rng.standard_normal((6, 2, s.head_dim))
    pos = np.array([0, 1, 2, 63, 64, 4000])
    c, sn = llama.rope_cos_sin(s, pos)
    ours = llama.apply_rope(x, c, sn)
    ref = torch_ref.rope_complex(torch.as_tensor(x), torch.as_tensor(pos),
                                 torch.as_tensor(llama.rope_inv_freq(s)))
    assert rel(ours, ref.numpy()) < 1e-13


def test_llama3_frequency_bands():
    """D=128, theta=5e5, orig 8192, low 1, high 4: wavelength 2*pi*theta^(2i/D) is below
    2048 for i <= 28 (kept), above 8192 for i >= 35 (divided by 8), and blended in between,
    continuously at both band edges."""
    s = Shape(4096, 32, 8, 128, 14336, 1e-5, 500000.0, llama.ROPE_LLAMA3, 8.0, 1.0, 4.0, 8192)
    plain = Shape(4096, 32, 8, 128, 14336, 1e-5, 500000.0, llama.ROPE_PLAIN)
    w = llama.rope_inv_freq(s)
    w0 = llama.rope_inv_freq(plain)
    assert w0[0] == 1.0 and abs(w0[1] - 500000.0 ** (-2 / 128)) < 1e-18
    assert np.array_equal(w[:29], w0[:29])
    assert np.allclose(w[35:], w0[35:] / 8.0, rtol=1e-15)
    mid = slice(29, 35)
    assert np.all(w[mid] < w0[mid]) and np.all(w[mid] > w0[mid] / 8.0)
    # blend weight s in (0,1) and monotone in i
    lam = 2 * math.pi / w0[mid]
    sm = (8192 / lam - 1.0) / 3.0
    assert np.all((sm > 0) & (sm < 1)) and np.all(np.diff(sm) < 0)


def _yarn(D=128, theta=1e6, L=2048, scale=4.0, alpha=1.0, beta=32.0):
    return Shape(4096, 32, 8, D, 14336, 1e-6, theta, llama.ROPE_YARN, scale, alpha, beta, L)


def test_yarn_at_scale_one_is_plain_rope():
    """s = 1: interpolation and extrapolation coincide, and the temperature is 1 (ln 1 = 0)."""
    for D, theta, L in ((128, 1e6, 2048), (64, 1e4, 256)):
        y = _yarn(D, theta, L, scale=1.0)
        plain = Shape(4096, 32, 8, D, 14336, 1e-6, theta, llama.ROPE_PLAIN)
        assert np.allclose(llama.rope_inv_freq(y), llama.rope_inv_freq(plain), rtol=1e-15, atol=0)
        assert llama.logit_scale(y) == llama.logit_scale(plain) == 1.0 / math.sqrt(D)


def test_yarn_bands_interpolate_and_keep():
    """Pairs that turn fewer than alpha times over the original context L are position-
    interpolated: their angle at position s*p equals the plain angle at p.  Pairs that
    turn more than beta times keep the plain angle.  In between the frequency lies
    strictly between the two and falls monotonically with the pair index."""
    y = _yarn()
    plain = Shape(4096, 32, 8, 128, 14336, 1e-6, 1e6, llama.ROPE_PLAIN)
    w0 = llama.rope_inv_freq(plain)
    turns = 2048 * w0 / (2 * math.pi)
    low, high, mid = turns < 1.0, turns > 32.0, (turns >= 1.0) & (turns <= 32.0)
    assert low.sum() > 10 and high.sum() > 5 and mid.sum() > 5
    p = np.array([0, 1, 3, 1000, 30000])
    cy, sy = llama.rope_cos_sin(y, 4 * p)
    c0, s0 = llama.rope_cos_sin(plain, p)
    assert np.allclose(cy[:, low], c0[:, low], atol=1e-9) and np.allclose(sy[:, low], s0[:, low], atol=1e-9)
    cy, sy = llama.rope_cos_sin(y, p)
    assert np.allclose(cy[:, high], c0[:, high], atol=1e-9) and np.allclose(sy[:, high], s0[:, high], atol=1e-9)
    w = llama.rope_inv_freq(y)
    assert np.all(w[mid] < w0[mid]) and np.all(w[mid] > w0[mid] / 4.0)
    assert np.all(np.diff(w) < 0)


def test_yarn_ramp_is_continuous_in_the_original_context():
    """gamma is continuous, so a pair's frequency moves continuously as L crosses the
    lengths at which it makes exactly alpha or beta turns."""
    plain = Shape(4096, 32, 8, 128, 14336, 1e-6, 1e6, llama.ROPE_PLAIN)
    w0 = llama.rope_inv_freq(plain)
    d = 40
    for n_turns in (1.0, 32.0):
        L_edge = n_turns * 2 * math.pi / w0[d]
        lo = llama.yarn_inv_freq(_yarn(L=L_edge * (1 - 1e-9)))[d]
        hi = llama.yarn_inv_freq(_yarn(L=L_edge * (1 + 1e-9)))[d]
        assert abs(lo - hi) < 1e-7 * w0[d]


def test_yarn_equals_llama3_rule_with_the_same_bounds():
    """Llama 3.1's frequency rule is the same NTK-by-parts blend (low/high frequency
    factors in the roles of alpha/beta), written here independently: with equal
    bounds the two definitions give the same frequencies."""
    for D, theta, L, s_, a, b in ((128, 5e5, 8192, 8.0, 1.0, 4.0), (64, 1e4, 300, 3.0, 2.0, 16.0)):
        y = _yarn(D, theta, L, s_, a, b)
        l3 = Shape(4096, 32, 8, D, 14336, 1e-6, theta, llama.ROPE_LLAMA3, s_, a, b, L)
        assert np.allclose(llama.rope_inv_freq(y), llama.rope_inv_freq(l3), rtol=1e-14, atol=0)


def test_yarn_temperature_closed_form():
    """Two keys, values 1 and 0: the output is the softmax weight of the first key,
    sigmoid(c * (q.k1 - q.k2)).  With s = e^10, sqrt(1/t) = 0.1*10 + 1 = 2, so
    c = 4/sqrt(D)."""
    D = 16
    y = Shape(64, 2, 1, D, 96, 1e-6, 1e4, llama.ROPE_YARN, math.exp(10.0), 1.0, 32.0, 64)
    rng = np.random.default_rng(7)
    q = rng.standard_normal((1, 2, D))
    k = rng.standard_normal((2, 1, D))
    v = np.zeros((2, 1, D)); v[0, 0, :] = 1.0
    out = llama.attention_rows(y, q, k, v, [1])
    for j in range(2):
        delta = float(q[0, j] @ k[0, 0] - q[0, j] @ k[1, 0])
        expect = 1.0 / (1.0 + math.exp(-4.0 * delta / math.sqrt(D)))
        assert np.allclose(out[0, j], expect, rtol=1e-13)


def test_qkv_bias_closed_form():
    """Zero projection weights: q, k are the rotated bias and v the bias itself; the
    key-only path adds the key slice of the same bias."""
    s = Shape.of(MINI_YARN)
    D, Hq, Hkv = s.head_dim, s.n_q_heads, s.n_kv_heads
    rng = np.random.default_rng(8)
    b = rng.standard_normal((Hq + 2 * Hkv) * D)
    lw = {"attn_norm": np.ones(64), "w_qkv": np.zeros(((Hq + 2 * Hkv) * D, 64)), "b_qkv": b}
    x = rng.standard_normal((3, 64))
    pos = np.array([0, 5, 40])
    q, k, v = llama.qkv_rows(s, lw, x, pos)
    c, sn = llama.rope_cos_sin(s, pos)
    assert np.allclose(q, llama.apply_rope(np.broadcast_to(b[: Hq * D].reshape(1, Hq, D), (3, Hq, D)), c, sn))
    kb = b[Hq * D: (Hq + Hkv) * D].reshape(1, Hkv, D)
    assert np.allclose(k, llama.apply_rope(np.broadcast_to(kb, (3, Hkv, D)), c, sn))
    assert np.allclose(v, np.broadcast_to(b[(Hq + Hkv) * D:].reshape(1, Hkv, D), (3, Hkv, D)))
    lw["w_qkv"] = rng.standard_normal(lw["w_qkv"].shape) * 0.1
    q, k, v = llama.qkv_rows(s, lw, x, pos)
    assert rel(llama.k_rows(s, lw, x, pos), k) < 1e-14


# ------------------------------------------------------------------------------------ block parts

def test_rmsnorm_and_silu_match_torch():
    rng = np.random.default_rng(3)
    x = rng.standard_normal((7, 64)) * 3
    g = rng.standard_normal(64)
    ref = torch.nn.functional.rms_norm(torch.as_tensor(x), (64,), torch.as_tensor(g), 1e-5)
    assert rel(llama.rmsnorm(x, g, 1e-5), ref.numpy()) < 1e-14
    assert np.allclose(np.sqrt(np.mean(llama.rmsnorm(x, np.ones(64), 0.0) ** 2, -1)), 1.0)
    assert rel(llama.silu(x), torch.nn.functional.silu(torch.as_tensor(x)).numpy()) < 1e-14


def _rand_qkv(m, n, Hq, Hkv, D, seed):
    rng = np.random.default_rng(seed)
    return (rng.standard_normal((m, Hq, D)), rng.standard_normal((n, Hkv, D)),
            rng.standard_normal((n, Hkv, D)))


def test_attention_matches_sdpa_causal_gqa():
    s = Shape.of(MINI)
    n = 37
    q, k, v = _rand_qkv(n, n, 4, 2, 16, 4)
    ours = llama.attention_rows(s, q, k, v, np.arange(n), block=8)
    qt, kt, vt = (torch.as_tensor(t).transpose(0, 1)[None] for t in (q, np.repeat(k, 2, 1), np.repeat(v, 2, 1)))
    ref = torch.nn.functional.scaled_dot_product_attention(qt, kt, vt, is_causal=True)[0].transpose(0, 1)
    assert rel(ours, ref.numpy()) < 1e-13


def test_attention_brute_force_sparse_rows():
    """Selected rows with key ranges [lo, hi], against explicit per-(row, head, key) loops."""
    s = Shape.of(MINI)
    n = 23
    rows = np.array([2, 5, 6, 15, 22])
    lo = np.array([0, 3, 3, 10, 0])
    q, k, v = _rand_qkv(len(rows), n, 4, 2, 16, 5)
    ours = llama.attention_rows(s, q, k, v, rows, lo)
    for a, (hi, l0) in enumerate(zip(rows, lo)):
        for j in range(4):
            g = j // 2
            sc = [sum(q[a, j, d] * k[t, g, d] for d in range(16)) / 4.0 for t in range(l0, hi + 1)]
            mx = max(sc)
            w = [math.exp(x - mx) for x in sc]
            z = sum(w)
            o = [sum(w[i] / z * v[l0 + i, g, d] for i in range(len(w))) for d in range(16)]
            assert np.allclose(ours[a, j], o, atol=1e-12)


def test_attention_special_cases():
    s = Shape.of(MINI)
    n = 9
    q, k, v = _rand_qkv(n, n, 4, 2, 16, 6)
    # a row that sees only itself returns its own value
    out = llama.attention_rows(s, q, k, v, np.arange(n), np.arange(n))
    assert np.allclose(out, np.repeat(v, 2, 1), atol=1e-15)
    # zero queries: uniform average of the visible values
    out = llama.attention_rows(s, np.zeros_like(q), k, v, np.arange(n))
    for t in range(n):
        assert np.allclose(out[t, 3], v[: t + 1, 1].mean(0), atol=1e-14)


def test_layer_matches_torch_library_block():
    m = model(MINI)
    s = Shape.of(MINI)
    n = 29
    x = llama.as64(synth.randn_bf16((n, 64), 11))
    lw = m["layers_np"][0]
    kc = np.zeros((n, 2, 16)); vc = np.zeros_like(kc)
    ours = llama.layer_rows(s, lw, x, np.arange(n), np.arange(n), kc, vc)
    inv = torch.as_tensor(llama.rope_inv_freq(s))
    ref, kr, vr = torch_ref.layer_full(s, lw, torch.as_tensor(x), inv, torch.arange(n))
    assert rel(ours, ref.numpy()) < 1e-12
    assert rel(kc, kr.numpy()) < 1e-12 and rel(vc, vr.numpy()) < 1e-12


def test_layer_llama3_scaled_block_diagonal_matches_torch():
    """Per-chunk isolated prefill as one block-diagonal pass equals torch with an explicit mask."""
    m = model(MINI_L3)
    s = Shape.of(MINI_L3)
    starts = [0, 5, 12, 20]
    n = starts[-1]
    seg = np.concatenate([[starts[c]] * (starts[c + 1] - starts[c]) for c in range(3)])
    pos = np.arange(n) - seg
    x = llama.as64(synth.randn_bf16((n, 64), 12))
    kc = np.zeros((n, 2, 16)); vc = np.zeros_like(kc)
    ours = llama.layer_rows(s, m["layers_np"][1], x, np.arange(n), pos, kc, vc, row_lo=seg)
    t = np.arange(n)
    mask = torch.as_tensor((t[None, :] >= seg[:, None]) & (t[None, :] <= t[:, None]))
    inv = torch.as_tensor(llama.rope_inv_freq(s))
    ref, _, _ = torch_ref.layer_full(s, m["layers_np"][1], torch.as_tensor(x), inv, torch.as_tensor(pos), mask)
    assert rel(ours, ref.numpy()) < 1e-12


def test_layer_yarn_gqa7_bias_matches_torch():
    """Seven q heads per kv head, YaRN frequencies and temperature, q/k/v bias: the oracle's
    layer against torch's block with the bias in F.linear and the temperature as SDPA's
    scale, over positions up to 4x the original context."""
    m = model(MINI_YARN)
    s = Shape.of(MINI_YARN)
    n = 64
    x = llama.as64(synth.randn_bf16((n, 64), 13))
    lw = m["layers_np"][0]
    assert "b_qkv" in lw
    kc = np.zeros((n, 1, 16)); vc = np.zeros_like(kc)
    ours = llama.layer_rows(s, lw, x, np.arange(n), np.arange(n), kc, vc)
    inv = torch.as_tensor(llama.rope_inv_freq(s))
    mult = (0.1 * math.log(4.0) + 1.0) ** 2
    ref, kr, vr = torch_ref.layer_full(s, lw, torch.as_tensor(x), inv, torch.arange(n), scale=mult / 4.0)
    assert rel(ours, ref.numpy()) < 1e-12
    assert rel(kc, kr.numpy()) < 1e-12 and rel(vc, vr.numpy()) < 1e-12
    # without the temperature or the bias the layer differs
    ref2, _, _ = torch_ref.layer_full(s, lw, torch.as_tensor(x), inv, torch.arange(n))
    assert rel(ours, ref2.numpy()) > 1e-4
    lw_nb = dict(lw); lw_nb.pop("b_qkv")
    ref3, _, _ = torch_ref.layer_full(s, lw_nb, torch.as_tensor(x), inv, torch.arange(n), scale=mult / 4.0)
    assert rel(ours, ref3.numpy()) > 1e-4


# ------------------------------------------------------------------------------------ the method

def _request(shape, starts, n_query, seed=0):
    m = model(shape, seed)
    toks = synth.make_tokens(shape, starts[-1] + n_query, seed + 1)
    x0 = blend.embed_rows(m["embed"], toks.numpy())
    return m, x0


def test_prefix_invariance_and_realign():
    """Chunk 0's isolated cache equals full-attention K/V (prefix caching is exact, Sec. 1),
    and at layer 0 the re-aligned keys of every chunk equal the fresh global-position keys."""
    s = Shape.of(MINI)
    starts = [0, 11, 20, 33]
    m, x0 = _request(MINI, starts, 0)
    cc = blend.chunk_caches(s, m["layers_np"], x0, starts)
    full = blend.full_prefill(s, m["layers_np"], x0)
    a, b = 0, starts[1]
    assert rel(cc["k"][:, a:b], full["k"][:, a:b]) < 1e-12
    assert rel(cc["v"][:, a:b], full["v"][:, a:b]) < 1e-12
    re = blend.realign(s, cc["k"], starts)
    assert rel(re[0], full["k"][0]) < 1e-12          # layer 0: depends on token and position only
    assert rel(cc["v"][0], full["v"][0]) < 1e-12
    assert rel(re[1, starts[1]:], full["k"][1, starts[1]:]) > 1e-3   # later chunks miss cross-attention


def test_hkvd_deviation_cases():
    rng = np.random.default_rng(7)
    k = rng.standard_normal((10, 2, 8))
    assert np.allclose(blend.hkvd_deviation(k, np.zeros_like(k)), np.sum(k.reshape(10, -1) ** 2, 1))
    assert np.all(blend.hkvd_deviation(k, k) == 0)
    d = np.zeros_like(k); d[3, 1, 5] = 2.0; d[7, 0, 0] = -3.0
    dev = blend.hkvd_deviation(k + d, k)
    assert np.allclose(dev, [0, 0, 0, 4, 0, 0, 0, 9, 0, 0])


def test_topk_brute_force_with_ties():
    rng = np.random.default_rng(8)
    for trial in range(30):
        n = int(rng.integers(1, 40))
        dev = rng.integers(0, 6, n).astype(np.float64)   # many ties
        for k in (0, 1, n // 3, n):
            got = blend.topk_select(dev, k)
            # brute force: rank of i = #{j: dev_j > dev_i or (dev_j == dev_i and j < i)}
            want = sorted(i for i in range(n)
                          if sum(1 for j in range(n) if dev[j] > dev[i] or (dev[j] == dev[i] and j < i)) < k)
            assert list(got) == want


def test_num_selected_matches_paper_ratio():
    with open(os.path.join(GOLDEN, "paper_constants.json")) as f:
        g = json.load(f)
    r = g["recompute_ratio"]["value"]
    assert r == 0.15
    # context sizes of the four workloads (chunks of at most 512 tokens, Sec. 4)
    assert [blend.num_selected(r, n) for n in (512, 3840, 32768, 123904)] == [76, 576, 4915, 18585]
    assert 242 * g["max_chunk_tokens"]["value"] + 128 <= g["long_context_tokens"]["value"]
    assert blend.num_selected(1.0, 123904) == 123904 and blend.num_selected(0.0, 777) == 0


def _sel(shape, starts, nq, r, check_layer=1, forced=None, seed=0):
    s = Shape.of(shape)
    m, x0 = _request(shape, starts, nq, seed)
    cc = blend.chunk_caches(s, m["layers_np"], x0[: starts[-1]], starts)
    res = blend.selective_prefill(s, m["layers_np"], x0, starts, nq, r, cc["k"], cc["v"],
                                  check_layer, forced, m["final_norm"])
    full = blend.full_prefill(s, m["layers_np"], x0, keep_layer_outputs=True)
    return s, m, x0, res, full


def test_full_ratio_equals_full_prefill():
    """r = 100 % recompute is full attention (Sec. 4.1)."""
    shape = MINI.with_layers(3)
    s, m, x0, res, full = _sel(shape, [0, 9, 16, 30], 5, 1.0)
    assert len(res["sel"]) == 30
    for l in range(3):
        assert rel(res["layer_out"][l], full["layer_out"][l]) < 1e-11
    assert rel(res["k"], full["k"]) < 1e-11 and rel(res["v"], full["v"]) < 1e-11
    fh = llama.rmsnorm(full["x"][-5:], np.ones(64), s.rms_eps)
    assert rel(res["final_hidden"], fh) < 1e-11


def test_single_chunk_concatenation_is_exact():
    """With one chunk the cache is a prefix cache: every r gives the full-attention result."""
    shape = MINI.with_layers(3)
    for r in (0.0, 0.15, 0.6):
        s, m, x0, res, full = _sel(shape, [0, 24], 6, r)
        assert rel(res["final_hidden"], llama.rmsnorm(full["x"][-6:], np.ones(64), s.rms_eps)) < 1e-11
        if res["dev"] is not None:
            assert np.max(res["dev"]) < 1e-20


def test_zero_ratio_is_plain_concatenation():
    """r = 0 %: only query rows are recomputed; they read the re-aligned cache as is."""
    shape = MINI.with_layers(3)
    starts = [0, 10, 21]
    s, m, x0, res, full = _sel(shape, starts, 4, 0.0)
    assert len(res["sel"]) == 0 and list(res["rows"]) == [21, 22, 23, 24]
    # the cached context rows of layers >= 1 are exactly the re-aligned chunk caches
    cc = blend.chunk_caches(s, m["layers_np"], x0[:21], starts)
    assert rel(res["k"][1:, :21], blend.realign(s, cc["k"], starts)[1:]) < 1e-14
    assert rel(res["v"][1:, :21], cc["v"][1:]) == 0.0
    # and the answer differs from full attention (cross-chunk attention is missing)
    fh = llama.rmsnorm(full["x"][-4:], np.ones(64), s.rms_eps)
    assert rel(res["final_hidden"], fh) > 1e-5


def test_check_layer_zero_deviation_is_rounding_only():
    """At layer 0 fresh keys equal re-aligned cached keys, so the deviation is ~0."""
    shape = MINI.with_layers(2)
    s, m, x0, res, full = _sel(shape, [0, 8, 20, 29], 3, 0.3, check_layer=0)
    assert np.max(res["dev"]) < 1e-20
    s, m, x0, res1, full = _sel(shape, [0, 8, 20, 29], 3, 0.3, check_layer=1)
    assert np.max(res1["dev"][8:]) > 1e-4        # later chunks deviate at layer 1
    assert np.max(res1["dev"][:8]) < 1e-20       # the first chunk is a prefix: exact


def test_forced_selection_reproduces_hkvd_choice():
    shape = MINI.with_layers(2)
    starts = [0, 8, 20, 29]
    s, m, x0, res, _ = _sel(shape, starts, 3, 0.3)
    s, m, x0, res2, _ = _sel(shape, starts, 3, 0.3, forced=res["sel"][::-1])
    assert np.array_equal(res["sel"], res2["sel"])
    assert rel(res["final_hidden"], res2["final_hidden"]) == 0.0
    # the HKVD choice never picks first-chunk tokens (their deviation is zero)
    assert res["sel"].min() >= 8


def test_selected_rows_recompute_to_full_attention_at_check_layer():
    """At the check layer, a recomputed row's K/V equal full-attention K/V of that layer
    (its input is the full-attention layer-0 output)."""
    shape = MINI.with_layers(2)
    starts = [0, 8, 20, 29]
    s, m, x0, res, full = _sel(shape, starts, 3, 0.3)
    rows = res["rows"]
    assert rel(res["k"][1, rows], full["k"][1, rows]) < 1e-12
    assert rel(res["v"][1, rows], full["v"][1, rows]) < 1e-12


# ------------------------------------------------------------------------------------ planted mistakes

def _pins_fail(monkeypatch, target, attr, bad):
    monkeypatch.setattr(target, attr, bad)
    failed = []
    for t in (test_layer_matches_torch_library_block, test_attention_matches_sdpa_causal_gqa,
              test_rope_direction_closed_form, test_full_ratio_equals_full_prefill,
              test_prefix_invariance_and_realign, test_rope_matches_complex_multiplication,
              test_llama3_frequency_bands, test_yarn_bands_interpolate_and_keep,
              test_yarn_equals_llama3_rule_with_the_same_bounds, test_yarn_temperature_closed_form,
              test_layer_yarn_gqa7_bias_matches_torch, test_qkv_bias_closed_form):
        try:
            t()
        except (AssertionError, ValueError):   # a wrong result, or operands that no longer fit
            failed.append(t.__name__)
    monkeypatch.undo()
    return failed


def test_planted_mistakes(monkeypatch):
    good_rope = llama.apply_rope
    def rope_sign(x, c, s):   # rotation in the wrong direction
        return good_rope(x, c, -s)
    assert _pins_fail(monkeypatch, llama, "apply_rope", rope_sign)

    good_attn = llama.attention_rows
    def attn_gqa(s, q, k, v, hi, lo=None, block=256):   # query head j -> kv head j % Hkv
        Hq, Hkv = q.shape[1], k.shape[1]
        perm = [(j % Hkv) * (Hq // Hkv) + j // Hkv for j in range(Hq)]
        return good_attn(s, q[:, perm], k, v, hi, lo, block)[:, np.argsort(perm)]
    assert _pins_fail(monkeypatch, llama, "attention_rows", attn_gqa)

    def attn_nocausal(s, q, k, v, hi, lo=None, block=256):   # mask dropped
        return good_attn(s, q, k, v, np.full_like(np.asarray(hi), k.shape[0] - 1), lo, block)
    assert _pins_fail(monkeypatch, llama, "attention_rows", attn_nocausal)

    good_mlp = llama.attn_out_mlp
    def mlp_no_resid(s, lw, x, attn):   # residual of the attention half dropped
        return good_mlp(s, lw, x, attn) - llama.as64(x)
    assert _pins_fail(monkeypatch, llama, "attn_out_mlp", mlp_no_resid)

    def mlp_wo_t(s, lw, x, attn):      # W_o applied transposed (square when Hq*D == H)
        lw2 = dict(lw); lw2["w_o"] = llama.as64(lw["w_o"]).T.copy()
        return good_mlp(s, lw2, x, attn)
    assert _pins_fail(monkeypatch, llama, "attn_out_mlp", mlp_wo_t)

    good_freq = llama.rope_inv_freq
    def freq_bad(s):                   # exponent -i/D instead of -2i/D
        return good_freq(s) ** 0.5
    assert _pins_fail(monkeypatch, llama, "rope_inv_freq", freq_bad)

    good_yarn = llama.yarn_inv_freq
    def yarn_swapped(s):               # interpolation on the fast pairs instead of the slow ones
        w = good_yarn(s)
        plain = s.rope_theta ** (-2.0 * np.arange(s.head_dim // 2) / s.head_dim)
        return plain * plain / w
    assert _pins_fail(monkeypatch, llama, "yarn_inv_freq", yarn_swapped)

    good_scale = llama.logit_scale
    def temp_once(s):                  # temperature applied as sqrt(1/t) instead of 1/t
        m = 0.1 * math.log(s.rs_factor) + 1.0 if s.rope_scaling == llama.ROPE_YARN else 1.0
        return good_scale(s) / m
    assert _pins_fail(monkeypatch, llama, "logit_scale", temp_once)

    good_qkv = llama.qkv_rows
    def qkv_bias_after_rope(s, lw, x, pos):   # bias added after the rotation
        if lw.get("b_qkv") is None:
            return good_qkv(s, lw, x, pos)
        lw2 = dict(lw); b = llama.as64(lw2.pop("b_qkv"))
        q, k, v = good_qkv(s, lw2, x, pos)
        D, Hq, Hkv = s.head_dim, s.n_q_heads, s.n_kv_heads
        return (q + b[: Hq * D].reshape(1, Hq, D), k + b[Hq * D:(Hq + Hkv) * D].reshape(1, Hkv, D),
                v + b[(Hq + Hkv) * D:].reshape(1, Hkv, D))
    assert _pins_fail(monkeypatch, llama, "qkv_rows", qkv_bias_after_rope)


# ------------------------------------------------------------------------------------ bf16 storage mode

def test_bf16_round_is_round_to_nearest_even():
    """Against the bit-level definition: keep the top 16 bits of the fp32 pattern,
    rounding the dropped 16 bits to nearest with ties to an even kept part."""
    rng = np.random.default_rng(11)
    x = np.concatenate([rng.standard_normal(5000) * 10.0 ** rng.integers(-6, 6, 5000),
                        [1.0 + 2.0 ** -8, 1.0 + 3 * 2.0 ** -8, -1.0 - 2.0 ** -8, 0.0, 65504.0]]).astype(np.float32)
    b = x.view(np.uint32).astype(np.uint64)
    r = ((b + 0x7FFF + ((b >> 16) & 1)) >> 16) << 16
    want = r.astype(np.uint32).view(np.float32).astype(np.float64)
    assert np.array_equal(llama.bf16_round(x), want)
    assert llama.bf16_round([1.0 + 2.0 ** -8])[0] == 1.0            # tie -> even
    assert llama.bf16_round([1.0 + 3 * 2.0 ** -8])[0] == 1.0 + 2.0 ** -6


def test_bf16_storage_mode_rounds_only_stored_activations():
    """With act_bf16 the cache entries are bf16 values, the residual stream is not, and the
    result stays within bf16 rounding of the float64 one; without it nothing is rounded."""
    shape = MINI.with_layers(2)
    m = model(shape)
    starts = [0, 9, 20]
    toks = synth.make_tokens(shape, 25, 1)
    x0 = blend.embed_rows(m["embed"], toks.numpy())
    s16, s64 = Shape.of(shape, act_bf16=True), Shape.of(shape)
    r16 = blend.full_prefill(s16, m["layers_np"], x0)
    r64 = blend.full_prefill(s64, m["layers_np"], x0)
    assert np.array_equal(llama.bf16_round(r16["k"]), r16["k"]) and np.array_equal(llama.bf16_round(r16["v"]), r16["v"])
    assert not np.array_equal(llama.bf16_round(r16["x"]), r16["x"])
    assert not np.array_equal(llama.bf16_round(r64["k"]), r64["k"])
    g = rel(r16["x"], r64["x"])
    assert 1e-5 < g < 2e-2
    cc = blend.chunk_caches(s16, m["layers_np"], x0[:20], starts)
    re = blend.realign(s16, cc["k"], starts)
    assert np.array_equal(llama.bf16_round(re), re)


def test_accum32_is_a_float32_accumulation_of_the_same_model():
    """accum32 changes only the accumulation precision of the linear layers: it agrees with
    a float32 torch matmul and with the float64 result to float32 accuracy."""
    rng = np.random.default_rng(12)
    x = rng.standard_normal((9, 64))
    w = rng.standard_normal((33, 64)) * 0.02
    y32 = llama.linear(x, w, accum32=True)
    ref32 = (torch.as_tensor(x, dtype=torch.float32) @ torch.as_tensor(w, dtype=torch.float32).T).double().numpy()
    assert rel(y32, ref32) < 1e-6
    assert 0 < rel(y32, llama.linear(x, w)) < 1e-6
    shape = MINI.with_layers(2)
    m = model(shape)
    x0 = blend.embed_rows(m["embed"], synth.make_tokens(shape, 20, 1).numpy())
    a = blend.full_prefill(Shape.of(shape, act_bf16=True), m["layers_np"], x0)["x"]
    b = blend.full_prefill(Shape.of(shape, act_bf16=True, accum32=True), m["layers_np"], x0)["x"]
    assert 0 < rel(a, b) < 1e-2


def test_first_token_is_argmax_with_lowest_id_on_ties():
    W = np.array([[1.0, 0.0], [0.0, 1.0], [1.0, 0.0], [0.5, 0.5]])
    tok, logits = blend.first_token(np.array([[2.0, 1.0], [1.0, 1.0]]), W)
    assert list(tok) == [0, 0]                      # row 0: ids 0 and 2 tie at 2 -> 0; row 1: all tie at 1 -> 0
    assert np.allclose(logits, [[2, 1, 2, 1.5], [1, 1, 1, 1]])
    rng = np.random.default_rng(13)
    h, w = rng.standard_normal((3, 16)), rng.standard_normal((50, 16))
    tok, logits = blend.first_token(h, w)
    for r in range(3):
        best = max(range(50), key=lambda v: (sum(h[r, d] * w[v, d] for d in range(16)), -v))
        assert tok[r] == best


# ------------------------------------------------------------------ separators, EPIC, deviation histogram

def test_separator_layout_and_tokens():
    from paper_2609_09768_gb300 import synth
    starts, seps = synth.separator_layout(3, 5, 2)
    assert starts == [0, 5, 7, 12, 14, 19] and seps == [5, 12]
    wl = synth.WORKLOADS["tiny_sep"]
    t = wl.tokens()
    assert len(t) == wl.n_total and wl.n_ctx == 4 * 126 + 3 * 2
    for s in wl.sep_starts():
        assert [int(t[s]), int(t[s + 1])] == [wl.shape.vocab - 2, wl.shape.vocab - 1]


def test_window_select_epic_and_kvlink():
    # EPIC: 20 rows from every separator start; windows overlap and run past the context end
    assert list(blend.window_select([3, 10], 20, 25)) == list(range(3, 25))
    assert list(blend.window_select([5, 12], 2, 19)) == [5, 6, 12, 13]              # KVLink: the separators
    assert list(blend.window_select([], 20, 10)) == []
    assert list(blend.window_select([9], 20, 10)) == [9]
    assert list(blend.window_select([4, 0], 3, 10)) == [0, 1, 2, 4, 5, 6]          # order of starts is free
    # closed form for disjoint windows inside the context
    sel = blend.window_select([100 * c for c in range(1, 9)], 20, 1000)
    assert len(sel) == 8 * 20 and np.all(np.diff(sel) > 0)


def test_zero_separator_rows_stay_zero_after_realign():
    s = Shape(hidden=16, n_q_heads=2, n_kv_heads=1, head_dim=8, mlp_dim=24, rms_eps=1e-5, rope_theta=1e4)
    rng = np.random.default_rng(3)
    cc = {"k": rng.standard_normal((2, 12, 1, 8)), "v": rng.standard_normal((2, 12, 1, 8))}
    z = blend.zero_kv_rows(cc, [5, 6])
    assert np.all(z["k"][:, [5, 6]] == 0) and np.all(z["v"][:, [5, 6]] == 0)
    assert np.array_equal(z["k"][:, :5], cc["k"][:, :5]) and np.array_equal(z["v"][:, 7:], cc["v"][:, 7:])
    r = blend.realign(s, z["k"], [0, 5, 7, 12])
    assert np.all(r[:, [5, 6]] == 0)


def test_deviation_histogram_bins():
    edges = np.array([1e-3, 1e-2, 1e-1, 1.0])
    dev = np.array([0.0, 1e-3, 5e-3, 1e-2, 0.5, 1.0, 7.0, 9e-4])
    assert list(blend.deviation_histogram(dev, edges)) == [2, 2, 1, 1, 2]
    rng = np.random.default_rng(4)
    d = rng.exponential(size=500)
    e = np.sort(rng.exponential(size=7))
    h = blend.deviation_histogram(d, e)
    assert h.sum() == 500
    assert np.array_equal(h, np.bincount(np.searchsorted(e, d, side="right"), minlength=8))


def test_selective_prefill_with_separators_recompute_all_equals_full():
    """r = 1 over a context with zeroed separator rows is still the full causal prefill:
    every context row, separators included, is recomputed before it is read."""
    s = Shape(hidden=16, n_q_heads=2, n_kv_heads=1, head_dim=8, mlp_dim=24, rms_eps=1e-5, rope_theta=1e4)
    rng = np.random.default_rng(8)
    layers = [{"attn_norm": np.ones(16), "mlp_norm": np.ones(16),
               "w_qkv": rng.standard_normal((32, 16)) * 0.2, "w_o": rng.standard_normal((16, 16)) * 0.2,
               "w_gate": rng.standard_normal((24, 16)) * 0.2, "w_up": rng.standard_normal((24, 16)) * 0.2,
               "w_down": rng.standard_normal((16, 24)) * 0.2} for _ in range(3)]
    starts, seps = [0, 5, 7, 12, 14, 19], [5, 12]
    x0 = rng.standard_normal((23, 16))
    cc = blend.zero_kv_rows(blend.chunk_caches(s, layers, x0[:19], starts), [5, 6, 12, 13])
    full = blend.full_prefill(s, layers, x0)
    sp = blend.selective_prefill(s, layers, x0, starts, 4, 1.0, cc["k"], cc["v"])
    assert np.array_equal(sp["layer_out"][-1][-4:], full["x"][-4:])
    # EPIC's rows are a valid forced selection; the separator rows it leaves out keep zero K/V
    epic = blend.window_select(seps, 3, 19)
    sp = blend.selective_prefill(s, layers, x0, starts, 4, 0.0, cc["k"], cc["v"], forced_sel=epic)
    assert list(sp["sel"]) == [5, 6, 7, 12, 13, 14]
    assert np.all(sp["k"][1:, [5, 6, 12, 13]] != 0)           # recomputed in the selective layers
    kv = blend.selective_prefill(s, layers, x0, starts, 4, 0.0, cc["k"], cc["v"], forced_sel=[7])
    assert np.all(kv["k"][1:, [5, 6, 12, 13]] == 0) and np.all(kv["v"][1:, [5, 6, 12, 13]] == 0)


def test_decode_steps_equal_a_longer_full_prefill():
    """Two greedy decode steps after a full prefill of n tokens give the final hidden
    states of a full prefill of n + 2 tokens at its last two rows (the appended K/V rows,
    positions and causal range must all be right)."""
    s = Shape(hidden=16, n_q_heads=4, n_kv_heads=2, head_dim=8, mlp_dim=24, rms_eps=1e-5, rope_theta=1e4)
    rng = np.random.default_rng(21)
    layers = [{"attn_norm": np.ones(16), "mlp_norm": np.ones(16),
               "w_qkv": rng.standard_normal((64, 16)) * 0.3, "w_o": rng.standard_normal((16, 32)) * 0.3,
               "w_gate": rng.standard_normal((24, 16)) * 0.3, "w_up": rng.standard_normal((24, 16)) * 0.3,
               "w_down": rng.standard_normal((16, 24)) * 0.3} for _ in range(2)]
    embed = rng.standard_normal((40, 16))
    lm = rng.standard_normal((40, 16)) * 0.3
    fn = np.ones(16)
    toks = rng.integers(0, 40, 9)
    n = 7
    pre = blend.full_prefill(s, layers, blend.embed_rows(embed, toks[:n]))
    kc = np.zeros((2, 9, 2, 8)); vc = np.zeros_like(kc)
    kc[:, :n] = pre["k"]; vc[:, :n] = pre["v"]
    t1, h1, _ = blend.decode_step(s, layers, embed, fn, lm, kc, vc, int(toks[n]), n)
    t2, h2, l2 = blend.decode_step(s, layers, embed, fn, lm, kc, vc, int(toks[n + 1]), n + 1)
    full = blend.full_prefill(s, layers, blend.embed_rows(embed, toks))
    fh = llama.rmsnorm(full["x"], fn, s.rms_eps)
    assert np.allclose(h1, fh[n], rtol=1e-10, atol=1e-12) and np.allclose(h2, fh[n + 1], rtol=1e-10, atol=1e-12)
    assert np.allclose(kc, full["k"], rtol=1e-10, atol=1e-12)
    assert t2 == int(np.argmax(fh[n + 1] @ lm.T)) and t1 == int(np.argmax(fh[n] @ lm.T))
