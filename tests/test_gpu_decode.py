"""Greedy decode after the prefill, through the C ABI, against the float64 oracle:
the split-KV decode attention alone (ragged positions and the 124k headline length),
and whole decode steps on the tiny and Llama-3.1-8B-shaped 2-layer models, teacher-forced
on the tokens the GPU produced (the oracle continues from the GPU's prefill cache)."""
import dataclasses

import numpy as np
import pytest
import torch

from oracle import blend, llama
from oracle.llama import Shape
from paper_2609_09768_gb300 import synth, workload
from tests.gpu_util import MEAN_ABS, assert_close_abs, assert_close_bf16, assert_close_rel, errs, np64

pytestmark = pytest.mark.gpu

TINY = synth.TINY
L8B = synth.LLAMA8B.with_layers(2)


@pytest.fixture(scope="module")
def kvb():
    from paper_2609_09768_gb300 import kvblend
    kvblend.lib()
    return kvblend


def dev(t):
    return t.to("cuda")


# ------------------------------------------------------------------------------ decode attention

@pytest.mark.parametrize("shape,n_rows,positions", [
    (L8B, 3000, [0, 1, 255, 256, 257, 2999]),      # split edges, a single key, the last row
    (TINY, 600, [0, 300, 599]),
    (L8B, 124160, [124031]),                        # the headline length (124,032 rows)
    (synth.YARN_GQA7, 3000, [0, 1, 1023, 1024, 2999]),   # 7 q heads per kv head, YaRN temperature
    (synth.YARN_GQA7_TINY, 600, [0, 300, 599]),
    (dataclasses.replace(L8B, n_q_heads=24), 1500, [15, 16, 17, 511, 512, 1499]),   # 3 per kv head
    (dataclasses.replace(L8B, n_q_heads=32, n_kv_heads=4), 700, [127, 128, 699]),   # 8 per kv head
    (dataclasses.replace(TINY, n_q_heads=2, n_kv_heads=2), 300, [0, 33, 299]),      # 1 per kv head
])
def test_decode_attention_matches_oracle(kvb, shape, n_rows, positions):
    cfg = kvb.config(shape)
    q = synth.randn_bf16((shape.n_q_heads, shape.head_dim), 31)
    k = synth.randn_bf16((n_rows, shape.n_kv_heads, shape.head_dim), 32)
    v = synth.randn_bf16((n_rows, shape.n_kv_heads, shape.head_dim), 33).to(torch.float16)
    dq, dk, dv = dev(q), dev(k), dev(v)
    ws = kvb.decode_workspace(cfg, n_rows)
    vs = float(np.sqrt(np.mean(np64(v) ** 2)))
    s = Shape.of(shape)
    for p in positions:
        pos = torch.tensor([p], dtype=torch.int32, device="cuda")
        out = kvb.decode_attention(cfg, dq, dk, dv, pos, n_rows, ws=ws)
        torch.cuda.synchronize()
        assert kvb.device_status(ws) == 0
        ref = llama.attention_rows(s, np64(q)[None], np64(k), np64(v), [p])
        e = assert_close_rel(out.cpu().reshape(1, -1), ref.reshape(1, -1), f"decode attention pos {p}", scale=vs)
        print("decode attn", shape.head_dim, n_rows, p, e)


def test_decode_attention_ignores_rows_past_the_position(kvb):
    """Cache rows after `pos` hold NaN (a cache the caller never wrote there): the output is
    that of the rows up to pos alone."""
    shape = L8B
    cfg = kvb.config(shape)
    n_rows = 700
    q = synth.randn_bf16((shape.n_q_heads, shape.head_dim), 51)
    k = synth.randn_bf16((n_rows, shape.n_kv_heads, shape.head_dim), 52)
    v = synth.randn_bf16((n_rows, shape.n_kv_heads, shape.head_dim), 53).to(torch.float16)
    ws = kvb.decode_workspace(cfg, n_rows)
    s = Shape.of(shape)
    for p in (0, 9, 130, 511, 600):
        kn, vn = k.clone(), v.clone()
        kn[p + 1:] = float("nan")
        vn[p + 1:] = float("nan")
        out = kvb.decode_attention(cfg, dev(q), dev(kn), dev(vn), torch.tensor([p], dtype=torch.int32, device="cuda"),
                                   n_rows, ws=ws)
        torch.cuda.synchronize()
        assert kvb.device_status(ws) == 0
        assert torch.isfinite(out.float()).all(), p
        ref = llama.attention_rows(s, np64(q)[None], np64(k), np64(v), [p])
        assert_close_rel(out.cpu().reshape(1, -1), ref.reshape(1, -1), f"decode attention pos {p} (NaN after)",
                         scale=float(np.sqrt(np.mean(np64(v) ** 2))))


def test_decode_attention_rejects_position_out_of_range(kvb):
    """pos >= max_pos: the kernels record KVB_ERR_INVALID_ARG and write nothing."""
    shape = L8B
    cfg = kvb.config(shape)
    n_rows = 512
    q = dev(synth.randn_bf16((shape.n_q_heads, shape.head_dim), 41))
    k = dev(synth.randn_bf16((n_rows, shape.n_kv_heads, shape.head_dim), 42))
    v = dev(synth.randn_bf16((n_rows, shape.n_kv_heads, shape.head_dim), 43).to(torch.float16))
    ws = kvb.decode_workspace(cfg, n_rows)
    out = torch.full((shape.n_q_heads, shape.head_dim), 7.0, dtype=torch.bfloat16, device="cuda")
    for p in (n_rows, -1):
        kvb.decode_attention(cfg, q, k, v, torch.tensor([p], dtype=torch.int32, device="cuda"), n_rows, out=out, ws=ws)
        assert kvb.device_status(ws) == kvb.KVB_ERR_INVALID_ARG
        assert torch.all(out == 7.0)


# ------------------------------------------------------------------------------- decode steps

class DecodeCase:
    """GPU prefill of a workload (HKVD selection on the device), then T decode steps on the
    GPU; the oracle repeats each step from the GPU's cache and token (teacher forcing)."""

    T = 3

    def __init__(self, kvb, wl: synth.Workload):
        self.wl, self.shape = wl, wl.shape
        shape = wl.shape
        N, n_ctx, nq = wl.n_total, wl.n_ctx, wl.n_query
        self.N = N
        cap = N + self.T + 1
        w = synth.make_model(shape, 0)
        lm = synth.make_lm_head(shape, 0)
        toks = wl.tokens()
        cfg = kvb.config(shape)
        self.cfg = cfg
        model = kvb.Model({"layers": [{k: v.cuda() for k, v in l.items()} for l in w["layers"]],
                           "embed": w["embed"].cuda(), "final_norm": w["final_norm"].cuda()})
        rope = kvb.RopeTable(cfg, cap)
        ws = kvb.workspace(cfg, N)
        starts = wl.chunk_starts()
        dtoks = toks.cuda()
        kch, vch = workload.chunk_caches(cfg, model, rope, dtoks[:n_ctx], starts, ws=ws, zero_rows=wl.sep_rows())
        L = shape.n_layers
        ck = torch.zeros(L, cap, shape.n_kv_heads, shape.head_dim, dtype=torch.bfloat16, device="cuda")
        cv = torch.zeros(L, cap, shape.n_kv_heads, shape.head_dim, dtype=torch.float16, device="cuda")
        fh, _, _ = kvb.selective_prefill(cfg, model, rope, kch, vch, ck, cv, dtoks,
                                         torch.tensor(starts, dtype=torch.int32, device="cuda"), n_ctx, nq, wl.r, 1,
                                         ws=ws)
        dlm = lm.cuda()
        tokens = torch.zeros(cap + 1, dtype=torch.int32, device="cuda")
        tokens[:N] = dtoks
        first, _ = kvb.lm_head_argmax(cfg, dlm, fh[nq - 1:].contiguous())                  # the first token
        tokens[N:N + 1] = first
        torch.cuda.synchronize()
        assert kvb.device_status(ws) == 0
        self.cache0_k, self.cache0_v = ck[:, :N].cpu(), cv[:, :N].cpu()
        pos = torch.tensor([N], dtype=torch.int32, device="cuda")
        dws = kvb.decode_workspace(cfg, cap)
        self.hidden = []
        for t in range(self.T):
            h = torch.empty(shape.hidden, dtype=torch.float32, device="cuda")
            kvb.decode_step(cfg, model, rope, ck, cv, dlm, tokens, pos, cap, hidden=h, ws=dws)
            self.hidden.append(h)
        torch.cuda.synchronize()
        assert kvb.device_status(dws) == 0
        assert int(pos.item()) == N + self.T
        self.tokens = tokens.cpu().numpy()
        self.hidden = [h.cpu() for h in self.hidden]
        self.ck, self.cv = ck.cpu(), cv.cpu()
        self.w, self.lm = w, lm


_CASES = {}


@pytest.fixture(scope="module", params=["tiny", "l8b_1layer", "yarn_tiny", "yarn_2l"])
def case(request, kvb):
    if request.param not in _CASES:
        _CASES[request.param] = DecodeCase(kvb, synth.WORKLOADS[request.param])
    return _CASES[request.param]


def test_decode_steps_match_oracle(kvb, case):
    shape, N, T = case.shape, case.N, case.T
    layers = [{k: llama.as64(v) for k, v in l.items()} for l in case.w["layers"]]
    s = Shape.of(shape, act_bf16=True)
    s32 = Shape.of(shape, act_bf16=True, accum32=True)
    embed, fn = case.w["embed"], case.w["final_norm"]
    lm64 = llama.as64(case.lm)
    abs_lm = np.abs(case.lm.float().numpy())
    L = shape.n_layers
    cap = N + T + 1
    kc = np.zeros((L, cap, shape.n_kv_heads, shape.head_dim))
    vc = np.zeros_like(kc)
    kc[:, :N] = np64(case.cache0_k)
    vc[:, :N] = np64(case.cache0_v)
    kc32, vc32 = kc.copy(), vc.copy()
    for t in range(T):
        p = N + t
        tok_in = int(case.tokens[p])
        tok_o, h_o, logits_o = blend.decode_step(s, layers, embed, fn, lm64, kc, vc, tok_in, p)
        _, h_32, _ = blend.decode_step(s32, layers, embed, fn, lm64, kc32, vc32, tok_in, p)
        floor = errs(h_32, h_o)["mean_abs"]
        h_g = np64(case.hidden[t])
        e = assert_close_abs(h_g, h_o, f"decode step {t} final hidden", mean_abs=max(MEAN_ABS, 1.5 * floor))
        # the row this step appended to every layer's cache
        for l in range(L):
            assert_close_bf16(case.ck[l, p], kc[l, p], f"decode step {t} layer {l} K row")
            assert_close_bf16(case.cv[l, p], vc[l, p], f"decode step {t} layer {l} V row")
        # the GPU's token: its exact logit reaches the maximum within the logit error that
        # the hidden-state difference and fp32 accumulation allow; equal where the gap is wider
        tok_g = int(case.tokens[p + 1])
        dh = np.abs(h_g - h_o)
        bound = (abs_lm @ dh.astype(np.float32)).astype(np.float64) * 1.001
        bound += shape.hidden * 2.0 ** -24 * 1.001 * (abs_lm @ np.abs(h_g).astype(np.float32))
        assert logits_o[tok_g] + bound[tok_g] >= logits_o[tok_o] - bound[tok_o], (t, tok_g, tok_o)
        srt = np.sort(logits_o)
        if srt[-1] - srt[-2] > 2 * bound.max():
            assert tok_g == tok_o
        # the oracle continues from the GPU's own row (teacher forcing keeps the two in step)
        kc[:, p], vc[:, p] = np64(case.ck[:, p]), np64(case.cv[:, p])
        kc32[:, p], vc32[:, p] = kc[:, p], vc[:, p]
        print("decode", shape.hidden, t, tok_g, tok_o, e, "floor", floor)


def test_decode_leaves_the_prompt_cache_untouched(kvb, case):
    N = case.N
    assert torch.equal(case.ck[:, :N], case.cache0_k) and torch.equal(case.cv[:, :N], case.cache0_v)
    assert np.all((case.tokens[N:N + case.T + 1] >= 0) & (case.tokens[N:N + case.T + 1] < case.shape.vocab))
