"""Per-step parity of the CUDA path (through the C ABI) against the float64 oracle,
on seeded synthetic inputs of both model shapes, with ragged sizes and edge cases."""
import numpy as np
import pytest
import torch

from oracle import blend, llama
from oracle.llama import Shape
from paper_2609_09768_gb300 import synth
from tests.attn_cases import assert_attn_close, peaked_queries, tagged_case
from tests.gpu_util import assert_close_abs, assert_close_bf16, check_selection, errs, np64

pytestmark = pytest.mark.gpu

TINY = synth.TINY
L8B = synth.LLAMA8B.with_layers(2)
YT = synth.YARN_GQA7_TINY            # YaRN, 7 q heads per kv head, q/k/v bias
Y2 = synth.YARN_GQA7


@pytest.fixture(scope="module")
def kvb():
    from paper_2609_09768_gb300 import kvblend
    kvblend.lib()
    return kvblend


def dev(t):
    return t.to("cuda")


# ------------------------------------------------------------------------------------------ realign

@pytest.mark.parametrize("shape,starts", [
    (TINY, [0, 128, 256, 384, 512]),
    (L8B, synth.chunk_starts_equal(8, 480)),
    (TINY, [0, 1, 70, 200, 203, 333]),            # ragged chunk lengths, a 1-token chunk
])
def test_realign_matches_oracle(kvb, shape, starts):
    cfg = kvb.config(shape)
    n_ctx, L, Hkv, D = starts[-1], shape.n_layers, shape.n_kv_heads, shape.head_dim
    k_src = synth.randn_bf16((L, n_ctx, Hkv, D), 101)
    v_src = synth.randn_bf16((L, n_ctx, Hkv, D), 102)            # chunk caches hold bf16 V
    rope = kvb.RopeTable(cfg, n_ctx)
    cs = dev(torch.tensor(starts, dtype=torch.int32))
    rows = n_ctx + 13
    k_dst = torch.zeros(L, rows, Hkv, D, dtype=torch.bfloat16, device="cuda")
    v_dst = torch.zeros(L, rows, Hkv, D, dtype=torch.float16, device="cuda")
    ws = torch.zeros(256, dtype=torch.uint8, device="cuda")
    kvb.rope_realign(cfg, rope, dev(k_src), dev(v_src), k_dst, v_dst, 0, L, cs, n_ctx, ws=ws)
    torch.cuda.synchronize()
    assert kvb.device_status(ws) == kvb.KVB_OK
    ref = blend.realign(Shape.of(shape, act_bf16=True), np64(k_src), starts)
    e = assert_close_bf16(k_dst[:, :n_ctx].cpu(), ref, "realigned K")
    # bf16 -> fp16 container: the same value (torch rounds to nearest-even like the kernel)
    assert torch.equal(v_dst[:, :n_ctx].cpu(), v_src.to(torch.float16)), "V must be converted exactly"
    # and come back unchanged wherever fp16 holds them exactly (zero and |v| >= 2^-14; smaller
    # magnitudes are fp16 subnormals, rounded to 2^-24)
    normal = (v_src == 0) | (v_src.float().abs() >= 2.0 ** -14)
    back = v_dst[:, :n_ctx].cpu().to(torch.bfloat16)
    assert torch.equal(back[normal], v_src[normal]), "V values must survive the round trip"
    assert (back[~normal].float() - v_src[~normal].float()).abs().max() <= 2.0 ** -25
    assert torch.count_nonzero(k_dst[:, n_ctx:]) == 0, "rows past n_ctx must be untouched"
    # in place gives the same bits as out of place
    k_in = dev(k_src).clone()
    kvb.rope_realign(cfg, rope, k_in, None, k_in, None, 0, L, cs, n_ctx)
    torch.cuda.synchronize()
    assert torch.equal(k_in, k_dst[:, :n_ctx])
    print("realign", shape.head_dim, e)


# ------------------------------------------------------------------------------------------ HKVD

@pytest.mark.parametrize("n,kv_dim,k", [
    (512, 128, 76), (3840, 1024, 576), (1000, 64, 333), (17, 128, 0), (17, 128, 17), (1, 128, 1),
    (123904, 1024, 18585), (5000, 1024, 1), (131072, 128, 20000), (131073, 128, 20000), (200000, 128, 30000),
])
def test_hkvd_select_matches_oracle(kvb, n, kv_dim, k):
    kf = synth.randn_bf16((n, kv_dim), 201)
    kc = synth.randn_bf16((n, kv_dim), 202)
    # a band of rows with zero deviation (a prefix chunk) and duplicated rows (exact ties)
    z = min(n // 4, 300)
    kc[:z] = kf[:z]
    if n > 40:
        kf[20:30] = kf[10]
        kc[20:30] = kc[10]
    sel, dv = kvb.hkvd_select(dev(kf), dev(kc), k)
    torch.cuda.synchronize()
    dref = blend.hkvd_deviation(np64(kf), np64(kc))
    e = errs(dv.cpu(), dref)
    assert e["max_abs"] <= 1e-5 * max(1.0, float(dref.max())), e
    s = sel.cpu().numpy()
    assert np.all(np.diff(s) > 0), "indices must be ascending and distinct"
    nd = check_selection(s, dref, k)
    print("hkvd", n, k, "dev err", e["max_abs"], "differing (near-tie) indices", nd)


@pytest.mark.parametrize("n", [123904, 131072, 200000])
def test_hkvd_all_equal_deviations_take_the_lowest_indices(kvb, n):
    """Every deviation equal: the top k are exactly indices 0..k-1, also where the k-th
    falls on the boundary between the key ranges of two CTAs of the select's cluster
    (16,384 keys each) and on the last key."""
    kv_dim = 8
    kf = torch.zeros(n, kv_dim, dtype=torch.bfloat16)
    kc = kf.clone()
    kc[:, 3] = 0.5
    for k in (1, 16383, 16384, 16385, 65536, n - 1, n):
        sel, _ = kvb.hkvd_select(dev(kf), dev(kc), k)
        assert torch.equal(sel.cpu(), torch.arange(k, dtype=torch.int32)), k


def test_hkvd_exact_ties_take_lowest_index(kvb):
    n, kv_dim = 4096, 256
    kf = synth.randn_bf16((n, kv_dim), 203)
    kc = kf.clone()
    kc[:, 0] = kc[:, 0] + 1.0      # same-magnitude offsets on many rows -> many equal deviations
    kc[::3, 1] = kc[::3, 1] + 2.0
    for k in (1, 100, 1365, 1366, 2000, n):
        sel, dv = kvb.hkvd_select(dev(kf), dev(kc), k)
        d32 = dv.cpu().numpy()
        want = blend.topk_select(d32.astype(np.float64), k)   # oracle rule on the GPU's own fp32 values
        assert np.array_equal(sel.cpu().numpy(), want), k


# ------------------------------------------------------------------------------------------ QKV GEMM

@pytest.mark.parametrize("shape,m,n_src", [(TINY, 108, 544), (L8B, 640, 3904), (L8B, 1, 7), (TINY, 129, 300),
                                           (L8B, 300, 300), (YT, 108, 544), (Y2, 640, 3904), (Y2, 1, 7)])
def test_gather_rmsnorm_qkv_matches_oracle(kvb, shape, m, n_src):
    cfg = kvb.config(shape)
    lw = synth.make_layer_weights(shape, 1, seed=5)
    lwd = {k: dev(v) for k, v in lw.items()}
    s = Shape.of(shape, act_bf16=True)
    g = torch.Generator().manual_seed(7)
    x = torch.randn(n_src, shape.hidden, generator=g) * 2.0
    row_idx = torch.sort(torch.randperm(n_src, generator=g)[:m]).values.to(torch.int32)
    max_pos = n_src + 50
    rope_pos = torch.randint(0, max_pos, (m,), generator=g, dtype=torch.int32)
    n_cache = n_src + 5
    kv_dst = torch.randperm(n_cache, generator=g)[:m].to(torch.int32)
    rope = kvb.RopeTable(cfg, max_pos)
    q = torch.zeros(m, shape.q_dim, dtype=torch.bfloat16, device="cuda")
    kc = torch.zeros(n_cache, shape.kv_dim, dtype=torch.bfloat16, device="cuda")
    vc = torch.zeros(n_cache, shape.kv_dim, dtype=torch.float16, device="cuda")
    ws = kvb.workspace(cfg, m)
    kvb.gather_rmsnorm_qkv(cfg, kvb.layer_struct(lwd), rope, dev(x), dev(row_idx), dev(rope_pos), m, q, kc, vc,
                           dev(kv_dst), ws)
    torch.cuda.synchronize()
    assert kvb.device_status(ws) == 0
    qr, kr, vr = llama.qkv_rows(s, lw, np64(x)[row_idx.numpy()], rope_pos.numpy())
    eq = assert_close_bf16(q.cpu(), qr.reshape(m, -1), "q")
    ek = assert_close_bf16(kc.cpu()[kv_dst.long()], kr.reshape(m, -1), "k")
    ev = assert_close_bf16(vc.cpu()[kv_dst.long()], vr.reshape(m, -1), "v")
    untouched = torch.ones(n_cache, dtype=torch.bool)
    untouched[kv_dst.long()] = False
    assert torch.count_nonzero(kc.cpu()[untouched]) == 0
    print("qkv", shape.hidden, m, eq, ek, ev)


# ------------------------------------------------------------------------------------------ attention

def _attn_case(kvb, shape, n_kv, q_rows, kv_lo=None, seed=11, tagged=False):
    """Runs the attention kernel on one case and the oracle on all its rows.  Default inputs:
    queries scaled for logits of standard deviation 5 (a peaked softmax) against N(0,1) keys;
    tagged=True: the tagged-key construction of tests/attn_cases.py, where each (row, head)
    reads essentially one chosen key, so a key range that is off by one key or one tile
    changes the output completely."""
    cfg = kvb.config(shape)
    m = len(q_rows)
    if tagged:
        q, k, v, _ = tagged_case(n_kv, q_rows, kv_lo, shape.n_q_heads, shape.n_kv_heads, shape.head_dim, seed)
        v = v.to(torch.float16)
    else:
        q = peaked_queries(m, shape.n_q_heads, shape.head_dim, seed)
        k = synth.randn_bf16((n_kv, shape.n_kv_heads, shape.head_dim), seed + 1)
        v = synth.randn_bf16((n_kv, shape.n_kv_heads, shape.head_dim), seed + 2).to(torch.float16)
    qi = torch.tensor(q_rows, dtype=torch.int32)
    lo = None if kv_lo is None else torch.tensor(kv_lo, dtype=torch.int32)
    out = torch.zeros(m, shape.q_dim, dtype=torch.bfloat16, device="cuda")
    ws = torch.zeros(256, dtype=torch.uint8, device="cuda")
    kvb.sparse_query_attn(cfg, dev(q), dev(qi), None if lo is None else dev(lo), dev(k), dev(v), out, ws)
    torch.cuda.synchronize()
    assert kvb.device_status(ws) == 0
    ref = llama.attention_rows(Shape.of(shape), np64(q), np64(k), np64(v), q_rows, kv_lo)
    return out.cpu(), ref.reshape(m, -1)


@pytest.mark.parametrize("tagged", [False, True])
@pytest.mark.parametrize("shape,n_kv", [(TINY, 544), (L8B, 3904), (TINY, 1), (L8B, 130), (L8B, 129), (YT, 544),
                                        (Y2, 3904), (Y2, 19), (YT, 1)])
def test_attention_dense_causal(kvb, shape, n_kv, tagged):
    out, ref = _attn_case(kvb, shape, n_kv, list(range(n_kv)), tagged=tagged)
    e = assert_attn_close(out, ref, "dense causal attention")
    print("attn dense", shape.head_dim, n_kv, tagged, e)


@pytest.mark.parametrize("tagged", [False, True])
@pytest.mark.parametrize("shape,n_kv,m", [(TINY, 544, 108), (L8B, 3904, 640), (L8B, 3904, 33), (L8B, 5000, 1),
                                          (TINY, 200, 3), (Y2, 3904, 640), (YT, 544, 37)])
def test_attention_sparse_rows(kvb, shape, n_kv, m, tagged):
    g = np.random.default_rng(m)
    rows = np.sort(g.choice(n_kv, size=m, replace=False))
    rows[-1] = n_kv - 1
    out, ref = _attn_case(kvb, shape, n_kv, rows.tolist(), tagged=tagged)
    e = assert_attn_close(out, ref, "sparse-query attention")
    print("attn sparse", shape.head_dim, n_kv, m, tagged, e)


@pytest.mark.parametrize("tagged", [False, True])
@pytest.mark.parametrize("shape,starts", [(TINY, [0, 128, 256, 384, 512]), (L8B, [0, 480, 960, 1440]),
                                          (TINY, [0, 5, 140, 141, 300]), (Y2, [0, 480, 960, 1440]),
                                          (YT, [0, 5, 140, 141, 300]), (L8B, [0, 143, 144, 289, 577, 1000])])
def test_attention_block_diagonal(kvb, shape, starts, tagged):
    n = starts[-1]
    lo = np.concatenate([[starts[c]] * (starts[c + 1] - starts[c]) for c in range(len(starts) - 1)])
    out, ref = _attn_case(kvb, shape, n, list(range(n)), lo.tolist(), tagged=tagged)
    e = assert_attn_close(out, ref, "block-diagonal attention")
    print("attn blockdiag", shape.head_dim, tagged, e)


# ------------------------------------------------------------------------------------------ MLP half

@pytest.mark.parametrize("shape,m", [(TINY, 108), (L8B, 640), (L8B, 1), (TINY, 300), (Y2, 640), (YT, 108)])
def test_mlp_rows_matches_oracle(kvb, shape, m):
    cfg = kvb.config(shape)
    lw = synth.make_layer_weights(shape, 0, seed=9)
    lwd = {k: dev(v) for k, v in lw.items()}
    attn = synth.randn_bf16((m, shape.q_dim), 301)
    g = torch.Generator().manual_seed(3)
    x = torch.randn(m, shape.hidden, generator=g) * 1.5
    xd = dev(x).contiguous()
    ws = kvb.workspace(cfg, m)
    kvb.mlp_rows(cfg, kvb.layer_struct(lwd), dev(attn), xd, ws)
    torch.cuda.synchronize()
    assert kvb.device_status(ws) == 0
    ref = llama.attn_out_mlp(Shape.of(shape, act_bf16=True), lw, np64(x), np64(attn))
    e = assert_close_abs(xd.cpu(), ref, "x after O-proj + MLP")
    print("mlp", shape.hidden, m, e)


# ------------------------------------------------------------------------------------------ scatter

@pytest.mark.parametrize("m,kv_dim,n_dst", [(576, 1024, 3904), (1, 128, 5), (108, 128, 544), (0, 128, 4)])
def test_kv_scatter_bit_exact(kvb, m, kv_dim, n_dst):
    g = torch.Generator().manual_seed(m)
    kr = synth.randn_bf16((m, kv_dim), 401)
    vr = synth.randn_bf16((m, kv_dim), 402).to(torch.float16)
    idx = torch.randperm(n_dst, generator=g)[:m].to(torch.int32)
    kd = torch.zeros(n_dst, kv_dim, dtype=torch.bfloat16, device="cuda")
    vd = torch.zeros(n_dst, kv_dim, dtype=torch.float16, device="cuda")
    kvb.kv_scatter(dev(kr), dev(vr), dev(idx), kd, vd)
    torch.cuda.synchronize()
    want_k = torch.zeros(n_dst, kv_dim, dtype=torch.bfloat16)
    want_v = torch.zeros(n_dst, kv_dim, dtype=torch.float16)
    want_k[idx.long()] = kr
    want_v[idx.long()] = vr
    assert torch.equal(kd.cpu(), want_k) and torch.equal(vd.cpu(), want_v)


def test_kv_scatter_skips_rows_outside_the_destination(kvb):
    """A destination index outside [0, n_dst_rows) is skipped, not written.  The
    destination is a view of the first rows of a larger buffer, so the row just past
    it is memory of this test and must stay untouched."""
    n_dst, kv_dim = 6, 128
    kr = synth.randn_bf16((3, kv_dim), 411)
    vr = synth.randn_bf16((3, kv_dim), 412).to(torch.float16)
    idx = torch.tensor([1, n_dst, 4], dtype=torch.int32)
    kpad = torch.zeros(n_dst + 1, kv_dim, dtype=torch.bfloat16, device="cuda")
    vpad = torch.zeros(n_dst + 1, kv_dim, dtype=torch.float16, device="cuda")
    kvb.kv_scatter(dev(kr), dev(vr), dev(idx), kpad[:n_dst], vpad[:n_dst])
    torch.cuda.synchronize()
    want_k = torch.zeros(n_dst + 1, kv_dim, dtype=torch.bfloat16)
    want_v = torch.zeros(n_dst + 1, kv_dim, dtype=torch.float16)
    want_k[[1, 4]] = kr[[0, 2]]
    want_v[[1, 4]] = vr[[0, 2]]
    assert torch.equal(kpad.cpu(), want_k) and torch.equal(vpad.cpu(), want_v)


@pytest.mark.parametrize("noalloc", [False, True])
def test_qkv_indices_outside_their_range_are_reported(kvb, noalloc):
    """Destinations outside [0, n_kv_rows) write no k/v row and positions outside the RoPE
    tables rotate by position 0; both set KVB_ERR_INVALID_ARG in the status word, and every
    other row comes out exactly as in a run with valid indices.  The k/v destination is a
    view that starts one row into a larger buffer, and the tables hold one row more than
    the struct declares, so the rows the bad indices name (-1, n_kv_rows, max_pos) are all
    memory of this test; they must stay untouched."""
    shape = L8B
    cfg = kvb.config(shape)
    lws = kvb.layer_struct({k: dev(v) for k, v in synth.make_layer_weights(shape, 1, seed=6).items()})
    m, n_rows, max_pos = 8, 40, 30
    g = torch.Generator().manual_seed(17)
    x = dev(torch.randn(m, shape.hidden, generator=g))
    good_dst = torch.tensor([3, 7, 11, 15, 19, 23, 27, 31], dtype=torch.int32)
    good_pos = torch.tensor([0, 1, 5, 9, 13, 17, 21, 29], dtype=torch.int32)
    bad_dst = good_dst.clone()
    bad_dst[2], bad_dst[5] = -1, n_rows                 # rows 2 and 5 must write nothing
    bad_pos = good_pos.clone()
    bad_pos[4] = max_pos                                # row 4 is rotated by position 0
    ref_pos = good_pos.clone()
    ref_pos[4] = 0
    rope = kvb.RopeTable(cfg, max_pos + 1)
    rope.struct.max_pos = max_pos

    def run(dst, pos):
        q = torch.zeros(m, shape.q_dim, dtype=torch.bfloat16, device="cuda")
        kbig = torch.zeros(n_rows + 2, shape.kv_dim, dtype=torch.bfloat16, device="cuda")
        vbig = torch.zeros(n_rows + 2, shape.kv_dim, dtype=torch.float16, device="cuda")
        kview, vview = kbig[1:n_rows + 1], vbig[1:n_rows + 1]
        if noalloc:
            st = torch.zeros(4, dtype=torch.int32, device="cuda")
            kvb.gather_rmsnorm_qkv_noalloc(cfg, lws, rope, x, None, dev(pos), m, q, kview, vview, dev(dst), st,
                                           n_kv_rows=n_rows)
            torch.cuda.synchronize()
            code = int(st[0])
        else:
            ws = kvb.workspace(cfg, m)
            kvb.gather_rmsnorm_qkv(cfg, lws, rope, x, None, dev(pos), m, q, kview, vview, dev(dst), ws,
                                   n_kv_rows=n_rows)
            code = kvb.device_status(ws)
        return code, q.cpu(), kbig.cpu(), vbig.cpu()

    code, q, kb, vb = run(bad_dst, bad_pos)
    assert code == kvb.KVB_ERR_INVALID_ARG
    code_ref, q_ref, kb_ref, vb_ref = run(good_dst, ref_pos)
    assert code_ref == kvb.KVB_OK
    assert torch.equal(q, q_ref), "q rows, including the one rotated by position 0"
    assert torch.count_nonzero(kb[0]) == 0 and torch.count_nonzero(kb[n_rows + 1]) == 0
    assert torch.count_nonzero(vb[0]) == 0 and torch.count_nonzero(vb[n_rows + 1]) == 0
    for r in range(m):
        row = int(good_dst[r]) + 1
        if r in (2, 5):
            assert torch.count_nonzero(kb[row]) == 0 and torch.count_nonzero(vb[row]) == 0
        else:
            assert torch.equal(kb[row], kb_ref[row]) and torch.equal(vb[row], vb_ref[row]), r


def test_realign_reports_v_outside_fp16_range(kvb):
    """A chunk-cache V value beyond fp16's finite range (|v| > 65504) cannot be held by the
    blended cache's fp16 containers: the merge writes it as +-65504, keeps NaN as NaN,
    converts every other value exactly and records KVB_ERR_RANGE; the largest bf16 value
    that fits (65280) and the smallest normal fp16 magnitude pass without a report."""
    shape = TINY
    cfg = kvb.config(shape)
    L, n_ctx, Hkv, D = 1, 8, shape.n_kv_heads, shape.head_dim
    starts = dev(torch.tensor([0, 5, 8], dtype=torch.int32))
    rope = kvb.RopeTable(cfg, n_ctx)
    k = dev(synth.randn_bf16((L, n_ctx, Hkv, D), 501))
    v = synth.randn_bf16((L, n_ctx, Hkv, D), 502)
    v[0, 1, 0, 3] = 65280.0                              # largest bf16 value below fp16's limit
    v[0, 2, 1, 0] = -(2.0 ** -14)                        # smallest normal fp16 magnitude
    ws = torch.zeros(256, dtype=torch.uint8, device="cuda")
    kd = torch.zeros(L, n_ctx, Hkv, D, dtype=torch.bfloat16, device="cuda")
    vd = torch.zeros(L, n_ctx, Hkv, D, dtype=torch.float16, device="cuda")
    kvb.rope_realign(cfg, rope, k, dev(v), kd, vd, 0, L, starts, n_ctx, ws=ws)
    assert kvb.device_status(ws) == kvb.KVB_OK
    assert torch.equal(vd.cpu(), v.to(torch.float16))
    vbad = v.clone()
    vbad[0, 3, 0, 5] = 65536.0
    vbad[0, 6, 1, 7] = -1.0e30
    vbad[0, 7, 0, 0] = float("inf")
    vbad[0, 4, 1, 1] = float("nan")
    kvb.rope_realign(cfg, rope, k, dev(vbad), kd, vd, 0, L, starts, n_ctx, ws=ws)
    assert kvb.device_status(ws) == kvb.KVB_ERR_RANGE
    got = vd.cpu().float()
    assert got[0, 3, 0, 5] == 65504.0 and got[0, 6, 1, 7] == -65504.0 and got[0, 7, 0, 0] == 65504.0
    assert torch.isnan(got[0, 4, 1, 1])
    want = v.to(torch.float16).float()
    mask = torch.ones_like(got, dtype=torch.bool)
    for idx in ((0, 3, 0, 5), (0, 6, 1, 7), (0, 7, 0, 0), (0, 4, 1, 1)):
        mask[idx] = False
    assert torch.equal(got[mask], want[mask])
    # in place (the same memory holds bf16 before and fp16 after) gives the same bits
    vin = dev(v).clone()
    kvb.rope_realign(cfg, rope, k, vin, kd, vin, 0, L, starts, n_ctx, ws=ws)
    assert kvb.device_status(ws) == kvb.KVB_OK
    assert torch.equal(vin.view(torch.float16).cpu(), v.to(torch.float16))


def _tiny_device_model(kvb, pad_embed_rows=0):
    w = synth.make_model(TINY, 0)
    emb = torch.zeros(TINY.vocab + pad_embed_rows, TINY.hidden, dtype=torch.bfloat16, device="cuda")
    emb[: TINY.vocab] = w["embed"].cuda()
    return kvb.Model({"layers": [{k: v.cuda() for k, v in l.items()} for l in w["layers"]],
                      "embed": emb[: TINY.vocab], "final_norm": w["final_norm"].cuda()})


def test_token_ids_outside_the_vocabulary_are_reported(kvb):
    """A token id outside [0, vocab) embeds as a zero row and sets KVB_ERR_INVALID_ARG in
    the status word; the next valid call reports nothing.  The embedding table is a view
    of a larger buffer, so the row just past the vocabulary is memory of this test."""
    cfg = kvb.config(TINY)
    model = _tiny_device_model(kvb, pad_embed_rows=1)
    n = 40
    rope = kvb.RopeTable(cfg, n)
    toks = synth.make_tokens(TINY, n, 3).cuda()
    ck = torch.zeros(TINY.n_layers, n, TINY.n_kv_heads, TINY.head_dim, dtype=torch.bfloat16, device="cuda")
    cv = torch.zeros(ck.shape, dtype=torch.float16, device="cuda")
    ws = kvb.workspace(cfg, n)
    bad = toks.clone()
    bad[7] = TINY.vocab
    kvb.full_prefill(cfg, model, rope, ck, cv, bad, n_out=1, ws=ws)
    assert kvb.device_status(ws) == kvb.KVB_ERR_INVALID_ARG
    fh, _ = kvb.full_prefill(cfg, model, rope, ck, cv, toks, n_out=1, ws=ws)
    assert kvb.device_status(ws) == kvb.KVB_OK
    assert torch.isfinite(fh).all()


def test_forced_selection_outside_the_context_is_reported(kvb):
    """A forced selected row outside [0, n_ctx) is reported as KVB_ERR_INVALID_ARG in the
    status word and replaced by row 0 (row n_ctx, the one named here, exists in the
    workspace and the cache, so nothing outside them is touched either way)."""
    wl = synth.WORKLOADS["tiny"]
    cfg = kvb.config(TINY)
    model = _tiny_device_model(kvb)
    rope = kvb.RopeTable(cfg, wl.n_total)
    toks = wl.tokens().cuda()
    kch = torch.zeros(TINY.n_layers, wl.n_ctx, TINY.n_kv_heads, TINY.head_dim, dtype=torch.bfloat16, device="cuda")
    vch = torch.zeros(kch.shape, dtype=torch.bfloat16, device="cuda")
    ck = torch.zeros(TINY.n_layers, wl.n_total, TINY.n_kv_heads, TINY.head_dim, dtype=torch.bfloat16, device="cuda")
    cv = torch.zeros(ck.shape, dtype=torch.float16, device="cuda")
    starts = torch.tensor(wl.chunk_starts(), dtype=torch.int32, device="cuda")
    ws = kvb.workspace(cfg, wl.n_total)
    for forced, want in (([3, 9, wl.n_ctx], kvb.KVB_ERR_INVALID_ARG), ([3, 9, wl.n_ctx - 1], kvb.KVB_OK)):
        sel = torch.tensor(forced, dtype=torch.int32, device="cuda")
        kvb.selective_prefill(cfg, model, rope, kch, vch, ck, cv, toks, starts, wl.n_ctx, wl.n_query, 0.0, 1,
                              forced_sel=sel, ws=ws)
        assert kvb.device_status(ws) == want


def test_bounded_wait_reports_timeout_and_context_survives(kvb):
    """A wait that nothing completes gives up after its limit and reports KVB_ERR_TIMEOUT
    through the status word; the context stays usable and the word is cleared on read."""
    ws = torch.zeros(256, dtype=torch.uint8, device="cuda")
    assert kvb.device_status(ws) == kvb.KVB_OK
    kvb.debug_wait_timeout(ws, 5_000_000)          # 5 ms
    assert kvb.device_status(ws) == kvb.KVB_ERR_TIMEOUT
    assert kvb.device_status(ws) == kvb.KVB_OK       # cleared
    # the device still runs the real kernels correctly afterwards
    kr = synth.randn_bf16((4, 128), 7)
    idx = torch.tensor([3, 0, 5, 1], dtype=torch.int32)
    kd = torch.zeros(6, 128, dtype=torch.bfloat16, device="cuda")
    vd = torch.zeros(6, 128, dtype=torch.float16, device="cuda")
    kvb.kv_scatter(dev(kr), dev(kr.to(torch.float16)), dev(idx), kd, vd)
    torch.cuda.synchronize()
    assert torch.equal(kd.cpu()[idx.long()], kr)


# ------------------------------------------------------------------------------------- first token

def _lm_head_bound(h64, w64):
    """Worst-case error of an fp32 dot product of length H against the exact value:
    gamma_H * sum_i |w_i x_i| with gamma_H = H u / (1 - H u), u = 2^-24 (round to nearest)."""
    u = 2.0 ** -24
    H = h64.shape[1]
    gamma = H * u / (1 - H * u)
    return gamma * (np.abs(h64) @ np.abs(w64).T)          # [n, vocab]


def _check_first_token(kvb, shape, h, w, with_logits=True):
    n = h.shape[0]
    cfg = kvb.config(shape)
    logits = torch.empty(n, shape.vocab, dtype=torch.float32, device="cuda") if with_logits else None
    tok, _ = kvb.lm_head_argmax(cfg, dev(w), dev(h), logits)
    torch.cuda.synchronize()
    tok = tok.cpu().numpy().astype(np.int64)
    h64, w64 = np64(h), np64(w)
    want_tok, want_logits = blend.first_token(h64, w64)
    bound = _lm_head_bound(h64, w64)
    if with_logits:
        got = np64(logits.cpu())
        assert np.all(np.abs(got - want_logits) <= bound), np.abs(got - want_logits).max()
    rows = np.arange(n)
    # the chosen token's exact logit is within two error bounds of the exact maximum ...
    assert np.all(want_logits[rows, tok] >= want_logits[rows, want_tok] - bound[rows, tok] - bound[rows, want_tok])
    # ... and is the oracle's token wherever the top-two gap exceeds those bounds
    srt = np.sort(want_logits, axis=1)
    gap = srt[:, -1] - srt[:, -2] if shape.vocab > 1 else np.full(n, np.inf)
    clear = gap > 2 * bound.max(axis=1)
    assert np.array_equal(tok[clear], want_tok[clear])
    return tok, want_tok


@pytest.mark.parametrize("vocab,hidden,n", [
    (128256, 4096, 1),          # Llama-3.1-8B output layer, one query row
    (128256, 4096, 4),          # the most rows one call takes
    (50001, 4096, 3),           # ragged vocabulary
    (1024, 256, 2),
    (1, 256, 1),                # a one-token vocabulary
])
def test_lm_head_argmax_matches_oracle(kvb, vocab, hidden, n):
    shape = synth.ModelShape(hidden, 4, 2, 64, 4 * hidden, 1, vocab)
    w = synth.randn_bf16((vocab, hidden), 501 + n, 0.02)
    h = torch.randn(n, hidden, generator=torch.Generator().manual_seed(vocab + n), dtype=torch.float64).float()
    _check_first_token(kvb, shape, h, w)
    if vocab > 1:
        _check_first_token(kvb, shape, h, w, with_logits=False)


def test_lm_head_argmax_ties_and_negative_logits(kvb):
    """Equal weight rows give bit-equal fp32 logits (same reduction order for every row);
    the lowest id must win.  All-negative logits exercise the sign handling of the key."""
    vocab, hidden = 4099, 512
    shape = synth.ModelShape(hidden, 4, 2, 64, 4 * hidden, 1, vocab)
    w = synth.randn_bf16((vocab, hidden), 511, 0.02)
    h = torch.randn(2, hidden, generator=torch.Generator().manual_seed(5), dtype=torch.float64).float()
    # row 0: make token 3000 the clear winner, duplicated at ids 17 and 4098
    w[3000] = (h[0].sign() * 0.05).to(torch.bfloat16)
    w[17] = w[3000]
    w[4098] = w[3000]
    tok, _ = _check_first_token(kvb, shape, h, w)
    assert tok[0] == 17
    # all logits negative: W rows anti-aligned with h, the least negative wins
    wn = -(h[1].sign() * (0.01 + 0.01 * torch.rand(vocab, 1, generator=torch.Generator().manual_seed(6)))).to(
        torch.bfloat16)
    tok, want = _check_first_token(kvb, shape, h[1:].contiguous(), wn.contiguous())
    assert tok[0] == want[0]


def test_lm_head_argmax_rejects_bad_arguments(kvb):
    shape = synth.ModelShape(256, 4, 2, 64, 1024, 1, 64)
    cfg = kvb.config(shape)
    w = dev(synth.randn_bf16((64, 256), 3))
    for n in (0, kvb.LMHEAD_MAX_ROWS + 1):
        h = torch.zeros(n, 256, device="cuda")
        with pytest.raises(kvb.KvbError):
            kvb.lm_head_argmax(cfg, w, h, tokens=torch.empty(max(n, 1), dtype=torch.int32, device="cuda"))
    with pytest.raises(kvb.KvbError):
        kvb.lm_head_argmax(cfg, w, torch.zeros(1, 256, device="cuda"),
                           ws=torch.zeros(64, dtype=torch.uint8, device="cuda"))


# ---------------------------------------------------------------- EPIC / KVLink windows, deviation histogram

@pytest.mark.parametrize("starts,window,n_ctx", [
    (synth.WORKLOADS["l8b_124k_sep"].sep_starts(), 20, synth.WORKLOADS["l8b_124k_sep"].n_ctx),   # EPIC, 124k
    (synth.WORKLOADS["l8b_124k_sep"].sep_starts(), 2, synth.WORKLOADS["l8b_124k_sep"].n_ctx),    # KVLink
    ([5, 3, 40, -7, 97, 1000, 99], 20, 100),       # overlapping, unsorted, outside the context
    ([], 20, 100),
    ([0, 10], 0, 100),
    ([0], 50000, 40000),                             # one window covering everything
])
def test_window_select_bit_exact(kvb, starts, window, n_ctx):
    sel, k = kvb.window_select(torch.tensor(starts, dtype=torch.int32, device="cuda"), window, n_ctx)
    want = blend.window_select(starts, window, n_ctx)
    assert k == len(want) and np.array_equal(sel.cpu().numpy(), want)


@pytest.mark.parametrize("n,kv_dim,ld", [(123904, 1024, 1024), (1000, 128, 256), (1, 8, 8), (0, 1024, 1024)])
def test_key_deviation_histogram(kvb, n, kv_dim, ld):
    a = synth.randn_bf16((max(n, 1), ld), 601)[:n]
    b = (a.float() + synth.randn_bf16((max(n, 1), ld), 602, 0.05)[:n].float()
         * torch.rand(max(n, 1), 1, generator=torch.Generator().manual_seed(3))[:n] ** 4).to(torch.bfloat16)
    b[: n // 3] = a[: n // 3]                        # exact zeros
    edges = torch.tensor([0.0] + [10.0 ** e for e in np.arange(-8, 3.01, 0.25)], dtype=torch.float32)
    da, db = dev(a), dev(b)
    d = torch.empty(max(n, 1), dtype=torch.float32, device="cuda")
    h = kvb.key_deviation_histogram(da[:, :kv_dim], db[:, :kv_dim], dev(edges), dev_out=d[:n] if n else None)
    h2 = kvb.key_deviation_histogram(da[:, :kv_dim], db[:, :kv_dim], dev(edges))   # deviation in the workspace
    torch.cuda.synchronize()
    got = d[:n].cpu().numpy()
    want = blend.hkvd_deviation(np64(a[:, :kv_dim]), np64(b[:, :kv_dim]))
    # fp32 sum of kv_dim exact squares of bf16 differences: relative bound kv_dim * 2^-24 (+ the square)
    assert np.all(np.abs(got - want) <= (kv_dim + 2) * 2.0 ** -24 * want)
    assert np.array_equal(h.cpu().numpy(), blend.deviation_histogram(got, edges.numpy()))
    assert torch.equal(h, h2) and int(h.sum()) == n
