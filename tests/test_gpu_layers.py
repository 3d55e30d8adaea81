"""Per-layer parity of the selective prefill, teacher-forced, on the Llama-3.1-8B-shaped
workloads: the 2-layer model (3.9k tokens) and the 32-layer stacks at 32.9k tokens
(64 x 512 + 128), 65.7k tokens (32 x 2048 + 128 at r = 0.25, the context of the r x
chunk-size sweep) and 124k tokens (242 x 512 + 128, the headline request); and on the
32-layer YaRN model with seven q heads per kv head and a q/k/v bias at 124k tokens.

One call of kvb_selective_prefill runs the whole path; layer taps capture the residual
rows entering each checked layer and leaving it, and the blended cache holds every
layer's K/V as that layer's attention read them (layer l's cache rows are not written
after layer l).  For each checked layer the oracle then recomputes, from the GPU's own
input rows and the GPU's cache (so that only this layer's rounding is judged), a sample
of at least 256 of the layer's rows with all heads: the rows' fresh q/k/v, attention over
the whole cache with the sampled rows' own K/V in place (Sec. 3.2: selected rows attend
the blended cache), O-proj and the SwiGLU MLP.  Layer 0 recomputes every row (Sec. 4);
its input rows are the token embeddings.

Bars.  The fresh K/V rows written into the cache: both sides store them in bf16, so one
bf16 ulp of the value per element (plus 2e-2 of the RMS) and mean-abs <= 2e-3 of the RMS.
The layer outputs: max-abs <= 2e-2 and mean-abs <= 2e-3 of the output's RMS, against the
float64 oracle with the bf16 storage points of the paper's bf16 model and against the
oracle's float32-accumulation run (the literal fp32 oracle).  The stated bar in absolute
units is asserted from layer 2 on (layers 15 and 31 of the 32-layer stacks) and reported for
layers 0 and 1 beside the distance between the two oracles themselves: at the first two
layers it lies within what fp32-level changes alone move the output
(tests/test_precision_floor.py), for this reason:
the residual rows have an RMS of 2.6 after layer 0 and grow with depth, and a perturbation
of one part in 10^7 before a bf16 rounding (an RMSNorm output, the attention output)
flips that rounding now and then; through the 4096 -> 14336 fan-out of the MLP a few
flips flip thousands of SwiGLU roundings, so two faithful fp32 implementations of this
random-weight model already differ by about 2e-3 mean-abs on a layer output.
"""
import numpy as np
import pytest
import torch

from oracle import blend, llama
from oracle.llama import Shape
from paper_2609_09768_gb300 import synth, workload
from tests.gpu_util import MAX_ABS, MEAN_ABS, assert_close_bf16, assert_close_rel, errs, np64

pytestmark = pytest.mark.gpu

N_SAMPLE = 256


@pytest.fixture(scope="module")
def kvb():
    from paper_2609_09768_gb300 import kvblend
    kvblend.lib()
    return kvblend


def _layers_checked(L):
    return sorted({0, 1, L // 2 - 1, L - 1} if L > 2 else set(range(L)))


def _run(kvb, wl_name):
    """Runs the selective prefill of one workload with taps around the checked layers;
    returns what the per-layer checks need (host copies of the taps, the selected set, the
    device cache and weights)."""
    wl = synth.WORKLOADS[wl_name]
    shape = wl.shape
    L = shape.n_layers
    cfg = kvb.config(shape)
    dev = torch.device("cuda")
    w = workload.device_model(shape, seed=0, device=dev, draw_on_device=L > 2)
    model = kvb.Model(w)
    N, n_ctx, nq = wl.n_total, wl.n_ctx, wl.n_query
    toks = wl.tokens(1, dev)
    rope = kvb.RopeTable(cfg, N, dev)
    ws = kvb.workspace(cfg, N, dev)
    starts = wl.chunk_starts()
    kch, vch = workload.chunk_caches(cfg, model, rope, toks[:n_ctx], starts, ws=ws)
    ck = torch.zeros(L, N, shape.n_kv_heads, shape.head_dim, dtype=torch.bfloat16, device=dev)
    cv = torch.zeros(ck.shape, dtype=torch.float16, device=dev)
    checked = _layers_checked(L)
    tap_layers = sorted({l for c in checked for l in (c, c + 1) if l >= 1})
    k = blend.num_selected(wl.r, n_ctx)
    m = k + nq
    taps = kvb.LayerTaps(tap_layers, m, shape.hidden, dev)
    dstarts = torch.tensor(starts, dtype=torch.int32, device=dev)
    fh, sel, _ = kvb.selective_prefill(cfg, model, rope, kch, vch, ck, cv, toks, dstarts, n_ctx, nq, wl.r, 1,
                                       ws=ws, taps=taps)
    torch.cuda.synchronize()
    assert kvb.device_status(ws) == kvb.KVB_OK
    for i, l in enumerate(tap_layers):
        assert taps.rows(i) == m, (l, taps.rows(i), m)
    rows = np.concatenate([np.sort(sel[:k].cpu().numpy().astype(np.int64)), np.arange(n_ctx, N)])
    assert np.all(np.diff(rows) > 0)
    del kch, vch
    return dict(wl=wl, shape=shape, L=L, w=w, toks=toks.cpu().numpy(), ck=ck, cv=cv, taps=taps,
                tap_layers=tap_layers, rows=rows, checked=checked, N=N, n_ctx=n_ctx, m=m, starts=starts,
                fh=fh.cpu())


def _sample(run, seed):
    """At least N_SAMPLE of the recomputed rows (indices into the m tap rows): the first and
    last selected rows, the first and last query rows, rows right after a chunk start if
    selected, the rest uniform."""
    m, rows, n_ctx = run["m"], run["rows"], run["n_ctx"]
    if m <= N_SAMPLE:
        return np.arange(m)
    k = m - run["wl"].n_query
    must = {0, max(k - 1, 0), k, m - 1}
    at_start = np.nonzero(np.isin(rows, np.asarray(run["starts"][:-1])))[0]
    must.update(at_start[:16].tolist())
    rng = np.random.default_rng(seed)
    rest = rng.choice(np.setdiff1d(np.arange(m), list(must)), N_SAMPLE - len(must), replace=False)
    return np.sort(np.concatenate([np.array(sorted(must)), rest]))


def _layer_np(w, l):
    return {k: llama.as64(v) for k, v in w["layers"][l].items()}


def _check_layer(run, l, smp, what):
    shape = run["shape"]
    s = Shape.of(shape, act_bf16=True)
    s32 = Shape.of(shape, act_bf16=True, accum32=True)
    pos = run["rows"][smp]
    taps = run["taps"]
    ti = {t: i for i, t in enumerate(run["tap_layers"])}
    if l == 0:
        x_in = blend.embed_rows(run["w"]["embed"], run["toks"][pos])
    else:
        x_in = np64(taps.get(ti[l])[torch.from_numpy(smp).cuda()])
    x_out = np64(taps.get(ti[l + 1])[torch.from_numpy(smp).cuda()])
    lw = _layer_np(run["w"], l)
    kc = np64(run["ck"][l, : int(pos.max()) + 1].cpu())
    vc = np64(run["cv"][l, : int(pos.max()) + 1].cpu())
    k_gpu, v_gpu = kc[pos].copy(), vc[pos].copy()
    outs, kv = {}, {}
    for name, sh in (("fp64", s), ("fp32acc", s32)):
        q, kr, vr = llama.qkv_rows(sh, lw, x_in, pos)
        kk, vv = kc.copy(), vc.copy()
        kk[pos], vv[pos] = kr, vr                      # the sampled rows' own K/V, as the oracle computes them
        a = llama.act(sh, llama.attention_rows(sh, q, kk, vv, pos))
        outs[name] = llama.attn_out_mlp(sh, lw, x_in, a.reshape(len(pos), -1))
        kv[name] = (kr.reshape(len(pos), -1), vr.reshape(len(pos), -1))
    e64, e32 = errs(x_out, outs["fp64"]), errs(x_out, outs["fp32acc"])
    floor = errs(outs["fp32acc"], outs["fp64"])        # two faithful oracles of the same bf16 model
    rms = e64["rms_ref"]
    absolute = e64["max_abs"] <= MAX_ABS and e64["mean_abs"] <= MEAN_ABS
    print(f"{what} layer {l}: {len(pos)} rows, output rms {rms:.3f}; GPU vs fp64 oracle max {e64['max_abs']:.3e} "
          f"mean {e64['mean_abs']:.3e}; GPU vs fp32-accumulation oracle max {e32['max_abs']:.3e} "
          f"mean {e32['mean_abs']:.3e}; fp32-accumulation vs fp64 oracle max {floor['max_abs']:.3e} "
          f"mean {floor['mean_abs']:.3e}; absolute bar (2e-2 / 2e-3) {'met' if absolute else 'NOT met'}")
    # fresh K/V rows: both sides store bf16, judged per element within one bf16 ulp + 2e-2 rms, mean 2e-3 rms
    ek = assert_close_bf16(k_gpu.reshape(len(pos), -1), kv["fp64"][0], f"{what} layer {l} K")
    ev = assert_close_bf16(v_gpu.reshape(len(pos), -1), kv["fp64"][1], f"{what} layer {l} V")
    print(f"{what} layer {l}: K {ek}, V {ev}")
    # layer output: the stated bar relative to the output's RMS, and in absolute units from layer 2 on
    assert_close_rel(x_out, outs["fp64"], f"{what} layer {l} output vs fp64 oracle")
    if l >= 2:
        assert absolute, f"{what} layer {l} output vs fp64 oracle, absolute bar: {e64}"
    assert_close_rel(x_out, outs["fp32acc"], f"{what} layer {l} output vs fp32-accumulation oracle")
    return dict(e64=e64, e32=e32, floor=floor, absolute=absolute)


_RUNS = {}


@pytest.fixture(scope="module", params=["l8b_1layer", "l8b_32k", "l8b_64k", "l8b_124k", "yarn_124k"])
def run(request, kvb):
    # one workload resident at a time (the 124k one holds ~40 GB of caches and weights)
    for key in list(_RUNS):
        if key != request.param:
            del _RUNS[key]
    torch.cuda.empty_cache()
    if request.param not in _RUNS:
        _RUNS[request.param] = _run(kvb, request.param)
    return _RUNS[request.param]


def test_layers_teacher_forced_match_oracle(run):
    smp = _sample(run, 7)
    assert len(smp) >= min(N_SAMPLE, run["m"])
    for l in run["checked"]:
        _check_layer(run, l, smp, run["wl"].name)


def test_final_hidden_is_the_last_tap_normalised(run):
    """The final hidden state the call returns is the final RMSNorm of the query rows that
    leave the last layer (the last tap), so the per-layer checks reach the output: the GPU's
    fp32 RMSNorm of those rows against the oracle's float64 one on the same rows."""
    L, nq = run["L"], run["wl"].n_query
    ti = {t: i for i, t in enumerate(run["tap_layers"])}
    last = np64(run["taps"].get(ti[L])[-nq:])
    want = llama.rmsnorm(last, np64(run["w"]["final_norm"].cpu()), run["shape"].rms_eps)
    e = errs(run["fh"], want)
    assert e["max_abs"] <= 1e-5 * max(1.0, float(np.abs(want).max())), e
