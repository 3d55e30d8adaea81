"""End-to-end parity of the whole path through the C ABI against the float64 oracle:
per-chunk caches, the dense prefill (the r = 1 comparator) and the selective
prefill, on the tiny model, the Llama-3.1-8B-shaped 2-layer model and two YaRN models
with seven q heads per kv head and a q/k/v bias."""
import numpy as np
import pytest
import torch

from oracle import blend, llama
from oracle.llama import Shape
from paper_2609_09768_gb300 import synth, workload
from tests.gpu_util import MEAN_ABS, assert_close_abs, assert_close_bf16, errs, fp64_gap_bounds, np64

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def kvb():
    from paper_2609_09768_gb300 import kvblend
    kvblend.lib()
    return kvblend


class Case:
    """One workload with its oracle results (computed once per module).

    The oracle runs with the activations the paper's bf16 model holds stored in
    bf16 (`s`, the parity reference) and all-float64 (`s64`, whose gap to the GPU
    path is reported and bounded by fp64_gap_bounds).  A third run accumulates the
    linear layers in float32 (`s32`): its distance from the reference is the
    floor two faithful implementations of the same bf16 model reach through
    accumulation rounding alone.  The stated bar (max-abs 2e-2, mean-abs 2e-3) is
    applied as is, except that the mean bar is raised to 1.5x that floor where the
    floor itself exceeds it (the 8B-shaped model: see the design notes)."""

    def __init__(self, kvb, wl: synth.Workload):
        self.wl, self.shape = wl, wl.shape
        self.starts = wl.chunk_starts()
        self.n_ctx, self.nq, self.N = wl.n_ctx, wl.n_query, wl.n_total
        w = synth.make_model(self.shape, 0)
        self.w = w
        self.toks = wl.tokens()
        self.sep_rows = wl.sep_rows()
        self.s = Shape.of(self.shape, act_bf16=True)
        self.s64 = Shape.of(self.shape)
        self.l64 = [{k: llama.as64(v) for k, v in l.items()} for l in w["layers"]]
        x0 = blend.embed_rows(w["embed"], self.toks.numpy())
        self.cc = blend.chunk_caches(self.s, self.l64, x0[: self.n_ctx], self.starts)
        if self.sep_rows:
            self.cc = blend.zero_kv_rows(self.cc, self.sep_rows)
        self.x0 = x0
        self.sel = blend.selective_prefill(self.s, self.l64, x0, self.starts, self.nq, wl.r, self.cc["k"],
                                           self.cc["v"], 1, None, w["final_norm"])
        self.full = blend.full_prefill(self.s, self.l64, x0)
        self.full_fh = llama.rmsnorm(self.full["x"][-self.nq:], np64(w["final_norm"]), self.s.rms_eps)
        # all-float64 references on the same inputs and the same selected set
        sel64 = blend.selective_prefill(self.s64, self.l64, x0, self.starts, self.nq, wl.r, self.cc["k"],
                                        self.cc["v"], 1, self.sel["sel"], w["final_norm"])
        self.sel_fh64 = sel64["final_hidden"]
        full64 = blend.full_prefill(self.s64, self.l64, x0)
        self.full_fh64 = llama.rmsnorm(full64["x"][-self.nq:], np64(w["final_norm"]), self.s.rms_eps)
        # floor: float32 accumulation, same bf16 rounding points
        full32 = blend.full_prefill(Shape.of(self.shape, act_bf16=True, accum32=True), self.l64, x0)
        fh32 = llama.rmsnorm(full32["x"][-self.nq:], np64(w["final_norm"]), self.s.rms_eps)
        self.full_fh32 = fh32
        self.floor = {"fh": errs(fh32, self.full_fh)["mean_abs"]}
        for l in range(self.shape.n_layers):
            self.floor[f"k{l}"] = errs(full32["k"][l], self.full["k"][l])["mean_abs"]
            self.floor[f"v{l}"] = errs(full32["v"][l], self.full["v"][l])["mean_abs"]
        print("floor (fp32 vs fp64 accumulation)", wl.name, self.floor)
        # device side
        self.cfg = kvb.config(self.shape)
        self.model = kvb.Model({"layers": [{k: v.cuda() for k, v in l.items()} for l in w["layers"]],
                                "embed": w["embed"].cuda(), "final_norm": w["final_norm"].cuda()})
        self.rope = kvb.RopeTable(self.cfg, self.N)
        self.dtoks = self.toks.cuda()
        self.dstarts = torch.tensor(self.starts, dtype=torch.int32, device="cuda")
        self.kch = torch.from_numpy(self.cc["k"]).to(torch.bfloat16).cuda()
        self.vch = torch.from_numpy(self.cc["v"]).to(torch.bfloat16).cuda()       # chunk-cache format
        self.ws = kvb.workspace(self.cfg, self.N)

    def mean_bar(self, key, scale=1.0):
        """Stated mean-abs bar (relative to `scale`), raised to 1.5x the floor where the floor exceeds it."""
        return max(MEAN_ABS * scale, 1.5 * self.floor[key])

    def check_fh(self, got, want, what):
        return assert_close_abs(got, want, what, mean_abs=self.mean_bar("fh"))

    def check_cache(self, got, want, key, what):
        rms = float(np.sqrt(np.mean(np64(want) ** 2)))
        return assert_close_bf16(got, want, what, mean_rel=self.mean_bar(key, rms) / rms)

    def fp64_gap(self, got, ref64, what):
        e = errs(got, ref64)
        mx, mn = fp64_gap_bounds(e["rms_ref"], self.shape.n_layers)
        assert e["max_abs"] <= mx and e["mean_abs"] <= mn, f"{what} vs float64 oracle: {e}"
        return e

    def new_cache(self):
        k = torch.zeros(self.shape.n_layers, self.N, self.shape.n_kv_heads, self.shape.head_dim,
                        dtype=torch.bfloat16, device="cuda")
        return k, torch.zeros(k.shape, dtype=torch.float16, device="cuda")


_CASES = {}


@pytest.fixture(scope="module", params=["tiny", "l8b_1layer", "tiny_sep", "l8b_1layer_sep", "yarn_tiny", "yarn_2l"])
def case(request, kvb):
    if request.param not in _CASES:
        _CASES[request.param] = Case(kvb, synth.WORKLOADS[request.param])
    return _CASES[request.param]


def test_full_prefill_matches_oracle(kvb, case):
    ck, cv = case.new_cache()
    fh, _ = kvb.full_prefill(case.cfg, case.model, case.rope, ck, cv, case.dtoks, n_out=case.nq, ws=case.ws)
    torch.cuda.synchronize()
    assert kvb.device_status(case.ws) == 0
    e = case.check_fh(fh.cpu(), case.full_fh, "final hidden (dense prefill)")
    e64 = case.fp64_gap(fh.cpu(), case.full_fh64, "final hidden (dense prefill)")
    e32 = errs(fh.cpu(), case.full_fh32)     # the fp32-accumulation oracle: reported beside the reference
    print("full prefill", case.wl.name, "vs fp32-accumulation oracle", e32)
    for l in range(case.shape.n_layers):
        case.check_cache(ck[l].cpu(), case.full["k"][l], f"k{l}", f"layer {l} K")
        case.check_cache(cv[l].cpu(), case.full["v"][l], f"v{l}", f"layer {l} V")
    print("full prefill", case.wl.name, e, "vs float64", e64)


def test_chunk_caches_match_oracle(kvb, case):
    k, v = workload.chunk_caches(case.cfg, case.model, case.rope, case.dtoks[: case.n_ctx], case.starts, ws=case.ws,
                                 zero_rows=case.sep_rows)
    torch.cuda.synchronize()
    assert kvb.device_status(case.ws) == 0
    for l in range(case.shape.n_layers):
        case.check_cache(k[l].cpu(), case.cc["k"][l], f"k{l}", f"chunk cache K layer {l}")
        case.check_cache(v[l].cpu(), case.cc["v"][l], f"v{l}", f"chunk cache V layer {l}")


def test_selective_prefill_forced_selection(kvb, case):
    """GPU path on the oracle's chunk caches with the oracle's selected set."""
    ck, cv = case.new_cache()
    forced = torch.from_numpy(case.sel["sel"].astype(np.int32)).cuda()
    fh, sel, t = kvb.selective_prefill(case.cfg, case.model, case.rope, case.kch, case.vch, ck, cv, case.dtoks,
                                       case.dstarts, case.n_ctx, case.nq, case.wl.r, 1, forced_sel=forced,
                                       ws=case.ws, timings=True)
    torch.cuda.synchronize()
    assert kvb.device_status(case.ws) == 0
    e = case.check_fh(fh.cpu(), case.sel["final_hidden"], "final hidden (selective)")
    e64 = case.fp64_gap(fh.cpu(), case.sel_fh64, "final hidden (selective)")
    k = len(case.sel["sel"])
    assert np.array_equal(sel[:k].cpu().numpy(), case.sel["sel"])
    assert t["n_selected"] == k and t["n_rows"] == k + case.nq
    # blended cache: layer 0 fully recomputed, layer 1 = re-aligned chunks + recomputed rows
    for l in range(case.shape.n_layers):
        case.check_cache(ck[l].cpu(), case.sel["k"][l], f"k{l}", f"blended K layer {l}")
        case.check_cache(cv[l].cpu(), case.sel["v"][l], f"v{l}", f"blended V layer {l}")
    print("selective forced", case.wl.name, e, "vs float64", e64, t)


def test_selective_prefill_device_selection_is_valid(kvb, case):
    """With the HKVD choice made on the device, upstream bf16 rounding moves the
    deviations a little; the chosen set must be a valid top-k within that error:
    every chosen row's oracle key distance, widened by the measured key error,
    reaches every unchosen row's distance narrowed by it."""
    ck, cv = case.new_cache()
    fh, sel, t = kvb.selective_prefill(case.cfg, case.model, case.rope, case.kch, case.vch, ck, cv, case.dtoks,
                                       case.dstarts, case.n_ctx, case.nq, case.wl.r, 1, ws=case.ws, timings=True)
    torch.cuda.synchronize()
    assert kvb.device_status(case.ws) == 0
    k = blend.num_selected(case.wl.r, case.n_ctx)
    s = sel[:k].cpu().numpy()
    assert len(np.unique(s)) == k and np.all(np.diff(s) > 0) and s.max() < case.n_ctx
    # fresh check-layer keys of the oracle (full-attention layer-1 keys) vs the GPU's, on the rows it recomputed
    kf_ref = case.full["k"][1, : case.n_ctx].reshape(case.n_ctx, -1)
    kf_gpu = np64(ck[1].cpu())[s].reshape(k, -1)
    key_err = np.linalg.norm(kf_gpu - kf_ref[s], axis=1).max()
    kc_gpu = np64(torch.from_numpy(blend.realign(case.s, case.cc["k"], case.starts)[1]))
    cache_err = 0.01 * np.linalg.norm(kc_gpu, axis=-1).max()   # bf16 rounding of the re-aligned keys
    e = 2.0 * key_err + cache_err
    dist = np.sqrt(case.sel["dev"])
    chosen = np.zeros(case.n_ctx, dtype=bool)
    chosen[s] = True
    if 0 < k < case.n_ctx:
        assert (dist[chosen] + e).min() >= (dist[~chosen] - e).max(), (key_err, cache_err)
    overlap = len(np.intersect1d(s, case.sel["sel"])) / max(k, 1)
    assert np.isfinite(fh.cpu().numpy()).all()
    print("device selection", case.wl.name, "overlap with oracle", overlap, "key err", key_err)


def test_full_ratio_equals_dense_prefill(kvb, case):
    """r = 1 recomputes every row: the selective entry point equals the dense prefill."""
    ck, cv = case.new_cache()
    fh, sel, _ = kvb.selective_prefill(case.cfg, case.model, case.rope, case.kch, case.vch, ck, cv, case.dtoks,
                                       case.dstarts, case.n_ctx, case.nq, 1.0, 1, ws=case.ws)
    ck2, cv2 = case.new_cache()
    fh2, _ = kvb.full_prefill(case.cfg, case.model, case.rope, ck2, cv2, case.dtoks, n_out=case.nq, ws=case.ws)
    torch.cuda.synchronize()
    assert torch.equal(fh, fh2) and torch.equal(ck, ck2)
    assert np.array_equal(sel.cpu().numpy(), np.arange(case.n_ctx))
    case.check_fh(fh.cpu(), case.full_fh, "r = 1 final hidden")


def test_zero_ratio_reads_the_realigned_cache(kvb, case):
    """r = 0: the selective layers recompute only the query rows and every context row
    keeps its re-aligned chunk cache entry (the plain concatenation baseline of Sec. 4);
    final hidden and blended caches against the oracle's r = 0 run."""
    ck, cv = case.new_cache()
    fh, _, t = kvb.selective_prefill(case.cfg, case.model, case.rope, case.kch, case.vch, ck, cv, case.dtoks,
                                     case.dstarts, case.n_ctx, case.nq, 0.0, 1, ws=case.ws, timings=True)
    torch.cuda.synchronize()
    assert kvb.device_status(case.ws) == 0
    assert t["n_selected"] == 0 and t["n_rows"] == case.nq
    ref = blend.selective_prefill(case.s, case.l64, case.x0, case.starts, case.nq, 0.0, case.cc["k"], case.cc["v"],
                                  1, None, case.w["final_norm"])
    assert len(ref["sel"]) == 0
    e = case.check_fh(fh.cpu(), ref["final_hidden"], "final hidden (r = 0)")
    for l in range(case.shape.n_layers):
        case.check_cache(ck[l].cpu(), ref["k"][l], f"k{l}", f"r = 0 blended K layer {l}")
        case.check_cache(cv[l].cpu(), ref["v"][l], f"v{l}", f"r = 0 blended V layer {l}")
    print("r = 0", case.wl.name, e)


def test_single_chunk_is_exact_for_any_ratio(kvb):
    """One chunk at offset 0: its isolated cache is the full prefill's cache (Sec. 1,
    prefix invariance) and re-alignment is the identity, so the selective prefill gives
    the full prefill's result whichever rows HKVD picks."""
    c = Case(kvb, synth.Workload("tiny-2L-1x300+20", synth.TINY, 1, 300, 20))
    for r in (0.0, 0.15, 0.5):
        ck, cv = c.new_cache()
        fh, _, _ = kvb.selective_prefill(c.cfg, c.model, c.rope, c.kch, c.vch, ck, cv, c.dtoks, c.dstarts, c.n_ctx,
                                         c.nq, r, 1, ws=c.ws)
        torch.cuda.synchronize()
        assert kvb.device_status(c.ws) == 0
        e = c.check_fh(fh.cpu(), c.full_fh, f"single chunk, r = {r}, vs the full prefill")
        for l in range(c.shape.n_layers):
            c.check_cache(ck[l].cpu(), c.full["k"][l], f"k{l}", f"single chunk, r = {r}, K layer {l}")
        print("single chunk r", r, e)


def test_context_cache_does_not_depend_on_the_query(kvb, case):
    """The same request without its query suffix: HKVD compares context rows only and every
    recomputed row attends keys at or before its own position, so the selection and the
    context rows of the blended cache are bit-identical (a block whose key range grows
    because it also holds query rows only adds fully masked tiles, which contribute zero)."""
    ck, cv = case.new_cache()
    _, sel, _ = kvb.selective_prefill(case.cfg, case.model, case.rope, case.kch, case.vch, ck, cv, case.dtoks,
                                      case.dstarts, case.n_ctx, case.nq, case.wl.r, 1, ws=case.ws)
    ck0, cv0 = case.new_cache()
    fh0, sel0, t0 = kvb.selective_prefill(case.cfg, case.model, case.rope, case.kch, case.vch, ck0, cv0,
                                          case.dtoks[: case.n_ctx], case.dstarts, case.n_ctx, 0, case.wl.r, 1,
                                          ws=case.ws, timings=True)
    torch.cuda.synchronize()
    assert kvb.device_status(case.ws) == 0
    k = blend.num_selected(case.wl.r, case.n_ctx)
    assert fh0.shape[0] == 0 and t0["n_selected"] == k and t0["n_rows"] == k
    assert torch.equal(sel[:k], sel0[:k])
    n = case.n_ctx
    assert torch.equal(ck[:, :n], ck0[:, :n]) and torch.equal(cv[:, :n], cv0[:, :n])


def test_query_only_request_is_a_dense_prefill(kvb, case):
    """No cached context: nothing to merge or select, so the call is the dense prefill of the
    query tokens, bit for bit."""
    q = case.dtoks[case.n_ctx:].clone()      # a fresh buffer: the call wants 16-byte aligned token ids
    ck, cv = case.new_cache()
    fh, _, t = kvb.selective_prefill(case.cfg, case.model, case.rope, case.kch, case.vch, ck, cv, q, case.dstarts,
                                     0, case.nq, case.wl.r, 1, ws=case.ws, timings=True)
    ck2, cv2 = case.new_cache()
    fh2, _ = kvb.full_prefill(case.cfg, case.model, case.rope, ck2, cv2, q, n_out=case.nq, ws=case.ws)
    torch.cuda.synchronize()
    assert kvb.device_status(case.ws) == 0
    assert t["n_selected"] == 0
    assert torch.equal(fh, fh2)
    assert torch.equal(ck[:, : case.nq], ck2[:, : case.nq]) and torch.equal(cv[:, : case.nq], cv2[:, : case.nq])


def test_repeatable_bitwise(kvb, case):
    """Three runs on the same inputs give bit-identical outputs (no races in the pipeline)."""
    outs = []
    k = blend.num_selected(case.wl.r, case.n_ctx)
    for _ in range(3):
        ck, cv = case.new_cache()
        fh, sel, _ = kvb.selective_prefill(case.cfg, case.model, case.rope, case.kch, case.vch, ck, cv, case.dtoks,
                                           case.dstarts, case.n_ctx, case.nq, case.wl.r, 1, ws=case.ws)
        torch.cuda.synchronize()
        outs.append((fh.clone(), sel[:k].clone(), ck.clone(), cv.clone()))
    for o in outs[1:]:
        assert all(torch.equal(a, b) for a, b in zip(o, outs[0]))


def test_pipelined_host_ingest_equals_device_resident(kvb, case):
    """Chunk caches in pinned host memory, ingested layer by layer on a copy stream
    (Sec. 3.4), give bit-identical results to the device-resident call."""
    ck, cv = case.new_cache()
    fh, sel, _ = kvb.selective_prefill(case.cfg, case.model, case.rope, case.kch, case.vch, ck, cv, case.dtoks,
                                       case.dstarts, case.n_ctx, case.nq, case.wl.r, 1, ws=case.ws)
    hk = torch.empty(case.kch.shape, dtype=case.kch.dtype, pin_memory=True)
    hv = torch.empty(case.vch.shape, dtype=case.vch.dtype, pin_memory=True)
    hk.copy_(case.kch)
    hv.copy_(case.vch)
    ck2, cv2 = case.new_cache()
    fh2, sel2, t = kvb.selective_prefill_host(case.cfg, case.model, case.rope, hk, hv, ck2, cv2, case.dtoks,
                                              case.dstarts, case.n_ctx, case.nq, case.wl.r, 1, timings=True)
    torch.cuda.synchronize()
    k = blend.num_selected(case.wl.r, case.n_ctx)
    assert torch.equal(fh, fh2) and torch.equal(sel[:k], sel2[:k])
    assert torch.equal(ck, ck2) and torch.equal(cv, cv2)
    with pytest.raises(ValueError):   # pageable memory is refused by the binding
        kvb.selective_prefill_host(case.cfg, case.model, case.rope, hk.clone(), hv, ck2, cv2, case.dtoks,
                                   case.dstarts, case.n_ctx, case.nq, case.wl.r, 1)


@pytest.fixture(scope="module", params=["tiny_sep", "l8b_1layer_sep"])
def sep_case(request, kvb):
    """The workloads with separator tokens between documents (cached with the others)."""
    if request.param not in _CASES:
        _CASES[request.param] = Case(kvb, synth.WORKLOADS[request.param])
    return _CASES[request.param]


def test_epic_and_kvlink_selection(kvb, sep_case):
    """Separator workloads: the EPIC set (20 rows from every separator) and the KVLink set
    (the separators) built on the device equal the oracle's; the selective prefill with the
    EPIC set matches the oracle; separator rows left out keep zero K/V in the selective layers."""
    case = sep_case
    assert case.sep_rows
    seps = case.wl.sep_starts()
    dseps = torch.tensor(seps, dtype=torch.int32, device="cuda")
    for window in (20, case.wl.n_sep):
        got, k = kvb.window_select(dseps, window, case.n_ctx)
        assert np.array_equal(got.cpu().numpy(), blend.window_select(seps, window, case.n_ctx))
    epic = blend.window_select(seps, 20, case.n_ctx)
    ref = blend.selective_prefill(case.s, case.l64, case.x0, case.starts, case.nq, 0.0, case.cc["k"], case.cc["v"], 1,
                                  epic, case.w["final_norm"])
    ck, cv = case.new_cache()
    sel_dev, _ = kvb.window_select(dseps, 20, case.n_ctx)
    fh, sel, _ = kvb.selective_prefill(case.cfg, case.model, case.rope, case.kch, case.vch, ck, cv, case.dtoks,
                                       case.dstarts, case.n_ctx, case.nq, 0.0, 1, forced_sel=sel_dev, ws=case.ws)
    torch.cuda.synchronize()
    assert kvb.device_status(case.ws) == 0
    e = case.check_fh(fh.cpu(), ref["final_hidden"], "final hidden (EPIC selection)")
    for l in range(1, case.shape.n_layers):
        case.check_cache(ck[l].cpu(), ref["k"][l], f"k{l}", f"EPIC blended K layer {l}")
    # KVLink's set recomputes exactly the separators; any other set leaves them zero
    one = torch.tensor([case.sep_rows[-1] + case.wl.n_sep], dtype=torch.int32, device="cuda")
    ck, cv = case.new_cache()
    kvb.selective_prefill(case.cfg, case.model, case.rope, case.kch, case.vch, ck, cv, case.dtoks, case.dstarts,
                          case.n_ctx, case.nq, 0.0, 1, forced_sel=one, ws=case.ws)
    torch.cuda.synchronize()
    rows = torch.tensor(case.sep_rows, device="cuda")
    assert torch.all(ck[1:, rows] == 0) and torch.all(cv[1:, rows] == 0)
    assert torch.all(ck[0, rows].abs().sum(dim=(-1, -2)) > 0)          # layer 0 is recomputed in full
    print("EPIC", case.wl.name, len(epic), "rows", e)


def test_key_deviation_histogram_at_check_layer(kvb, case):
    """Distribution of squared key differences against the full prefill at the check layer:
    plain concatenation (r = 0) gives the deviations HKVD ranks (bit-equal to the ones it
    ranked); the r = 0.15 blend zeroes exactly its k rows, which are the k largest; EPIC
    zeroes its windows.  Counts are exact against the oracle's binning of the same values."""
    nc = case.n_ctx
    ckf, cvf = case.new_cache()
    kvb.full_prefill(case.cfg, case.model, case.rope, ckf, cvf, case.dtoks, n_out=case.nq, ws=case.ws)
    kd = case.shape.kv_dim

    def blend_cache(r, forced=None):
        ck, cv = case.new_cache()
        _, sel, _ = kvb.selective_prefill(case.cfg, case.model, case.rope, case.kch, case.vch, ck, cv, case.dtoks,
                                          case.dstarts, nc, case.nq, r, 1, forced_sel=forced, ws=case.ws)
        return ck, sel

    edges = torch.tensor([0.0] + [10.0 ** e for e in np.arange(-6, 3.01, 0.5)], dtype=torch.float32, device="cuda")
    ed = edges.cpu().numpy()

    def dev_hist(ck):
        dev = torch.empty(nc, dtype=torch.float32, device="cuda")
        h = kvb.key_deviation_histogram(ck[1, :nc].view(nc, kd), ckf[1, :nc].view(nc, kd), edges, dev_out=dev)
        torch.cuda.synchronize()
        d = dev.cpu().numpy()
        assert np.array_equal(h.cpu().numpy(), blend.deviation_histogram(d, ed))
        return d, h.cpu().numpy()

    ck0, _ = blend_cache(0.0)
    d0, h0 = dev_hist(ck0)
    ref = blend.hkvd_deviation(np64(ck0[1, :nc].cpu()), np64(ckf[1, :nc].cpu()))
    assert np.allclose(d0, ref, rtol=1e-5, atol=1e-30)
    k = blend.num_selected(case.wl.r, nc)
    cks, sel = blend_cache(case.wl.r)
    s = sel[:k].cpu().numpy().astype(np.int64)
    assert np.array_equal(s, blend.topk_select(d0, k))          # HKVD ranked these very values
    ds, hs = dev_hist(cks)
    want = d0.copy()
    want[s] = 0.0
    assert np.array_equal(ds, want)
    assert hs.sum() == nc
    if 0 < k < nc:
        assert ds.max() <= np.sort(d0)[-k - 1]                    # the k largest deviations are gone
    epic = blend.window_select(case.wl.sep_starts(), 20, nc)
    if len(epic):
        cke, _ = blend_cache(0.0, torch.from_numpy(epic.astype(np.int32)).cuda())
        de, _ = dev_hist(cke)
        want = d0.copy()
        want[epic] = 0.0
        assert np.array_equal(de, want)
    print("check-layer deviation", case.wl.name, "r=0", h0.tolist(), "hkvd", hs.tolist())
