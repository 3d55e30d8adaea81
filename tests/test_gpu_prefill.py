"""End-to-end parity of the whole path through the C ABI against the float64 oracle:
per-chunk caches, the dense prefill (the r = 1 comparator) and the selective
prefill, on the tiny model and the Llama-3.1-8B-shaped 2-layer model."""
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
        self.toks = synth.make_tokens(self.shape, self.N, 1)
        self.s = Shape.of(self.shape, act_bf16=True)
        self.s64 = Shape.of(self.shape)
        self.l64 = [{k: llama.as64(v) for k, v in l.items()} for l in w["layers"]]
        x0 = blend.embed_rows(w["embed"], self.toks.numpy())
        self.cc = blend.chunk_caches(self.s, self.l64, x0[: self.n_ctx], self.starts)
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
        self.vch = torch.from_numpy(self.cc["v"]).to(torch.bfloat16).to(torch.float16).cuda()
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


@pytest.fixture(scope="module", params=["tiny", "l8b_1layer"])
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
    for l in range(case.shape.n_layers):
        case.check_cache(ck[l].cpu(), case.full["k"][l], f"k{l}", f"layer {l} K")
        case.check_cache(cv[l].cpu(), case.full["v"][l], f"v{l}", f"layer {l} V")
    print("full prefill", case.wl.name, e, "vs float64", e64)


def test_chunk_caches_match_oracle(kvb, case):
    k, v = workload.chunk_caches(case.cfg, case.model, case.rope, case.dtoks[: case.n_ctx], case.starts, ws=case.ws)
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
