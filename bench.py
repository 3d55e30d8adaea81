#!/usr/bin/env python
"""Benchmark: time to first token of the selective-recompute prefill on one GB300.

A step is one call of kvb_selective_prefill on the headline workload: a 32-layer
Llama-3.1-8B-shaped bf16 model (random weights), 242 chunks x 512 tokens of
per-chunk KV caches resident in HBM plus a 128-token query (124,032 tokens),
recompute ratio r = 0.15.  The step covers merge + re-alignment of the chunk
caches, the dense layer 0, the HKVD selection and the 31 selective layers, up
to the query rows' final hidden state.  `value` is the mean TTFT in ms over the
timed steps (lower is better).  Next to it the line reports the library's own
dense r = 1.0 prefill of the same request, the end-to-end TTFT with the chunk
caches copied from pinned host memory inside the timed region, a live roofline
of the dominant kernel and the CPU oracle's time on a bounded sample.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]

With --gpus N under torchrun every rank serves its own replica of the request
(no data-path collective; the path has no exchange step).
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "TTFT (ms) at 124k tokens r=0.15 vs own r=1.0 prefill; attn TFLOP/s, % of bf16 peak"

# DRAM bytes (read + write) per launch of the selective-layer attention at this workload's
# size (18,713 rows over a 124,032-row cache), from one ncu capture of that launch; valid
# only for the kernel sources it was taken on (sha1 prefixes of attn.cu and common.cuh),
# otherwise reported as null.
ATTN_TRAFFIC = {"bytes": 0.878205e9 + 0.142111e9, "sha1": {"attn.cu": "0b224fed4482", "common.cuh": "ac1f1dda7832"}}


def attn_traffic():
    import hashlib
    d = os.path.join(ROOT, "paper_2609_09768_gb300", "csrc")
    for f, h in ATTN_TRAFFIC["sha1"].items():
        with open(os.path.join(d, f), "rb") as fh:
            if hashlib.sha1(fh.read()).hexdigest()[:12] != h:
                return None
    return ATTN_TRAFFIC["bytes"]


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=5)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--workload", default="l8b_124k")
    ap.add_argument("--model-config", default=None,
                    help="JSON model configuration (published-checkpoint layout) whose shape replaces the "
                         "workload's model; chunk layout, query and r stay the workload's")
    ap.add_argument("--r", type=float, default=None)
    ap.add_argument("--r1-steps", type=int, default=1, help="timed steps of the r = 1.0 comparator (0: skip)")
    ap.add_argument("--e2e-steps", type=int, default=2, help="timed end-to-end steps (0: skip)")
    ap.add_argument("--decode-steps", type=int, default=16, help="greedy decode steps timed after the prefill (0: skip)")
    ap.add_argument("--cpu-rows", type=int, default=128,
                    help="rows in the oracle's timed sample (the same for the cpu_baseline leg and the reference arm)")
    ap.add_argument("--no-cpu", action="store_true")
    ap.add_argument("--sweep", action="store_true",
                    help="64k-context sweep: r x chunk size, per-kernel times (prints one JSON line per point)")
    ap.add_argument("--kernel", default=None,
                    choices=["attn", "dense", "gemm", "realign", "decode_attn", "decode_step", "topk", "hkvd"],
                    help="time one kernel of the library on a seeded synthetic Llama-3.1-8B-shaped case "
                         "(for ncu captures); prints one JSON line")
    ap.add_argument("--m", type=int, default=18713, help="--kernel attn / gemm: query rows")
    ap.add_argument("--n-kv", type=int, default=124032, help="--kernel attn / dense / decode_*: cache rows")
    ap.add_argument("--n-ctx", type=int, default=123904, help="--kernel realign: context rows")
    ap.add_argument("--layers", type=int, default=2, help="--kernel realign / decode_step: layers")
    ap.add_argument("--which", default="qkv", choices=["qkv", "o", "gateup", "down"], help="--kernel gemm")
    ap.add_argument("--reps", type=int, default=2, help="--kernel: calls, the last one timed")
    ap.add_argument("--timed", type=int, default=1, help="--kernel: calls between the timing events (mean)")
    ap.add_argument("--selectors", action="store_true",
                    help="separator workload: TTFT and per-layer key-deviation histograms against the full "
                         "prefill for plain concatenation, HKVD, EPIC and KVLink selections (one JSON line each)")
    return ap.parse_args()


def max_over_ranks(value: float, world: int, device=None) -> float:
    """The slowest replica's step time: max over the ranks of the process group (the
    replicas share nothing else, so this is the only collective of the benchmark)."""
    if world <= 1:
        return value
    import torch
    import torch.distributed as dist
    t = torch.tensor([value], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def replica_tokens_per_s(n_tokens: int, world: int, ms: float) -> float:
    """Whole-job throughput of `world` replicas that each prefill `n_tokens` in `ms`."""
    return world * n_tokens / (ms * 1e-3)


def peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            p = json.load(f)
        return {"hbm_gbs": p["hbm_gbs"], "bf16": p["bf16_tflops"], "bf16_sustained": p["bf16_tflops_sustained"],
                "source": "measured"}
    except Exception:
        return {"hbm_gbs": 6800.0, "bf16": 1900.0, "bf16_sustained": 1700.0, "source": "fallback"}


class Clocks:
    """nvidia-smi sampling (200 ms) while the timed region runs."""
    Q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,clocks_event_reasons.hw_slowdown,"
         "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
         "clocks_event_reasons.sw_power_cap")

    def __init__(self, index: int):
        self.index, self.rows, self.proc = index, [], None

    def start(self):
        try:
            self.proc = subprocess.Popen(["nvidia-smi", f"--id={self.index}", f"--query-gpu={self.Q}",
                                          "--format=csv,noheader,nounits", "-lms", "200"],
                                         stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            threading.Thread(target=self._read, daemon=True).start()
        except Exception:
            self.proc = None

    def _read(self):
        for line in self.proc.stdout:
            self.rows.append([c.strip() for c in line.split(",")])

    def stop(self) -> dict:
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        time.sleep(0.1)
        sm = [float(r[1]) for r in self.rows if len(r) >= 9 and r[1].replace(".", "").isdigit()]
        mx = [float(r[2]) for r in self.rows if len(r) >= 9 and r[2].replace(".", "").isdigit()]
        reasons = set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for r in self.rows:
            if len(r) >= 9:
                for n, v in zip(names, r[5:9]):
                    if v.lower() == "active":
                        reasons.add(n)
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": max(mx) if mx else None,
                "reasons": sorted(reasons), "samples": len(sm)}


# ------------------------------------------------------------------------------------ oracle (CPU) leg

ORACLE_BLOCK = 256     # rows per block of the oracle's attention (oracle.llama.attention_rows)


def oracle_attention_work(hi, lo=None, block: int = ORACLE_BLOCK) -> float:
    """The oracle's attention work for a set of rows, in (row, key) pairs: it takes the rows in
    blocks of `block` consecutive rows and scores each block against the union of its rows' key
    ranges [min lo, max hi], so its cost is the sum over blocks of rows x keys in that union."""
    import numpy as np
    hi = np.asarray(hi, dtype=np.int64)
    lo = np.zeros_like(hi) if lo is None else np.asarray(lo, dtype=np.int64)
    w = 0.0
    for b0 in range(0, len(hi), block):
        h, l = hi[b0:b0 + block], lo[b0:b0 + block]
        w += float(len(h)) * float(h.max() - l.min() + 1)
    return w


class OracleSample:
    """A bounded sample of the workload for the CPU oracle: one selective decoder layer
    over `n_rows` rows spread uniformly over the context, attending a float64 cache of
    the full request length.  Inputs are drawn once; run() times the oracle's steps in two
    parts: the per-row part (RMSNorm, q/k/v projection and RoPE, O-projection, RMSNorm and
    SwiGLU MLP), and the attention, whose cost per row depends on the key range the
    oracle scores it against."""

    def __init__(self, wl, n_rows: int, seed: int = 0):
        import numpy as np
        from oracle import llama
        from oracle.llama import Shape
        from paper_2609_09768_gb300 import synth
        shape = wl.shape
        self.s = Shape.of(shape, act_bf16=True)
        self.lw = {k: llama.as64(v) for k, v in synth.make_layer_weights(shape, 1, seed).items()}
        N = wl.n_total
        rng = np.random.default_rng(seed)
        self.kc = rng.standard_normal((N, shape.n_kv_heads, shape.head_dim))
        self.vc = rng.standard_normal((N, shape.n_kv_heads, shape.head_dim))
        self.rows = np.sort(rng.choice(wl.n_ctx, size=n_rows, replace=False))
        self.x = rng.standard_normal((n_rows, shape.hidden))
        self.n_rows = n_rows
        self.work = oracle_attention_work(self.rows)

    def run(self):
        """(seconds of the per-row part, seconds of the attention) for one oracle layer."""
        from oracle import llama
        t0 = time.perf_counter()
        q, k, v = llama.qkv_rows(self.s, self.lw, self.x, self.rows)
        t1 = time.perf_counter()
        self.kc[self.rows] = k
        self.vc[self.rows] = v
        a = llama.act(self.s, llama.attention_rows(self.s, q, self.kc, self.vc, self.rows))
        t2 = time.perf_counter()
        llama.attn_out_mlp(self.s, self.lw, self.x, a.reshape(a.shape[0], -1))
        t3 = time.perf_counter()
        return (t1 - t0) + (t3 - t2), t2 - t1


def sample_rows(args, wl, k: int) -> int:
    """Rows in the oracle's timed sample: --cpu-rows within [16, 256], and no more than the
    rows the method recomputes (k + n_query) or the context holds."""
    return max(1, min(max(16, min(256, args.cpu_rows)), k + wl.n_query, wl.n_ctx))


def cpu_cores() -> int:
    try:
        return len(os.sched_getaffinity(0))
    except Exception:
        return os.cpu_count() or 1


def oracle_ttft_ms(wl, smp: "OracleSample", t_rows: float, t_attn: float, k: int, sel=None) -> float:
    """The oracle's prefill time from one timed sample layer:
         per-row part:  t_rows / sample rows  x  (N + (L - 1) m) row-layers
         attention:     t_attn / sample work  x  (work of layer 0 + (L - 1) x work of a selective layer)
    with the work of oracle_attention_work: layer 0 scores all N rows causally, a selective
    layer the m = k + n_query recomputed rows (the selected context rows `sel`, or k rows
    spread uniformly when they are not known, then the query rows) over [0, own row]."""
    import numpy as np
    N, L, nq = wl.n_total, wl.shape.n_layers, wl.n_query
    m = k + nq
    if sel is None:
        sel = np.linspace(0, wl.n_ctx - 1, num=k).round().astype(np.int64) if k else np.zeros(0, np.int64)
    rows_sel = np.concatenate([np.sort(np.asarray(sel, dtype=np.int64)), np.arange(wl.n_ctx, N)])
    work = oracle_attention_work(np.arange(N)) + (L - 1) * oracle_attention_work(rows_sel)
    return (t_rows / smp.n_rows * (N + (L - 1) * m) + t_attn / smp.work * work) * 1e3


def run_reference(args, wl, rank: int, world: int) -> None:
    """The reference arm: the CPU oracle as it stands, on the host cores."""
    if rank != 0:
        return
    from oracle import blend
    r = wl.r if args.r is None else args.r
    k = blend.num_selected(r, wl.n_ctx)
    rows = sample_rows(args, wl, k)
    smp = OracleSample(wl, rows)
    for _ in range(args.warmup):
        smp.run()
    vals = []
    for _ in range(args.steps):
        vals.append(oracle_ttft_ms(wl, smp, *smp.run(), k))
    v = statistics.mean(vals)
    sample = (f"oracle selective layer on {rows} of {k + wl.n_query} recomputed rows (uniform over the context) "
              f"attending a {wl.n_total}-row cache, per step; per-row part scaled by (N + (L-1) m) row-layers, "
              f"attention by the oracle's (row, key) block work of the whole prefill (extrapolated)")
    print(json.dumps({
        "impl": "reference", "metric": METRIC, "value": round(v, 3), "unit": "ms", "n_gpus": args.gpus,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(v, 3), "higher_is_better": False,
        "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": {"workload": wl.name, "n_ctx": wl.n_ctx, "n_query": wl.n_query, "r": r, "k": k},
        "cpu_baseline": {"value": round(v, 3), "unit": "ms", "cores": cpu_cores(), "kind": "oracle", "sample": sample},
        "e2e": {"value": round(v, 3), "unit": "ms", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }))


# ------------------------------------------------------------------------------------ our arm

def run_ours(args, wl, rank: int, world: int) -> None:
    import numpy as np
    import torch
    import torch.distributed as dist
    from paper_2609_09768_gb300 import build, synth, workload
    from paper_2609_09768_gb300 import kvblend as kvb

    build.build()
    dev = torch.device("cuda", torch.cuda.current_device())
    shape = wl.shape
    r = wl.r if args.r is None else args.r
    cfg = kvb.config(shape)
    N, n_ctx, nq, L = wl.n_total, wl.n_ctx, wl.n_query, shape.n_layers
    Hq, Hkv, D, H, F = shape.n_q_heads, shape.n_kv_heads, shape.head_dim, shape.hidden, shape.mlp_dim
    pk = peaks()

    weights = workload.device_model(shape, seed=0, device=dev, draw_on_device=True)
    model = kvb.Model(weights)
    toks = synth.make_tokens(shape, N, 1).to(dev)
    n_dec = max(args.decode_steps, 0)
    cap = N + n_dec + 1                      # cache rows: the prompt, then the decoded tokens
    rope = kvb.RopeTable(cfg, cap, dev)
    ws = kvb.workspace(cfg, N, dev)
    starts = wl.chunk_starts()
    dstarts = torch.tensor(starts, dtype=torch.int32, device=dev)
    kch, vch = workload.chunk_caches(cfg, model, rope, toks[:n_ctx], starts, ws=ws)
    ck = torch.empty(L, cap, Hkv, D, dtype=torch.bfloat16, device=dev)
    cv = torch.empty(L, cap, Hkv, D, dtype=torch.float16, device=dev)
    fh = torch.empty(nq, H, dtype=torch.float32, device=dev)
    sel = torch.empty(n_ctx, dtype=torch.int32, device=dev)
    lm = synth.make_lm_head(shape, 0, dev)
    tok = torch.empty(1, dtype=torch.int32, device=dev)
    lm_ws = torch.zeros(512, dtype=torch.uint8, device=dev)
    lm_ev = []
    torch.cuda.synchronize()

    def first_token():
        """Logits of the last query row over the vocabulary and their argmax."""
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record()
        kvb.lm_head_argmax(cfg, lm, fh[nq - 1:], tokens=tok, ws=lm_ws)
        b.record()
        lm_ev.append((a, b))

    def step(rr=r, timings=True):
        t = kvb.selective_prefill(cfg, model, rope, kch, vch, ck, cv, toks, dstarts, n_ctx, nq, rr, 1,
                                  final_hidden=fh, sel_out=sel, ws=ws, timings=timings)[2]
        first_token()
        return t

    def barrier():
        if world > 1:
            dist.barrier()

    for _ in range(max(args.warmup, 3)):
        step()
    torch.cuda.synchronize()
    clocks = Clocks(torch.cuda.current_device())
    clocks.start()
    barrier()
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    lm_ev.clear()
    e0.record()
    tims = [step() for _ in range(args.steps)]
    e1.record()
    torch.cuda.synchronize()
    barrier()
    clk = clocks.stop()
    ms = e0.elapsed_time(e1) / args.steps
    ms = max_over_ranks(ms, world, dev)
    assert kvb.device_status(ws) == 0, "device wait timed out"

    # algorithmic work of the step (from the chosen rows, read back after the timed region)
    k = int(tims[-1]["n_selected"])
    m = k + nq
    rows = np.concatenate([sel[:k].cpu().numpy().astype(np.int64), np.arange(n_ctx, N)])
    attn_sel_flop = 4.0 * Hq * D * float(np.sum(rows + 1))          # per selective layer
    attn_dense_flop = 4.0 * Hq * D * N * (N + 1) / 2.0               # layer 0
    gemm_row_flop = 2.0 * H * (shape.qkv_dim + shape.q_dim) + 2.0 * 3 * H * F
    gemm_flop = gemm_row_flop * (N + (L - 1) * m) + 2.0 * n_ctx * H * shape.kv_dim
    total_flop = attn_dense_flop + (L - 1) * attn_sel_flop + gemm_flop

    def avg(key):
        return statistics.mean(t[key] for t in tims)

    kern = {
        "attn_selective": {"ms": avg("attn_sel_ms"), "launches": int(tims[-1]["n_attn_sel"]),
                           "flop": attn_sel_flop * (L - 1)},
        "attn_dense": {"ms": avg("attn_dense_ms"), "launches": int(tims[-1]["n_attn_dense"]), "flop": attn_dense_flop},
        "gemm": {"ms": avg("gemm_ms"), "launches": int(tims[-1]["n_gemm"]), "flop": gemm_flop},
    }
    lm_ms = statistics.mean(a.elapsed_time(b) for a, b in lm_ev[:args.steps])
    lm_bytes = float(shape.vocab * H * 2)
    lm_head = {"ms": round(lm_ms, 4), "launches": 2, "bytes": lm_bytes,
               "gbs": round(lm_bytes / (lm_ms * 1e-3) / 1e9, 1),
               "frac_of_hbm": round(lm_bytes / (lm_ms * 1e-3) / 1e9 / pk["hbm_gbs"], 4)}
    for v in kern.values():
        v["tflops"] = v["flop"] / (v["ms"] * 1e-3) / 1e12 if v["ms"] > 0 else None
        v["frac_of_sustained_peak"] = (v["tflops"] / pk["bf16_sustained"]) if v["tflops"] else None
    dom_name = max(kern, key=lambda n: kern[n]["ms"])
    dom = kern[dom_name]
    per_launch_ms = dom["ms"] / max(dom["launches"], 1)
    per_launch_flop = dom["flop"] / max(dom["launches"], 1)
    achieved = per_launch_flop / (per_launch_ms * 1e-3) / 1e12
    roofline = {"kernel": dom_name, "bound": "tensor", "achieved": round(achieved, 2),
                "peak": pk["bf16_sustained"], "unit": "TFLOP/s", "frac": round(achieved / pk["bf16_sustained"], 4),
                "traffic": attn_traffic() if dom_name == "attn_selective" else None,
                "peak_source": f"{pk['source']} bf16 sustained",
                "flop_per_launch": per_launch_flop, "ms_per_launch": round(per_launch_ms, 4)}

    # the library's own dense r = 1.0 prefill of the same request
    r1 = None
    if args.r1_steps > 0:
        step(1.0)
        torch.cuda.synchronize()
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record()
        r1t = [step(1.0) for _ in range(args.r1_steps)]
        b.record()
        torch.cuda.synchronize()
        r1_ms = a.elapsed_time(b) / args.r1_steps
        r1 = {"ttft_ms": round(r1_ms, 3), "attn_dense_ms": round(statistics.mean(t["attn_dense_ms"] for t in r1t), 3),
              "gemm_ms": round(statistics.mean(t["gemm_ms"] for t in r1t), 3),
              "attn_tflops": round(4.0 * Hq * D * N * (N + 1) / 2.0 * L /
                                   (statistics.mean(t["attn_dense_ms"] for t in r1t) * 1e-3) / 1e12, 2)}

    # end to end through the public API: chunk caches in pinned host memory, ingested layer by
    # layer under the compute (kvb_selective_prefill_host), tokens copied in and the final
    # hidden copied back, all inside the timed region
    e2e = None
    if args.e2e_steps > 0:
        hk = torch.empty(kch.shape, dtype=kch.dtype, pin_memory=True)
        hv = torch.empty(vch.shape, dtype=vch.dtype, pin_memory=True)
        ht = torch.empty(toks.shape, dtype=toks.dtype, pin_memory=True)
        hf = torch.empty(fh.shape, dtype=fh.dtype, pin_memory=True)
        htok = torch.empty(tok.shape, dtype=tok.dtype, pin_memory=True)
        hk.copy_(kch); hv.copy_(vch); ht.copy_(toks)
        torch.cuda.synchronize()
        # the bare host->device copy of the same caches before any e2e step, for reference
        kd = torch.empty_like(kch)
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record(); kd.copy_(hk, non_blocking=True); b.record()
        torch.cuda.synchronize()
        h2d_k_ms = a.elapsed_time(b)
        del kd
        td = torch.empty_like(toks)
        wsp = torch.zeros(kvb.workspace_size_pipelined(cfg, N, n_ctx), dtype=torch.uint8, device=dev)
        cs = torch.cuda.Stream(device=dev)
        torch.cuda.synchronize()

        e2e_t = []

        def e2e_step(timings=False):
            td.copy_(ht, non_blocking=True)
            t = kvb.selective_prefill_host(cfg, model, rope, hk, hv, ck, cv, td, dstarts, n_ctx, nq, r, 1,
                                           copy_stream=cs, final_hidden=fh, sel_out=sel, ws=wsp,
                                           timings=timings)[2]
            if t:
                e2e_t.append(t)
            kvb.lm_head_argmax(cfg, lm, fh[nq - 1:], tokens=tok, ws=lm_ws)
            hf.copy_(fh, non_blocking=True)
            htok.copy_(tok, non_blocking=True)

        e2e_step(timings=True)           # untimed: its stage times show where the ingest waits
        torch.cuda.synchronize()
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record()
        for _ in range(args.e2e_steps):
            e2e_step()
        b.record()
        torch.cuda.synchronize()
        e2e_ms = a.elapsed_time(b) / args.e2e_steps
        # the bare host->device copy of the same caches, for reference
        kd = torch.empty_like(kch)
        a.record(); kd.copy_(hk, non_blocking=True); kd.copy_(hv, non_blocking=True); b.record()
        torch.cuda.synchronize()
        h2d_ms = a.elapsed_time(b)
        h2d = hk.numel() * 2 + hv.numel() * 2 + ht.numel() * 4
        e2e = {"value": round(e2e_ms, 3), "unit": "ms", "h2d_bytes_per_step": int(h2d),
               "d2h_bytes_per_step": int(hf.numel() * 4 + htok.numel() * 4), "path": "kvb_selective_prefill_host (layer-wise ingest)",
               "bare_h2d_ms": round(h2d_ms, 2), "bare_h2d_gbs": round(h2d / (h2d_ms * 1e-3) / 1e9, 1),
               "bare_h2d_k_before_gbs": round(hk.numel() * 2 / (h2d_k_ms * 1e-3) / 1e9, 1),
               "stages_ms_untimed_step": {k_: round(v_, 3) for k_, v_ in e2e_t[0].items() if k_.endswith("_ms")}
               if e2e_t else None}
        del hk, hv, kd, wsp

    # greedy decode after the prefill (first token already decoded by the step): n_dec steps
    # through kvb_decode_step, position and tokens on the device; eager launches, then the
    # same step replayed as a CUDA graph
    decode = None
    if n_dec > 0:
        step()                                             # fresh prefill cache + first token
        tokens = torch.zeros(cap + 1, dtype=torch.int32, device=dev)
        tokens[:N] = toks
        tokens[N:N + 1] = tok
        pos = torch.tensor([N], dtype=torch.int32, device=dev)
        dws = kvb.decode_workspace(cfg, cap, dev)
        kvb.decode_step(cfg, model, rope, ck, cv, lm, tokens, pos, cap, ws=dws)   # warm-up (position N)
        torch.cuda.synchronize()
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record()
        for _ in range(n_dec - 1):
            kvb.decode_step(cfg, model, rope, ck, cv, lm, tokens, pos, cap, ws=dws)
        b.record()
        torch.cuda.synchronize()
        # embed; per layer 4 GEMVs (RMSNorm, RoPE and the K/V append fused into them),
        # attention + combine; final norm, lm_head + argmax, position/token update
        launches = 1 + 6 * L + 1 + 2 + 1
        dec_ms = a.elapsed_time(b) / max(n_dec - 1, 1)
        assert kvb.device_status(dws) == 0 and int(pos.item()) == N + n_dec
        p_mid = N + n_dec // 2
        w_bytes = float(L * 2 * (shape.qkv_dim * H + H * shape.q_dim + 3 * H * F) + shape.vocab * H * 2)
        kv_bytes = float(L * (p_mid + 1) * shape.kv_dim * 2 * 2)
        graph_ms = None
        try:
            pos.fill_(N)
            g = torch.cuda.CUDAGraph()
            cs = torch.cuda.Stream(device=dev)
            cs.wait_stream(torch.cuda.current_stream())
            with torch.cuda.stream(cs):
                with torch.cuda.graph(g, stream=cs):
                    kvb.decode_step(cfg, model, rope, ck, cv, lm, tokens, pos, cap, ws=dws)
            torch.cuda.current_stream().wait_stream(cs)
            pos.fill_(N)
            g.replay()
            torch.cuda.synchronize()
            a.record()
            for _ in range(n_dec - 1):
                g.replay()
            b.record()
            torch.cuda.synchronize()
            assert kvb.device_status(dws) == 0 and int(pos.item()) == N + n_dec
            graph_ms = a.elapsed_time(b) / max(n_dec - 1, 1)
        except Exception as exc:                          # report the eager number alone
            print(f"decode graph capture skipped: {exc}", file=sys.stderr)
        best = min(dec_ms, graph_ms) if graph_ms else dec_ms
        decode = {"tokens": n_dec, "positions": [N, N + n_dec], "ms_per_token": round(dec_ms, 4),
                  "graph_ms_per_token": round(graph_ms, 4) if graph_ms else None,
                  "bytes_per_token": w_bytes + kv_bytes, "weights_bytes": w_bytes, "kv_bytes": kv_bytes,
                  "gbs": round((w_bytes + kv_bytes) / (best * 1e-3) / 1e9, 1),
                  "frac_of_hbm": round((w_bytes + kv_bytes) / (best * 1e-3) / 1e9 / pk["hbm_gbs"], 4),
                  "launches_per_token": int(launches)}

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu:
        n = sample_rows(args, wl, k)
        smp = OracleSample(wl, n)
        t_rows, t_attn = smp.run()
        sel_np = sel[:k].cpu().numpy() if k > 0 else None
        cpu = {"value": round(oracle_ttft_ms(wl, smp, t_rows, t_attn, k, sel_np), 1), "unit": "ms",
               "cores": cpu_cores(), "kind": "oracle",
               "sample": (f"oracle selective layer on {n} of {m} recomputed rows (uniform over the context) "
                          f"attending a {N}-row float64 cache: {t_rows:.1f} s per-row part + {t_attn:.1f} s "
                          f"attention; per-row part scaled by (N + (L-1) m) row-layers, attention by the oracle's "
                          f"(row, key) block work of the whole prefill with the selection this run made "
                          f"(extrapolated)")}

    if rank == 0:
        stages = {k_: round(avg(k_), 3) for k_ in ("realign_ms", "dense_ms", "select_ms", "selective_ms", "final_ms")}
        kdict = {n: {kk: (round(vv, 4) if isinstance(vv, float) else vv) for kk, vv in v.items()}
                 for n, v in kern.items()}
        out = {
            "metric": METRIC, "value": round(ms, 3), "unit": "ms", "n_gpus": world, "steps": args.steps,
            "warmup": max(args.warmup, 3), "ms_per_step": round(ms, 3), "higher_is_better": False,
            "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
            "data": "synthetic (random N(0,0.02) weights, uniform token ids, per-chunk caches from isolated prefill)",
            "config": {"workload": wl.name, "n_layers": L, "n_chunks": wl.n_chunks, "chunk_len": wl.chunk_len,
                       "n_ctx": n_ctx, "n_query": nq, "n_tokens": N, "r": r, "k": k, "check_layer": 1,
                       "l2": "inputs larger than L2 (16.3 GB of chunk KV caches read per step)",
                       "parallelism": f"replicas x{world}"},
            "tokens_per_s": round(replica_tokens_per_s(N, world, ms), 1),
            "r1_dense": r1,
            "ttft_reduction_vs_r1": (round(1.0 - ms / r1["ttft_ms"], 4) if r1 else None),
            "algorithmic_tflops": round(total_flop / (ms * 1e-3) / 1e12, 2),
            "stages_ms": stages, "kernels": dict(kdict, first_token_lm_head=lm_head),
            "first_token": int(tok.item()),
            "roofline": roofline, "cpu_baseline": cpu, "e2e": e2e, "decode": decode,
            "gpu_launches": int(sum(t["n_launches"] for t in tims)) + 2 * args.steps,
            "clocks": clk,
        }
        print(json.dumps(out))


def run_sweep(args) -> None:
    """The 64k-context sweep: 32 layers, chunk sizes 256/512/1024/2048 (count adjusted to fill
    65,536 context tokens) + 128 query tokens, r in {0.05, 0.10, 0.15, 0.25, 0.5, 1.0}; per point
    the TTFT and the per-kernel times of re-align, HKVD (deviation + top-k), row GEMMs and
    sparse-query attention."""
    import torch
    from paper_2609_09768_gb300 import build, synth, workload
    from paper_2609_09768_gb300 import kvblend as kvb

    build.build()
    dev = torch.device("cuda", torch.cuda.current_device())
    shape = synth.LLAMA8B
    cfg = kvb.config(shape)
    nq, n_ctx = 128, 65536
    N, L = n_ctx + nq, shape.n_layers
    weights = workload.device_model(shape, seed=0, device=dev, draw_on_device=True)
    model = kvb.Model(weights)
    toks = synth.make_tokens(shape, N, 1).to(dev)
    rope = kvb.RopeTable(cfg, N, dev)
    ws = kvb.workspace(cfg, N, dev)
    ck = torch.empty(L, N, shape.n_kv_heads, shape.head_dim, dtype=torch.bfloat16, device=dev)
    cv = torch.empty(L, N, shape.n_kv_heads, shape.head_dim, dtype=torch.float16, device=dev)
    fh = torch.empty(nq, shape.hidden, dtype=torch.float32, device=dev)
    sel = torch.empty(n_ctx, dtype=torch.int32, device=dev)
    for chunk in (256, 512, 1024, 2048):
        starts = synth.chunk_starts_equal(n_ctx // chunk, chunk)
        dstarts = torch.tensor(starts, dtype=torch.int32, device=dev)
        kch, vch = workload.chunk_caches(cfg, model, rope, toks[:n_ctx], starts, ws=ws)
        for r in (0.05, 0.10, 0.15, 0.25, 0.5, 1.0):
            run = lambda: kvb.selective_prefill(cfg, model, rope, kch, vch, ck, cv, toks, dstarts, n_ctx, nq, r, 1,
                                                final_hidden=fh, sel_out=sel, ws=ws, timings=True)[2]
            for _ in range(max(1, args.warmup - 1)):
                run()
            reps = [run() for _ in range(max(1, min(args.steps, 3)))]
            avg = {k: statistics.mean(t[k] for t in reps) for k in reps[0]}
            print(json.dumps({"sweep": "l8b-32L-64k", "chunk": chunk, "n_chunks": n_ctx // chunk, "r": r,
                              "k": int(avg["n_selected"]), "ttft_ms": round(avg["total_ms"], 2),
                              "realign_ms": round(avg["realign_ms"], 3), "hkvd_ms": round(avg["hkvd_ms"], 3),
                              "gemm_ms": round(avg["gemm_ms"], 2),
                              "attn_sel_ms": round(avg["attn_sel_ms"], 2),
                              "attn_dense_ms": round(avg["attn_dense_ms"], 2)}), flush=True)
        del kch, vch
    assert kvb.device_status(ws) == 0


def run_selectors(args) -> None:
    """Selections compared on a request with two zero-KV separator tokens between documents:
    plain concatenation (r = 0), CacheBlend's HKVD at r, EPIC (20 rows from every separator)
    and KVLink's rows (the separators).  Per selection: TTFT and, for every layer, the
    histogram of per-token squared key differences of the blended cache against the
    full prefill's cache (the quantity of the paper's deviation figures)."""
    import numpy as np
    import torch
    from paper_2609_09768_gb300 import build, synth, workload
    from paper_2609_09768_gb300 import kvblend as kvb

    build.build()
    wl = synth.WORKLOADS[args.workload if args.workload.endswith("_sep") else "l8b_124k_sep"]
    dev = torch.device("cuda", torch.cuda.current_device())
    shape = wl.shape
    cfg = kvb.config(shape)
    N, n_ctx, nq, L = wl.n_total, wl.n_ctx, wl.n_query, shape.n_layers
    r = wl.r if args.r is None else args.r
    model = kvb.Model(workload.device_model(shape, seed=0, device=dev, draw_on_device=True))
    toks = wl.tokens(1, dev)
    rope = kvb.RopeTable(cfg, N, dev)
    ws = kvb.workspace(cfg, N, dev)
    starts = wl.chunk_starts()
    dstarts = torch.tensor(starts, dtype=torch.int32, device=dev)
    kch, vch = workload.chunk_caches(cfg, model, rope, toks[:n_ctx], starts, ws=ws, zero_rows=wl.sep_rows())
    shp = (L, N, shape.n_kv_heads, shape.head_dim)
    ckf = torch.empty(shp, dtype=torch.bfloat16, device=dev)
    cvf = torch.empty(shp, dtype=torch.float16, device=dev)
    ck = torch.empty(shp, dtype=torch.bfloat16, device=dev)
    cv = torch.empty(shp, dtype=torch.float16, device=dev)
    fh = torch.empty(nq, shape.hidden, dtype=torch.float32, device=dev)
    sel = torch.empty(n_ctx, dtype=torch.int32, device=dev)
    seps = torch.tensor(wl.sep_starts(), dtype=torch.int32, device=dev)
    epic, k_epic = kvb.window_select(seps, 20, n_ctx)
    kvlink, k_kvlink = kvb.window_select(seps, wl.n_sep, n_ctx)
    edges_l = [0.0] + [float(10.0 ** e) for e in np.arange(-4, 3.01, 0.5)]
    edges = torch.tensor(edges_l, dtype=torch.float32, device=dev)
    kd = shape.kv_dim

    def run(rr, forced=None, cache=(ck, cv)):
        return kvb.selective_prefill(cfg, model, rope, kch, vch, cache[0], cache[1], toks, dstarts, n_ctx, nq, rr, 1,
                                     forced_sel=forced, final_hidden=fh, sel_out=sel, ws=ws, timings=True)[2]

    def timed(fn, reps):
        fn()
        torch.cuda.synchronize()
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record()
        for _ in range(reps):
            t = fn()
        b.record()
        torch.cuda.synchronize()
        return a.elapsed_time(b) / reps, t

    full_ms, _ = timed(lambda: run(1.0, cache=(ckf, cvf)), 1)
    print(json.dumps({"selectors": wl.name, "selection": "full prefill (r = 1)", "k": n_ctx,
                      "ttft_ms": round(full_ms, 2)}), flush=True)
    for name, rr, forced in (("concatenation (r = 0)", 0.0, None), (f"CacheBlend HKVD r = {r}", r, None),
                             ("EPIC: 20 rows from every separator", 0.0, epic),
                             ("KVLink rows: the separators", 0.0, kvlink)):
        ms, t = timed(lambda: run(rr, forced), max(1, min(args.steps, 3)))
        hist = {}
        mean_dev = []
        d = torch.empty(n_ctx, dtype=torch.float32, device=dev)
        for l in range(1, L):
            h = kvb.key_deviation_histogram(ck[l, :n_ctx].view(n_ctx, kd), ckf[l, :n_ctx].view(n_ctx, kd), edges,
                                            dev_out=d)
            mean_dev.append(round(float(d.mean()), 5))
            if l in (1, 2, L // 2, L - 1):
                hist[l] = h.cpu().tolist()
        print(json.dumps({"selectors": wl.name, "selection": name, "k": int(t["n_selected"]),
                          "ttft_ms": round(ms, 2), "ttft_vs_full": round(ms / full_ms, 4),
                          "hist_edges": edges_l, "hist_by_layer": hist, "mean_dev_by_layer": mean_dev}), flush=True)
    assert kvb.device_status(ws) == 0


def run_kernel(args) -> None:
    """One kernel on a seeded synthetic case of the Llama-3.1-8B layer shape (H 4096, 32 q / 8
    kv heads, D 128, F 14336).  attn: --m query rows drawn uniformly over the cache (as the
    HKVD choice at r = m / n_kv would spread them) plus the last row; dense: causal over all
    --n-kv rows; gemm: the QKV GEMM or the back half of a layer on --m rows; realign: --layers
    layers of --n-ctx rows of chunk caches in 512-row chunks; decode_attn / decode_step: one
    decode row at position --n-kv - 1.  Prints the CUDA-event time of the last call (or the
    mean of --timed calls) and its algorithmic throughput."""
    import torch
    from paper_2609_09768_gb300 import build, synth
    from paper_2609_09768_gb300 import kvblend as kvb
    build.build()
    shape = synth.LLAMA8B
    cfg = kvb.config(shape)
    dev = torch.device("cuda")
    Hq, Hkv, D, H, F = shape.n_q_heads, shape.n_kv_heads, shape.head_dim, shape.hidden, shape.mlp_dim
    g = torch.Generator(device=dev)
    g.manual_seed(0)
    ws = torch.zeros(256, dtype=torch.uint8, device=dev)
    out, flop = {}, None
    if args.kernel in ("attn", "dense"):
        n_kv = args.n_kv
        if args.kernel == "dense":
            rows = torch.arange(n_kv, device=dev, dtype=torch.int32)
        else:
            perm = torch.randperm(n_kv - 1, generator=g, device=dev)[: args.m - 1]
            rows = torch.cat([torch.sort(perm).values, torch.tensor([n_kv - 1], device=dev)]).to(torch.int32)
        m = rows.numel()
        q = torch.randn(m, Hq, D, generator=g, device=dev).to(torch.bfloat16)
        kc = torch.randn(n_kv, Hkv, D, generator=g, device=dev).to(torch.bfloat16)
        vc = torch.randn(n_kv, Hkv, D, generator=g, device=dev).to(torch.bfloat16).to(torch.float16)
        o = torch.empty(m, Hq * D, dtype=torch.bfloat16, device=dev)
        fn = lambda: kvb.sparse_query_attn(cfg, q, rows, None, kc, vc, o, ws)
        flop = 4.0 * Hq * D * float((rows.to(torch.float64) + 1).sum())
        out.update(m=m, n_kv=n_kv)
    elif args.kernel == "gemm":
        m = args.m
        lws = kvb.layer_struct(synth.make_layer_weights(shape, 0, 0, dev))
        wsl = kvb.workspace(cfg, m, dev)
        if args.which == "qkv":
            x = torch.randn(m, H, generator=g, device=dev)
            pos = torch.arange(m, dtype=torch.int32, device=dev)
            rope = kvb.RopeTable(cfg, m, dev)
            qo = torch.empty(m, Hq * D, dtype=torch.bfloat16, device=dev)
            ko = torch.empty(m, Hkv * D, dtype=torch.bfloat16, device=dev)
            vo = torch.empty(m, Hkv * D, dtype=torch.float16, device=dev)
            fn = lambda: kvb.gather_rmsnorm_qkv(cfg, lws, rope, x, None, pos, m, qo, ko, vo, None, wsl)
            flop = 2.0 * m * H * shape.qkv_dim
        else:
            attn = torch.randn(m, Hq * D, generator=g, device=dev).to(torch.bfloat16)
            x = torch.randn(m, H, generator=g, device=dev)
            fn = lambda: kvb.mlp_rows(cfg, lws, attn, x, wsl)
            flop = 2.0 * m * H * (Hq * D + 3 * F)
        out.update(m=m, which=("o+gateup+down (mlp_rows)" if args.which != "qkv" else "qkv"))
    elif args.kernel == "decode_attn":
        n_kv = args.n_kv
        q = torch.randn(Hq, D, generator=g, device=dev).to(torch.bfloat16)
        kc = torch.randn(n_kv, Hkv, D, generator=g, device=dev).to(torch.bfloat16)
        vc = torch.randn(n_kv, Hkv, D, generator=g, device=dev).to(torch.bfloat16).to(torch.float16)
        pos = torch.tensor([n_kv - 1], dtype=torch.int32, device=dev)
        ws = kvb.decode_workspace(cfg, n_kv, dev)
        o = torch.empty(Hq, D, dtype=torch.bfloat16, device=dev)
        fn = lambda: kvb.decode_attention(cfg, q, kc, vc, pos, n_kv, out=o, ws=ws)
        out.update(bytes=float(n_kv) * Hkv * D * 2 * 2, n_kv=n_kv)
    elif args.kernel == "decode_step":
        # a decode step of a --layers-layer model at position n_kv - 1
        shp = shape.with_layers(args.layers)
        cfgl = kvb.config(shp)
        model = kvb.Model(synth.make_model(shp, 0, dev))
        lm = synth.make_lm_head(shp, 0, dev)
        n_kv = args.n_kv
        rope = kvb.RopeTable(cfgl, n_kv, dev)
        kc = torch.randn(args.layers, n_kv, Hkv, D, generator=g, device=dev).to(torch.bfloat16)
        vc = torch.randn(args.layers, n_kv, Hkv, D, generator=g, device=dev).to(torch.bfloat16).to(torch.float16)
        tokens = torch.zeros(n_kv + 1, dtype=torch.int32, device=dev)
        pos = torch.tensor([n_kv - 1], dtype=torch.int32, device=dev)
        ws = kvb.decode_workspace(cfgl, n_kv, dev)

        def fn():
            pos.fill_(n_kv - 1)
            kvb.decode_step(cfgl, model, rope, kc, vc, lm, tokens, pos, n_kv, ws=ws)
        wb = args.layers * 2.0 * (shp.qkv_dim * H + H * shp.q_dim + 3 * H * F) + shp.vocab * H * 2.0
        out.update(bytes=wb + args.layers * float(n_kv) * Hkv * D * 4, layers=args.layers, n_kv=n_kv)
    elif args.kernel in ("topk", "hkvd"):
        # HKVD selection over --n-ctx context rows at r = 0.15: the deviation over the 1,024
        # key entries of a row, then the top-k (topk: 8 entries per row, so that the time is
        # the top-k's)
        n_ctx = args.n_ctx
        kvd = 8 if args.kernel == "topk" else Hkv * D
        kf = torch.randn(n_ctx, kvd, generator=g, device=dev).to(torch.bfloat16)
        kc = torch.randn(n_ctx, kvd, generator=g, device=dev).to(torch.bfloat16)
        kk = int(0.15 * n_ctx)
        sel = torch.empty(kk, dtype=torch.int32, device=dev)
        dv = torch.empty(n_ctx, dtype=torch.float32, device=dev)
        fn = lambda: kvb.hkvd_select(kf, kc, kk, sel_out=sel, dev_out=dv)
        out.update(n_ctx=n_ctx, k=kk, kv_dim=kvd, bytes=4.0 * n_ctx * kvd)
    else:
        L, n_ctx = args.layers, args.n_ctx
        ks = torch.randn(L, n_ctx, Hkv, D, generator=g, device=dev).to(torch.bfloat16)
        vs = torch.randn(L, n_ctx, Hkv, D, generator=g, device=dev).to(torch.bfloat16)
        kd = torch.empty_like(ks)
        vd = torch.empty(vs.shape, dtype=torch.float16, device=dev)
        rope = kvb.RopeTable(cfg, n_ctx, dev)
        starts = torch.arange(0, n_ctx + 1, 512, dtype=torch.int32, device=dev)
        fn = lambda: kvb.rope_realign(cfg, rope, ks, vs, kd, vd, 0, L, starts, n_ctx, ws=ws)
        out.update(bytes=4.0 * ks.numel() * 2, layers=L, n_ctx=n_ctx)
    for _ in range(args.reps - 1):
        fn()
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record()
    for _ in range(max(args.timed, 1)):
        fn()
    e1.record()
    torch.cuda.synchronize()
    ms = e0.elapsed_time(e1) / max(args.timed, 1)
    assert kvb.device_status(ws) == 0
    out.update(kernel=args.kernel, ms=round(ms, 4))
    if flop:
        out["tflops"] = round(flop / (ms * 1e-3) / 1e12, 1)
    if "bytes" in out:
        out["gbs"] = round(out["bytes"] / (ms * 1e-3) / 1e9, 1)
    print(json.dumps(out))


def main():
    args = parse()
    if args.kernel:
        run_kernel(args)
        return
    from paper_2609_09768_gb300 import synth
    wl = synth.WORKLOADS[args.workload]
    if args.model_config:
        import dataclasses
        with open(args.model_config) as fh:
            shape = synth.shape_from_config(json.load(fh))
        name = os.path.splitext(os.path.basename(args.model_config))[0]
        wl = dataclasses.replace(wl, shape=shape, name=f"{name}-{shape.n_layers}L-{wl.n_chunks}x{wl.chunk_len}+{wl.n_query}")
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    if args.impl == "reference":
        run_reference(args, wl, rank, world)
        return
    if args.sweep:
        run_sweep(args)
        return
    if args.selectors:
        run_selectors(args)
        return
    import torch
    if world > 1:
        import torch.distributed as dist
        torch.cuda.set_device(int(os.environ.get("LOCAL_RANK", "0")))
        dist.init_process_group("nccl")
    run_ours(args, wl, rank, world)
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
