"""Run one kernel of the library on a seeded synthetic case (for timing and ncu captures).

    python -m paper_2609_09768_gb300.profile_case attn  --m 18713 --n-kv 124032 [--reps 2]
    python -m paper_2609_09768_gb300.profile_case dense --n-kv 16384
    python -m paper_2609_09768_gb300.profile_case gemm  --m 18713 --which qkv|o|gateup|down
    python -m paper_2609_09768_gb300.profile_case realign --n-ctx 123904 --layers 2
    python -m paper_2609_09768_gb300.profile_case decode_attn --n-kv 124032
    python -m paper_2609_09768_gb300.profile_case decode_step --n-kv 128 --layers 4

Shapes are the Llama-3.1-8B layer (H 4096, 32 q / 8 kv heads, D 128, F 14336).  The
selected rows of `attn` are drawn uniformly over the context (as the HKVD choice of
r = m / n_kv would spread them) and always include the last row.  Prints the CUDA-event
time of the last repetition (the mean of the last --timed calls) and its algorithmic
throughput.
"""
from __future__ import annotations

import argparse
import json

import torch

from . import build, synth
from . import kvblend as kvb


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("kernel", choices=["attn", "dense", "gemm", "realign", "decode_attn", "decode_step"])
    ap.add_argument("--m", type=int, default=18713)
    ap.add_argument("--n-kv", type=int, default=124032)
    ap.add_argument("--n-ctx", type=int, default=123904)
    ap.add_argument("--layers", type=int, default=2)
    ap.add_argument("--which", default="qkv", choices=["qkv", "o", "gateup", "down"])
    ap.add_argument("--reps", type=int, default=2)
    ap.add_argument("--timed", type=int, default=1,
                    help="calls between the timing events (the mean is reported); more than one keeps the "
                         "host's launch overhead out of short kernels' times")
    a = ap.parse_args()
    build.build()
    shape = synth.LLAMA8B
    cfg = kvb.config(shape)
    dev = torch.device("cuda")
    Hq, Hkv, D, H, F = shape.n_q_heads, shape.n_kv_heads, shape.head_dim, shape.hidden, shape.mlp_dim
    g = torch.Generator(device=dev)
    g.manual_seed(0)
    ws = torch.zeros(256, dtype=torch.uint8, device=dev)
    out = {}
    if a.kernel in ("attn", "dense"):
        n_kv = a.n_kv
        if a.kernel == "dense":
            rows = torch.arange(n_kv, device=dev, dtype=torch.int32)
        else:
            perm = torch.randperm(n_kv - 1, generator=g, device=dev)[: a.m - 1]
            rows = torch.cat([torch.sort(perm).values, torch.tensor([n_kv - 1], device=dev)]).to(torch.int32)
        m = rows.numel()
        q = torch.randn(m, Hq, D, generator=g, device=dev).to(torch.bfloat16)
        kc = torch.randn(n_kv, Hkv, D, generator=g, device=dev).to(torch.bfloat16)
        vc = torch.randn(n_kv, Hkv, D, generator=g, device=dev).to(torch.bfloat16).to(torch.float16)
        o = torch.empty(m, Hq * D, dtype=torch.bfloat16, device=dev)
        fn = lambda: kvb.sparse_query_attn(cfg, q, rows, None, kc, vc, o, ws)
        flop = 4.0 * Hq * D * float((rows.to(torch.float64) + 1).sum())
        out.update(m=m, n_kv=n_kv)
    elif a.kernel == "gemm":
        m = a.m
        lw = {k: v for k, v in synth.make_layer_weights(shape, 0, 0, dev).items()}
        lws = kvb.layer_struct(lw)
        wsl = kvb.workspace(cfg, m, dev)
        if a.which == "qkv":
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
        out.update(m=m, which=("o+gateup+down (mlp_rows)" if a.which != "qkv" else "qkv"))
    elif a.kernel == "decode_attn":
        n_kv = a.n_kv
        q = torch.randn(Hq, D, generator=g, device=dev).to(torch.bfloat16)
        kc = torch.randn(n_kv, Hkv, D, generator=g, device=dev).to(torch.bfloat16)
        vc = torch.randn(n_kv, Hkv, D, generator=g, device=dev).to(torch.bfloat16).to(torch.float16)
        pos = torch.tensor([n_kv - 1], dtype=torch.int32, device=dev)
        ws = kvb.decode_workspace(cfg, n_kv, dev)
        o = torch.empty(Hq, D, dtype=torch.bfloat16, device=dev)
        fn = lambda: kvb.decode_attention(cfg, q, kc, vc, pos, n_kv, out=o, ws=ws)
        flop = None
        out.update(bytes=float(n_kv) * Hkv * D * 2 * 2, n_kv=n_kv)
    elif a.kernel == "decode_step":
        # a decode step of an a.layers-layer model at position n_kv - 1 (step time minus the
        # lm_head is per-layer GEMV + attention time)
        shp = shape.with_layers(a.layers)
        cfgl = kvb.config(shp)
        model = kvb.Model(synth.make_model(shp, 0, dev))
        lm = synth.make_lm_head(shp, 0, dev)
        n_kv = a.n_kv
        rope = kvb.RopeTable(cfgl, n_kv, dev)
        kc = torch.randn(a.layers, n_kv, Hkv, D, generator=g, device=dev).to(torch.bfloat16)
        vc = torch.randn(a.layers, n_kv, Hkv, D, generator=g, device=dev).to(torch.bfloat16).to(torch.float16)
        tokens = torch.zeros(n_kv + 1, dtype=torch.int32, device=dev)
        pos = torch.tensor([n_kv - 1], dtype=torch.int32, device=dev)
        ws = kvb.decode_workspace(cfgl, n_kv, dev)

        def fn():
            pos.fill_(n_kv - 1)
            kvb.decode_step(cfgl, model, rope, kc, vc, lm, tokens, pos, n_kv, ws=ws)
        flop = None
        wb = a.layers * 2.0 * (shp.qkv_dim * H + H * shp.q_dim + 3 * H * F) + shp.vocab * H * 2.0
        out.update(bytes=wb + a.layers * float(n_kv) * Hkv * D * 4, layers=a.layers, n_kv=n_kv)
    else:
        L, n_ctx = a.layers, a.n_ctx
        ks = torch.randn(L, n_ctx, Hkv, D, generator=g, device=dev).to(torch.bfloat16)
        vs = torch.randn(L, n_ctx, Hkv, D, generator=g, device=dev).to(torch.float16)
        kd, vd = torch.empty_like(ks), torch.empty_like(vs)
        rope = kvb.RopeTable(cfg, n_ctx, dev)
        starts = torch.arange(0, n_ctx + 1, 512, dtype=torch.int32, device=dev)
        fn = lambda: kvb.rope_realign(cfg, rope, ks, vs, kd, vd, 0, L, starts, n_ctx)
        flop = None
        out.update(bytes=4.0 * ks.numel() * 2, layers=L, n_ctx=n_ctx)
    for _ in range(a.reps - 1):
        fn()
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record()
    for _ in range(max(a.timed, 1)):
        fn()
    e1.record()
    torch.cuda.synchronize()
    ms = e0.elapsed_time(e1) / max(a.timed, 1)
    assert kvb.device_status(ws) == 0
    out.update(kernel=a.kernel, ms=round(ms, 4))
    if flop:
        out["tflops"] = round(flop / (ms * 1e-3) / 1e12, 1)
    if "bytes" in out:
        out["gbs"] = round(out["bytes"] / (ms * 1e-3) / 1e9, 1)
    print(json.dumps(out))


if __name__ == "__main__":
    main()
