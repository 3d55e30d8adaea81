"""Device-side set-up of a request for the library: weights, RoPE tables and the
per-chunk KV caches (each chunk prefilled alone through kvb_full_prefill with
block-diagonal key ranges and chunk-local RoPE positions)."""
from __future__ import annotations

from typing import List, Optional

import torch

from . import kvblend as kvb
from . import synth


def device_model(shape: synth.ModelShape, seed: int = 0, device="cuda", draw_on_device: bool = True) -> dict:
    """Random weights of `shape` on `device`.  draw_on_device=False draws them on the
    CPU (the generator the oracle's inputs come from) and copies them over."""
    if draw_on_device:
        return synth.make_model(shape, seed, device)
    w = synth.make_model(shape, seed, "cpu")
    return {"layers": [{k: v.to(device) for k, v in l.items()} for l in w["layers"]],
            "embed": w["embed"].to(device), "final_norm": w["final_norm"].to(device)}


def chunk_layout(chunk_starts: List[int], device="cuda"):
    """(rope_pos, kv_lo) int32 for the isolated per-chunk prefill of the context rows."""
    n = chunk_starts[-1]
    lo = torch.empty(n, dtype=torch.int32)
    for c in range(len(chunk_starts) - 1):
        lo[chunk_starts[c]:chunk_starts[c + 1]] = chunk_starts[c]
    pos = torch.arange(n, dtype=torch.int32) - lo
    return pos.to(device), lo.to(device)


def chunk_caches(cfg: kvb.Config, model: kvb.Model, rope: kvb.RopeTable, ctx_tokens: torch.Tensor,
                 chunk_starts: List[int], ws: Optional[torch.Tensor] = None, zero_rows: Optional[List[int]] = None):
    """Per-chunk caches in the chunk-cache format: K and V bf16 [L][n_ctx][Hkv][D], keys at
    chunk-local positions.  Rows in `zero_rows` (separator tokens) are set to zero in every layer."""
    n_ctx = chunk_starts[-1]
    L = cfg.n_layers
    dev = ctx_tokens.device
    k = torch.empty(L, n_ctx, cfg.n_kv_heads, cfg.head_dim, dtype=torch.bfloat16, device=dev)
    v = torch.empty(L, n_ctx, cfg.n_kv_heads, cfg.head_dim, dtype=torch.bfloat16, device=dev)
    v_att = torch.empty(L, n_ctx, cfg.n_kv_heads, cfg.head_dim, dtype=torch.float16, device=dev)  # read by attention
    pos, lo = chunk_layout(chunk_starts, dev)
    kvb.full_prefill(cfg, model, rope, k, v_att, ctx_tokens, rope_pos=pos, kv_lo=lo, ws=ws, v_chunk_out=v)
    del v_att
    if zero_rows:
        idx = torch.tensor(zero_rows, dtype=torch.long, device=dev)
        k[:, idx] = 0
        v[:, idx] = 0
    return k, v
