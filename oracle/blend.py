"""The selective-recompute prefill after KV-cache concatenation, float64 (oracle).

Test infrastructure only.  Follows the paper's description of the method:

* Per-chunk caches (Sec. 1, Sec. 3.4): every retrieved chunk is prefilled alone,
  at chunk-local positions 0..len-1, and its per-layer K (rotated at those local
  positions) and V are stored.
* Concatenation with position adjustment (Sec. 2 on PIE, Sec. 3.4, Sec. 4): the
  chunk caches are merged into one cache in context order and the keys of chunk
  c, which starts at global position o_c, are rotated by the extra angle o_c*w_i
  so they sit at their global positions.  Values are unchanged.
* Full recompute of layer 0 in causal mode (Sec. 4).
* CacheBlend selection (Sec. 2, Sec. 3.2): at the check layer the fresh keys of
  every context token (computed with full attention at global positions) are
  compared with the concatenated cache's keys; the per-token deviation is the
  sum over kv heads and head dims of the squared difference, and the r = 15 %
  tokens with the largest deviation are recomputed.
* Selective layers: from the check layer on, only the selected context rows and
  the query-suffix rows are recomputed; their fresh K/V replace the cached ones
  before the layer's attention, and each recomputed row attends the whole
  blended cache up to its own position (the causal mask of Limitation 1).
* r = 100 % is full attention (Sec. 4.1, Tables 1-2); r = 0 % is plain
  concatenation.

Readings where the paper is silent (each is listed with its reason in the
design notes): the check layer defaults to 1 (layer-0 keys depend only on token
and position, so their deviation is zero in exact arithmetic); k = floor(r *
N_ctx) with r taken as a float32 value; ties in the deviation go to the lower
token index; the residual stream is kept in full precision.
"""
from __future__ import annotations

import math
from typing import Sequence

import numpy as np

from .llama import (F64, Shape, act, as64, apply_rope, k_rows, layer_rows, rmsnorm, rope_cos_sin)


def embed_rows(embed, tokens) -> np.ndarray:
    """x0[i] = E[token_i] (rows of the embedding table), float64."""
    tokens = np.asarray(tokens, dtype=np.int64)
    if hasattr(embed, "detach"):
        import torch
        return as64(embed[torch.as_tensor(tokens)])
    return as64(np.asarray(embed)[tokens])


def full_prefill(s: Shape, layers: Sequence[dict], x0, rope_pos=None, row_lo=None,
                 keep_layer_outputs: bool = False) -> dict:
    """Every layer over all n rows, causal (row t reads cache rows [lo_t, t]).

    rope_pos defaults to the row index; with row_lo = chunk start and rope_pos =
    index - chunk start this is the block-diagonal per-chunk isolated prefill.
    Returns k/v caches [L, n, Hkv, D], the last hidden x [n, H] and optionally
    every layer's output.
    """
    x = as64(x0)
    n = x.shape[0]
    L = len(layers)
    rows = np.arange(n)
    rope_pos = rows if rope_pos is None else np.asarray(rope_pos)
    kc = np.zeros((L, n, s.n_kv_heads, s.head_dim), dtype=F64)
    vc = np.zeros_like(kc)
    outs = []
    for l, lw in enumerate(layers):
        x = layer_rows(s, lw, x, rows, rope_pos, kc[l], vc[l], row_lo)
        if keep_layer_outputs:
            outs.append(x.copy())
    return {"k": kc, "v": vc, "x": x, "layer_out": outs}


def chunk_caches(s: Shape, layers: Sequence[dict], x0_ctx, chunk_starts: Sequence[int]) -> dict:
    """Per-chunk caches, each chunk prefilled alone at positions 0..len_c-1, laid end to end.

    Returns k (rotated at chunk-local positions) and v, each [L, N_ctx, Hkv, D].
    """
    x0_ctx = as64(x0_ctx)
    L = len(layers)
    n_ctx = chunk_starts[-1]
    kc = np.zeros((L, n_ctx, s.n_kv_heads, s.head_dim), dtype=F64)
    vc = np.zeros_like(kc)
    for c in range(len(chunk_starts) - 1):
        a, b = chunk_starts[c], chunk_starts[c + 1]
        r = full_prefill(s, layers, x0_ctx[a:b])
        kc[:, a:b] = r["k"]
        vc[:, a:b] = r["v"]
    return {"k": kc, "v": vc}


def realign(s: Shape, k_local: np.ndarray, chunk_starts: Sequence[int]) -> np.ndarray:
    """Rotate the keys of chunk c by o_c = chunk_starts[c]: R(o_c) applied to every
    (head, pair), turning chunk-local positions into global ones.  k_local: [..., N_ctx, Hkv, D]
    (any number of leading layer axes)."""
    k = as64(k_local).copy()
    for c in range(len(chunk_starts) - 1):
        a, b = chunk_starts[c], chunk_starts[c + 1]
        cos, sin = rope_cos_sin(s, [chunk_starts[c]])
        blk = k[..., a:b, :, :]
        shp = blk.shape
        flat = blk.reshape(-1, shp[-2], shp[-1])
        rot = apply_rope(flat, np.broadcast_to(cos, (flat.shape[0], cos.shape[1])),
                         np.broadcast_to(sin, (flat.shape[0], sin.shape[1])))
        k[..., a:b, :, :] = rot.reshape(shp)
    return act(s, k)


def hkvd_deviation(k_fresh, k_cached) -> np.ndarray:
    """dev[i] = sum over kv heads h and dims d of (K_fresh[i,h,d] - K_cached[i,h,d])^2."""
    a = as64(k_fresh)
    b = as64(k_cached)
    d = (a - b).reshape(a.shape[0], int(np.prod(a.shape[1:])))
    return np.sum(d * d, axis=1)


def num_selected(r: float, n_ctx: int) -> int:
    """k = floor(r * N_ctx) with r rounded to float32 first (the ABI passes r as float)."""
    r32 = float(np.float32(r))
    return int(math.floor(r32 * n_ctx + 1e-9))


def topk_select(dev, k: int) -> np.ndarray:
    """Indices of the k largest deviations (ties -> lower index), returned ascending."""
    dev = np.asarray(dev)
    n = dev.shape[0]
    order = np.lexsort((np.arange(n), -dev))  # primary: dev descending, then index ascending
    return np.sort(order[:k]).astype(np.int64)


def selective_prefill(s: Shape, layers: Sequence[dict], x0, chunk_starts: Sequence[int],
                      n_query: int, r: float, k_local, v_local, check_layer: int = 1,
                      forced_sel=None, final_norm=None) -> dict:
    """Selective-recompute prefill over concatenated per-chunk caches.

    x0:      [N, H] embedded tokens (context rows then the query suffix)
    k_local, v_local: [L, N_ctx, Hkv, D] per-chunk caches at chunk-local positions
    forced_sel: optional context indices to recompute instead of the HKVD choice

    Returns final_hidden [n_query, H] (after the final RMSNorm when `final_norm`
    is given), the selected indices, the deviation, the recomputed row set, every
    layer's output rows and the blended caches.
    """
    L = len(layers)
    x_all = as64(x0)
    n_ctx = chunk_starts[-1]
    N = n_ctx + n_query
    assert x_all.shape[0] == N
    assert 0 <= check_layer <= L

    # concatenated cache with every chunk's keys moved to global positions
    kc = np.zeros((L, N, s.n_kv_heads, s.head_dim), dtype=F64)
    vc = np.zeros_like(kc)
    kc[:, :n_ctx] = realign(s, k_local, chunk_starts)
    vc[:, :n_ctx] = as64(v_local)

    all_rows = np.arange(N)
    layer_out = []
    # layers before the check layer (layer 0 at least): full causal recompute
    for l in range(min(check_layer, L)):
        x_all = layer_rows(s, layers[l], x_all, all_rows, all_rows, kc[l], vc[l])
        layer_out.append(x_all.copy())

    dev = None
    if check_layer >= L:
        sel = np.arange(n_ctx, dtype=np.int64)
        rows = all_rows
        x = x_all
    else:
        if forced_sel is not None:
            sel = np.sort(np.asarray(forced_sel, dtype=np.int64))
        else:
            lc = check_layer
            ctx = np.arange(n_ctx)
            k_fresh = k_rows(s, layers[lc], x_all[:n_ctx], ctx)
            dev = hkvd_deviation(k_fresh, kc[lc, :n_ctx])
            sel = topk_select(dev, num_selected(r, n_ctx))
        rows = np.concatenate([sel, np.arange(n_ctx, N)])
        x = x_all[rows]
        for l in range(check_layer, L):
            x = layer_rows(s, layers[l], x, rows, rows, kc[l], vc[l])
            layer_out.append(x.copy())

    q_rows = x[-n_query:] if n_query > 0 else x[:0]
    fh = q_rows if final_norm is None else rmsnorm(q_rows, final_norm, s.rms_eps)
    return {"final_hidden": fh, "sel": sel, "dev": dev, "rows": rows,
            "layer_out": layer_out, "k": kc, "v": vc}


def first_token(hidden, lm_head) -> tuple:
    """The first generated token (greedy decoding, Sec. 4): logits = h W^T over the vocabulary,
    token = argmax (the lowest id among equal maxima).  hidden: [n, H] final hidden states."""
    logits = as64(hidden) @ as64(lm_head).T
    return np.argmax(logits, axis=-1).astype(np.int64), logits


def zero_kv_rows(caches: dict, rows) -> dict:
    """Separator tokens (Sec. 3.1, Sec. 4): two special tokens sit between consecutive
    documents and their entries in the concatenated cache are all zero, K and V, every
    layer.  Returns a copy of the caches {"k", "v"} ([L, N_ctx, Hkv, D]) with `rows` zeroed."""
    k = as64(caches["k"]).copy()
    v = as64(caches["v"]).copy()
    rows = np.asarray(rows, dtype=np.int64)
    k[:, rows] = 0.0
    v[:, rows] = 0.0
    return {"k": k, "v": v}


def window_select(win_starts, window: int, n_ctx: int) -> np.ndarray:
    """Fixed-position selection of the compared methods (Sec. 2, Sec. 3.1): EPIC recomputes
    the `window` = 20 tokens that start at each separator position; KVLink recomputes
    the separator tokens themselves (window = number of separator tokens).  The set is
    the union of [s, s + window) over the window starts s, cut to [0, n_ctx), ascending."""
    mark = [False] * n_ctx
    for s in win_starts:
        for i in range(int(s), int(s) + int(window)):
            if 0 <= i < n_ctx:
                mark[i] = True
    return np.array([i for i in range(n_ctx) if mark[i]], dtype=np.int64)


def deviation_histogram(dev, edges) -> np.ndarray:
    """Distribution of per-token squared key differences (the figures of Sec. 3.2 and 3.3).
    Each value d falls in bin j = #(edges e with d >= e); for ascending edges that is
    counts[0] = #(d < edges[0]), counts[j] = #(edges[j-1] <= d < edges[j]),
    counts[len(edges)] = #(d >= edges[-1]).  The comparisons are made in the precision
    of `dev` and `edges` as given."""
    dev = np.asarray(dev)
    edges = np.asarray(edges)
    counts = np.zeros(len(edges) + 1, dtype=np.int64)
    for d in dev:
        counts[sum(1 for e in edges if d >= e)] += 1
    return counts


def decode_step(s: Shape, layers: Sequence[dict], embed, final_norm, lm_head, k_cache: np.ndarray,
                v_cache: np.ndarray, token: int, pos: int) -> tuple:
    """One step of greedy decoding (Sec. 4): the token at position `pos` runs through
    every layer as a single row (its K/V written into cache row `pos` of each layer,
    attention over rows [0, pos]), then the final RMSNorm, the logits and their argmax.
    k_cache, v_cache: [L, n_rows, Hkv, D] float64, updated in place.
    Returns (next token, final hidden [H], logits [vocab])."""
    x = embed_rows(embed, np.array([token]))
    for l, lw in enumerate(layers):
        x = layer_rows(s, lw, x, [pos], [pos], k_cache[l], v_cache[l])
    h = rmsnorm(x, final_norm, s.rms_eps)
    tok, logits = first_token(h, lm_head)
    return int(tok[0]), h[0], logits[0]
