"""Thin ctypes binding of libkvblend.so (the C ABI in include/kvblend.h).

Argument marshalling only: tensors are checked for device, dtype and layout and
their data pointers are handed to the C entry points together with the current
torch CUDA stream.  Every step of the computation runs in the library's CUDA
kernels; there is no fallback.  If the library is missing, `lib()` raises.
"""
from __future__ import annotations

import ctypes as C
import os
from typing import Dict, Optional, Tuple

import numpy as np
import torch

from .build import LIB

c_i32, c_i64, c_f32, c_sz, c_vp = C.c_int32, C.c_int64, C.c_float, C.c_size_t, C.c_void_p


class KvbError(RuntimeError):
    """A kvb_* call returned a status other than KVB_OK."""

    def __init__(self, fn: str, status: int, msg: str):
        super().__init__(f"{fn}: status {status} ({STATUS.get(status, '?')}): {msg}")
        self.status = status


STATUS = {0: "ok", 1: "invalid argument", 2: "unsupported", 3: "CUDA error", 4: "device wait timed out",
          5: "workspace too small", 6: "value out of range"}
(KVB_OK, KVB_ERR_INVALID_ARG, KVB_ERR_UNSUPPORTED, KVB_ERR_CUDA, KVB_ERR_TIMEOUT, KVB_ERR_WORKSPACE,
 KVB_ERR_RANGE) = range(7)
KVB_ROPE_PLAIN, KVB_ROPE_LLAMA3, KVB_ROPE_YARN = range(3)


class Config(C.Structure):
    _fields_ = [("hidden", c_i32), ("n_q_heads", c_i32), ("n_kv_heads", c_i32), ("head_dim", c_i32),
                ("mlp_dim", c_i32), ("n_layers", c_i32), ("vocab", c_i32), ("rms_eps", c_f32),
                ("rope_theta", c_f32), ("rope_scaling", c_i32), ("rs_factor", c_f32), ("rs_low", c_f32),
                ("rs_high", c_f32), ("rs_orig_ctx", c_i32)]


class LayerWeights(C.Structure):
    _fields_ = [("attn_norm", c_vp), ("w_qkv", c_vp), ("w_o", c_vp), ("mlp_norm", c_vp), ("w_gate", c_vp),
                ("w_up", c_vp), ("w_down", c_vp), ("b_qkv", c_vp)]


class ModelStruct(C.Structure):
    _fields_ = [("layers", C.POINTER(LayerWeights)), ("embed", c_vp), ("final_norm", c_vp)]


class RopeTableStruct(C.Structure):
    _fields_ = [("cos", c_vp), ("sin", c_vp), ("max_pos", c_i64)]


class KVCache(C.Structure):
    _fields_ = [("k", c_vp), ("v", c_vp), ("n_rows", c_i64), ("n_layers", c_i32)]


class Timings(C.Structure):
    _fields_ = [("total_ms", c_f32), ("realign_ms", c_f32), ("dense_ms", c_f32), ("select_ms", c_f32),
                ("selective_ms", c_f32), ("final_ms", c_f32), ("attn_dense_ms", c_f32), ("attn_sel_ms", c_f32),
                ("gemm_ms", c_f32), ("hkvd_ms", c_f32), ("n_attn_dense", c_i32), ("n_attn_sel", c_i32), ("n_gemm", c_i32),
                ("n_launches", c_i32), ("n_selected", c_i64), ("n_rows", c_i64)]

    def as_dict(self) -> dict:
        return {f: getattr(self, f) for f, _ in self._fields_}


class LayerTapsStruct(C.Structure):
    _fields_ = [("n", c_i32), ("layers", C.POINTER(c_i32)), ("x_out", c_vp), ("rows_cap", c_i64),
                ("rows_out", C.POINTER(c_i64))]


P = C.POINTER
_SIGS = {
    "kvb_status_string": (C.c_char_p, [c_i32]),
    "kvb_last_error": (C.c_char_p, []),
    "kvb_version": (c_i32, []),
    "kvb_rope_table_fill": (c_i32, [P(Config), c_i64, c_vp, c_vp]),
    "kvb_attention_scale": (c_i32, [P(Config), P(c_f32)]),
    "kvb_rope_realign": (c_i32, [P(Config), P(RopeTableStruct), c_vp, c_vp, c_i64, c_vp, c_vp, c_i64, c_i32, c_i32,
                                 c_vp, c_i32, c_i64, c_vp, c_sz, c_vp]),
    "kvb_hkvd_workspace_size": (c_sz, [c_i64]),
    "kvb_hkvd_select": (c_i32, [c_vp, c_i64, c_vp, c_i64, c_i64, c_i32, c_i64, c_vp, c_vp, c_vp, c_sz, c_vp]),
    "kvb_gather_rmsnorm_qkv": (c_i32, [P(Config), P(LayerWeights), P(RopeTableStruct), c_vp, c_vp, c_vp, c_i64,
                                       c_vp, c_vp, c_vp, c_vp, c_i64, c_vp, c_sz, c_vp]),
    "kvb_gather_rmsnorm_qkv_noalloc": (c_i32, [P(Config), P(LayerWeights), P(RopeTableStruct), c_vp, c_vp, c_vp,
                                               c_i64, c_vp, c_vp, c_vp, c_vp, c_i64, c_vp, c_vp]),
    "kvb_kv_scatter": (c_i32, [c_vp, c_vp, c_vp, c_i64, c_i32, c_vp, c_vp, c_i64, c_vp]),
    "kvb_sparse_query_attn": (c_i32, [P(Config), c_vp, c_vp, c_vp, c_i64, c_vp, c_vp, c_i64, c_vp, c_vp, c_sz,
                                      c_vp]),
    "kvb_mlp_rows": (c_i32, [P(Config), P(LayerWeights), c_vp, c_i64, c_vp, c_vp, c_sz, c_vp]),
    "kvb_workspace_size": (c_i32, [P(Config), c_i64, P(c_sz)]),
    "kvb_selective_prefill": (c_i32, [P(Config), P(ModelStruct), P(RopeTableStruct), c_vp, c_vp, P(KVCache), c_vp,
                                      c_vp, c_i32, c_i64, c_i64, c_f32, c_i32, c_vp, c_i64, c_vp, c_vp, P(Timings),
                                      P(LayerTapsStruct), c_vp, c_sz, c_vp]),
    "kvb_selective_prefill_host": (c_i32, [P(Config), P(ModelStruct), P(RopeTableStruct), c_vp, c_vp, P(KVCache),
                                           c_vp, c_vp, c_i32, c_i64, c_i64, c_f32, c_i32, c_vp, c_i64, c_vp, c_vp,
                                           P(Timings), P(LayerTapsStruct), c_vp, c_sz, c_vp, c_vp]),
    "kvb_workspace_size_pipelined": (c_i32, [P(Config), c_i64, c_i64, P(c_sz)]),
    "kvb_full_prefill": (c_i32, [P(Config), P(ModelStruct), P(RopeTableStruct), P(KVCache), c_vp, c_vp, c_i64, c_vp,
                                 c_vp, c_vp, c_i64, P(Timings), P(LayerTapsStruct), c_vp, c_sz, c_vp]),
    "kvb_device_status": (c_i32, [c_vp, c_sz, c_vp, P(c_i32)]),
    "kvb_debug_wait_timeout": (c_i32, [c_vp, c_sz, c_i64, c_vp]),
    "kvb_lm_head_argmax": (c_i32, [P(Config), c_vp, c_vp, c_i32, c_vp, c_vp, c_vp, c_sz, c_vp]),
    "kvb_decode_workspace_size": (c_i32, [P(Config), c_i64, P(c_sz)]),
    "kvb_decode_step": (c_i32, [P(Config), P(ModelStruct), P(RopeTableStruct), P(KVCache), c_vp, c_vp, c_vp, c_i64,
                                c_vp, c_vp, c_sz, c_vp]),
    "kvb_decode_attention": (c_i32, [P(Config), c_vp, c_vp, c_vp, c_i64, c_vp, c_i64, c_vp, c_vp, c_sz, c_vp]),
    "kvb_window_select_workspace_size": (c_sz, [c_i64]),
    "kvb_window_select": (c_i32, [c_vp, c_i32, c_i32, c_i64, c_vp, c_vp, c_vp, c_sz, c_vp]),
    "kvb_key_deviation_histogram": (c_i32, [c_vp, c_i64, c_vp, c_i64, c_i64, c_i32, c_vp, c_i32, c_vp, c_vp, c_vp,
                                            c_sz, c_vp]),
}
EXPORTED = tuple(_SIGS)

_LIB: Optional[C.CDLL] = None


def lib_path() -> str:
    return LIB


def lib() -> C.CDLL:
    """Load libkvblend.so (built by `build.build()`); raises if it is missing."""
    global _LIB
    if _LIB is None:
        if not os.path.exists(LIB):
            raise RuntimeError(f"libkvblend.so not built ({LIB}); run __graft_entry__.build() first")
        L = C.CDLL(LIB)
        for name, (res, args) in _SIGS.items():
            f = getattr(L, name)
            f.restype, f.argtypes = res, args
        _LIB = L
    return _LIB


def _call(name: str, *args) -> None:
    st = getattr(lib(), name)(*args)
    if st != KVB_OK:
        raise KvbError(name, st, lib().kvb_last_error().decode())


def _stream() -> int:
    return torch.cuda.current_stream().cuda_stream


def _ptr(t: Optional[torch.Tensor], dtype=None, name: str = "tensor") -> Optional[int]:
    if t is None:
        return None
    if not t.is_cuda:
        raise ValueError(f"{name} must be a CUDA tensor")
    if dtype is not None and t.dtype != dtype:
        raise ValueError(f"{name} must be {dtype}, got {t.dtype}")
    if not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")
    return t.data_ptr()


def config(shape, n_layers: Optional[int] = None) -> Config:
    """kvb_config from any object with ModelShape's fields."""
    return Config(shape.hidden, shape.n_q_heads, shape.n_kv_heads, shape.head_dim, shape.mlp_dim,
                  shape.n_layers if n_layers is None else n_layers, shape.vocab, shape.rms_eps, shape.rope_theta,
                  int(shape.rope_scaling), shape.rs_factor, shape.rs_low, shape.rs_high, shape.rs_orig_ctx)


# ---------------------------------------------------------------------------------- RoPE

def rope_table_fill(cfg: Config, max_pos: int) -> Tuple[np.ndarray, np.ndarray]:
    half = cfg.head_dim // 2
    cos = np.empty((max_pos, half), dtype=np.float32)
    sin = np.empty((max_pos, half), dtype=np.float32)
    _call("kvb_rope_table_fill", C.byref(cfg), max_pos, cos.ctypes.data, sin.ctypes.data)
    return cos, sin


def attention_scale(cfg: Config) -> float:
    """The q.k factor of every attention kernel (1/sqrt(D), times YaRN's temperature)."""
    out = c_f32(0.0)
    _call("kvb_attention_scale", C.byref(cfg), C.byref(out))
    return out.value


class RopeTable:
    """Device cos/sin tables [max_pos][D/2] (fp32) and the struct pointing at them."""

    def __init__(self, cfg: Config, max_pos: int, device="cuda"):
        cos, sin = rope_table_fill(cfg, max_pos)
        self.cos = torch.from_numpy(cos).to(device)
        self.sin = torch.from_numpy(sin).to(device)
        self.struct = RopeTableStruct(self.cos.data_ptr(), self.sin.data_ptr(), max_pos)


# ---------------------------------------------------------------------------------- model

def layer_struct(lw: Dict[str, torch.Tensor]) -> LayerWeights:
    return LayerWeights(_ptr(lw["attn_norm"], torch.float32, "attn_norm"), _ptr(lw["w_qkv"], torch.bfloat16, "w_qkv"),
                        _ptr(lw["w_o"], torch.bfloat16, "w_o"), _ptr(lw["mlp_norm"], torch.float32, "mlp_norm"),
                        _ptr(lw["w_gate"], torch.bfloat16, "w_gate"), _ptr(lw["w_up"], torch.bfloat16, "w_up"),
                        _ptr(lw["w_down"], torch.bfloat16, "w_down"), _ptr(lw.get("b_qkv"), torch.float32, "b_qkv"))


class Model:
    """Device weights ({'layers': [...], 'embed', 'final_norm'}) and the kvb_model struct."""

    def __init__(self, weights: dict):
        self.weights = weights
        self.layers = (LayerWeights * len(weights["layers"]))(*[layer_struct(l) for l in weights["layers"]])
        self.struct = ModelStruct(C.cast(self.layers, P(LayerWeights)),
                                  _ptr(weights["embed"], torch.bfloat16, "embed"),
                                  _ptr(weights["final_norm"], torch.float32, "final_norm"))


def kv_cache_struct(k: torch.Tensor, v: torch.Tensor) -> KVCache:
    """Blended cache: k [L][n_rows][Hkv][D] bf16; v the same shape, fp16 (bf16-precision values)."""
    assert k.shape == v.shape and k.dim() == 4
    return KVCache(_ptr(k, torch.bfloat16, "cache k"), _ptr(v, torch.float16, "cache v"), k.shape[1], k.shape[0])


class LayerTaps:
    """Residual rows captured at layer boundaries (kvb_layer_taps): slot i holds the fp32 rows
    entering layer layers[i] (n_layers: leaving the last layer), rows_cap rows per slot.
    After the call, `rows(i)` is the number of rows captured in slot i and `get(i)` the
    [rows][H] view of them."""

    def __init__(self, layers, rows_cap: int, hidden: int, device="cuda"):
        self.layers = list(int(l) for l in layers)
        self.hidden = hidden
        self.x = torch.zeros(max(len(self.layers), 1), rows_cap, hidden, dtype=torch.float32, device=device)
        self._layers = (c_i32 * max(len(self.layers), 1))(*self.layers)
        self._rows = (c_i64 * max(len(self.layers), 1))()
        self.struct = LayerTapsStruct(len(self.layers), self._layers, self.x.data_ptr(), rows_cap, self._rows)

    def rows(self, i: int) -> int:
        return int(self._rows[i])

    def get(self, i: int) -> torch.Tensor:
        return self.x[i, : self.rows(i)]


def _taps(taps: Optional[LayerTaps]):
    return C.byref(taps.struct) if taps is not None else None


# ---------------------------------------------------------------------------------- workspace

def workspace_size(cfg: Config, n_rows: int) -> int:
    n = c_sz(0)
    _call("kvb_workspace_size", C.byref(cfg), n_rows, C.byref(n))
    return n.value


def workspace(cfg: Config, n_rows: int, device="cuda") -> torch.Tensor:
    """A zeroed workspace (the zeroed head is the device status word)."""
    return torch.zeros(workspace_size(cfg, n_rows), dtype=torch.uint8, device=device)


LMHEAD_MAX_ROWS = 4


def lm_head_argmax(cfg: Config, lm_head: torch.Tensor, hidden: torch.Tensor, logits: Optional[torch.Tensor] = None,
                   tokens: Optional[torch.Tensor] = None, ws: Optional[torch.Tensor] = None):
    """First-token logits and argmax for up to LMHEAD_MAX_ROWS rows of final hidden states."""
    n = hidden.shape[0]
    dev = hidden.device
    if tokens is None:
        tokens = torch.empty(n, dtype=torch.int32, device=dev)
    if ws is None:
        ws = torch.zeros(256 + 8 * LMHEAD_MAX_ROWS, dtype=torch.uint8, device=dev)
    _call("kvb_lm_head_argmax", C.byref(cfg), _ptr(lm_head, torch.bfloat16, "lm_head"),
          _ptr(hidden, torch.float32, "hidden"), n, _ptr(logits, torch.float32, "logits"),
          _ptr(tokens, torch.int32, "tokens"), _ptr(ws), ws.numel(), _stream())
    return tokens, logits


def window_select(win_start: torch.Tensor, window: int, n_ctx: int, sel_out: Optional[torch.Tensor] = None,
                  ws: Optional[torch.Tensor] = None) -> Tuple[torch.Tensor, int]:
    """EPIC / KVLink selection: the union of [s, s + window) over the window starts, cut to
    the context, ascending.  Returns (the selection, its length); reading the length waits
    for the stream."""
    dev = win_start.device
    n_win = win_start.numel()
    if sel_out is None:
        sel_out = torch.empty(max(min(n_ctx, n_win * window), 1), dtype=torch.int32, device=dev)
    need = lib().kvb_window_select_workspace_size(n_ctx)
    if ws is None:
        ws = torch.zeros(need, dtype=torch.uint8, device=dev)
    k_out = torch.zeros(1, dtype=torch.int64, device=dev)
    _call("kvb_window_select", _ptr(win_start, torch.int32, "win_start"), n_win, window, n_ctx,
          _ptr(sel_out, torch.int32, "sel_out"), _ptr(k_out, torch.int64, "k_out"), _ptr(ws), ws.numel(), _stream())
    k = int(k_out.item())
    return sel_out[:k], k


def key_deviation_histogram(k_a: torch.Tensor, k_b: torch.Tensor, edges: torch.Tensor,
                            dev_out: Optional[torch.Tensor] = None, ws: Optional[torch.Tensor] = None) -> torch.Tensor:
    """Per-token squared key difference between two [n][kv_dim] bf16 key sets (row strides
    taken from the tensors), binned by `edges`; returns int64 counts [len(edges) + 1]."""
    n = k_a.shape[0]
    kv_dim = k_a[0].numel() if n else k_a.shape[-1]
    if k_b.shape[0] != n:
        raise ValueError("k_a and k_b need the same number of rows")
    for t, nm in ((k_a, "k_a"), (k_b, "k_b")):
        if t.dtype != torch.bfloat16 or not t.is_cuda:
            raise ValueError(f"{nm} must be a CUDA bf16 tensor")
        if n and not t[0].is_contiguous():
            raise ValueError(f"{nm} rows must be contiguous")
    ld_a = k_a.stride(0)
    ld_b = k_b.stride(0)
    hist = torch.empty(edges.numel() + 1, dtype=torch.int64, device=k_a.device)
    if ws is None:
        ws = torch.zeros(256 + (0 if dev_out is not None else 4 * n + 16), dtype=torch.uint8, device=k_a.device)
    _call("kvb_key_deviation_histogram", k_a.data_ptr(), ld_a, k_b.data_ptr(), ld_b, n, kv_dim,
          _ptr(edges, torch.float32, "edges"), edges.numel(), _ptr(dev_out, torch.float32, "dev_out"),
          _ptr(hist, torch.int64, "hist"), _ptr(ws), ws.numel(), _stream())
    return hist


def debug_wait_timeout(ws: torch.Tensor, limit_ns: int) -> None:
    _call("kvb_debug_wait_timeout", _ptr(ws), ws.numel(), limit_ns, _stream())


def device_status(ws: torch.Tensor) -> int:
    code = c_i32(0)
    _call("kvb_device_status", _ptr(ws), ws.numel(), _stream(), C.byref(code))
    return code.value


# ---------------------------------------------------------------------------------- steps

def rope_realign(cfg: Config, rope: RopeTable, k_src, v_src, k_dst, v_dst, layer_begin: int, layer_end: int,
                 chunk_start: torch.Tensor, n_ctx: int, ws: Optional[torch.Tensor] = None) -> None:
    """Chunk caches (k_src, v_src: bf16 [L][src_rows][Hkv][D]) -> blended-cache layers (k_dst bf16,
    v_dst fp16).  v_src / v_dst may be None (V untouched); a V value outside fp16's range is
    recorded as KVB_ERR_RANGE in the status word of `ws` (256 bytes, allocated if None)."""
    if ws is None and v_src is not None and v_dst is not None:
        ws = torch.zeros(256, dtype=torch.uint8, device=k_src.device)
    if v_src is not None and v_dst is not None and v_src.data_ptr() == v_dst.data_ptr():
        # in place: the same memory holds bf16 before and fp16 after the call
        vs, vd = _ptr(v_src, None, "v_src"), _ptr(v_dst, None, "v_dst")
    else:
        vs, vd = _ptr(v_src, torch.bfloat16, "v_src"), _ptr(v_dst, torch.float16, "v_dst")
    _call("kvb_rope_realign", C.byref(cfg), C.byref(rope.struct), _ptr(k_src, torch.bfloat16, "k_src"),
          vs, k_src.shape[1], _ptr(k_dst, torch.bfloat16, "k_dst"),
          vd, k_dst.shape[1], layer_begin, layer_end,
          _ptr(chunk_start, torch.int32, "chunk_start"), chunk_start.numel() - 1, n_ctx,
          _ptr(ws) if ws is not None else None, ws.numel() if ws is not None else 0, _stream())


def hkvd_select(k_fresh: torch.Tensor, k_cached: torch.Tensor, k: int, sel_out=None, dev_out=None,
                ws: Optional[torch.Tensor] = None) -> Tuple[torch.Tensor, torch.Tensor]:
    """k_fresh, k_cached: [n_ctx][kv_dim] bf16 (or any row-major view with that row count)."""
    n = k_fresh.shape[0]
    kv_dim = k_fresh[0].numel() if n else 0
    dev = dev_out if dev_out is not None else torch.empty(n, dtype=torch.float32, device=k_fresh.device)
    sel = sel_out if sel_out is not None else torch.empty(max(k, 1), dtype=torch.int32, device=k_fresh.device)
    need = lib().kvb_hkvd_workspace_size(n)
    if ws is None and need:
        ws = torch.zeros(need, dtype=torch.uint8, device=k_fresh.device)
    _call("kvb_hkvd_select", _ptr(k_fresh, torch.bfloat16, "k_fresh"), kv_dim, _ptr(k_cached, torch.bfloat16, "k_cached"),
          kv_dim, n, kv_dim, k, _ptr(sel, torch.int32, "sel"), _ptr(dev, torch.float32, "dev"),
          _ptr(ws) if ws is not None else None, ws.numel() if ws is not None else 0, _stream())
    return sel[:k], dev


def gather_rmsnorm_qkv(cfg: Config, lw: LayerWeights, rope: RopeTable, x: torch.Tensor, row_idx, rope_pos, m: int,
                       q_out, k_out, v_out, kv_dst, ws: torch.Tensor, n_kv_rows: Optional[int] = None) -> None:
    """k_out / v_out hold n_kv_rows rows (default: k_out's first dimension)."""
    if n_kv_rows is None:
        n_kv_rows = k_out.shape[0]
    _call("kvb_gather_rmsnorm_qkv", C.byref(cfg), C.byref(lw), C.byref(rope.struct), _ptr(x, torch.float32, "x"),
          _ptr(row_idx, torch.int32, "row_idx"), _ptr(rope_pos, torch.int32, "rope_pos"), m,
          _ptr(q_out, torch.bfloat16, "q_out"), _ptr(k_out, torch.bfloat16, "k_out"), _ptr(v_out, torch.float16, "v_out"),
          _ptr(kv_dst, torch.int32, "kv_dst"), n_kv_rows, _ptr(ws), ws.numel(), _stream())


NOALLOC_MAX_ELEMS = 4 * 1024 * 1024


def gather_rmsnorm_qkv_noalloc(cfg: Config, lw: LayerWeights, rope: RopeTable, x: torch.Tensor, row_idx, rope_pos,
                               m: int, q_out, k_out, v_out, kv_dst, status_out: Optional[torch.Tensor] = None,
                               n_kv_rows: Optional[int] = None) -> None:
    """kvb_gather_rmsnorm_qkv without a workspace: the library's fixed scratch holds the
    normalised rows (m * hidden <= NOALLOC_MAX_ELEMS), for callers that cannot allocate."""
    if n_kv_rows is None:
        n_kv_rows = k_out.shape[0]
    _call("kvb_gather_rmsnorm_qkv_noalloc", C.byref(cfg), C.byref(lw), C.byref(rope.struct),
          _ptr(x, torch.float32, "x"), _ptr(row_idx, torch.int32, "row_idx"), _ptr(rope_pos, torch.int32, "rope_pos"),
          m, _ptr(q_out, torch.bfloat16, "q_out"), _ptr(k_out, torch.bfloat16, "k_out"),
          _ptr(v_out, torch.float16, "v_out"), _ptr(kv_dst, torch.int32, "kv_dst"), n_kv_rows,
          _ptr(status_out, torch.int32, "status_out"), _stream())


def kv_scatter(k_rows, v_rows, dst_idx, k_dst, v_dst) -> None:
    m = dst_idx.numel()
    kv_dim = k_rows[0].numel() if m else 8
    _call("kvb_kv_scatter", _ptr(k_rows, torch.bfloat16, "k_rows"), _ptr(v_rows, torch.float16, "v_rows"),
          _ptr(dst_idx, torch.int32, "dst_idx"), m, kv_dim, _ptr(k_dst, torch.bfloat16, "k_dst"),
          _ptr(v_dst, torch.float16, "v_dst"), k_dst.shape[0], _stream())


def sparse_query_attn(cfg: Config, q, q_idx, kv_lo, k_cache, v_cache, out, ws: torch.Tensor) -> None:
    _call("kvb_sparse_query_attn", C.byref(cfg), _ptr(q, torch.bfloat16, "q"), _ptr(q_idx, torch.int32, "q_idx"),
          _ptr(kv_lo, torch.int32, "kv_lo"), q_idx.numel(), _ptr(k_cache, torch.bfloat16, "k_cache"),
          _ptr(v_cache, torch.float16, "v_cache"), k_cache.shape[0], _ptr(out, torch.bfloat16, "out"), _ptr(ws),
          ws.numel(), _stream())


def mlp_rows(cfg: Config, lw: LayerWeights, attn, x, ws: torch.Tensor) -> None:
    _call("kvb_mlp_rows", C.byref(cfg), C.byref(lw), _ptr(attn, torch.bfloat16, "attn"), x.shape[0],
          _ptr(x, torch.float32, "x"), _ptr(ws), ws.numel(), _stream())


# ---------------------------------------------------------------------------------- whole prefill

def selective_prefill(cfg: Config, model: Model, rope: RopeTable, k_chunks, v_chunks, cache_k, cache_v, token_ids,
                      chunk_start: torch.Tensor, n_ctx: int, n_query: int, r: float, check_layer: int = 1,
                      forced_sel: Optional[torch.Tensor] = None, final_hidden=None, sel_out=None,
                      ws: Optional[torch.Tensor] = None, timings: bool = False, taps: Optional[LayerTaps] = None):
    """Runs kvb_selective_prefill on chunk caches k_chunks / v_chunks (bf16 [L][n_ctx][Hkv][D]) into the
    blended cache (cache_k bf16, cache_v fp16).  Returns (final_hidden [n_query][H] fp32, sel_out,
    timings dict or None)."""
    dev = token_ids.device
    if final_hidden is None:
        final_hidden = torch.empty(max(n_query, 1), cfg.hidden, dtype=torch.float32, device=dev)
    if sel_out is None:
        sel_out = torch.empty(max(n_ctx, 1), dtype=torch.int32, device=dev)
    if ws is None:
        ws = workspace(cfg, n_ctx + n_query, dev)
    cache = kv_cache_struct(cache_k, cache_v)
    t = Timings()
    _call("kvb_selective_prefill", C.byref(cfg), C.byref(model.struct), C.byref(rope.struct),
          _ptr(k_chunks, torch.bfloat16, "k_chunks"), _ptr(v_chunks, torch.bfloat16, "v_chunks"), C.byref(cache),
          _ptr(token_ids, torch.int32, "token_ids"), _ptr(chunk_start, torch.int32, "chunk_start"),
          (chunk_start.numel() - 1) if chunk_start is not None else 0, n_ctx, n_query, r, check_layer,
          _ptr(forced_sel, torch.int32, "forced_sel"), forced_sel.numel() if forced_sel is not None else 0,
          _ptr(final_hidden, torch.float32, "final_hidden"), _ptr(sel_out, torch.int32, "sel_out"),
          C.byref(t) if timings else None, _taps(taps), _ptr(ws), ws.numel(), _stream())
    return final_hidden[:n_query], sel_out, (t.as_dict() if timings else None)


def workspace_size_pipelined(cfg: Config, n_rows: int, n_ctx: int) -> int:
    n = c_sz(0)
    _call("kvb_workspace_size_pipelined", C.byref(cfg), n_rows, n_ctx, C.byref(n))
    return n.value


def _host_ptr(t: torch.Tensor, dtype, name: str) -> int:
    if t.is_cuda or not t.is_pinned():
        raise ValueError(f"{name} must be a pinned host tensor")
    if t.dtype != dtype or not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous {dtype}")
    return t.data_ptr()


def selective_prefill_host(cfg: Config, model: Model, rope: RopeTable, k_chunks_host, v_chunks_host, cache_k, cache_v,
                           token_ids, chunk_start: torch.Tensor, n_ctx: int, n_query: int, r: float,
                           check_layer: int = 1, copy_stream: Optional[torch.cuda.Stream] = None,
                           forced_sel: Optional[torch.Tensor] = None, final_hidden=None, sel_out=None,
                           ws: Optional[torch.Tensor] = None, timings: bool = False,
                           taps: Optional[LayerTaps] = None):
    """kvb_selective_prefill_host: chunk caches in pinned host memory, ingested layer by layer
    on `copy_stream` under the compute on the current stream."""
    dev = token_ids.device
    if final_hidden is None:
        final_hidden = torch.empty(max(n_query, 1), cfg.hidden, dtype=torch.float32, device=dev)
    if sel_out is None:
        sel_out = torch.empty(max(n_ctx, 1), dtype=torch.int32, device=dev)
    if ws is None:
        ws = torch.zeros(workspace_size_pipelined(cfg, n_ctx + n_query, n_ctx), dtype=torch.uint8, device=dev)
    if copy_stream is None:
        copy_stream = torch.cuda.Stream(device=dev)
    cache = kv_cache_struct(cache_k, cache_v)
    t = Timings()
    _call("kvb_selective_prefill_host", C.byref(cfg), C.byref(model.struct), C.byref(rope.struct),
          _host_ptr(k_chunks_host, torch.bfloat16, "k_chunks_host"), _host_ptr(v_chunks_host, torch.bfloat16, "v_chunks_host"),
          C.byref(cache), _ptr(token_ids, torch.int32, "token_ids"), _ptr(chunk_start, torch.int32, "chunk_start"),
          chunk_start.numel() - 1, n_ctx, n_query, r, check_layer,
          _ptr(forced_sel, torch.int32, "forced_sel"), forced_sel.numel() if forced_sel is not None else 0,
          _ptr(final_hidden, torch.float32, "final_hidden"), _ptr(sel_out, torch.int32, "sel_out"),
          C.byref(t) if timings else None, _taps(taps), _ptr(ws), ws.numel(), _stream(), copy_stream.cuda_stream)
    return final_hidden[:n_query], sel_out, (t.as_dict() if timings else None)


def full_prefill(cfg: Config, model: Model, rope: RopeTable, cache_k, cache_v, token_ids, rope_pos=None, kv_lo=None,
                 n_out: int = 0, final_hidden=None, ws: Optional[torch.Tensor] = None, timings: bool = False,
                 v_chunk_out: Optional[torch.Tensor] = None, taps: Optional[LayerTaps] = None):
    """Runs kvb_full_prefill over all rows of token_ids into the blended cache (cache_k bf16, cache_v
    fp16); v_chunk_out (bf16 [L][n][Hkv][D]) also receives every layer's V in the chunk-cache format.
    Returns (final_hidden or None, timings or None)."""
    n = token_ids.numel()
    dev = token_ids.device
    if n_out and final_hidden is None:
        final_hidden = torch.empty(n_out, cfg.hidden, dtype=torch.float32, device=dev)
    if ws is None:
        ws = workspace(cfg, n, dev)
    cache = kv_cache_struct(cache_k, cache_v)
    t = Timings()
    _call("kvb_full_prefill", C.byref(cfg), C.byref(model.struct), C.byref(rope.struct), C.byref(cache),
          _ptr(v_chunk_out, torch.bfloat16, "v_chunk_out"),
          _ptr(token_ids, torch.int32, "token_ids"), n, _ptr(rope_pos, torch.int32, "rope_pos"),
          _ptr(kv_lo, torch.int32, "kv_lo"), _ptr(final_hidden, torch.float32, "final_hidden") if n_out else None,
          n_out, C.byref(t) if timings else None, _taps(taps), _ptr(ws), ws.numel(), _stream())
    return final_hidden, (t.as_dict() if timings else None)


# ---------------------------------------------------------------------------------- decode

def decode_workspace(cfg: Config, max_pos: int, device="cuda") -> torch.Tensor:
    """A zeroed workspace for kvb_decode_step / kvb_decode_attention up to max_pos."""
    n = c_sz(0)
    _call("kvb_decode_workspace_size", C.byref(cfg), max_pos, C.byref(n))
    return torch.zeros(n.value, dtype=torch.uint8, device=device)


def decode_step(cfg: Config, model: Model, rope: RopeTable, cache_k, cache_v, lm_head: torch.Tensor,
                tokens: torch.Tensor, pos: torch.Tensor, max_pos: int, hidden: Optional[torch.Tensor] = None,
                ws: Optional[torch.Tensor] = None):
    """One greedy decode step on the device: reads tokens[pos], writes tokens[pos + 1] and
    the new K/V at cache row pos, increments pos (int32 [1] on the device)."""
    if ws is None:
        ws = decode_workspace(cfg, max_pos, tokens.device)
    if tokens.numel() < max_pos + 1:
        raise ValueError("tokens needs room for max_pos + 1 ids")
    cache = kv_cache_struct(cache_k, cache_v)
    _call("kvb_decode_step", C.byref(cfg), C.byref(model.struct), C.byref(rope.struct), C.byref(cache),
          _ptr(lm_head, torch.bfloat16, "lm_head"), _ptr(tokens, torch.int32, "tokens"), _ptr(pos, torch.int32, "pos"),
          max_pos, _ptr(hidden, torch.float32, "hidden"), _ptr(ws), ws.numel(), _stream())
    return ws


def decode_attention(cfg: Config, q: torch.Tensor, k_layer: torch.Tensor, v_layer: torch.Tensor, pos: torch.Tensor,
                     max_pos: int, out: Optional[torch.Tensor] = None, ws: Optional[torch.Tensor] = None):
    """Attention of one new row (q bf16 [Hq][D]) over cache rows [0, pos] of one layer
    (k bf16 / v fp16, [n_rows][Hkv][D]).  Returns bf16 [Hq][D]."""
    if out is None:
        out = torch.empty(cfg.n_q_heads, cfg.head_dim, dtype=torch.bfloat16, device=q.device)
    if ws is None:
        ws = decode_workspace(cfg, max_pos, q.device)
    _call("kvb_decode_attention", C.byref(cfg), _ptr(q, torch.bfloat16, "q"), _ptr(k_layer, torch.bfloat16, "k"),
          _ptr(v_layer, torch.float16, "v"), k_layer.shape[0], _ptr(pos, torch.int32, "pos"), max_pos,
          _ptr(out, torch.bfloat16, "out"), _ptr(ws), ws.numel(), _stream())
    return out
