"""Seeded synthetic inputs for the selective-recompute prefill.

This module only draws numbers: model shapes, random weights, token ids and the
chunk layout of a request.  It holds none of the method's arithmetic, so that the
CUDA path and the CPU oracle can both be fed from it without sharing any code
that computes the method.

Workload recipe (stand-in for the paper's RULER HQA inputs, Sec. 4 and Tables
9-10: a long context made of retrieved documents of at most 512 tokens each,
followed by the question):

* token ids: uniform over the vocabulary;
* embedding table: N(0, 1), rounded to bf16;
* linear weights: N(0, 0.02), rounded to bf16 (so both sides read the same values);
* RMSNorm gains: 1.0;
* q/k/v projection bias (shapes that have one): N(0, 0.5^2), rounded to bf16, held as fp32;
* chunks of equal length laid end to end, then a query suffix;
* optionally two special tokens between consecutive documents (the last two ids of
  the vocabulary), whose rows of the concatenated cache are zero.

Every tensor is drawn from its own generator, seeded from (seed, layer, name), so
one layer can be regenerated without drawing the others.
"""
from __future__ import annotations

import dataclasses
from typing import Dict, List, Sequence

import torch

__all__ = [
    "ModelShape", "Workload", "SHAPES", "WORKLOADS", "tensor_seed", "shape_from_config",
    "make_layer_weights", "make_embed", "make_lm_head", "make_model", "make_tokens",
    "chunk_starts_equal", "separator_layout", "separator_ids", "randn_bf16",
]


@dataclasses.dataclass(frozen=True)
class ModelShape:
    """Decoder shape (hidden, heads, head dim, MLP dim, layers, RoPE).

    rope_scaling: 0 plain RoPE, 1 Llama 3.1 frequency scaling (rs_factor, low/high
    frequency factors rs_low/rs_high, original context rs_orig_ctx), 2 YaRN (scale
    rs_factor, ramp bounds alpha = rs_low and beta = rs_high, original context
    rs_orig_ctx).  qkv_bias: the q/k/v projections carry an additive bias."""
    hidden: int
    n_q_heads: int
    n_kv_heads: int
    head_dim: int
    mlp_dim: int
    n_layers: int
    vocab: int
    rms_eps: float = 1e-5
    rope_theta: float = 10000.0
    rope_scaling: int = 0
    rs_factor: float = 8.0
    rs_low: float = 1.0
    rs_high: float = 4.0
    rs_orig_ctx: int = 8192
    qkv_bias: bool = False

    @property
    def q_dim(self) -> int:
        return self.n_q_heads * self.head_dim

    @property
    def kv_dim(self) -> int:
        return self.n_kv_heads * self.head_dim

    @property
    def qkv_dim(self) -> int:
        return self.q_dim + 2 * self.kv_dim

    def with_layers(self, n_layers: int) -> "ModelShape":
        return dataclasses.replace(self, n_layers=n_layers)


@dataclasses.dataclass(frozen=True)
class Workload:
    """A request: `n_chunks` chunks of `chunk_len` tokens, a query suffix, ratio r.

    With n_sep > 0, n_sep special tokens sit between consecutive chunks (documents);
    their cache rows are zero in the concatenated cache."""
    name: str
    shape: ModelShape
    n_chunks: int
    chunk_len: int
    n_query: int
    r: float = 0.15
    check_layer: int = 1
    n_sep: int = 0

    @property
    def n_ctx(self) -> int:
        return self.n_chunks * self.chunk_len + max(self.n_chunks - 1, 0) * self.n_sep

    @property
    def n_total(self) -> int:
        return self.n_ctx + self.n_query

    def chunk_starts(self) -> List[int]:
        """Boundaries of every segment of the context (documents and separator groups), then n_ctx."""
        return separator_layout(self.n_chunks, self.chunk_len, self.n_sep)[0]

    def sep_starts(self) -> List[int]:
        """First row of each separator group."""
        return separator_layout(self.n_chunks, self.chunk_len, self.n_sep)[1]

    def sep_rows(self) -> List[int]:
        return [s + j for s in self.sep_starts() for j in range(self.n_sep)]

    def tokens(self, seed: int = 1, device: str | torch.device = "cpu") -> torch.Tensor:
        """Uniform token ids, with the separator ids at the separator rows."""
        t = make_tokens(self.shape, self.n_total, seed)
        ids = separator_ids(self.shape, self.n_sep)
        for s in self.sep_starts():
            for j, tok in enumerate(ids):
                t[s + j] = tok
        return t.to(device)


TINY = ModelShape(hidden=256, n_q_heads=4, n_kv_heads=2, head_dim=64, mlp_dim=688,
                  n_layers=2, vocab=1024, rms_eps=1e-5, rope_theta=10000.0)
LLAMA8B = ModelShape(hidden=4096, n_q_heads=32, n_kv_heads=8, head_dim=128, mlp_dim=14336,
                     n_layers=32, vocab=128256, rms_eps=1e-5, rope_theta=500000.0,
                     rope_scaling=1, rs_factor=8.0, rs_low=1.0, rs_high=4.0, rs_orig_ctx=8192)
# Seven query heads per kv head, YaRN scaling (factor 4 over an original context shorter
# than the workloads below, ramp between 1 and 32 turns) and a q/k/v bias: the features
# of the paper's second model family, at sizes chosen here (not that model's own).
YARN_GQA7_TINY = ModelShape(hidden=512, n_q_heads=7, n_kv_heads=1, head_dim=64, mlp_dim=1376,
                            n_layers=2, vocab=1024, rms_eps=1e-6, rope_theta=1000000.0,
                            rope_scaling=2, rs_factor=4.0, rs_low=1.0, rs_high=32.0, rs_orig_ctx=256,
                            qkv_bias=True)
YARN_GQA7 = ModelShape(hidden=1792, n_q_heads=14, n_kv_heads=2, head_dim=128, mlp_dim=4864,
                       n_layers=2, vocab=32768, rms_eps=1e-6, rope_theta=1000000.0,
                       rope_scaling=2, rs_factor=4.0, rs_low=1.0, rs_high=32.0, rs_orig_ctx=2048,
                       qkv_bias=True)

SHAPES: Dict[str, ModelShape] = {"tiny": TINY, "llama8b": LLAMA8B, "yarn_gqa7_tiny": YARN_GQA7_TINY,
                                 "yarn_gqa7": YARN_GQA7}

# The single-layer configurations are instantiated with two layers: layer 0 is the
# full-recompute layer and layer 1 the selective layer under test.
WORKLOADS: Dict[str, Workload] = {
    "tiny": Workload("tiny-2L-4x128+32", TINY, 4, 128, 32),
    "l8b_1layer": Workload("llama8b-2L-8x480+64", LLAMA8B.with_layers(2), 8, 480, 64),
    "l8b_32k": Workload("llama8b-32L-64x512+128", LLAMA8B, 64, 512, 128),
    "l8b_124k": Workload("llama8b-32L-242x512+128", LLAMA8B, 242, 512, 128),
    # the 64k-context request of the r x chunk-size sweep, at its largest chunks and r = 0.25
    "l8b_64k": Workload("llama8b-32L-32x2048+128", LLAMA8B, 32, 2048, 128, r=0.25),
    # two special tokens between documents, their cache rows zero
    "tiny_sep": Workload("tiny-2L-4x126+sep2+32", TINY, 4, 126, 32, n_sep=2),
    "l8b_1layer_sep": Workload("llama8b-2L-8x478+sep2+64", LLAMA8B.with_layers(2), 8, 478, 64, n_sep=2),
    "l8b_124k_sep": Workload("llama8b-32L-242x512+sep2+128", LLAMA8B, 242, 512, 128, n_sep=2),
    # YaRN RoPE, seven q heads per kv head, q/k/v bias
    "yarn_tiny": Workload("yarn-gqa7-tiny-2L-4x128+32", YARN_GQA7_TINY, 4, 128, 32),
    "yarn_2l": Workload("yarn-gqa7-2L-8x480+64", YARN_GQA7, 8, 480, 64),
    "yarn_124k": Workload("yarn-gqa7-32L-242x512+128", YARN_GQA7.with_layers(32), 242, 512, 128),
}


def shape_from_config(cfg: dict) -> ModelShape:
    """A ModelShape from a model configuration in the common JSON layout of published
    decoder checkpoints (hidden_size, num_attention_heads, num_key_value_heads,
    intermediate_size, num_hidden_layers, vocab_size, rms_norm_eps, rope_theta and an
    optional rope_scaling block of type "llama3" or "yarn").  The q/k/v bias is taken from
    "attention_bias" when present, else from a "qkv_bias" key (False if neither).  YaRN's
    ramp bounds default to alpha = 1, beta = 32 when the block does not give them."""
    H = int(cfg["hidden_size"])
    Hq = int(cfg["num_attention_heads"])
    Hkv = int(cfg.get("num_key_value_heads", Hq))
    D = int(cfg.get("head_dim") or H // Hq)
    kw = {}
    rs = cfg.get("rope_scaling") or {}
    kind = (rs.get("rope_type") or rs.get("type") or "default").lower()
    if kind == "llama3":
        kw = dict(rope_scaling=1, rs_factor=float(rs["factor"]), rs_low=float(rs["low_freq_factor"]),
                  rs_high=float(rs["high_freq_factor"]), rs_orig_ctx=int(rs["original_max_position_embeddings"]))
    elif kind == "yarn":
        kw = dict(rope_scaling=2, rs_factor=float(rs["factor"]), rs_low=float(rs.get("beta_slow", 1.0)),
                  rs_high=float(rs.get("beta_fast", 32.0)), rs_orig_ctx=int(rs["original_max_position_embeddings"]))
    elif kind not in ("default", "none"):
        raise ValueError(f"rope_scaling type {kind!r} is not supported")
    bias = bool(cfg.get("attention_bias", cfg.get("qkv_bias", False)))
    return ModelShape(hidden=H, n_q_heads=Hq, n_kv_heads=Hkv, head_dim=D, mlp_dim=int(cfg["intermediate_size"]),
                      n_layers=int(cfg["num_hidden_layers"]), vocab=int(cfg["vocab_size"]),
                      rms_eps=float(cfg.get("rms_norm_eps", 1e-5)), rope_theta=float(cfg.get("rope_theta", 10000.0)),
                      qkv_bias=bias, **kw)


def tensor_seed(seed: int, layer: int, name: str) -> int:
    """Deterministic 63-bit seed for one tensor (FNV-1a over the identifiers)."""
    h = 0xCBF29CE484222325
    for b in f"{seed}/{layer}/{name}".encode():
        h ^= b
        h = (h * 0x100000001B3) & 0xFFFFFFFFFFFFFFFF
    return h & 0x7FFFFFFFFFFFFFFF


def randn_bf16(shape: Sequence[int], seed: int, std: float = 1.0,
               device: str | torch.device = "cpu") -> torch.Tensor:
    """N(0, std^2) drawn in fp32 from a generator on `device`, rounded to bf16."""
    g = torch.Generator(device=device)
    g.manual_seed(seed)
    t = torch.randn(*shape, generator=g, device=device, dtype=torch.float32)
    if std != 1.0:
        t.mul_(std)
    return t.to(torch.bfloat16)


LAYER_TENSORS = ("w_qkv", "w_o", "w_gate", "w_up", "w_down")


def make_layer_weights(shape: ModelShape, layer: int, seed: int = 0,
                       device: str | torch.device = "cpu") -> Dict[str, torch.Tensor]:
    """One decoder layer: bf16 matrices (out_features x in_features), fp32 gains and,
    for shapes with one, the fp32 q/k/v bias `b_qkv` [qkv_dim].

    w_qkv rows are [q heads | k heads | v heads], each head `head_dim` rows.
    """
    H, F = shape.hidden, shape.mlp_dim
    dims = {
        "w_qkv": (shape.qkv_dim, H),
        "w_o": (H, shape.q_dim),
        "w_gate": (F, H),
        "w_up": (F, H),
        "w_down": (H, F),
    }
    w = {n: randn_bf16(dims[n], tensor_seed(seed, layer, n), 0.02, device) for n in LAYER_TENSORS}
    if shape.qkv_bias:
        w["b_qkv"] = randn_bf16((shape.qkv_dim,), tensor_seed(seed, layer, "b_qkv"), 0.5, device).float()
    w["attn_norm"] = torch.ones(H, dtype=torch.float32, device=device)
    w["mlp_norm"] = torch.ones(H, dtype=torch.float32, device=device)
    return w


def make_embed(shape: ModelShape, seed: int = 0, device: str | torch.device = "cpu") -> torch.Tensor:
    return randn_bf16((shape.vocab, shape.hidden), tensor_seed(seed, -1, "embed"), 1.0, device)


def make_lm_head(shape: ModelShape, seed: int = 0, device: str | torch.device = "cpu") -> torch.Tensor:
    """Output projection [vocab][hidden], N(0, 0.02) rounded to bf16."""
    return randn_bf16((shape.vocab, shape.hidden), tensor_seed(seed, -3, "lm_head"), 0.02, device)


def make_model(shape: ModelShape, seed: int = 0, device: str | torch.device = "cpu") -> dict:
    return {
        "layers": [make_layer_weights(shape, l, seed, device) for l in range(shape.n_layers)],
        "embed": make_embed(shape, seed, device),
        "final_norm": torch.ones(shape.hidden, dtype=torch.float32, device=device),
    }


def make_tokens(shape: ModelShape, n: int, seed: int = 1, device: str | torch.device = "cpu") -> torch.Tensor:
    g = torch.Generator(device="cpu")
    g.manual_seed(tensor_seed(seed, -2, "tokens"))
    return torch.randint(0, shape.vocab, (n,), generator=g, dtype=torch.int64).to(torch.int32).to(device)


def chunk_starts_equal(n_chunks: int, chunk_len: int) -> List[int]:
    return [c * chunk_len for c in range(n_chunks + 1)]


def separator_layout(n_chunks: int, chunk_len: int, n_sep: int):
    """Documents of chunk_len tokens with n_sep special tokens between consecutive ones.
    Returns (segment boundaries ending with n_ctx, first row of each separator group)."""
    starts, seps, pos = [0], [], 0
    for c in range(n_chunks):
        pos += chunk_len
        starts.append(pos)
        if c + 1 < n_chunks and n_sep > 0:
            seps.append(pos)
            pos += n_sep
            starts.append(pos)
    return starts, seps


def separator_ids(shape: ModelShape, n_sep: int) -> List[int]:
    """Token ids of the special separator tokens: the last n_sep ids of the vocabulary."""
    return [shape.vocab - n_sep + j for j in range(n_sep)]

