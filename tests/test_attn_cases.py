"""The attention parity cases can fail: on the CPU, with the oracle as the expectation, a
slip planted in a copy of the key-range predicate (the row's own key left out, the next
key taken in, the key before a block-diagonal range taken in) or one key tile left out
moves the tagged-key outputs far beyond the bar the GPU tests apply, while a computation
with the kernel's own roundings (fp32 logits and sums, fp16 softmax weights, a bf16
output) stays well inside it."""
import numpy as np
import pytest
import torch

from oracle import llama
from oracle.llama import Shape
from paper_2609_09768_gb300 import synth
from tests.attn_cases import TILE, assert_attn_close, tagged_case

SHAPE = synth.ModelShape(hidden=256, n_q_heads=8, n_kv_heads=2, head_dim=128, mlp_dim=256, n_layers=1, vocab=16,
                         rms_eps=1e-5, rope_theta=10000.0)
N_KV = 700


def _rows():
    """Rows whose own key sits on every residue of a 144-key tile, plus a few more."""
    hi = np.unique(np.concatenate([np.arange(2 * TILE, 3 * TILE), [0, 1, 143, 144, 287, 599, N_KV - 1]]))
    return hi


def _case(block_diag: bool):
    hi = _rows()
    lo = (hi // 230) * 230 if block_diag else np.zeros_like(hi)     # ragged, not tile-aligned chunk starts
    q, k, v, tg = tagged_case(N_KV, hi, lo, SHAPE.n_q_heads, SHAPE.n_kv_heads, SHAPE.head_dim, seed=3)
    s = Shape.of(SHAPE)
    qn, kn, vn = (t.float().numpy().astype(np.float64) for t in (q, k, v))
    return s, qn, kn, vn, hi, lo


def _oracle(s, q, k, v, hi, lo):
    return llama.attention_rows(s, q, k, v, hi, lo).reshape(len(hi), -1)


def _kernel_like(s, q, k, v, hi, lo):
    """The kernel's roundings on the same inputs: fp32 logits and sums, softmax weights
    rounded to fp16, output rounded to bf16 (no blocking: only the roundings differ)."""
    m, Hq, D = q.shape
    G = Hq // k.shape[1]
    out = np.zeros((m, Hq, D), dtype=np.float32)
    scale = np.float32(llama.logit_scale(s))
    for r in range(m):
        t = np.arange(lo[r], hi[r] + 1)
        for h in range(Hq):
            sc = (q[r, h].astype(np.float32) @ k[t, h // G].astype(np.float32).T) * scale
            p = np.exp(sc - sc.max()).astype(np.float16).astype(np.float32)
            out[r, h] = (p @ v[t, h // G].astype(np.float32)) / p.astype(np.float32).sum()
    return torch.from_numpy(out.reshape(m, -1)).to(torch.bfloat16).float().numpy()


@pytest.mark.parametrize("block_diag", [False, True])
def test_kernel_roundings_pass_the_bar(block_diag):
    s, q, k, v, hi, lo = _case(block_diag)
    assert_attn_close(_kernel_like(s, q, k, v, hi, lo), _oracle(s, q, k, v, hi, lo), "kernel-like roundings")


@pytest.mark.parametrize("block_diag", [False, True])
def test_planted_key_range_slips_fail_the_bar(block_diag):
    s, q, k, v, hi, lo = _case(block_diag)
    want = _oracle(s, q, k, v, hi, lo)
    slips = {
        "next key taken in": (np.minimum(hi + 1, N_KV - 1), lo),
        "own key left out": (np.maximum(hi - 1, lo), lo),
    }
    if block_diag:
        slips["key before the range taken in"] = (hi, np.maximum(lo - 1, 0))
    for name, (h2, l2) in slips.items():
        with pytest.raises(AssertionError):
            assert_attn_close(_oracle(s, q, k, v, h2, l2), want, name)
    # one key tile left out: its keys can match nothing (logit 0, e^-32 of the target's weight)
    k_drop = k.copy()
    k_drop[2 * TILE: 3 * TILE] = 0.0
    with pytest.raises(AssertionError):
        assert_attn_close(_oracle(s, q, k_drop, v, hi, lo), want, "tile 2 left out")


def test_target_key_carries_the_mass():
    """Each (row, head) whose target lies in its range reads essentially that key's value:
    the output is within 5 % of V[target] (the near matches share the rest)."""
    s, q, k, v, hi, lo = _case(False)
    hi_ = np.asarray(hi)
    _, _, _, tg = tagged_case(N_KV, hi, lo, SHAPE.n_q_heads, SHAPE.n_kv_heads, SHAPE.head_dim, seed=3)
    out = _oracle(s, q, k, v, hi, lo).reshape(len(hi), SHAPE.n_q_heads, -1)
    G = SHAPE.n_q_heads // SHAPE.n_kv_heads
    n_in = 0
    for r in range(len(hi_)):
        for h in range(SHAPE.n_q_heads):
            c = tg[r, h]
            if lo[r] <= c <= hi_[r]:
                n_in += 1
                vv = v[c, h // G]
                assert np.abs(out[r, h] - vv).max() <= 0.05 * np.abs(vv).max() + 0.05, (r, h, c)
    assert n_in > len(hi_) * SHAPE.n_q_heads // 2
