"""The CPU baseline's cost model (bench.py): how the oracle's time on a bounded sample is
scaled to the whole prefill (CPU only, no oracle timing).

The oracle's attention scores each block of consecutive rows against the union of the
rows' key ranges, so its work is counted block by block in (row, key) pairs; the rest of
a layer costs the same per row.  These tests pin the counting to hand-counted cases and to
the oracle's own block size, and the extrapolation to its two stated parts.
"""
import inspect
from types import SimpleNamespace

import numpy as np
import pytest

import bench
from oracle import llama


def test_block_size_is_the_oracles():
    assert bench.ORACLE_BLOCK == inspect.signature(llama.attention_rows).parameters["block"].default


def test_attention_work_hand_counted():
    # one row: its own key range
    assert bench.oracle_attention_work([7]) == 8
    assert bench.oracle_attention_work([7], [3]) == 5
    # ten causal rows in blocks of 4: 4 x 4 + 4 x 8 + 2 x 10
    assert bench.oracle_attention_work(np.arange(10), block=4) == 16 + 32 + 20
    # a block is scored against the union of its rows' ranges, not each row's own
    assert bench.oracle_attention_work([5, 100], [0, 90], block=2) == 2 * 101
    assert bench.oracle_attention_work([5, 100], [0, 90], block=1) == 6 + 11


def test_attention_work_is_additive_over_blocks():
    rng = np.random.default_rng(0)
    hi = np.sort(rng.integers(0, 5000, 1000))
    whole = bench.oracle_attention_work(hi, block=256)
    parts = sum(bench.oracle_attention_work(hi[b:b + 256], block=256) for b in range(0, len(hi), 256))
    assert whole == parts


def _wl(N, n_ctx, L):
    return SimpleNamespace(n_total=N, n_ctx=n_ctx, n_query=N - n_ctx, shape=SimpleNamespace(n_layers=L))


def test_ttft_model_per_row_part():
    wl = _wl(N=1000, n_ctx=900, L=4)
    smp = SimpleNamespace(n_rows=10, work=1.0)
    k = 90
    # 2 s for 10 sample rows -> 0.2 s per row-layer, over N + (L - 1)(k + n_query) row-layers
    got = bench.oracle_ttft_ms(wl, smp, 2.0, 0.0, k)
    assert got == pytest.approx(0.2 * (1000 + 3 * (90 + 100)) * 1e3)


def test_ttft_model_attention_part():
    wl = _wl(N=1000, n_ctx=900, L=4)
    smp = SimpleNamespace(n_rows=10, work=5000.0)
    sel = np.array([3, 50, 400, 899])
    rows = np.concatenate([sel, np.arange(900, 1000)])
    expect_work = bench.oracle_attention_work(np.arange(1000)) + 3 * bench.oracle_attention_work(rows)
    got = bench.oracle_ttft_ms(wl, smp, 0.0, 1.0, len(sel), sel=sel)
    assert got == pytest.approx(1.0 / 5000.0 * expect_work * 1e3)
    # the selection's order does not matter (the oracle takes rows in ascending order)
    assert bench.oracle_ttft_ms(wl, smp, 0.0, 1.0, len(sel), sel=sel[::-1]) == pytest.approx(got)


def test_ttft_model_without_a_selection_spreads_rows_uniformly():
    wl = _wl(N=1000, n_ctx=900, L=2)
    smp = SimpleNamespace(n_rows=10, work=1.0)
    k = 90
    spread = np.linspace(0, 899, num=k).round().astype(np.int64)
    assert bench.oracle_ttft_ms(wl, smp, 0.0, 1.0, k) == pytest.approx(
        bench.oracle_ttft_ms(wl, smp, 0.0, 1.0, k, sel=spread))
