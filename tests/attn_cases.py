"""Attention inputs whose outputs expose a wrong key range, and the bar they are judged by.

Random N(0,1) queries and keys give logits of standard deviation 1, so over thousands of
keys the softmax is nearly uniform and the output is an average far smaller than the
values; a key wrongly taken in or left out then moves the output by less than rounding.
The "tagged" case here makes each (row, head) look for one chosen key instead:

  * key t holds the base-b digits of t (b = D/4, four digits, unique for t < b^4: 65,536
    at D = 64, 1,048,576 at D = 128) as four one-hot groups of b dims, each set to KAPPA_K;
  * query (r, h) holds the digits of its target key c as one-hot groups set to KAPPA_Q;
  * so q.k_t = KAPPA_K * KAPPA_Q * (number of digits t shares with c), and with the logit
    scale 1/sqrt(D) every shared digit is worth about 8 in the exponent: the target key,
    when the row may read it, carries ~96 % of the softmax mass, and a key sharing three
    digits e^-8 of it.  All entries are small multiples of powers of two, so the GPU's
    bf16 operands and the oracle hold the same values and the logits are exact.

Values are random per key, so the output of (r, h) is essentially the value row of its
target: a target the row may not read (hi + 1, lo - 1) gives an average of near matches
instead, and a dropped key tile or an off-by-one mask changes the output completely.
Targets are spread over the kinds below so that every boundary a kernel handles (the
row's own key, the first key of its range, the edges of the 144-key tiles) is someone's
target.  The same construction serves the GPU parity tests and the CPU check that a
planted slip in the expectation fails the bar.
"""
import numpy as np
import torch

KAPPA_K, KAPPA_Q = 8.0, 11.25        # bf16-exact; product 90, times 1/sqrt(128) = 7.95 per digit
TILE = 144                           # key tile of the prefill attention kernel
MAX_REL, MEAN_REL = 2e-2, 2e-3       # the stated bar, relative to the output's own RMS

KINDS = ("hi", "hi+1", "lo", "lo-1", "tile_start", "prev_tile_end", "hi-tile", "random")


def digits(t: np.ndarray, base: int) -> np.ndarray:
    t = np.asarray(t, dtype=np.int64)
    return np.stack([(t // base ** j) % base for j in range(4)], axis=-1)


def onehot_digits(t: np.ndarray, D: int, kappa: float) -> np.ndarray:
    """[..., D] float32 with the four digits of t one-hot in groups of D/4."""
    base = D // 4
    dg = digits(t, base)
    out = np.zeros(dg.shape[:-1] + (D,), dtype=np.float32)
    idx = np.arange(4) * base + dg
    np.put_along_axis(out.reshape(-1, D), idx.reshape(-1, 4), kappa, axis=1)
    return out


def targets(hi: np.ndarray, lo: np.ndarray, Hq: int, n_kv: int, seed: int) -> np.ndarray:
    """Target key per (row, head), int64 [m, Hq]; head h of row r takes kind (r + h) % len(KINDS)."""
    rng = np.random.default_rng(seed)
    m = len(hi)
    c = np.empty((m, Hq), dtype=np.int64)
    for h in range(Hq):
        kind = (np.arange(m) + h) % len(KINDS)
        ts = (hi // TILE) * TILE                        # first key of the tile that holds hi
        choices = np.stack([
            hi, hi + 1, lo, lo - 1, np.maximum(ts, lo), np.maximum(ts - 1, lo),
            np.maximum(hi - TILE, lo), lo + (rng.random(m) * (hi - lo + 1)).astype(np.int64)], axis=1)
        c[:, h] = choices[np.arange(m), kind]
    # a target outside [0, n_kv) names no key at all (the row sees only near matches)
    return np.where((c >= 0) & (c < n_kv), c, n_kv + 7)


def tagged_case(n_kv: int, hi, lo, Hq: int, Hkv: int, D: int, seed: int = 0):
    """q [m, Hq, D] bf16, k [n_kv, Hkv, D] bf16, v [n_kv, Hkv, D] (bf16 values, returned as
    bf16) and the targets.  Every kv head holds the same digit keys; values differ."""
    hi = np.asarray(hi, dtype=np.int64)
    lo = np.zeros_like(hi) if lo is None else np.asarray(lo, dtype=np.int64)
    tg = targets(hi, lo, Hq, n_kv, seed)
    q = torch.from_numpy(onehot_digits(tg, D, KAPPA_Q)).to(torch.bfloat16)
    kk = onehot_digits(np.arange(n_kv), D, KAPPA_K)
    k = torch.from_numpy(np.repeat(kk[:, None, :], Hkv, axis=1)).to(torch.bfloat16)
    g = torch.Generator().manual_seed(seed + 1)
    v = torch.randn(n_kv, Hkv, D, generator=g).to(torch.bfloat16)
    return q, k, v, tg


def peaked_queries(m: int, Hq: int, D: int, seed: int, logit_std: float = 5.0) -> torch.Tensor:
    """Random queries scaled so that, against N(0,1) keys, the logits have standard deviation
    `logit_std` (a peaked softmax rather than a near-uniform average)."""
    g = torch.Generator().manual_seed(seed)
    return (torch.randn(m, Hq, D, generator=g) * logit_std).to(torch.bfloat16)


def _f64(a) -> np.ndarray:
    if isinstance(a, torch.Tensor):
        return a.detach().cpu().float().numpy().astype(np.float64)
    return np.asarray(a, dtype=np.float64)


def attn_errors(got, want) -> dict:
    g, w = _f64(got), _f64(want)
    d = np.abs(g - w)
    rms = float(np.sqrt(np.mean(w * w))) if w.size else 0.0
    return {"max_abs": float(d.max()) if d.size else 0.0, "mean_abs": float(d.mean()) if d.size else 0.0,
            "rms_out": rms}


def assert_attn_close(got, want, what: str = "") -> dict:
    """The stated bar relative to the attention output's own RMS: every element within
    2e-2 rms + 2^-7 |want| (the second term is one bf16 ulp of the value: the output is
    stored in bf16) and mean-abs <= 2e-3 rms."""
    e = attn_errors(got, want)
    g, w = _f64(got), _f64(want)
    assert np.all(np.isfinite(g)), f"{what}: non-finite values"
    s = max(e["rms_out"], 1e-30)
    bad = np.abs(g - w) > MAX_REL * s + 2.0 ** -7 * np.abs(w)
    assert not bad.any() and e["mean_abs"] <= MEAN_REL * s, f"{what}: {e}, {int(bad.sum())} elements over the bar"
    return e
