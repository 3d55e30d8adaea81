"""Helpers shared by the GPU parity tests: error metrics and the tolerances.

Tolerances (float outputs are compared with the float64 oracle on the same
bf16-representable inputs):
  * layer outputs / final hidden states: max-abs <= 2e-2 and mean-abs <= 2e-3
    (the bar the method's specification states for bf16 outputs);
  * bf16 intermediates (q, k, v, realigned keys): errors are judged relative to
    the reference RMS, max <= 2e-2 * rms and mean <= 2e-3 * rms, i.e. the same bar
    applied to a unit-scale signal.  One bf16 rounding of the result alone
    contributes up to 2^-9 (0.2 %) relative per element.
  * tensors that both sides store in bf16 (q, k, v, caches, re-aligned keys):
    fp32 and fp64 accumulation can land on opposite sides of a bf16 rounding
    boundary, so single elements may differ by one bf16 ulp of the value (2^-7
    relative at most), and an input element rounded to the other side moves an
    output by |w| * ulp(input); the bar is |err| <= 2^-7 |ref| + 2e-2 rms
    elementwise and mean-abs <= 2e-3 rms.
  * attention outputs: the same bar relative to the RMS of V.  The output is a
    convex combination of value rows; rounding each softmax weight to bf16 (the
    P operand of the P.V product) perturbs it by at most 2^-9 * max|v - out|,
    which scales with the values, not with the (much smaller) RMS of the average.
"""
import numpy as np
import torch

MAX_ABS, MEAN_ABS = 2e-2, 2e-3


def fp64_gap_bounds(rms: float, n_layers: int) -> tuple:
    """Bound on the gap between the GPU path and the all-float64 oracle.

    The CUDA path holds five activations per layer in bf16 (the oracle's act_bf16
    mode rounds the same ones); each rounding is at most 2^-9 relative, RMS
    2^-9/sqrt(3), and the layer maps carry it into the residual with gain ~1, so
    the RMS gap after L layers is about 2^-9 * sqrt(5 L / 3) of the signal.  We
    allow mean-abs <= 2^-9 * sqrt(5 L) * rms and max-abs <= 8x that.
    """
    mean = 2.0 ** -9 * np.sqrt(5.0 * n_layers) * rms
    return 8.0 * mean, mean


def np64(t) -> np.ndarray:
    if isinstance(t, torch.Tensor):
        t = t.detach().to("cpu")
        if t.dtype in (torch.bfloat16, torch.float16):
            t = t.float()
        return t.numpy().astype(np.float64)
    return np.asarray(t, dtype=np.float64)


def errs(got, want) -> dict:
    g, w = np64(got), np64(want)
    assert g.shape == w.shape, (g.shape, w.shape)
    d = np.abs(g - w)
    rms = float(np.sqrt(np.mean(w * w))) if w.size else 0.0
    return {"max_abs": float(d.max()) if d.size else 0.0, "mean_abs": float(d.mean()) if d.size else 0.0,
            "rms_ref": rms}


def assert_close_abs(got, want, what="", max_abs=MAX_ABS, mean_abs=MEAN_ABS):
    e = errs(got, want)
    assert np.all(np.isfinite(np64(got))), f"{what}: non-finite values"
    assert e["max_abs"] <= max_abs and e["mean_abs"] <= mean_abs, f"{what}: {e}"
    return e


def assert_close_rel(got, want, what="", max_rel=MAX_ABS, mean_rel=MEAN_ABS, scale=None):
    e = errs(got, want)
    assert np.all(np.isfinite(np64(got))), f"{what}: non-finite values"
    s = max(e["rms_ref"] if scale is None else scale, 1e-30)
    assert e["max_abs"] <= max_rel * s and e["mean_abs"] <= mean_rel * s, f"{what}: {e}"
    return e


def assert_close_bf16(got, want, what="", mean_rel=MEAN_ABS):
    g, w = np64(got), np64(want)
    e = errs(g, w)
    assert np.all(np.isfinite(g)), f"{what}: non-finite values"
    s = max(e["rms_ref"], 1e-30)
    bad = np.abs(g - w) > 2.0 ** -7 * np.abs(w) + MAX_ABS * s
    assert not bad.any() and e["mean_abs"] <= mean_rel * s, f"{what}: {e}, {int(bad.sum())} elements over 1 ulp"
    return e


def bf16_round(a: np.ndarray) -> np.ndarray:
    return torch.from_numpy(np.asarray(a, dtype=np.float32)).to(torch.bfloat16).float().numpy().astype(np.float64)


def check_selection(sel_gpu, dev_ref, k, tie_rel=1e-3):
    """Selected indices must equal the oracle's top-k, except where the oracle's
    deviation is within tie_rel (relative) of its k-th largest value."""
    sel_gpu = np.sort(np.asarray(sel_gpu, dtype=np.int64))
    assert len(sel_gpu) == k and len(np.unique(sel_gpu)) == k
    if k == 0:
        return 0
    dev_ref = np.asarray(dev_ref, dtype=np.float64)
    order = np.lexsort((np.arange(len(dev_ref)), -dev_ref))
    want = np.sort(order[:k])
    kth = dev_ref[order[k - 1]]
    band = tie_rel * max(abs(kth), 1e-30)
    diff = np.setxor1d(sel_gpu, want)
    for i in diff:
        assert abs(dev_ref[i] - kth) <= band, f"index {i}: dev {dev_ref[i]} vs k-th {kth}"
    return len(diff)
