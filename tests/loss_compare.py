"""Tolerances of the GPU loss against the oracle, written once for every loss test.

  logp      |gpu - oracle| <= 2e-5 (absolute)
  loss      |gpu - oracle| <= 1e-5 * |oracle| + 1e-12
  dlogits   bf16: within 1 ulp (ordered-integer distance, +0 == -0); f32: |diff| <= 1e-6
Rows whose ratio lies within 1e-5 (relative) of a clip boundary may take either branch; their
dlogits and loss terms are not compared, and they are counted.
"""
import numpy as np

from helpers import bf16_ulp_distance

LOGP_ATOL = 2e-5
LOSS_RTOL = 1e-5
LOSS_ATOL = 1e-12
F32_ATOL = 1e-6
BF16_ULPS = 1


def boundary_rows(rho, eps_low, eps_high):
    lo, hi = 1.0 - np.float64(np.float32(eps_low)), 1.0 + np.float64(np.float32(eps_high))
    return (np.abs(rho - lo) <= 1e-5 * lo) | (np.abs(rho - hi) <= 1e-5 * hi)


def compare(gpu_logp, gpu_dlogits, gpu_loss, ref, dlogits_dtype, eps_low=0.2, eps_high=0.2,
            gpu_row_loss=None, rows=None):
    """ref: the oracle's dict.  gpu_dlogits: uint16 bf16 bits or float32, [n, V].  rows: which
    oracle rows the GPU arrays correspond to (default: all, in order)."""
    o_logp = ref["logp"] if rows is None else ref["logp"][rows]
    o_rho = ref["rho"] if rows is None else ref["rho"][rows]
    valid = ~np.isnan(o_logp)
    assert np.all(np.isnan(gpu_logp[~valid]))
    err = np.abs(gpu_logp[valid].astype(np.float64) - o_logp[valid])
    assert err.max(initial=0.0) <= LOGP_ATOL, "logp max abs err %g" % err.max()
    skip = boundary_rows(o_rho, eps_low, eps_high) & valid
    keep_rows = ~skip
    o_d = ref["dlogits"] if rows is None else ref["dlogits"][rows]
    if dlogits_dtype == "bf16":
        dist = bf16_ulp_distance(gpu_dlogits[keep_rows], o_d[keep_rows])
        worst = int(dist.max(initial=0))
        assert worst <= BF16_ULPS, "dlogits bf16 max ulp distance %d" % worst
    else:
        diff = np.abs(gpu_dlogits[keep_rows].astype(np.float64) - o_d[keep_rows].astype(np.float64))
        worst = float(diff.max(initial=0.0))
        assert worst <= F32_ATOL, "dlogits f32 max abs err %g" % worst
    if gpu_row_loss is not None:
        o_rl = ref["row_loss"] if rows is None else ref["row_loss"][rows]
        d = np.abs(gpu_row_loss[keep_rows] - o_rl[keep_rows])
        assert np.all(d <= LOSS_RTOL * np.abs(o_rl[keep_rows]) + 1e-9 * np.abs(o_rl).max(initial=0) + LOSS_ATOL)
    if gpu_loss is not None and not skip.any():
        assert abs(gpu_loss - ref["loss"]) <= LOSS_RTOL * abs(ref["loss"]) + LOSS_ATOL, \
            "loss %r vs oracle %r" % (gpu_loss, ref["loss"])
    return dict(worst=worst, boundary_rows=int(skip.sum()), logp_err=float(err.max(initial=0.0)))
