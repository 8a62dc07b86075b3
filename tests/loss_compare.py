"""Tolerances of the GPU loss against the oracle, written once for every loss test.

  logp      |gpu - oracle| <= 2e-5 (absolute)
  loss      |gpu - oracle| <= 1e-5 * |oracle| + 1e-12; each row's term w_t l_t likewise, plus,
            given `cond`, w_t times the error its logp error carries into l_t (d l_t / d logp =
            g_t) and f32 rounding of l_t's terms: a row whose l_t is the KL term alone (A = 0)
            is tiny and cancels in f32
  dlogits   bf16: within 1 ulp (ordered-integer distance, +0 == -0); f32: |diff| <= 1e-6
Rows whose ratio lies within 1e-5 (relative) of a clip boundary may take either branch; their
dlogits and loss terms are not compared, and they are counted.  The loss is then compared as the
sum of every other row's term on both sides (which needs the GPU's per-row terms); the check is
never dropped.

A row's dlogits are w_t * g_t * (onehot(y) - softmax), with g_t = -(c*rho*A + beta*(e^x - 1)),
x = ref_logp - logp (Eq. 3; GSPO: the sequence ratio s in place of rho).  Where the two terms of
g_t nearly cancel (for instance A = 0 and ref_logp close to logp), the error that the logp
tolerance allows is amplified in g_t's relative error, and one bf16 ulp is not reachable from an
f32 log-probability.  Given the inputs (`cond`), such rows get the ulps that the log-probability
errors propagate into g_t: |c rho A| * e_ratio + beta e^x * e over |g_t|, with e the row's own
logp error and e_ratio the error of log(rho) (the row's e; for GSPO the largest e of its
sequence), plus f32 rounding of g_t's terms; every other row keeps the 1-ulp bar.  Those rows are
counted.
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


def row_loss_slack(gpu_logp, ref, cond, rows=None):
    """Per row, the absolute error that the row's log-probability error and f32 rounding allow
    its loss term w_t l_t beyond the relative bar (module docstring: d l_t / d logp = g_t).  It
    matters where the KL term alone makes up l_t (A = 0): beta (e^x - x - 1) is then tiny and
    cancels in f32.  Zero without `cond` or without the oracle's weights."""
    o_logp = ref["logp"] if rows is None else ref["logp"][rows]
    if cond is None or "w" not in ref:
        return np.zeros(o_logp.size)
    g = ref["g"] if rows is None else ref["g"][rows]
    w = ref["w"] if rows is None else ref["w"][rows]
    rl = ref["row_loss"] if rows is None else ref["row_loss"][rows]
    beta = float(np.float32(cond["beta"]))
    x = np.asarray(cond["ref_logp"], np.float64) - o_logp
    em1 = np.expm1(x)
    u = np.abs(-g - beta * em1)  # |c rho A|
    e = np.abs(np.asarray(gpu_logp, np.float64) - o_logp) + 2.0 ** -24 * np.abs(o_logp)
    e_r = np.asarray(cond["e_ratio"], np.float64) if "e_ratio" in cond else e
    with np.errstate(invalid="ignore", divide="ignore"):
        ell = np.abs(rl) / w
        prop = u * e_r + beta * (np.abs(em1) * e + np.exp(x) * e * e)
        rnd = 2.0 ** -22 * (ell + 2.0 * beta * (np.abs(em1) + np.abs(x)))
        s = w * (prop + rnd)
    return np.where(np.isfinite(s), s, 0.0)


def compare_rows(gpu_logp, gpu_loss, gpu_row_loss, ref, eps_low=0.2, eps_high=0.2, rows=None,
                 cond=None):
    """logp of every row, the per-row loss terms (when given) and the total loss against the
    oracle's dict.  Returns (valid rows, rows compared, boundary rows skipped, max logp error)."""
    o_logp = ref["logp"] if rows is None else ref["logp"][rows]
    o_rho = ref["rho"] if rows is None else ref["rho"][rows]
    valid = ~np.isnan(o_logp)
    assert np.all(np.isnan(gpu_logp[~valid]))
    err = np.abs(gpu_logp[valid].astype(np.float64) - o_logp[valid])
    assert err.max(initial=0.0) <= LOGP_ATOL, "logp max abs err %g" % err.max()
    skip = boundary_rows(o_rho, eps_low, eps_high) & valid
    keep_rows = ~skip
    o_rl = None
    if gpu_row_loss is not None:
        o_rl = ref["row_loss"] if rows is None else ref["row_loss"][rows]
        slack = row_loss_slack(gpu_logp, ref, cond, rows)
        d = np.abs(gpu_row_loss[keep_rows] - o_rl[keep_rows])
        bar = (LOSS_RTOL * np.abs(o_rl[keep_rows]) + 1e-9 * np.abs(o_rl).max(initial=0)
               + LOSS_ATOL + slack[keep_rows])
        assert np.all(d <= bar), "row loss: %d rows beyond their bar (worst %g at bar %g)" % (
            int((d > bar).sum()), d.max(initial=0), bar[d.argmax()] if d.size else 0)
    n_skip = int(skip.sum())
    if gpu_loss is not None:
        if n_skip == 0:
            assert abs(gpu_loss - ref["loss"]) <= LOSS_RTOL * abs(ref["loss"]) + LOSS_ATOL, \
                "loss %r vs oracle %r" % (gpu_loss, ref["loss"])
        else:
            # both sums without the boundary rows' terms; the GPU's total is its terms' sum
            assert gpu_row_loss is not None, \
                "%d rows sit at a clip boundary: pass the GPU's per-row terms" % n_skip
            g_all = float(np.sum(gpu_row_loss))
            assert abs(gpu_loss - g_all) <= 1e-12 * np.abs(gpu_row_loss).sum() + LOSS_ATOL
            g_part = float(np.sum(gpu_row_loss[keep_rows]))
            o_part = float(np.sum(o_rl[keep_rows]))
            assert abs(g_part - o_part) <= LOSS_RTOL * abs(o_part) + LOSS_ATOL, \
                "loss without %d boundary rows %r vs oracle %r" % (n_skip, g_part, o_part)
            print("loss compared without %d clip-boundary rows" % n_skip)
    return keep_rows, n_skip, float(err.max(initial=0.0))


def allowed_ulps(gpu_logp, ref, cond, rows=None):
    """Per row, the bf16 ulps its dlogits may differ by (1 unless g_t is ill-conditioned, see the
    module docstring).  cond = dict(ref_logp=the rows' ref_logp inputs, beta=beta)."""
    o_logp = ref["logp"] if rows is None else ref["logp"][rows]
    g = ref["g"] if rows is None else ref["g"][rows]
    n = o_logp.size
    if cond is None:
        return np.full(n, BF16_ULPS)
    beta = float(np.float32(cond["beta"]))
    x = np.asarray(cond["ref_logp"], np.float64) - o_logp
    ex = np.exp(x)
    u = np.abs(-g - beta * (ex - 1))  # |c rho A|: g's clipped-surrogate term
    k = beta * ex                      # beta e^x: its KL term's derivative
    e = np.abs(np.asarray(gpu_logp, np.float64) - o_logp) + 2.0 ** -24 * np.abs(o_logp)
    e_r = np.asarray(cond["e_ratio"], np.float64) if "e_ratio" in cond else e
    with np.errstate(divide="ignore", invalid="ignore"):
        rel = e + (u * e_r + k * e + 2.0 ** -22 * (u + k)) / np.abs(g) + 1e-5
    n_ulp = np.where(np.isfinite(rel), np.ceil(rel * 256.0), BF16_ULPS)  # ulp >= 2^-8 relative
    n_ulp = np.where(g == 0, BF16_ULPS, n_ulp)
    return np.maximum(BF16_ULPS, n_ulp).astype(np.int64)


def compare(gpu_logp, gpu_dlogits, gpu_loss, ref, dlogits_dtype, eps_low=0.2, eps_high=0.2,
            gpu_row_loss=None, rows=None, cond=None):
    """ref: the oracle's dict.  gpu_dlogits: uint16 bf16 bits or float32, [n, V].  rows: which
    oracle rows the GPU arrays correspond to (default: all, in order).  cond: the rows'
    ref_logp inputs and beta, for the conditioning of g_t (module docstring)."""
    keep_rows, n_skip, logp_err = compare_rows(gpu_logp, gpu_loss, gpu_row_loss, ref, eps_low,
                                               eps_high, rows, cond)
    o_d = ref["dlogits"] if rows is None else ref["dlogits"][rows]
    n_wide = 0
    if dlogits_dtype == "bf16":
        k = allowed_ulps(gpu_logp, ref, cond, rows)
        dist = bf16_ulp_distance(gpu_dlogits[keep_rows], o_d[keep_rows])
        row_worst = dist.max(axis=1, initial=0) if dist.ndim == 2 else dist
        worst = int(row_worst.max(initial=0))
        bad = row_worst > k[keep_rows]
        assert not bad.any(), "dlogits bf16: %d rows beyond their bar (worst %d ulps, bar %s)" % (
            int(bad.sum()), worst, k[keep_rows][bad][:5])
        n_wide = int((k[keep_rows] > BF16_ULPS).sum())
        if n_wide:
            print("dlogits: %d rows with an ill-conditioned g_t, bar up to %d ulps; worst %d"
                  % (n_wide, int(k.max()), worst))
    else:
        diff = np.abs(gpu_dlogits[keep_rows].astype(np.float64) - o_d[keep_rows].astype(np.float64))
        worst = float(diff.max(initial=0.0))
        assert worst <= F32_ATOL, "dlogits f32 max abs err %g" % worst
    return dict(worst=worst, boundary_rows=n_skip, logp_err=logp_err, widened_rows=n_wide)
