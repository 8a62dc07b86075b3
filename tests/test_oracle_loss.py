"""Pins of the oracle's GRPO loss and dlogits (Eqs. 1-3): hand-worked tokens, a library
log-sum-exp, finite differences of the loss, and invariants of the gradient."""
import math

import numpy as np
import pytest
import scipy.special

from helpers import golden


def one_token(oracle_mod, case, **kw):
    z = np.asarray(case["z"], np.float32)[None, :]
    return oracle_mod.loss(z, case["V"], [case["y"]], [case["old_logp"]], [case["ref_logp"]],
                           [case["A"]], [0], eps_low=case["eps"], eps_high=case["eps"],
                           beta=case["beta"], denom_tokens=1, want_f64=True, **kw)


def test_hand_worked(oracle_mod):
    for case in golden("loss_hand.json")["cases"]:
        out = one_token(oracle_mod, case)
        msg = case["name"] + ": " + case["derivation"]
        assert out["logp"][0] == pytest.approx(case["logp"], abs=1e-7), msg
        if case["name"].startswith("ratio at the upper boundary"):
            # rho lands on 1+eps up to one rounding: the indicator follows the computed rho
            unclipped = out["rho"][0] <= 1.0 + case["eps"]
            expect = case["dlogits"] if unclipped else [0.0, 0.0]
            np.testing.assert_allclose(out["dlogits_f64"][0], expect, atol=1e-6, err_msg=msg)
            continue
        assert out["loss"] == pytest.approx(case["loss"], rel=1e-6, abs=1e-7), msg
        np.testing.assert_allclose(out["dlogits_f64"][0], case["dlogits"], atol=1e-7, err_msg=msg)


def rows(rng, n, V, scale=2.0, grid=None):
    z = rng.standard_normal((n, V)) * scale
    if grid:
        z = np.round(z * grid) / grid  # values with few significant bits: z + c is exact
    return z.astype(np.float32)


def inputs(rng, z, A_values=(1.0, -0.7, 0.0), old_sd=0.05, ref_sd=0.1):
    n, V = z.shape
    y = rng.integers(0, V, size=n).astype(np.int32)
    zz = z.astype(np.float64)
    logp = zz[np.arange(n), y] - scipy.special.logsumexp(zz, axis=1)
    old = (logp + old_sd * rng.standard_normal(n)).astype(np.float32)
    ref = (logp + ref_sd * rng.standard_normal(n)).astype(np.float32)
    adv = np.asarray(A_values, np.float32)
    rr = (np.arange(n) % adv.size).astype(np.int32)
    return y, old, ref, adv, rr


def test_logp_matches_library_logsumexp(oracle_mod):
    rng = np.random.default_rng(10)
    for V, scale in ((7, 1.0), (1024, 2.0), (5000, 8.0)):
        z = rows(rng, 6, V, scale)
        y, old, ref, adv, rr = inputs(rng, z)
        out = oracle_mod.loss(z, V, y, old, ref, adv, rr, want_dlogits=False)
        zz = z.astype(np.float64)
        expect = zz[np.arange(6), y] - scipy.special.logsumexp(zz, axis=1)
        np.testing.assert_allclose(out["logp"], expect, rtol=0, atol=1e-12)


def test_bf16_inputs_are_read_exactly(oracle_mod):
    rng = np.random.default_rng(11)
    z = rows(rng, 4, 300, 3.0)
    bits = (z.view(np.uint32) >> 16).astype(np.uint16)  # truncate to bf16 patterns
    zb = (bits.astype(np.uint32) << 16).view(np.float32)
    y, old, ref, adv, rr = inputs(rng, zb)
    a = oracle_mod.loss(bits, 300, y, old, ref, adv, rr, want_f64=True)
    b = oracle_mod.loss(zb, 300, y, old, ref, adv, rr, want_f64=True)
    assert a["loss"] == b["loss"]
    assert np.array_equal(a["dlogits_f64"], b["dlogits_f64"])


def loss_only(oracle_mod, z, y, old, ref, adv, rr, **kw):
    return oracle_mod.loss(z, z.shape[1], y, old, ref, adv, rr, want_dlogits=False, **kw)["loss"]


@pytest.mark.parametrize("agg_mode", [0, 1])
def test_gradient_matches_finite_differences(oracle_mod, agg_mode):
    """dlogits equals the derivative of the summed loss, by a fourth-order central difference
    on a grid where every perturbed logit is exact in f32 (away from the clip kinks)."""
    rng = np.random.default_rng(12)
    n, V = 5, 9
    z = rows(rng, n, V, 1.5, grid=64)
    y, old, ref, adv, rr = inputs(rng, z, A_values=(1.3, -0.8))
    kw = dict(beta=0.3, denom_tokens=7)
    if agg_mode == 1:
        kw.update(agg_mode=1, seq_off=np.array([0, 3, 5], np.int64), n_seq=2)
    out = oracle_mod.loss(z, V, y, old, ref, adv, rr, want_f64=True, **kw)
    assert np.all(np.abs(out["rho"] - 0.8) > 1e-2) and np.all(np.abs(out["rho"] - 1.2) > 1e-2)
    h = 2.0 ** -9
    fd = np.zeros((n, V))
    for t in range(n):
        for v in range(V):
            vals = []
            for k in (2, 1, -1, -2):
                zp = z.copy()
                zp[t, v] += np.float32(k * h)
                assert zp[t, v] - z[t, v] == np.float32(k * h)
                vals.append(loss_only(oracle_mod, zp, y, old, ref, adv, rr, **kw))
            fd[t, v] = (-vals[0] + 8 * vals[1] - 8 * vals[2] + vals[3]) / (12 * h)
    np.testing.assert_allclose(out["dlogits_f64"], fd, rtol=1e-6, atol=1e-9)


def test_gradient_invariants(oracle_mod):
    rng = np.random.default_rng(13)
    z = rows(rng, 8, 200, 2.0, grid=64)
    y, old, ref, adv, rr = inputs(rng, z)
    out = oracle_mod.loss(z, 200, y, old, ref, adv, rr, want_f64=True)
    d = out["dlogits_f64"]
    # each row of dlogits is w*g*(e_y - p): it sums to zero
    np.testing.assert_allclose(d.sum(1), 0.0, atol=1e-15)
    # softmax is shift invariant: z + 1 gives the same loss and gradient
    sh = oracle_mod.loss(z + np.float32(1.0), 200, y, old, ref, adv, rr, want_f64=True)
    assert sh["loss"] == pytest.approx(out["loss"], rel=1e-12, abs=1e-15)
    np.testing.assert_allclose(sh["dlogits_f64"], d, rtol=1e-10, atol=1e-18)
    # the gradient coefficient is the only row factor: d / (e_y - p) is constant per row
    p = np.exp(z.astype(np.float64) - scipy.special.logsumexp(z.astype(np.float64), 1, keepdims=True))
    e = np.zeros_like(p)
    e[np.arange(8), y] = 1.0
    ratio = d / (e - p)
    np.testing.assert_allclose(ratio, ratio[:, :1].repeat(200, 1), rtol=1e-9)


def test_gradient_factor_g(oracle_mod):
    """The oracle's per-row g: (1) dlogits[t] / (e_y - p) = w * g_t; (2) g_t is the derivative of
    the row's loss term l_t with respect to log pi(y), by a central difference that moves old_logp
    and ref_logp together (rho and x then move as if logp moved the other way); (3) its own
    derivative with respect to log pi(y) is g + beta * (2 e^x - 1), the identity the GPU tests use
    to bound how far an error in logp moves g."""
    rng = np.random.default_rng(16)
    n, V = 12, 50
    z = rows(rng, n, V, 2.0)
    y, old, ref, adv, rr = inputs(rng, z, A_values=(1.1, -0.6, 0.0))
    beta = 0.3
    out = oracle_mod.loss(z, V, y, old, ref, adv, rr, beta=beta, denom_tokens=4, want_f64=True)
    assert np.all(np.abs(out["rho"] - 0.8) > 1e-3) and np.all(np.abs(out["rho"] - 1.2) > 1e-3)
    zz = z.astype(np.float64)
    p = np.exp(zz - scipy.special.logsumexp(zz, 1, keepdims=True))
    e = np.zeros_like(p)
    e[np.arange(n), y] = 1.0
    np.testing.assert_allclose(out["dlogits_f64"] / (e - p), (out["g"] / 4.0)[:, None]
                               .repeat(V, 1), rtol=1e-9)
    h = 1e-5
    # old and ref moved by -h (as if logp moved by +h) and by +h; they are f32 in the oracle's
    # interface, so the shift actually applied is measured, and must be the same for both
    old_p, old_m = old - np.float32(h), old + np.float32(h)
    ref_p, ref_m = ref - np.float32(h), ref + np.float32(h)
    dh = (old_m.astype(np.float64) - old_p.astype(np.float64)) / 2  # the shift actually applied
    assert np.allclose((ref_m.astype(np.float64) - ref_p.astype(np.float64)) / 2, dh, rtol=0, atol=0)
    lp = oracle_mod.loss(z, V, y, old_p, ref_p, adv, rr, beta=beta, denom_tokens=1,
                         want_dlogits=False)
    lm = oracle_mod.loss(z, V, y, old_m, ref_m, adv, rr, beta=beta, denom_tokens=1,
                         want_dlogits=False)
    np.testing.assert_allclose((lp["row_loss"] - lm["row_loss"]) / (2 * dh), out["g"], rtol=1e-5,
                               atol=1e-9)
    x = ref.astype(np.float64) - out["logp"]
    np.testing.assert_allclose((lp["g"] - lm["g"]) / (2 * dh), out["g"] + beta * (2 * np.exp(x) - 1),
                               rtol=1e-5, atol=1e-9)


def test_asymmetric_clip_regions(oracle_mod):
    """Eq. 2 with eps_low = 0.2, eps_high = 0.28 against the clipped surrogate's closed form,
    one token at a time (beta = 0, denominator 1): loss = -min(rho*A, clip(rho)*A), and dlogits
    = -A*rho*(e_y - p) where the unclipped term is the minimum, else 0.  The ratios sit between
    the two widths (1.25, 0.75) and outside both (1.3, 0.7), so a swapped or shared width fails."""
    z = np.array([0.5, -1.0, 2.0, 0.25, -0.5], np.float32)
    zz = z.astype(np.float64)
    logp = zz[0] - scipy.special.logsumexp(zz)
    p = np.exp(zz - scipy.special.logsumexp(zz))
    e = np.zeros(5)
    e[0] = 1.0
    for rho_t, A, clipped in ((1.25, 1.0, False), (1.3, 1.0, True), (0.85, 1.0, False),
                              (0.75, -1.0, True), (0.7, -1.0, True), (0.85, -1.0, False),
                              (1.25, -1.0, False), (0.75, 1.0, False)):
        old = np.float32(logp - math.log(rho_t))
        out = oracle_mod.loss(z[None, :], 5, [0], [old], [old], [A], [0], eps_low=0.2,
                              eps_high=0.28, beta=0.0, denom_tokens=1, want_f64=True)
        rho = math.exp(logp - float(old))
        cl = min(max(rho, 1.0 - float(np.float32(0.2))), 1.0 + float(np.float32(0.28)))
        assert out["loss"] == pytest.approx(-min(rho * A, cl * A), rel=1e-12)
        expect = np.zeros(5) if clipped else -A * rho * (e - p)
        np.testing.assert_allclose(out["dlogits_f64"][0], expect, rtol=1e-12, atol=1e-15)


def test_zero_advantage_without_kl_gives_zero_gradient(oracle_mod):
    rng = np.random.default_rng(14)
    z = rows(rng, 5, 64)
    y, old, ref, _, rr = inputs(rng, z)
    out = oracle_mod.loss(z, 64, y, old, ref, np.zeros(3, np.float32), rr, beta=0.0,
                          want_f64=True, dlogits_dtype=1)
    assert np.all(out["dlogits_f64"] == 0.0)
    assert np.all((out["dlogits"] & 0x7FFF) == 0)
    assert out["loss"] == 0.0


def test_seq_mean_weights(oracle_mod):
    rng = np.random.default_rng(15)
    z = rows(rng, 5, 32)
    y, old, ref, adv, _ = inputs(rng, z)
    rr = np.array([0, 0, 1, 1, 1], np.int32)  # rollouts of lengths 2 and 3
    tok = oracle_mod.loss(z, 32, y, old, ref, adv, rr, denom_tokens=5, want_dlogits=False)
    seq = oracle_mod.loss(z, 32, y, old, ref, adv, rr, agg_mode=1,
                          seq_off=np.array([0, 2, 5], np.int64), n_seq=2, want_dlogits=False)
    # token mean weights 1/5; Eq. 1's weights 1/(2*2) and 1/(2*3)
    scale = np.array([5 / 4, 5 / 4, 5 / 6, 5 / 6, 5 / 6])
    np.testing.assert_allclose(seq["row_loss"], tok["row_loss"] * scale, rtol=1e-14)
    # the weights the oracle reports are those weights: both give the same unweighted l_t
    np.testing.assert_allclose(tok["w"], np.full(5, 1 / 5), rtol=1e-15)
    np.testing.assert_allclose(seq["w"], [1 / 4, 1 / 4, 1 / 6, 1 / 6, 1 / 6], rtol=1e-15)
    np.testing.assert_allclose(seq["row_loss"] / seq["w"], tok["row_loss"] / tok["w"], rtol=1e-14)


def test_invalid_token_row_is_zero(oracle_mod):
    z = np.zeros((2, 8), np.float32)
    out = oracle_mod.loss(z, 8, [3, 9], [-2.0, -2.0], [-2.0, -2.0], [1.0], [0, 0], want_f64=True)
    assert math.isnan(out["logp"][1]) and np.all(out["dlogits_f64"][1] == 0)
    assert out["row_loss"][1] == 0.0 and out["row_loss"][0] != 0.0


def test_round_bf16(oracle_mod):
    import torch
    rng = np.random.default_rng(16)
    x = np.concatenate([rng.standard_normal(2000) * 10.0 ** rng.integers(-40, 38, size=2000),
                        [0.0, -0.0, 1e-45, -3e-41, 3.3e38, 3.4e38, -3.4e38]]).astype(np.float32)
    expect = torch.from_numpy(x).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    got = oracle_mod.round_bf16(x.astype(np.float64))
    assert np.array_equal(got, expect)
    # one rounding from fp64: 1 + 2^-8 + 2^-40 lies above the tie, so it rounds up; rounding
    # through f32 first would land on the tie and then round to even (down)
    assert oracle_mod.round_bf16(np.array([1.0 + 2.0 ** -8 + 2.0 ** -40]))[0] == 0x3F81
    assert oracle_mod.round_bf16(np.array([1.0 + 2.0 ** -8]))[0] == 0x3F80
    assert oracle_mod.round_bf16(np.array([float("inf"), float("nan")])).tolist()[0] == 0x7F80


def test_logp_only_matches_library_logsumexp_and_the_loss(oracle_mod):
    """oracle_logp is the plain z_y - logsumexp(z); it agrees with scipy and with the logp the
    loss reports, including gathered rows and invalid ids."""
    rng = np.random.default_rng(17)
    for V, scale in ((5, 1.0), (3000, 4.0)):
        z = rows(rng, 9, V, scale)
        y = rng.integers(0, V, size=9).astype(np.int32)
        y[4] = V  # invalid
        idx = np.array([8, 0, 4, 3], np.int64)
        got = oracle_mod.logp(z, V, y, row_index=idx)
        zz = z.astype(np.float64)
        for k, r in enumerate(idx):
            if y[r] >= V:
                assert math.isnan(got[k])
            else:
                assert got[k] == pytest.approx(zz[r, y[r]] - scipy.special.logsumexp(zz[r]), abs=1e-12)
        yl = np.where(y >= V, 0, y).astype(np.int32)
        lo = oracle_mod.loss(z, V, yl, np.zeros(9, np.float32), np.zeros(9, np.float32),
                             np.zeros(1, np.float32), np.zeros(9, np.int32), want_dlogits=False)
        np.testing.assert_array_equal(oracle_mod.logp(z, V, yl), lo["logp"])
