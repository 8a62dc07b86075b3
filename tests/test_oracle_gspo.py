"""Pins of the oracle's GSPO sequence-level loss: hand-worked sequences, the reduction to the
token-level loss (Eq. 1's sequence mean) when every sequence has one token, finite differences
across the tokens of a sequence, and invariants of the sequence ratio."""
import numpy as np
import pytest
import scipy.special

from helpers import golden


def seq_case(oracle_mod, case, **kw):
    z = np.asarray([r["z"] for r in case["rows"]], np.float32)
    y = [r["y"] for r in case["rows"]]
    old = [r["old_logp"] for r in case["rows"]]
    ref = [r["ref_logp"] for r in case["rows"]]
    seq_off = [case["sequences"][0]["rows"][0]] + [s["rows"][1] for s in case["sequences"]]
    adv = [s["A"] for s in case["sequences"]]
    return oracle_mod.gspo_loss(z, case["V"], y, old, ref, adv, np.arange(len(adv)), seq_off,
                                n_seq=case["n_seq"], eps_low=case["eps_low"],
                                eps_high=case["eps_high"], beta=case["beta"], want_f64=True, **kw)


def test_hand_worked(oracle_mod):
    for case in golden("gspo_hand.json")["cases"]:
        out = seq_case(oracle_mod, case)
        msg = case["name"] + ": " + case["derivation"]
        assert out["loss"] == pytest.approx(case["loss"], rel=1e-6, abs=1e-7), msg
        np.testing.assert_allclose(out["seq_ratio"], case["seq_ratio"], rtol=1e-6, err_msg=msg)
        np.testing.assert_allclose(out["dlogits_f64"], case["dlogits"], atol=1e-7, err_msg=msg)


def batch(rng, lens, V, old_sd=0.05, scale=2.0, grid=None):
    n = int(sum(lens))
    z = rng.standard_normal((n, V)) * scale
    if grid:
        z = np.round(z * grid) / grid
    z = z.astype(np.float32)
    y = rng.integers(0, V, size=n).astype(np.int32)
    zz = z.astype(np.float64)
    logp = zz[np.arange(n), y] - scipy.special.logsumexp(zz, axis=1)
    old = (logp + old_sd * rng.standard_normal(n)).astype(np.float32)
    ref = (logp + 0.1 * rng.standard_normal(n)).astype(np.float32)
    off = np.concatenate([[0], np.cumsum(lens)]).astype(np.int64)
    return z, y, old, ref, off


def test_one_token_sequences_reduce_to_the_token_level_sequence_mean(oracle_mod):
    """With every sequence one token long, s_k is the token ratio and the sequence mean is
    Eq. 1's: the loss, logp and dlogits equal the token-level oracle's with agg_mode 1."""
    rng = np.random.default_rng(30)
    K, V = 40, 300
    z, y, old, ref, off = batch(rng, [1] * K, V, old_sd=0.4)
    adv = rng.standard_normal(K).astype(np.float32)
    kw = dict(eps_low=0.2, eps_high=0.28, beta=0.04)
    g = oracle_mod.gspo_loss(z, V, y, old, ref, adv, np.arange(K), off, want_f64=True, **kw)
    t = oracle_mod.loss(z, V, y, old, ref, adv, np.arange(K, dtype=np.int32), agg_mode=1,
                        seq_off=off, n_seq=K, want_f64=True, **kw)
    assert g["loss"] == pytest.approx(t["loss"], rel=1e-13)
    np.testing.assert_allclose(g["logp"], t["logp"], rtol=0, atol=1e-14)
    np.testing.assert_allclose(g["seq_ratio"], t["rho"], rtol=1e-13)
    np.testing.assert_allclose(g["dlogits_f64"], t["dlogits_f64"], rtol=1e-12, atol=1e-18)
    lo, hi = 0.8, 1.28
    clipped = ((adv > 0) & (t["rho"] > hi)) | ((adv < 0) & (t["rho"] < lo))
    assert 3 <= clipped.sum() <= K - 3  # both branches are exercised


def loss_only(oracle_mod, z, *a, **kw):
    return oracle_mod.gspo_loss(z, z.shape[1], *a, want_dlogits=False, **kw)["loss"]


def test_gradient_matches_finite_differences(oracle_mod):
    """dlogits equals the derivative of the loss, through the sequence ratio that couples the
    tokens of a sequence (fourth-order central differences on an f32-exact grid)."""
    rng = np.random.default_rng(31)
    lens, V = [3, 1, 2], 7
    z, y, old, ref, off = batch(rng, lens, V, old_sd=0.1, scale=1.5, grid=64)
    adv = np.array([1.1, -0.6, 0.8], np.float32)
    kw = dict(eps_low=0.2, eps_high=0.28, beta=0.3, n_seq=4)
    args = (y, old, ref, adv, np.arange(3), off)
    out = oracle_mod.gspo_loss(z, V, *args, want_f64=True, **kw)
    s = out["seq_ratio"]
    assert np.all(np.abs(s - 0.8) > 1e-2) and np.all(np.abs(s - 1.28) > 1e-2)
    h = 2.0 ** -9
    fd = np.zeros_like(out["dlogits_f64"])
    for t in range(z.shape[0]):
        for v in range(V):
            vals = []
            for k in (2, 1, -1, -2):
                zp = z.copy()
                zp[t, v] += np.float32(k * h)
                assert zp[t, v] - z[t, v] == np.float32(k * h)
                vals.append(loss_only(oracle_mod, zp, *args, **kw))
            fd[t, v] = (-vals[0] + 8 * vals[1] - 8 * vals[2] + vals[3]) / (12 * h)
    np.testing.assert_allclose(out["dlogits_f64"], fd, rtol=1e-6, atol=1e-9)


def test_gradient_factor_g(oracle_mod):
    """The oracle's per-row g_t: dlogits[t] / (e_y - p) = g_t / (n_seq L_k) for every row (the
    dlogits themselves are pinned by finite differences above), NaN in a sequence without a
    ratio."""
    rng = np.random.default_rng(33)
    lens, V = [4, 1, 3, 0, 2], 11
    z, y, old, ref, off = batch(rng, lens, V, old_sd=0.1, scale=1.5)
    y = y.copy()
    y[-1] = V + 2  # the last sequence has an invalid token: no ratio
    adv = np.array([0.9, -0.4, 0.0, 1.0, 0.5], np.float32)
    out = oracle_mod.gspo_loss(z, V, y, old, ref, adv, np.arange(5), off, n_seq=6, eps_low=0.2,
                               eps_high=0.28, beta=0.3, want_f64=True)
    zz = z.astype(np.float64)
    p = np.exp(zz - scipy.special.logsumexp(zz, 1, keepdims=True))
    e = np.zeros_like(p)
    ok = (y >= 0) & (y < V)
    e[np.flatnonzero(ok), y[ok]] = 1.0
    L = np.repeat(np.asarray(lens), lens).astype(np.float64)
    g = out["g"]
    assert np.all(np.isnan(g[-2:])) and np.all(np.isfinite(g[:-2]))
    np.testing.assert_allclose(out["dlogits_f64"][:-2] / (e - p)[:-2],
                               (g[:-2] / (6 * L[:-2]))[:, None].repeat(V, 1), rtol=1e-9)


def test_clipping_is_per_sequence(oracle_mod):
    """A sequence whose ratio is clipped (A > 0, s > 1 + eps_high, beta = 0) gets zero gradient
    on every token, including tokens whose own ratio lies inside the clip range; the token-level
    loss on the same rows keeps those tokens."""
    rng = np.random.default_rng(32)
    V = 50
    z, y, old, ref, off = batch(rng, [6, 6], V)
    zz = z.astype(np.float64)
    logp = zz[np.arange(12), y] - scipy.special.logsumexp(zz, axis=1)
    shift = np.array([1.5, 1.5, 1.5, 0.1, 0.1, 0.1, 0.05, -0.05, 0.1, -0.1, 0.0, 0.02])
    old = (logp - shift).astype(np.float32)  # token log-ratios = shift
    adv = np.array([1.0, 1.0], np.float32)
    g = oracle_mod.gspo_loss(z, V, y, old, ref, adv, [0, 1], off, eps_low=0.2, eps_high=0.2,
                             beta=0.0, want_f64=True)
    assert g["seq_ratio"][0] > 1.2 and 0.8 < g["seq_ratio"][1] < 1.2
    assert np.all(g["dlogits_f64"][:6] == 0.0)
    assert np.all(np.any(g["dlogits_f64"][6:] != 0.0, axis=1))
    t = oracle_mod.loss(z, V, y, old, ref, adv, np.repeat([0, 1], 6).astype(np.int32),
                        agg_mode=1, seq_off=off, n_seq=2, eps_low=0.2, eps_high=0.2, beta=0.0,
                        want_f64=True)
    assert np.all(np.any(t["dlogits_f64"][3:6] != 0.0, axis=1))  # token-level keeps them


def test_ratio_ignores_token_order_within_a_sequence(oracle_mod):
    """s_k is a mean over the sequence: reading a sequence's rows in reverse order (through
    row_index) leaves s_k and the loss unchanged and permutes the dlogits rows."""
    rng = np.random.default_rng(33)
    lens, V = [5, 3, 4], 64
    z, y, old, ref, off = batch(rng, lens, V, old_sd=0.2)
    adv = rng.standard_normal(3).astype(np.float32)
    kw = dict(eps_low=0.2, eps_high=0.28, beta=0.04, want_f64=True)
    a = oracle_mod.gspo_loss(z, V, y, old, ref, adv, np.arange(3), off, **kw)
    perm = np.concatenate([np.arange(off[k], off[k + 1])[::-1] for k in range(3)])
    b = oracle_mod.gspo_loss(z, V, y, old, ref, adv, np.arange(3), off, row_index=perm, **kw)
    np.testing.assert_allclose(b["seq_ratio"], a["seq_ratio"], rtol=1e-14)
    assert b["loss"] == pytest.approx(a["loss"], rel=1e-13)
    np.testing.assert_allclose(b["dlogits_f64"], a["dlogits_f64"][perm], rtol=1e-12, atol=1e-20)


def test_invalid_token_and_empty_sequences(oracle_mod):
    """A sequence holding a token id outside [0, V) has no ratio: NaN, zero loss term, zero
    rows; an empty sequence contributes nothing; the other sequences are unaffected."""
    rng = np.random.default_rng(34)
    lens, V = [4, 0, 3, 2], 40
    z, y, old, ref, off = batch(rng, lens, V, old_sd=0.2)
    adv = rng.standard_normal(4).astype(np.float32)
    kw = dict(eps_low=0.2, eps_high=0.2, beta=0.04, n_seq=4, want_f64=True)
    good = oracle_mod.gspo_loss(z, V, y, old, ref, adv, np.arange(4), off, **kw)
    y_bad = y.copy()
    y_bad[5] = V  # row 5 belongs to sequence 2 (rows 4..6)
    bad = oracle_mod.gspo_loss(z, V, y_bad, old, ref, adv, np.arange(4), off, **kw)
    assert np.isnan(bad["seq_ratio"][2]) and np.isnan(bad["seq_ratio"][1])
    assert bad["seq_loss"][2] == 0.0 and bad["seq_loss"][1] == 0.0
    assert np.all(bad["dlogits_f64"][4:7] == 0.0)
    np.testing.assert_array_equal(bad["dlogits_f64"][:4], good["dlogits_f64"][:4])
    np.testing.assert_array_equal(bad["dlogits_f64"][7:], good["dlogits_f64"][7:])
    assert bad["loss"] == pytest.approx(good["loss"] - good["seq_loss"][2], rel=1e-12)
