"""Pins of the oracle's output layer fused with the GRPO loss (z = h W^T, then Eqs. 1-3, then the
chain rule): a library matrix product, a hand-worked two-word vocabulary, finite differences of
the loss with respect to every hidden and weight entry, and invariances of the softmax; and the
same for GSPO's sequence-level ratio."""
import math

import numpy as np
import pytest


def problem(rng, T=6, V=9, D=5, n_roll=2, old_shift=0.0, beta=0.04):
    h = rng.standard_normal((T, D))
    w = rng.standard_normal((V, D)) * 0.7
    y = rng.integers(0, V, T)
    rr = np.sort(rng.integers(0, n_roll, T))
    adv = rng.standard_normal(n_roll)
    z = h @ w.T
    logp = z[np.arange(T), y] - np.log(np.exp(z).sum(1))
    old = (logp + old_shift + rng.normal(0, 0.05, T)).astype(np.float32)
    ref = (logp + rng.normal(0, 0.1, T)).astype(np.float32)
    return dict(hidden=h, weight=w, y=y, old_logp=old, ref_logp=ref, adv=adv.astype(np.float32),
                row_rollout=rr.astype(np.int32)), dict(beta=beta)


def run(oracle_mod, p, kw, **extra):
    return oracle_mod.lmhead_loss(p["hidden"], p["weight"], p["y"], p["old_logp"], p["ref_logp"],
                                  p["adv"], p["row_rollout"], **kw, **extra)


def test_logits_equal_a_library_matrix_product_and_feed_the_loss(oracle_mod):
    rng = np.random.default_rng(1)
    p, kw = problem(rng, T=7, V=13, D=6)
    out = run(oracle_mod, p, kw, want_logits=True, want_dlogits=True)
    z = np.matmul(p["hidden"], p["weight"].T)
    np.testing.assert_allclose(out["logits"], z, rtol=1e-13, atol=1e-13)
    # The loss part is the (separately pinned) token loss evaluated on those logits.
    ref = oracle_mod.loss(z, 13, p["y"], p["old_logp"], p["ref_logp"], p["adv"], p["row_rollout"],
                          logits_dtype=2, want_f64=True, **kw)
    np.testing.assert_allclose(out["logp"], ref["logp"], rtol=1e-12, atol=1e-12)
    np.testing.assert_allclose(out["dlogits"], ref["dlogits_f64"], rtol=1e-11, atol=1e-15)
    assert out["loss"] == pytest.approx(ref["loss"], rel=1e-12, abs=1e-15)


def test_hand_worked_two_word_vocabulary(oracle_mod):
    # V = 2, D = 1: z = (h w0, h w1), y = 0, so logp = -log(1 + e^{z1 - z0}).  With beta = 0 and
    # A = 1 inside the clip range, loss = -rho and d loss / d logp = -rho, while
    # d logp / d z0 = sigma(z1 - z0) = -d logp / d z1.  By the chain rule:
    #   d loss / d h  = -rho * sigma(z1 - z0) * (w0 - w1)
    #   d loss / d w0 = -rho * sigma(z1 - z0) * h,   d loss / d w1 = +rho * sigma(z1 - z0) * h
    h, w0, w1 = 0.5, 2.0, -1.0
    z0, z1 = h * w0, h * w1                      # 1.0, -0.5
    logp = -math.log1p(math.exp(z1 - z0))        # log sigma(1.5)
    old = np.float32(logp - 0.05)                # rho = e^{0.05...} inside [0.8, 1.2]
    rho = math.exp(logp - float(old))
    sig = 1.0 / (1.0 + math.exp(-(z1 - z0)))
    out = oracle_mod.lmhead_loss([[h]], [[w0], [w1]], [0], [old], [logp], [1.0], [0], beta=0.0,
                                 denom_tokens=1)
    assert out["logp"][0] == pytest.approx(logp, rel=1e-14)
    assert out["loss"] == pytest.approx(-rho, rel=1e-14)
    assert out["dhidden"][0, 0] == pytest.approx(-rho * sig * (w0 - w1), rel=1e-13)
    assert out["dweight"][0, 0] == pytest.approx(-rho * sig * h, rel=1e-13)
    assert out["dweight"][1, 0] == pytest.approx(rho * sig * h, rel=1e-13)


def finite_difference(oracle_mod, p, kw, key, idx, step=1e-6):
    q = {k: (v.copy() if isinstance(v, np.ndarray) else v) for k, v in p.items()}
    q[key] = q[key].astype(np.float64)
    q[key][idx] += step
    up = run(oracle_mod, q, kw, want_dhidden=False, want_dweight=False)["loss"]
    q[key][idx] -= 2 * step
    down = run(oracle_mod, q, kw, want_dhidden=False, want_dweight=False)["loss"]
    return (up - down) / (2 * step)


@pytest.mark.parametrize("case", ["token-mean", "seq-mean", "beta 0, clipped tokens"])
def test_gradients_are_the_derivatives_of_the_loss(oracle_mod, case):
    rng = np.random.default_rng({"token-mean": 3, "seq-mean": 4, "beta 0, clipped tokens": 5}[case])
    if case == "beta 0, clipped tokens":
        p, kw = problem(rng, old_shift=-0.6, beta=0.0)  # rho ~ e^0.6: clipped where A > 0
        p["adv"] = np.array([0.8, -1.1], np.float32)
    else:
        p, kw = problem(rng)
    if case == "seq-mean":
        rr = p["row_rollout"]
        kw.update(agg_mode=1, seq_off=np.r_[0, np.cumsum(np.bincount(rr, minlength=2))],
                  n_seq=2)
    out = run(oracle_mod, p, kw)
    # no ratio sits on a clip boundary, where the loss has a kink
    z = p["hidden"] @ p["weight"].T
    logp = z[np.arange(len(p["y"])), p["y"]] - np.log(np.exp(z).sum(1))
    rho = np.exp(logp - p["old_logp"])
    assert np.min(np.abs(rho - 0.8)) > 1e-3 and np.min(np.abs(rho - 1.2)) > 1e-3
    if case == "beta 0, clipped tokens":
        assert (rho > 1.2).any()
    T, D = p["hidden"].shape
    V = p["weight"].shape[0]
    for t in range(T):
        for d in range(D):
            fd = finite_difference(oracle_mod, p, kw, "hidden", (t, d))
            assert out["dhidden"][t, d] == pytest.approx(fd, rel=1e-6, abs=1e-9), (t, d)
    for v in range(V):
        for d in range(D):
            fd = finite_difference(oracle_mod, p, kw, "weight", (v, d))
            assert out["dweight"][v, d] == pytest.approx(fd, rel=1e-6, abs=1e-9), (v, d)


def test_common_shift_of_the_weight_rows_changes_nothing(oracle_mod):
    # Adding one vector c to every weight row adds h_t . c to every logit of row t: the softmax,
    # the loss and dlogits are unchanged, and so is dh = dlogits W because each dlogits row sums
    # to zero.
    rng = np.random.default_rng(6)
    p, kw = problem(rng, T=8, V=11, D=4)
    base = run(oracle_mod, p, kw)
    q = dict(p)
    q["weight"] = p["weight"] + rng.standard_normal(4)[None, :]
    moved = run(oracle_mod, q, kw)
    np.testing.assert_allclose(moved["logp"], base["logp"], rtol=1e-12, atol=1e-12)
    assert moved["loss"] == pytest.approx(base["loss"], rel=1e-11, abs=1e-14)
    np.testing.assert_allclose(moved["dhidden"], base["dhidden"], rtol=1e-9, atol=1e-13)
    np.testing.assert_allclose(moved["dweight"], base["dweight"], rtol=1e-9, atol=1e-13)


def test_weight_gradient_rows_sum_to_zero_and_bounds_dominate(oracle_mod):
    rng = np.random.default_rng(7)
    p, kw = problem(rng, T=10, V=17, D=6)
    out = run(oracle_mod, p, kw, want_dlogits=True, want_bounds=True)
    np.testing.assert_allclose(out["dlogits"].sum(1), 0.0, atol=1e-15)
    np.testing.assert_allclose(out["dweight"].sum(0), 0.0, atol=1e-14)
    assert (np.abs(out["dhidden"]) <= out["dhidden_abs"] * (1 + 1e-12)).all()
    assert (np.abs(out["dweight"]) <= out["dweight_abs"] * (1 + 1e-12)).all()
    np.testing.assert_allclose(out["dhidden_abs"], np.abs(out["dlogits"]) @ np.abs(p["weight"]),
                               rtol=1e-12)


def test_invalid_token_rows_carry_no_gradient(oracle_mod):
    rng = np.random.default_rng(8)
    p, kw = problem(rng, T=5, V=7, D=3)
    p["y"] = p["y"].copy()
    p["y"][2] = 7  # outside [0, V)
    out = run(oracle_mod, p, kw)
    assert math.isnan(out["logp"][2]) and out["row_loss"][2] == 0.0
    np.testing.assert_array_equal(out["dhidden"][2], 0.0)
    assert np.isfinite(out["dweight"]).all()


def gspo_problem(rng, lens=(3, 1, 4), V=8, D=5, old_shift=0.0, beta=0.03):
    T = int(sum(lens))
    p, kw = problem(rng, T=T, V=V, D=D, n_roll=len(lens), old_shift=old_shift, beta=beta)
    so = np.r_[0, np.cumsum(lens)].astype(np.int64)
    return p, so, dict(beta=beta, eps_low=0.2, eps_high=0.28)


def run_gspo(oracle_mod, p, so, kw, **extra):
    return oracle_mod.lmhead_gspo_loss(p["hidden"], p["weight"], p["y"], p["old_logp"],
                                       p["ref_logp"], p["adv"], np.arange(len(so) - 1), so,
                                       **kw, **extra)


def test_gspo_logits_feed_the_gspo_loss(oracle_mod):
    rng = np.random.default_rng(11)
    p, so, kw = gspo_problem(rng)
    out = run_gspo(oracle_mod, p, so, kw, want_dlogits=True)
    z = np.matmul(p["hidden"], p["weight"].T)
    ref = oracle_mod.gspo_loss(z, z.shape[1], p["y"], p["old_logp"], p["ref_logp"], p["adv"],
                               np.arange(len(so) - 1), so, logits_dtype=2, want_f64=True, **kw)
    np.testing.assert_allclose(out["logp"], ref["logp"], rtol=1e-12, atol=1e-12)
    np.testing.assert_allclose(out["seq_ratio"], ref["seq_ratio"], rtol=1e-12)
    np.testing.assert_allclose(out["dlogits"], ref["dlogits_f64"], rtol=1e-11, atol=1e-15)
    assert out["loss"] == pytest.approx(ref["loss"], rel=1e-12, abs=1e-15)


@pytest.mark.parametrize("case", ["inside the clip range", "clipped sequences"])
def test_gspo_gradients_are_the_derivatives_of_the_loss(oracle_mod, case):
    rng = np.random.default_rng(12 if case == "inside the clip range" else 13)
    p, so, kw = gspo_problem(rng, old_shift=0.0 if case == "inside the clip range" else -0.5)
    if case == "clipped sequences":
        p["adv"] = np.array([0.9, -0.7, 1.3], np.float32)
    out = run_gspo(oracle_mod, p, so, kw)
    s_k = out["seq_ratio"]
    assert np.min(np.abs(s_k - 0.8)) > 1e-3 and np.min(np.abs(s_k - 1.28)) > 1e-3
    if case == "clipped sequences":
        assert (s_k > 1.28).any()

    def loss_of(key, idx, step):
        q = {k: (v.copy() if isinstance(v, np.ndarray) else v) for k, v in p.items()}
        q[key] = q[key].astype(np.float64)
        q[key][idx] += step
        return run_gspo(oracle_mod, q, so, kw, want_dhidden=False, want_dweight=False)["loss"]

    T, D = p["hidden"].shape
    V = p["weight"].shape[0]
    h = 1e-6
    for key, shape, grad in (("hidden", (T, D), out["dhidden"]), ("weight", (V, D), out["dweight"])):
        for idx in np.ndindex(*shape):
            fd = (loss_of(key, idx, h) - loss_of(key, idx, -h)) / (2 * h)
            assert grad[idx] == pytest.approx(fd, rel=1e-6, abs=1e-9), (key, idx)


def test_chain_rule_alone_equals_library_matrix_products(oracle_mod):
    """oracle.lmhead_grad (the chain rule for given dlogits) equals numpy's matrix products, and
    its absolute sums equal the products of the absolute values; on the fused oracle's own dlogits
    it returns the fused oracle's dhidden and dweight."""
    rng = np.random.default_rng(31)
    for T, V, D in ((1, 1, 1), (7, 13, 6), (40, 33, 24)):
        dl = rng.standard_normal((T, V))
        h = rng.standard_normal((T, D))
        w = rng.standard_normal((V, D))
        out = oracle_mod.lmhead_grad(dl, h, w, want_bounds=True)
        np.testing.assert_allclose(out["dhidden"], dl @ w, rtol=1e-12, atol=1e-12)
        np.testing.assert_allclose(out["dweight"], dl.T @ h, rtol=1e-12, atol=1e-12)
        np.testing.assert_allclose(out["dhidden_abs"], np.abs(dl) @ np.abs(w), rtol=1e-12)
        np.testing.assert_allclose(out["dweight_abs"], np.abs(dl).T @ np.abs(h), rtol=1e-12)
    p, kw = problem(np.random.default_rng(32), T=9, V=11, D=7)
    fused = run(oracle_mod, p, kw, want_dlogits=True)
    alone = oracle_mod.lmhead_grad(fused["dlogits"], p["hidden"], p["weight"])
    assert np.array_equal(alone["dhidden"], fused["dhidden"])
    assert np.array_equal(alone["dweight"], fused["dweight"])
