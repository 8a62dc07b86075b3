"""Pins of the oracle's advantage (Eq. 5) against hand-worked groups and invariants."""
import numpy as np
import pytest

from helpers import golden


def test_hand_worked(oracle_mod):
    g = golden("advantage_hand.json")
    for case in g["cases"]:
        adv, _ = oracle_mod.advantage(case["rewards"], case["G"], case["std_mode"])
        np.testing.assert_allclose(adv, case["adv"], rtol=1e-7, atol=1e-7, err_msg=case["derivation"])


@pytest.mark.parametrize("G", [2, 3, 4, 8, 16, 32])
def test_equal_rewards_give_zero(oracle_mod, G):
    for v in (0.0, 1.0, 0.1, -3.5):
        adv, key = oracle_mod.advantage(np.full(G, v, np.float32), G)
        assert np.all(adv == 0.0) and np.all(key == 0.0)


def test_single_rollout_is_zero(oracle_mod):
    adv, _ = oracle_mod.advantage([0.7, 0.2, 1.0], 1, 0)
    assert np.all(adv == 0.0)


@pytest.mark.parametrize("std_mode", [0, 1])
def test_zero_sum_unit_std(oracle_mod, std_mode):
    rng = np.random.default_rng(1)
    G = 8
    r = rng.random((20, G)).astype(np.float32)
    adv, _ = oracle_mod.advantage(r.ravel(), G, std_mode)
    a = adv.reshape(20, G).astype(np.float64)
    np.testing.assert_allclose(a.sum(1), 0.0, atol=1e-6)
    np.testing.assert_allclose(a.std(1, ddof=1 if std_mode == 0 else 0), 1.0, rtol=1e-6)


def test_affine_invariance(oracle_mod):
    """A is unchanged by r -> a*r + b for a > 0 and negated for a < 0 (Eq. 5 is a z-score)."""
    rng = np.random.default_rng(2)
    G = 8
    r = rng.integers(0, 5, size=(16, G)).astype(np.float64)
    base, _ = oracle_mod.advantage(r.ravel().astype(np.float32), G)
    for a, b in ((2.0, 3.0), (0.5, -1.0), (-1.0, 0.0), (-4.0, 1.0)):
        adv, _ = oracle_mod.advantage((a * r + b).ravel().astype(np.float32), G)
        np.testing.assert_allclose(adv, np.sign(a) * base, atol=1e-6)


def test_key_is_distance_to_mean(oracle_mod):
    r = np.array([1, 0, 0, 0, 0.9, 0.1, 1.0, 0.0], np.float32)
    _, key = oracle_mod.advantage(r, 4)
    np.testing.assert_allclose(key[:4], [0.75, 0.25, 0.25, 0.25])
    m = np.mean(r[4:].astype(np.float64))
    np.testing.assert_allclose(key[4:], np.abs(r[4:].astype(np.float64) - m), rtol=1e-15)
