"""Pins of the oracle's adaptive rollout sampling (Eqs. 10-14, Algorithm 1) and parity of the
library's host implementation with it (no GPU involved)."""
import numpy as np
import pytest

from helpers import golden


def run_trace(step_fn, g):
    out = []
    spe, M = g["steps_per_epoch"], g["total_steps"]
    for s, kept in enumerate(g["kept_per_step"], start=1):
        out.append(step_fn(kept, s, M, s % spe == 0))
    return out


def test_hand_trace(oracle_mod):
    g = golden("ars_trace.json")
    st = oracle_mod.Ars(g["G1"])
    gts = []

    def step(kept, s, M, end):
        n = st.step(kept, s, M, end)
        if end:
            gts.append(st.g_t)
        return n

    assert run_trace(step, g) == g["n_after_step"]
    assert st.g_ref == pytest.approx(g["g_ref"])
    assert gts == pytest.approx(g["g_t_at_epoch_end"])


def test_before_first_epoch_end_n_is_g1(oracle_mod):
    st = oracle_mod.Ars(16)
    for s in range(1, 10):
        assert st.step([1, 1, 1], s, 100, False) == 16
    assert st.g_ref is None and st.g_t is None


def test_range_property(oracle_mod):
    rng = np.random.default_rng(3)
    for trial in range(50):
        G1 = int(rng.integers(2, 33))
        M = int(rng.integers(2, 60))
        spe = int(rng.integers(1, 8))
        st = oracle_mod.Ars(G1)
        n = G1
        for s in range(1, M + 1):
            kept = rng.integers(0, n + 1, size=int(rng.integers(1, 6)))
            n = st.step(kept, s, M, s % spe == 0)
            assert 2 <= n <= G1
