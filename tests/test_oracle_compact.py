"""Pin of the oracle's compaction: it is a prefix sum and a gather, restated with numpy."""
import numpy as np


def test_compaction_matches_numpy(oracle_mod):
    rng = np.random.default_rng(9)
    for _ in range(50):
        n = int(rng.integers(0, 300))
        L = rng.integers(0, 40, size=n)
        off = np.zeros(n + 1, np.int64)
        off[1:] = np.cumsum(L)
        keep = (rng.random(n) < 0.4).astype(np.uint8)
        out = oracle_mod.compact(keep, off)
        idx = np.nonzero(keep)[0]
        assert out["K"] == idx.size and out["T_kept"] == int(L[idx].sum())
        assert np.array_equal(out["kept_idx"], idx)
        assert np.array_equal(out["kept_off"], np.concatenate([[0], np.cumsum(L[idx])]))
        src = np.concatenate([np.arange(off[i], off[i + 1]) for i in idx]) if idx.size else np.zeros(0)
        assert np.array_equal(out["src_token"], src)
        assert np.array_equal(out["token_rollout"], np.repeat(idx, L[idx]))
