"""Pins of the oracle's MDAP pruning (Eqs. 6-9, Algorithm 1): hand-worked cases, brute-force
enumeration on every small instance drawn, special values of tau, the cap and the DP fill."""
import numpy as np
import pytest

from helpers import golden, pack_rollouts
from mdap_ref import brute_force_mdap, cap_by_sort, ngram_set, random_structured_prompt, theta


def run_oracle(oracle_mod, rewards, seqs, G, n, tau, cap=None, dp=1):
    ids, off = pack_rollouts(seqs)
    return oracle_mod.prune(np.asarray(rewards, np.float32), ids, off, G, n, tau, cap, dp)


def test_hand_worked(oracle_mod):
    for case in golden("mdap_hand.json")["cases"]:
        keep, kpp = run_oracle(oracle_mod, case["rewards"], case["rollouts"], case["G"], case["n"],
                               case["tau"], case["keep_cap"], case["dp"])
        assert keep.tolist() == case["keep"], case["name"] + ": " + case["derivation"]
        G = case["G"]
        assert kpp.tolist() == [sum(case["keep"][p * G:(p + 1) * G]) for p in range(len(kpp))]


def test_jaccard_matches_python_sets(oracle_mod):
    rng = np.random.default_rng(5)
    for _ in range(200):
        n = int(rng.integers(1, 4))
        a = rng.integers(0, 5, size=int(rng.integers(0, 9))).tolist()
        b = rng.integers(0, 5, size=int(rng.integers(0, 9))).tolist()
        ids, off = pack_rollouts([a, b])
        got = oracle_mod.jaccard_distance(ids, off, 0, 1, n)
        assert got == theta(ngram_set(a, n), ngram_set(b, n))


@pytest.mark.parametrize("G", [2, 3, 5, 8])
@pytest.mark.parametrize("n", [1, 2, 3])
@pytest.mark.parametrize("tau", [0.3, 0.5, 0.8, 1.0])
def test_brute_force_small_groups(oracle_mod, G, n, tau):
    rng = np.random.default_rng(100 * G + 10 * n + int(10 * tau))
    for trial in range(25):
        q = [0.1, 0.3, 0.6][trial % 3]
        rewards, seqs = random_structured_prompt(rng, G, vocab=6, max_len=7, q=q)
        keep, _ = run_oracle(oracle_mod, rewards, seqs, G, n, tau)
        assert keep.astype(bool).tolist() == brute_force_mdap(rewards, seqs, n, tau), (rewards, seqs)


def test_every_class_keeps_one_and_tau_limits(oracle_mod):
    rng = np.random.default_rng(6)
    for _ in range(200):
        G = int(rng.integers(1, 9))
        rewards, seqs = random_structured_prompt(rng, G, vocab=4, max_len=6, q=0.2)
        for tau, expect in ((0.0, "all"), (-1.0, "all"), (1.01, "one"), (0.8, None)):
            keep, _ = run_oracle(oracle_mod, rewards, seqs, G, 1, tau)
            r = np.float32(rewards)
            for c in set(r.tolist()):
                members = np.nonzero(r == c)[0]
                k = int(keep[members].sum())
                assert k >= 1  # |S'_k| >= 1 (Algorithm 1)
                if expect == "all":
                    assert k == len(members)
                if expect == "one":
                    assert k == 1 and keep[members[0]] == 1


def test_cap_matches_sort_statement(oracle_mod):
    rng = np.random.default_rng(7)
    for _ in range(300):
        G = int(rng.integers(2, 17))
        rewards, seqs = random_structured_prompt(rng, G, vocab=50, max_len=6, q=0.9)
        uncapped, _ = run_oracle(oracle_mod, rewards, seqs, G, 1, 0.8)
        cap = int(rng.integers(1, G + 1))
        capped, kpp = run_oracle(oracle_mod, rewards, seqs, G, 1, 0.8, cap)
        assert capped.astype(bool).tolist() == cap_by_sort(rewards, uncapped.astype(bool), cap)
        assert kpp[0] == min(cap, int(uncapped.sum()))


def test_dp_fill_properties(oracle_mod):
    rng = np.random.default_rng(8)
    for _ in range(200):
        P = int(rng.integers(1, 6))
        G = int(rng.integers(2, 9))
        rewards, seqs = [], []
        for _p in range(P):
            r, s = random_structured_prompt(rng, G, vocab=30, max_len=5, q=0.8)
            rewards += r
            seqs += s
        cap = int(rng.integers(1, G + 1))
        d = int(rng.integers(1, 7))
        base, _ = run_oracle(oracle_mod, rewards, seqs, G, 1, 0.8, cap, 1)
        filled, kpp = run_oracle(oracle_mod, rewards, seqs, G, 1, 0.8, cap, d)
        assert np.all(filled >= base)  # only additions
        total = int(filled.sum())
        assert total % d == 0 or total == P * G
        added = (filled.astype(int) - base.astype(int)).reshape(P, G)
        per_prompt = added.sum(1)
        # round-robin from prompt 0: prompts that never ran out differ by at most one addition,
        # earlier prompts first
        full = [p for p in range(P) if base.reshape(P, G)[p].sum() + per_prompt[p] == G]
        open_ = [p for p in range(P) if p not in full]
        if open_:
            counts = per_prompt[open_]
            assert counts.max() - counts.min() <= 1
            assert all(counts[i] >= counts[i + 1] for i in range(len(counts) - 1))
        # each addition is the largest |r - mean| left in its prompt (lowest index on ties)
        r = np.float32(rewards).reshape(P, G).astype(np.float64)
        dist = np.abs(r - r.mean(1, keepdims=True))
        for p in range(P):
            for i in np.nonzero(added[p])[0]:
                left = [j for j in range(G) if not base.reshape(P, G)[p][j]]
                best = sorted(left, key=lambda j: (-dist[p][j], j))[:int(per_prompt[p])]
                assert i in best
        assert kpp.tolist() == filled.reshape(P, G).sum(1).tolist()


from mdap_ref import (brute_force_mdap_labels, cap_by_sort_labels, chain_classes,
                      clustered_rewards)


def run_oracle_cont(oracle_mod, rewards, seqs, G, n, tau, eps, cap=None, dp=1):
    ids, off = pack_rollouts(seqs)
    adv, _ = oracle_mod.advantage(np.asarray(rewards, np.float32), G)
    keep, kpp = oracle_mod.prune(np.asarray(rewards, np.float32), ids, off, G, n, tau, cap, dp,
                                 adv=adv, class_eps=eps)
    return keep, kpp, adv


@pytest.mark.parametrize("G", [3, 5, 8])
@pytest.mark.parametrize("eps", [1e-4, 1e-2, 0.5])
def test_continuous_grouping_brute_force(oracle_mod, G, eps):
    """Chained-advantage classes (the continuous-reward extension), then per class the
    lexicographically largest independent set, found by enumeration."""
    rng = np.random.default_rng(int(G * 1000 + eps * 1e4))
    for trial in range(20):
        _, seqs = random_structured_prompt(rng, G, vocab=5, max_len=6, q=0.3)
        rewards = clustered_rewards(rng, G)
        keep, _, adv = run_oracle_cont(oracle_mod, rewards, seqs, G, 1, 0.8, eps)
        labels = chain_classes(adv, eps)
        assert keep.astype(bool).tolist() == brute_force_mdap_labels(rewards, seqs, 1, 0.8, labels)


def test_continuous_grouping_limits(oracle_mod):
    rng = np.random.default_rng(31)
    for _ in range(100):
        G = int(rng.integers(2, 9))
        rewards, seqs = random_structured_prompt(rng, G, vocab=4, max_len=6, q=0.3)
        ids, off = pack_rollouts(seqs)
        r = np.asarray(rewards, np.float32)
        exact, _ = oracle_mod.prune(r, ids, off, G, 1, 0.8)
        adv, _ = oracle_mod.advantage(r, G)
        # eps below every gap between distinct advantages: the exact-equality classes
        tiny, _ = oracle_mod.prune(r, ids, off, G, 1, 0.8, adv=adv, class_eps=1e-30)
        assert np.array_equal(tiny, exact)
        # eps above every gap: one class, so the greedy runs over the whole group
        one, _ = oracle_mod.prune(r, ids, off, G, 1, 0.8, adv=adv, class_eps=1e30)
        assert one.astype(bool).tolist() == brute_force_mdap_labels(rewards, seqs, 1, 0.8, [0] * G)


def test_continuous_cap_in_visiting_order(oracle_mod):
    rng = np.random.default_rng(32)
    for _ in range(200):
        G = int(rng.integers(2, 17))
        _, seqs = random_structured_prompt(rng, G, vocab=40, max_len=5, q=0.9)
        rewards = clustered_rewards(rng, G, spread=3e-3)
        eps = float(rng.choice([1e-4, 1e-2, 0.2]))
        uncapped, _, adv = run_oracle_cont(oracle_mod, rewards, seqs, G, 1, 0.8, eps)
        cap = int(rng.integers(1, G + 1))
        capped, kpp, _ = run_oracle_cont(oracle_mod, rewards, seqs, G, 1, 0.8, eps, cap)
        labels = chain_classes(adv, eps)
        assert capped.astype(bool).tolist() == cap_by_sort_labels(rewards, uncapped.astype(bool),
                                                                  cap, labels)
