"""GPU parity of grpo_advantage (Eq. 5), grpo_prune (Eqs. 6-9, Algorithm 1) and grpo_compact
with the oracle: bit-exact advantages, keep masks, kept counts and compaction offsets."""
import numpy as np
import pytest

from helpers import golden, pack_rollouts
from mdap_ref import random_structured_prompt
from paper_2609_36932_gb300 import workloads

pytestmark = pytest.mark.gpu


def t(a):
    import torch
    return torch.from_numpy(np.ascontiguousarray(a)).cuda()


def gpu_prune(grpo, rewards, ids, off, G, V, n, tau, cap, dp):
    import torch
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    keep, kpp = grpo.grpo_prune(t(np.asarray(rewards, np.float32)), t(ids), t(off), G, V, n, tau,
                                cap, dp, status=status)
    torch.cuda.synchronize()
    return keep.cpu().numpy(), kpp.cpu().numpy(), int(status.item())


@pytest.mark.parametrize("G", [1, 2, 3, 8, 16, 32, 100, 1024])
@pytest.mark.parametrize("std_mode", [0, 1])
def test_advantage_bit_exact(grpo, oracle_mod, G, std_mode):
    rng = np.random.default_rng(G + std_mode)
    P = 37
    r = rng.choice([0.0, 0.1, 0.5, 0.9, 1.0, 1.5], size=P * G).astype(np.float32)
    r[:G] = 0.7  # one all-equal group
    r[G:2 * G] = rng.standard_normal(G).astype(np.float32) * 1e3
    import torch
    key = torch.empty(P * G, dtype=torch.float64, device="cuda")
    adv, _ = grpo.grpo_advantage(t(r), G, std_mode, key=key)
    o_adv, o_key = oracle_mod.advantage(r, G, std_mode)
    assert np.array_equal(adv.cpu().numpy().view(np.uint32), o_adv.view(np.uint32))
    assert np.array_equal(key.cpu().numpy().view(np.uint64), o_key.view(np.uint64))


@pytest.mark.parametrize("name", list(workloads.WORKLOADS))
def test_advantage_workloads(grpo, oracle_mod, name):
    w = workloads.get(name)
    r = workloads.rewards(w, seed=0)
    adv, _ = grpo.grpo_advantage(t(r), w.G)
    o_adv, _ = oracle_mod.advantage(r, w.G)
    assert np.array_equal(adv.cpu().numpy().view(np.uint32), o_adv.view(np.uint32))


def test_prune_hand_worked(grpo):
    for case in golden("mdap_hand.json")["cases"]:
        ids, off = pack_rollouts(case["rollouts"])
        keep, kpp, st = gpu_prune(grpo, case["rewards"], ids, off, case["G"], 64, case["n"],
                                  case["tau"], case["keep_cap"], case["dp"])
        assert st == 0
        assert keep.tolist() == case["keep"], case["name"]


@pytest.mark.parametrize("n", [1, 2, 3])
@pytest.mark.parametrize("tau", [0.0, 0.5, 0.8, 1.0, 1.5])
def test_prune_random_structured(grpo, oracle_mod, n, tau):
    rng = np.random.default_rng(int(100 * tau) + n)
    for trial in range(6):
        P = int(rng.integers(1, 12))
        G = int(rng.integers(1, 33))
        rewards, seqs = [], []
        for _ in range(P):
            r, s = random_structured_prompt(rng, G, vocab=int(rng.integers(3, 40)), max_len=30,
                                            q=float(rng.choice([0.05, 0.3, 0.7])))
            rewards += r
            seqs += s
        ids, off = pack_rollouts(seqs)
        cap = int(rng.integers(1, G + 2))
        dp = int(rng.choice([1, 2, 3, 8]))
        keep, kpp, st = gpu_prune(grpo, rewards, ids, off, G, 64, n, tau, cap, dp)
        o_keep, o_kpp = oracle_mod.prune(np.asarray(rewards, np.float32), ids, off, G, n, tau, cap, dp)
        assert st == 0
        assert np.array_equal(keep, o_keep), (trial, P, G, cap, dp)
        assert np.array_equal(kpp, o_kpp)


@pytest.mark.parametrize("name", list(workloads.WORKLOADS))
@pytest.mark.parametrize("q", [None, 0.1, 0.3, 0.6])
def test_prune_workloads(grpo, oracle_mod, name, q):
    w = workloads.get(name)
    b = workloads.make_batch(w, seed=0, structured_q=q)
    for n in (1, 2, 3):
        keep, kpp, st = gpu_prune(grpo, b["rewards"], b["ids"], b["off"], w.G, w.V, n, w.tau,
                                  w.keep_cap, 1)
        o_keep, o_kpp = oracle_mod.prune(b["rewards"], b["ids"], b["off"], w.G, n, w.tau,
                                         w.keep_cap, 1)
        assert st == 0
        assert np.array_equal(keep, o_keep) and np.array_equal(kpp, o_kpp)


def test_prune_long_rollouts_sort_in_workspace(grpo, oracle_mod):
    """Rollouts with more windows than the shared-memory sort holds are sorted in the workspace."""
    rng = np.random.default_rng(12)
    G = 4
    base = rng.integers(0, 3000, size=20000)
    seqs = []
    for i in range(G):
        s = base.copy()
        flip = rng.random(s.size) < [0.05, 0.9, 0.1, 0.5][i]
        s[flip] = rng.integers(0, 3000, size=int(flip.sum()))
        seqs.append(s[: [20000, 9000, 8193, 16385][i]].tolist())
    ids, off = pack_rollouts(seqs)
    for n in (1, 2):
        for tau in (0.3, 0.6, 0.9):
            keep, kpp, _ = gpu_prune(grpo, [1, 1, 1, 1], ids, off, G, 3000, n, tau, G, 1)
            o_keep, _ = oracle_mod.prune(np.ones(4, np.float32), ids, off, G, n, tau, G, 1)
            assert np.array_equal(keep, o_keep), (n, tau)


def test_prune_bad_token_flag(grpo):
    ids, off = pack_rollouts([[1, 2, 3], [4, 99, 5]])
    _, _, st = gpu_prune(grpo, [1, 1], ids, off, 2, 50, 1, 0.8, 2, 1)
    assert st & grpo.binding.DEVFLAG_BAD_TOKEN


def test_prune_empty_rollouts(grpo, oracle_mod):
    seqs = [[], [], [3], [], [1, 2], [1, 2]]
    ids, off = pack_rollouts(seqs)
    for n in (1, 2, 3):
        keep, kpp, _ = gpu_prune(grpo, [0, 0, 0, 1, 1, 1], ids, off, 3, 10, n, 0.8, 3, 1)
        o_keep, o_kpp = oracle_mod.prune(np.float32([0, 0, 0, 1, 1, 1]), ids, off, 3, n, 0.8, 3, 1)
        assert np.array_equal(keep, o_keep) and np.array_equal(kpp, o_kpp)


@pytest.mark.parametrize("n", [0, 1, 5, 1023, 1024, 1025, 5000])
def test_compact_bit_exact(grpo, oracle_mod, n):
    import torch
    rng = np.random.default_rng(n)
    L = rng.integers(0, 50, size=n)
    off = np.zeros(n + 1, np.int64)
    off[1:] = np.cumsum(L)
    for p in (0.0, 0.3, 1.0):
        keep = (rng.random(n) < p).astype(np.uint8)
        host = torch.empty(2, dtype=torch.int64, pin_memory=True)
        out = grpo.grpo_compact(t(keep), t(off), counts_host=host)
        torch.cuda.synchronize()
        o = oracle_mod.compact(keep, off)
        K, TK = int(host[0]), int(host[1])
        assert (K, TK) == (o["K"], o["T_kept"])
        assert np.array_equal(out["counts"].cpu().numpy(), [K, TK])
        assert np.array_equal(out["kept_idx"][:K].cpu().numpy(), o["kept_idx"])
        assert np.array_equal(out["kept_off"][:K + 1].cpu().numpy(), o["kept_off"])
        assert np.array_equal(out["src_token"][:TK].cpu().numpy(), o["src_token"])
        assert np.array_equal(out["token_rollout"][:TK].cpu().numpy(), o["token_rollout"])


@pytest.mark.parametrize("eps", [1e-4, 1e-2, 0.5])
@pytest.mark.parametrize("n", [1, 2])
def test_prune_continuous_grouping(grpo, oracle_mod, eps, n):
    """Classes by chained advantages (continuous rewards): the GPU takes grpo_advantage's
    advantages, the oracle its own; both keep masks agree bit for bit."""
    import torch
    from mdap_ref import clustered_rewards
    rng = np.random.default_rng(int(eps * 1e4) + n)
    for trial in range(6):
        P = int(rng.integers(1, 10))
        G = int(rng.integers(2, 33))
        rewards, seqs = [], []
        for _ in range(P):
            _, s = random_structured_prompt(rng, G, vocab=int(rng.integers(3, 30)), max_len=25,
                                            q=float(rng.choice([0.1, 0.4])))
            rewards += clustered_rewards(rng, G, spread=float(rng.choice([1e-5, 1e-3])))
            seqs += s
        ids, off = pack_rollouts(seqs)
        r = np.asarray(rewards, np.float32)
        cap = int(rng.integers(1, G + 2))
        dp = int(rng.choice([1, 3]))
        adv_g, _ = grpo.grpo_advantage(t(r), G)
        status = torch.zeros(1, dtype=torch.int32, device="cuda")
        keep, kpp = grpo.grpo_prune(t(r), t(ids), t(off), G, 64, n, 0.8, cap, dp, status=status,
                                    adv=adv_g, class_eps=eps)
        torch.cuda.synchronize()
        adv_o, _ = oracle_mod.advantage(r, G)
        o_keep, o_kpp = oracle_mod.prune(r, ids, off, G, n, 0.8, cap, dp, adv=adv_o, class_eps=eps)
        assert np.array_equal(keep.cpu().numpy(), o_keep), (trial, P, G, cap, dp)
        assert np.array_equal(kpp.cpu().numpy(), o_kpp)
