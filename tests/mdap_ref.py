"""Independent statements of MDAP used to pin the oracle (no code shared with it):
brute-force enumeration of independent sets over exact Python n-gram sets, and the cap as a
sort rather than a loop."""
from itertools import combinations

import numpy as np


def ngram_set(seq, n):
    return {tuple(seq[t:t + n]) for t in range(len(seq) - n + 1)}


def theta(a, b):
    inter = len(a & b)
    uni = len(a | b)
    return 0.0 if uni == 0 else 1.0 - inter / uni


def visit_order(r):
    r = [float(np.float32(x)) for x in r]
    mean = 0.0
    for x in r:
        mean += x
    mean /= len(r)
    d = [abs(x - mean) for x in r]
    return sorted(range(len(r)), key=lambda i: (-d[i], i)), d


def brute_force_mdap(rewards, seqs, n, tau):
    """Per class, the independent set (no pair with theta < tau) whose membership vector in
    visiting order is lexicographically largest, found by enumerating all subsets."""
    tau = float(np.float32(tau))
    G = len(rewards)
    r = [float(np.float32(x)) for x in rewards]
    order, _ = visit_order(r)
    sets = [ngram_set(list(s), n) for s in seqs]
    keep = [False] * G
    for cls in sorted(set(r)):
        members = [i for i in order if r[i] == cls]
        best = None
        for mask in range(1 << len(members)):
            chosen = [members[k] for k in range(len(members)) if (mask >> k) & 1]
            if any(theta(sets[a], sets[b]) < tau for a, b in combinations(chosen, 2)):
                continue
            outside = [x for x in members if x not in chosen]
            if any(all(theta(sets[x], sets[c]) >= tau for c in chosen) for x in outside):
                continue  # not maximal
            vec = tuple((mask >> k) & 1 for k in range(len(members)))
            if best is None or vec > best[0]:
                best = (vec, chosen)
        for i in best[1]:
            keep[i] = True
    return keep


def cap_by_sort(rewards, keep, cap):
    """Round-robin cap restated as a sort: each kept rollout gets (its rank inside its class,
    its class's rank), classes ranked by |r - mean| descending then lowest member; the cap
    smallest keys stay."""
    r = [float(np.float32(x)) for x in rewards]
    _, d = visit_order(r)
    kept = [i for i in range(len(r)) if keep[i]]
    if len(kept) <= cap:
        return list(keep)
    classes = sorted({r[i] for i in kept}, key=lambda c: (-d[[i for i in kept if r[i] == c][0]],
                                                           min(i for i in kept if r[i] == c)))
    keys = []
    for i in kept:
        same = [j for j in kept if r[j] == r[i]]
        keys.append(((same.index(i), classes.index(r[i])), i))
    chosen = {i for _, i in sorted(keys)[:cap]}
    return [i in chosen for i in range(len(r))]


def random_structured_prompt(rng, G, vocab, max_len, q):
    templ = rng.integers(0, vocab, size=max_len)
    seqs = []
    for _ in range(G):
        L = int(rng.integers(0, max_len + 1))
        s = templ[:L].copy()
        flip = rng.random(L) < q
        s[flip] = rng.integers(0, vocab, size=int(flip.sum()))
        seqs.append([int(t) for t in s])
    rewards = [float(x) for x in rng.choice([0.0, 0.5, 1.0], size=G)]
    return rewards, seqs


def chain_classes(adv, eps):
    """Continuous-reward classes: sort by advantage (ties by index), start a new class where the
    gap to the previous value is >= eps; label = smallest index in the class."""
    a = [float(np.float32(x)) for x in adv]
    order = sorted(range(len(a)), key=lambda i: (a[i], i))
    chain = {}
    c = 0
    for k, i in enumerate(order):
        if k > 0 and a[i] - a[order[k - 1]] >= float(np.float32(eps)):
            c += 1
        chain[i] = c
    return [min(j for j in range(len(a)) if chain[j] == chain[i]) for i in range(len(a))]


def brute_force_mdap_labels(rewards, seqs, n, tau, labels):
    """brute_force_mdap with explicit class labels; members of a class are visited by
    |r - mean| descending, lower index first."""
    tau = float(np.float32(tau))
    G = len(rewards)
    order, _ = visit_order(rewards)
    sets = [ngram_set(list(s), n) for s in seqs]
    keep = [False] * G
    for cls in sorted(set(labels)):
        members = [i for i in order if labels[i] == cls]
        best = None
        for mask in range(1 << len(members)):
            chosen = [members[k] for k in range(len(members)) if (mask >> k) & 1]
            if any(theta(sets[a], sets[b]) < tau for a, b in combinations(chosen, 2)):
                continue
            vec = tuple((mask >> k) & 1 for k in range(len(members)))
            if best is None or vec > best[0]:
                best = (vec, chosen)
        for i in best[1]:
            keep[i] = True
    return keep


def cap_by_sort_labels(rewards, keep, cap, labels):
    """The cap as a sort: key = (rank of the rollout among its class's kept members in visiting
    order, visiting position of the class's first kept member)."""
    order, _ = visit_order(rewards)
    pos = {i: k for k, i in enumerate(order)}
    kept = [i for i in range(len(keep)) if keep[i]]
    if len(kept) <= cap:
        return list(keep)
    keys = []
    for i in kept:
        same = sorted((j for j in kept if labels[j] == labels[i]), key=lambda j: pos[j])
        keys.append(((same.index(i), pos[same[0]]), i))
    chosen = {i for _, i in sorted(keys)[:cap]}
    return [i in chosen for i in range(len(keep))]


def clustered_rewards(rng, G, spread=1e-5):
    """Continuous rewards around a few centres: advantage gaps inside a cluster are ~1e-5."""
    centres = rng.random(int(rng.integers(1, 4)))
    r = centres[rng.integers(0, centres.size, size=G)] + spread * rng.standard_normal(G)
    return [float(x) for x in r.astype(np.float32)]
