"""Seeded synthetic workloads shaped like the paper's GRPO batches.

This module only draws inputs: rollout lengths, token ids, rewards, logits and the old/reference
log-probabilities.  It holds none of the path's arithmetic (no advantage, pruning, compaction or
loss code) and serves both the CUDA path and the CPU oracle with the same arrays.

The five workloads (sizes, value distributions and structure of the batches the paper trains on:
groups of 8-16 rollouts per prompt, a Qwen2.5-size vocabulary of 152064 tokens, binary
accuracy+format rewards, Sec. 4 and Table 6) are:

  tiny    4 prompts x G=4,  lengths U{8..32},   V=1024,   f32 logits N(0, 2^2)
  small   8 prompts x G=8,  lengths U{64..512}, V=32000,  bf16 logits N(0, 3^2), +8 on one id/row
  qwen    16 x G=8,  lengths lognormal(median 384, sigma 0.4) <= 1024,  V=152064, Zipf(1.1) bias
  large   16 x G=16, lengths lognormal(median 768) <= 2048, keep ratio 0.25
  long    16 x G=16, lengths lognormal(median 1024) <= 4096, f32 dlogits

For the output layer fused with the loss, the same batches carry hidden states of width 3584
(Qwen2.5-7B) ~ N(0, 1) and an output-layer weight ~ N(0, 4 / D), both bf16, in place of logits.

Host arrays come from numpy's PCG64 seeded with (seed, stream id); logits come from torch's
generator on the target device, seeded per block of 256 token rows, so any row range can be
regenerated on its own.  old_logp and ref_logp are the current log-probability plus Gaussian
noise (sd 0.05 and 0.1); the current log-probability is taken with torch.logsumexp in f32 only
to centre that noise (any error there changes the inputs, which both sides share, not a result).
"""
from __future__ import annotations

import dataclasses
import math

import numpy as np

ROW_BLOCK = 256  # rows per independently seeded logits block


@dataclasses.dataclass(frozen=True)
class Workload:
    name: str
    P: int
    G: int
    length: tuple          # ("uniform", lo, hi) or ("lognormal", median, sigma, cap)
    V: int
    logits_kind: str       # "normal" | "normal_peak" | "zipf"
    logits_dtype: str      # "f32" | "bf16"
    logits_sd: float
    reward_kind: str       # "bern05" | "bern_p" | "acc_fmt"
    zero_adv_frac: float
    keep_ratio: float
    dlogits_dtype: str     # "f32" | "bf16"
    eps: float = 0.2
    beta: float = 0.04
    tau: float = 0.8
    ngram_n: int = 1
    chunk_rows: int = 0    # >0: the loss is run over kept rows in chunks of this many rows

    @property
    def n_rollouts(self) -> int:
        return self.P * self.G

    @property
    def keep_cap(self) -> int:
        """Per-prompt cap max(1, ceil(keep_ratio * G)) from the workload's keep ratio."""
        return max(1, int(math.ceil(self.keep_ratio * self.G - 1e-9)))

    @property
    def in_bytes(self) -> int:
        return 4 if self.logits_dtype == "f32" else 2

    @property
    def out_bytes(self) -> int:
        return 4 if self.dlogits_dtype == "f32" else 2


WORKLOADS = {
    "tiny": Workload("tiny", 4, 4, ("uniform", 8, 32), 1024, "normal", "f32", 2.0, "bern05", 0.0,
                     0.5, "f32"),
    "small": Workload("small", 8, 8, ("uniform", 64, 512), 32000, "normal_peak", "bf16", 3.0,
                      "bern_p", 0.0, 0.5, "bf16"),
    "qwen": Workload("qwen", 16, 8, ("lognormal", 384, 0.4, 1024), 152064, "zipf", "bf16", 2.0,
                     "acc_fmt", 0.25, 0.5, "bf16"),
    "large": Workload("large", 16, 16, ("lognormal", 768, 0.4, 2048), 152064, "zipf", "bf16", 2.0,
                      "acc_fmt", 0.30, 0.25, "bf16"),
    "long": Workload("long", 16, 16, ("lognormal", 1024, 0.4, 4096), 152064, "zipf", "bf16", 2.0,
                     "acc_fmt", 0.25, 0.5, "f32", chunk_rows=16384),
}
# The same five, by position.
BY_INDEX = ["tiny", "small", "qwen", "large", "long"]


def get(name_or_index) -> Workload:
    if isinstance(name_or_index, int) or str(name_or_index).isdigit():
        return WORKLOADS[BY_INDEX[int(name_or_index)]]
    return WORKLOADS[name_or_index]


def _rng(seed: int, stream: int) -> np.random.Generator:
    return np.random.default_rng([int(seed), int(stream)])


def lengths(w: Workload, seed: int = 0) -> np.ndarray:
    rng = _rng(seed, 1)
    n = w.n_rollouts
    if w.length[0] == "uniform":
        _, lo, hi = w.length
        L = rng.integers(lo, hi + 1, size=n)
    else:
        _, median, sigma, cap = w.length
        L = np.rint(median * np.exp(sigma * rng.standard_normal(n)))
        L = np.clip(L, 1, cap)
    return L.astype(np.int64)


def rewards(w: Workload, seed: int = 0) -> np.ndarray:
    rng = _rng(seed, 2)
    P, G = w.P, w.G
    if w.reward_kind == "bern05":
        r = (rng.random((P, G)) < 0.5).astype(np.float64)
    elif w.reward_kind == "bern_p":
        p = rng.random(P)
        r = (rng.random((P, G)) < p[:, None]).astype(np.float64)
    else:  # accuracy (0.9) plus format (0.1)
        p = rng.random(P)
        acc = (rng.random((P, G)) < p[:, None]).astype(np.float64)
        fmt = (rng.random((P, G)) < 0.8).astype(np.float64)
        r = 0.9 * acc + 0.1 * fmt
    n_zero = int(round(w.zero_adv_frac * P))
    if n_zero:
        for q in rng.choice(P, n_zero, replace=False):
            r[q, :] = r[q, 0]
    return r.astype(np.float32).ravel()


def token_ids(w: Workload, L: np.ndarray, seed: int = 0, structured_q=None) -> np.ndarray:
    """Completion token ids, packed.  structured_q: per-token resample probability of a per-prompt
    template (rollouts of one prompt then share n-grams, which exercises Eq. 8's pruning)."""
    rng = _rng(seed, 3)
    T = int(L.sum())
    if structured_q is None:
        return rng.integers(0, w.V, size=T, dtype=np.int64).astype(np.int32)
    out = np.empty(T, np.int32)
    pos = 0
    for q in range(w.P):
        Lg = L[q * w.G:(q + 1) * w.G]
        templ = rng.integers(0, w.V, size=int(Lg.max()), dtype=np.int64)
        for i in range(w.G):
            li = int(Lg[i])
            seq = templ[:li].copy()
            flip = rng.random(li) < structured_q
            seq[flip] = rng.integers(0, w.V, size=int(flip.sum()), dtype=np.int64)
            out[pos:pos + li] = seq
            pos += li
    return out


def make_batch(w: Workload, seed: int = 0, structured_q=None) -> dict:
    """Host arrays of one step: rewards, lengths, offsets, ids (= sampled tokens y), noise."""
    L = lengths(w, seed)
    off = np.zeros(w.n_rollouts + 1, np.int64)
    np.cumsum(L, out=off[1:])
    T = int(off[-1])
    rng = _rng(seed, 4)
    return dict(
        workload=w, seed=seed, rewards=rewards(w, seed), lengths=L, off=off, T=T,
        ids=token_ids(w, L, seed, structured_q),
        noise_old=(0.05 * rng.standard_normal(T)).astype(np.float32),
        noise_ref=(0.1 * rng.standard_normal(T)).astype(np.float32),
    )


def _torch():
    import torch
    return torch


_zipf_cache: dict = {}


def _zipf_bias(w: Workload, seed: int, device):
    key = (w.V, seed, str(device))
    if key not in _zipf_cache:
        torch = _torch()
        rank = _rng(seed, 5).permutation(w.V) + 1
        bias = -1.1 * np.log(rank.astype(np.float64))
        _zipf_cache.clear()
        _zipf_cache[key] = torch.from_numpy(bias.astype(np.float32)).to(device)
    return _zipf_cache[key]


def logits_block(w: Workload, seed: int, block: int, device):
    """Rows [block*ROW_BLOCK, (block+1)*ROW_BLOCK) of the full [T, V] logits (f32 tensor)."""
    torch = _torch()
    g = torch.Generator(device=device)
    g.manual_seed((int(seed) * 1_000_003 + 7919 * int(block) + 17) % (2**63))
    x = torch.randn((ROW_BLOCK, w.V), generator=g, device=device, dtype=torch.float32)
    x.mul_(w.logits_sd)
    if w.logits_kind == "zipf":
        x.add_(_zipf_bias(w, seed, device))
    elif w.logits_kind == "normal_peak":
        peak = torch.randint(0, w.V, (ROW_BLOCK,), generator=g, device=device)
        x[torch.arange(ROW_BLOCK, device=device), peak] += 8.0
    return x


def logits_rows(w: Workload, seed: int, rows, device, out=None):
    """Logits of the given token rows (a range or an int64 index array), in the workload's dtype.

    Each row's values depend only on (seed, row), not on which other rows are asked for."""
    torch = _torch()
    dt = torch.float32 if w.logits_dtype == "f32" else torch.bfloat16
    if isinstance(rows, range):
        idx = np.arange(rows.start, rows.stop, dtype=np.int64)
    else:
        idx = np.asarray(rows, np.int64)
    n = idx.size
    if out is None:
        out = torch.empty((n, w.V), dtype=dt, device=device)
    if n == 0:
        return out
    blocks = np.unique(idx // ROW_BLOCK)
    idx_t = torch.from_numpy(idx).to(device)
    for b in blocks:
        blk = logits_block(w, seed, int(b), device).to(dt)
        sel = np.nonzero(idx // ROW_BLOCK == b)[0]
        sel_t = torch.from_numpy(sel).to(device)
        out[sel_t] = blk[idx_t[sel_t] - int(b) * ROW_BLOCK]
        del blk
    return out


def old_ref_logp(logits, y, noise_old, noise_ref):
    """old_logp / ref_logp for rows of `logits` (torch, any device): centred on the current
    log-probability of the sampled token (torch.logsumexp in f32) plus the given noise."""
    torch = _torch()
    dev = logits.device
    n = logits.shape[0]
    center = torch.empty(n, dtype=torch.float32, device=dev)
    yt = torch.as_tensor(np.asarray(y, np.int64), device=dev)
    step = 4096
    for s in range(0, n, step):
        blk = logits[s:s + step].float()
        center[s:s + step] = blk.gather(1, yt[s:s + step, None])[:, 0] - torch.logsumexp(blk, 1)
    old = center + torch.as_tensor(np.asarray(noise_old, np.float32), device=dev)
    ref = center + torch.as_tensor(np.asarray(noise_ref, np.float32), device=dev)
    return old, ref


# Output-layer inputs: a batch's tokens as hidden states of Qwen2.5-7B's width.
LMHEAD_D = 3584


def lmhead_hidden(n_rows: int, D: int, seed: int, device, rows=None):
    """Hidden states [n, D] ~ N(0, 1) in bf16 (torch's generator on `device`, seeded per block of
    ROW_BLOCK rows, so any rows can be regenerated on their own).  rows: a range or index array
    (default: range(n_rows))."""
    torch = _torch()
    idx = np.arange(n_rows, dtype=np.int64) if rows is None else (
        np.arange(rows.start, rows.stop, dtype=np.int64) if isinstance(rows, range)
        else np.asarray(rows, np.int64))
    out = torch.empty((idx.size, D), dtype=torch.bfloat16, device=device)
    for b in np.unique(idx // ROW_BLOCK):
        g = torch.Generator(device=device)
        g.manual_seed((int(seed) * 1_000_033 + 104_729 * int(b) + 29) % (2**63))
        blk = torch.randn((ROW_BLOCK, D), generator=g, device=device).to(torch.bfloat16)
        sel = np.nonzero(idx // ROW_BLOCK == b)[0]
        out[torch.from_numpy(sel).to(device)] = blk[torch.from_numpy(idx[sel] - int(b) * ROW_BLOCK).to(device)]
    return out


def lmhead_weight(V: int, D: int, seed: int, device, logit_sd: float = 2.0):
    """Output-layer weight [V, D] ~ N(0, logit_sd^2 / D) in bf16, so that the logits h W^T of
    N(0, 1) hidden states have standard deviation about logit_sd (2, like the qwen logits)."""
    torch = _torch()
    g = torch.Generator(device=device)
    g.manual_seed((int(seed) * 7_919 + 3) % (2**63))
    w = torch.empty((V, D), dtype=torch.bfloat16, device=device)
    step = 8192
    for s in range(0, V, step):
        n = min(step, V - s)
        w[s:s + n] = (torch.randn((n, D), generator=g, device=device) * (logit_sd / math.sqrt(D))).to(
            torch.bfloat16)
    return w


def lmhead_old_ref(hidden, weight, y, noise_old, noise_ref):
    """old_logp / ref_logp for rows of `hidden`: the current log-probability of the sampled token
    (logits h W^T and torch.logsumexp in f32, block by block) plus the given noise."""
    torch = _torch()
    dev = hidden.device
    n = hidden.shape[0]
    center = torch.empty(n, dtype=torch.float32, device=dev)
    yt = torch.as_tensor(np.asarray(y, np.int64), device=dev)
    wt = weight if dev.type == "cuda" else weight.float()
    step = 2048
    for s in range(0, n, step):
        h = hidden[s:s + step] if dev.type == "cuda" else hidden[s:s + step].float()
        blk = (h @ wt.t()).float()
        center[s:s + step] = blk.gather(1, yt[s:s + step, None])[:, 0] - torch.logsumexp(blk, 1)
        del blk
    old = center + torch.as_tensor(np.asarray(noise_old, np.float32), device=dev)
    ref = center + torch.as_tensor(np.asarray(noise_ref, np.float32), device=dev)
    return old, ref


def ars_pruning_ratios(seed: int, steps: int, P: int) -> np.ndarray:
    """Synthetic per-step, per-prompt pruning ratios U(0.1, 0.6) for the ARS closed loop."""
    return _rng(seed, 6).uniform(0.1, 0.6, size=(steps, P))


def synthetic_kept_counts(ratios_row: np.ndarray, n: int) -> np.ndarray:
    """Kept counts of one step when a fraction `ratios_row` of n rollouts is pruned:
    clamp(round_half_even((1 - ratio) * n), 1, n)."""
    k = np.rint((1.0 - ratios_row) * n).astype(np.int64)
    return np.clip(k, 1, n).astype(np.int32)
