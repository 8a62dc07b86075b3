"""Whole-step parity on the five workloads, in the launch configuration bench.py times:
advantage -> prune -> compact -> loss over the kept rows.  'tiny' and 'small' are compared
with the oracle row by row in full.  The three Qwen-vocabulary workloads at full size are
compared with the oracle on every kept row's log-probability and loss term and on the total
loss, and on the dlogits of at least 1024 rows (every row of two whole kept rollouts among
them)."""
import dataclasses

import numpy as np
import pytest

from loss_compare import LOSS_RTOL, allowed_ulps, compare, compare_rows
from paper_2609_36932_gb300 import workloads
from paper_2609_36932_gb300.pipeline import GrpoStep, StepParams

pytestmark = pytest.mark.gpu


def build(name, seed=0, chunk_rows=None, **overrides):
    import torch
    w = workloads.get(name)
    b = workloads.make_batch(w, seed)
    dev = torch.device("cuda", 0)
    rewards = torch.from_numpy(b["rewards"]).to(dev)
    ids = torch.from_numpy(b["ids"]).to(dev)
    off = torch.from_numpy(b["off"]).to(dev)
    logits = workloads.logits_rows(w, seed, range(b["T"]), dev)
    old, ref = workloads.old_ref_logp(logits, b["ids"], b["noise_old"], b["noise_ref"])
    p = StepParams(G=w.G, V=w.V, ngram_n=w.ngram_n, tau=w.tau, keep_cap=w.keep_cap,
                   eps_low=w.eps, eps_high=w.eps, beta=w.beta, dlogits_dtype=w.dlogits_dtype,
                   chunk_rows=w.chunk_rows if chunk_rows is None else chunk_rows)
    p = dataclasses.replace(p, **overrides)
    step = GrpoStep(p, rewards, ids, off, logits, old, ref)
    return w, b, step, dict(logits=logits, old=old.cpu().numpy(), ref=ref.cpu().numpy())


def host_bits(t):
    import torch
    if t.dtype == torch.bfloat16:
        return t.view(torch.int16).cpu().numpy().view(np.uint16)
    return t.cpu().numpy()


def check_selection(oracle_mod, w, b, step):
    adv, _ = oracle_mod.advantage(b["rewards"], w.G)
    keep, kpp = oracle_mod.prune(b["rewards"], b["ids"], b["off"], w.G, w.ngram_n, w.tau,
                                 w.keep_cap, 1)
    comp = oracle_mod.compact(keep, b["off"])
    assert np.array_equal(step.adv.cpu().numpy().view(np.uint32), adv.view(np.uint32))
    assert np.array_equal(step.keep.cpu().numpy(), keep)
    assert np.array_equal(step.kpp[:w.P].cpu().numpy(), kpp)
    assert (step.K, step.T_kept) == (comp["K"], comp["T_kept"])
    src, tr = step.kept_rows()
    assert np.array_equal(src, comp["src_token"]) and np.array_equal(tr, comp["token_rollout"])
    return adv, comp


@pytest.mark.parametrize("name", ["tiny", "small"])
def test_full_comparison(oracle_mod, name):
    import torch
    w, b, step, h = build(name)
    step.run()
    torch.cuda.synchronize()
    assert int(step.status.item()) == 0
    adv, comp = check_selection(oracle_mod, w, b, step)
    TK = step.T_kept
    lg = host_bits(h["logits"])
    ref = oracle_mod.loss(lg, w.V, b["ids"], h["old"], h["ref"], adv, comp["token_rollout"],
                          row_index=comp["src_token"], eps_low=w.eps, eps_high=w.eps,
                          beta=w.beta, denom_tokens=TK,
                          dlogits_dtype=1 if w.dlogits_dtype == "bf16" else 0)
    compare(step.logp[:TK].cpu().numpy(), host_bits(step.dlogits[:TK]), float(step.loss.item()),
            ref, w.dlogits_dtype, gpu_row_loss=step.row_loss[:TK].cpu().numpy(),
            cond=dict(ref_logp=h["ref"][comp["src_token"]], beta=w.beta))


def oracle_all_rows(oracle_mod, w, b, h, adv, comp, TK, block=8192):
    """The oracle over every kept row, without dlogits: logits copied to the host a block of rows
    at a time.  Returns its dict (logp, rho, row_loss per row and the total loss)."""
    import torch
    st, tr = comp["src_token"], comp["token_rollout"]
    out = dict(logp=np.empty(TK), rho=np.empty(TK), row_loss=np.empty(TK), loss=0.0)
    for r0 in range(0, TK, block):
        r1 = min(TK, r0 + block)
        src = st[r0:r1]
        lg = host_bits(h["logits"][torch.from_numpy(src).cuda()])
        o = oracle_mod.loss(lg, w.V, b["ids"][src], h["old"][src], h["ref"][src], adv, tr[r0:r1],
                            eps_low=w.eps, eps_high=w.eps, beta=w.beta, denom_tokens=TK,
                            want_dlogits=False)
        for k in ("logp", "rho", "row_loss"):
            out[k][r0:r1] = o[k]
        out["loss"] += o["loss"]
    return out


def sample_rows(comp, K, TK, n=1024, seed=7):
    """Every row of two whole kept rollouts (the first and the longest), the first and last 8
    rows, and random rows up to n."""
    ko = comp["kept_off"]
    lens = np.diff(ko[:K + 1])
    whole = [0, int(np.argmax(lens))]
    rows = [np.arange(ko[k], ko[k + 1]) for k in whole]
    rows += [np.arange(min(8, TK)), np.arange(max(TK - 8, 0), TK)]
    have = np.unique(np.concatenate(rows))
    rng = np.random.default_rng(seed)
    rest = np.setdiff1d(np.arange(TK), have)
    extra = rng.choice(rest, size=min(rest.size, max(n - have.size, 0)), replace=False)
    return np.unique(np.concatenate([have, extra])).astype(np.int64), whole


@pytest.mark.parametrize("name", ["qwen", "large", "long"])
def test_full_size_against_oracle(oracle_mod, name):
    import torch
    w, b, step, h = build(name, chunk_rows=0)
    step.run()
    torch.cuda.synchronize()
    assert int(step.status.item()) == 0
    adv, comp = check_selection(oracle_mod, w, b, step)
    TK, K = step.T_kept, step.K
    logp = step.logp[:TK].cpu().numpy()
    row_loss = step.row_loss[:TK].cpu().numpy()
    total = float(step.loss.item())
    # every kept row: logp, loss term and the total loss against the oracle's
    o_all = oracle_all_rows(oracle_mod, w, b, h, adv, comp, TK)
    _, n_skip, logp_err = compare_rows(logp, total, row_loss, o_all, w.eps, w.eps)
    print("%s: %d kept rows, max logp error %.3g, %d clip-boundary rows, loss %.12g (oracle %.12g)"
          % (name, TK, logp_err, n_skip, total, o_all["loss"]))
    # dlogits: >= 1024 rows, every row of two whole kept rollouts among them
    rows, whole = sample_rows(comp, K, TK)
    ko = comp["kept_off"]
    assert all(np.isin(np.arange(ko[k], ko[k + 1]), rows).all() for k in whole)
    assert rows.size >= min(1024, TK)
    src = comp["src_token"][rows]
    lg = host_bits(h["logits"][torch.from_numpy(src).cuda()])
    o = oracle_mod.loss(lg, w.V, b["ids"][src], h["old"][src], h["ref"][src], adv,
                        comp["token_rollout"][rows], eps_low=w.eps, eps_high=w.eps, beta=w.beta,
                        denom_tokens=TK, dlogits_dtype=1 if w.dlogits_dtype == "bf16" else 0)
    idx = torch.from_numpy(rows).cuda()
    res = compare(logp[rows], host_bits(step.dlogits[:TK][idx]), None, o, w.dlogits_dtype,
                  gpu_row_loss=row_loss[rows], cond=dict(ref_logp=h["ref"][src], beta=w.beta))
    print("%s: dlogits of %d rows, worst %s, %d rows with an ill-conditioned g_t"
          % (name, rows.size, res["worst"], res["widened_rows"]))
    # the same step again is bitwise identical
    loss0 = total
    step.run()
    torch.cuda.synchronize()
    assert float(step.loss.item()) == loss0
    if name == "long":
        # chunks of 16384 kept rows sharing one dlogits buffer sum to the single call's loss
        d_last = step.dlogits[:TK][-100:].clone()
        step.p.chunk_rows = w.chunk_rows
        step.dlogits = None
        step.run()
        torch.cuda.synchronize()
        assert float(step.loss.item()) == loss0
        assert np.array_equal(step.logp[:TK].cpu().numpy(), logp)
        assert np.array_equal(step.row_loss[:TK].cpu().numpy(), row_loss)
        n_last = TK - (TK - 1) // w.chunk_rows * w.chunk_rows
        assert torch.equal(step.dlogits[:n_last][-100:], d_last)


@pytest.mark.parametrize("name,ratio", [("tiny", "token"), ("qwen", "token"), ("tiny", "sequence"),
                                        ("small", "sequence")])
def test_graph_mode_equals_host_synced_step(name, ratio):
    """The step captured as two CUDA graphs (the loss reads the kept counts on the device) gives
    the same selection, loss, logp and dlogits as the host-synced step, on two replays, for the
    token-level loss and for GSPO's sequence-level loss."""
    import torch
    w, b, step, h = build(name, chunk_rows=0, ratio_level=ratio)
    step.run()
    torch.cuda.synchronize()
    TK = step.T_kept
    ref_loss = float(step.loss.item())
    ref_logp = step.logp[:TK].clone()
    ref_dl = step.dlogits[:TK].clone()
    ref_keep = step.keep.clone()
    step.capture()
    for _ in range(2):
        step.loss.zero_()
        assert step.run_graph() == TK
        assert float(step.loss.item()) == ref_loss
        assert torch.equal(step.keep, ref_keep)
        assert torch.equal(step.logp[:TK], ref_logp)
        assert torch.equal(step.dlogits[:TK], ref_dl)
        assert int(step.status.item()) == 0


VARIANTS = {
    # DP fill to a multiple of 7, a keep cap of 3, Eq. 1's per-sequence mean, clip-higher
    # widths and no KL term, bigram sets
    "small-dp7-cap3-seqmean-cliphigher": ("small", dict(ngram_n=2, keep_cap=3, dp_divisor=7,
                                                         agg_mode=1, eps_low=0.2, eps_high=0.28,
                                                         beta=0.0)),
    # population std, trigram sets, a tight tau, continuous-reward grouping
    "tiny-popstd-tri-classeps": ("tiny", dict(std_mode=1, ngram_n=3, tau=0.3, class_eps=1e-4,
                                              dp_divisor=3)),
}


@pytest.mark.parametrize("variant", list(VARIANTS))
def test_step_variants(oracle_mod, variant):
    """The whole step under non-default step parameters, compared with the oracle in full, then
    replayed as CUDA graphs and compared with itself bit for bit."""
    import torch
    name, kw = VARIANTS[variant]
    w, b, step, h = build(name, chunk_rows=0, **kw)
    p = step.p
    step.run()
    torch.cuda.synchronize()
    assert int(step.status.item()) == 0
    adv, _ = oracle_mod.advantage(b["rewards"], w.G, p.std_mode)
    keep, kpp = oracle_mod.prune(b["rewards"], b["ids"], b["off"], w.G, p.ngram_n, p.tau,
                                 p.keep_cap, p.dp_divisor, adv=adv, class_eps=p.class_eps)
    comp = oracle_mod.compact(keep, b["off"])
    assert np.array_equal(step.adv.cpu().numpy().view(np.uint32), adv.view(np.uint32))
    assert np.array_equal(step.keep.cpu().numpy(), keep)
    assert np.array_equal(step.kpp[:w.P].cpu().numpy(), kpp)
    assert (step.K, step.T_kept) == (comp["K"], comp["T_kept"])
    assert comp["K"] % p.dp_divisor == 0
    TK = step.T_kept
    ref = oracle_mod.loss(host_bits(h["logits"]), w.V, b["ids"], h["old"], h["ref"], adv,
                          comp["token_rollout"], row_index=comp["src_token"],
                          eps_low=p.eps_low, eps_high=p.eps_high, beta=p.beta,
                          agg_mode=p.agg_mode, denom_tokens=TK, seq_off=b["off"],
                          n_seq=comp["K"], dlogits_dtype=1 if w.dlogits_dtype == "bf16" else 0)
    compare(step.logp[:TK].cpu().numpy(), host_bits(step.dlogits[:TK]), float(step.loss.item()),
            ref, w.dlogits_dtype, eps_low=p.eps_low, eps_high=p.eps_high,
            gpu_row_loss=step.row_loss[:TK].cpu().numpy(),
            cond=dict(ref_logp=h["ref"][comp["src_token"]], beta=p.beta))
    loss0, dl0 = float(step.loss.item()), step.dlogits[:TK].clone()
    step.capture()
    assert step.run_graph() == TK
    assert float(step.loss.item()) == loss0 and torch.equal(step.dlogits[:TK], dl0)


@pytest.mark.parametrize("name", ["tiny", "small"])
def test_step_with_every_group_zero_advantage(oracle_mod, name):
    """Every prompt's rewards equal (a different value per prompt): every advantage is 0, each
    group is one advantage class, and the loss and dlogits carry the KL term alone; the step
    matches the oracle in full."""
    import torch
    w, b, step, h = build(name, chunk_rows=0)
    r = np.repeat(np.arange(w.P, dtype=np.float32) * 0.25, w.G)
    b["rewards"] = r
    step.rewards.copy_(torch.from_numpy(r))
    step.run()
    torch.cuda.synchronize()
    assert int(step.status.item()) == 0
    adv, comp = check_selection(oracle_mod, w, b, step)
    assert np.all(adv == 0) and comp["K"] >= w.P
    TK = step.T_kept
    ref = oracle_mod.loss(host_bits(h["logits"]), w.V, b["ids"], h["old"], h["ref"], adv,
                          comp["token_rollout"], row_index=comp["src_token"], eps_low=w.eps,
                          eps_high=w.eps, beta=w.beta, denom_tokens=TK,
                          dlogits_dtype=1 if w.dlogits_dtype == "bf16" else 0)
    compare(step.logp[:TK].cpu().numpy(), host_bits(step.dlogits[:TK]), float(step.loss.item()),
            ref, w.dlogits_dtype, gpu_row_loss=step.row_loss[:TK].cpu().numpy(),
            cond=dict(ref_logp=h["ref"][comp["src_token"]], beta=w.beta))


def test_upload_kept_copies_only_kept_rows():
    """grpo_upload_kept: kept rollouts' rows arrive intact, pruned rows keep their old contents,
    one copy per run of consecutive kept rollouts, on two row widths."""
    import torch
    from paper_2609_36932_gb300 import binding as B
    rng = np.random.default_rng(21)
    for n, width, dtype in ((37, 1000, torch.bfloat16), (200, 33, torch.float32)):
        lens = rng.integers(0, 9, size=n)
        off = torch.from_numpy(np.concatenate([[0], np.cumsum(lens)]).astype(np.int64))
        T = int(off[-1])
        keep = torch.from_numpy((rng.random(n) < 0.5).astype(np.uint8))
        src = torch.randn(T, width).to(dtype).pin_memory()
        dst = torch.full((T, width), -7.0, dtype=dtype, device="cuda")
        nbytes, copies = B.grpo_upload_kept(src, dst, keep, off)
        torch.cuda.synchronize()
        kept_row = np.repeat(keep.numpy().astype(bool), lens)
        got = dst.cpu()
        assert torch.equal(got[torch.from_numpy(kept_row)], src[torch.from_numpy(kept_row)])
        assert bool((got[torch.from_numpy(~kept_row)] == -7.0).all())
        assert nbytes == int(kept_row.sum()) * width * src.element_size()
        # runs of kept rollouts, counting only runs that hold at least one token
        runs, r = 0, 0
        kk = keep.numpy().astype(bool)
        while r < n:
            if not kk[r]:
                r += 1
                continue
            e = r
            while e < n and kk[e]:
                e += 1
            runs += int(lens[r:e].sum() > 0)
            r = e
        assert copies == runs and runs >= 1


@pytest.mark.parametrize("name,graph,groups", [("tiny", False, 1), ("tiny", True, 4),
                                               ("small", True, 1), ("small", False, 4),
                                               ("qwen", True, 4)])
def test_host_inputs_step_equals_resident_step(name, graph, groups):
    """A step from pinned host inputs copies only the kept rollouts' logit rows, whole (groups = 1)
    or in groups whose loss starts as each lands (groups = 4).  It gives the resident step's
    selection, loss, logp and dlogits bit for bit, although every device input was poisoned
    beforehand (NaN logits everywhere): no pruned row is read."""
    import torch
    w, b, step, h = build(name, chunk_rows=0)
    step.run()
    torch.cuda.synchronize()
    TK, K = step.T_kept, step.K
    ref_loss = float(step.loss.item())
    ref_logp, ref_dl = step.logp[:TK].clone(), step.dlogits[:TK].clone()
    ref_keep = step.keep.clone()
    host = {}
    for k in ("rewards", "ids", "off", "old", "ref", "logits"):
        d = getattr(step, k)
        host[k] = torch.empty(d.shape, dtype=d.dtype, pin_memory=True)
        host[k].copy_(d)
    if graph:
        step.capture()
    step.logits.fill_(float("nan"))
    for t in (step.old, step.ref, step.rewards):
        t.fill_(float("nan"))
    step.ids.fill_(-1)
    step.off.fill_(0)
    step.status.zero_()
    loss_host = torch.empty(1, dtype=torch.float64, pin_memory=True)
    small = sum(host[k].numel() * host[k].element_size() for k in step.SMALL_INPUTS)
    for _ in range(2):
        h2d, d2h = step.run_from_host(host, loss_host, overlap_groups=groups)
        assert (step.T_kept, step.K) == (TK, K)
        assert float(loss_host.item()) == ref_loss
        assert torch.equal(step.keep, ref_keep)
        assert torch.equal(step.logp[:TK], ref_logp) and torch.equal(step.dlogits[:TK], ref_dl)
        assert int(step.status.item()) == 0
        assert h2d == small + TK * w.V * host["logits"].element_size()
        n = step.keep.numel()
        assert d2h == 16 + 4 * step.P + n + 8 * (n + 1) + 8


@pytest.mark.parametrize("name", ["tiny", "small"])
def test_gspo_step_matches_oracle(oracle_mod, name):
    """The whole step with GSPO's sequence-level ratio: the compaction's kept offsets and kept
    rollout indices are the sequences; loss, logp, ratios and dlogits against the oracle."""
    import torch
    from test_gpu_gspo import RATIO_RTOL
    w, b, step, h = build(name, chunk_rows=0, ratio_level="sequence", eps_low=0.2,
                          eps_high=0.28)
    step.run()
    torch.cuda.synchronize()
    assert int(step.status.item()) == 0
    adv, comp = check_selection(oracle_mod, w, b, step)
    TK, K = step.T_kept, step.K
    ref = oracle_mod.gspo_loss(host_bits(h["logits"]), w.V, b["ids"], h["old"], h["ref"], adv,
                               comp["kept_idx"][:K], comp["kept_off"][:K + 1], eps_low=0.2, eps_high=0.28,
                               beta=w.beta, row_index=comp["src_token"],
                               dlogits_dtype=1 if w.dlogits_dtype == "bf16" else 0)
    np.testing.assert_allclose(step.seq_ratio[:K].cpu().numpy(), ref["seq_ratio"], rtol=RATIO_RTOL)
    assert np.abs(step.logp[:TK].cpu().numpy().astype(np.float64) - ref["logp"]).max() <= 2e-5
    d = host_bits(step.dlogits[:TK])
    if w.dlogits_dtype == "bf16":
        from helpers import bf16_ulp_distance
        assert int(bf16_ulp_distance(d, ref["dlogits"]).max()) <= 1
    else:
        assert np.abs(d.astype(np.float64) - ref["dlogits"].astype(np.float64)).max() <= 1e-6
    assert abs(float(step.loss.item()) - ref["loss"]) <= LOSS_RTOL * abs(ref["loss"]) + 1e-12


def test_gspo_full_size_against_oracle(oracle_mod):
    """GSPO's sequence-level loss on the full qwen step: every kept row's logp, every kept
    sequence's ratio and the total loss against the oracle run over all kept rows (without
    dlogits), and the dlogits of whole sequences (the first ones and the longest, at least 1024
    rows) against the oracle run on those sequences alone with the same sequence count."""
    import torch
    from helpers import bf16_ulp_distance
    from test_gpu_gspo import RATIO_RTOL
    w, b, step, h = build("qwen", chunk_rows=0, ratio_level="sequence", eps_low=0.2,
                          eps_high=0.28)
    step.run()
    torch.cuda.synchronize()
    assert int(step.status.item()) == 0
    adv, comp = check_selection(oracle_mod, w, b, step)
    TK, K = step.T_kept, step.K
    st, ko, kidx = comp["src_token"], comp["kept_off"][:K + 1], comp["kept_idx"][:K]
    lg = host_bits(h["logits"][torch.from_numpy(st).cuda()])  # the kept rows, in order
    kw = dict(eps_low=0.2, eps_high=0.28, beta=w.beta)
    o = oracle_mod.gspo_loss(lg, w.V, b["ids"][st], h["old"][st], h["ref"][st], adv, kidx, ko,
                             want_dlogits=False, **kw)
    logp = step.logp[:TK].cpu().numpy().astype(np.float64)
    assert np.abs(logp - o["logp"]).max() <= 2e-5
    s_gpu, s_o = step.seq_ratio[:K].cpu().numpy(), o["seq_ratio"]
    np.testing.assert_allclose(s_gpu, s_o, rtol=RATIO_RTOL)
    lo, hi = 0.8, 1.0 + np.float64(np.float32(0.28))
    near = (np.abs(s_o - lo) <= RATIO_RTOL * lo) | (np.abs(s_o - hi) <= RATIO_RTOL * hi)
    widen = float(np.sum(np.abs(adv[kidx][near].astype(np.float64)) * RATIO_RTOL * hi)) / K
    loss = float(step.loss.item())
    assert abs(loss - o["loss"]) <= LOSS_RTOL * abs(o["loss"]) + 1e-12 + widen
    # dlogits of whole sequences: the first ones up to 1024 rows, and the longest
    lens = np.diff(ko)
    pick = sorted(set(list(range(int(np.searchsorted(np.cumsum(lens), 1024)) + 1)) +
                      [int(np.argmax(lens))]) - set(np.flatnonzero(near).tolist()))
    rows = np.concatenate([np.arange(ko[k], ko[k + 1]) for k in pick])
    sub_off = np.concatenate([[0], np.cumsum(lens[pick])]).astype(np.int64)
    src = st[rows]
    od = oracle_mod.gspo_loss(host_bits(h["logits"][torch.from_numpy(src).cuda()]), w.V,
                              b["ids"][src], h["old"][src], h["ref"][src], adv, kidx[pick],
                              sub_off, n_seq=K, dlogits_dtype=1, **kw)
    d = host_bits(step.dlogits[:TK][torch.from_numpy(rows).cuda()])
    assert rows.size >= 1024
    # the bar of each row: 1 ulp, widened where g_t is ill-conditioned (loss_compare); the error
    # of log s is bounded by the largest logp error of the sequence
    e = np.abs(logp - o["logp"]) + 2.0 ** -24 * np.abs(o["logp"])
    e_seq = np.repeat([e[ko[k]:ko[k + 1]].max() for k in pick], lens[pick])
    bar = allowed_ulps(logp[rows], dict(logp=o["logp"][rows], g=od["g"]),
                       dict(ref_logp=h["ref"][src], beta=w.beta, e_ratio=e_seq))
    dist = bf16_ulp_distance(d, od["dlogits"]).max(axis=1)
    assert np.all(dist <= bar), (int(dist.max()), bar[dist > bar][:5])
    print("qwen GSPO: %d rows, %d sequences, %d at a clip boundary, loss %.12g (oracle %.12g), "
          "dlogits of %d sequences (%d rows, worst %d ulps, %d rows with an ill-conditioned g_t)"
          % (TK, K, int(near.sum()), loss, o["loss"], len(pick), rows.size, int(dist.max()),
             int((bar > 1).sum())))


@pytest.mark.parametrize("name,ratio", [("small", "token"), ("small", "sequence")])
def test_graph_replay_follows_new_inputs(name, ratio):
    """Graphs captured on one batch, replayed after new rewards are written into the same device
    buffers (rewards permuted within each prompt: other advantages, another kept set, other
    counts), give what a fresh host-synced step computes from the new rewards: no host value is
    baked into the captured graphs."""
    import torch
    w, b, step, h = build(name, chunk_rows=0, ratio_level=ratio)
    step.capture()
    rng = np.random.default_rng(5)
    r2 = b["rewards"].reshape(w.P, w.G).copy()
    for p in range(w.P):
        r2[p] = r2[p][rng.permutation(w.G)]
    r2 = torch.from_numpy(r2.reshape(-1)).cuda()
    k0 = step.run_graph()
    keep0 = step.keep.clone()
    step.rewards.copy_(r2)
    k1 = step.run_graph()
    assert not torch.equal(step.keep, keep0)  # the permutation changed the kept set
    loss, logp, dl = float(step.loss.item()), step.logp[:k1].clone(), step.dlogits[:k1].clone()
    keep = step.keep.clone()
    w2, b2, fresh, h2 = build(name, chunk_rows=0, ratio_level=ratio)
    fresh.rewards.copy_(r2)
    fresh.run()
    torch.cuda.synchronize()
    assert fresh.T_kept == k1 and torch.equal(fresh.keep, keep)
    assert float(fresh.loss.item()) == loss
    assert torch.equal(fresh.logp[:k1], logp) and torch.equal(fresh.dlogits[:k1], dl)
