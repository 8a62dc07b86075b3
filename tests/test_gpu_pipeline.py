"""Whole-step parity on the five workloads, in the launch configuration bench.py times:
advantage -> prune -> compact -> loss over the kept rows.  'tiny' and 'small' are compared
with the oracle row by row in full; the three Qwen-vocabulary workloads at full size are
compared on sampled rows, and their total loss through a property that holds at any size
(the loss is the weighted sum of Eq. 1's per-token terms evaluated at the kernel's logp)."""
import numpy as np
import pytest

from loss_compare import LOSS_RTOL, compare
from paper_2609_36932_gb300 import workloads
from paper_2609_36932_gb300.pipeline import GrpoStep, StepParams

pytestmark = pytest.mark.gpu


def build(name, seed=0, chunk_rows=None):
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


def eq1_terms(logp, old, ref, A, eps, beta, w):
    """Eq. 1's per-token loss terms at the given log-probs (fp64)."""
    logp = logp.astype(np.float64)
    rho = np.exp(logp - old)
    lo, hi = 1.0 - np.float64(np.float32(eps)), 1.0 + np.float64(np.float32(eps))
    surr = np.minimum(rho * A, np.clip(rho, lo, hi) * A)
    x = ref - logp
    kl = np.expm1(x) - x
    return -w * (surr - np.float64(np.float32(beta)) * kl)


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
            ref, w.dlogits_dtype)


@pytest.mark.parametrize("name", ["qwen", "large", "long"])
def test_full_size_sampled(oracle_mod, name):
    import torch
    w, b, step, h = build(name, chunk_rows=0)
    step.run()
    torch.cuda.synchronize()
    assert int(step.status.item()) == 0
    adv, comp = check_selection(oracle_mod, w, b, step)
    TK = step.T_kept
    rng = np.random.default_rng(7)
    rows = np.unique(np.concatenate([np.arange(8), np.arange(TK - 8, TK),
                                     rng.choice(TK, 32, replace=False)]))
    src = comp["src_token"][rows]
    lg = host_bits(h["logits"][torch.from_numpy(src).cuda()])
    o = oracle_mod.loss(lg, w.V, b["ids"][src], h["old"][src], h["ref"][src], adv,
                        comp["token_rollout"][rows], eps_low=w.eps, eps_high=w.eps, beta=w.beta,
                        denom_tokens=TK, dlogits_dtype=1 if w.dlogits_dtype == "bf16" else 0)
    idx = torch.from_numpy(rows).cuda()
    logp = step.logp[:TK].cpu().numpy()
    compare(logp[rows], host_bits(step.dlogits[:TK][idx]), None, o, w.dlogits_dtype)
    # the total: Eq. 1's terms at the kernel's logp, summed in fp64
    st = comp["src_token"]
    terms = eq1_terms(logp, h["old"][st].astype(np.float64), h["ref"][st].astype(np.float64),
                      adv[comp["token_rollout"]].astype(np.float64), w.eps, w.beta, 1.0 / TK)
    total = float(step.loss.item())
    assert abs(total - terms.sum()) <= LOSS_RTOL * abs(terms.sum()) + 1e-12
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
        n_last = TK - (TK - 1) // w.chunk_rows * w.chunk_rows
        assert torch.equal(step.dlogits[:n_last][-100:], d_last)


@pytest.mark.parametrize("name", ["tiny", "qwen"])
def test_graph_mode_equals_host_synced_step(name):
    """The step captured as two CUDA graphs (the loss reads the kept count on the device) gives
    the same selection, loss, logp and dlogits as the host-synced step, on two replays."""
    import torch
    w, b, step, h = build(name, chunk_rows=0)
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
