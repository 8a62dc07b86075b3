"""GPU parity of grpo_lmhead_loss_fwd_bwd (the output layer fused with the GRPO loss, logits on
the tensor cores) with the oracle, through the C ABI.

Tolerances follow from the arithmetic (u = 2^-23: one f32 rounding of the tensor cores'
accumulation, taken at twice IEEE's unit roundoff; S[t, v] = sum_d |h[t, d]| |W[v, d]|):
  logits    |dz[t, v]| <= D * u * S[t, v]    (bf16 x bf16 products are exact in f32; D additions)
  logp      |dlogp_t| <= 2 * max_v |dz[t, v]| + 1e-5      (z_y and the log-sum-exp; f32 exp/log)
  dlogits   |dd| <= |d| * (2^-8 + 4 * max_v |dz[t, v]|) + 2^-133   (one bf16 rounding of a value
            whose softmax factor moved by at most exp(2 max |dz|))
  dhidden   |d dh[t, d]| <= (2^-8 + 4 * max|dz| + V * u) * sum_v |d[t, v]| |W[v, d]| (+ one bf16
            rounding of the output when dhidden is bf16)
  dweight   |d dW[v, d]| <= (2^-8 + 4 * max|dz| + T * u) * sum_t |d[t, v]| |h[t, d]|
  loss      |dloss| <= sum_t w_t |g_t| |dlogp_t| + 1e-6 |loss|
The oracle's dhidden_abs / dweight_abs give the sums of absolute products.  A wrong tile, k-block,
swizzle or operand moves results by the size of those sums, far outside these bounds."""
import math

import numpy as np
import pytest

pytestmark = pytest.mark.gpu

U = 2.0 ** -23


def bf16_round(x):
    import torch
    return torch.from_numpy(np.ascontiguousarray(x, np.float32)).to(torch.bfloat16).float().numpy()


class LmCase:
    def __init__(self, seed, T, V, D, n_roll=None, beta=0.04, eps=(0.2, 0.2), bad_rows=(),
                 agg_mode=0, old_sd=0.05, logit_sd=2.0):
        rng = np.random.default_rng(seed)
        self.T, self.V, self.D, self.beta, self.eps, self.agg_mode = T, V, D, beta, eps, agg_mode
        self.h = bf16_round(rng.standard_normal((T, D)))
        self.w = bf16_round(rng.standard_normal((V, D)) * (logit_sd / np.sqrt(D)))
        self.y = rng.integers(0, V, T).astype(np.int32)
        for r in bad_rows:
            self.y[r] = V + 3 if r % 2 else -1
        n_roll = n_roll or max(1, T // 37)
        self.rr = np.sort(rng.integers(0, n_roll, T)).astype(np.int32)
        self.seq_off = np.r_[0, np.cumsum(np.bincount(self.rr, minlength=n_roll))].astype(np.int64)
        self.n_seq = int((np.diff(self.seq_off) > 0).sum()) if agg_mode == 1 else 0
        self.adv = rng.standard_normal(n_roll).astype(np.float32)
        z = self.h.astype(np.float64) @ self.w.astype(np.float64).T
        m = z.max(1)
        lse = m + np.log(np.exp(z - m[:, None]).sum(1))
        yc = np.clip(self.y, 0, V - 1)
        logp = z[np.arange(T), yc] - lse
        self.old = (logp + rng.normal(0, old_sd, T)).astype(np.float32)
        self.ref = (logp + rng.normal(0, 0.1, T)).astype(np.float32)
        # Bound ingredients: S = |h| |W|^T and the logit error bound per row.
        S = np.abs(self.h).astype(np.float64) @ np.abs(self.w).astype(np.float64).T
        self.dz = D * U * S.max(1)

    def kw(self):
        kw = dict(eps_low=self.eps[0], eps_high=self.eps[1], beta=self.beta, agg_mode=self.agg_mode)
        if self.agg_mode == 1:
            kw.update(seq_off=self.seq_off, n_seq=self.n_seq)
        return kw

    def oracle(self, oracle_mod):
        return oracle_mod.lmhead_loss(self.h, self.w, self.y, self.old, self.ref, self.adv, self.rr,
                                      want_dlogits=True, want_bounds=True, **self.kw())

    def gpu(self, grpo, chunk_rows=0, dhidden_dtype="bf16", with_dlogits=True, dweight=None,
            accumulate=False):
        import torch
        dev = "cuda"
        t = lambda a, dt: torch.from_numpy(np.ascontiguousarray(a)).to(dev, dt)
        args = (t(self.h, torch.bfloat16), t(self.w, torch.bfloat16), t(self.y, torch.int32),
                t(self.old, torch.float32), t(self.ref, torch.float32), t(self.adv, torch.float32),
                t(self.rr, torch.int32))
        kw = self.kw()
        if self.agg_mode == 1:
            kw["seq_off"] = t(self.seq_off, torch.int64)
        ldd = grpo.grpo_lmhead_dlogits_stride(self.V)
        dl = torch.full((self.T, ldd), float("nan"), dtype=torch.bfloat16, device=dev) \
            if with_dlogits else None
        logp = torch.empty(self.T, dtype=torch.float32, device=dev)
        rl = torch.empty(self.T, dtype=torch.float64, device=dev)
        status = torch.zeros(1, dtype=torch.int32, device=dev)
        out = grpo.grpo_lmhead_loss_fwd_bwd(*args, dhidden_dtype=dhidden_dtype, dlogits_out=dl,
                                            logp_out=logp, row_loss_out=rl, status=status,
                                            chunk_rows=chunk_rows, dweight=dweight,
                                            accumulate_dweight=accumulate, **kw)
        torch.cuda.synchronize()
        res = dict(loss=float(out["loss"].item()), logp=logp.cpu().numpy(),
                   row_loss=rl.cpu().numpy(), dhidden=out["dhidden"].float().cpu().numpy(),
                   dweight=out["dweight"].cpu().numpy(), status=int(status.item()))
        if dl is not None:
            res["dlogits"] = dl.float().cpu().numpy()
            res["ldd"] = ldd
        return res


def check(case, g, o, dhidden_bf16=True):
    valid = (case.y >= 0) & (case.y < case.V)
    # logp
    assert np.all(np.isnan(g["logp"][~valid]))
    tol_logp = 2 * case.dz + 1e-5
    err = np.abs(g["logp"][valid] - o["logp"][valid])
    assert np.all(err <= tol_logp[valid]), "logp err %g (bound %g)" % (err.max(), tol_logp.min())
    # dlogits (when asked for): columns past V are 0
    if "dlogits" in g:
        d = g["dlogits"][:, :case.V].astype(np.float64)
        tol = np.abs(o["dlogits"]) * (2.0 ** -8 + 4 * case.dz[:, None]) + 2.0 ** -133
        bad = np.abs(d - o["dlogits"]) > tol
        assert not bad.any(), "dlogits: %d entries outside the bound, worst %g" % (
            bad.sum(), np.abs(d - o["dlogits"]).max())
        assert np.all(g["dlogits"][:, case.V:] == 0)
    # dhidden
    rel = 2.0 ** -8 + 4 * case.dz.max() + case.V * U
    tol = rel * o["dhidden_abs"] + (2.0 ** -8 * np.abs(o["dhidden"]) if dhidden_bf16 else 0) + 1e-30
    e = np.abs(g["dhidden"] - o["dhidden"])
    assert np.all(e <= tol), "dhidden: worst err %g at bound %g" % (e.max(), tol.flat[e.argmax()])
    # dweight
    rel = 2.0 ** -8 + 4 * case.dz.max() + case.T * U
    tol = rel * o["dweight_abs"] + 1e-30
    e = np.abs(g["dweight"] - o["dweight"])
    assert np.all(e <= tol), "dweight: worst err %g at bound %g" % (e.max(), tol.flat[e.argmax()])
    # loss and row terms
    rho = np.exp(np.where(valid, o["logp"], 0) - case.old)
    A = case.adv[case.rr]
    gbound = rho * np.abs(A) + case.beta * np.abs(np.exp(case.ref - np.where(valid, o["logp"], 0)) - 1)
    w = np.abs(o["row_loss"]) + 0  # sign-free size of each term, for scale only
    wt = (1.0 / case.T) if case.agg_mode == 0 else (
        1.0 / (case.n_seq * np.diff(case.seq_off)[case.rr]))
    row_tol = wt * gbound * tol_logp + 1e-6 * w + 1e-12
    assert np.all(np.abs(g["row_loss"] - o["row_loss"]) <= np.where(valid, row_tol, 0))
    assert abs(g["loss"] - o["loss"]) <= np.sum(np.where(valid, row_tol, 0)) + 1e-6 * abs(o["loss"])


@pytest.mark.parametrize("T,V,D", [(300, 1000, 256), (129, 257, 64), (64, 1, 8), (1, 300, 200)])
def test_parity_ragged_shapes(grpo, oracle_mod, T, V, D):
    # ragged row blocks (300 = 2*128 + 44), vocabulary tiles (1000 = 3*256 + 232), a vocabulary of
    # one word, a single row, and D not a multiple of 64 (zero-filled k tail)
    case = LmCase(11 + T, T, V, D)
    check(case, case.gpu(grpo), case.oracle(oracle_mod))


def test_parity_many_tiles_and_chunks(grpo, oracle_mod):
    case = LmCase(21, 600, 8192, 512, beta=0.0, eps=(0.2, 0.28))
    o = case.oracle(oracle_mod)
    one = case.gpu(grpo)
    check(case, one, o)
    chunked = case.gpu(grpo, chunk_rows=128, with_dlogits=False, dhidden_dtype="f32")
    check(case, chunked, o, dhidden_bf16=False)
    # The chunking changes only how dW is summed: the forward quantities are identical.
    np.testing.assert_array_equal(chunked["logp"], one["logp"])
    assert chunked["loss"] == one["loss"]


def test_seq_mean_aggregation_and_invalid_tokens(grpo, oracle_mod):
    case = LmCase(31, 200, 700, 128, agg_mode=1, bad_rows=(3, 150))
    g = case.gpu(grpo)
    assert g["status"] & 1  # GRPO_DEVFLAG_BAD_TOKEN
    check(case, g, case.oracle(oracle_mod))
    np.testing.assert_array_equal(g["dhidden"][[3, 150]], 0.0)


def test_accumulate_dweight_adds_to_the_buffer(grpo, oracle_mod):
    import torch
    case = LmCase(41, 150, 600, 64)
    o = case.oracle(oracle_mod)
    base = np.random.default_rng(5).standard_normal((case.V, case.D)).astype(np.float32)
    g = case.gpu(grpo, dweight=torch.from_numpy(base.copy()).cuda(), accumulate=True)
    rel = 2.0 ** -8 + 4 * case.dz.max() + case.T * U
    e = np.abs(g["dweight"] - (base + o["dweight"]))
    assert np.all(e <= rel * o["dweight_abs"] + 1e-6 * np.abs(base) + 1e-30)


def test_zero_rows(grpo):
    import torch
    h = torch.zeros((0, 64), dtype=torch.bfloat16, device="cuda")
    w = torch.ones((100, 64), dtype=torch.bfloat16, device="cuda")
    e32 = lambda dt: torch.zeros(0, dtype=dt, device="cuda")
    dw = torch.full((100, 64), 7.0, device="cuda")
    out = grpo.grpo_lmhead_loss_fwd_bwd(h, w, e32(torch.int32), e32(torch.float32),
                                        e32(torch.float32), torch.zeros(1, device="cuda"),
                                        e32(torch.int32), dweight=dw)
    torch.cuda.synchronize()
    assert float(out["loss"].item()) == 0.0
    assert float(dw.abs().max().item()) == 0.0


def test_parity_rows_gathered_through_row_index(grpo, oracle_mod):
    import torch
    case = LmCase(51, 260, 900, 192)
    o = case.oracle(oracle_mod)
    # the case's rows scattered into a larger buffer; y/old/ref at the same source rows
    rng = np.random.default_rng(52)
    n_src = case.T + 57
    src = rng.permutation(n_src)[:case.T].astype(np.int64)
    big_h = np.zeros((n_src, case.D), np.float32)
    big_h[src] = case.h
    big = {k: np.zeros(n_src, dt) for k, dt in (("y", np.int32), ("old", np.float32),
                                                 ("ref", np.float32))}
    big["y"][src], big["old"][src], big["ref"][src] = case.y, case.old, case.ref
    t = lambda a, dt: torch.from_numpy(np.ascontiguousarray(a)).cuda().to(dt)
    logp = torch.empty(case.T, dtype=torch.float32, device="cuda")
    rl = torch.empty(case.T, dtype=torch.float64, device="cuda")
    out = grpo.grpo_lmhead_loss_fwd_bwd(
        t(big_h, torch.bfloat16), t(case.w, torch.bfloat16), t(big["y"], torch.int32),
        t(big["old"], torch.float32), t(big["ref"], torch.float32), t(case.adv, torch.float32),
        t(case.rr, torch.int32), row_index=t(src, torch.int64), logp_out=logp, row_loss_out=rl,
        **case.kw())
    torch.cuda.synchronize()
    g = dict(loss=float(out["loss"].item()), logp=logp.cpu().numpy(), row_loss=rl.cpu().numpy(),
             dhidden=out["dhidden"].float().cpu().numpy(), dweight=out["dweight"].cpu().numpy())
    check(case, g, o)
    # the gathered call equals the dense one bit for bit
    dense = case.gpu(grpo, with_dlogits=False)
    np.testing.assert_array_equal(g["logp"], dense["logp"])
    np.testing.assert_array_equal(g["dhidden"], dense["dhidden"])


def test_logp_forward_entry_equals_the_loss_entrys_logp(grpo, oracle_mod):
    import torch
    case = LmCase(61, 333, 1500, 128, bad_rows=(7,))
    full = case.gpu(grpo, with_dlogits=False)
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    t = lambda a, dt: torch.from_numpy(np.ascontiguousarray(a)).cuda().to(dt)
    lp = grpo.grpo_lmhead_logp_fwd(t(case.h, torch.bfloat16), t(case.w, torch.bfloat16),
                                   t(case.y, torch.int32), status=status)["logp"]
    torch.cuda.synchronize()
    np.testing.assert_array_equal(lp.cpu().numpy(), full["logp"])
    assert status.item() & 1
    o = case.oracle(oracle_mod)
    ok = ~np.isnan(o["logp"])
    assert np.all(np.abs(lp.cpu().numpy()[ok] - o["logp"][ok]) <= 2 * case.dz[ok] + 1e-5)


def test_full_size_step_sampled_rows(grpo, oracle_mod):
    """The benchmark's output-layer configuration: the qwen batch (16 prompts x 8 rollouts,
    V = 152064) with hidden states of width 3584, through GrpoStep (selection, then the fused
    output layer and loss over the kept rows, gathered by row index).  Sampled kept rows are
    checked against the oracle one by one; dweight by the zero sum of its rows over v."""
    import torch
    from paper_2609_36932_gb300 import workloads
    from paper_2609_36932_gb300.pipeline import GrpoStep, StepParams
    w = workloads.get("qwen")
    D = workloads.LMHEAD_D
    b = workloads.make_batch(w, 0)
    dev = torch.device("cuda")
    hid = workloads.lmhead_hidden(b["T"], D, 0, dev)
    wt = workloads.lmhead_weight(w.V, D, 0, dev)
    old, ref = workloads.lmhead_old_ref(hid, wt, b["ids"], b["noise_old"], b["noise_ref"])
    p = StepParams(G=w.G, V=w.V, ngram_n=w.ngram_n, tau=w.tau, keep_cap=w.keep_cap,
                   eps_low=w.eps, eps_high=w.eps, beta=w.beta)
    step = GrpoStep(p, torch.from_numpy(b["rewards"]).to(dev), torch.from_numpy(b["ids"]).to(dev),
                    torch.from_numpy(b["off"]).to(dev), None, old, ref, hidden=hid, weight=wt)
    step.run()
    torch.cuda.synchronize()
    assert step.status.item() == 0
    T_kept = step.T_kept
    assert T_kept > 20000
    src, rr = step.kept_rows()
    sample = np.array([0, 1, T_kept // 2, T_kept - 129, T_kept - 1])
    adv, _ = oracle_mod.advantage(b["rewards"], w.G)
    o = oracle_mod.lmhead_loss(hid[torch.from_numpy(src[sample]).to(dev)].float().cpu().numpy(),
                               wt.float().cpu().numpy(), b["ids"][src[sample]],
                               old.cpu().numpy()[src[sample]], ref.cpu().numpy()[src[sample]],
                               adv, rr[sample], eps_low=w.eps, eps_high=w.eps, beta=w.beta,
                               denom_tokens=T_kept, want_dweight=False, want_bounds=True)
    S = (hid[torch.from_numpy(src[sample]).to(dev)].float().abs() @ wt.float().abs().t()).max(1)[0]
    dz = (D * U * S).cpu().numpy().astype(np.float64)
    g_logp = step.logp[:T_kept].cpu().numpy()[sample]
    assert np.all(np.abs(g_logp - o["logp"]) <= 2 * dz + 1e-5)
    dh = step.dhidden[:T_kept].float().cpu().numpy()[sample]
    rel = 2.0 ** -8 + 4 * dz.max() + w.V * U
    tol = rel * o["dhidden_abs"] + 2.0 ** -8 * np.abs(o["dhidden"])
    assert np.all(np.abs(dh - o["dhidden"]) <= tol)
    # dW: each dlogits row sums to zero, so the rows of dW sum to zero over v, up to the bf16
    # rounding of dlogits and the f32 sums
    dW = step.dweight
    col = dW.sum(0).abs().double()
    scale = dW.abs().sum(0).double()
    assert bool((col <= 2.0 ** -6 * scale).all())
    assert math.isfinite(float(step.loss.item()))


class GspoCase(LmCase):
    """LmCase rows grouped into sequences (lengths `lens`; rows after the last sequence belong to
    none), GSPO's clip widths."""

    def __init__(self, seed, lens, V, D, extra_rows=0, bad_rows=(), beta=0.02, old_sd=0.05):
        T = int(sum(lens)) + extra_rows
        super().__init__(seed, T, V, D, n_roll=len(lens), beta=beta, eps=(0.2, 0.28),
                         bad_rows=bad_rows, old_sd=old_sd)
        self.lens = np.asarray(lens, np.int64)
        self.so = np.r_[0, np.cumsum(self.lens)].astype(np.int64)
        # sequence log-ratios near 0, +0.35 or -0.35 in turn: inside the clip range, or clipped
        # on either side, and far from its edges
        for k in range(len(lens)):
            self.old[self.so[k]:self.so[k + 1]] -= (0.0, 0.35, -0.35)[k % 3]
        self.seq_rollout = np.random.default_rng(seed + 1).permutation(len(lens)).astype(np.int32)

    def oracle(self, oracle_mod):
        return oracle_mod.lmhead_gspo_loss(self.h, self.w, self.y, self.old, self.ref, self.adv,
                                           self.seq_rollout, self.so, eps_low=self.eps[0],
                                           eps_high=self.eps[1], beta=self.beta,
                                           want_dlogits=True, want_bounds=True)

    def gpu(self, grpo, chunk_rows=0):
        import torch
        t = lambda a, dt: torch.from_numpy(np.ascontiguousarray(a)).cuda().to(dt)
        K = len(self.lens)
        ldd = grpo.grpo_lmhead_dlogits_stride(self.V)
        dl = torch.full((self.T, ldd), float("nan"), dtype=torch.bfloat16, device="cuda")
        ratio = torch.empty(K, dtype=torch.float32, device="cuda")
        status = torch.zeros(1, dtype=torch.int32, device="cuda")
        out = grpo.grpo_lmhead_gspo_loss_fwd_bwd(
            t(self.h, torch.bfloat16), t(self.w, torch.bfloat16), t(self.y, torch.int32),
            t(self.old, torch.float32), t(self.ref, torch.float32), t(self.adv, torch.float32),
            t(self.seq_rollout, torch.int32), t(self.so, torch.int64), eps_low=self.eps[0],
            eps_high=self.eps[1], beta=self.beta, dlogits_out=dl, seq_ratio_out=ratio,
            status=status, chunk_rows=chunk_rows)
        torch.cuda.synchronize()
        return dict(loss=float(out["loss"].item()), logp=out["logp"][:self.T].cpu().numpy(),
                    dhidden=out["dhidden"].float().cpu().numpy(),
                    dweight=out["dweight"].cpu().numpy(), dlogits=dl.float().cpu().numpy(),
                    seq_ratio=ratio.cpu().numpy(), status=int(status.item()))


def check_gspo(case, g, o):
    # logp is compared on the rows of sequences (the oracle leaves rows in no sequence at 0)
    valid = (case.y >= 0) & (case.y < case.V) & (np.arange(case.T) < case.so[-1])
    tol_logp = 2 * case.dz + 1e-5
    assert np.all(np.abs(g["logp"][valid] - o["logp"][valid]) <= tol_logp[valid])
    # the ratio of a sequence moves with the mean of its rows' logp errors
    good = ~np.isnan(o["seq_ratio"])
    np.testing.assert_array_equal(np.isnan(g["seq_ratio"]), ~good)
    sr = o["seq_ratio"][good]
    assert np.min(np.abs(sr - 0.8), initial=1) > 1e-3 and np.min(np.abs(sr - 1.28), initial=1) > 1e-3
    r_tol = o["seq_ratio"][good] * (tol_logp.max() + 1e-6)
    assert np.all(np.abs(g["seq_ratio"][good] - o["seq_ratio"][good]) <= r_tol)
    d = g["dlogits"][:, :case.V].astype(np.float64)
    tol = np.abs(o["dlogits"]) * (2.0 ** -8 + 4 * case.dz[:, None] + 1e-5) + 2.0 ** -133
    assert not (np.abs(d - o["dlogits"]) > tol).any()
    rel = 2.0 ** -8 + 4 * case.dz.max() + 1e-5 + case.V * U
    assert np.all(np.abs(g["dhidden"] - o["dhidden"]) <=
                  rel * o["dhidden_abs"] + 2.0 ** -8 * np.abs(o["dhidden"]) + 1e-30)
    rel = 2.0 ** -8 + 4 * case.dz.max() + 1e-5 + case.T * U
    assert np.all(np.abs(g["dweight"] - o["dweight"]) <= rel * o["dweight_abs"] + 1e-30)
    K = len(case.lens)
    A = np.abs(case.adv[case.seq_rollout])
    s = np.where(good, o["seq_ratio"], 0)
    loss_tol = np.sum((s * A * 1.01 + 2 * case.beta) * tol_logp.max()) / K
    assert abs(g["loss"] - o["loss"]) <= loss_tol + 1e-6 * abs(o["loss"]) + 1e-12


@pytest.mark.parametrize("lens,V,D,extra", [((40, 1, 97, 0, 130), 1000, 128, 0),
                                            ((300, 260), 2000, 256, 37)])
def test_gspo_parity(grpo, oracle_mod, lens, V, D, extra):
    # sequences of one row, an empty sequence, a sequence across row blocks, rows in no sequence
    case = GspoCase(71 + V, lens, V, D, extra_rows=extra)
    g = case.gpu(grpo)
    check_gspo(case, g, case.oracle(oracle_mod))
    if extra:
        np.testing.assert_array_equal(g["dhidden"][-extra:], 0.0)


def test_gspo_invalid_token_sequence_and_chunks(grpo, oracle_mod):
    case = GspoCase(81, (50, 70, 90), 700, 64, bad_rows=(60,))
    g = case.gpu(grpo, chunk_rows=128)
    assert g["status"] & 1
    o = case.oracle(oracle_mod)
    assert np.isnan(o["seq_ratio"][1]) and np.isnan(g["seq_ratio"][1])
    check_gspo(case, g, o)
    np.testing.assert_array_equal(g["dhidden"][50:120], 0.0)


@pytest.mark.parametrize("chunk", [128, 0])
def test_gspo_kept_first_chunk_and_recomputed_logits_give_the_same_bits(grpo, oracle_mod, chunk):
    """GSPO's entry keeps the first chunk's f32 logits from pass 1 and recomputes the later
    chunks' in pass 2; with recompute_logits set every chunk is recomputed.  Sequences cross the
    128-row chunk boundaries (and with the default chunk all rows are one chunk): every output is
    bit-identical, and matches the oracle."""
    case = GspoCase(91, (50, 70, 90, 35), 700, 64, bad_rows=(60,))
    kept = case.gpu(grpo, chunk_rows=chunk)
    try:
        grpo.grpo_lmhead_tune(0, 0, 1)
        rec = case.gpu(grpo, chunk_rows=chunk)
    finally:
        grpo.grpo_lmhead_tune(0, 0, 0)
    for k in ("logp", "dhidden", "dweight", "dlogits", "seq_ratio"):
        np.testing.assert_array_equal(kept[k], rec[k], err_msg=k)
    assert kept["loss"] == rec["loss"] and kept["status"] == rec["status"]
    check_gspo(case, kept, case.oracle(oracle_mod))


def test_step_with_the_output_layer_and_gspo(grpo, oracle_mod):
    """GrpoStep in output-layer mode with GSPO's ratio on the small workload's batch: selection,
    then grpo_lmhead_gspo_loss_fwd_bwd over the kept rollouts as sequences, against the oracle."""
    import torch
    from paper_2609_36932_gb300 import workloads
    from paper_2609_36932_gb300.pipeline import GrpoStep, StepParams
    w = workloads.get("small")
    D = 128
    b = workloads.make_batch(w, 3)
    dev = torch.device("cuda")
    hid = workloads.lmhead_hidden(b["T"], D, 3, dev)
    wt = workloads.lmhead_weight(w.V, D, 3, dev)
    old, ref = workloads.lmhead_old_ref(hid, wt, b["ids"], b["noise_old"], b["noise_ref"])
    p = StepParams(G=w.G, V=w.V, keep_cap=w.keep_cap, eps_low=3e-4, eps_high=4e-4, beta=0.0,
                   ratio_level="sequence")
    step = GrpoStep(p, torch.from_numpy(b["rewards"]).to(dev), torch.from_numpy(b["ids"]).to(dev),
                    torch.from_numpy(b["off"]).to(dev), None, old, ref, hidden=hid, weight=wt)
    step.run()
    torch.cuda.synchronize()
    adv, _ = oracle_mod.advantage(b["rewards"], w.G)
    keep, _ = oracle_mod.prune(b["rewards"], b["ids"], b["off"], w.G, w.ngram_n, w.tau,
                               w.keep_cap, 1)
    comp = oracle_mod.compact(keep, b["off"])
    K, TK = comp["K"], comp["T_kept"]
    assert (step.K, step.T_kept) == (K, TK)
    src = comp["src_token"][:TK]
    o = oracle_mod.lmhead_gspo_loss(hid.float().cpu().numpy()[src], wt.float().cpu().numpy(),
                                    b["ids"][src], old.cpu().numpy()[src], ref.cpu().numpy()[src],
                                    adv, comp["kept_idx"][:K], comp["kept_off"][:K + 1],
                                    eps_low=3e-4, eps_high=4e-4, beta=0.0, want_bounds=True)
    S = (hid[torch.from_numpy(src).to(dev)].float().abs() @ wt.float().abs().t()).max(1)[0]
    dz = (D * U * S).cpu().numpy().astype(np.float64)
    lp = step.logp[:TK].cpu().numpy()
    assert np.all(np.abs(lp - o["logp"]) <= 2 * dz + 1e-5)
    # sequences whose ratio sits within the logp error of a clip edge may take either branch
    s_o = o["seq_ratio"]
    edge = (np.abs(s_o - (1 - 3e-4)) < 1e-4) | (np.abs(s_o - (1 + 4e-4)) < 1e-4)
    rows_ok = np.ones(TK, bool)
    for k in np.flatnonzero(edge):
        rows_ok[comp["kept_off"][k]:comp["kept_off"][k + 1]] = False
    dh = step.dhidden[:TK].float().cpu().numpy()
    rel = 2.0 ** -8 + 4 * dz.max() + 1e-5 + w.V * U
    tol = rel * o["dhidden_abs"] + 2.0 ** -8 * np.abs(o["dhidden"]) + 1e-30
    assert np.all((np.abs(dh - o["dhidden"]) <= tol)[rows_ok])
    if not edge.any():
        assert abs(float(step.loss.item()) - o["loss"]) <= 1e-4 * abs(o["loss"]) + 1e-9


def test_non_finite_hidden_row_is_flagged(grpo):
    """A NaN in one row's hidden state makes that row's logits NaN: its logp is NaN and the status
    word carries GRPO_DEVFLAG_NONFINITE; the other rows' logp are unaffected."""
    import torch
    case = LmCase(91, 200, 600, 64)
    clean = case.gpu(grpo, with_dlogits=False)
    case.h = case.h.copy()
    case.h[17, 5] = np.nan
    g = case.gpu(grpo, with_dlogits=False)
    assert g["status"] & 2  # GRPO_DEVFLAG_NONFINITE
    assert np.isnan(g["logp"][17])
    others = np.arange(case.T) != 17
    np.testing.assert_array_equal(g["logp"][others], clean["logp"][others])


@pytest.mark.parametrize("T,V,D", [(400, 32000, 4096), (300, 8192, 8192)])
def test_large_hidden_sizes_sampled_rows(grpo, oracle_mod, T, V, D):
    """Long reductions (64 and 128 k-blocks of 64 per tile): the GPU runs every row; the oracle
    checks sampled rows one by one (logp and dhidden, token-mean weights over all T rows)."""
    import torch
    rng = np.random.default_rng(D)
    h = bf16_round(rng.standard_normal((T, D)))
    w = bf16_round(rng.standard_normal((V, D)) * (2.0 / np.sqrt(D)))
    y = rng.integers(0, V, T).astype(np.int32)
    rr = np.sort(rng.integers(0, 8, T)).astype(np.int32)
    adv = rng.standard_normal(8).astype(np.float32)
    ht = torch.from_numpy(h).cuda().to(torch.bfloat16)
    wt = torch.from_numpy(w).cuda().to(torch.bfloat16)
    z = (ht.float() @ wt.float().t()).double()
    logp_c = (z.gather(1, torch.from_numpy(y.astype(np.int64)).cuda()[:, None])[:, 0]
              - torch.logsumexp(z, 1)).cpu().numpy()
    old = (logp_c + rng.normal(0, 0.05, T)).astype(np.float32)
    ref = (logp_c + rng.normal(0, 0.1, T)).astype(np.float32)
    t = lambda a, dt: torch.from_numpy(np.ascontiguousarray(a)).cuda().to(dt)
    lp = torch.empty(T, dtype=torch.float32, device="cuda")
    out = grpo.grpo_lmhead_loss_fwd_bwd(ht, wt, t(y, torch.int32), t(old, torch.float32),
                                        t(ref, torch.float32), t(adv, torch.float32),
                                        t(rr, torch.int32), logp_out=lp, dhidden_dtype="f32")
    torch.cuda.synchronize()
    rows = np.array([0, 1, T // 2, T - 1])
    o = oracle_mod.lmhead_loss(h[rows], w, y[rows], old[rows], ref[rows], adv, rr[rows],
                               denom_tokens=T, want_dweight=False, want_bounds=True)
    S = np.abs(h[rows]).astype(np.float64) @ np.abs(w).astype(np.float64).T
    dz = D * U * S.max(1)
    assert np.all(np.abs(lp.cpu().numpy()[rows] - o["logp"]) <= 2 * dz + 1e-5)
    rel = 2.0 ** -8 + 4 * dz.max() + V * U
    dh = out["dhidden"].cpu().numpy()[rows]
    assert np.all(np.abs(dh - o["dhidden"]) <= rel * o["dhidden_abs"] + 1e-30)


def assert_same_bits(a, b):
    for k in ("logp", "row_loss", "dhidden", "dweight", "dlogits"):
        if k in a or k in b:
            np.testing.assert_array_equal(a[k], b[k], err_msg=k)
    assert a["loss"] == b["loss"]


@pytest.mark.parametrize("prefetch,lanes", [(0, 1), (0, 8), (4, 3)])
def test_parity_under_other_schedules(grpo, oracle_mod, prefetch, lanes):
    """grpo_lmhead_tune changes the grid (pair lanes x vocabulary lanes) and adds L2 prefetches;
    every setting computes the same function, to the bit: each row's softmax sums are combined per
    vocabulary tile in a fixed order, whichever CTA visited the tile."""
    case = LmCase(101 + lanes, 900, 3000, 192)
    o = case.oracle(oracle_mod)
    ref = case.gpu(grpo)
    try:
        grpo.grpo_lmhead_tune(prefetch, lanes)
        g = case.gpu(grpo)
    finally:
        grpo.grpo_lmhead_tune(0, 0)
    check(case, g, o)
    assert_same_bits(g, ref)


@pytest.mark.parametrize("T,V,D,chunk", [(700, 5000, 192, 256), (333, 257, 64, 0),
                                         (600, 152064, 64, 256)])
def test_stored_and_recomputed_logits_give_the_same_bits(grpo, oracle_mod, T, V, D, chunk):
    """The token loss keeps each chunk's f32 logits from pass 1 and forms dlogits from them; with
    recompute_logits set it recomputes the tiles in a second tensor-core pass instead.  Both apply
    the same arithmetic to the same f32 logits: every output is bit-identical, and matches the
    oracle (ragged chunks, a ragged vocabulary tile, invalid tokens)."""
    case = LmCase(71 + T, T, V, D, bad_rows=(5, T - 1))
    stored = case.gpu(grpo, chunk_rows=chunk)
    # without dlogits_out the library's own chunk buffer holds each chunk's dlogits in turn
    own = case.gpu(grpo, chunk_rows=chunk, with_dlogits=False)
    try:
        grpo.grpo_lmhead_tune(0, 0, 1)
        rec = case.gpu(grpo, chunk_rows=chunk)
    finally:
        grpo.grpo_lmhead_tune(0, 0, 0)
    assert_same_bits(stored, rec)
    assert_same_bits(own, {k: v for k, v in rec.items() if k != "dlogits"})
    assert stored["status"] == rec["status"] == own["status"] == 1  # GRPO_DEVFLAG_BAD_TOKEN
    if V * T <= 5000 * 700:
        check(case, stored, case.oracle(oracle_mod))
