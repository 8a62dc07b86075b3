"""GPU parity of grpo_gspo_loss_fwd_bwd (GSPO's sequence-level loss, FastRL's GSPO variant) with
the oracle, through the C ABI: vocabulary sizes with ragged tails, both dtypes, gathered rows,
GSPO's narrow clip range, sequences of one token, invalid tokens, empty sequences."""
import numpy as np
import pytest

from helpers import bf16_bits_to_f32, bf16_ulp_distance
from loss_compare import F32_ATOL, LOGP_ATOL, LOSS_ATOL, LOSS_RTOL

pytestmark = pytest.mark.gpu

RATIO_RTOL = 3e-5  # s_k from f32 log-probs (each within 2e-5 of the oracle's)


def bf16_bits(x):
    import torch
    return torch.from_numpy(np.ascontiguousarray(x, np.float32)).to(torch.bfloat16).view(
        torch.int16).numpy().view(np.uint16)


class SeqCase:
    def __init__(self, rng, lens, V, in_dtype="bf16", out_dtype="bf16", old_sd=0.05, beta=0.04,
                 eps=(0.2, 0.28), gather=False):
        import torch
        self.lens = np.asarray(lens, np.int64)
        self.K = len(lens)
        self.n = int(self.lens.sum())
        self.V, self.out_dtype, self.beta, self.eps = V, out_dtype, beta, eps
        n_src = self.n + (7 if gather else 0)
        z = (rng.standard_normal((n_src, V)) * 2.5).astype(np.float32)
        if in_dtype == "bf16":
            self.host = bf16_bits(z)
            zf = bf16_bits_to_f32(self.host)
            self.dev = torch.from_numpy(self.host.view(np.int16)).cuda().view(torch.bfloat16)
        else:
            self.host, zf = z, z
            self.dev = torch.from_numpy(z).cuda()
        self.y = rng.integers(0, V, size=n_src).astype(np.int32)
        zz = zf.astype(np.float64)
        m = zz.max(1, keepdims=True)
        logp = zz[np.arange(n_src), self.y] - (m[:, 0] + np.log(np.exp(zz - m).sum(1)))
        # a per-sequence drift of the old policy, so whole sequences leave the clip range
        drift = np.repeat(rng.standard_normal(self.K) * old_sd * 2, lens)
        drift = np.concatenate([drift, np.zeros(n_src - self.n)])
        self.old = (logp - drift + old_sd * rng.standard_normal(n_src)).astype(np.float32)
        self.ref = (logp + 0.1 * rng.standard_normal(n_src)).astype(np.float32)
        self.adv = rng.standard_normal(self.K + 3).astype(np.float32)
        self.seq_rollout = rng.permutation(self.K + 3)[:self.K].astype(np.int32)
        self.seq_row_off = np.concatenate([[0], np.cumsum(self.lens)]).astype(np.int64)
        self.row_index = rng.permutation(n_src)[:self.n].astype(np.int64) if gather else None

    def t(self, a):
        import torch
        return torch.from_numpy(np.ascontiguousarray(a)).cuda()

    def run_gpu(self, grpo, n_seq=None):
        import torch
        status = torch.zeros(1, dtype=torch.int32, device="cuda")
        ratio = torch.empty(max(self.K, 1), dtype=torch.float32, device="cuda")
        out = grpo.grpo_gspo_loss_fwd_bwd(
            self.dev, self.t(self.y), self.t(self.old), self.t(self.ref), self.t(self.adv),
            self.t(self.seq_rollout), self.t(self.seq_row_off), n_rows=self.n, n_seq=n_seq,
            row_index=None if self.row_index is None else self.t(self.row_index),
            eps_low=self.eps[0], eps_high=self.eps[1], beta=self.beta,
            dlogits_dtype=self.out_dtype, seq_ratio_out=ratio, status=status)
        torch.cuda.synchronize()
        d = out["dlogits"][:self.n]
        d = d.view(torch.int16).cpu().numpy().view(np.uint16) if self.out_dtype == "bf16" else d.cpu().numpy()
        return dict(loss=float(out["loss"].item()), dlogits=d, logp=out["logp"][:self.n].cpu().numpy(),
                    ratio=ratio[:self.K].cpu().numpy(), status=int(status.item()))

    def run_oracle(self, oracle_mod, n_seq=None):
        return oracle_mod.gspo_loss(self.host, self.V, self.y, self.old, self.ref, self.adv,
                                    self.seq_rollout, self.seq_row_off, n_seq=n_seq,
                                    eps_low=self.eps[0], eps_high=self.eps[1], beta=self.beta,
                                    row_index=self.row_index,
                                    dlogits_dtype=1 if self.out_dtype == "bf16" else 0)


def compare_gspo(g, r, case, n_seq=None):
    """Tolerances as the token-level loss; rows of sequences whose ratio lies within RATIO_RTOL
    of a clip boundary may take either branch and are not compared.  The loss is always compared:
    such a sequence's two branches give surrogates s*A and b*A (b the boundary), which differ by at
    most |A| * RATIO_RTOL * b, so its term widens the loss tolerance by that over n_seq."""
    valid = ~np.isnan(r["logp"])
    assert np.all(np.isnan(g["logp"][~valid]) | ~np.isfinite(g["logp"][~valid]))
    assert np.abs(g["logp"][valid].astype(np.float64) - r["logp"][valid]).max(initial=0) <= LOGP_ATOL
    s = r["seq_ratio"]
    ok = ~np.isnan(s)
    assert np.array_equal(np.isnan(g["ratio"]), ~ok)
    np.testing.assert_allclose(g["ratio"][ok], s[ok], rtol=RATIO_RTOL)
    lo, hi = 1.0 - np.float64(np.float32(case.eps[0])), 1.0 + np.float64(np.float32(case.eps[1]))
    near = ok & ((np.abs(s - lo) <= RATIO_RTOL * lo) | (np.abs(s - hi) <= RATIO_RTOL * hi))
    rows = ~np.repeat(near, case.lens)
    if case.out_dtype == "bf16":
        assert int(bf16_ulp_distance(g["dlogits"][rows], r["dlogits"][rows]).max(initial=0)) <= 1
    else:
        diff = np.abs(g["dlogits"][rows].astype(np.float64) - r["dlogits"][rows].astype(np.float64))
        assert diff.max(initial=0.0) <= F32_ATOL
    A = np.abs(case.adv[case.seq_rollout].astype(np.float64))
    widen = float(np.sum(A[near] * RATIO_RTOL * hi)) / (n_seq or case.K)
    assert abs(g["loss"] - r["loss"]) <= LOSS_RTOL * abs(r["loss"]) + LOSS_ATOL + widen, \
        "GSPO loss %r vs oracle %r (%d sequences at a clip boundary)" % (g["loss"], r["loss"],
                                                                          int(near.sum()))
    return int(near.sum())


SHAPES = [(1000, "bf16", "bf16"), (1001, "f32", "f32"), (4097, "f32", "bf16"),
          (32000, "bf16", "bf16"), (152064, "bf16", "bf16"), (152067, "bf16", "f32")]


@pytest.mark.parametrize("V,ind,outd", SHAPES)
def test_gspo_matches_oracle(grpo, oracle_mod, V, ind, outd):
    rng = np.random.default_rng(V)
    lens = list(rng.integers(4, 24 if V > 100000 else 48, size=7)) + [0, 9]
    c = SeqCase(rng, lens, V, ind, outd, old_sd=0.15)
    g, r = c.run_gpu(grpo), c.run_oracle(oracle_mod)
    assert g["status"] == 0
    compare_gspo(g, r, c)
    s = r["seq_ratio"][~np.isnan(r["seq_ratio"])]
    assert ((s > 1.28) | (s < 0.8)).any() and ((s < 1.28) & (s > 0.8)).any()


@pytest.mark.parametrize("V,ind,outd,off,pad,out_off", [
    (152064, "bf16", "bf16", 1, 0, 0), (152064, "bf16", "bf16", 0, 0, 1),
    (32000, "bf16", "f32", 0, 3, 1), (4096, "f32", "bf16", 1, 1, 3), (1000, "f32", "f32", 2, 1, 1)])
def test_gspo_unaligned_rows_give_the_aligned_bits(grpo, V, ind, outd, off, pad, out_off):
    """Logits or dlogits rows that do not start on a 16-byte boundary run the realigning
    instances (forward rows and dlogits): the same values at another alignment give the same
    loss, logp, sequence ratios and dlogits bits."""
    import torch
    rng = np.random.default_rng(V + off + 10 * pad + 100 * out_off)
    lens = list(rng.integers(4, 24, size=6)) + [0, 9]
    c = SeqCase(rng, lens, V, ind, outd, old_sd=0.15)
    odt = torch.bfloat16 if outd == "bf16" else torch.float32

    def call(logits, dlogits, S):
        ratio = torch.empty(c.K, dtype=torch.float32, device="cuda")
        logp = torch.empty(c.n, dtype=torch.float32, device="cuda")
        out = grpo.grpo_gspo_loss_fwd_bwd(
            logits, c.t(c.y), c.t(c.old), c.t(c.ref), c.t(c.adv), c.t(c.seq_rollout),
            c.t(c.seq_row_off), n_rows=c.n, V=V, row_stride=S, eps_low=c.eps[0],
            eps_high=c.eps[1], beta=c.beta, dlogits=dlogits, logp_out=logp, seq_ratio_out=ratio)
        torch.cuda.synchronize()
        bits = torch.int16 if outd == "bf16" else torch.int32
        return (out["loss"].view(torch.int64).item(), logp.view(torch.int32).cpu().numpy(),
                ratio.view(torch.int32).cpu().numpy(), dlogits.view(bits).cpu().numpy())

    ref = call(c.dev.view(-1, V)[:c.n], torch.empty(c.n, V, dtype=odt, device="cuda"), V)
    S = V + pad
    flat = torch.zeros(off + c.n * S, dtype=c.dev.dtype, device="cuda")
    rows = flat[off:].view(c.n, S)
    rows[:, :V] = c.dev.view(-1, V)[:c.n]
    out_flat = torch.empty(out_off + c.n * V, dtype=odt, device="cuda")
    got = call(rows[:, :V], out_flat[out_off:].view(c.n, V), S)
    assert got[0] == ref[0]
    for a, b in zip(got[1:], ref[1:]):
        assert np.array_equal(a, b)


def test_gspo_misaligned_element_pointer_is_rejected(grpo):
    """A dlogits pointer that is not a multiple of its element size is refused before any launch."""
    import ctypes
    import torch
    rng = np.random.default_rng(6)
    c = SeqCase(rng, [3, 5], 64)
    raw = torch.zeros(c.n * 64 * 2 + 2, dtype=torch.uint8, device="cuda")
    logp = torch.empty(c.n, dtype=torch.float32, device="cuda")
    loss = torch.empty(1, dtype=torch.float64, device="cuda")
    ws = torch.empty(1 << 16, dtype=torch.uint8, device="cuda")
    ws_bytes = ctypes.c_size_t(ws.numel())
    y, old, ref, adv, sr, so = (c.t(a) for a in (c.y, c.old, c.ref, c.adv, c.seq_rollout, c.seq_row_off))
    lib = grpo.lib()
    st = lib.grpo_gspo_loss_fwd_bwd(c.dev.data_ptr(), 1, 64, None, c.n, 64, y.data_ptr(),
                                    old.data_ptr(), ref.data_ptr(), adv.data_ptr(), sr.data_ptr(),
                                    so.data_ptr(), c.K, c.K, 0.2, 0.2, 0.0, raw.data_ptr() + 1, 1,
                                    logp.data_ptr(), None, loss.data_ptr(), None, ws.data_ptr(),
                                    ctypes.byref(ws_bytes), None)
    assert st == 1, st  # GRPO_ERR_INVALID_ARG
    assert b"element size" in lib.grpo_last_error()


def test_gspo_gathered_rows_and_global_sequence_count(grpo, oracle_mod):
    """Rows gathered through row_index from a larger buffer; n_seq larger than the local
    sequence count (data parallelism: the global count)."""
    rng = np.random.default_rng(41)
    c = SeqCase(rng, [5, 17, 1, 30, 8], 32000, gather=True)
    g, r = c.run_gpu(grpo, n_seq=13), c.run_oracle(oracle_mod, n_seq=13)
    compare_gspo(g, r, c, n_seq=13)


def test_gspo_narrow_clip_range(grpo, oracle_mod):
    """GSPO's own clip widths are far narrower than the token-level ones (3e-4 / 4e-4 here):
    most sequences are clipped and get zero gradient when beta = 0."""
    rng = np.random.default_rng(42)
    c = SeqCase(rng, list(rng.integers(8, 40, size=16)), 32000, old_sd=0.01, beta=0.0,
                eps=(3e-4, 4e-4))
    g, r = c.run_gpu(grpo), c.run_oracle(oracle_mod)
    compare_gspo(g, r, c)
    A = c.adv[c.seq_rollout].astype(np.float64)
    s = r["seq_ratio"]
    active = ((A > 0) & (s > (1 + 4e-4) * (1 + RATIO_RTOL))) | ((A < 0) & (s < (1 - 3e-4) * (1 - RATIO_RTOL)))
    assert active.sum() >= 4
    zero_rows = np.repeat(active, c.lens)
    assert np.all((g["dlogits"][zero_rows] & 0x7FFF) == 0)


def test_gspo_one_token_sequences(grpo, oracle_mod):
    """Every sequence one token long: the case where GSPO's ratio is the token ratio."""
    rng = np.random.default_rng(43)
    c = SeqCase(rng, [1] * 64, 32000, old_sd=0.2)
    compare_gspo(c.run_gpu(grpo), c.run_oracle(oracle_mod), c)


def test_gspo_invalid_token_drops_its_sequence(grpo, oracle_mod):
    rng = np.random.default_rng(44)
    c = SeqCase(rng, [6, 6, 6], 5000)
    c.y[8] = 5000  # row 8 belongs to sequence 1
    g, r = c.run_gpu(grpo), c.run_oracle(oracle_mod)
    assert g["status"] & grpo.binding.DEVFLAG_BAD_TOKEN
    assert np.isnan(g["ratio"][1]) and np.all((g["dlogits"][6:12] & 0x7FFF) == 0)
    compare_gspo(g, r, c)


def test_gspo_deterministic(grpo):
    rng = np.random.default_rng(45)
    c = SeqCase(rng, list(rng.integers(10, 200, size=12)), 152064)
    a, b = c.run_gpu(grpo), c.run_gpu(grpo)
    assert a["loss"] == b["loss"] and np.array_equal(a["dlogits"], b["dlogits"])
    assert np.array_equal(a["ratio"], b["ratio"])


def test_gspo_no_rows(grpo):
    """Two empty sequences (no rows gathered from a 7-row buffer): the loss is 0."""
    rng = np.random.default_rng(46)
    c = SeqCase(rng, [0, 0], 1000, gather=True)
    g = c.run_gpu(grpo)
    assert g["loss"] == 0.0 and g["status"] == 0 and np.all(np.isnan(g["ratio"]))


def test_gspo_device_counts_match_host_counts(grpo):
    """grpo_gspo_loss_fwd_bwd_dev over min(max_seqs, K) sequences and min(max_rows, T_kept) rows,
    with the mean over K, equals grpo_gspo_loss_fwd_bwd given the same numbers on the host, bit
    for bit; entries past the counts are not written."""
    import torch
    rng = np.random.default_rng(47)
    lens = [9, 0, 14, 5, 21, 3]
    c = SeqCase(rng, lens, 32000, old_sd=0.15)
    off = c.seq_row_off
    for K in (0, 1, 3, 6):
        TK = int(off[K])
        counts = c.t(np.array([K, TK], np.int64))
        dl_a = torch.zeros((c.n, c.V), dtype=torch.bfloat16, device="cuda")
        dl_b = torch.zeros_like(dl_a)
        lp_a = torch.zeros(c.n, dtype=torch.float32, device="cuda")
        lp_b = torch.zeros_like(lp_a)
        sr_a = torch.zeros(c.K, dtype=torch.float32, device="cuda")
        sr_b = torch.zeros_like(sr_a)
        la = torch.empty(1, dtype=torch.float64, device="cuda")
        lb = torch.empty(1, dtype=torch.float64, device="cuda")
        ws = torch.empty(1 << 20, dtype=torch.uint8, device="cuda")
        grpo.binding.grpo_gspo_loss_fwd_bwd_dev(
            c.dev, c.t(c.y), c.t(c.old), c.t(c.ref), c.t(c.adv), c.t(c.seq_rollout),
            c.t(c.seq_row_off), counts, max_rows=c.n, max_seqs=c.K, dlogits=dl_a, loss_out=la,
            ws=ws, eps_low=0.2, eps_high=0.28, beta=0.04, logp_out=lp_a, seq_ratio_out=sr_a)
        if K:
            grpo.grpo_gspo_loss_fwd_bwd(
                c.dev, c.t(c.y), c.t(c.old), c.t(c.ref), c.t(c.adv), c.t(c.seq_rollout),
                c.t(c.seq_row_off), n_rows=TK, n_seq_rows=K, n_seq=K, eps_low=0.2,
                eps_high=0.28, beta=0.04, dlogits=dl_b, logp_out=lp_b, seq_ratio_out=sr_b,
                loss_out=lb)
        else:
            lb.zero_()
        torch.cuda.synchronize()
        assert la.item() == lb.item()
        assert torch.equal(dl_a, dl_b) and torch.equal(lp_a, lp_b)  # untouched past TK in both
        assert np.array_equal(np.isnan(sr_a.cpu().numpy()), np.isnan(sr_b.cpu().numpy()))
        ok = ~np.isnan(sr_b.cpu().numpy())
        assert np.array_equal(sr_a.cpu().numpy()[ok], sr_b.cpu().numpy()[ok])
