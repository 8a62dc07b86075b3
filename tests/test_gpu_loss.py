"""GPU parity of grpo_loss_fwd_bwd (Eqs. 1-3) with the oracle, through the C ABI: vocabulary
sizes with ragged tails, both input and output dtypes, launch shapes, gathered and strided
rows, Eq. 1's sequence mean, and the documented edge cases."""
import numpy as np
import pytest

from helpers import bf16_bits_to_f32
from loss_compare import compare

pytestmark = pytest.mark.gpu


def bf16_bits(x):
    import torch
    return torch.from_numpy(np.ascontiguousarray(x, np.float32)).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)


class Case:
    def __init__(self, rng, n, V, in_dtype="bf16", out_dtype="bf16", scale=2.0, n_roll=4,
                 stride=None, beta=0.04, A=None, old_noise=0.05):
        import torch
        self.n, self.V, self.in_dtype, self.out_dtype = n, V, in_dtype, out_dtype
        self.stride = V if stride is None else stride
        z = (rng.standard_normal((n, self.stride)) * scale).astype(np.float32)
        if in_dtype == "bf16":
            self.host = bf16_bits(z)
            zf = bf16_bits_to_f32(self.host)
            self.dev = torch.from_numpy(self.host.view(np.int16)).cuda().view(torch.bfloat16)
        else:
            self.host = z
            zf = z
            self.dev = torch.from_numpy(z).cuda()
        self.y = rng.integers(0, V, size=n).astype(np.int32)
        zz = zf[:, :V].astype(np.float64)
        m = zz.max(1, keepdims=True)
        logp = zz[np.arange(n), self.y] - (m[:, 0] + np.log(np.exp(zz - m).sum(1)))
        self.old = (logp + old_noise * rng.standard_normal(n)).astype(np.float32)
        self.ref = (logp + 0.1 * rng.standard_normal(n)).astype(np.float32)
        self.adv = (rng.standard_normal(n_roll) if A is None else np.asarray(A)).astype(np.float32)
        self.rr = rng.integers(0, self.adv.size, size=n).astype(np.int32)
        self.beta = beta

    def t(self, a):
        import torch
        return torch.from_numpy(np.ascontiguousarray(a)).cuda()

    def cond(self, idx=None):
        """The rows' ref_logp inputs and beta, for compare()'s conditioning of g_t."""
        return dict(ref_logp=self.ref[:self.n] if idx is None else self.ref[idx], beta=self.beta)

    def run_gpu(self, grpo, **kw):
        import torch
        n = kw.pop("n_rows", self.n)
        rr = kw.pop("rr", self.rr)
        logp = torch.empty(max(n, 1), dtype=torch.float32, device="cuda")
        rl = torch.empty(max(n, 1), dtype=torch.float64, device="cuda")
        status = torch.zeros(1, dtype=torch.int32, device="cuda")
        logits = self.dev.view(self.n, self.stride)[:, :self.V] if self.stride != self.V else self.dev
        args = dict(V=self.V, row_stride=self.stride, beta=self.beta,
                    dlogits_dtype=self.out_dtype, logp_out=logp, row_loss_out=rl, status=status)
        args.update(kw)
        out = grpo.grpo_loss_fwd_bwd(logits, self.t(self.y), self.t(self.old), self.t(self.ref),
                                     self.t(self.adv), self.t(rr), n_rows=n, **args)
        torch.cuda.synchronize()
        d = out["dlogits"]
        if self.out_dtype == "bf16":
            d = d.view(torch.int16).cpu().numpy().view(np.uint16)
        else:
            d = d.cpu().numpy()
        return dict(loss=float(out["loss"].item()), dlogits=d.reshape(n, self.V) if n else d,
                    logp=logp[:n].cpu().numpy(), row_loss=rl[:n].cpu().numpy(),
                    status=int(status.item()))

    def run_oracle(self, oracle_mod, **kw):
        kw.setdefault("beta", self.beta)
        return oracle_mod.loss(self.host, self.V, self.y, self.old, self.ref, self.adv, self.rr,
                               row_stride=self.stride, n_rows=kw.pop("n_rows", self.n),
                               dlogits_dtype=1 if self.out_dtype == "bf16" else 0, **kw)


SHAPES = [(1, "f32", "f32"), (7, "bf16", "bf16"), (8, "bf16", "bf16"), (9, "f32", "bf16"),
          (1000, "bf16", "f32"), (1001, "bf16", "bf16"), (1024, "f32", "f32"),
          (4097, "bf16", "bf16"), (32000, "bf16", "bf16"), (32001, "f32", "f32"),
          (152064, "bf16", "bf16"), (152067, "bf16", "f32")]


@pytest.mark.parametrize("V,ind,outd", SHAPES)
def test_vocab_sizes_and_dtypes(grpo, oracle_mod, V, ind, outd):
    rng = np.random.default_rng(V)
    n = 37 if V < 100000 else 19
    c = Case(rng, n, V, ind, outd)
    g = c.run_gpu(grpo)
    r = c.run_oracle(oracle_mod)
    assert g["status"] == 0
    compare(g["logp"], g["dlogits"], g["loss"], r, outd, gpu_row_loss=g["row_loss"],
            cond=c.cond())


@pytest.mark.parametrize("cluster,threads,chunks", [(2, 256, 0), (3, 128, 3), (4, 512, 5),
                                                    (5, 256, 7), (8, 256, 1), (8, 128, 16),
                                                    (16, 128, 4), (16, 512, 2)])
def test_launch_shapes(grpo, oracle_mod, cluster, threads, chunks):
    rng = np.random.default_rng(cluster * 100 + threads + chunks)
    c = Case(rng, 23, 152064, "bf16", "bf16")
    r = c.run_oracle(oracle_mod)
    try:
        grpo.grpo_loss_tune(cluster, threads, chunks)
        g = c.run_gpu(grpo)
        g2 = c.run_gpu(grpo)
    finally:
        grpo.grpo_loss_tune(0, 0, 0)
    compare(g["logp"], g["dlogits"], g["loss"], r, "bf16", gpu_row_loss=g["row_loss"],
            cond=c.cond())
    assert g["loss"] == g2["loss"] and np.array_equal(g["dlogits"], g2["dlogits"])


@pytest.mark.parametrize("V,ind,outd", [(32001, "bf16", "bf16"), (5003, "f32", "bf16"),
                                        (152067, "bf16", "f32")])
def test_many_rows_per_cluster_with_unaligned_rows(grpo, oracle_mod, V, ind, outd):
    """More rows than resident clusters, with row lengths that are not a multiple of 16 bytes:
    every CTA runs many rows in a row and realigns its slice (the kernel's kAny instance), so the warp that
    read z_y and the warps that combine the row's entries differ from row to row."""
    rng = np.random.default_rng(V + 17)
    n = 1200 if V < 100000 else 700
    c = Case(rng, n, V, ind, outd)
    g = c.run_gpu(grpo)
    r = c.run_oracle(oracle_mod)
    assert g["status"] == 0
    compare(g["logp"], g["dlogits"], g["loss"], r, outd, gpu_row_loss=g["row_loss"],
            cond=c.cond())
    g2 = c.run_gpu(grpo)
    assert g2["loss"] == g["loss"] and np.array_equal(g2["dlogits"], g["dlogits"])


def test_single_cta_row_too_large_is_rejected(grpo):
    rng = np.random.default_rng(1)
    c = Case(rng, 2, 152064, "bf16", "bf16")
    try:
        grpo.grpo_loss_tune(1, 0, 0)
        with pytest.raises(grpo.GrpoError) as ei:
            c.run_gpu(grpo)
        assert ei.value.status == 2
    finally:
        grpo.grpo_loss_tune(0, 0, 0)


@pytest.mark.parametrize("V,ind", [(32000, "bf16"), (1001, "bf16"), (4096, "f32")])
def test_gathered_strided_rows(grpo, oracle_mod, V, ind):
    """row_index gathers rows from a larger buffer with a padded row stride."""
    import torch
    rng = np.random.default_rng(2)
    c = Case(rng, 64, V, ind, "bf16", stride=V + 24)
    idx = rng.choice(64, size=29, replace=False).astype(np.int64)
    rr = rng.integers(0, c.adv.size, size=29).astype(np.int32)
    g = c.run_gpu(grpo, n_rows=29, row_index=c.t(idx), rr=rr)
    r = oracle_mod.loss(c.host, V, c.y, c.old, c.ref, c.adv, rr, row_stride=c.stride,
                        row_index=idx, dlogits_dtype=1, beta=c.beta)
    compare(g["logp"], g["dlogits"], g["loss"], r, "bf16", gpu_row_loss=g["row_loss"],
            cond=c.cond(idx))


def test_unaligned_rows_take_the_realigning_path(grpo, oracle_mod):
    """A base pointer one element past a 16-byte boundary disables the bulk copies: the slices
    are realigned by the consumer threads."""
    import torch
    rng = np.random.default_rng(3)
    V = 5000
    c = Case(rng, 11, V, "bf16", "f32", stride=V + 8)
    full = c.dev.view(11, V + 8)
    logits = full[:, 1:V + 1]
    host = bf16_bits_to_f32(c.host).reshape(11, V + 8)[:, 1:V + 1]
    zz = host.astype(np.float64)
    m = zz.max(1, keepdims=True)
    logp = zz[np.arange(11), c.y] - (m[:, 0] + np.log(np.exp(zz - m).sum(1)))
    old = (logp + 0.05 * rng.standard_normal(11)).astype(np.float32)
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    lp = torch.empty(11, dtype=torch.float32, device="cuda")
    out = grpo.grpo_loss_fwd_bwd(logits, c.t(c.y), c.t(old), c.t(c.ref), c.t(c.adv), c.t(c.rr),
                                 dlogits_dtype="f32", logp_out=lp, status=status, beta=c.beta)
    torch.cuda.synchronize()
    r = oracle_mod.loss(np.ascontiguousarray(host), V, c.y, old, c.ref, c.adv, c.rr, beta=c.beta)
    compare(lp.cpu().numpy(), out["dlogits"].cpu().numpy(), float(out["loss"].item()), r, "f32",
            cond=c.cond())


def _loss_bits(grpo, c, logits, dlogits):
    """One call over c's rows with the given logits view and dlogits buffer; every output's bits."""
    import torch
    n = c.n
    logp = torch.empty(n, dtype=torch.float32, device="cuda")
    rl = torch.empty(n, dtype=torch.float64, device="cuda")
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    out = grpo.grpo_loss_fwd_bwd(logits, c.t(c.y), c.t(c.old), c.t(c.ref), c.t(c.adv), c.t(c.rr),
                                 V=c.V, beta=c.beta, dlogits=dlogits, logp_out=logp,
                                 row_loss_out=rl, status=status)
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    ibits = torch.int16 if dlogits.dtype == torch.bfloat16 else torch.int32
    return (out["loss"].view(torch.int64).item(), logp.view(torch.int32).cpu().numpy(),
            rl.view(torch.int64).cpu().numpy(), dlogits.view(ibits).cpu().numpy())


@pytest.mark.parametrize("V,ind,outd,in_off,stride_pad,out_off", [
    (32000, "bf16", "bf16", 1, 0, 0),        # every row one element past a boundary
    (32000, "bf16", "bf16", 0, 3, 0),        # row stride V + 3: each row a different offset
    (32000, "bf16", "bf16", 0, 0, 1),        # dlogits one element past a boundary
    (152064, "bf16", "bf16", 5, 1, 3),       # both, 7 CTAs per row
    (152064, "bf16", "f32", 3, 0, 1),
    (4096, "f32", "bf16", 1, 2, 3),
    (1024, "f32", "f32", 2, 1, 1),
    (61, "bf16", "bf16", 1, 1, 1),           # a row shorter than one slice's vectors
])
def test_unaligned_rows_give_the_aligned_bits(grpo, V, ind, outd, in_off, stride_pad, out_off):
    """Logits rows or dlogits rows that do not start on a 16-byte boundary (a base pointer past a
    boundary, a row stride that is not a multiple of 16 bytes) run the kernel's realigning
    instance: its vectors hold the same elements for the same threads, and its element-wise
    stores use the vector path's arithmetic, so it must reproduce the aligned call's bits (loss,
    logp, per-row terms, every dlogits entry) on the same values."""
    import torch
    rng = np.random.default_rng(V + 7 * in_off + 11 * stride_pad + 13 * out_off)
    n = 96 if V > 100000 else 257
    c = Case(rng, n, V, ind, outd)
    odt = torch.bfloat16 if outd == "bf16" else torch.float32
    ref = _loss_bits(grpo, c, c.dev, torch.empty(n, V, dtype=odt, device="cuda"))
    S = V + stride_pad
    flat = torch.zeros(in_off + n * S, dtype=c.dev.dtype, device="cuda")
    rows = flat[in_off:].view(n, S)
    rows[:, :V] = c.dev
    out_flat = torch.empty(out_off + n * V, dtype=odt, device="cuda")
    got = _loss_bits(grpo, c, rows[:, :V], out_flat[out_off:].view(n, V))
    assert got[0] == ref[0]
    for a, b in zip(got[1:], ref[1:]):
        assert np.array_equal(a, b)


def test_misaligned_element_pointer_is_rejected(grpo):
    """A logits pointer that is not a multiple of its element size is refused before any launch
    (the kernels' element loads need element-aligned addresses)."""
    import ctypes
    import torch
    rng = np.random.default_rng(4)
    n, V = 4, 64
    c = Case(rng, n, V, "bf16", "bf16")
    raw = torch.zeros(n * V * 2 + 2, dtype=torch.uint8, device="cuda")
    dl = torch.empty(n, V, dtype=torch.bfloat16, device="cuda")
    loss = torch.empty(1, dtype=torch.float64, device="cuda")
    rl = torch.empty(n, dtype=torch.float64, device="cuda")
    y, old, ref, adv, rr = (c.t(a) for a in (c.y, c.old, c.ref, c.adv, c.rr))
    lib = grpo.lib()
    st = lib.grpo_loss_fwd_bwd(raw.data_ptr() + 1, 1, V, None, n, V, y.data_ptr(), old.data_ptr(),
                               ref.data_ptr(), adv.data_ptr(), rr.data_ptr(), 0.2, 0.2, 0.04, 0, n,
                               None, 0, dl.data_ptr(), 1, None, rl.data_ptr(), loss.data_ptr(),
                               None, None, None, None)
    assert st == 1, st  # GRPO_ERR_INVALID_ARG
    assert b"element size" in lib.grpo_last_error()


def test_padding_an_odd_vocabulary_with_minus_inf_is_exact(grpo, oracle_mod):
    """Dense rows of an odd vocabulary (GPT-2's V = 50257) are not 16-byte aligned, so the fused
    loss realigns them, at under half of its streaming rate.  Padding
    the vocabulary to a multiple of 8 with -inf logits is exact: a padded column adds exp(-inf) = 0
    to every sum and gets a zero gradient, and the rows take the vector path.  Both calls match the
    oracle on the true vocabulary, and the padded columns' dlogits are exactly 0."""
    import torch
    rng = np.random.default_rng(50257)
    V, Vp, n = 50257, 50264, 300
    c = Case(rng, n, V, "bf16", "bf16")
    r = c.run_oracle(oracle_mod)
    dense = c.run_gpu(grpo)
    assert dense["status"] == 0
    compare(dense["logp"], dense["dlogits"], dense["loss"], r, "bf16",
            gpu_row_loss=dense["row_loss"], cond=c.cond())
    padded = torch.full((n, Vp), float("-inf"), dtype=torch.bfloat16, device="cuda")
    padded[:, :V] = c.dev.view(n, V)
    logp = torch.empty(n, dtype=torch.float32, device="cuda")
    rl = torch.empty(n, dtype=torch.float64, device="cuda")
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    out = grpo.grpo_loss_fwd_bwd(padded, c.t(c.y), c.t(c.old), c.t(c.ref), c.t(c.adv), c.t(c.rr),
                                 beta=c.beta, logp_out=logp, row_loss_out=rl, status=status)
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    dl = out["dlogits"].view(torch.int16).cpu().numpy().view(np.uint16)
    assert np.all((dl[:, V:] & 0x7FFF) == 0)  # +0 or -0 (a negative scale times exp(-inf))
    compare(logp.cpu().numpy(), dl[:, :V], float(out["loss"].item()), r, "bf16",
            gpu_row_loss=rl.cpu().numpy(), cond=c.cond())


def test_sequence_mean(grpo, oracle_mod):
    import torch
    rng = np.random.default_rng(4)
    c = Case(rng, 40, 32000, "bf16", "bf16", n_roll=5)
    rr = np.sort(rng.integers(0, 5, size=40)).astype(np.int32)
    lens = np.bincount(rr, minlength=5)
    seq_off = np.concatenate([[0], np.cumsum(lens)]).astype(np.int64)
    n_seq = int((lens > 0).sum())
    g = c.run_gpu(grpo, rr=rr, agg_mode=1, seq_off=c.t(seq_off), n_seq=n_seq)
    r = oracle_mod.loss(c.host, c.V, c.y, c.old, c.ref, c.adv, rr, agg_mode=1, seq_off=seq_off,
                        n_seq=n_seq, dlogits_dtype=1, beta=c.beta)
    compare(g["logp"], g["dlogits"], g["loss"], r, "bf16", gpu_row_loss=g["row_loss"],
            cond=c.cond())


@pytest.mark.parametrize("beta", [0.0, 0.04])
def test_asymmetric_clip(grpo, oracle_mod, beta):
    """Eq. 2 with different lower and upper clip widths (eps_low 0.2, eps_high 0.28).  Old
    log-probs far from the current ones put many rows outside the clip range on both sides.
    Where the clip is active (A > 0 above 1 + eps_high, A < 0 below 1 - eps_low) the surrogate
    is constant, so with beta = 0 those rows' gradient is exactly zero."""
    rng = np.random.default_rng(12)
    c = Case(rng, 96, 32000, "bf16", "bf16", beta=beta, old_noise=0.35, n_roll=8)
    g = c.run_gpu(grpo, eps_low=0.2, eps_high=0.28)
    r = c.run_oracle(oracle_mod, eps_low=0.2, eps_high=0.28)
    assert g["status"] == 0
    compare(g["logp"], g["dlogits"], g["loss"], r, "bf16", eps_low=0.2, eps_high=0.28,
            gpu_row_loss=g["row_loss"], cond=c.cond())
    A = c.adv[c.rr].astype(np.float64)
    rho = r["rho"][:c.n]
    active = ((A > 0) & (rho > 1.28 * (1 + 1e-5))) | ((A < 0) & (rho < 0.8 * (1 - 1e-5)))
    inside = (rho > 0.8 * (1 + 1e-5)) & (rho < 1.28 * (1 - 1e-5)) & (A != 0)
    assert active.sum() >= 10 and inside.sum() >= 10
    if beta == 0.0:
        assert np.all((g["dlogits"][active] & 0x7FFF) == 0)
        assert np.all(np.any(g["dlogits"][inside] & 0x7FFF, axis=1))


def test_deterministic(grpo):
    rng = np.random.default_rng(5)
    c = Case(rng, 50, 152064, "bf16", "bf16")
    a, b = c.run_gpu(grpo), c.run_gpu(grpo)
    assert a["loss"] == b["loss"]
    assert np.array_equal(a["dlogits"], b["dlogits"]) and np.array_equal(a["logp"], b["logp"])


def test_no_rows(grpo):
    rng = np.random.default_rng(6)
    c = Case(rng, 3, 1000, "bf16", "bf16")
    g = c.run_gpu(grpo, n_rows=0)
    assert g["loss"] == 0.0 and g["status"] == 0


def test_zero_advantage_without_kl_is_exactly_zero(grpo):
    rng = np.random.default_rng(7)
    c = Case(rng, 9, 32000, "bf16", "bf16", beta=0.0, A=[0.0, 0.0])
    g = c.run_gpu(grpo)
    assert np.all((g["dlogits"] & 0x7FFF) == 0) and g["loss"] == 0.0


def test_bad_token_sets_status_and_zero_row(grpo, oracle_mod):
    rng = np.random.default_rng(8)
    c = Case(rng, 6, 1000, "bf16", "bf16")
    c.y[2] = 1000
    c.y[4] = -5
    g = c.run_gpu(grpo)
    assert g["status"] & grpo.binding.DEVFLAG_BAD_TOKEN
    r = c.run_oracle(oracle_mod)
    assert np.isnan(g["logp"][2]) and np.isnan(g["logp"][4])
    assert np.all((g["dlogits"][[2, 4]] & 0x7FFF) == 0)
    compare(g["logp"], g["dlogits"], g["loss"], r, "bf16", cond=c.cond())


def test_nonfinite_logits_set_status(grpo):
    import torch
    rng = np.random.default_rng(9)
    c = Case(rng, 4, 2000, "f32", "f32")
    host = c.host.copy()
    host[1, 17] = np.nan
    c.host = host
    c.dev = torch.from_numpy(host).cuda()
    g = c.run_gpu(grpo)
    assert g["status"] & grpo.binding.DEVFLAG_NONFINITE
    assert np.isnan(g["logp"][1]) and np.all(np.isfinite(g["logp"][[0, 2, 3]]))


def test_masked_vocabulary(grpo, oracle_mod):
    """-inf logits (a masked vocabulary range, whole slices included) contribute nothing."""
    import torch
    rng = np.random.default_rng(10)
    c = Case(rng, 8, 152064, "bf16", "bf16")
    host = c.host.copy()
    host[:, 40000:120000] = 0xFF80  # bf16 -inf
    c.y = rng.integers(0, 40000, size=8).astype(np.int32)
    c.host = host
    c.dev = torch.from_numpy(host.view(np.int16)).cuda().view(torch.bfloat16)
    zz = bf16_bits_to_f32(host).astype(np.float64)
    m = zz.max(1, keepdims=True)
    logp = zz[np.arange(8), c.y] - (m[:, 0] + np.log(np.exp(zz - m).sum(1)))
    c.old = (logp + 0.05 * rng.standard_normal(8)).astype(np.float32)
    g = c.run_gpu(grpo)
    r = c.run_oracle(oracle_mod)
    assert g["status"] == 0
    compare(g["logp"], g["dlogits"], g["loss"], r, "bf16", gpu_row_loss=g["row_loss"],
            cond=c.cond())


def test_peaked_rows_keep_one_minus_p_accurate(grpo, oracle_mod):
    """When p_y is close to 1 the y entry is coef*(1 - p_y); it is formed from the sum that
    leaves y out, so it keeps full relative accuracy."""
    rng = np.random.default_rng(11)
    c = Case(rng, 12, 32000, "bf16", "bf16", scale=1.0)
    host = bf16_bits_to_f32(c.host).reshape(12, 32000).copy()
    host[np.arange(12), c.y] = 24.0
    c.host = bf16_bits(host)
    import torch
    c.dev = torch.from_numpy(c.host.view(np.int16)).cuda().view(torch.bfloat16)
    zz = host.astype(np.float64)
    m = zz.max(1, keepdims=True)
    logp = zz[np.arange(12), c.y] - (m[:, 0] + np.log(np.exp(zz - m).sum(1)))
    c.old = (logp + 0.05 * rng.standard_normal(12)).astype(np.float32)
    c.ref = (logp + 0.1 * rng.standard_normal(12)).astype(np.float32)
    g = c.run_gpu(grpo)
    r = c.run_oracle(oracle_mod)
    compare(g["logp"], g["dlogits"], g["loss"], r, "bf16", cond=c.cond())


@pytest.mark.parametrize("agg_mode", [0, 1])
def test_device_row_count_matches_host_count(grpo, agg_mode):
    """grpo_loss_fwd_bwd_dev over min(max_rows, T_kept) rows, with its denominators from the
    device counts, equals grpo_loss_fwd_bwd given the same numbers on the host, bit for bit."""
    import torch
    rng = np.random.default_rng(40 + agg_mode)
    c = Case(rng, 64, 32000, "bf16", "bf16", n_roll=6)
    rr = np.sort(rng.integers(0, 6, size=64)).astype(np.int32)
    lens = np.bincount(rr, minlength=6)
    seq_off = c.t(np.concatenate([[0], np.cumsum(lens)]).astype(np.int64))
    for t_kept in (0, 1, 37, 64):
        K = int((lens[:6] > 0).sum())
        counts = c.t(np.array([K, t_kept], np.int64))
        dl_a = torch.zeros((64, 32000), dtype=torch.bfloat16, device="cuda")
        dl_b = torch.zeros_like(dl_a)
        la = torch.empty(1, dtype=torch.float64, device="cuda")
        lb = torch.empty(1, dtype=torch.float64, device="cuda")
        ws = torch.empty(64 * 8 + 512, dtype=torch.uint8, device="cuda")
        grpo.grpo_loss_fwd_bwd_dev(c.dev, c.t(c.y), c.t(c.old), c.t(c.ref), c.t(c.adv), c.t(rr),
                                   counts, max_rows=64, dlogits=dl_a, loss_out=la, ws=ws,
                                   beta=c.beta, agg_mode=agg_mode, seq_off=seq_off)
        if t_kept:
            grpo.grpo_loss_fwd_bwd(c.dev, c.t(c.y), c.t(c.old), c.t(c.ref), c.t(c.adv), c.t(rr),
                                   n_rows=t_kept, beta=c.beta, agg_mode=agg_mode,
                                   denom_tokens=t_kept, seq_off=seq_off, n_seq=K, dlogits=dl_b,
                                   loss_out=lb)
        else:
            lb.zero_()
        torch.cuda.synchronize()
        assert la.item() == lb.item()
        assert torch.equal(dl_a, dl_b)  # rows past T_kept untouched (still zero) in both


def test_lost_copy_times_out_and_the_context_stays_usable(grpo, oracle_mod):
    """Failure detection without a fault: the test hook arms one copy that is never issued.  The
    waiting CTA gives up after about a second, the kernel reports GRPO_DEVFLAG_TIMEOUT and
    returns; the next launch on the same context is correct."""
    import time
    rng = np.random.default_rng(99)
    c = Case(rng, 24, 152064, "bf16", "bf16")
    grpo.binding.lib().grpo_test_skip_copy(1)
    t0 = time.time()
    bad = c.run_gpu(grpo)
    elapsed = time.time() - t0
    assert bad["status"] & grpo.binding.DEVFLAG_TIMEOUT
    assert elapsed < 30.0
    good = c.run_gpu(grpo)
    assert good["status"] == 0
    compare(good["logp"], good["dlogits"], good["loss"], c.run_oracle(oracle_mod), "bf16",
            gpu_row_loss=good["row_loss"], cond=c.cond())


@pytest.mark.parametrize("V", [262144, 600000])
def test_large_vocabularies(grpo, oracle_mod, V):
    """Vocabularies beyond today's common sizes: 7 CTAs per row at V = 262144, and 11 at
    V = 600000 (a cluster above the portable size of 8)."""
    rng = np.random.default_rng(V)
    c = Case(rng, 5, V, "bf16", "bf16")
    g = c.run_gpu(grpo)
    r = c.run_oracle(oracle_mod)
    assert g["status"] == 0
    compare(g["logp"], g["dlogits"], g["loss"], r, "bf16", gpu_row_loss=g["row_loss"],
            cond=c.cond())
    lp = grpo.grpo_logp_fwd(c.dev, c.t(c.y)).cpu().numpy()[:5]
    assert np.abs(lp.astype(np.float64) - r["logp"]).max() <= 2e-5


def test_injected_launch_failure_is_reported_and_the_next_call_is_clean(grpo, oracle_mod):
    """Host-side fault injection: the test hook makes one launch check report an error.  The call
    raises GrpoError with the injected message; the next call, with nothing armed, matches the
    oracle.  Nothing faults on the device."""
    rng = np.random.default_rng(98)
    c = Case(rng, 24, 1000, "bf16", "bf16")
    grpo.binding.lib().grpo_test_fail_launch(1)
    try:
        with pytest.raises(grpo.GrpoError) as err:
            c.run_gpu(grpo)
    finally:
        grpo.binding.lib().grpo_test_fail_launch(0)
    assert "injected launch failure" in str(err.value)
    assert err.value.status == 4  # GRPO_ERR_CUDA
    good = c.run_gpu(grpo)
    assert good["status"] == 0
    compare(good["logp"], good["dlogits"], good["loss"], c.run_oracle(oracle_mod), "bf16",
            gpu_row_loss=good["row_loss"], cond=c.cond())
