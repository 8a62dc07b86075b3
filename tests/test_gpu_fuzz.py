"""Randomised parity of the fused loss and GSPO's loss with the oracle: vocabulary sizes from 1
to 70000 (odd ones included), both dtypes in and out, padded and gathered rows, clip widths,
beta and the aggregation mode drawn at random (seeded, so every failure is reproducible); and
the fused loss's bits under random row alignments against an aligned layout of the same rows."""
import numpy as np
import pytest

from loss_compare import compare
from test_gpu_gspo import SeqCase, compare_gspo
from test_gpu_loss import Case

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("seed", range(12))
def test_fused_loss_random_configurations(grpo, oracle_mod, seed):
    rng = np.random.default_rng(1000 + seed)
    V = int(rng.choice([1, 2, 7, 33, 1000, 4097]) if seed % 3 == 0 else rng.integers(1, 70000))
    ind, outd = rng.choice(["bf16", "f32"]), rng.choice(["bf16", "f32"])
    n = int(rng.integers(1, 24 if V > 20000 else 60))
    pad = int(rng.choice([0, 0, 8, 5]))
    c = Case(rng, n + 3, V, ind, outd, stride=V + pad, n_roll=5, beta=float(rng.choice([0.0, 0.04])),
             old_noise=float(rng.choice([0.05, 0.3])))
    eps_low, eps_high = float(rng.choice([0.1, 0.2])), float(rng.choice([0.2, 0.28]))
    idx = rng.choice(n + 3, size=n, replace=False).astype(np.int64)
    rr = np.sort(rng.integers(0, 5, size=n)).astype(np.int32)
    agg = int(rng.integers(0, 2))
    kw = dict(eps_low=eps_low, eps_high=eps_high)
    if agg:
        lens = np.bincount(rr, minlength=5)
        seq_off = np.concatenate([[0], np.cumsum(lens)]).astype(np.int64)
        kw.update(agg_mode=1, n_seq=int((lens > 0).sum()))
        g = c.run_gpu(grpo, n_rows=n, row_index=c.t(idx), rr=rr, seq_off=c.t(seq_off), **kw)
        r = oracle_mod.loss(c.host, V, c.y, c.old, c.ref, c.adv, rr, row_stride=c.stride,
                            row_index=idx, seq_off=seq_off, beta=c.beta,
                            dlogits_dtype=1 if outd == "bf16" else 0, **kw)
    else:
        g = c.run_gpu(grpo, n_rows=n, row_index=c.t(idx), rr=rr, **kw)
        r = oracle_mod.loss(c.host, V, c.y, c.old, c.ref, c.adv, rr, row_stride=c.stride,
                            row_index=idx, beta=c.beta, dlogits_dtype=1 if outd == "bf16" else 0,
                            **kw)
    assert g["status"] == 0
    compare(g["logp"], g["dlogits"], g["loss"], r, outd, eps_low=eps_low, eps_high=eps_high,
            gpu_row_loss=g["row_loss"], cond=c.cond(idx))


@pytest.mark.parametrize("seed", range(8))
def test_gspo_random_configurations(grpo, oracle_mod, seed):
    rng = np.random.default_rng(2000 + seed)
    V = int(rng.choice([5, 1000, 4097]) if seed % 3 == 0 else rng.integers(8, 60000))
    ind, outd = rng.choice(["bf16", "f32"]), rng.choice(["bf16", "f32"])
    K = int(rng.integers(1, 9))
    lens = list(rng.integers(0, 30 if V > 20000 else 60, size=K))
    if sum(lens) == 0:
        lens[0] = 3
    c = SeqCase(rng, lens, V, ind, outd, old_sd=float(rng.choice([0.02, 0.2])),
                beta=float(rng.choice([0.0, 0.04])), eps=(0.2, float(rng.choice([0.2, 0.28]))),
                gather=bool(rng.integers(0, 2)))
    g, r = c.run_gpu(grpo), c.run_oracle(oracle_mod)
    compare_gspo(g, r, c)


@pytest.mark.parametrize("seed", range(12))
def test_fused_loss_bits_do_not_depend_on_alignment(grpo, seed):
    """The same gathered rows, once from a buffer whose rows start on 16-byte boundaries and once
    from one whose base, row stride and dlogits base are drawn at random (an element past a
    boundary, a stride of V + 0..9): every output must have the same bits, whichever kernel
    instance each layout selects."""
    import torch
    rng = np.random.default_rng(3000 + seed)
    V = int(rng.choice([1, 3, 9, 61, 1001, 4099]) if seed % 3 == 0 else rng.integers(1, 70000))
    ind, outd = str(rng.choice(["bf16", "f32"])), str(rng.choice(["bf16", "f32"]))
    n_src = int(rng.integers(2, 20 if V > 20000 else 80))
    c = Case(rng, n_src, V, ind, outd, n_roll=5, beta=float(rng.choice([0.0, 0.04])))
    n = int(rng.integers(1, n_src + 1))
    idx = rng.choice(n_src, size=n, replace=False).astype(np.int64)
    rr = rng.integers(0, 5, size=n).astype(np.int32)
    elem = 8 if ind == "bf16" else 4
    odt = torch.bfloat16 if outd == "bf16" else torch.float32

    def call(rows, S, dl):
        logp = torch.empty(n, dtype=torch.float32, device="cuda")
        rl = torch.empty(n, dtype=torch.float64, device="cuda")
        status = torch.zeros(1, dtype=torch.int32, device="cuda")
        out = grpo.grpo_loss_fwd_bwd(rows, c.t(c.y), c.t(c.old), c.t(c.ref), c.t(c.adv), c.t(rr),
                                     V=V, row_stride=S, row_index=c.t(idx), n_rows=n,
                                     beta=c.beta, dlogits=dl, logp_out=logp, row_loss_out=rl,
                                     status=status)
        torch.cuda.synchronize()
        assert int(status.item()) == 0
        bits = torch.int16 if outd == "bf16" else torch.int32
        return (out["loss"].view(torch.int64).item(), logp.view(torch.int32).cpu().numpy(),
                rl.view(torch.int64).cpu().numpy(), dl.view(bits).cpu().numpy())

    def layout(off, S, out_off):
        flat = torch.zeros(off + n_src * S, dtype=c.dev.dtype, device="cuda")
        rows = flat[off:].view(n_src, S)
        rows[:, :V] = c.dev.view(n_src, V)
        out = torch.empty(out_off + n * V, dtype=odt, device="cuda")
        return call(rows[:, :V], S, out[out_off:].view(n, V))

    ref = layout(0, -(-V // elem) * elem, 0)
    got = layout(int(rng.integers(0, elem)), V + int(rng.integers(0, 10)), int(rng.integers(0, 8)))
    assert got[0] == ref[0]
    for a, b in zip(got[1:], ref[1:]):
        assert np.array_equal(a, b)
