"""The allocation-free loss entry (grpo_loss_fwd_bwd_noalloc), for callers that cannot allocate
device memory when the loss runs (a host that hands over only inputs and outputs, or a runtime
that forbids allocation after start-up).  It runs the same kernel, launch shape and summation
order as grpo_loss_fwd_bwd, so its loss, logp and dlogits must equal that entry's bit for bit,
call after call, although its scratch is one fixed array inside the library that every call
reuses.  This file is collected last so that a run stopping at the first failure has already
run every other test."""

import numpy as np
import pytest


def _case(rng, n, V, n_roll=5):
    import torch
    z = torch.from_numpy((rng.standard_normal((n, V)) * 2.0).astype(np.float32)).to(torch.bfloat16)
    y = rng.integers(0, V, size=n).astype(np.int32)
    zz = z.float().double().numpy()
    m = zz.max(1, keepdims=True)
    logp = zz[np.arange(n), y] - (m[:, 0] + np.log(np.exp(zz - m).sum(1)))
    old = (logp + 0.05 * rng.standard_normal(n)).astype(np.float32)
    ref = (logp + 0.1 * rng.standard_normal(n)).astype(np.float32)
    adv = rng.standard_normal(n_roll).astype(np.float32)
    rr = np.sort(rng.integers(0, n_roll, size=n)).astype(np.int32)
    lens = np.bincount(rr, minlength=n_roll)
    seq_off = np.concatenate([[0], np.cumsum(lens)]).astype(np.int64)
    dev = dict(logits=z.cuda(), y=torch.from_numpy(y).cuda(), old=torch.from_numpy(old).cuda(),
               ref=torch.from_numpy(ref).cuda(), adv=torch.from_numpy(adv).cuda(),
               rr=torch.from_numpy(rr).cuda(), seq_off=torch.from_numpy(seq_off).cuda(),
               n_seq=int((lens > 0).sum()))
    return dev


def _outputs(n, V, row_loss):
    import torch
    return dict(dlogits=torch.empty((max(n, 1), V), dtype=torch.bfloat16, device="cuda"),
                logp=torch.empty(max(n, 1), dtype=torch.float32, device="cuda"),
                row_loss=(torch.empty(max(n, 1), dtype=torch.float64, device="cuda")
                          if row_loss else None),
                loss=torch.full((1,), 12345.0, dtype=torch.float64, device="cuda"),
                status=torch.zeros(1, dtype=torch.int32, device="cuda"))


def _host(o, n):
    import torch
    return dict(loss=float(o["loss"].item()), logp=o["logp"][:n].cpu().numpy().view(np.uint32),
                dlogits=o["dlogits"][:n].view(torch.int16).cpu().numpy().view(np.uint16),
                row_loss=None if o["row_loss"] is None else o["row_loss"][:n].cpu().numpy(),
                status=int(o["status"].item()))


def _run(fn, d, o, n, agg):
    kw = dict(agg_mode=agg, seq_off=d["seq_off"], n_seq=d["n_seq"]) if agg else {}
    fn(d["logits"], d["y"], d["old"], d["ref"], d["adv"], d["rr"], n_rows=n,
       dlogits=o["dlogits"], logp_out=o["logp"], row_loss_out=o["row_loss"], loss_out=o["loss"],
       status=o["status"], **kw)


# The larger batch comes first, so that the smaller calls after it find the shared scratch full
# of the earlier call's rows; then Eq. 1's sequence mean, the caller's own row-loss buffer, and
# an empty call.
CALLS = [(777, 32001, 0, False), (301, 152064, 1, False), (5, 1000, 0, False),
         (64, 4097, 0, True), (0, 1000, 0, False)]


@pytest.mark.gpu
def test_noalloc_equals_workspace_entry_bit_for_bit_call_after_call(grpo):
    import torch
    rng = np.random.default_rng(2024)
    for n, V, agg, own_rows in CALLS:
        d = _case(rng, max(n, 1), V)
        ref_o, got_o = _outputs(n, V, own_rows), _outputs(n, V, own_rows)
        _run(grpo.grpo_loss_fwd_bwd, d, ref_o, n, agg)
        _run(grpo.grpo_loss_fwd_bwd_noalloc, d, got_o, n, agg)
        torch.cuda.synchronize()
        a, b = _host(ref_o, n), _host(got_o, n)
        assert a["status"] == 0 and b["status"] == 0
        assert b["loss"] == a["loss"], (n, V, agg, b["loss"], a["loss"])
        assert np.array_equal(b["logp"], a["logp"])
        assert np.array_equal(b["dlogits"], a["dlogits"])
        if own_rows:
            assert np.array_equal(b["row_loss"], a["row_loss"])
        if n == 0:
            assert b["loss"] == 0.0


def test_noalloc_rejects_rows_beyond_its_scratch(grpo):
    """Checked on the host before any GPU work: no device needed."""
    L = grpo.lib()
    rc = L.grpo_loss_fwd_bwd_noalloc(None, 1, 1000, None, 262145, 1000, None, None, None, None,
                                     None, 0.2, 0.2, 0.04, 0, 1, None, 0, None, 1, None, None,
                                     None, None, None)
    assert rc == 2
    assert b"262144" in L.grpo_last_error()
