"""The allocation-free loss entry (grpo_loss_fwd_bwd_noalloc), for callers that cannot allocate
device memory when the loss runs (a host that hands over only inputs and outputs, or a runtime
that forbids allocation after start-up).  It must give the same results as grpo_loss_fwd_bwd,
call after call, although its scratch is one fixed array inside the library that every call
reuses.  This file is collected last so that a run stopping at the first failure has already
run every other test."""

import numpy as np
import pytest

from loss_compare import compare


def _case(rng, n, V):
    import torch
    z = torch.from_numpy((rng.standard_normal((n, V)) * 2.0).astype(np.float32)).to(torch.bfloat16)
    y = rng.integers(0, V, size=n).astype(np.int32)
    zz = z.float().double().numpy()
    m = zz.max(1, keepdims=True)
    logp = zz[np.arange(n), y] - (m[:, 0] + np.log(np.exp(zz - m).sum(1)))
    old = (logp + 0.05 * rng.standard_normal(n)).astype(np.float32)
    ref = (logp + 0.1 * rng.standard_normal(n)).astype(np.float32)
    adv = rng.standard_normal(5).astype(np.float32)
    rr = rng.integers(0, 5, size=n).astype(np.int32)
    dev = dict(logits=z.cuda(), y=torch.from_numpy(y).cuda(), old=torch.from_numpy(old).cuda(),
               ref=torch.from_numpy(ref).cuda(), adv=torch.from_numpy(adv).cuda(),
               rr=torch.from_numpy(rr).cuda())
    return dev


def _outputs(n, V):
    import torch
    return dict(dlogits=torch.empty((n, V), dtype=torch.bfloat16, device="cuda"),
                logp=torch.empty(n, dtype=torch.float32, device="cuda"),
                loss=torch.empty(1, dtype=torch.float64, device="cuda"),
                status=torch.zeros(1, dtype=torch.int32, device="cuda"))


def _host(o):
    import torch
    return dict(loss=float(o["loss"].item()), logp=o["logp"].cpu().numpy(),
                dlogits=o["dlogits"].view(torch.int16).cpu().numpy().view(np.uint16),
                status=int(o["status"].item()))


@pytest.mark.gpu
def test_noalloc_matches_workspace_entry_on_two_calls_in_a_row(grpo):
    import torch
    rng = np.random.default_rng(2024)
    # two different batches, so the second call cannot pass on the first call's scratch
    for n, V in ((301, 152064), (777, 32001)):
        d = _case(rng, n, V)
        ref_o = _outputs(n, V)
        grpo.grpo_loss_fwd_bwd(d["logits"], d["y"], d["old"], d["ref"], d["adv"], d["rr"],
                               dlogits=ref_o["dlogits"], logp_out=ref_o["logp"],
                               loss_out=ref_o["loss"], status=ref_o["status"])
        got_o = _outputs(n, V)
        grpo.grpo_loss_fwd_bwd_noalloc(d["logits"], d["y"], d["old"], d["ref"], d["adv"], d["rr"],
                                       dlogits=got_o["dlogits"], logp_out=got_o["logp"],
                                       loss_out=got_o["loss"], status=got_o["status"])
        torch.cuda.synchronize()
        a, b = _host(ref_o), _host(got_o)
        assert a["status"] == 0 and b["status"] == 0
        ref_like = dict(logp=a["logp"].astype(np.float64), rho=np.ones(n), dlogits=a["dlogits"],
                        loss=a["loss"], row_loss=None)
        compare(b["logp"], b["dlogits"], b["loss"], ref_like, "bf16")


def test_noalloc_rejects_rows_beyond_its_scratch(grpo):
    """Checked on the host before any GPU work: no device needed."""
    L = grpo.lib()
    rc = L.grpo_loss_fwd_bwd_noalloc(None, 1, 1000, None, 262145, 1000, None, None, None, None,
                                     None, 0.2, 0.2, 0.04, 0, 1, None, 0, None, 1, None, None,
                                     None, None, None)
    assert rc == 2
    assert b"262144" in L.grpo_last_error()
