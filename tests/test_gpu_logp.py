"""GPU parity of grpo_logp_fwd (the old/reference policy evaluation: log pi(y) alone) with the
oracle's logp: within 2e-5 absolute, over vocabularies with ragged tails, both input dtypes,
launch shapes, gathered rows, invalid ids and the workloads' full size."""
import numpy as np
import pytest


pytestmark = pytest.mark.gpu
LOGP_ATOL = 2e-5


def case(rng, n, V, dtype, stride=None, scale=3.0):
    import torch
    stride = V if stride is None else stride
    z = (rng.standard_normal((n, stride)) * scale).astype(np.float32)
    if dtype == "bf16":
        host = torch.from_numpy(z).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
        dev = torch.from_numpy(host.view(np.int16)).cuda().view(torch.bfloat16)
    else:
        host, dev = z, torch.from_numpy(z).cuda()
    y = rng.integers(0, V, size=n).astype(np.int32)
    return host, dev, y


def run(grpo, dev, y, V, stride, **kw):
    import torch
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    logits = dev.view(-1, stride)[:, :V]
    out = grpo.grpo_logp_fwd(logits, torch.from_numpy(y).cuda(), V=V, row_stride=stride,
                             status=status, **kw)
    torch.cuda.synchronize()
    return out.cpu().numpy(), int(status.item())


@pytest.mark.parametrize("V,dtype", [(1, "f32"), (9, "bf16"), (1001, "bf16"), (4096, "f32"),
                                     (32000, "bf16"), (32001, "f32"), (152064, "bf16"),
                                     (152067, "bf16")])
def test_logp_matches_oracle(grpo, oracle_mod, V, dtype):
    rng = np.random.default_rng(V + 3)
    n = 41 if V < 100000 else 17
    host, dev, y = case(rng, n, V, dtype)
    got, st = run(grpo, dev, y, V, V)
    assert st == 0
    ref = oracle_mod.logp(host, V, y)
    assert np.abs(got[:n].astype(np.float64) - ref).max() <= LOGP_ATOL


@pytest.mark.parametrize("V,ind", [(5000, "bf16"), (32001, "f32"), (152064, "bf16")])
def test_logp_unaligned_rows(grpo, oracle_mod, V, ind):
    """Rows that start one element past a 16-byte boundary are realigned: each 16-byte vector
    from the two aligned words that hold it."""
    import torch
    rng = np.random.default_rng(V + 1)
    stride = V + 8
    host, dev, y = case(rng, 13, stride, ind)
    y = rng.integers(0, V, size=13).astype(np.int32)
    full = dev.view(13, stride)
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    out = grpo.grpo_logp_fwd(full[:, 1:V + 1], torch.from_numpy(y).cuda(), V=V, row_stride=stride,
                             status=status)
    torch.cuda.synchronize()
    hv = (host.reshape(13, stride)[:, 1:V + 1]).copy()
    ref = oracle_mod.logp(hv, V, y)
    assert int(status.item()) == 0
    assert np.abs(out.cpu().numpy()[:13].astype(np.float64) - ref).max() <= LOGP_ATOL


def test_logp_gathered_rows_and_bad_ids(grpo, oracle_mod):
    import torch
    rng = np.random.default_rng(5)
    V, stride = 32000, 32008
    host, dev, y = case(rng, 50, V, "bf16", stride=stride)
    y[7] = V
    idx = rng.choice(50, 23, replace=False).astype(np.int64)
    idx[0] = 7
    got, st = run(grpo, dev, y, V, stride, row_index=torch.from_numpy(idx).cuda(), n_rows=23)
    assert st & grpo.binding.DEVFLAG_BAD_TOKEN
    ref = oracle_mod.logp(host, V, y, row_index=idx, row_stride=stride)
    got = got[:23].astype(np.float64)
    assert np.isnan(got[0]) and np.array_equal(np.isnan(got), np.isnan(ref))
    ok = ~np.isnan(ref)
    assert np.abs(got[ok] - ref[ok]).max() <= LOGP_ATOL


@pytest.mark.parametrize("V", [32000, 152064])
def test_logp_agrees_with_the_loss_kernel(grpo, V):
    """The forward-only kernel and the fused loss report the same log-probabilities to within a
    few ulps (their sums run in different orders), so the ratio of a policy to itself is 1 to
    within ~1e-6."""
    import torch
    rng = np.random.default_rng(6)
    host, dev, y = case(rng, 64, V, "bf16")
    yt = torch.from_numpy(y).cuda()
    z = torch.zeros(64, dtype=torch.float32, device="cuda")
    lp2 = torch.empty(64, dtype=torch.float32, device="cuda")
    grpo.grpo_loss_fwd_bwd(dev.view(64, V), yt, z, z, torch.zeros(1, device="cuda"),
                           torch.zeros(64, dtype=torch.int32, device="cuda"), logp_out=lp2)
    torch.cuda.synchronize()
    lp, lp2 = run(grpo, dev, y, V, V)[0], lp2.cpu().numpy()
    ulp = np.spacing(np.abs(lp2).astype(np.float32)).astype(np.float64)
    assert np.all(np.abs(lp.astype(np.float64) - lp2) <= 4 * ulp)


def test_logp_ignores_the_loss_launch_shape(grpo):
    """grpo_loss_tune shapes the fused loss only: the forward-only kernel gives the same bits
    under any setting."""
    rng = np.random.default_rng(7)
    host, dev, y = case(rng, 33, 152064, "bf16")
    base = run(grpo, dev, y, 152064, 152064)[0]
    try:
        for shape in ((4, 256, 2), (2, 128, 1), (8, 512, 3)):
            grpo.grpo_loss_tune(*shape)
            assert np.array_equal(run(grpo, dev, y, 152064, 152064)[0], base)
    finally:
        grpo.grpo_loss_tune(0, 0, 0)


def test_logp_full_size_sampled(grpo, oracle_mod):
    """All 52779 token rows of the qwen workload; 48 sampled rows against the oracle."""
    import torch
    from paper_2609_36932_gb300 import workloads
    w = workloads.get("qwen")
    b = workloads.make_batch(w, 0)
    logits = workloads.logits_rows(w, 0, range(b["T"]), torch.device("cuda", 0))
    y = torch.from_numpy(b["ids"]).cuda()
    out = grpo.grpo_logp_fwd(logits, y)
    torch.cuda.synchronize()
    rows = np.random.default_rng(1).choice(b["T"], 48, replace=False)
    host = logits[torch.from_numpy(rows).cuda()].view(torch.int16).cpu().numpy().view(np.uint16)
    ref = oracle_mod.logp(host, w.V, b["ids"][rows])
    assert np.abs(out.cpu().numpy()[rows].astype(np.float64) - ref).max() <= LOGP_ATOL


@pytest.mark.parametrize("V,dtype,off,pad", [(152064, "bf16", 1, 0), (152064, "bf16", 0, 3),
                                             (50257, "bf16", 0, 0), (32001, "f32", 1, 1),
                                             (61, "bf16", 3, 1)])
def test_logp_unaligned_rows_give_the_aligned_bits(grpo, V, dtype, off, pad):
    """The realigning instance gives each thread the same vectors as the aligned one: the same
    values at another alignment (base off elements past a boundary, row stride V + pad) give
    the same logp bits."""
    import torch
    rng = np.random.default_rng(V + off + 10 * pad)
    n = 64
    host, dev, y = case(rng, n, V, dtype)
    yd = torch.from_numpy(y).cuda()
    ref = grpo.grpo_logp_fwd(dev.view(n, V), yd).view(torch.int32).cpu().numpy()
    S = V + pad
    flat = torch.zeros(off + n * S, dtype=dev.dtype, device="cuda")
    rows = flat[off:].view(n, S)
    rows[:, :V] = dev.view(n, V)
    got = grpo.grpo_logp_fwd(rows[:, :V], yd, V=V, row_stride=S).view(torch.int32).cpu().numpy()
    assert np.array_equal(got[:n], ref[:n])


def test_logp_misaligned_element_pointer_is_rejected(grpo):
    """A logits pointer that is not a multiple of its element size is refused before any launch."""
    import torch
    n, V = 4, 64
    raw = torch.zeros(n * V * 2 + 2, dtype=torch.uint8, device="cuda")
    y = torch.zeros(n, dtype=torch.int32, device="cuda")
    logp = torch.empty(n, dtype=torch.float32, device="cuda")
    lib = grpo.lib()
    st = lib.grpo_logp_fwd(raw.data_ptr() + 1, 1, V, None, n, V, y.data_ptr(), logp.data_ptr(),
                           None, None)
    assert st == 1, st  # GRPO_ERR_INVALID_ARG
    assert b"element size" in lib.grpo_last_error()
