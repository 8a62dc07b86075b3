"""grpo_sum_f64, the fixed-order fp64 sum that ends every loss call (and lets a loss computed in
chunks sum to the bits of one call), against exact sums: math.fsum gives the exactly rounded sum,
and any summation order in fp64 stays within (n - 1) * 2^-53 * sum |v| of it; terms whose partial
sums are all representable (multiples of a power of two, integers below 2^53) must give the exact
value bit for bit, whatever the order.  The terms are written by a device kernel launched just
before the sum, on the same stream and without a host synchronisation, so that a sum that read
them before that kernel completed would show."""
import math

import numpy as np
import pytest

pytestmark = pytest.mark.gpu

SIZES = [0, 1, 2, 7, 8, 9, 255, 256, 257, 2047, 2048, 2049, 8715, 24976, 132670, 1 << 20]


@pytest.mark.parametrize("n", SIZES)
def test_random_terms_within_the_fp64_bound_and_reproducible(grpo, n):
    import torch
    g = torch.Generator(device="cuda").manual_seed(n + 1)
    v = torch.randn(max(n, 1), generator=g, device="cuda", dtype=torch.float64)[:n] * 3.0 + 0.25
    out = grpo.grpo_sum_f64(v, n)
    again = grpo.grpo_sum_f64(v, n)
    h = v.cpu().numpy()
    exact = math.fsum(h.tolist())
    bound = max(n - 1, 0) * 2.0 ** -53 * float(np.abs(h).sum())
    got = float(out.item())
    assert abs(got - exact) <= bound, (n, got, exact, bound)
    assert out.view(torch.int64).item() == again.view(torch.int64).item()  # same bits


@pytest.mark.parametrize("n", SIZES)
def test_representable_partial_sums_are_exact(grpo, n):
    import torch
    # k * 2^-3 for k in [-1000, 1000]: every partial sum of at most 2^20 terms is a multiple of
    # 2^-3 below 2^31 in magnitude, so every fp64 addition is exact in any order
    idx = torch.arange(n, device="cuda", dtype=torch.int64)
    v = (((idx * 7919 + 13) % 2001) - 1000).to(torch.float64) * 0.125
    out = grpo.grpo_sum_f64(v, n).item()
    exact = float(sum(((i * 7919 + 13) % 2001 - 1000) for i in range(n))) * 0.125
    assert out == exact, (n, out, exact)


def test_a_prefix_of_the_terms(grpo):
    import torch
    v = torch.arange(1, 10001, device="cuda", dtype=torch.float64)
    for m in (0, 1, 99, 4096, 9999):
        assert grpo.grpo_sum_f64(v, m).item() == m * (m + 1) / 2
