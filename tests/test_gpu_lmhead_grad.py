"""GPU parity of grpo_lmhead_grad (the chain rule through the output layer z = h W^T for given
dlogits: dhidden = dlogits W, dweight = dlogits^T h, Sec. 3.2 with Eqs. 1-3) with the oracle,
through the C ABI.  These are the two products grpo_lmhead_loss_fwd_bwd runs after its dlogits
pass, on the library's own tcgen05 kernel.

Tolerances follow from the arithmetic (u = 2^-23, twice IEEE's f32 unit roundoff, per addition of
the tensor cores' f32 accumulation; bf16 x bf16 products are exact in f32):
  dhidden  |err[t, d]| <= V * u * sum_v |dl[t, v]| |W[v, d]|   (+ 2^-8 |dh| when dhidden is bf16)
  dweight  |err[v, d]| <= T * u * sum_t |dl[t, v]| |h[t, d]|
A split K adds its S partial sums in f32 as well: S <= 8 additions, inside the same bound.  A
wrong tile, k-block, swizzle or operand layout moves results by the size of those sums."""
import numpy as np
import pytest

pytestmark = pytest.mark.gpu

U = 2.0 ** -23


def bf16(x):
    import torch
    return torch.from_numpy(np.ascontiguousarray(x, np.float32)).to(torch.bfloat16)


class GradCase:
    def __init__(self, seed, T, V, D, dl_pad=0, h_pad=0, scale=1e-3):
        rng = np.random.default_rng(seed)
        self.T, self.V, self.D = T, V, D
        self.dl_t = bf16(rng.standard_normal((T, V)) * scale)
        self.h_t = bf16(rng.standard_normal((T, D)))
        self.w_t = bf16(rng.standard_normal((V, D)) / np.sqrt(D))
        self.dl = self.dl_t.float().double().numpy()
        self.h = self.h_t.float().double().numpy()
        self.w = self.w_t.float().double().numpy()
        self.dl_pad, self.h_pad = dl_pad, h_pad

    def device_inputs(self):
        """dlogits and hidden inside wider rows (the padding is NaN: it must never be read).
        dlogits rows are padded to a multiple of 8 elements, as the call requires."""
        import torch
        width = self.V + (-self.V) % 8 + self.dl_pad
        dl = torch.full((self.T, width), float("nan"), dtype=torch.bfloat16)
        dl[:, :self.V] = self.dl_t
        h = torch.full((self.T, self.D + self.h_pad), float("nan"), dtype=torch.bfloat16)
        h[:, :self.D] = self.h_t
        return dl.cuda()[:, :self.V], h.cuda()[:, :self.D], self.w_t.cuda()

    def oracle(self, oracle_mod):
        return oracle_mod.lmhead_grad(self.dl, self.h, self.w, want_bounds=True)


def check(case, o, dh, dw, dh_bf16, base_dw=None):
    if dh is not None:
        tol = case.V * U * o["dhidden_abs"] + (2.0 ** -8 * np.abs(o["dhidden"]) if dh_bf16 else 0)
        e = np.abs(dh.astype(np.float64) - o["dhidden"])
        assert np.all(e <= tol + 1e-30), "dhidden: worst err %g at bound %g" % (
            e.max(), tol.flat[e.argmax()])
    if dw is not None:
        ref = o["dweight"] + (0 if base_dw is None else base_dw)
        tol = case.T * U * o["dweight_abs"] + (0 if base_dw is None else 2 * U * np.abs(ref))
        e = np.abs(dw.astype(np.float64) - ref)
        assert np.all(e <= tol + 1e-30), "dweight: worst err %g at bound %g" % (
            e.max(), tol.flat[e.argmax()])


def run(grpo, case, **kw):
    import torch
    dl, h, w = case.device_inputs()
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    out = grpo.grpo_lmhead_grad(dl, h, w, status=status, **kw)
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    dh = out["dhidden"].float().cpu().numpy()[:case.T] if out["dhidden"] is not None else None
    dw = out["dweight"].cpu().numpy() if out["dweight"] is not None else None
    return dh, dw


# (T, V, D): one row and one word; ragged row blocks, vocabularies and hidden sizes; D not a
# multiple of 64; a product whose K is split (few output tiles, long K); and one with many tiles.
SHAPES = [(1, 1, 8), (5, 300, 24), (257, 1000, 200), (300, 4097, 72), (600, 40000, 264),
          (130, 70001, 136), (1000, 2048, 520)]


@pytest.mark.parametrize("T,V,D", SHAPES)
@pytest.mark.parametrize("dh_dtype", ["bf16", "f32"])
def test_parity_ragged_shapes(grpo, oracle_mod, T, V, D, dh_dtype):
    case = GradCase(T * 7 + V + D, T, V, D)
    o = case.oracle(oracle_mod)
    dh, dw = run(grpo, case, dhidden_dtype=dh_dtype)
    check(case, o, dh, dw, dh_dtype == "bf16")


def test_padded_strides_and_determinism(grpo, oracle_mod):
    """dlogits and hidden inside wider rows whose padding is NaN (never read); two calls give the
    same bits."""
    case = GradCase(5, 333, 5000, 96, dl_pad=40, h_pad=24)
    o = case.oracle(oracle_mod)
    dh, dw = run(grpo, case, dhidden_dtype="f32")
    check(case, o, dh, dw, False)
    dh2, dw2 = run(grpo, case, dhidden_dtype="f32")
    assert np.array_equal(dh, dh2) and np.array_equal(dw, dw2)


def test_accumulate_and_single_outputs(grpo, oracle_mod):
    """dweight added to an existing buffer; either product alone."""
    import torch
    case = GradCase(6, 200, 3000, 64)
    o = case.oracle(oracle_mod)
    base = np.random.default_rng(1).standard_normal((case.V, case.D)).astype(np.float32)
    dl, h, w = case.device_inputs()
    dwt = torch.from_numpy(base.copy()).cuda()
    out = grpo.grpo_lmhead_grad(dl, h, w, dweight=dwt, accumulate_dweight=True, want_dhidden=False)
    torch.cuda.synchronize()
    assert out["dhidden"] is None
    check(case, o, None, dwt.cpu().numpy(), False, base_dw=base.astype(np.float64))
    out = grpo.grpo_lmhead_grad(dl, h, w, want_dweight=False, dhidden_dtype="f32")
    torch.cuda.synchronize()
    assert out["dweight"] is None
    check(case, o, out["dhidden"].cpu().numpy(), None, False)


def test_unaligned_bf16_dhidden(grpo, oracle_mod):
    """A dhidden buffer two bytes past an 8-byte boundary takes the element-wise store path."""
    import torch
    case = GradCase(7, 70, 900, 40)
    o = case.oracle(oracle_mod)
    dl, h, w = case.device_inputs()
    flat = torch.zeros(case.T * case.D + 8, dtype=torch.bfloat16, device="cuda")
    dh = flat[1:1 + case.T * case.D].view(case.T, case.D)
    grpo.grpo_lmhead_grad(dl, h, w, dhidden=dh, want_dweight=False)
    torch.cuda.synchronize()
    check(case, o, dh.float().cpu().numpy(), None, True)
    assert float(flat[0]) == 0.0 and float(flat[1 + case.T * case.D]) == 0.0


def test_zero_rows(grpo):
    import torch
    w = torch.ones((16, 16), dtype=torch.bfloat16, device="cuda")
    dl = torch.empty((0, 16), dtype=torch.bfloat16, device="cuda")
    h = torch.empty((0, 16), dtype=torch.bfloat16, device="cuda")
    dw = torch.full((16, 16), 3.0, device="cuda")
    grpo.grpo_lmhead_grad(dl, h, w, dweight=dw, want_dhidden=False)
    torch.cuda.synchronize()
    assert float(dw.abs().max()) == 0.0
