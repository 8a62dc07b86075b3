"""Host-side parts of the C-ABI library, checked without a GPU: the library loads and exports
every function include/fastrl_grpo.h declares, argument errors come back as statuses before any
GPU work, workspace queries answer without a device, and the host adaptive rollout sampling
equals the oracle's."""
import ctypes
import os
import re

import numpy as np
import pytest

from helpers import golden
from test_oracle_ars import run_trace

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def declared_functions():
    text = open(os.path.join(ROOT, "include", "fastrl_grpo.h")).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b([a-z_][a-z0-9_]*)\s*\(", text)) - {"sizeof"})


def test_exports_every_declared_function(grpo):
    names = declared_functions()
    assert len(names) >= 10
    lib = ctypes.CDLL(grpo.library_path())
    for nm in names:
        assert hasattr(lib, nm), nm
    assert sorted(grpo.binding.EXPORTS) == names


def test_version_and_counter(grpo):
    assert "sm_103a" in grpo.version()
    assert grpo.grpo_kernel_launches() >= 0


def test_check_status_maps_device_bits(grpo):
    """grpo_check_status: 0 is OK, a timed-out wait is GRPO_ERR_TIMEOUT (it wins over data bits),
    data bits are GRPO_ERR_DEVICE_CHECK, and the message names every bit."""
    B = grpo.binding
    L = B.lib()
    assert L.grpo_check_status(0) == 0
    for word, rc, words in ((B.DEVFLAG_BAD_TOKEN, 6, [b"token id"]),
                            (B.DEVFLAG_NONFINITE, 6, [b"non-finite"]),
                            (B.DEVFLAG_TIMEOUT, 5, [b"timed out"]),
                            (B.DEVFLAG_TIMEOUT | B.DEVFLAG_BAD_TOKEN, 5, [b"timed out", b"token id"]),
                            (64, 6, [b"unknown"])):
        assert L.grpo_check_status(word) == rc
        msg = L.grpo_last_error()
        assert all(w in msg for w in words), msg
    with pytest.raises(grpo.GrpoError) as e:
        B.check_status(B.DEVFLAG_NONFINITE)
    assert e.value.status == 6
    assert B.check_status(0) == 0


def test_library_host_ars_matches_oracle(oracle_mod, grpo):
    """adaptive_rollout_count (host C++ in the library) equals the oracle step for step."""
    rng = np.random.default_rng(4)
    g = golden("ars_trace.json")
    st = grpo.grpo_ars_init(g["G1"])
    assert run_trace(lambda k, s, M, e: grpo.adaptive_rollout_count(st, k, s, M, e), g) == g["n_after_step"]
    for trial in range(100):
        G1 = int(rng.integers(2, 33))
        M = int(rng.integers(2, 80))
        spe = int(rng.integers(1, 10))
        P = int(rng.integers(1, 40))
        o = oracle_mod.Ars(G1)
        lib_st = grpo.grpo_ars_init(G1)
        n = G1
        for s in range(1, M + 1):
            kept = np.minimum(rng.integers(0, G1 + 1, size=P), n).astype(np.int32)
            end = (s % spe == 0)
            n_o = o.step(kept, s, M, end)
            n_l = grpo.adaptive_rollout_count(lib_st, kept, s, M, end)
            assert n_o == n_l, (trial, s)
            n = n_l


def test_library_host_ars_rejects_bad_args(grpo):
    st = grpo.grpo_ars_init(8)
    with pytest.raises(grpo.GrpoError):
        grpo.adaptive_rollout_count(st, [1, 2], 0, 10, False)
    with pytest.raises(grpo.GrpoError):
        grpo.adaptive_rollout_count(st, [1, 2], 11, 10, False)
    with pytest.raises(grpo.GrpoError):
        grpo.grpo_ars_init(1)


def raw():
    import paper_2609_36932_gb300 as g
    return g.lib()


def test_argument_errors_return_status_without_gpu_work(grpo):
    L = raw()
    assert L.grpo_advantage(None, 4, 0, 0, None, None, None) == 1
    assert L.grpo_advantage(None, 4, 4, 2, None, None, None) == 1
    assert L.grpo_advantage(None, 0, 4, 0, None, None, None) == 0  # P = 0 is a no-op
    size = ctypes.c_size_t(0)
    # G above 32, V above 2^18, n-gram order 4 are outside the supported limits
    assert L.grpo_prune(None, None, 0.0, None, None, 4, 33, 10, 100, 1, 0.8, 4, 1, None, None, None, None,
                        ctypes.byref(size), None) == 2
    assert L.grpo_prune(None, None, 0.0, None, None, 4, 8, 10, (1 << 18) + 1, 1, 0.8, 4, 1, None, None, None,
                        None, ctypes.byref(size), None) == 2
    assert L.grpo_prune(None, None, 0.0, None, None, 4, 8, 10, 100, 4, 0.8, 4, 1, None, None, None, None,
                        ctypes.byref(size), None) == 2
    assert L.grpo_prune(None, None, 0.0, None, None, 4, 8, 10, 100, 1, 0.8, 0, 1, None, None, None, None,
                        ctypes.byref(size), None) == 1
    assert L.grpo_compact(None, None, -1, None, None, None, None, None, None, None) == 1
    assert L.grpo_loss_tune(17, 0, 0) == 1 and L.grpo_loss_tune(0, 96, 0) == 1
    assert L.grpo_loss_tune(0, 0, 0) == 0
    assert b"cluster" in L.grpo_last_error() or L.grpo_last_error() == b""


def test_upload_kept_argument_errors(grpo):
    """grpo_upload_kept validates everything before its first copy; with nothing kept it
    enqueues nothing, so these calls need no device."""
    L = raw()
    keep = np.array([1, 0, 1, 1], np.uint8)
    off = np.array([0, 3, 5, 9, 12], np.int64)
    src, dst = ctypes.c_void_p(4096), ctypes.c_void_p(8192)  # never dereferenced here
    nb, nc = ctypes.c_int64(-1), ctypes.c_int32(-1)

    def call(k, o, n, row_bytes=64, s=src, d=dst):
        return L.grpo_upload_kept(s, d, row_bytes, k.ctypes.data if k is not None else None,
                                  o.ctypes.data if o is not None else None, n,
                                  ctypes.byref(nb), ctypes.byref(nc), None)

    assert call(keep, off, -1) == 1
    assert call(keep, off, 4, row_bytes=0) == 1
    assert call(None, off, 4) == 1 and call(keep, None, 4) == 1
    assert call(keep, off, 4, s=None) == 1 and call(keep, off, 4, d=None) == 1
    assert call(keep, np.array([0, 3, 2, 9, 12], np.int64), 4) == 1  # decreasing
    assert call(keep, np.array([-1, 3, 5, 9, 12], np.int64), 4) == 1
    assert call(keep, np.array([0, 3, 5, 9, 1 << 40], np.int64), 4, row_bytes=1 << 30) == 1
    assert b"overflow" in L.grpo_last_error()
    assert call(keep, off, 0) == 0 and (nb.value, nc.value) == (0, 0)
    assert call(np.zeros(4, np.uint8), off, 4) == 0 and (nb.value, nc.value) == (0, 0)


def gspo_call(L, n_rows, V, K, ws, size_p, n_seq=1, ldt=1, beta=0.0, eps=0.2, logp=4096):
    return L.grpo_gspo_loss_fwd_bwd(None, ldt, V, None, n_rows, V, None, None, None, None, None,
                                    None, K, n_seq, eps, eps, beta, None, 1,
                                    ctypes.c_void_p(logp) if logp else None, None, None, None,
                                    ws, size_p, None)


def test_gspo_workspace_query_and_argument_errors(grpo):
    L = raw()
    size = ctypes.c_size_t(0)
    def up(x):
        return (x + 255) // 256 * 256
    assert gspo_call(L, 1000, 152064, 16, None, ctypes.byref(size)) == 0
    assert size.value == up(1000 * 16) + up(1000 * 4) + up(16 * 8)  # stats, coef, seq terms
    assert gspo_call(L, 1000, 152064, 16, None, ctypes.byref(size), n_seq=0) == 1
    assert gspo_call(L, 1000, 152064, -1, None, ctypes.byref(size)) == 1
    assert gspo_call(L, -1, 152064, 16, None, ctypes.byref(size)) == 1
    assert gspo_call(L, 10, 0, 1, None, ctypes.byref(size)) == 1
    assert gspo_call(L, 10, 100, 1, None, ctypes.byref(size), ldt=5) == 1
    assert gspo_call(L, 10, 100, 1, None, ctypes.byref(size), beta=-1.0) == 1
    small = ctypes.c_size_t(8)
    assert gspo_call(L, 1000, 152064, 16, ctypes.c_void_p(4096), ctypes.byref(small)) == 3
    # a real call with NULL sequence arrays is refused before any launch
    big = ctypes.c_size_t(1 << 20)
    assert gspo_call(L, 1000, 152064, 16, ctypes.c_void_p(4096), ctypes.byref(big)) == 1
    # the device-count variant: counts are required; the size query matches the host variant's
    def dev_call(counts, size_p):
        return L.grpo_gspo_loss_fwd_bwd_dev(None, 1, 152064, None, 1000, 16, counts, 152064, None,
                                            None, None, None, None, None, 0, 0.2, 0.2, 0.0, None,
                                            1, ctypes.c_void_p(4096), None, None, None, None,
                                            size_p, None)
    assert dev_call(None, ctypes.byref(size)) == 1
    assert dev_call(ctypes.c_void_p(4096), ctypes.byref(size)) == 0
    assert size.value == up(1000 * 16) + up(1000 * 4) + up(16 * 8)


def loss_call(L, n_rows, V, ws, size_p, ldt=1, agg=0, denom=1, row_loss=None, beta=0.04):
    return L.grpo_loss_fwd_bwd(None, ldt, V, None, n_rows, V, None, None, None, None, None, 0.2,
                               0.2, beta, agg, denom, None, 0, None, 1, None, row_loss, None, None,
                               ws, size_p, None)


def test_workspace_queries_answer_without_a_device(grpo):
    L = raw()
    size = ctypes.c_size_t(0)
    assert L.grpo_prune(None, None, 0.0, None, None, 16, 8, 5000, 152064, 2, 0.8, 4, 1, None, None, None,
                        None, ctypes.byref(size), None) == 0
    def up(x):
        return (x + 255) // 256 * 256
    # bigrams: sorted keys (2T u64), set sizes, one byte per ordered pair
    assert size.value == up(2 * 5000 * 8) + 3 * up(16 * 8 * 4) + up(16 * 8 * 8)
    assert L.grpo_prune(None, None, 0.0, None, None, 16, 8, 5000, 152064, 1, 0.8, 4, 1, None, None, None,
                        None, ctypes.byref(size), None) == 0
    # unigrams: a vocabulary bitmap per rollout instead of keys
    assert size.value == up(16 * 8 * ((152064 + 63) // 64) * 8) + 3 * up(16 * 8 * 4) + up(16 * 8 * 8)
    assert loss_call(L, 1000, 152064, None, ctypes.byref(size)) == 0
    assert size.value == up(1000 * 8)
    # with a row-loss output the loss needs no workspace
    assert loss_call(L, 1000, 152064, None, ctypes.byref(size), row_loss=ctypes.c_void_p(256)) == 0
    assert size.value == 0
    # too small a workspace is refused before any launch
    small = ctypes.c_size_t(8)
    assert loss_call(L, 1000, 152064, ctypes.c_void_p(4096), ctypes.byref(small)) == 3


def test_loss_argument_errors(grpo):
    L = raw()
    size = ctypes.c_size_t(0)
    assert loss_call(L, 10, 100, None, ctypes.byref(size), ldt=7) == 1
    assert loss_call(L, -1, 100, None, ctypes.byref(size)) == 1
    assert loss_call(L, 10, 0, None, ctypes.byref(size)) == 1
    assert loss_call(L, 10, 100, None, ctypes.byref(size), denom=0) == 1
    assert loss_call(L, 10, 100, None, ctypes.byref(size), agg=1) == 1  # needs seq_off
    assert loss_call(L, 10, 100, None, ctypes.byref(size), beta=-1.0) == 1


def test_ars_closed_loop_of_the_large_group_workload(oracle_mod, grpo):
    """20 steps, G1 = 16, 5 steps per epoch, pruning ratios U(0.1, 0.6) per prompt: the library's
    host ARS and the oracle choose the same rollout count at every step."""
    from paper_2609_36932_gb300 import workloads
    w = workloads.get("large")
    steps, spe = 20, 5
    ratios = workloads.ars_pruning_ratios(0, steps, w.P)

    def loop(step_fn):
        n, seq = w.G, []
        for s in range(1, steps + 1):
            kept = workloads.synthetic_kept_counts(ratios[s - 1], n)
            n = step_fn(kept, s, s % spe == 0)
            seq.append(n)
        return seq

    o = oracle_mod.Ars(w.G)
    st = grpo.grpo_ars_init(w.G)
    seq_o = loop(lambda k, s, e: o.step(k, s, steps, e))
    seq_l = loop(lambda k, s, e: grpo.adaptive_rollout_count(st, k, s, steps, e))
    assert seq_o == seq_l
    assert all(2 <= n <= w.G for n in seq_o)


def lmhead_call(L, n_rows, V, D, ws, ws_bytes, *, stride=None, chunk=0, agg=0, denom=None,
                beta=0.04, dh_dtype=0, dl=None, ri=None):
    f = ctypes.c_float
    L.grpo_lmhead_loss_fwd_bwd.restype = ctypes.c_int32
    return L.grpo_lmhead_loss_fwd_bwd(
        None, ctypes.c_int64(D if stride is None else stride), ri, ctypes.c_int64(n_rows), None,
        ctypes.c_int32(V), ctypes.c_int32(D), None, None, None, None, None, f(0.2), f(0.2),
        f(beta), ctypes.c_int32(agg), ctypes.c_int64(max(n_rows, 1) if denom is None else denom),
        None, ctypes.c_int64(0), None, ctypes.c_int32(dh_dtype), None, ctypes.c_int32(0), dl, None,
        None, None, None, ctypes.c_int64(chunk), ws, ws_bytes, None)


def test_lmhead_workspace_query_and_argument_errors(grpo):
    L = raw()
    size = ctypes.c_size_t(0)
    assert lmhead_call(L, 1000, 152064, 3584, None, ctypes.byref(size)) == 0
    full = size.value
    # per row: a partial (max, sum) pair per 256-entry vocabulary tile (594), z_y, the row
    # scalars and the row loss; one chunk of f32 logits and one of bf16 dlogits (1000 rows round
    # up to 1024); and the f32 partial products of dhidden's split K: S copies of the chunk's
    # [rows, D] (1 <= S <= 8; 56 output tiles on 152 SMs split)
    def up(x):
        return (x + 255) // 256 * 256
    base = up(1000 * 594 * 8) + up(1000 * 4) + up(1000 * 16) + up(1000 * 8)
    gp = full - base - up(1024 * 152064 * 4) - up(1024 * 152064 * 2)
    unit = 1000 * 3584 * 4
    assert 2 * unit <= gp <= 8 * unit and gp % unit == 0
    assert lmhead_call(L, 1000, 152064, 3584, None, ctypes.byref(size), chunk=256) == 0
    gp = size.value - base - up(256 * 152064 * 4) - up(256 * 152064 * 2)
    assert 2 * 256 * 3584 * 4 <= gp <= 8 * 256 * 3584 * 4 and gp % (256 * 3584 * 4) == 0
    # recomputed logits: no chunk of f32 logits
    L.grpo_lmhead_tune.restype = ctypes.c_int32
    assert L.grpo_lmhead_tune(ctypes.c_int32(0), ctypes.c_int32(0), ctypes.c_int32(1)) == 0
    try:
        assert lmhead_call(L, 1000, 152064, 3584, None, ctypes.byref(size)) == 0
        assert size.value == full - up(1024 * 152064 * 4)
    finally:
        assert L.grpo_lmhead_tune(ctypes.c_int32(0), ctypes.c_int32(0), ctypes.c_int32(0)) == 0
    assert lmhead_call(L, 1000, 152064, 3584, None, ctypes.byref(size),
                       dl=ctypes.c_void_p(4096)) == 0
    assert size.value == full - up(1024 * 152064 * 2)
    # rows taken through row_index are gathered: D bf16 values and y, old, ref per row
    assert lmhead_call(L, 1000, 152064, 3584, None, ctypes.byref(size),
                       ri=ctypes.c_void_p(4096)) == 0
    assert size.value == full + up(1000 * 3584 * 2) + 3 * up(1000 * 4)
    assert lmhead_call(L, 10, 100, 12, None, ctypes.byref(size)) == 1      # D not a multiple of 8
    assert lmhead_call(L, 10, 100, 64, None, ctypes.byref(size), stride=60) == 1
    assert lmhead_call(L, 10, 0, 64, None, ctypes.byref(size)) == 1
    assert lmhead_call(L, -1, 100, 64, None, ctypes.byref(size)) == 1
    assert lmhead_call(L, 10, 100, 64, None, ctypes.byref(size), denom=0) == 1
    assert lmhead_call(L, 10, 100, 64, None, ctypes.byref(size), agg=1) == 1   # needs seq_off
    assert lmhead_call(L, 10, 100, 64, None, ctypes.byref(size), beta=-1.0) == 1
    assert lmhead_call(L, 10, 100, 64, None, ctypes.byref(size), dh_dtype=9) == 1
    # a real call with NULL buffers is refused before any launch
    big = ctypes.c_size_t(1 << 40)
    assert lmhead_call(L, 10, 100, 64, ctypes.c_void_p(4096), ctypes.byref(big)) == 1


def test_lmhead_tune_rejects_out_of_range_settings(grpo):
    L = raw()
    L.grpo_lmhead_tune.restype = ctypes.c_int32
    i32 = ctypes.c_int32
    assert L.grpo_lmhead_tune(i32(-1), i32(0), i32(0)) == 1
    assert L.grpo_lmhead_tune(i32(65), i32(0), i32(0)) == 1
    assert L.grpo_lmhead_tune(i32(0), i32(9), i32(0)) == 1
    assert L.grpo_lmhead_tune(i32(0), i32(0), i32(2)) == 1
    assert L.grpo_lmhead_tune(i32(0), i32(0), i32(-1)) == 1
    assert L.grpo_lmhead_tune(i32(0), i32(0), i32(1)) == 0
    assert L.grpo_lmhead_tune(i32(0), i32(0), i32(0)) == 0


def test_ars_checkpoint_resumes_the_rollout_counts(oracle_mod, grpo):
    """The ARS state saved mid-run (mid-epoch and at an epoch end) and restored into a fresh state
    continues with exactly the rollout counts of the uninterrupted run, which equal the oracle's."""
    import struct
    from paper_2609_36932_gb300 import workloads
    w = workloads.get("large")
    steps, spe = 20, 5
    ratios = workloads.ars_pruning_ratios(1, steps, w.P)

    def run(st, first, last, n):
        seq = []
        for s in range(first, last + 1):
            kept = workloads.synthetic_kept_counts(ratios[s - 1], n)
            n = grpo.adaptive_rollout_count(st, kept, s, steps, s % spe == 0)
            seq.append(n)
        return seq, n

    full, _ = run(grpo.grpo_ars_init(w.G), 1, steps, w.G)
    o = oracle_mod.Ars(w.G)
    n, seq_o = w.G, []
    for s in range(1, steps + 1):
        n = o.step(workloads.synthetic_kept_counts(ratios[s - 1], n), s, steps, s % spe == 0)
        seq_o.append(n)
    assert full == seq_o
    for cut in (3, 5, 7, 12):
        st = grpo.grpo_ars_init(w.G)
        head, n = run(st, 1, cut, w.G)
        rec = grpo.grpo_ars_serialize(st)
        assert len(rec) == 64 and rec[:8] == b"FRLARS01"
        assert struct.unpack_from("<iiii", rec, 8) == (st.G1, st.n, st.have_ref, st.have_gt)
        assert struct.unpack_from("<ddddq", rec, 24) == (st.g_ref, st.g_t, st.buf_mean_sum,
                                                         st.buf_max_sum, st.buf_count)
        back = grpo.grpo_ars_deserialize(rec)
        assert grpo.grpo_ars_serialize(back) == rec
        tail, _ = run(back, cut + 1, steps, n)
        assert head + tail == full, cut


def test_ars_checkpoint_rejects_bad_records(grpo):
    import struct
    st = grpo.grpo_ars_init(8)
    good = bytearray(grpo.grpo_ars_serialize(st))

    def bad(rec):
        with pytest.raises(grpo.GrpoError):
            grpo.grpo_ars_deserialize(bytes(rec))

    bad(good[:63])
    r = bytearray(good); r[0:8] = b"FRLARS02"; bad(r)
    r = bytearray(good); struct.pack_into("<i", r, 12, 9); bad(r)          # n > G1
    r = bytearray(good); struct.pack_into("<i", r, 8, 1); bad(r)           # G1 < 2
    r = bytearray(good); struct.pack_into("<i", r, 16, 2); bad(r)          # have_ref not 0/1
    r = bytearray(good); struct.pack_into("<d", r, 24, float("nan")); bad(r)
    r = bytearray(good); struct.pack_into("<q", r, 56, -1); bad(r)
    assert grpo.grpo_ars_deserialize(bytes(good)).G1 == 8


def test_fail_launch_hook_rejects_negative_counts(grpo):
    L = raw()
    L.grpo_test_fail_launch.restype = ctypes.c_int32
    assert L.grpo_test_fail_launch(ctypes.c_int32(-1)) == 1
    assert L.grpo_test_fail_launch(ctypes.c_int32(0)) == 0


def test_lmhead_grad_workspace_query_and_argument_errors(grpo):
    """grpo_lmhead_grad answers its size query and rejects bad arguments without a device; a
    query on a qwen-sized chunk (14122 rows, V = 152064, D = 3584) asks for the split partials
    of dhidden's product (its 784 output tiles would leave most of a seventh wave idle)."""
    L = grpo.binding.lib()
    size = ctypes.c_size_t(0)
    out = ctypes.c_void_p(256)  # never dereferenced by a size query

    def call(n, V, D, dstride, hstride, dtype=1, dh=out, dw=out):
        return L.grpo_lmhead_grad(None, dstride, n, V, None, hstride, None, D, dh, dtype, dw, 0,
                                  None, None, ctypes.byref(size), None)

    assert call(14122, 152064, 3584, 152064, 3584) == 0
    assert size.value >= 2 * 14122 * 3584 * 4 and size.value % 256 == 0
    assert call(14122, 152064, 3584, 152064, 3584, dh=None) == 0  # dweight alone: no split
    assert size.value == 0
    assert call(0, 100, 64, 104, 64) == 0 and size.value == 0
    assert call(10, 100, 12, 104, 16) == 1                  # D not a multiple of 8
    assert call(10, 100, 64, 100, 64) == 1                  # dlogits stride not a multiple of 8
    assert call(10, 100, 64, 96, 64) == 1                   # dlogits stride < V
    assert call(10, 100, 64, 104, 60) == 1                  # hidden stride < D
    assert call(10, 100, 64, 104, 64, dtype=7) == 1         # dhidden dtype
    assert b"grpo_lmhead_grad" in L.grpo_last_error()



def test_normal_build_has_no_index_check_report(grpo):
    """grpo_debug_checks answers GRPO_ERR_UNSUPPORTED in the normal build, without touching a
    device, and names the checked build in its message."""
    if grpo.checked_build():
        pytest.skip("the checked build reports")
    L = raw()
    mask, site = ctypes.c_int32(7), ctypes.c_int32(7)
    L.grpo_debug_checks.restype = ctypes.c_int32
    assert L.grpo_debug_checks(ctypes.c_int32(1), ctypes.byref(mask), ctypes.byref(site)) == 2
    assert mask.value == 0 and site.value == 0
    assert "checked build" in grpo.grpo_last_error()
    L.grpo_version.restype = ctypes.c_char_p
    assert b"checked" not in L.grpo_version()
