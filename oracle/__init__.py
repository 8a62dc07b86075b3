"""CPU oracle for the FastRL kept-token GRPO path — TEST INFRASTRUCTURE ONLY.

A plain fp64 restatement of the paper's definitions (Eqs. 1-14, Algorithm 1) in C++
(oracle/*.cpp), loaded through ctypes with numpy arrays.  Only the tests, the smoke check and the
benchmark's CPU-baseline leg may import this package.  It shares no code with the CUDA library
and never imports it.
"""
from __future__ import annotations

import ctypes
import math

import numpy as np

from .build import build_oracle

_lib = None

_c_p = ctypes.c_void_p
_i32 = ctypes.c_int32
_i64 = ctypes.c_int64
_f32 = ctypes.c_float
_f64 = ctypes.c_double


def lib():
    """Load (building if needed) liboracle.so."""
    global _lib
    if _lib is None:
        L = ctypes.CDLL(build_oracle())
        L.oracle_advantage.argtypes = [_c_p, _i32, _i32, _i32, _c_p, _c_p]
        L.oracle_advantage.restype = _i32
        L.oracle_prune.argtypes = [_c_p, _c_p, _c_p, _i32, _i32, _i32, _f32, _i32, _i32, _c_p, _c_p]
        L.oracle_prune.restype = _i32
        L.oracle_prune_classes.argtypes = [_c_p, _c_p, _f32, _c_p, _c_p, _i32, _i32, _i32, _f32,
                                           _i32, _i32, _c_p, _c_p]
        L.oracle_prune_classes.restype = _i32
        L.oracle_jaccard_distance.argtypes = [_c_p, _c_p, _i32, _i32, _i32]
        L.oracle_jaccard_distance.restype = _f64
        L.oracle_compact.argtypes = [_c_p, _c_p, _i32, _c_p, _c_p, _c_p, _c_p, _c_p]
        L.oracle_compact.restype = _i32
        L.oracle_loss.argtypes = [_c_p, _i32, _i64, _c_p, _i64, _i32, _c_p, _c_p, _c_p, _c_p, _c_p,
                                  _f32, _f32, _f32, _i32, _i64, _c_p, _i64, _c_p, _i32, _c_p,
                                  _c_p, _c_p, _c_p, _c_p, _c_p]
        L.oracle_loss.restype = _i32
        L.oracle_gspo_loss.argtypes = [_c_p, _i32, _i64, _c_p, _i32, _c_p, _c_p, _c_p, _c_p,
                                       _c_p, _c_p, _i64, _i64, _f32, _f32, _f32, _c_p, _i32,
                                       _c_p, _c_p, _c_p, _c_p, _c_p, _c_p]
        L.oracle_gspo_loss.restype = _i32
        L.oracle_lmhead_loss.argtypes = [_c_p, _c_p, _i64, _i32, _i32, _c_p, _c_p, _c_p, _c_p,
                                         _c_p, _f32, _f32, _f32, _i32, _i64, _c_p, _i64, _c_p,
                                         _c_p, _c_p, _c_p, _c_p, _c_p, _c_p, _c_p, _c_p]
        L.oracle_lmhead_loss.restype = _i32
        L.oracle_lmhead_gspo_loss.argtypes = [_c_p, _c_p, _i64, _i32, _i32, _c_p, _c_p, _c_p,
                                              _c_p, _c_p, _c_p, _i64, _i64, _f32, _f32, _f32,
                                              _c_p, _c_p, _c_p, _c_p, _c_p, _c_p, _c_p, _c_p, _c_p]
        L.oracle_lmhead_gspo_loss.restype = _i32
        L.oracle_lmhead_grad.argtypes = [_c_p, _c_p, _c_p, _i64, _i32, _i32, _c_p, _c_p, _c_p,
                                         _c_p]
        L.oracle_lmhead_grad.restype = _i32
        L.oracle_logp.argtypes = [_c_p, _i32, _i64, _c_p, _i64, _i32, _c_p, _c_p]
        L.oracle_logp.restype = _i32
        L.oracle_round_bf16.argtypes = [_f64]
        L.oracle_round_bf16.restype = ctypes.c_uint16
        L.oracle_ars_new.argtypes = [_i32]
        L.oracle_ars_new.restype = _c_p
        L.oracle_ars_free.argtypes = [_c_p]
        L.oracle_ars_free.restype = None
        L.oracle_ars_step.argtypes = [_c_p, _c_p, _i32, _i64, _i64, _i32]
        L.oracle_ars_step.restype = _i32
        L.oracle_ars_get.argtypes = [_c_p, _i32]
        L.oracle_ars_get.restype = _f64
        L.oracle_set_threads.argtypes = [_i32]
        L.oracle_set_threads.restype = _i32
        _lib = L
    return _lib


def _p(a):
    return None if a is None else a.ctypes.data_as(_c_p)


def _arr(a, dtype):
    return np.ascontiguousarray(np.asarray(a), dtype=dtype)


def set_threads(n: int = 0) -> int:
    """Set the loss's OpenMP thread count (0 = keep); return the count in effect."""
    return int(lib().oracle_set_threads(int(n)))


def advantage(rewards, G: int, std_mode: int = 0):
    """Eq. 5.  Returns (adv f32 [P*G], key f64 [P*G] = |r - mean|)."""
    r = _arr(rewards, np.float32)
    P = r.size // G
    adv = np.empty(P * G, np.float32)
    key = np.empty(P * G, np.float64)
    if lib().oracle_advantage(_p(r), P, G, std_mode, _p(adv), _p(key)) != 0:
        raise ValueError("oracle_advantage: bad arguments")
    return adv, key


def prune(rewards, ids, off, G: int, ngram_n: int = 1, tau: float = 0.8, keep_cap=None,
          dp_divisor: int = 1, adv=None, class_eps: float = 0.0):
    """Eqs. 6-9 + Algorithm 1.  Returns (keep u8 [P*G], kept_per_prompt i32 [P]).
    class_eps > 0 (with adv) groups by chained advantages (the continuous-reward extension)."""
    r = _arr(rewards, np.float32)
    P = r.size // G
    ids_ = _arr(ids, np.int32)
    off_ = _arr(off, np.int64)
    keep = np.zeros(P * G, np.uint8)
    kpp = np.zeros(max(P, 1), np.int32)
    cap = G if keep_cap is None else int(keep_cap)
    a = None if adv is None else _arr(adv, np.float32)
    if class_eps > 0 or a is not None:
        rc = lib().oracle_prune_classes(_p(r), _p(a), float(class_eps), _p(ids_), _p(off_), P, G,
                                        ngram_n, float(tau), cap, dp_divisor, _p(keep), _p(kpp))
    else:
        rc = lib().oracle_prune(_p(r), _p(ids_), _p(off_), P, G, ngram_n, float(tau), cap,
                                dp_divisor, _p(keep), _p(kpp))
    if rc != 0:
        raise ValueError("oracle_prune: bad arguments")
    return keep, kpp[:P]


def jaccard_distance(ids, off, i: int, j: int, ngram_n: int = 1) -> float:
    """Eq. 7 for rollouts i and j."""
    ids_ = _arr(ids, np.int32)
    off_ = _arr(off, np.int64)
    return float(lib().oracle_jaccard_distance(_p(ids_), _p(off_), i, j, ngram_n))


def compact(keep, off):
    """Token compaction.  Returns dict(kept_idx, kept_off, src_token, token_rollout, K, T_kept)."""
    k = _arr(keep, np.uint8)
    off_ = _arr(off, np.int64)
    n = k.size
    T = int(off_[n]) if n else 0
    kept_idx = np.zeros(max(n, 1), np.int32)
    kept_off = np.zeros(n + 1, np.int64)
    src = np.zeros(max(T, 1), np.int64)
    tr = np.zeros(max(T, 1), np.int32)
    counts = np.zeros(2, np.int64)
    lib().oracle_compact(_p(k), _p(off_), n, _p(kept_idx), _p(kept_off), _p(src), _p(tr),
                         _p(counts))
    K, TK = int(counts[0]), int(counts[1])
    return dict(kept_idx=kept_idx[:K], kept_off=kept_off[:K + 1], src_token=src[:TK],
                token_rollout=tr[:TK], K=K, T_kept=TK)


def loss(logits, V: int, y, old_logp, ref_logp, adv, row_rollout, *, eps_low=0.2, eps_high=0.2,
         beta=0.04, agg_mode=0, denom_tokens=None, seq_off=None, n_seq=0, row_index=None,
         n_rows=None, row_stride=None, logits_dtype=None, dlogits_dtype=0, want_f64=False,
         want_dlogits=True):
    """Eqs. 1-3.  `logits` is a float32 array or a uint16 array of bf16 bit patterns (or, with
    logits_dtype=2, float64).

    Returns dict(loss, logp [n_rows] f64, rho, row_loss, g (each row's gradient factor g_t, so
    that dlogits[t] = w_t * g_t * (onehot(y) - softmax)), w (the weights w_t), dlogits (f32 array
    or uint16 bf16 bits, [n_rows, V]) and, with want_f64, dlogits_f64).
    """
    lg = np.ascontiguousarray(logits)
    if logits_dtype is None:
        logits_dtype = 1 if lg.dtype == np.uint16 else 0
    if logits_dtype == 0:
        lg = lg.astype(np.float32, copy=False)
    elif logits_dtype == 2:
        lg = lg.astype(np.float64, copy=False)
    stride = V if row_stride is None else int(row_stride)
    ri = None if row_index is None else _arr(row_index, np.int64)
    if n_rows is None:
        n_rows = ri.size if ri is not None else lg.size // stride
    y_ = _arr(y, np.int32)
    old = _arr(old_logp, np.float32)
    ref = _arr(ref_logp, np.float32)
    a = _arr(adv, np.float32)
    rr = _arr(row_rollout, np.int32)
    so = None if seq_off is None else _arr(seq_off, np.int64)
    if denom_tokens is None:
        denom_tokens = n_rows
    out_np = np.float32 if dlogits_dtype == 0 else np.uint16
    dl = np.empty((n_rows, V), out_np) if want_dlogits else None
    d64 = np.empty((n_rows, V), np.float64) if want_f64 else None
    logp = np.empty(max(n_rows, 1), np.float64)
    rho = np.empty(max(n_rows, 1), np.float64)
    rl = np.empty(max(n_rows, 1), np.float64)
    g = np.empty(max(n_rows, 1), np.float64)
    total = np.zeros(1, np.float64)
    rc = lib().oracle_loss(_p(lg), logits_dtype, stride, _p(ri), n_rows, V, _p(y_), _p(old), _p(ref),
                           _p(a), _p(rr), float(eps_low), float(eps_high), float(beta), agg_mode,
                           int(denom_tokens), _p(so), int(n_seq), _p(dl), dlogits_dtype, _p(d64),
                           _p(logp), _p(rho), _p(rl), _p(total), _p(g))
    if rc != 0:
        raise ValueError("oracle_loss: bad arguments")
    # each row's aggregation weight w_t (1/denom_tokens, or 1/(n_seq |o_i|) per sequence)
    if agg_mode == 0:
        w = np.full(n_rows, 1.0 / float(denom_tokens))
    else:
        lens = (so[1:] - so[:-1]).astype(np.float64)
        w = 1.0 / (float(n_seq) * lens[rr[:n_rows]]) if n_rows else np.zeros(0)
    return dict(loss=float(total[0]), logp=logp[:n_rows], rho=rho[:n_rows], row_loss=rl[:n_rows],
                g=g[:n_rows], w=w, dlogits=dl, dlogits_f64=d64)


def lmhead_loss(hidden, weight, y, old_logp, ref_logp, adv, row_rollout, *, eps_low=0.2,
                eps_high=0.2, beta=0.04, agg_mode=0, denom_tokens=None, seq_off=None, n_seq=0,
                want_logits=False, want_dlogits=False, want_dhidden=True, want_dweight=True,
                want_bounds=False):
    """The output layer z = hidden @ weight.T fused with Eqs. 1-3, and the chain rule.

    hidden [n_rows, D] and weight [V, D] are taken as float64 (bf16 values widen exactly).
    Returns dict(loss, logp, row_loss, and as asked: logits, dlogits (f64), dhidden [n_rows, D],
    dweight [V, D], dhidden_abs, dweight_abs).
    """
    h = np.ascontiguousarray(hidden, dtype=np.float64)
    w = np.ascontiguousarray(weight, dtype=np.float64)
    n_rows, D = h.shape
    V = w.shape[0]
    if w.shape[1] != D:
        raise ValueError("hidden and weight disagree on D")
    y_ = _arr(y, np.int32)
    old = _arr(old_logp, np.float32)
    ref = _arr(ref_logp, np.float32)
    a = _arr(adv, np.float32)
    rr = _arr(row_rollout, np.int32)
    so = None if seq_off is None else _arr(seq_off, np.int64)
    if denom_tokens is None:
        denom_tokens = n_rows

    def buf(want, shape):
        return np.empty(shape, np.float64) if want else None

    lg = buf(want_logits, (n_rows, V))
    dl = buf(want_dlogits, (n_rows, V))
    dh = buf(want_dhidden, (n_rows, D))
    dw = buf(want_dweight, (V, D))
    dha = buf(want_bounds and want_dhidden, (n_rows, D))
    dwa = buf(want_bounds and want_dweight, (V, D))
    logp = np.empty(max(n_rows, 1), np.float64)
    rl = np.empty(max(n_rows, 1), np.float64)
    total = np.zeros(1, np.float64)
    rc = lib().oracle_lmhead_loss(_p(h), _p(w), n_rows, V, D, _p(y_), _p(old), _p(ref), _p(a),
                                  _p(rr), float(eps_low), float(eps_high), float(beta), agg_mode,
                                  int(denom_tokens), _p(so), int(n_seq), _p(lg), _p(dl), _p(logp),
                                  _p(rl), _p(total), _p(dh), _p(dw), _p(dha), _p(dwa))
    if rc != 0:
        raise ValueError("oracle_lmhead_loss: bad arguments")
    return dict(loss=float(total[0]), logp=logp[:n_rows], row_loss=rl[:n_rows], logits=lg,
                dlogits=dl, dhidden=dh, dweight=dw, dhidden_abs=dha, dweight_abs=dwa)


def lmhead_grad(dlogits, hidden, weight, want_bounds=False):
    """The chain rule through z = hidden @ weight.T for given dlogits [n_rows, V]: returns
    dict(dhidden = dlogits @ weight, dweight = dlogits.T @ hidden and, with want_bounds, the sums
    of absolute products dhidden_abs and dweight_abs), all fp64 (bf16 inputs widen exactly)."""
    dl = np.ascontiguousarray(dlogits, dtype=np.float64)
    h = np.ascontiguousarray(hidden, dtype=np.float64)
    w = np.ascontiguousarray(weight, dtype=np.float64)
    n_rows, V = dl.shape
    D = w.shape[1]
    if w.shape[0] != V or h.shape != (n_rows, D):
        raise ValueError("dlogits, hidden and weight disagree on their sizes")
    dh = np.empty((n_rows, D), np.float64)
    dw = np.empty((V, D), np.float64)
    dha = np.empty((n_rows, D), np.float64) if want_bounds else None
    dwa = np.empty((V, D), np.float64) if want_bounds else None
    if lib().oracle_lmhead_grad(_p(h), _p(w), _p(dl), n_rows, V, D, _p(dh), _p(dw), _p(dha),
                                _p(dwa)) != 0:
        raise ValueError("oracle_lmhead_grad: bad arguments")
    return dict(dhidden=dh, dweight=dw, dhidden_abs=dha, dweight_abs=dwa)


def lmhead_gspo_loss(hidden, weight, y, old_logp, ref_logp, adv, seq_rollout, seq_row_off, *,
                     n_seq=None, eps_low=0.2, eps_high=0.2, beta=0.0, want_dlogits=False,
                     want_dhidden=True, want_dweight=True, want_bounds=False):
    """The output layer fused with GSPO's sequence-level loss: gspo_loss on z = hidden @ weight.T
    (sequence k owns rows [seq_row_off[k], seq_row_off[k+1])), then the chain rule.  Returns
    dict(loss, logp, seq_ratio, seq_loss, and as asked dlogits, dhidden, dweight, *_abs)."""
    h = np.ascontiguousarray(hidden, dtype=np.float64)
    w = np.ascontiguousarray(weight, dtype=np.float64)
    n_rows, D = h.shape
    V = w.shape[0]
    so = _arr(seq_row_off, np.int64)
    K = so.size - 1
    if n_seq is None:
        n_seq = K

    def buf(want, shape):
        return np.empty(shape, np.float64) if want else None

    dl = buf(want_dlogits, (n_rows, V))
    dh = buf(want_dhidden, (n_rows, D))
    dw = buf(want_dweight, (V, D))
    dha = buf(want_bounds and want_dhidden, (n_rows, D))
    dwa = buf(want_bounds and want_dweight, (V, D))
    lp = np.empty(max(n_rows, 1), np.float64)
    sr = np.empty(max(K, 1), np.float64)
    sl = np.empty(max(K, 1), np.float64)
    total = np.zeros(1, np.float64)
    rc = lib().oracle_lmhead_gspo_loss(
        _p(h), _p(w), n_rows, V, D, _p(_arr(y, np.int32)), _p(_arr(old_logp, np.float32)),
        _p(_arr(ref_logp, np.float32)), _p(_arr(adv, np.float32)),
        _p(_arr(seq_rollout, np.int32)), _p(so), K, int(n_seq), float(eps_low), float(eps_high),
        float(beta), _p(dl), _p(lp), _p(sr), _p(sl), _p(total), _p(dh), _p(dw), _p(dha), _p(dwa))
    if rc != 0:
        raise ValueError("oracle_lmhead_gspo_loss: bad arguments")
    return dict(loss=float(total[0]), logp=lp[:n_rows], seq_ratio=sr[:K], seq_loss=sl[:K],
                dlogits=dl, dhidden=dh, dweight=dw, dhidden_abs=dha, dweight_abs=dwa)


def gspo_loss(logits, V: int, y, old_logp, ref_logp, adv, seq_rollout, seq_row_off, *,
              n_seq=None, eps_low=0.2, eps_high=0.2, beta=0.0, row_index=None, row_stride=None,
              logits_dtype=None, dlogits_dtype=0, want_f64=False, want_dlogits=True):
    """GSPO's sequence-level loss over kept rollouts (see loss.cpp).  Sequence k owns rows
    [seq_row_off[k], seq_row_off[k+1]) and rollout seq_rollout[k].  n_seq defaults to the number
    of sequences.  Returns dict(loss, logp [rows], seq_ratio [seqs], seq_loss [seqs], g (each
    row's gradient factor, dlogits[t] = g_t / (n_seq L_k) (onehot(y) - softmax); NaN in a sequence
    without a ratio), dlogits, dlogits_f64)."""
    lg = np.ascontiguousarray(logits)
    if logits_dtype is None:
        logits_dtype = 1 if lg.dtype == np.uint16 else 0
    if logits_dtype == 0:
        lg = lg.astype(np.float32, copy=False)
    elif logits_dtype == 2:
        lg = lg.astype(np.float64, copy=False)
    stride = V if row_stride is None else int(row_stride)
    ri = None if row_index is None else _arr(row_index, np.int64)
    so = _arr(seq_row_off, np.int64)
    K = so.size - 1
    n_rows = int(so[-1])
    if n_seq is None:
        n_seq = K
    out_np = np.float32 if dlogits_dtype == 0 else np.uint16
    dl = np.empty((n_rows, V), out_np) if want_dlogits else None
    d64 = np.empty((n_rows, V), np.float64) if want_f64 else None
    lp = np.empty(max(n_rows, 1), np.float64)
    sr = np.empty(max(K, 1), np.float64)
    sl = np.empty(max(K, 1), np.float64)
    g = np.empty(max(n_rows, 1), np.float64)
    total = np.zeros(1, np.float64)
    rc = lib().oracle_gspo_loss(_p(lg), logits_dtype, stride, _p(ri), V, _p(_arr(y, np.int32)),
                                _p(_arr(old_logp, np.float32)), _p(_arr(ref_logp, np.float32)),
                                _p(_arr(adv, np.float32)), _p(_arr(seq_rollout, np.int32)),
                                _p(so), K, int(n_seq), float(eps_low), float(eps_high),
                                float(beta), _p(dl), dlogits_dtype, _p(d64), _p(lp), _p(sr),
                                _p(sl), _p(total), _p(g))
    if rc != 0:
        raise ValueError("oracle_gspo_loss: bad arguments")
    return dict(loss=float(total[0]), logp=lp[:n_rows], seq_ratio=sr[:K], seq_loss=sl[:K],
                g=g[:n_rows], dlogits=dl, dlogits_f64=d64)


def logp(logits, V: int, y, *, row_index=None, n_rows=None, row_stride=None, logits_dtype=None):
    """log pi(y) per row: the old/reference policy evaluation.  Returns f64 [n_rows]."""
    lg = np.ascontiguousarray(logits)
    if logits_dtype is None:
        logits_dtype = 1 if lg.dtype == np.uint16 else 0
    if logits_dtype == 0:
        lg = lg.astype(np.float32, copy=False)
    stride = V if row_stride is None else int(row_stride)
    ri = None if row_index is None else _arr(row_index, np.int64)
    if n_rows is None:
        n_rows = ri.size if ri is not None else lg.size // stride
    y_ = _arr(y, np.int32)
    out = np.empty(max(n_rows, 1), np.float64)
    if lib().oracle_logp(_p(lg), logits_dtype, stride, _p(ri), n_rows, V, _p(y_), _p(out)) != 0:
        raise ValueError("oracle_logp: bad arguments")
    return out[:n_rows]


def round_bf16(x) -> np.ndarray:
    """fp64 -> bf16 bits, nearest-even, one rounding."""
    L = lib()
    flat = np.asarray(x, np.float64).ravel()
    return np.array([L.oracle_round_bf16(float(v)) for v in flat], np.uint16).reshape(np.shape(x))


class Ars:
    """Eqs. 10-14 / Algorithm 1 controller state (oracle)."""

    def __init__(self, G1: int):
        self._h = lib().oracle_ars_new(G1)

    def step(self, kept_per_prompt, step: int, total_steps: int, epoch_end: bool) -> int:
        k = _arr(kept_per_prompt, np.int32)
        return int(lib().oracle_ars_step(self._h, _p(k), k.size, step, total_steps, int(epoch_end)))

    @property
    def g_ref(self):
        v = lib().oracle_ars_get(self._h, 0)
        return None if math.isnan(v) else v

    @property
    def g_t(self):
        v = lib().oracle_ars_get(self._h, 1)
        return None if math.isnan(v) else v

    def __del__(self):
        if getattr(self, "_h", None) and _lib is not None:
            _lib.oracle_ars_free(self._h)
            self._h = None
