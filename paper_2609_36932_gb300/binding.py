"""Python binding of libfastrl_grpo: the C ABI of include/fastrl_grpo.h, one function per entry.

Argument marshalling only: tensors become device pointers, outputs that the caller does not
pass are allocated with torch on the input's device, and the work is enqueued on the current
torch CUDA stream.  Every computation runs in the library's CUDA kernels; there is no CPU or
PyTorch fallback, and loading fails loudly if the library cannot be built or loaded.
"""
from __future__ import annotations

import ctypes
import os

import numpy as np

from . import build as _build

_c_p = ctypes.c_void_p
_i32 = ctypes.c_int32
_i64 = ctypes.c_int64
_f32 = ctypes.c_float

GRPO_DTYPE_F32 = 0
GRPO_DTYPE_BF16 = 1
DEVFLAG_BAD_TOKEN = 1
DEVFLAG_NONFINITE = 2
DEVFLAG_TIMEOUT = 4

STATUS_NAMES = {0: "GRPO_OK", 1: "GRPO_ERR_INVALID_ARG", 2: "GRPO_ERR_UNSUPPORTED",
                3: "GRPO_ERR_WORKSPACE", 4: "GRPO_ERR_CUDA", 5: "GRPO_ERR_TIMEOUT",
                6: "GRPO_ERR_DEVICE_CHECK"}

# Every function include/fastrl_grpo.h declares.
EXPORTS = ["grpo_last_error", "grpo_version", "grpo_kernel_launches", "grpo_debug_checks",
           "grpo_check_status",
           "grpo_advantage",
           "grpo_prune", "grpo_compact", "grpo_upload_kept", "grpo_loss_fwd_bwd", "grpo_loss_fwd_bwd_dev", "grpo_loss_fwd_bwd_noalloc", "grpo_gspo_loss_fwd_bwd", "grpo_gspo_loss_fwd_bwd_dev",
           "grpo_sum_f64", "grpo_logp_fwd", "grpo_lmhead_loss_fwd_bwd", "grpo_lmhead_dlogits_stride",
           "grpo_lmhead_logp_fwd", "grpo_lmhead_tune", "grpo_lmhead_gspo_loss_fwd_bwd",
           "grpo_lmhead_grad",
           "grpo_loss_tune", "grpo_test_skip_copy", "grpo_test_fail_launch", "grpo_ars_init",
           "adaptive_rollout_count",
           "grpo_ars_serialize", "grpo_ars_deserialize"]


class GrpoError(RuntimeError):
    def __init__(self, status: int, message: str):
        super().__init__("%s: %s" % (STATUS_NAMES.get(status, str(status)), message))
        self.status = status


class ArsState(ctypes.Structure):
    """grpo_ars_state (Algorithm 1's adaptive sampling state)."""
    _fields_ = [("G1", _i32), ("n", _i32), ("have_ref", _i32), ("have_gt", _i32),
                ("g_ref", ctypes.c_double), ("g_t", ctypes.c_double),
                ("buf_mean_sum", ctypes.c_double), ("buf_max_sum", ctypes.c_double),
                ("buf_count", _i64)]


_lib = None


def checked_build() -> bool:
    """True when FASTRL_GRPO_CHECKED=1 selects the checked build (device index checks, reported
    by grpo_debug_checks) for this process."""
    return os.environ.get("FASTRL_GRPO_CHECKED", "0") == "1"


def library_path() -> str:
    return _build.LIB_CHECKED if checked_build() else _build.LIB


def lib():
    """Load libfastrl_grpo.so, or libfastrl_grpo_checked.so with FASTRL_GRPO_CHECKED=1 (building
    it first if it is missing or stale)."""
    global _lib
    if _lib is not None:
        return _lib
    path = _build.build(checked=checked_build())
    if not os.path.exists(path):
        raise RuntimeError("%s is missing" % path)
    L = ctypes.CDLL(path)
    L.grpo_last_error.restype = ctypes.c_char_p
    L.grpo_last_error.argtypes = []
    L.grpo_version.restype = ctypes.c_char_p
    L.grpo_version.argtypes = []
    L.grpo_kernel_launches.restype = ctypes.c_uint64
    L.grpo_kernel_launches.argtypes = []
    L.grpo_check_status.argtypes = [_i32]
    L.grpo_debug_checks.argtypes = [_i32, _c_p, _c_p]
    L.grpo_debug_checks.restype = _i32
    L.grpo_check_status.restype = _i32
    L.grpo_advantage.argtypes = [_c_p, _i32, _i32, _i32, _c_p, _c_p, _c_p]
    L.grpo_advantage.restype = _i32
    L.grpo_prune.argtypes = [_c_p, _c_p, _f32, _c_p, _c_p, _i32, _i32, _i64, _i32, _i32, _f32, _i32,
                             _i32, _c_p, _c_p, _c_p, _c_p, ctypes.POINTER(ctypes.c_size_t), _c_p]
    L.grpo_prune.restype = _i32
    L.grpo_compact.argtypes = [_c_p, _c_p, _i32, _c_p, _c_p, _c_p, _c_p, _c_p, _c_p, _c_p]
    L.grpo_compact.restype = _i32
    L.grpo_upload_kept.argtypes = [_c_p, _c_p, _i64, _c_p, _c_p, _i32, _c_p, _c_p, _c_p]
    L.grpo_upload_kept.restype = _i32
    L.grpo_loss_fwd_bwd.argtypes = [_c_p, _i32, _i64, _c_p, _i64, _i32, _c_p, _c_p, _c_p, _c_p, _c_p,
                                    _f32, _f32, _f32, _i32, _i64, _c_p, _i64, _c_p, _i32, _c_p, _c_p,
                                    _c_p, _c_p, _c_p, ctypes.POINTER(ctypes.c_size_t), _c_p]
    L.grpo_loss_fwd_bwd.restype = _i32
    L.grpo_loss_fwd_bwd_dev.argtypes = [_c_p, _i32, _i64, _c_p, _i64, _c_p, _i32, _c_p, _c_p, _c_p,
                                        _c_p, _c_p, _f32, _f32, _f32, _i32, _i64, _c_p, _i64, _c_p,
                                        _i32, _c_p, _c_p, _c_p, _c_p, _c_p,
                                        ctypes.POINTER(ctypes.c_size_t), _c_p]
    L.grpo_loss_fwd_bwd_dev.restype = _i32
    L.grpo_loss_fwd_bwd_noalloc.argtypes = [_c_p, _i32, _i64, _c_p, _i64, _i32, _c_p, _c_p, _c_p,
                                            _c_p, _c_p, _f32, _f32, _f32, _i32, _i64, _c_p, _i64,
                                            _c_p, _i32, _c_p, _c_p, _c_p, _c_p, _c_p]
    L.grpo_loss_fwd_bwd_noalloc.restype = _i32
    L.grpo_gspo_loss_fwd_bwd.argtypes = [_c_p, _i32, _i64, _c_p, _i64, _i32, _c_p, _c_p, _c_p,
                                         _c_p, _c_p, _c_p, _i32, _i64, _f32, _f32, _f32, _c_p,
                                         _i32, _c_p, _c_p, _c_p, _c_p, _c_p,
                                         ctypes.POINTER(ctypes.c_size_t), _c_p]
    L.grpo_gspo_loss_fwd_bwd.restype = _i32
    L.grpo_gspo_loss_fwd_bwd_dev.argtypes = [_c_p, _i32, _i64, _c_p, _i64, _i32, _c_p, _i32, _c_p,
                                             _c_p, _c_p, _c_p, _c_p, _c_p, _i64, _f32, _f32, _f32,
                                             _c_p, _i32, _c_p, _c_p, _c_p, _c_p, _c_p,
                                             ctypes.POINTER(ctypes.c_size_t), _c_p]
    L.grpo_gspo_loss_fwd_bwd_dev.restype = _i32
    L.grpo_logp_fwd.argtypes = [_c_p, _i32, _i64, _c_p, _i64, _i32, _c_p, _c_p, _c_p, _c_p]
    L.grpo_logp_fwd.restype = _i32
    L.grpo_lmhead_loss_fwd_bwd.argtypes = [_c_p, _i64, _c_p, _i64, _c_p, _i32, _i32, _c_p, _c_p, _c_p,
                                           _c_p, _c_p, _f32, _f32, _f32, _i32, _i64, _c_p, _i64,
                                           _c_p, _i32, _c_p, _i32, _c_p, _c_p, _c_p, _c_p, _c_p,
                                           _i64, _c_p, _c_p, _c_p]
    L.grpo_lmhead_loss_fwd_bwd.restype = _i32
    L.grpo_lmhead_logp_fwd.argtypes = [_c_p, _i64, _c_p, _i64, _c_p, _i32, _i32, _c_p, _c_p, _c_p,
                                       _c_p, _c_p, _c_p]
    L.grpo_lmhead_logp_fwd.restype = _i32
    L.grpo_lmhead_grad.argtypes = [_c_p, _i64, _i64, _i32, _c_p, _i64, _c_p, _i32, _c_p, _i32,
                                   _c_p, _i32, _c_p, _c_p, ctypes.POINTER(ctypes.c_size_t), _c_p]
    L.grpo_lmhead_grad.restype = _i32
    L.grpo_lmhead_gspo_loss_fwd_bwd.argtypes = [_c_p, _i64, _c_p, _i64, _c_p, _i32, _i32, _c_p,
                                                _c_p, _c_p, _c_p, _c_p, _c_p, _i32, _i64, _f32,
                                                _f32, _f32, _c_p, _i32, _c_p, _i32, _c_p, _c_p,
                                                _c_p, _c_p, _c_p, _i64, _c_p, _c_p, _c_p]
    L.grpo_lmhead_gspo_loss_fwd_bwd.restype = _i32
    L.grpo_lmhead_tune.argtypes = [_i32, _i32, _i32]
    L.grpo_lmhead_tune.restype = _i32
    L.grpo_lmhead_dlogits_stride.argtypes = [_i32]
    L.grpo_lmhead_dlogits_stride.restype = _i64
    L.grpo_sum_f64.argtypes = [_c_p, _i64, _c_p, _c_p]
    L.grpo_sum_f64.restype = _i32
    L.grpo_test_fail_launch.argtypes = [_i32]
    L.grpo_test_fail_launch.restype = _i32
    L.grpo_test_skip_copy.argtypes = [_i32]
    L.grpo_test_skip_copy.restype = _i32
    L.grpo_loss_tune.argtypes = [_i32, _i32, _i32]
    L.grpo_loss_tune.restype = _i32
    L.grpo_ars_init.argtypes = [ctypes.POINTER(ArsState), _i32]
    L.grpo_ars_init.restype = _i32
    L.adaptive_rollout_count.argtypes = [ctypes.POINTER(ArsState), _c_p, _i32, _i64, _i64, _i32]
    L.adaptive_rollout_count.restype = _i32
    L.grpo_ars_serialize.argtypes = [ctypes.POINTER(ArsState), _c_p, ctypes.POINTER(ctypes.c_size_t)]
    L.grpo_ars_serialize.restype = _i32
    L.grpo_ars_deserialize.argtypes = [ctypes.POINTER(ArsState), _c_p, ctypes.c_size_t]
    L.grpo_ars_deserialize.restype = _i32
    _lib = L
    return L


def _check(rc: int):
    if rc != 0:
        raise GrpoError(rc, lib().grpo_last_error().decode(errors="replace"))


def _torch():
    import torch
    return torch


def _ptr(t):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _stream(stream=None):
    torch = _torch()
    s = torch.cuda.current_stream() if stream is None else stream
    return ctypes.c_void_p(s.cuda_stream)


def _need(t, dtype, n, what):
    torch = _torch()
    if t.dtype != dtype:
        raise TypeError("%s must be %s, got %s" % (what, dtype, t.dtype))
    if not t.is_cuda:
        raise TypeError("%s must be a CUDA tensor" % what)
    if not t.is_contiguous():
        raise ValueError("%s must be contiguous" % what)
    if n is not None and t.numel() < n:
        raise ValueError("%s has %d elements, needs %d" % (what, t.numel(), n))
    return t


def _workspace(nbytes: int, device, ws=None):
    torch = _torch()
    if nbytes == 0:
        return None
    if ws is not None and ws.numel() >= nbytes + 256:
        return ws
    return torch.empty(nbytes + 256, dtype=torch.uint8, device=device)


def _aligned(ws):
    """A 256-byte aligned view of a workspace tensor."""
    if ws is None:
        return None, 0
    p = ws.data_ptr()
    pad = (-p) % 256
    return ctypes.c_void_p(p + pad), ws.numel() - pad


def _ws_args(wst):
    """(ws pointer, pointer to its size) for a real call; (NULL, NULL) when no workspace."""
    if wst is None:
        return None, None
    wp, wn = _aligned(wst)
    return wp, ctypes.byref(ctypes.c_size_t(wn))


def version() -> str:
    return lib().grpo_version().decode()


def grpo_kernel_launches() -> int:
    return int(lib().grpo_kernel_launches())


def grpo_last_error() -> str:
    return lib().grpo_last_error().decode(errors="replace")


def grpo_loss_tune(cluster_ctas: int = 0, threads: int = 0, chunks: int = 0):
    _check(lib().grpo_loss_tune(cluster_ctas, threads, chunks))


def grpo_advantage(rewards, G: int, std_mode: int = 0, adv=None, key=None, stream=None):
    """Eq. 5 on the GPU.  Returns (adv f32, key f64 or None)."""
    torch = _torch()
    _need(rewards, torch.float32, None, "rewards")
    n = rewards.numel()
    if G < 1 or n % G:
        raise ValueError("rewards has %d elements, not a multiple of G=%d" % (n, G))
    P = n // G
    if adv is None:
        adv = torch.empty(n, dtype=torch.float32, device=rewards.device)
    _need(adv, torch.float32, n, "adv")
    if key is not None:
        _need(key, torch.float64, n, "key")
    _check(lib().grpo_advantage(_ptr(rewards), P, G, std_mode, _ptr(adv), _ptr(key), _stream(stream)))
    return adv, key


def grpo_prune(rewards, ids, off, G: int, V: int, ngram_n: int = 1, tau: float = 0.8,
               keep_cap: int | None = None, dp_divisor: int = 1, keep=None, kept_per_prompt=None,
               status=None, ws=None, stream=None, adv=None, class_eps: float = 0.0):
    """Eqs. 6-9 + Algorithm 1 on the GPU.  Returns (keep u8 [P*G], kept_per_prompt i32 [P]).
    class_eps > 0 with adv: classes by chained advantages (continuous rewards)."""
    torch = _torch()
    _need(rewards, torch.float32, None, "rewards")
    n = rewards.numel()
    P = n // G
    _need(off, torch.int64, n + 1, "off")
    _need(ids, torch.int32, None, "ids")
    T = ids.numel()
    cap = G if keep_cap is None else int(keep_cap)
    if keep is None:
        keep = torch.empty(n, dtype=torch.uint8, device=rewards.device)
    if kept_per_prompt is None:
        kept_per_prompt = torch.empty(max(P, 1), dtype=torch.int32, device=rewards.device)
    if adv is not None:
        _need(adv, torch.float32, n, "adv")
    L = lib()
    head = (_ptr(rewards), _ptr(adv), float(class_eps), _ptr(ids), _ptr(off), P, G, T, V, ngram_n,
            float(tau), cap, dp_divisor, _ptr(keep), _ptr(kept_per_prompt), _ptr(status))
    need = ctypes.c_size_t(0)
    _check(L.grpo_prune(*head, None, ctypes.byref(need), _stream(stream)))
    wst = _workspace(need.value, rewards.device, ws)
    wp, size = _ws_args(wst)
    _check(L.grpo_prune(*head, wp, size, _stream(stream)))
    return keep, kept_per_prompt[:P]


def grpo_compact(keep, off, kept_idx=None, kept_off=None, src_token=None, token_rollout=None,
                 counts=None, counts_host=None, stream=None):
    """Token compaction on the GPU.  Returns a dict of the output tensors (full capacity)."""
    torch = _torch()
    _need(keep, torch.uint8, None, "keep")
    n = keep.numel()
    _need(off, torch.int64, n + 1, "off")
    dev = keep.device
    T = None
    if src_token is None or token_rollout is None:
        T = int(off[n].item())
    if kept_idx is None:
        kept_idx = torch.empty(max(n, 1), dtype=torch.int32, device=dev)
    if kept_off is None:
        kept_off = torch.empty(n + 1, dtype=torch.int64, device=dev)
    if src_token is None:
        src_token = torch.empty(max(T, 1), dtype=torch.int64, device=dev)
    if token_rollout is None:
        token_rollout = torch.empty(max(T, 1), dtype=torch.int32, device=dev)
    if counts is None:
        counts = torch.empty(2, dtype=torch.int64, device=dev)
    hp = None if counts_host is None else ctypes.c_void_p(counts_host.data_ptr())
    _check(lib().grpo_compact(_ptr(keep), _ptr(off), n, _ptr(kept_idx), _ptr(kept_off),
                              _ptr(src_token), _ptr(token_rollout), _ptr(counts), hp, _stream(stream)))
    return dict(kept_idx=kept_idx, kept_off=kept_off, src_token=src_token,
                token_rollout=token_rollout, counts=counts)


def grpo_upload_kept(src_host, dst, keep_host, off_host, stream=None):
    """Copy the kept rollouts' token rows of `src_host` (a host tensor, pinned for the copies to be
    asynchronous) into the same rows of the device tensor `dst`.  keep_host: host u8
    [n_rollouts]; off_host: host i64 [n_rollouts+1].  Rows are dim 0 of src_host and dst.
    Returns (bytes, copies) enqueued on the stream."""
    torch = _torch()
    if src_host.is_cuda or not dst.is_cuda:
        raise ValueError("grpo_upload_kept: src_host must be a host tensor and dst a device tensor")
    if src_host.shape != dst.shape or src_host.dtype != dst.dtype:
        raise ValueError("grpo_upload_kept: src_host and dst differ in shape or dtype")
    if not (src_host.is_contiguous() and dst.is_contiguous()):
        raise ValueError("grpo_upload_kept: src_host and dst must be contiguous")
    if keep_host.is_cuda or off_host.is_cuda:
        raise ValueError("grpo_upload_kept: keep_host and off_host must be host tensors")
    if keep_host.dtype != torch.uint8 or off_host.dtype != torch.int64:
        raise TypeError("grpo_upload_kept: keep_host must be uint8 and off_host int64")
    if not (keep_host.is_contiguous() and off_host.is_contiguous()):
        raise ValueError("grpo_upload_kept: keep_host and off_host must be contiguous")
    n = keep_host.numel()
    if off_host.numel() < n + 1:
        raise ValueError("grpo_upload_kept: off_host needs n_rollouts + 1 entries")
    rows = src_host.shape[0] if src_host.dim() else 1
    if n and int(off_host[n]) > rows:
        raise ValueError("grpo_upload_kept: off_host[-1] = %d exceeds the %d rows"
                         % (int(off_host[n]), rows))
    row_bytes = src_host.numel() * src_host.element_size() // max(rows, 1)
    nbytes, ncopies = ctypes.c_int64(0), ctypes.c_int32(0)
    _check(lib().grpo_upload_kept(_ptr(src_host), _ptr(dst), row_bytes, _ptr(keep_host),
                                  _ptr(off_host), n, ctypes.byref(nbytes), ctypes.byref(ncopies),
                                  _stream(stream)))
    return nbytes.value, ncopies.value


def grpo_loss_fwd_bwd(logits, y, old_logp, ref_logp, adv, row_rollout, *, V: int | None = None,
                      row_stride: int | None = None, row_index=None, n_rows: int | None = None,
                      eps_low: float = 0.2, eps_high: float = 0.2, beta: float = 0.04,
                      agg_mode: int = 0, denom_tokens: int | None = None, seq_off=None,
                      n_seq: int = 0, dlogits=None, dlogits_dtype=None, logp_out=None,
                      row_loss_out=None, loss_out=None, status=None, ws=None, stream=None):
    """Eqs. 1-3 on the GPU.  Returns dict(loss (f64 [1] tensor), dlogits, logp, row_loss)."""
    torch = _torch()
    if logits.dtype == torch.bfloat16:
        ldt = GRPO_DTYPE_BF16
    elif logits.dtype == torch.float32:
        ldt = GRPO_DTYPE_F32
    else:
        raise TypeError("logits must be bf16 or f32")
    if not logits.is_cuda:
        raise TypeError("logits must be a CUDA tensor")
    if logits.dim() != 2 or logits.stride(1) != 1:
        raise ValueError("logits must be 2-D with unit stride along the vocabulary")
    if V is None:
        V = logits.shape[1]
    stride = logits.stride(0) if row_stride is None else int(row_stride)
    if n_rows is None:
        n_rows = row_index.numel() if row_index is not None else logits.shape[0]
    dev = logits.device
    if dlogits_dtype is None:
        if dlogits is not None:
            dlogits_dtype = GRPO_DTYPE_BF16 if dlogits.dtype == torch.bfloat16 else GRPO_DTYPE_F32
        else:
            dlogits_dtype = ldt
    elif dlogits_dtype in (torch.bfloat16, "bf16"):
        dlogits_dtype = GRPO_DTYPE_BF16
    elif dlogits_dtype in (torch.float32, "f32"):
        dlogits_dtype = GRPO_DTYPE_F32
    out_t = torch.bfloat16 if dlogits_dtype == GRPO_DTYPE_BF16 else torch.float32
    if dlogits is None:
        dlogits = torch.empty((n_rows, V), dtype=out_t, device=dev)
    _need(dlogits, out_t, n_rows * V, "dlogits")
    if loss_out is None:
        loss_out = torch.empty(1, dtype=torch.float64, device=dev)
    if denom_tokens is None:
        denom_tokens = max(int(n_rows), 1)
    _need(y, torch.int32, None, "y")
    _need(old_logp, torch.float32, None, "old_logp")
    _need(ref_logp, torch.float32, None, "ref_logp")
    _need(adv, torch.float32, None, "adv")
    _need(row_rollout, torch.int32, n_rows, "row_rollout")
    if row_index is not None:
        _need(row_index, torch.int64, n_rows, "row_index")
    L = lib()
    args_head = (_ptr(logits), ldt, stride, _ptr(row_index), int(n_rows), int(V), _ptr(y),
                 _ptr(old_logp), _ptr(ref_logp), _ptr(adv), _ptr(row_rollout), float(eps_low),
                 float(eps_high), float(beta), int(agg_mode), int(denom_tokens), _ptr(seq_off),
                 int(n_seq), _ptr(dlogits), dlogits_dtype, _ptr(logp_out), _ptr(row_loss_out),
                 _ptr(loss_out), _ptr(status))
    need = ctypes.c_size_t(0)
    _check(L.grpo_loss_fwd_bwd(*args_head, None, ctypes.byref(need), _stream(stream)))
    wst = _workspace(need.value, dev, ws)
    wp, size = _ws_args(wst)
    _check(L.grpo_loss_fwd_bwd(*args_head, wp, size, _stream(stream)))
    return dict(loss=loss_out, dlogits=dlogits, logp=logp_out, row_loss=row_loss_out, ws=wst)


def grpo_debug_checks(reset: bool = True):
    """The checked build's report: (mask of files whose index checks failed, first failing site
    as 100000 * file + line), after synchronising the device.  GrpoError(GRPO_ERR_UNSUPPORTED)
    from the normal build."""
    mask, site = _i32(0), _i32(0)
    _check(lib().grpo_debug_checks(int(bool(reset)), ctypes.byref(mask), ctypes.byref(site)))
    return mask.value, site.value


def grpo_lmhead_tune(prefetch: int = 0, row_lanes: int = 0, recompute_logits: int = 0):
    """Launch settings of the output-layer kernels for this process (see the header)."""
    _check(lib().grpo_lmhead_tune(int(prefetch), int(row_lanes), int(recompute_logits)))


def grpo_lmhead_dlogits_stride(V: int) -> int:
    """Row stride (elements) of grpo_lmhead_loss_fwd_bwd's dlogits_out."""
    return int(lib().grpo_lmhead_dlogits_stride(int(V)))


def grpo_lmhead_logp_fwd(hidden, weight, y, *, row_index=None, n_rows: int | None = None,
                         logp_out=None, status=None, ws=None, stream=None):
    """log pi(y) from hidden states through the output layer (see the header).  Returns
    dict(logp, ws)."""
    torch = _torch()
    if hidden.dtype != torch.bfloat16 or weight.dtype != torch.bfloat16:
        raise TypeError("hidden and weight must be bf16")
    if hidden.dim() != 2 or hidden.stride(1) != 1 or not hidden.is_cuda:
        raise ValueError("hidden must be a 2-D CUDA tensor with unit stride along D")
    if weight.dim() != 2 or not weight.is_contiguous() or weight.shape[1] != hidden.shape[1]:
        raise ValueError("weight must be a contiguous [V, D] tensor")
    D = hidden.shape[1]
    V = weight.shape[0]
    if n_rows is None:
        n_rows = row_index.numel() if row_index is not None else hidden.shape[0]
    if row_index is not None:
        _need(row_index, torch.int64, n_rows, "row_index")
    _need(y, torch.int32, None if row_index is not None else n_rows, "y")
    if logp_out is None:
        logp_out = torch.empty(max(int(n_rows), 1), dtype=torch.float32, device=hidden.device)
    L = lib()
    head = (_ptr(hidden), int(hidden.stride(0)), _ptr(row_index), int(n_rows), _ptr(weight), int(V),
            int(D), _ptr(y), _ptr(logp_out), _ptr(status))
    need = ctypes.c_size_t(0)
    _check(L.grpo_lmhead_logp_fwd(*head, None, ctypes.byref(need), _stream(stream)))
    wst = _workspace(need.value, hidden.device, ws)
    wp, size = _ws_args(wst)
    _check(L.grpo_lmhead_logp_fwd(*head, wp, size, _stream(stream)))
    return dict(logp=logp_out, ws=wst)


def grpo_lmhead_grad(dlogits, hidden, weight, *, n_rows: int | None = None, dhidden=None,
                     dhidden_dtype=None, dweight=None, accumulate_dweight: bool = False,
                     want_dhidden: bool = True, want_dweight: bool = True, status=None, ws=None,
                     stream=None):
    """dhidden = dlogits @ weight and dweight (+)= dlogits^T @ hidden on the tensor cores (the
    chain rule through the output layer, see the header).  dlogits bf16 [n_rows, >= V] with unit
    stride along V; hidden bf16 [n_rows, D]; weight bf16 [V, D].  Returns dict(dhidden, dweight,
    ws)."""
    torch = _torch()
    for t, nm in ((dlogits, "dlogits"), (hidden, "hidden"), (weight, "weight")):
        if t.dtype != torch.bfloat16 or not t.is_cuda or t.dim() != 2 or t.stride(1) != 1:
            raise TypeError("%s must be a 2-D bf16 CUDA tensor with unit inner stride" % nm)
    if not weight.is_contiguous() or weight.shape[1] != hidden.shape[1]:
        raise ValueError("weight must be a contiguous [V, D] tensor")
    V, D = weight.shape
    if n_rows is None:
        n_rows = dlogits.shape[0]
    dev = dlogits.device
    if dhidden_dtype is None:
        dhidden_dtype = dhidden.dtype if dhidden is not None else torch.bfloat16
    dht = GRPO_DTYPE_BF16 if dhidden_dtype in (torch.bfloat16, "bf16") else GRPO_DTYPE_F32
    ht = torch.bfloat16 if dht == GRPO_DTYPE_BF16 else torch.float32
    if want_dhidden and dhidden is None:
        dhidden = torch.empty((max(int(n_rows), 1), D), dtype=ht, device=dev)
    if want_dhidden:
        _need(dhidden, ht, n_rows * D, "dhidden")
    if want_dweight and dweight is None:
        dweight = torch.empty((V, D), dtype=torch.float32, device=dev)
    if want_dweight:
        _need(dweight, torch.float32, V * D, "dweight")
    L = lib()
    head = (_ptr(dlogits), int(dlogits.stride(0)), int(n_rows), int(V), _ptr(hidden),
            int(hidden.stride(0)), _ptr(weight), int(D), _ptr(dhidden if want_dhidden else None),
            dht, _ptr(dweight if want_dweight else None), int(bool(accumulate_dweight)),
            _ptr(status))
    need = ctypes.c_size_t(0)
    _check(L.grpo_lmhead_grad(*head, None, ctypes.byref(need), _stream(stream)))
    wst = _workspace(need.value, dev, ws)
    wp, size = _ws_args(wst)
    _check(L.grpo_lmhead_grad(*head, wp, size, _stream(stream)))
    return dict(dhidden=dhidden, dweight=dweight, ws=wst)


def _lmhead_common(hidden, weight, row_index, n_rows, dhidden, dhidden_dtype, dweight,
                   dlogits_out):
    torch = _torch()
    if hidden.dtype != torch.bfloat16 or weight.dtype != torch.bfloat16:
        raise TypeError("hidden and weight must be bf16")
    if not (hidden.is_cuda and weight.is_cuda):
        raise TypeError("hidden and weight must be CUDA tensors")
    if hidden.dim() != 2 or hidden.stride(1) != 1:
        raise ValueError("hidden must be 2-D with unit stride along D")
    if weight.dim() != 2 or not weight.is_contiguous() or weight.shape[1] != hidden.shape[1]:
        raise ValueError("weight must be a contiguous [V, D] tensor")
    D = hidden.shape[1]
    V = weight.shape[0]
    if n_rows is None:
        n_rows = row_index.numel() if row_index is not None else hidden.shape[0]
    if row_index is not None:
        _need(row_index, torch.int64, n_rows, "row_index")
    dev = hidden.device
    if dhidden_dtype is None:
        dhidden_dtype = dhidden.dtype if dhidden is not None else torch.bfloat16
    if dhidden_dtype in (torch.bfloat16, "bf16"):
        dht, ht = GRPO_DTYPE_BF16, torch.bfloat16
    elif dhidden_dtype in (torch.float32, "f32"):
        dht, ht = GRPO_DTYPE_F32, torch.float32
    else:
        raise TypeError("dhidden must be bf16 or f32")
    if dhidden is None:
        dhidden = torch.empty((max(int(n_rows), 1), D), dtype=ht, device=dev)
    _need(dhidden, ht, n_rows * D, "dhidden")
    if dweight is None:
        dweight = torch.empty((V, D), dtype=torch.float32, device=dev)
    _need(dweight, torch.float32, V * D, "dweight")
    if dlogits_out is not None:
        _need(dlogits_out, torch.bfloat16, n_rows * grpo_lmhead_dlogits_stride(V), "dlogits_out")
    return int(n_rows), V, D, dht, dhidden, dweight


def grpo_lmhead_gspo_loss_fwd_bwd(hidden, weight, y, old_logp, ref_logp, adv, seq_rollout,
                                  seq_row_off, *, n_seq_rows: int | None = None,
                                  n_seq: int | None = None, eps_low: float = 0.2,
                                  eps_high: float = 0.2, beta: float = 0.0, dhidden=None,
                                  dhidden_dtype=None, dweight=None,
                                  accumulate_dweight: bool = False, dlogits_out=None,
                                  logp_out=None, seq_ratio_out=None, loss_out=None, status=None,
                                  chunk_rows: int = 0, row_index=None, n_rows: int | None = None,
                                  ws=None, stream=None):
    """The output layer fused with GSPO's sequence-level loss (see the header).  seq_row_off /
    seq_rollout: device i64 [K+1] / i32 [K] over the rows in order.  Returns dict(loss, dhidden,
    dweight, logp, seq_ratio, dlogits)."""
    torch = _torch()
    n_rows, V, D, dht, dhidden, dweight = _lmhead_common(hidden, weight, row_index, n_rows,
                                                         dhidden, dhidden_dtype, dweight,
                                                         dlogits_out)
    dev = hidden.device
    if n_seq_rows is None:
        n_seq_rows = seq_rollout.numel()
    if n_seq is None:
        n_seq = max(int(n_seq_rows), 1)
    _need(seq_rollout, torch.int32, n_seq_rows, "seq_rollout")
    _need(seq_row_off, torch.int64, n_seq_rows + 1, "seq_row_off")
    _need(adv, torch.float32, None, "adv")
    n_src = None if row_index is not None else n_rows
    _need(y, torch.int32, n_src, "y")
    _need(old_logp, torch.float32, n_src, "old_logp")
    _need(ref_logp, torch.float32, n_src, "ref_logp")
    if logp_out is None:
        logp_out = torch.empty(max(n_rows, 1), dtype=torch.float32, device=dev)
    if loss_out is None:
        loss_out = torch.empty(1, dtype=torch.float64, device=dev)
    L = lib()
    head = (_ptr(hidden), int(hidden.stride(0)), _ptr(row_index), n_rows, _ptr(weight), V, D,
            _ptr(y), _ptr(old_logp), _ptr(ref_logp), _ptr(adv), _ptr(seq_rollout),
            _ptr(seq_row_off), int(n_seq_rows), int(n_seq), float(eps_low), float(eps_high),
            float(beta), _ptr(dhidden), dht, _ptr(dweight), 1 if accumulate_dweight else 0,
            _ptr(dlogits_out), _ptr(logp_out), _ptr(seq_ratio_out), _ptr(loss_out), _ptr(status),
            int(chunk_rows))
    need = ctypes.c_size_t(0)
    _check(L.grpo_lmhead_gspo_loss_fwd_bwd(*head, None, ctypes.byref(need), _stream(stream)))
    wst = _workspace(need.value, dev, ws)
    wp, size = _ws_args(wst)
    _check(L.grpo_lmhead_gspo_loss_fwd_bwd(*head, wp, size, _stream(stream)))
    return dict(loss=loss_out, dhidden=dhidden, dweight=dweight, logp=logp_out,
                seq_ratio=seq_ratio_out, dlogits=dlogits_out, ws=wst)


def grpo_lmhead_loss_fwd_bwd(hidden, weight, y, old_logp, ref_logp, adv, row_rollout, *,
                             eps_low: float = 0.2, eps_high: float = 0.2, beta: float = 0.04,
                             agg_mode: int = 0, denom_tokens: int | None = None, seq_off=None,
                             n_seq: int = 0, dhidden=None, dhidden_dtype=None, dweight=None,
                             accumulate_dweight: bool = False, dlogits_out=None, logp_out=None,
                             row_loss_out=None, loss_out=None, status=None, chunk_rows: int = 0,
                             row_index=None, n_rows: int | None = None, ws=None, stream=None):
    """The output layer fused with the GRPO loss (see the header): hidden bf16 [*, D] (rows taken
    through row_index when given), weight bf16 [V, D].  Returns dict(loss, dhidden, dweight, logp,
    row_loss, dlogits)."""
    torch = _torch()
    if hidden.dtype != torch.bfloat16 or weight.dtype != torch.bfloat16:
        raise TypeError("hidden and weight must be bf16")
    if not (hidden.is_cuda and weight.is_cuda):
        raise TypeError("hidden and weight must be CUDA tensors")
    if hidden.dim() != 2 or hidden.stride(1) != 1:
        raise ValueError("hidden must be 2-D with unit stride along D")
    if weight.dim() != 2 or not weight.is_contiguous():
        raise ValueError("weight must be a contiguous [V, D] tensor")
    D = hidden.shape[1]
    if n_rows is None:
        n_rows = row_index.numel() if row_index is not None else hidden.shape[0]
    if row_index is not None:
        _need(row_index, torch.int64, n_rows, "row_index")
    V = weight.shape[0]
    if weight.shape[1] != D:
        raise ValueError("hidden and weight disagree on D")
    dev = hidden.device
    if dhidden_dtype is None:
        dhidden_dtype = dhidden.dtype if dhidden is not None else torch.bfloat16
    if dhidden_dtype in (torch.bfloat16, "bf16"):
        dht, ht = GRPO_DTYPE_BF16, torch.bfloat16
    elif dhidden_dtype in (torch.float32, "f32"):
        dht, ht = GRPO_DTYPE_F32, torch.float32
    else:
        raise TypeError("dhidden must be bf16 or f32")
    if dhidden is None:
        dhidden = torch.empty((n_rows, D), dtype=ht, device=dev)
    _need(dhidden, ht, n_rows * D, "dhidden")
    if dweight is None:
        dweight = torch.empty((V, D), dtype=torch.float32, device=dev)
    _need(dweight, torch.float32, V * D, "dweight")
    if dlogits_out is not None:
        _need(dlogits_out, torch.bfloat16, n_rows * grpo_lmhead_dlogits_stride(V), "dlogits_out")
    if loss_out is None:
        loss_out = torch.empty(1, dtype=torch.float64, device=dev)
    if denom_tokens is None:
        denom_tokens = max(int(n_rows), 1)
    n_src = None if row_index is not None else n_rows
    _need(y, torch.int32, n_src, "y")
    _need(old_logp, torch.float32, n_src, "old_logp")
    _need(ref_logp, torch.float32, n_src, "ref_logp")
    _need(adv, torch.float32, None, "adv")
    _need(row_rollout, torch.int32, n_rows, "row_rollout")
    L = lib()
    head = (_ptr(hidden), int(hidden.stride(0)), _ptr(row_index), int(n_rows), _ptr(weight),
            int(V), int(D),
            _ptr(y), _ptr(old_logp), _ptr(ref_logp), _ptr(adv), _ptr(row_rollout),
            float(eps_low), float(eps_high), float(beta), int(agg_mode), int(denom_tokens),
            _ptr(seq_off), int(n_seq), _ptr(dhidden), dht, _ptr(dweight),
            1 if accumulate_dweight else 0, _ptr(dlogits_out), _ptr(logp_out),
            _ptr(row_loss_out), _ptr(loss_out), _ptr(status), int(chunk_rows))
    need = ctypes.c_size_t(0)
    _check(L.grpo_lmhead_loss_fwd_bwd(*head, None, ctypes.byref(need), _stream(stream)))
    wst = _workspace(need.value, dev, ws)
    wp, size = _ws_args(wst)
    _check(L.grpo_lmhead_loss_fwd_bwd(*head, wp, size, _stream(stream)))
    return dict(loss=loss_out, dhidden=dhidden, dweight=dweight, logp=logp_out,
                row_loss=row_loss_out, dlogits=dlogits_out, ws=wst)


def grpo_gspo_loss_fwd_bwd(logits, y, old_logp, ref_logp, adv, seq_rollout, seq_row_off, *,
                           n_rows: int, n_seq_rows: int | None = None, n_seq: int | None = None,
                           V: int | None = None, row_stride: int | None = None, row_index=None,
                           eps_low: float = 0.2, eps_high: float = 0.2, beta: float = 0.0,
                           dlogits=None, dlogits_dtype=None, logp_out=None, seq_ratio_out=None,
                           loss_out=None, status=None, ws=None, stream=None):
    """GSPO's sequence-level loss on the GPU (see the header).  seq_row_off / seq_rollout: device
    i64 [K+1] / i32 [K] (grpo_compact's kept_off and kept_idx); n_rows: the rows they cover
    (T_kept).  n_seq_rows defaults to seq_rollout.numel(), n_seq to n_seq_rows.  Returns
    dict(loss, dlogits, logp, seq_ratio)."""
    torch = _torch()
    if logits.dtype == torch.bfloat16:
        ldt = GRPO_DTYPE_BF16
    elif logits.dtype == torch.float32:
        ldt = GRPO_DTYPE_F32
    else:
        raise TypeError("logits must be bf16 or f32")
    if not logits.is_cuda:
        raise TypeError("logits must be a CUDA tensor")
    if logits.dim() != 2 or logits.stride(1) != 1:
        raise ValueError("logits must be 2-D with unit stride along the vocabulary")
    if V is None:
        V = logits.shape[1]
    stride = logits.stride(0) if row_stride is None else int(row_stride)
    if n_seq_rows is None:
        n_seq_rows = seq_rollout.numel()
    if n_seq is None:
        n_seq = max(int(n_seq_rows), 1)
    dev = logits.device
    if dlogits_dtype is None:
        if dlogits is not None:
            dlogits_dtype = GRPO_DTYPE_BF16 if dlogits.dtype == torch.bfloat16 else GRPO_DTYPE_F32
        else:
            dlogits_dtype = ldt
    elif dlogits_dtype in (torch.bfloat16, "bf16"):
        dlogits_dtype = GRPO_DTYPE_BF16
    elif dlogits_dtype in (torch.float32, "f32"):
        dlogits_dtype = GRPO_DTYPE_F32
    out_t = torch.bfloat16 if dlogits_dtype == GRPO_DTYPE_BF16 else torch.float32
    if dlogits is None:
        dlogits = torch.empty((max(n_rows, 1), V), dtype=out_t, device=dev)
    _need(dlogits, out_t, n_rows * V, "dlogits")
    if logp_out is None:
        logp_out = torch.empty(max(n_rows, 1), dtype=torch.float32, device=dev)
    _need(logp_out, torch.float32, n_rows, "logp_out")
    if seq_ratio_out is not None:
        _need(seq_ratio_out, torch.float32, n_seq_rows, "seq_ratio_out")
    if loss_out is None:
        loss_out = torch.empty(1, dtype=torch.float64, device=dev)
    _need(y, torch.int32, None, "y")
    _need(old_logp, torch.float32, None, "old_logp")
    _need(ref_logp, torch.float32, None, "ref_logp")
    _need(adv, torch.float32, None, "adv")
    _need(seq_rollout, torch.int32, n_seq_rows, "seq_rollout")
    _need(seq_row_off, torch.int64, n_seq_rows + 1, "seq_row_off")
    if row_index is not None:
        _need(row_index, torch.int64, n_rows, "row_index")
    L = lib()
    head = (_ptr(logits), ldt, stride, _ptr(row_index), int(n_rows), int(V), _ptr(y),
            _ptr(old_logp), _ptr(ref_logp), _ptr(adv), _ptr(seq_rollout), _ptr(seq_row_off),
            int(n_seq_rows), int(n_seq), float(eps_low), float(eps_high), float(beta),
            _ptr(dlogits), dlogits_dtype, _ptr(logp_out), _ptr(seq_ratio_out), _ptr(loss_out),
            _ptr(status))
    need = ctypes.c_size_t(0)
    _check(L.grpo_gspo_loss_fwd_bwd(*head, None, ctypes.byref(need), _stream(stream)))
    wst = _workspace(need.value, dev, ws)
    wp, size = _ws_args(wst)
    _check(L.grpo_gspo_loss_fwd_bwd(*head, wp, size, _stream(stream)))
    return dict(loss=loss_out, dlogits=dlogits, logp=logp_out, seq_ratio=seq_ratio_out, ws=wst)


def grpo_gspo_loss_fwd_bwd_dev(logits, y, old_logp, ref_logp, adv, seq_rollout, seq_row_off,
                               counts, *, max_rows: int, max_seqs: int, dlogits, loss_out, ws,
                               n_seq: int = 0, V: int | None = None, row_stride: int | None = None,
                               row_index=None, eps_low: float = 0.2, eps_high: float = 0.2,
                               beta: float = 0.0, logp_out=None, seq_ratio_out=None, status=None,
                               stream=None):
    """GSPO's loss with {K, T_kept} read from the device `counts` (CUDA-graph capturable): the
    caller passes every buffer, sized for max_rows and max_seqs, and a workspace tensor."""
    torch = _torch()
    ldt = GRPO_DTYPE_BF16 if logits.dtype == torch.bfloat16 else GRPO_DTYPE_F32
    if V is None:
        V = logits.shape[1]
    stride = logits.stride(0) if row_stride is None else int(row_stride)
    odt = GRPO_DTYPE_BF16 if dlogits.dtype == torch.bfloat16 else GRPO_DTYPE_F32
    _need(counts, torch.int64, 2, "counts")
    _need(dlogits, dlogits.dtype, max_rows * V, "dlogits")
    _need(seq_rollout, torch.int32, max_seqs, "seq_rollout")
    _need(seq_row_off, torch.int64, max_seqs + 1, "seq_row_off")
    if logp_out is None:
        raise ValueError("grpo_gspo_loss_fwd_bwd_dev: logp_out is required")
    head = (_ptr(logits), ldt, stride, _ptr(row_index), int(max_rows), int(max_seqs), _ptr(counts),
            int(V), _ptr(y), _ptr(old_logp), _ptr(ref_logp), _ptr(adv), _ptr(seq_rollout),
            _ptr(seq_row_off), int(n_seq), float(eps_low), float(eps_high), float(beta),
            _ptr(dlogits), odt, _ptr(logp_out), _ptr(seq_ratio_out), _ptr(loss_out), _ptr(status))
    L = lib()
    need = ctypes.c_size_t(0)
    _check(L.grpo_gspo_loss_fwd_bwd_dev(*head, None, ctypes.byref(need), _stream(stream)))
    wst = _workspace(need.value, logits.device, ws)
    wp, size = _ws_args(wst)
    _check(L.grpo_gspo_loss_fwd_bwd_dev(*head, wp, size, _stream(stream)))
    return dict(loss=loss_out, dlogits=dlogits, logp=logp_out, seq_ratio=seq_ratio_out, ws=wst)


def grpo_loss_fwd_bwd_noalloc(logits, y, old_logp, ref_logp, adv, row_rollout, *, dlogits,
                              logp_out=None, row_loss_out=None, loss_out, status=None,
                              row_index=None, n_rows: int | None = None, V: int | None = None,
                              row_stride: int | None = None, eps_low: float = 0.2,
                              eps_high: float = 0.2, beta: float = 0.04, agg_mode: int = 0,
                              denom_tokens: int | None = None, seq_off=None, n_seq: int = 0,
                              stream=None):
    """The allocation-free loss entry: for callers that cannot allocate device memory when the
    loss runs (a host that passes only inputs and outputs and has no workspace hook, or a
    runtime that forbids allocation after start-up).  Every output buffer must be passed in;
    the library's fixed scratch holds the per-row loss terms (at most 262144 rows per call
    unless row_loss_out is given).  Nothing here allocates."""
    torch = _torch()
    if logits.dtype == torch.bfloat16:
        ldt = GRPO_DTYPE_BF16
    elif logits.dtype == torch.float32:
        ldt = GRPO_DTYPE_F32
    else:
        raise TypeError("logits must be bf16 or f32")
    if logits.dim() != 2 or logits.stride(1) != 1 or not logits.is_cuda:
        raise ValueError("logits must be a 2-D CUDA tensor with unit stride along the vocabulary")
    if V is None:
        V = logits.shape[1]
    stride = logits.stride(0) if row_stride is None else int(row_stride)
    if n_rows is None:
        n_rows = row_index.numel() if row_index is not None else logits.shape[0]
    if dlogits.dtype == torch.bfloat16:
        odt = GRPO_DTYPE_BF16
    elif dlogits.dtype == torch.float32:
        odt = GRPO_DTYPE_F32
    else:
        raise TypeError("dlogits must be bf16 or f32")
    _need(dlogits, dlogits.dtype, n_rows * V, "dlogits")
    _need(loss_out, torch.float64, 1, "loss_out")
    if denom_tokens is None:
        denom_tokens = max(int(n_rows), 1)
    _check(lib().grpo_loss_fwd_bwd_noalloc(
        _ptr(logits), ldt, stride, _ptr(row_index), int(n_rows), int(V), _ptr(y), _ptr(old_logp),
        _ptr(ref_logp), _ptr(adv), _ptr(row_rollout), float(eps_low), float(eps_high),
        float(beta), int(agg_mode), int(denom_tokens), _ptr(seq_off), int(n_seq), _ptr(dlogits),
        odt, _ptr(logp_out), _ptr(row_loss_out), _ptr(loss_out), _ptr(status), _stream(stream)))
    return dict(loss=loss_out, dlogits=dlogits, logp=logp_out, row_loss=row_loss_out)


def grpo_loss_fwd_bwd_dev(logits, y, old_logp, ref_logp, adv, row_rollout, counts, *,
                          max_rows: int, dlogits, loss_out, ws, V: int | None = None,
                          row_stride: int | None = None, row_index=None, eps_low: float = 0.2,
                          eps_high: float = 0.2, beta: float = 0.04, agg_mode: int = 0,
                          denom_tokens: int = 0, seq_off=None, n_seq: int = 0, logp_out=None,
                          row_loss_out=None, status=None, stream=None):
    """Eqs. 1-3 with the row count {K, T_kept} read on the device (capturable in a CUDA graph).
    All buffers are passed in, sized for max_rows; nothing is allocated here."""
    torch = _torch()
    ldt = GRPO_DTYPE_BF16 if logits.dtype == torch.bfloat16 else GRPO_DTYPE_F32
    odt = GRPO_DTYPE_BF16 if dlogits.dtype == torch.bfloat16 else GRPO_DTYPE_F32
    if V is None:
        V = logits.shape[1]
    stride = logits.stride(0) if row_stride is None else int(row_stride)
    _need(counts, torch.int64, 2, "counts")
    wp, size = _ws_args(ws)
    _check(lib().grpo_loss_fwd_bwd_dev(
        _ptr(logits), ldt, stride, _ptr(row_index), int(max_rows), _ptr(counts), int(V), _ptr(y),
        _ptr(old_logp), _ptr(ref_logp), _ptr(adv), _ptr(row_rollout), float(eps_low),
        float(eps_high), float(beta), int(agg_mode), int(denom_tokens), _ptr(seq_off), int(n_seq),
        _ptr(dlogits), odt, _ptr(logp_out), _ptr(row_loss_out), _ptr(loss_out), _ptr(status), wp,
        size, _stream(stream)))
    return loss_out


def grpo_logp_fwd(logits, y, *, V: int | None = None, row_stride: int | None = None,
                  row_index=None, n_rows: int | None = None, logp_out=None, status=None,
                  stream=None):
    """log pi(y) of each row on the GPU (old/reference policy evaluation).  Returns logp f32."""
    torch = _torch()
    if logits.dtype == torch.bfloat16:
        ldt = GRPO_DTYPE_BF16
    elif logits.dtype == torch.float32:
        ldt = GRPO_DTYPE_F32
    else:
        raise TypeError("logits must be bf16 or f32")
    if logits.dim() != 2 or logits.stride(1) != 1 or not logits.is_cuda:
        raise ValueError("logits must be a 2-D CUDA tensor with unit stride along the vocabulary")
    if V is None:
        V = logits.shape[1]
    stride = logits.stride(0) if row_stride is None else int(row_stride)
    if n_rows is None:
        n_rows = row_index.numel() if row_index is not None else logits.shape[0]
    _need(y, torch.int32, None, "y")
    if row_index is not None:
        _need(row_index, torch.int64, n_rows, "row_index")
    if logp_out is None:
        logp_out = torch.empty(max(int(n_rows), 1), dtype=torch.float32, device=logits.device)
    _need(logp_out, torch.float32, n_rows, "logp_out")
    _check(lib().grpo_logp_fwd(_ptr(logits), ldt, stride, _ptr(row_index), int(n_rows), int(V),
                               _ptr(y), _ptr(logp_out), _ptr(status), _stream(stream)))
    return logp_out


def grpo_sum_f64(v, n: int | None = None, out=None, stream=None):
    """Fixed-order fp64 sum of v[:n] on the GPU (the loss's own reduction)."""
    torch = _torch()
    _need(v, torch.float64, n, "v")
    if n is None:
        n = v.numel()
    if out is None:
        out = torch.empty(1, dtype=torch.float64, device=v.device)
    _check(lib().grpo_sum_f64(_ptr(v), int(n), _ptr(out), _stream(stream)))
    return out


def grpo_ars_init(G1: int) -> ArsState:
    st = ArsState()
    _check(lib().grpo_ars_init(ctypes.byref(st), G1))
    return st


def grpo_ars_serialize(state: ArsState) -> bytes:
    """The ARS state as its 64-byte checkpoint record (see the header)."""
    n = ctypes.c_size_t(0)
    _check(lib().grpo_ars_serialize(ctypes.byref(state), None, ctypes.byref(n)))
    buf = ctypes.create_string_buffer(n.value)
    _check(lib().grpo_ars_serialize(ctypes.byref(state), buf, ctypes.byref(n)))
    return buf.raw[:n.value]


def grpo_ars_deserialize(record: bytes) -> ArsState:
    """An ARS state restored from grpo_ars_serialize's record."""
    st = ArsState()
    buf = ctypes.create_string_buffer(bytes(record), len(record))
    _check(lib().grpo_ars_deserialize(ctypes.byref(st), buf, len(record)))
    return st


def adaptive_rollout_count(state: ArsState, kept_per_prompt, step: int, total_steps: int,
                           epoch_end: bool) -> int:
    """Eqs. 10-14 (host).  kept_per_prompt: host integers."""
    k = np.ascontiguousarray(np.asarray(kept_per_prompt), dtype=np.int32)
    n = lib().adaptive_rollout_count(ctypes.byref(state), k.ctypes.data_as(_c_p), k.size, step,
                                     total_steps, int(bool(epoch_end)))
    if n < 0:
        _check(-n)
    return int(n)


def check_status(status) -> int:
    """grpo_check_status on a device status word (a tensor, read back here, or an int): raises
    GrpoError (GRPO_ERR_TIMEOUT or GRPO_ERR_DEVICE_CHECK) if any bit is set; returns the word."""
    v = int(status.item()) if hasattr(status, "item") else int(status)
    _check(lib().grpo_check_status(ctypes.c_int32(v)))
    return v
