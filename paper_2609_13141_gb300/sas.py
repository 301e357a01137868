"""ctypes binding of the SAS C ABI (include/sas.h).

Argument marshalling only: every function here converts torch tensors to
device pointers, checks dtype/device/contiguity, and calls the entry point
of the same name in libsas.so.  No arithmetic of the method happens here, and
there is no fallback: if the library is missing or the device is not sm_103,
the calls raise.
"""
from __future__ import annotations

import ctypes
import os
import re

import torch

from . import _build

SAS_OK = 0
SAS_ERR_INVALID_ARG = 1
SAS_ERR_UNSUPPORTED = 2
SAS_ERR_CUDA = 3
SAS_ERR_TIMEOUT = 4
SAS_ERR_OOM = 5

SAS_MODE_TRAIN_SOFT = 0
SAS_MODE_INFER_HARD = 1
SAS_MODE_TRAIN_HARD_STE = 2
SAS_SEL_SCORES_GIVEN = 0
SAS_SEL_MEANPOOL_PROJ = 1
SAS_GATE_SOFTMAX = 0
SAS_GATE_SIGMOID = 1
SAS_GATE_LOGIT = 2
SAS_GATE_INNER = 0
SAS_GATE_OUTER = 1
SAS_SCOPE_SPARSE = 0
SAS_SCOPE_FULL = 1
SAS_NUM_KERNEL_KINDS = 7
KERNEL_KINDS = ["block_summaries", "query_projection", "selection", "attention", "mlp_up_gelu", "mlp_down",
                "attention_bwd"]

HEADER = os.path.join(_build.ROOT, "include", "sas.h")


class SasConfig(ctypes.Structure):
    _fields_ = [("B", ctypes.c_int32), ("H", ctypes.c_int32), ("N", ctypes.c_int32), ("d", ctypes.c_int32),
                ("block", ctypes.c_int32), ("topk", ctypes.c_int32), ("sm_scale", ctypes.c_float),
                ("mode", ctypes.c_int32), ("selector", ctypes.c_int32), ("d_sel", ctypes.c_int32),
                ("gate_act", ctypes.c_int32), ("gate_pos", ctypes.c_int32), ("Hkv", ctypes.c_int32),
                ("max_seqs", ctypes.c_int32), ("max_seqlen", ctypes.c_int32), ("scope", ctypes.c_int32)]


class SasDecodeConfig(ctypes.Structure):
    _fields_ = [("B", ctypes.c_int32), ("Hq", ctypes.c_int32), ("Hkv", ctypes.c_int32), ("d", ctypes.c_int32),
                ("d_sel", ctypes.c_int32), ("block", ctypes.c_int32), ("topk", ctypes.c_int32),
                ("max_blocks", ctypes.c_int32), ("num_pages", ctypes.c_int32), ("sm_scale", ctypes.c_float),
                ("dense", ctypes.c_int32)]


SAS_DECODE_NUM_KERNEL_KINDS = 4
DECODE_KERNEL_KINDS = ["prep", "select", "attention", "summarize"]


class SasError(RuntimeError):
    def __init__(self, status, message):
        super().__init__(f"{message} (status {status})")
        self.status = status


_lib = None


def lib():
    """Loads libsas.so (built in-tree by _build.build())."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(_build.LIB_PATH):
        raise RuntimeError("libsas.so is not built; run paper_2609_13141_gb300._build.build() first")
    L = ctypes.CDLL(_build.LIB_PATH)
    vp, i32, i64 = ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64
    L.sas_create.argtypes = [ctypes.POINTER(SasConfig), ctypes.POINTER(vp)]
    L.sas_create.restype = i32
    L.sas_destroy.argtypes = [vp]
    L.sas_destroy.restype = None
    L.sas_attention_fwd.argtypes = [vp] * 12
    L.sas_attention_fwd.restype = i32
    L.sas_attention_fwd_noisy.argtypes = [vp] * 13
    L.sas_attention_fwd_noisy.restype = i32
    L.sas_attention_fwd_varlen.argtypes = [vp, vp, i32] + [vp] * 11
    L.sas_attention_fwd_varlen.restype = i32
    L.sas_attention_bwd.argtypes = [vp] * 16
    L.sas_attention_bwd.restype = i32
    L.sas_mlp_fwd.argtypes = [vp] * 7 + [i64, i64, i64, vp]
    L.sas_mlp_fwd.restype = i32
    L.sas_status_str.argtypes = [i32]
    L.sas_status_str.restype = ctypes.c_char_p
    L.sas_last_error.argtypes = [vp]
    L.sas_last_error.restype = ctypes.c_char_p
    L.sas_get_device_status.argtypes = [vp, ctypes.POINTER(i32)]
    L.sas_get_device_status.restype = i32
    L.sas_set_timing.argtypes = [vp, i32]
    L.sas_set_timing.restype = i32
    L.sas_get_timings.argtypes = [vp, ctypes.POINTER(i64), ctypes.POINTER(ctypes.c_double), i32]
    L.sas_get_timings.restype = i32
    L.sas_launch_count.argtypes = [vp]
    L.sas_launch_count.restype = i64
    L.sas_set_wait_limit.argtypes = [vp, i64]
    L.sas_set_wait_limit.restype = i32
    L.sas_get_tile_union_counts.argtypes = [vp, ctypes.POINTER(i32), i64]
    L.sas_get_tile_union_counts.restype = i32
    L.sas_get_attention_work.argtypes = [vp, ctypes.POINTER(i64), ctypes.POINTER(i64)]
    L.sas_get_attention_work.restype = i32
    L.sas_mlp_fwd_noalloc.argtypes = [vp] * 6 + [i64, i64, i64, vp]
    L.sas_mlp_fwd_noalloc.restype = i32
    L.sas_mlp_noalloc_get_device_status.argtypes = [ctypes.POINTER(i32)]
    L.sas_mlp_noalloc_get_device_status.restype = i32
    L.sas_selftest_wait_timeout.argtypes = [i64, ctypes.POINTER(i32)]
    L.sas_selftest_wait_timeout.restype = i32
    L.sas_decode_create.argtypes = [ctypes.POINTER(SasDecodeConfig), ctypes.POINTER(vp)]
    L.sas_decode_create.restype = i32
    L.sas_decode_destroy.argtypes = [vp]
    L.sas_decode_destroy.restype = None
    L.sas_decode_summarize.argtypes = [vp] * 7
    L.sas_decode_summarize.restype = i32
    L.sas_decode_step.argtypes = [vp] * 15
    L.sas_decode_step.restype = i32
    L.sas_decode_last_error.argtypes = [vp]
    L.sas_decode_last_error.restype = ctypes.c_char_p
    L.sas_decode_get_device_status.argtypes = [vp, ctypes.POINTER(i32)]
    L.sas_decode_get_device_status.restype = i32
    L.sas_decode_set_timing.argtypes = [vp, i32]
    L.sas_decode_set_timing.restype = i32
    L.sas_decode_get_timings.argtypes = [vp, ctypes.POINTER(i64), ctypes.POINTER(ctypes.c_double), i32]
    L.sas_decode_get_timings.restype = i32
    L.sas_decode_launch_count.argtypes = [vp]
    L.sas_decode_launch_count.restype = i64
    _lib = L
    return L


def header_functions():
    """Names of the functions include/sas.h declares."""
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(sas_[a-z_]+)\s*\(", text)))


def _ptr(t, dtype, name, required=True):
    if t is None:
        if required:
            raise ValueError(f"{name} is required")
        return None
    if not isinstance(t, torch.Tensor) or t.device.type != "cuda":
        raise ValueError(f"{name} must be a CUDA tensor")
    if t.dtype != dtype:
        raise ValueError(f"{name} must be {dtype}, got {t.dtype}")
    if not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")
    return ctypes.c_void_p(t.data_ptr())


def _stream(stream):
    if stream is None:
        stream = torch.cuda.current_stream()
    return ctypes.c_void_p(stream.cuda_stream if hasattr(stream, "cuda_stream") else int(stream))


def _check(status, handle=None, what="sas"):
    if status != SAS_OK:
        L = lib()
        msg = L.sas_status_str(status).decode()
        if handle is not None:
            detail = L.sas_last_error(handle).decode()
            if detail:
                msg += ": " + detail
        raise SasError(status, f"{what}: {msg}")


def sas_status_str(status):
    return lib().sas_status_str(int(status)).decode()


def sas_create(B, H, N, d, topk, mode=SAS_MODE_TRAIN_SOFT, selector=SAS_SEL_SCORES_GIVEN, d_sel=0,
               sm_scale=0.0, block=64, gate_act=SAS_GATE_SOFTMAX, gate_pos=SAS_GATE_INNER, Hkv=0, max_seqs=0,
               max_seqlen=0, scope=SAS_SCOPE_SPARSE):
    cfg = SasConfig(B, H, N, d, block, topk, sm_scale, mode, selector, d_sel, gate_act, gate_pos, Hkv, max_seqs,
                    max_seqlen, scope)
    h = ctypes.c_void_p()
    _check(lib().sas_create(ctypes.byref(cfg), ctypes.byref(h)), None, "sas_create")
    return h


def sas_create_status(B, H, N, d, topk, mode=0, selector=0, d_sel=0, sm_scale=0.0, block=64,
                      gate_act=SAS_GATE_SOFTMAX, gate_pos=SAS_GATE_INNER, Hkv=0, max_seqs=0, max_seqlen=0,
                      scope=SAS_SCOPE_SPARSE):
    """Raw status of sas_create (for argument-check tests); destroys the handle on success."""
    cfg = SasConfig(B, H, N, d, block, topk, sm_scale, mode, selector, d_sel, gate_act, gate_pos, Hkv, max_seqs,
                    max_seqlen, scope)
    h = ctypes.c_void_p()
    st = lib().sas_create(ctypes.byref(cfg), ctypes.byref(h))
    if st == SAS_OK:
        lib().sas_destroy(h)
    return st


def sas_destroy(h):
    lib().sas_destroy(h)


def sas_attention_fwd_varlen(h, cu_seqlens, Q, K, V, scores, O, LSE=None, sel_idx=None, sel_logg=None,
                             stream=None, Wq=None, Wk=None):
    bf = torch.bfloat16
    st = lib().sas_attention_fwd_varlen(
        h, _ptr(cu_seqlens, torch.int32, "cu_seqlens"), ctypes.c_int32(cu_seqlens.numel() - 1),
        _ptr(Q, bf, "Q"), _ptr(K, bf, "K"), _ptr(V, bf, "V"), _ptr(scores, torch.float32, "scores", False),
        _ptr(Wq, bf, "Wq", False), _ptr(Wk, bf, "Wk", False), _ptr(O, bf, "O"), _ptr(LSE, torch.float32, "LSE", False), _ptr(sel_idx, torch.int32, "sel_idx", False),
        _ptr(sel_logg, torch.float32, "sel_logg", False), _stream(stream))
    _check(st, h, "sas_attention_fwd_varlen")


def sas_attention_fwd(h, Q, K, V, O, scores=None, Wq=None, Wk=None, LSE=None, sel_idx=None, sel_logg=None,
                      stream=None):
    bf = torch.bfloat16
    st = lib().sas_attention_fwd(
        h, _ptr(Q, bf, "Q"), _ptr(K, bf, "K"), _ptr(V, bf, "V"),
        _ptr(scores, torch.float32, "scores", False), _ptr(Wq, bf, "Wq", False), _ptr(Wk, bf, "Wk", False),
        _ptr(O, bf, "O"), _ptr(LSE, torch.float32, "LSE", False), _ptr(sel_idx, torch.int32, "sel_idx", False),
        _ptr(sel_logg, torch.float32, "sel_logg", False), _stream(stream))
    _check(st, h, "sas_attention_fwd")


def sas_attention_fwd_noisy(h, Q, K, V, O, noise, scores=None, Wq=None, Wk=None, LSE=None, sel_idx=None,
                            sel_logg=None, stream=None):
    bf = torch.bfloat16
    st = lib().sas_attention_fwd_noisy(
        h, _ptr(Q, bf, "Q"), _ptr(K, bf, "K"), _ptr(V, bf, "V"),
        _ptr(scores, torch.float32, "scores", False), _ptr(Wq, bf, "Wq", False), _ptr(Wk, bf, "Wk", False),
        _ptr(noise, torch.float32, "noise"), _ptr(O, bf, "O"), _ptr(LSE, torch.float32, "LSE", False),
        _ptr(sel_idx, torch.int32, "sel_idx", False), _ptr(sel_logg, torch.float32, "sel_logg", False),
        _stream(stream))
    _check(st, h, "sas_attention_fwd_noisy")


def sas_attention_bwd(h, Q, K, V, O, LSE, dO, dQ, dK, dV, scores=None, sel_idx=None, sel_logg=None, dlogg=None,
                      dscores=None, stream=None):
    bf, f32 = torch.bfloat16, torch.float32
    st = lib().sas_attention_bwd(
        h, _ptr(Q, bf, "Q"), _ptr(K, bf, "K"), _ptr(V, bf, "V"), _ptr(scores, f32, "scores", False),
        _ptr(O, bf, "O"), _ptr(LSE, f32, "LSE"), _ptr(dO, bf, "dO"), _ptr(sel_idx, torch.int32, "sel_idx", False),
        _ptr(sel_logg, f32, "sel_logg", False), _ptr(dQ, bf, "dQ"), _ptr(dK, bf, "dK"), _ptr(dV, bf, "dV"),
        _ptr(dlogg, f32, "dlogg", False), _ptr(dscores, f32, "dscores", False), _stream(stream))
    _check(st, h, "sas_attention_bwd")


def sas_mlp_fwd(h, X, W1, W2, Y, b1=None, b2=None, stream=None):
    bf = torch.bfloat16
    T, D = X.shape
    F = W1.shape[0]
    st = lib().sas_mlp_fwd(h, _ptr(X, bf, "X"), _ptr(W1, bf, "W1"), _ptr(b1, bf, "b1", False), _ptr(W2, bf, "W2"),
                           _ptr(b2, bf, "b2", False), _ptr(Y, bf, "Y"), T, D, F, _stream(stream))
    _check(st, h, "sas_mlp_fwd")


SAS_MLP_NOALLOC_MAX_HIDDEN_BYTES = 32 * 1024 * 1024


def sas_mlp_fwd_noalloc(X, W1, W2, Y, b1=None, b2=None, stream=None):
    """The MLP without a handle and without any device allocation (see sas.h):
    the hidden activation lives in a fixed 32 MiB array inside the library,
    shared by every call on the device."""
    bf = torch.bfloat16
    T, D = X.shape
    F = W1.shape[0]
    st = lib().sas_mlp_fwd_noalloc(_ptr(X, bf, "X"), _ptr(W1, bf, "W1"), _ptr(b1, bf, "b1", False),
                                   _ptr(W2, bf, "W2"), _ptr(b2, bf, "b2", False), _ptr(Y, bf, "Y"), T, D, F,
                                   _stream(stream))
    if st == SAS_ERR_UNSUPPORTED and T * F * 2 > SAS_MLP_NOALLOC_MAX_HIDDEN_BYTES:
        raise SasError(st, f"sas_mlp_fwd_noalloc: hidden activation of {T}x{F} bf16 ({T * F * 2} bytes) exceeds "
                           f"the fixed {SAS_MLP_NOALLOC_MAX_HIDDEN_BYTES}-byte array")
    _check(st, None, "sas_mlp_fwd_noalloc")


def sas_mlp_noalloc_get_device_status():
    """Reads and clears the status word of sas_mlp_fwd_noalloc on the current
    device (synchronises the device)."""
    v = ctypes.c_int32(-1)
    _check(lib().sas_mlp_noalloc_get_device_status(ctypes.byref(v)), None, "sas_mlp_noalloc_get_device_status")
    return v.value


def sas_get_device_status(h):
    v = ctypes.c_int32(0)
    _check(lib().sas_get_device_status(h, ctypes.byref(v)), h, "sas_get_device_status")
    return v.value


def sas_set_timing(h, enable):
    _check(lib().sas_set_timing(h, 1 if enable else 0), h, "sas_set_timing")


def sas_get_timings(h):
    """{kind: (launches, total_ms)} for the kernel kinds of sas.h."""
    n = SAS_NUM_KERNEL_KINDS
    launches = (ctypes.c_int64 * n)()
    ms = (ctypes.c_double * n)()
    _check(lib().sas_get_timings(h, launches, ms, n), h, "sas_get_timings")
    return {KERNEL_KINDS[k]: (launches[k], ms[k]) for k in range(n)}


def sas_launch_count(h):
    return lib().sas_launch_count(h)


def sas_set_wait_limit(h, cycles):
    """Failure-path diagnostics: main-loop wait budget in SM cycles (0: default)."""
    _check(lib().sas_set_wait_limit(h, int(cycles)), h, "sas_set_wait_limit")


def sas_get_tile_union_counts(h, n):
    out = (ctypes.c_int32 * n)()
    _check(lib().sas_get_tile_union_counts(h, out, n), h, "sas_get_tile_union_counts")
    return list(out)


def sas_get_attention_work(h):
    """(tiles, tile_blocks) of the last attention forward (see sas.h)."""
    t, b = ctypes.c_int64(0), ctypes.c_int64(0)
    _check(lib().sas_get_attention_work(h, ctypes.byref(t), ctypes.byref(b)), h, "sas_get_attention_work")
    return t.value, b.value


def sas_selftest_wait_timeout(limit_cycles):
    v = ctypes.c_int32(-1)
    _check(lib().sas_selftest_wait_timeout(int(limit_cycles), ctypes.byref(v)), None, "sas_selftest_wait_timeout")
    return v.value


class SasLayer:
    """Owns one handle; allocates outputs and calls the C ABI."""

    def __init__(self, B, H, N, d, topk, mode=SAS_MODE_TRAIN_SOFT, selector=SAS_SEL_SCORES_GIVEN, d_sel=0,
                 sm_scale=0.0, gate_act=SAS_GATE_SOFTMAX, gate_pos=SAS_GATE_INNER, Hkv=0, max_seqs=0, max_seqlen=0,
                 scope=SAS_SCOPE_SPARSE):
        self.B, self.H, self.N, self.d, self.topk = B, H, N, d, topk
        self.mode = mode
        self.Hkv = Hkv or H                      # kept lists are per KV group
        self.selector = selector
        self.scope = scope
        self.h = sas_create(B, H, N, d, topk, mode, selector, d_sel, sm_scale, 64, gate_act, gate_pos, Hkv,
                            max_seqs, max_seqlen, scope)

    def attention_varlen(self, cu_seqlens, Q, K, V, scores=None, want_sel=True, stream=None, sel_fill=-1, Wq=None,
                         Wk=None):
        """Packed sequences (handle made with max_seqs > 0): Q [H, N, d], K/V [Hkv, N, d],
        scores [Hkv, N, C] (or the learned selector's Wq, Wk), cu_seqlens int32 on the
        device.  The library does not write rows past cu[-1]: they keep the fill of
        the tensors made here (0, and sel_fill in sel_idx)."""
        dev = Q.device
        O = torch.zeros_like(Q)
        LSE = torch.zeros(self.H, self.N, device=dev, dtype=torch.float32)
        sel_idx = sel_logg = None
        if want_sel:
            k = max(self.topk, 1)
            sel_idx = torch.full((self.Hkv, self.N, k), sel_fill, device=dev, dtype=torch.int32)
            sel_logg = torch.zeros(self.Hkv, self.N, k, device=dev, dtype=torch.float32)
        sas_attention_fwd_varlen(self.h, cu_seqlens, Q, K, V, scores, O, LSE, sel_idx, sel_logg, stream, Wq, Wk)
        return O, LSE, sel_idx, sel_logg

    def _outputs(self, Q, want_sel):
        dev = Q.device
        O = torch.empty_like(Q)
        LSE = torch.empty(self.B, self.H, self.N, device=dev, dtype=torch.float32)
        sel_idx = sel_logg = None
        if want_sel and self.scope == SAS_SCOPE_SPARSE:
            k = max(self.topk, 1)
            sel_idx = torch.empty(self.B, self.Hkv, self.N, k, device=dev, dtype=torch.int32)
            sel_logg = torch.empty(self.B, self.Hkv, self.N, k, device=dev, dtype=torch.float32)
        return O, LSE, sel_idx, sel_logg

    def attention(self, Q, K, V, scores=None, Wq=None, Wk=None, want_sel=True, stream=None):
        """Returns (O, LSE, sel_idx, sel_logg); the full scope keeps no Top-K (sel_* None)."""
        O, LSE, sel_idx, sel_logg = self._outputs(Q, want_sel)
        sas_attention_fwd(self.h, Q, K, V, O, scores, Wq, Wk, LSE, sel_idx, sel_logg, stream)
        return O, LSE, sel_idx, sel_logg

    def attention_noisy(self, Q, K, V, noise, scores=None, Wq=None, Wk=None, want_sel=True, stream=None):
        """full*: the scores plus `noise` (fp32, the layout of given scores) choose and gate the blocks."""
        O, LSE, sel_idx, sel_logg = self._outputs(Q, want_sel)
        sas_attention_fwd_noisy(self.h, Q, K, V, O, noise, scores, Wq, Wk, LSE, sel_idx, sel_logg, stream)
        return O, LSE, sel_idx, sel_logg

    def attention_bwd(self, Q, K, V, O, LSE, dO, scores=None, sel_idx=None, sel_logg=None, want_ds=False,
                      stream=None):
        """Returns (dQ, dK, dV, dlogg, dscores); dscores only with want_ds (given scores).
        With Hkv < H, dK, dV, dlogg and dscores are per KV group (sums over its heads).
        The full scope and the hard-STE mode report dlogg for every block: [B, Hkv, N, C]."""
        dQ, dK, dV = torch.empty_like(Q), torch.empty_like(K), torch.empty_like(V)
        C = -(-self.N // 64)
        width = C if (self.scope == SAS_SCOPE_FULL or self.mode == SAS_MODE_TRAIN_HARD_STE) else max(self.topk, 1)
        dlogg = torch.empty(self.B, self.Hkv, self.N, width, device=Q.device, dtype=torch.float32)
        ds = None
        if want_ds:
            ds = torch.empty(self.B, self.Hkv, self.N, -(-self.N // 64), device=Q.device, dtype=torch.float32)
        sas_attention_bwd(self.h, Q, K, V, O, LSE, dO, dQ, dK, dV, scores, sel_idx, sel_logg, dlogg, ds, stream)
        return dQ, dK, dV, dlogg, ds

    def attention_bwd_varlen(self, Q, K, V, O, LSE, dO, scores=None, sel_idx=None, sel_logg=None, want_ds=False,
                             stream=None):
        """Backward of the last attention_varlen on this handle: Q, O, dO [H, N, d],
        K, V [Hkv, N, d].  Returns (dQ, dK, dV, dlogg [Hkv, N, topk], dscores [Hkv, N, C]
        or None); rows past cu[-1] keep the zero fill of the tensors made here."""
        dev = Q.device
        dQ, dK, dV = torch.zeros_like(Q), torch.zeros_like(K), torch.zeros_like(V)
        dlogg = torch.zeros(self.Hkv, self.N, max(self.topk, 1), device=dev, dtype=torch.float32)
        ds = None
        if want_ds:
            ds = torch.zeros(self.Hkv, self.N, scores.shape[-1], device=dev, dtype=torch.float32)
        sas_attention_bwd(self.h, Q, K, V, O, LSE, dO, dQ, dK, dV, scores, sel_idx, sel_logg, dlogg, ds, stream)
        return dQ, dK, dV, dlogg, ds

    def mlp(self, X, W1, W2, b1=None, b2=None, stream=None):
        Y = torch.empty(X.shape[0], W2.shape[0], device=X.device, dtype=torch.bfloat16)
        sas_mlp_fwd(self.h, X, W1, W2, Y, b1, b2, stream)
        return Y

    def close(self):
        if self.h is not None:
            sas_destroy(self.h)
            self.h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


# ------------------------------------------------------------------ decode


def _dcheck(status, handle, what):
    if status != SAS_OK:
        L = lib()
        msg = L.sas_status_str(status).decode()
        if handle is not None:
            detail = L.sas_decode_last_error(handle).decode()
            if detail:
                msg += ": " + detail
        raise SasError(status, f"{what}: {msg}")


def sas_decode_create(B, Hq, Hkv, d, topk, max_blocks, num_pages, d_sel=0, sm_scale=0.0, dense=False, block=64):
    cfg = SasDecodeConfig(B, Hq, Hkv, d, d_sel, block, topk, max_blocks, num_pages, sm_scale, 1 if dense else 0)
    h = ctypes.c_void_p()
    _dcheck(lib().sas_decode_create(ctypes.byref(cfg), ctypes.byref(h)), None, "sas_decode_create")
    return h


def sas_decode_create_status(B, Hq, Hkv, d, topk, max_blocks, num_pages, d_sel=0, sm_scale=0.0, dense=0, block=64):
    """Raw status of sas_decode_create (argument-check tests); destroys the handle on success."""
    cfg = SasDecodeConfig(B, Hq, Hkv, d, d_sel, block, topk, max_blocks, num_pages, sm_scale, dense)
    h = ctypes.c_void_p()
    st = lib().sas_decode_create(ctypes.byref(cfg), ctypes.byref(h))
    if st == SAS_OK:
        lib().sas_decode_destroy(h)
    return st


def sas_decode_destroy(h):
    lib().sas_decode_destroy(h)


def sas_decode_summarize(h, K_cache, block_table, seq_lens, Wk, Ksum, stream=None):
    bf, i32 = torch.bfloat16, torch.int32
    st = lib().sas_decode_summarize(h, _ptr(K_cache, bf, "K_cache"), _ptr(block_table, i32, "block_table"),
                                    _ptr(seq_lens, i32, "seq_lens"), _ptr(Wk, bf, "Wk"), _ptr(Ksum, bf, "Ksum"),
                                    _stream(stream))
    _dcheck(st, h, "sas_decode_summarize")


def sas_decode_step(h, q, K_cache, V_cache, block_table, seq_lens, O, k_new=None, v_new=None, Wq=None, Wk=None,
                    Ksum=None, LSE=None, sel_idx=None, stream=None):
    bf, i32 = torch.bfloat16, torch.int32
    st = lib().sas_decode_step(
        h, _ptr(q, bf, "q"), _ptr(k_new, bf, "k_new", False), _ptr(v_new, bf, "v_new", False),
        _ptr(K_cache, bf, "K_cache"), _ptr(V_cache, bf, "V_cache"), _ptr(block_table, i32, "block_table"),
        _ptr(seq_lens, i32, "seq_lens"), _ptr(Wq, bf, "Wq", False), _ptr(Wk, bf, "Wk", False),
        _ptr(Ksum, bf, "Ksum", False), _ptr(O, bf, "O"), _ptr(LSE, torch.float32, "LSE", False),
        _ptr(sel_idx, i32, "sel_idx", False), _stream(stream))
    _dcheck(st, h, "sas_decode_step")


def sas_decode_get_device_status(h):
    v = ctypes.c_int32(0)
    _dcheck(lib().sas_decode_get_device_status(h, ctypes.byref(v)), h, "sas_decode_get_device_status")
    return v.value


def sas_decode_set_timing(h, enable):
    _dcheck(lib().sas_decode_set_timing(h, 1 if enable else 0), h, "sas_decode_set_timing")


def sas_decode_get_timings(h):
    n = SAS_DECODE_NUM_KERNEL_KINDS
    launches = (ctypes.c_int64 * n)()
    ms = (ctypes.c_double * n)()
    _dcheck(lib().sas_decode_get_timings(h, launches, ms, n), h, "sas_decode_get_timings")
    return {DECODE_KERNEL_KINDS[k]: (launches[k], ms[k]) for k in range(n)}


def sas_decode_launch_count(h):
    return lib().sas_decode_launch_count(h)


class SasDecoder:
    """Owns one decode handle; allocates the step's outputs and calls the C ABI."""

    def __init__(self, B, Hq, Hkv, d, topk, max_blocks, num_pages, d_sel=0, sm_scale=0.0, dense=False):
        self.B, self.Hq, self.Hkv, self.d, self.topk = B, Hq, Hkv, d, topk
        self.dense = dense
        self.h = sas_decode_create(B, Hq, Hkv, d, topk, max_blocks, num_pages, d_sel, sm_scale, dense)

    def summarize(self, K_cache, block_table, seq_lens, Wk, Ksum, stream=None):
        sas_decode_summarize(self.h, K_cache, block_table, seq_lens, Wk, Ksum, stream)

    def step(self, q, K_cache, V_cache, block_table, seq_lens, k_new=None, v_new=None, Wq=None, Wk=None, Ksum=None,
             out=None, stream=None):
        """Returns (O, LSE, sel_idx); sel_idx is None in dense mode.  out = (O, LSE, sel_idx)
        reuses caller buffers (as a captured graph needs)."""
        if out is None:
            O = torch.empty(self.B, self.Hq, self.d, device=q.device, dtype=torch.bfloat16)
            LSE = torch.empty(self.B, self.Hq, device=q.device, dtype=torch.float32)
            sel = None if self.dense else torch.empty(self.B, self.Hkv, max(self.topk, 1), device=q.device,
                                                      dtype=torch.int32)
        else:
            O, LSE, sel = out
        sas_decode_step(self.h, q, K_cache, V_cache, block_table, seq_lens, O, k_new, v_new, Wq, Wk, Ksum, LSE,
                        sel, stream)
        return O, LSE, sel

    def close(self):
        if self.h is not None:
            sas_decode_destroy(self.h)
            self.h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass
