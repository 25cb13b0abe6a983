"""ctypes binding of libjab.so (include/jab.h). Argument marshalling only.

Each function has the name of its C entry point, takes torch tensors where the C function takes
device pointers, checks dtype / device / contiguity (the C side checks shapes, alignment and
workspace size), calls the library on the current CUDA stream (or the one given), and raises
JabError on a non-OK status.
"""
from __future__ import annotations

import ctypes
import os
from typing import Optional, Sequence

import torch

JAB_OK = 0
_STATUS_NAMES = {0: "JAB_OK", 1: "JAB_ERR_INVALID_ARG", 2: "JAB_ERR_UNSUPPORTED", 3: "JAB_ERR_CUDA",
                 4: "JAB_ERR_NONFINITE", 5: "JAB_ERR_RANGE", 6: "JAB_ERR_TIMEOUT",
                 7: "JAB_ERR_SCRATCH_LIMIT", 8: "JAB_ERR_INTERNAL", 9: "JAB_ERR_DEVICE_ASSERT"}

_HERE = os.path.dirname(os.path.abspath(__file__))


def lib_path() -> str:
    """libjab.so, or the checked build libjab_checked.so when the environment sets JAB_CHECKED=1."""
    name = "libjab_checked.so" if os.environ.get("JAB_CHECKED", "0") == "1" else "libjab.so"
    return os.path.join(_HERE, name)


class JabError(RuntimeError):
    def __init__(self, status: int, where: str):
        self.status = int(status)
        super().__init__(f"{where}: {_STATUS_NAMES.get(self.status, self.status)} "
                         f"({jab_status_string(self.status)})")


class BlockDesc(ctypes.Structure):
    """jab_block_desc: one attention block (Section 2.1; App. C)."""

    _fields_ = [("d_model", ctypes.c_int32), ("n_q_heads", ctypes.c_int32),
                ("n_kv_heads", ctypes.c_int32), ("head_dim", ctypes.c_int32),
                ("group_size", ctypes.c_int32), ("use_rope", ctypes.c_int32),
                ("rope_theta", ctypes.c_float), ("softmax_scale", ctypes.c_float)]

    def as_dict(self) -> dict:
        return {name: getattr(self, name) for name, _ in self._fields_}


def desc_from_shape(shape, group_size: int) -> BlockDesc:
    """BlockDesc from a workloads.BlockShape-like object (d_model, heads, head_dim, RoPE)."""
    return BlockDesc(shape.d_model, shape.n_q_heads, shape.n_kv_heads, shape.head_dim, group_size,
                     1 if shape.use_rope else 0, float(shape.rope_theta), 0.0)


_P = ctypes.c_void_p
_LIB = None


def lib() -> ctypes.CDLL:
    """Loads libjab.so; raises if it has not been built (there is no fallback)."""
    global _LIB
    if _LIB is not None:
        return _LIB
    path = lib_path()
    if not os.path.exists(path):
        raise RuntimeError(f"{path} is missing: build it with `python -m paper_2609_34866_gb300.build` "
                           "or __graft_entry__.build()")
    L = ctypes.CDLL(path)
    D = ctypes.POINTER(BlockDesc)
    i32, f32, sz = ctypes.c_int32, ctypes.c_float, ctypes.c_size_t
    L.jab_workspace_size.argtypes = [D, i32, i32, i32, i32]
    L.jab_workspace_size.restype = sz
    L.jab_reference_forward.argtypes = [D, i32, i32, _P, _P, _P, _P, _P, _P, sz, _P]
    L.jab_loss_forward.argtypes = [D, i32, i32, _P, _P, _P, i32, ctypes.POINTER(i32),
                                   ctypes.POINTER(_P), _P, _P, _P, sz, _P]
    L.jab_loss_forward_noalloc.argtypes = [D, i32, i32, _P, _P, _P, i32, ctypes.POINTER(i32),
                                           ctypes.POINTER(_P), _P, _P, _P]
    L.jab_loss_backward_scales.argtypes = [D, i32, i32, _P, _P, _P, i32, _P, f32, _P, _P, _P, sz, _P]
    L.jab_loss_backward_weights.argtypes = [D, i32, i32, _P, _P, _P, i32, _P, _P, _P, _P, _P, sz, _P]
    L.jab_prepare_x.argtypes = [D, i32, i32, _P, _P, sz, _P]
    L.jab_loss_backward_scales_prepared.argtypes = [D, i32, i32, _P, _P, _P, i32, _P, f32, _P, _P,
                                                    _P, sz, _P]
    L.jab_loss_backward_scales_kl.argtypes = [D, i32, i32, _P, _P, _P, _P, _P, i32, _P, f32, f32,
                                              _P, _P, _P, _P, sz, _P]
    L.jab_flip_rate.argtypes = [_P, _P, ctypes.c_int64, _P, _P]
    L.jab_reference_projection.argtypes = [D, i32, i32, _P, _P, _P, _P, sz, _P]
    L.jab_hutchinson_trace.argtypes = [D, i32, i32, _P, _P, _P, _P, i32, ctypes.c_uint64, _P, _P,
                                       _P, sz, _P]
    L.jab_rademacher_probes.argtypes = [ctypes.c_uint64, ctypes.c_int64, ctypes.c_int64, _P, _P]
    L.jab_omega_scores.argtypes = [D, _P, i32, ctypes.POINTER(i32), ctypes.POINTER(_P), _P, i32,
                                   _P, _P, _P, sz, _P]
    L.jab_loss_forward_kl.argtypes = [D, i32, i32, _P, _P, _P, _P, i32, ctypes.POINTER(i32),
                                      ctypes.POINTER(_P), f32, _P, _P, _P, _P, _P, sz, _P]
    L.jab_quantize.argtypes = [D, i32, _P, _P, _P, _P, _P]
    L.jab_allocate_bits.argtypes = [_P, _P, _P, i32, i32, ctypes.c_double, i32, _P]
    L.jab_init_scales.argtypes = [D, i32, i32, _P, _P, _P]
    L.jab_get_device_status.argtypes = [_P]
    L.jab_set_deterministic.argtypes = [i32]
    L.jab_selftest_bounds_check.argtypes = [_P, i32, _P]
    L.jab_selftest_wait_timeout.argtypes = [_P]
    L.jab_status_string.argtypes = [i32]
    L.jab_status_string.restype = ctypes.c_char_p
    L.jab_timing_enable.argtypes = [i32]
    L.jab_timing_collect.argtypes = []
    L.jab_timing_count.argtypes = []
    L.jab_timing_count.restype = i32
    L.jab_timing_get.argtypes = [i32, ctypes.POINTER(ctypes.c_char_p), ctypes.POINTER(ctypes.c_double),
                                 ctypes.POINTER(ctypes.c_int64), ctypes.POINTER(ctypes.c_int64)]
    L.jab_timing_reset.argtypes = []
    for fn in ("jab_reference_forward", "jab_loss_forward", "jab_loss_forward_noalloc",
               "jab_loss_backward_scales", "jab_loss_backward_weights", "jab_allocate_bits",
               "jab_prepare_x", "jab_loss_backward_scales_prepared", "jab_flip_rate",
               "jab_loss_backward_scales_kl",
               "jab_reference_projection", "jab_loss_forward_kl", "jab_hutchinson_trace",
               "jab_omega_scores", "jab_rademacher_probes",
               "jab_quantize", "jab_init_scales", "jab_get_device_status", "jab_timing_enable",
               "jab_selftest_wait_timeout", "jab_set_deterministic", "jab_selftest_bounds_check",
               "jab_timing_collect", "jab_timing_get", "jab_timing_reset"):
        getattr(L, fn).restype = i32
    _LIB = L
    return L


def jab_status_string(status: int) -> str:
    try:
        return lib().jab_status_string(int(status)).decode()
    except RuntimeError:
        return _STATUS_NAMES.get(int(status), "unknown")


def _ptr(t: Optional[torch.Tensor], dtype=None, name="tensor") -> Optional[int]:
    if t is None:
        return None
    if not t.is_cuda:
        raise ValueError(f"{name} must be a CUDA tensor")
    if dtype is not None and t.dtype != dtype:
        raise ValueError(f"{name} must be {dtype}, got {t.dtype}")
    if not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")
    return t.data_ptr()


def _stream(stream) -> Optional[int]:
    if stream is None:
        stream = torch.cuda.current_stream()
    return stream.cuda_stream if hasattr(stream, "cuda_stream") else int(stream)


def _check(status: int, where: str):
    if status != JAB_OK:
        raise JabError(status, where)


def jab_workspace_size(desc: BlockDesc, B: int, T: int, n_cand: int = 1, with_bwd: bool = True) -> int:
    return int(lib().jab_workspace_size(ctypes.byref(desc), B, T, n_cand, 1 if with_bwd else 0))


class Workspace:
    """A caller-owned device workspace (a uint8 torch tensor) sized by jab_workspace_size."""

    def __init__(self, desc: BlockDesc, B: int, T: int, n_cand: int = 1, with_bwd: bool = True,
                 device=None):
        self.nbytes = jab_workspace_size(desc, B, T, n_cand, with_bwd)
        if self.nbytes == 0:
            raise JabError(1, "jab_workspace_size")
        self.buf = torch.empty(self.nbytes, dtype=torch.uint8,
                               device=device or torch.device("cuda", torch.cuda.current_device()))

    @property
    def ptr(self) -> int:
        return self.buf.data_ptr()


def jab_reference_forward(desc, B, T, X, W, A_ref, ws: Workspace, lse=None, a_sqnorm=None,
                          stream=None):
    st = lib().jab_reference_forward(
        ctypes.byref(desc), B, T, _ptr(X, torch.bfloat16, "X"), _ptr(W, torch.bfloat16, "W"),
        _ptr(A_ref, torch.float32, "A_ref"), _ptr(lse, torch.float32, "lse"),
        _ptr(a_sqnorm, torch.float64, "a_sqnorm"), ws.ptr, ws.nbytes, _stream(stream))
    _check(st, "jab_reference_forward")


def jab_loss_forward(desc, B, T, X, W, A_ref, bits: Sequence[int], scales: Sequence[torch.Tensor],
                     loss, ws: Workspace, sse_parts=None, stream=None):
    n = len(bits)
    if len(scales) != n:
        raise ValueError("bits and scales must have the same length")
    bits_arr = (ctypes.c_int32 * n)(*[int(b) for b in bits])
    sc_arr = (ctypes.c_void_p * n)(*[_ptr(s, torch.float32, "scales") for s in scales])
    st = lib().jab_loss_forward(
        ctypes.byref(desc), B, T, _ptr(X, torch.bfloat16, "X"), _ptr(W, torch.bfloat16, "W"),
        _ptr(A_ref, torch.float32, "A_ref"), n, bits_arr, sc_arr,
        _ptr(loss, torch.float64, "loss"), _ptr(sse_parts, torch.float64, "sse_parts"), ws.ptr,
        ws.nbytes, _stream(stream))
    _check(st, "jab_loss_forward")


def jab_reference_projection(desc, B, T, X, W, QKV_ref, ws: Workspace, stream=None):
    """Teacher [Q|K|V] (rotated, fp16 [B, T, D]) for the KL term."""
    st = lib().jab_reference_projection(
        ctypes.byref(desc), B, T, _ptr(X, torch.bfloat16, "X"), _ptr(W, torch.bfloat16, "W"),
        _ptr(QKV_ref, torch.float16, "QKV_ref"), ws.ptr, ws.nbytes, _stream(stream))
    _check(st, "jab_reference_projection")


def jab_loss_forward_kl(desc, B, T, X, W, A_ref, QKV_ref, bits: Sequence[int],
                        scales: Sequence[torch.Tensor], lambda_kl: float, loss, ws: Workspace,
                        mse=None, kl=None, kl_rows=None, stream=None):
    """Both terms of Eq. 3 per candidate: loss = mse + lambda_kl * kl (fp64 [n_cand] each)."""
    n = len(bits)
    if len(scales) != n:
        raise ValueError("bits and scales must have the same length")
    bits_arr = (ctypes.c_int32 * n)(*[int(b) for b in bits])
    sc_arr = (ctypes.c_void_p * n)(*[_ptr(s, torch.float32, "scales") for s in scales])
    st = lib().jab_loss_forward_kl(
        ctypes.byref(desc), B, T, _ptr(X, torch.bfloat16, "X"), _ptr(W, torch.bfloat16, "W"),
        _ptr(A_ref, torch.float32, "A_ref"), _ptr(QKV_ref, torch.float16, "QKV_ref"), n, bits_arr,
        sc_arr, float(lambda_kl), _ptr(loss, torch.float64, "loss"), _ptr(mse, torch.float64, "mse"),
        _ptr(kl, torch.float64, "kl"), _ptr(kl_rows, torch.float32, "kl_rows"), ws.ptr, ws.nbytes,
        _stream(stream))
    _check(st, "jab_loss_forward_kl")


def jab_hutchinson_trace(desc, B, T, X, W, A_ref, lse_ref, n_probes: int, seed: int, trace,
                         ws: Workspace, vhv=None, stream=None):
    """Tr(H) of L_JAB at the float weights from n_probes Rademacher probes (Section 2.4, Eq. 5)."""
    st = lib().jab_hutchinson_trace(
        ctypes.byref(desc), B, T, _ptr(X, torch.bfloat16, "X"), _ptr(W, torch.bfloat16, "W"),
        _ptr(A_ref, torch.float32, "A_ref"), _ptr(lse_ref, torch.float32, "lse_ref"), int(n_probes),
        int(seed) & ((1 << 64) - 1), _ptr(trace, torch.float64, "trace"),
        _ptr(vhv, torch.float64, "vhv"), ws.ptr, ws.nbytes, _stream(stream))
    _check(st, "jab_hutchinson_trace")


def jab_rademacher_probes(seed: int, first: int, out, stream=None):
    """Probe entries first .. first + out.numel() - 1 of jab_hutchinson_trace's sequence (fp16 +-1)."""
    st = lib().jab_rademacher_probes(int(seed) & ((1 << 64) - 1), int(first), int(out.numel()),
                                     _ptr(out, torch.float16, "out"), _stream(stream))
    _check(st, "jab_rademacher_probes")


def jab_omega_scores(desc, W, bits: Sequence[int], scales: Sequence[torch.Tensor], trace,
                     layers_after: int, c1, ws: Workspace, c2=None, stream=None):
    """Eq. 6: C1 = Tr(H) ||Q_b(W) - W||^2 per candidate (and C2 = layers_after * C1)."""
    n = len(bits)
    if len(scales) != n:
        raise ValueError("bits and scales must have the same length")
    bits_arr = (ctypes.c_int32 * n)(*[int(b) for b in bits])
    sc_arr = (ctypes.c_void_p * n)(*[_ptr(s, torch.float32, "scales") for s in scales])
    st = lib().jab_omega_scores(ctypes.byref(desc), _ptr(W, torch.bfloat16, "W"), n, bits_arr,
                                sc_arr, _ptr(trace, torch.float64, "trace"), int(layers_after),
                                _ptr(c1, torch.float64, "c1"), _ptr(c2, torch.float64, "c2"),
                                ws.ptr, ws.nbytes, _stream(stream))
    _check(st, "jab_omega_scores")


def jab_loss_forward_noalloc(desc, B, T, X, W, A_ref, bits: Sequence[int],
                             scales: Sequence[torch.Tensor], loss, sse_parts=None, stream=None):
    """jab_loss_forward on the library's fixed device scratch (no workspace argument): for callers
    that cannot allocate device memory. Raises JabError(JAB_ERR_SCRATCH_LIMIT) when the problem
    needs more scratch than JAB_NOALLOC_SCRATCH_BYTES."""
    n = len(bits)
    if len(scales) != n:
        raise ValueError("bits and scales must have the same length")
    bits_arr = (ctypes.c_int32 * n)(*[int(b) for b in bits])
    sc_arr = (ctypes.c_void_p * n)(*[_ptr(s, torch.float32, "scales") for s in scales])
    st = lib().jab_loss_forward_noalloc(
        ctypes.byref(desc), B, T, _ptr(X, torch.bfloat16, "X"), _ptr(W, torch.bfloat16, "W"),
        _ptr(A_ref, torch.float32, "A_ref"), n, bits_arr, sc_arr,
        _ptr(loss, torch.float64, "loss"), _ptr(sse_parts, torch.float64, "sse_parts"),
        _stream(stream))
    _check(st, "jab_loss_forward_noalloc")


def jab_loss_backward_scales(desc, B, T, X, W, A_ref, bits: int, scales, kappa: float, loss,
                             grad_scales, ws: Workspace, stream=None):
    st = lib().jab_loss_backward_scales(
        ctypes.byref(desc), B, T, _ptr(X, torch.bfloat16, "X"), _ptr(W, torch.bfloat16, "W"),
        _ptr(A_ref, torch.float32, "A_ref"), int(bits), _ptr(scales, torch.float32, "scales"),
        float(kappa), _ptr(loss, torch.float64, "loss"),
        _ptr(grad_scales, torch.float32, "grad_scales"), ws.ptr, ws.nbytes, _stream(stream))
    _check(st, "jab_loss_backward_scales")


def jab_prepare_x(desc, B, T, X, ws: Workspace, stream=None):
    """Converts X into the workspace's fp16 copy for jab_loss_backward_scales_prepared."""
    st = lib().jab_prepare_x(ctypes.byref(desc), B, T, _ptr(X, torch.bfloat16, "X"), ws.ptr,
                             ws.nbytes, _stream(stream))
    _check(st, "jab_prepare_x")


def jab_loss_backward_scales_prepared(desc, B, T, X, W, A_ref, bits: int, scales, kappa: float,
                                      loss, grad_scales, ws: Workspace, stream=None):
    """jab_loss_backward_scales on the fp16 X that jab_prepare_x left in `ws`."""
    st = lib().jab_loss_backward_scales_prepared(
        ctypes.byref(desc), B, T, _ptr(X, torch.bfloat16, "X"), _ptr(W, torch.bfloat16, "W"),
        _ptr(A_ref, torch.float32, "A_ref"), int(bits), _ptr(scales, torch.float32, "scales"),
        float(kappa), _ptr(loss, torch.float64, "loss"),
        _ptr(grad_scales, torch.float32, "grad_scales"), ws.ptr, ws.nbytes, _stream(stream))
    _check(st, "jab_loss_backward_scales_prepared")


def jab_loss_backward_scales_kl(desc, B, T, X, W, A_ref, QKV_ref, lse_ref, bits: int, scales,
                                kappa: float, lambda_kl: float, loss, grad_scales, ws: Workspace,
                                kl=None, stream=None):
    """Scale gradient of MSE + lambda_kl * KL (Eq. 3 with both terms); the teacher's projection and
    log-sum-exp from jab_reference_projection / jab_reference_forward."""
    st = lib().jab_loss_backward_scales_kl(
        ctypes.byref(desc), B, T, _ptr(X, torch.bfloat16, "X"), _ptr(W, torch.bfloat16, "W"),
        _ptr(A_ref, torch.float32, "A_ref"), _ptr(QKV_ref, torch.float16, "QKV_ref"),
        _ptr(lse_ref, torch.float32, "lse_ref"), int(bits), _ptr(scales, torch.float32, "scales"),
        float(kappa), float(lambda_kl), _ptr(loss, torch.float64, "loss"),
        _ptr(kl, torch.float64, "kl"), _ptr(grad_scales, torch.float32, "grad_scales"), ws.ptr,
        ws.nbytes, _stream(stream))
    _check(st, "jab_loss_backward_scales_kl")


def jab_flip_rate(codes_a, codes_b, count, stream=None):
    """Number of positions where two int8 code tensors differ (Eq. 15), into count (int64 [1])."""
    if codes_a.numel() != codes_b.numel():
        raise ValueError("code arrays differ in size")
    if codes_a.numel() == 0:
        codes_a = codes_b = None
    n = 0 if codes_a is None else int(codes_a.numel())
    st = lib().jab_flip_rate(_ptr(codes_a, torch.int8, "codes_a"), _ptr(codes_b, torch.int8, "codes_b"),
                             n, _ptr(count, torch.int64, "count"), _stream(stream))
    _check(st, "jab_flip_rate")


def jab_loss_backward_weights(desc, B, T, X, W, A_ref, bits: int, scales, loss, grad_w=None,
                              grad_sqnorm=None, ws: Workspace = None, stream=None):
    """Loss and the STE weight gradient dL/dw_hat (fp32 [D, d]) and/or its squared norm (fp64 [1])."""
    st = lib().jab_loss_backward_weights(
        ctypes.byref(desc), B, T, _ptr(X, torch.bfloat16, "X"), _ptr(W, torch.bfloat16, "W"),
        _ptr(A_ref, torch.float32, "A_ref"), int(bits), _ptr(scales, torch.float32, "scales"),
        _ptr(loss, torch.float64, "loss"), _ptr(grad_w, torch.float32, "grad_w"),
        _ptr(grad_sqnorm, torch.float64, "grad_sqnorm"), ws.ptr, ws.nbytes, _stream(stream))
    _check(st, "jab_loss_backward_weights")


def jab_allocate_bits(omega, widths, n_weights, avg_bits: float, method: str = "greedy"):
    """Width per layer minimising the summed score within avg_bits per weight (Eq. 7). Host only.

    omega: [L, K] scores (any array-like of floats); widths: K increasing ints; n_weights: L ints.
    method: "greedy" or "pareto". Returns a list of L widths."""
    import numpy as np
    om = np.ascontiguousarray(np.asarray(omega, dtype=np.float64))
    w = np.ascontiguousarray(np.asarray(widths, dtype=np.int32))
    n = np.ascontiguousarray(np.asarray(n_weights, dtype=np.int64))
    if om.ndim != 2 or om.shape != (n.size, w.size):
        raise ValueError("omega must be [len(n_weights), len(widths)]")
    out = np.zeros(n.size, dtype=np.int32)
    st = lib().jab_allocate_bits(om.ctypes.data, w.ctypes.data, n.ctypes.data, int(n.size),
                                 int(w.size), float(avg_bits), {"greedy": 0, "pareto": 1}[method],
                                 out.ctypes.data)
    _check(st, "jab_allocate_bits")
    return [int(b) for b in out]


def jab_quantize(desc, bits, W, scales, codes=None, w_hat=None, stream=None):
    st = lib().jab_quantize(ctypes.byref(desc), int(bits), _ptr(W, torch.bfloat16, "W"),
                            _ptr(scales, torch.float32, "scales"), _ptr(codes, torch.int8, "codes"),
                            _ptr(w_hat, torch.float32, "w_hat"), _stream(stream))
    _check(st, "jab_quantize")


def jab_init_scales(desc, bits, mode, W, scales, stream=None):
    st = lib().jab_init_scales(ctypes.byref(desc), int(bits), int(mode),
                               _ptr(W, torch.bfloat16, "W"), _ptr(scales, torch.float32, "scales"),
                               _stream(stream))
    _check(st, "jab_init_scales")


def jab_selftest_wait_timeout(stream=None):
    """Launches the bounded-wait self-test kernel (its wait runs out after 2 s)."""
    _check(lib().jab_selftest_wait_timeout(_stream(stream)), "jab_selftest_wait_timeout")


def jab_set_deterministic(on: bool):
    """Deterministic-reduction mode, process-wide: every floating-point reduction in a fixed order
    (repeated calls bit-identical). Off by default: the STE weight gradient may then split its GEMM's
    token range and add the partial tiles with atomics."""
    _check(lib().jab_set_deterministic(int(on)), "jab_set_deterministic")


def jab_selftest_bounds_check(buf, n: int, stream=None) -> int:
    """Checked build only: writes buf[0..n] behind bounds checks against an n-element extent (the
    last write is skipped, JAB_ERR_DEVICE_ASSERT raised on the device). Returns the call's status
    (JAB_ERR_UNSUPPORTED from the normal build, which launches nothing)."""
    return int(lib().jab_selftest_bounds_check(_ptr(buf, torch.int32, "buf"), int(n), _stream(stream)))


def jab_get_device_status(stream=None) -> int:
    """Synchronises the stream and returns (and clears) the device-side status word."""
    return int(lib().jab_get_device_status(_stream(stream)))


def jab_timing_enable(on: bool = True):
    _check(lib().jab_timing_enable(1 if on else 0), "jab_timing_enable")


def jab_timing_reset():
    _check(lib().jab_timing_reset(), "jab_timing_reset")


def jab_timing_read() -> dict:
    """Synchronises the recorded events; returns {site: (total_ms, ranges, kernels)}."""
    L = lib()
    _check(L.jab_timing_collect(), "jab_timing_collect")
    out = {}
    for i in range(L.jab_timing_count()):
        name = ctypes.c_char_p()
        ms = ctypes.c_double()
        rng = ctypes.c_int64()
        nk = ctypes.c_int64()
        _check(L.jab_timing_get(i, ctypes.byref(name), ctypes.byref(ms), ctypes.byref(rng),
                                ctypes.byref(nk)), "jab_timing_get")
        out[name.value.decode()] = (ms.value, rng.value, nk.value)
    return out
