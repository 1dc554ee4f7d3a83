"""Python binding of libdptq (include/dptq.h): argument marshalling only.

Every function here forwards to the C ABI of the same name; all computation runs in the
library's CUDA kernels.  Tensors are torch CUDA tensors used as device buffers, and the
current torch stream is passed as the cudaStream_t.  There is no fallback: if the
library is missing or fails to load, every call raises.
"""
from __future__ import annotations

import ctypes
import os
import threading

from . import build as _build

_lock = threading.Lock()
_lib = None

DPTQ_OK = 0
_STATUS = {0: "ok", 1: "invalid argument", 2: "unsupported shape", 3: "CUDA error",
           4: "out of device memory", 5: "device wait timed out"}

EXPORTS = ("dptq_pack_weights", "dptq_rotate_quant_act", "dptq_rotate_act", "dptq_qlinear",
           "dptq_qlinear_quantize", "dptq_qlinear_gemm", "dptq_qlinear_static",
           "dptq_qgemm_codes", "dptq_reserve", "dptq_get_packed", "dptq_get_shape",
           "dptq_last_device_error", "dptq_destroy", "dptq_status_str", "dptq_last_error_message",
           "dptq_pack_weights_rh", "dptq_rotate_quant_act_rh", "dptq_rotate_act_rh", "dptq_kv4_quantize",
           "dptq_sensitivity_policy", "dptq_plan_info", "dptq_scratch_buffers")


class DptqError(RuntimeError):
    def __init__(self, status: int, msg: str):
        super().__init__(f"{_STATUS.get(status, status)}: {msg}")
        self.status = status


def lib_path() -> str:
    return _build.LIB


def load(build_if_missing: bool = True):
    """Load libdptq.so (building it first when it is missing or stale)."""
    global _lib
    with _lock:
        if _lib is None:
            path = _build.build() if build_if_missing else _build.LIB
            if not os.path.exists(path):
                raise RuntimeError(f"libdptq is not built ({path}); run paper_2606_12487_gb300.build")
            lib = ctypes.CDLL(path)
            P, I = ctypes.c_void_p, ctypes.c_int
            sig = {
                "dptq_pack_weights": ([P, I, I, I, I, ctypes.POINTER(P)], I),
                "dptq_rotate_quant_act": ([P, I, I, I, I, P, P, P], I),
                "dptq_rotate_act": ([P, I, I, I, P, P], I),
                "dptq_qlinear": ([P, P, I, I, P, P], I),
                "dptq_qlinear_quantize": ([P, P, I, I, P], I),
                "dptq_qlinear_gemm": ([P, I, I, P, P], I),
                "dptq_qlinear_static": ([P, P, I, I, P, P], I),
                "dptq_qgemm_codes": ([P, P, P, I, I, P, P, P], I),
                "dptq_reserve": ([I, I, I], I),
                "dptq_get_packed": ([P, P, P], I),
                "dptq_get_shape": ([P, P, P, P], I),
                "dptq_last_device_error": ([P], I),
                "dptq_destroy": ([P], None),
                "dptq_status_str": ([I], ctypes.c_char_p),
                "dptq_last_error_message": ([], ctypes.c_char_p),
                "dptq_pack_weights_rh": ([P, I, I, I, P, I, ctypes.POINTER(P)], I),
                "dptq_rotate_quant_act_rh": ([P, I, I, I, I, P, P, P, P], I),
                "dptq_rotate_act_rh": ([P, I, I, I, P, P, P], I),
                "dptq_kv4_quantize": ([P, I, I, I, P, P, P], I),
                "dptq_sensitivity_policy": ([P, P, I, I, I, I, ctypes.c_double, ctypes.c_double, ctypes.c_double,
                                             P, P, P, P], I),
                "dptq_plan_info": ([I, I, I, I, I, I, ctypes.POINTER(I), I], I),
                "dptq_scratch_buffers": ([ctypes.POINTER(P), ctypes.POINTER(ctypes.c_size_t), ctypes.POINTER(I), I,
                                          ctypes.POINTER(I)], I),
            }
            for name, (args, res) in sig.items():
                fn = getattr(lib, name)
                fn.argtypes = args
                fn.restype = res
            _lib = lib
    return _lib


def _check(status: int):
    if status != DPTQ_OK:
        msg = load().dptq_last_error_message().decode(errors="replace")
        raise DptqError(status, msg)


def _ptr(t) -> ctypes.c_void_p:
    if t is None:
        return None
    return ctypes.c_void_p(t.data_ptr())


def _stream(stream=None):
    import torch
    s = stream if stream is not None else torch.cuda.current_stream()
    return ctypes.c_void_p(s.cuda_stream)


def _check_tensor(t, dtype, shape, name):
    import torch
    if not isinstance(t, torch.Tensor) or not t.is_cuda:
        raise TypeError(f"{name} must be a CUDA tensor")
    if t.dtype != dtype:
        raise TypeError(f"{name} must be {dtype}, got {t.dtype}")
    if tuple(t.shape) != tuple(shape):
        raise ValueError(f"{name} must have shape {tuple(shape)}, got {tuple(t.shape)}")
    if not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")


class QLinear:
    """A packed quantized linear layer (owns the library handle)."""

    def __init__(self, handle: ctypes.c_void_p, N: int, K: int, had_block: int):
        self._h = handle
        self.N, self.K, self.had_block = N, K, had_block

    @property
    def handle(self):
        return self._h

    def close(self):
        if self._h:
            load().dptq_destroy(self._h)
            self._h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


def dptq_pack_weights(W, had_block: int) -> QLinear:
    """Pack fp16 weights [N, K] (CUDA or CPU tensor) into a QLinear (RTN int4, Eq. 5 fold)."""
    import torch
    if W.dtype != torch.float16 or W.dim() != 2 or not W.is_contiguous():
        raise TypeError("W must be a contiguous 2-D float16 tensor")
    N, K = W.shape
    h = ctypes.c_void_p()
    _check(load().dptq_pack_weights(ctypes.c_void_p(W.data_ptr()), N, K, had_block, int(W.is_cuda),
                                    ctypes.byref(h)))
    return QLinear(h, N, K, had_block)


def dptq_pack_weights_rh(W, had_block: int, signs) -> QLinear:
    """dptq_pack_weights with the randomized Hadamard D R; `signs`: K values of +1 / -1
    (a host int8 numpy array or CPU tensor)."""
    import numpy as np
    import torch
    if W.dtype != torch.float16 or W.dim() != 2 or not W.is_contiguous():
        raise TypeError("W must be a contiguous 2-D float16 tensor")
    N, K = W.shape
    d = np.ascontiguousarray(signs.cpu().numpy() if isinstance(signs, torch.Tensor) else signs, dtype=np.int8)
    if d.shape != (K,):
        raise ValueError(f"signs must have shape ({K},)")
    h = ctypes.c_void_p()
    _check(load().dptq_pack_weights_rh(ctypes.c_void_p(W.data_ptr()), N, K, had_block,
                                       d.ctypes.data_as(ctypes.c_void_p), int(W.is_cuda), ctypes.byref(h)))
    return QLinear(h, N, K, had_block)


def dptq_rotate_quant_act_rh(x, had_block: int, bits: int, signs, codes, scales, stream=None):
    """dptq_rotate_quant_act with the randomized Hadamard: `signs` a CUDA int8 tensor [K]."""
    import torch
    M, K = x.shape
    _check_tensor(x, torch.float16, (M, K), "x")
    _check_tensor(signs, torch.int8, (K,), "signs")
    _check_tensor(codes, torch.uint8 if bits == 4 else torch.int8, (M, K // 2 if bits == 4 else K), "codes")
    _check_tensor(scales, torch.float32, (M,), "scales")
    _check(load().dptq_rotate_quant_act_rh(_ptr(x), M, K, had_block, bits, _ptr(signs), _ptr(codes), _ptr(scales),
                                           _stream(stream)))


def dptq_rotate_act_rh(x, had_block: int, signs, y, stream=None):
    import torch
    M, K = x.shape
    _check_tensor(x, torch.float16, (M, K), "x")
    _check_tensor(signs, torch.int8, (K,), "signs")
    _check_tensor(y, torch.float32, (M, K), "y")
    _check(load().dptq_rotate_act_rh(_ptr(x), M, K, had_block, _ptr(signs), _ptr(y), _stream(stream)))


def dptq_kv4_quantize(kv, group: int, codes, scales, stream=None):
    """Group-wise symmetric 4-bit KV codes: kv float16 [rows, cols] -> codes uint8
    [rows, cols/2] (two's complement nibbles, low nibble first), scales float32
    [rows, cols/group]."""
    import torch
    R, C = kv.shape
    _check_tensor(kv, torch.float16, (R, C), "kv")
    _check_tensor(codes, torch.uint8, (R, C // 2), "codes")
    _check_tensor(scales, torch.float32, (R, C // group if group > 0 else 0), "scales")
    _check(load().dptq_kv4_quantize(_ptr(kv), R, C, group, _ptr(codes), _ptr(scales), _stream(stream)))


def dptq_sensitivity_policy(x, dx, bits: int, eps: float, tau_jr: float, tau_snr: float, jr, snr, bits_out,
                            stream=None):
    """Per-layer JR and historical SNR of residual states x and updates dx (float32
    [L, T, d]) and the activation bits (8 on the sensitive set): jr, snr float64 [L],
    bits_out uint8 [L]."""
    import torch
    L, T, d = x.shape
    _check_tensor(x, torch.float32, (L, T, d), "x")
    _check_tensor(dx, torch.float32, (L, T, d), "dx")
    _check_tensor(jr, torch.float64, (L,), "jr")
    _check_tensor(snr, torch.float64, (L,), "snr")
    _check_tensor(bits_out, torch.uint8, (L,), "bits_out")
    _check(load().dptq_sensitivity_policy(_ptr(x), _ptr(dx), L, T, d, bits, eps, tau_jr, tau_snr, _ptr(jr), _ptr(snr),
                                          _ptr(bits_out), _stream(stream)))


def dptq_rotate_quant_act(x, had_block: int, bits: int, codes, scales, stream=None):
    import torch
    M, K = x.shape
    _check_tensor(x, torch.float16, (M, K), "x")
    _check_tensor(codes, torch.uint8 if bits == 4 else torch.int8, (M, K // 2 if bits == 4 else K), "codes")
    _check_tensor(scales, torch.float32, (M,), "scales")
    _check(load().dptq_rotate_quant_act(_ptr(x), M, K, had_block, bits, _ptr(codes), _ptr(scales),
                                        _stream(stream)))


def dptq_rotate_act(x, had_block: int, y, stream=None):
    import torch
    M, K = x.shape
    _check_tensor(x, torch.float16, (M, K), "x")
    _check_tensor(y, torch.float32, (M, K), "y")
    _check(load().dptq_rotate_act(_ptr(x), M, K, had_block, _ptr(y), _stream(stream)))


def dptq_qlinear(layer: QLinear, x, bits: int, out, stream=None):
    import torch
    M = x.shape[0]
    _check_tensor(x, torch.float16, (M, layer.K), "x")
    _check_tensor(out, torch.float16, (M, layer.N), "out")
    _check(load().dptq_qlinear(layer.handle, _ptr(x), M, bits, _ptr(out), _stream(stream)))


def dptq_qlinear_static(layer: QLinear, x, bits: int, out, stream=None):
    """dptq_qlinear without any device allocation: the library's fixed scratch array is
    used instead (M <= 32, K <= 16384)."""
    import torch
    M = x.shape[0]
    _check_tensor(x, torch.float16, (M, layer.K), "x")
    _check_tensor(out, torch.float16, (M, layer.N), "out")
    _check(load().dptq_qlinear_static(layer.handle, _ptr(x), M, bits, _ptr(out), _stream(stream)))


def dptq_qlinear_quantize(layer: QLinear, x, bits: int, stream=None):
    import torch
    M = x.shape[0]
    _check_tensor(x, torch.float16, (M, layer.K), "x")
    _check(load().dptq_qlinear_quantize(layer.handle, _ptr(x), M, bits, _stream(stream)))


def dptq_qlinear_gemm(layer: QLinear, M: int, bits: int, out, stream=None):
    import torch
    _check_tensor(out, torch.float16, (M, layer.N), "out")
    _check(load().dptq_qlinear_gemm(layer.handle, M, bits, _ptr(out), _stream(stream)))


def dptq_qgemm_codes(layer: QLinear, codes, scales, bits: int, out, acc=None, stream=None):
    import torch
    M = scales.shape[0]
    _check_tensor(codes, torch.uint8 if bits == 4 else torch.int8,
                  (M, layer.K // 2 if bits == 4 else layer.K), "codes")
    _check_tensor(scales, torch.float32, (M,), "scales")
    _check_tensor(out, torch.float16, (M, layer.N), "out")
    if acc is not None:
        _check_tensor(acc, torch.int32, (M, layer.N), "acc")
    _check(load().dptq_qgemm_codes(layer.handle, _ptr(codes), _ptr(scales), M, bits, _ptr(out), _ptr(acc),
                                   _stream(stream)))


def dptq_reserve(max_M: int, max_K: int, max_N: int = 0):
    _check(load().dptq_reserve(max_M, max_K, max_N))


PLAN_INFO_FIELDS = ("nt", "kps", "M_pad", "grid", "smem_bytes", "stages", "conv_slots", "a_tmem", "nbuf",
                    "segs", "seg_iters", "tmem_cols", "acc_cols", "KI", "n_wtiles", "m_tiles", "dp_tiles",
                    "sk_iters", "rq_np", "fused")


def dptq_plan_info(M: int, N: int, K: int, bits: int, num_sms: int, fused: bool = False) -> dict:
    """The GEMM launch plan for a shape (host only, no GPU): a dict of PLAN_INFO_FIELDS."""
    buf = (ctypes.c_int * len(PLAN_INFO_FIELDS))()
    _check(load().dptq_plan_info(M, N, K, bits, num_sms, 1 if fused else 0, buf, len(PLAN_INFO_FIELDS)))
    return dict(zip(PLAN_INFO_FIELDS, list(buf)))


def dptq_get_packed(layer: QLinear):
    """(packed int4 uint8 [N, K/2] in the public nibble format, s_w float32 [N]) as numpy."""
    import numpy as np
    wq = np.empty((layer.N, layer.K // 2), dtype=np.uint8)
    sw = np.empty((layer.N,), dtype=np.float32)
    _check(load().dptq_get_packed(layer.handle, wq.ctypes.data_as(ctypes.c_void_p),
                                  sw.ctypes.data_as(ctypes.c_void_p)))
    return wq, sw


def dptq_last_device_error():
    _check(load().dptq_last_device_error(None))


def dptq_scratch_buffers(max_entries: int = 64):
    """Test hook: [(device address, bytes, still allocated)] of the current device's
    activation-plane and scale scratch, current buffers first, then superseded ones."""
    P = ctypes.c_void_p
    ptrs = (P * max_entries)()
    sizes = (ctypes.c_size_t * max_entries)()
    alloc = (ctypes.c_int * max_entries)()
    count = ctypes.c_int(0)
    _check(load().dptq_scratch_buffers(ptrs, sizes, alloc, max_entries, ctypes.byref(count)))
    n = min(count.value, max_entries)
    return [(int(ptrs[i] or 0), int(sizes[i]), bool(alloc[i])) for i in range(n)]
