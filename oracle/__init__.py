"""CPU oracle for the DynamicPTQ quantized linear layer (ctypes wrapper over dptq_oracle.c).

TEST INFRASTRUCTURE ONLY: the test suite, ``__graft_entry__.smoke()`` and the CPU-baseline
leg of ``bench.py`` may use it; the product path (``paper_2606_12487_gb300``) never does.
It shares no code with the CUDA library.  See ``dptq_oracle.c`` for the definitions and the
paper passages each function follows (Section 2 Eqs. 2-5, Section 4.2, Section 3.1 Eqs. 8-11).

Parity status: every exported function is pinned by tests under ``tests/test_oracle_*.py``
against closed forms, textbook constructions and library routines.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "dptq_oracle.c")
_LIB = os.path.join(_HERE, "_build", "libdptq_oracle.so")
_lock = threading.Lock()
_lib = None


def build(force: bool = False) -> str:
    """Compile the oracle with the host C compiler (plain C11, no fast-math)."""
    os.makedirs(os.path.dirname(_LIB), exist_ok=True)
    if force or not os.path.exists(_LIB) or os.path.getmtime(_LIB) < os.path.getmtime(_SRC):
        tmp = _LIB + f".tmp{os.getpid()}"
        subprocess.check_call(
            ["cc", "-O2", "-std=c11", "-ffp-contract=off", "-fno-fast-math", "-fPIC", "-shared",
             _SRC, "-o", tmp, "-lm"])
        os.replace(tmp, _LIB)
    return _LIB


def _load():
    global _lib
    with _lock:
        if _lib is None:
            lib = ctypes.CDLL(build())
            P = ctypes.c_void_p
            I = ctypes.c_int
            lib.orc_half_to_double.argtypes = [ctypes.c_uint16]
            lib.orc_half_to_double.restype = ctypes.c_double
            lib.orc_float_to_half.argtypes = [ctypes.c_float]
            lib.orc_float_to_half.restype = ctypes.c_uint16
            lib.orc_hadamard_entry.argtypes = [I, I]
            lib.orc_hadamard_entry.restype = I
            lib.orc_paley_entry.argtypes = [I, I, I]
            lib.orc_paley_entry.restype = I
            lib.orc_tail_factor.argtypes = [I, P, P]
            lib.orc_tail_factor.restype = I
            lib.orc_tail_entry.argtypes = [I, I, I]
            lib.orc_tail_entry.restype = I
            lib.orc_block_layout.argtypes = [I, I, P, P]
            lib.orc_block_layout.restype = I
            lib.orc_rotate_row_f64.argtypes = [P, P, I, I]
            lib.orc_rotate_row_f64.restype = I
            lib.orc_rotate_f16.argtypes = [P, P, I, I, I]
            lib.orc_rotate_f16.restype = I
            lib.orc_quant_rows.argtypes = [P, I, I, I, P, P]
            lib.orc_quant_rows.restype = I
            lib.orc_rotate_quant_act.argtypes = [P, I, I, I, I, P, P]
            lib.orc_rotate_quant_act.restype = I
            lib.orc_pack_weights.argtypes = [P, I, I, I, P, P]
            lib.orc_pack_weights.restype = I
            lib.orc_gemm_i32.argtypes = [P, P, I, I, I, P]
            lib.orc_gemm_i32.restype = I
            lib.orc_epilogue.argtypes = [P, P, P, I, I, P]
            lib.orc_epilogue.restype = None
            lib.orc_qlinear.argtypes = [P, I, I, I, I, P, P, I, P, P, P, P]
            lib.orc_qlinear.restype = I
            lib.orc_pack_nibbles.argtypes = [P, I, I, P]
            lib.orc_pack_nibbles.restype = None
            lib.orc_unpack_nibbles.argtypes = [P, I, I, P]
            lib.orc_unpack_nibbles.restype = None
            lib.orc_residual_stats.argtypes = [P, P, I, I, I, ctypes.c_double, P, P]
            lib.orc_residual_stats.restype = I
            lib.orc_rotate_f16_signed.argtypes = [P, P, I, I, I, P]
            lib.orc_rotate_f16_signed.restype = I
            lib.orc_rotate_quant_act_signed.argtypes = [P, I, I, I, I, P, P, P]
            lib.orc_rotate_quant_act_signed.restype = I
            lib.orc_pack_weights_signed.argtypes = [P, I, I, I, P, P, P]
            lib.orc_pack_weights_signed.restype = I
            lib.orc_qlinear_signed.argtypes = [P, I, I, I, I, P, P, P, I, P, P, P, P]
            lib.orc_qlinear_signed.restype = I
            lib.orc_kv4_quantize.argtypes = [P, I, I, I, P, P]
            lib.orc_kv4_quantize.restype = I
            lib.orc_policy_mask.argtypes = [P, P, I, ctypes.c_double, ctypes.c_double, P]
            lib.orc_policy_mask.restype = None
            _lib = lib
    return _lib


def _p(a: np.ndarray):
    assert a.flags["C_CONTIGUOUS"]
    return a.ctypes.data_as(ctypes.c_void_p)


def _as_half_bits(x) -> np.ndarray:
    x = np.ascontiguousarray(x)
    if x.dtype == np.float16:
        return x.view(np.uint16)
    assert x.dtype == np.uint16, x.dtype
    return x


# ---------------------------------------------------------------------------------------
def half_to_double(bits: int) -> float:
    return _load().orc_half_to_double(int(bits))


def float_to_half(v: float) -> int:
    return int(_load().orc_float_to_half(float(v)))


def hadamard_entry(i: int, j: int) -> int:
    return int(_load().orc_hadamard_entry(i, j))


def paley_entry(p: int, i: int, j: int) -> int:
    """Entry of Paley's type-I Hadamard matrix of order p (p - 1 prime, = 3 mod 4); 0 when
    p is not such an order."""
    return int(_load().orc_paley_entry(p, i, j))


def tail_factor(r: int):
    """(p, k) with r = p 2^k for a tail block (p = 1 for a power of two), or None."""
    p = ctypes.c_int(0)
    k = ctypes.c_int(0)
    return (p.value, k.value) if _load().orc_tail_factor(r, ctypes.byref(p), ctypes.byref(k)) else None


def tail_entry(r: int, i: int, j: int) -> int:
    """Entry (i, j) of the tail block's Hadamard matrix H_p (x) H_(2^k) of order r."""
    return int(_load().orc_tail_entry(r, i, j))


def block_layout(K: int, B: int):
    q = ctypes.c_int(0)
    r = ctypes.c_int(0)
    ok = _load().orc_block_layout(K, B, ctypes.byref(q), ctypes.byref(r))
    return (q.value, r.value) if ok else None


def rotate_row_f64(x: np.ndarray, B: int) -> np.ndarray:
    x = np.ascontiguousarray(x, dtype=np.float64)
    y = np.empty_like(x)
    if not _load().orc_rotate_row_f64(_p(x), _p(y), x.shape[0], B):
        raise ValueError("bad block layout")
    return y


def _signs(signs, K):
    if signs is None:
        return None
    d = np.ascontiguousarray(signs, dtype=np.int8)
    assert d.shape == (K,) and np.all(np.abs(d) == 1), "signs must be K values of +1 / -1"
    return d


def rotate(x_f16: np.ndarray, B: int, signs=None) -> np.ndarray:
    """fp16 [M, K] -> fp32 [M, K]: x R with R = blockdiag(H/sqrt(block)) (Eq. 4); with
    `signs` (K values of +-1) the randomized Hadamard x diag(signs) R."""
    xb = _as_half_bits(x_f16)
    M, K = xb.shape
    y = np.empty((M, K), dtype=np.float32)
    d = _signs(signs, K)
    if not _load().orc_rotate_f16_signed(_p(xb), _p(y), M, K, B, None if d is None else _p(d)):
        raise ValueError("bad block layout")
    return y


def quant_rows(y: np.ndarray, bits: int):
    """Per-token symmetric quantizer (Eq. 2, Section 4.2): returns (codes int8, scales fp32)."""
    y = np.ascontiguousarray(y, dtype=np.float32)
    M, K = y.shape
    c = np.empty((M, K), dtype=np.int8)
    s = np.empty((M,), dtype=np.float32)
    if not _load().orc_quant_rows(_p(y), M, K, bits, _p(c), _p(s)):
        raise ValueError("bits must be 4 or 8")
    return c, s


def rotate_quant_act(x_f16: np.ndarray, B: int, bits: int, signs=None):
    xb = _as_half_bits(x_f16)
    M, K = xb.shape
    c = np.empty((M, K), dtype=np.int8)
    s = np.empty((M,), dtype=np.float32)
    d = _signs(signs, K)
    if not _load().orc_rotate_quant_act_signed(_p(xb), M, K, B, bits, None if d is None else _p(d), _p(c), _p(s)):
        raise ValueError("bad shape or bits")
    return c, s


def pack_weights(W_f16: np.ndarray, B: int, signs=None):
    """RTN int4 per-channel symmetric weights with R folded in (Eq. 5): (q int8 [N,K], s_w fp32 [N])."""
    wb = _as_half_bits(W_f16)
    N, K = wb.shape
    q = np.empty((N, K), dtype=np.int8)
    s = np.empty((N,), dtype=np.float32)
    d = _signs(signs, K)
    if not _load().orc_pack_weights_signed(_p(wb), N, K, B, None if d is None else _p(d), _p(q), _p(s)):
        raise ValueError("bad shape")
    return q, s


def gemm_i32(a: np.ndarray, w: np.ndarray) -> np.ndarray:
    a = np.ascontiguousarray(a, dtype=np.int8)
    w = np.ascontiguousarray(w, dtype=np.int8)
    M, K = a.shape
    N, K2 = w.shape
    assert K == K2
    acc = np.empty((M, N), dtype=np.int32)
    if not _load().orc_gemm_i32(_p(a), _p(w), M, N, K, _p(acc)):
        raise OverflowError("accumulator leaves int32")
    return acc


def epilogue(acc: np.ndarray, sa: np.ndarray, sw: np.ndarray) -> np.ndarray:
    acc = np.ascontiguousarray(acc, dtype=np.int32)
    sa = np.ascontiguousarray(sa, dtype=np.float32)
    sw = np.ascontiguousarray(sw, dtype=np.float32)
    M, N = acc.shape
    out = np.empty((M, N), dtype=np.uint16)
    _load().orc_epilogue(_p(acc), _p(sa), _p(sw), M, N, _p(out))
    return out.view(np.float16)


def qlinear(x_f16: np.ndarray, B: int, bits: int, q: np.ndarray, sw: np.ndarray, signs=None):
    """Whole layer: returns dict(out fp16 [M,N], acc int32, codes int8, sa fp32)."""
    xb = _as_half_bits(x_f16)
    M, K = xb.shape
    q = np.ascontiguousarray(q, dtype=np.int8)
    sw = np.ascontiguousarray(sw, dtype=np.float32)
    N = q.shape[0]
    out = np.empty((M, N), dtype=np.uint16)
    acc = np.empty((M, N), dtype=np.int32)
    codes = np.empty((M, K), dtype=np.int8)
    sa = np.empty((M,), dtype=np.float32)
    d = _signs(signs, K)
    if not _load().orc_qlinear_signed(_p(xb), M, K, B, bits, None if d is None else _p(d), _p(q), _p(sw), N,
                                      _p(out), _p(acc), _p(codes), _p(sa)):
        raise ValueError("bad shape, bits or int32 overflow")
    return {"out": out.view(np.float16), "acc": acc, "codes": codes, "sa": sa}


def pack_nibbles(codes: np.ndarray) -> np.ndarray:
    codes = np.ascontiguousarray(codes, dtype=np.int8)
    R, K = codes.shape
    assert K % 2 == 0
    out = np.empty((R, K // 2), dtype=np.uint8)
    _load().orc_pack_nibbles(_p(codes), R, K, _p(out))
    return out


def unpack_nibbles(packed: np.ndarray, K: int) -> np.ndarray:
    packed = np.ascontiguousarray(packed, dtype=np.uint8)
    R = packed.shape[0]
    out = np.empty((R, K), dtype=np.int8)
    _load().orc_unpack_nibbles(_p(packed), R, K, _p(out))
    return out


def residual_stats(x: np.ndarray, dx: np.ndarray, bits: int, eps: float = 1e-6):
    """(JR_l, SNR_hist_l) of Eqs. 8-11 for one layer's residual state x and update dx [T, d]."""
    x = np.ascontiguousarray(x, dtype=np.float32)
    dx = np.ascontiguousarray(dx, dtype=np.float32)
    T, d = x.shape
    jr = ctypes.c_double(0)
    snr = ctypes.c_double(0)
    if not _load().orc_residual_stats(_p(x), _p(dx), T, d, bits, eps, ctypes.byref(jr),
                                      ctypes.byref(snr)):
        raise MemoryError
    return jr.value, snr.value


def kv4_quantize(x_f16: np.ndarray, group: int = 128):
    """Group-wise symmetric 4-bit KV-cache codes (Section 4.2, group 128):
    (codes int8 [rows, cols], scales fp32 [rows, cols // group])."""
    xb = _as_half_bits(x_f16)
    R, C = xb.shape
    c = np.empty((R, C), dtype=np.int8)
    s = np.empty((R, C // group if group > 0 else 0), dtype=np.float32)
    if not _load().orc_kv4_quantize(_p(xb), R, C, group, _p(c), _p(s)):
        raise ValueError("group must divide the number of columns")
    return c, s


def policy_mask(jr, snr, tau_jr: float, tau_snr: float) -> np.ndarray:
    """Per-layer activation bits (Section 3.3 Eq. 20, Algorithm 1 step 2): 8 on the
    sensitive set {l: JR_l > tau_jr and SNR_l < tau_snr}, else 4."""
    jr = np.ascontiguousarray(jr, dtype=np.float64)
    snr = np.ascontiguousarray(snr, dtype=np.float64)
    L = jr.shape[0]
    bits = np.empty((L,), dtype=np.uint8)
    _load().orc_policy_mask(_p(jr), _p(snr), L, tau_jr, tau_snr, _p(bits))
    return bits
