"""Comparison rules between the CUDA path and the oracle.

Tolerances (the parity contract):
  * rotated activations: |y_gpu - y_oracle| <= 1e-5 * max|y_oracle row|;
  * codes: bit-exact, except at rounding ties inside that tolerance -- each mismatch is
    off by one code, sits where the oracle's y/s lies within 1e-5 * qmax of a half
    integer (the rotation tolerance expressed in code units), and there are at most
    1e-5 of all codes of them;
  * accumulators: bit-exact on identical codes;
  * fp16 outputs: within 1 fp16 ulp given identical accumulators and scales.
"""
import numpy as np

Y_TOL = 1e-5
TIE_FRAC = 1e-5


def check_rotation(y_gpu, y_ref):
    y_gpu = np.asarray(y_gpu, dtype=np.float64)
    y_ref = np.asarray(y_ref, dtype=np.float64)
    rowmax = np.max(np.abs(y_ref), axis=1, keepdims=True)
    err = np.abs(y_gpu - y_ref)
    bad = err > Y_TOL * rowmax
    assert not bad.any(), f"rotation off at {np.argwhere(bad)[:5].tolist()}: max rel {np.max(err / np.maximum(rowmax, 1e-30)):.3e}"
    return float(np.max(err / np.maximum(rowmax, 1e-30)))


def check_codes(c_gpu, c_ref, y_ref, s_ref, bits, total=None):
    """Returns the number of tie mismatches (asserts they follow the contract)."""
    c_gpu = np.asarray(c_gpu, dtype=np.int32)
    c_ref = np.asarray(c_ref, dtype=np.int32)
    qmax = (1 << (bits - 1)) - 1
    mism = c_gpu != c_ref
    n = int(mism.sum())
    if n == 0:
        return 0
    assert np.all(np.abs(c_gpu - c_ref)[mism] == 1), "a code is off by more than one"
    rows, cols = np.nonzero(mism)
    t = np.abs(y_ref[rows, cols].astype(np.float64) / s_ref[rows].astype(np.float64))
    dist = np.abs(t - (np.floor(t) + 0.5))
    assert np.all(dist <= Y_TOL * qmax), f"non-tie mismatch: distance to .5 {dist.max():.3e}"
    total = c_ref.size if total is None else total
    assert n <= TIE_FRAC * total, f"{n} tie mismatches out of {total} codes exceed 1e-5"
    return n


def check_scales(s_gpu, s_ref):
    s_gpu = np.asarray(s_gpu, dtype=np.float64)
    s_ref = np.asarray(s_ref, dtype=np.float64)
    rel = np.abs(s_gpu - s_ref) / np.maximum(np.abs(s_ref), 1e-30)
    assert np.all(rel <= Y_TOL), f"scale off by {rel.max():.3e}"


def fp16_ulp_distance(a, b):
    """Distance in representable fp16 steps (monotone integer mapping of the bits)."""
    def key(v):
        u = np.asarray(v, dtype=np.float16).view(np.uint16).astype(np.int32)
        return np.where(u & 0x8000, -(u & 0x7FFF), u)
    return np.abs(key(a) - key(b))


def check_out(out_gpu, out_ref, max_ulp=1):
    d = fp16_ulp_distance(out_gpu, out_ref)
    assert d.max() <= max_ulp, f"output off by {int(d.max())} fp16 ulp at {np.argwhere(d > max_ulp)[:5].tolist()}"
    return int(d.max())


def unpack_public_a4(packed, K):
    p = np.asarray(packed, dtype=np.uint8)
    lo = (p & 0x0F).astype(np.int16)
    hi = (p >> 4).astype(np.int16)
    lo = np.where(lo >= 8, lo - 16, lo)
    hi = np.where(hi >= 8, hi - 16, hi)
    out = np.empty((p.shape[0], K), dtype=np.int8)
    out[:, 0::2] = lo
    out[:, 1::2] = hi
    return out
