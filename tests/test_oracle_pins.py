"""Pins of the CPU oracle against things other than itself (no GPU).

Each test ties one oracle function to a closed form, a textbook construction, a value
worked by hand (tests/golden), a library routine, or a mathematical invariant the paper
states, chosen so that a dropped term, a flipped sign, a wrong index or a transposed
operand fails at least one of them.
"""
import math
import os

import numpy as np
import pytest

from paper_2606_12487_gb300 import inputs

GOLD = os.path.join(os.path.dirname(__file__), "golden")


def _rows(name):
    with open(os.path.join(GOLD, name)) as f:
        return [ln.strip() for ln in f if ln.strip() and not ln.startswith("#")]


def sylvester(n):
    """Textbook recursion H_2n = [[H, H], [H, -H]] (independent of the popcount form)."""
    h = np.array([[1]], dtype=np.int64)
    while h.shape[0] < n:
        h = np.block([[h, h], [h, -h]])
    return h


# ---------------------------------------------------------------- fp16 conversions
def test_half_decode_matches_numpy_for_every_pattern(orc):
    bits = np.arange(65536, dtype=np.uint32).astype(np.uint16)
    ref = bits.view(np.float16).astype(np.float64)
    got = np.array([orc.half_to_double(int(b)) for b in bits])
    finite = ~np.isnan(ref)
    assert np.array_equal(got[finite], ref[finite])
    assert np.all(np.isnan(got[~finite]))


def test_float_to_half_matches_numpy(orc):
    rng = np.random.default_rng(3)
    vals = np.concatenate([
        rng.standard_normal(4000).astype(np.float32) * np.float32(10.0) ** rng.integers(-9, 6, 4000),
        # exact ties between neighbouring halves at several binades
        (np.arange(1, 2048, dtype=np.float64) * 2.0 ** -11 + 1.0).astype(np.float32),
        np.array([65504, 65519.996, 65520, 65536, 1e9, -65520, 2 ** -24, 2 ** -25,
                  3 * 2 ** -26, 2 ** -14, 2 ** -14 - 2 ** -25, 0.0, -0.0], dtype=np.float32),
    ]).astype(np.float32)
    got = np.array([orc.float_to_half(float(v)) for v in vals], dtype=np.uint16)
    with np.errstate(over="ignore"):
        ref = vals.astype(np.float16).view(np.uint16)
    assert np.array_equal(got, ref)


# ---------------------------------------------------------------- Hadamard (Section 2, Eq. 4)
def test_hadamard_h4_golden(orc):
    gold = np.array([[int(v) for v in ln.split()] for ln in _rows("hadamard_h4.txt")])
    got = np.array([[orc.hadamard_entry(i, j) for j in range(4)] for i in range(4)])
    assert np.array_equal(got, gold)


@pytest.mark.parametrize("n", [1, 2, 4, 8, 16, 32, 64])
def test_hadamard_entry_equals_sylvester_recursion(orc, n):
    got = np.array([[orc.hadamard_entry(i, j) for j in range(n)] for i in range(n)])
    assert np.array_equal(got, sylvester(n))


@pytest.mark.parametrize("B", [2, 16, 256, 2048, 4096])
def test_rotation_rows_are_scaled_sylvester_rows(orc, B):
    H = sylvester(B)
    for j in sorted({0, 1, B // 3, B - 1}):
        e = np.zeros(B)
        e[j] = 1.0
        y = orc.rotate_row_f64(e, B)
        assert np.allclose(y, H[j] / math.sqrt(B), rtol=0, atol=1e-15)


@pytest.mark.parametrize("B", [2, 8, 64, 256])
def test_hadamard_orthogonality_exact(orc, B):
    # rows of R for the identity give R itself; H H^T = B I exactly
    R = np.stack([orc.rotate_row_f64(np.eye(B)[i], B) for i in range(B)])
    HHt = np.rint(R @ R.T * B).astype(np.int64)
    assert np.array_equal(HHt, B * np.eye(B, dtype=np.int64))


@pytest.mark.parametrize("K,B", [(4096, 4096), (11008, 256), (13824, 1024), (768, 512)])
def test_rotation_preserves_norm_and_is_involution(orc, K, B):
    rng = np.random.default_rng(11)
    x = rng.standard_normal(K)
    y = orc.rotate_row_f64(x, B)
    assert abs(np.linalg.norm(y) - np.linalg.norm(x)) <= 1e-12 * np.linalg.norm(x)   # Eq. 12
    z = orc.rotate_row_f64(y, B)                                                     # R R = I
    assert np.max(np.abs(z - x)) <= 1e-12 * np.max(np.abs(x))


def test_all_ones_block_maps_to_first_axis(orc):
    B = 1024
    y = orc.rotate_row_f64(np.ones(B), B)
    exp = np.zeros(B)
    exp[0] = math.sqrt(B)
    assert np.allclose(y, exp, atol=1e-12)


def test_block_structure_and_tail(orc):
    # K = 13 * 1024 + 512: a vector living in block 2 stays in block 2; the tail uses H_512
    K, B = 13824, 1024
    assert orc.block_layout(K, B) == (13, 512)
    rng = np.random.default_rng(5)
    x = np.zeros(K)
    x[2048:3072] = rng.standard_normal(1024)
    y = orc.rotate_row_f64(x, B)
    assert np.all(y[:2048] == 0) and np.all(y[3072:] == 0)
    assert np.allclose(y[2048:3072], sylvester(1024) @ x[2048:3072] / 32.0, atol=1e-12)
    t = np.zeros(K)
    t[13312:] = rng.standard_normal(512)
    yt = orc.rotate_row_f64(t, B)
    assert np.allclose(yt[13312:], sylvester(512) @ t[13312:] / math.sqrt(512), atol=1e-12)
    assert np.all(yt[:13312] == 0)


def test_bad_block_layouts_rejected(orc):
    assert orc.block_layout(1536 + 100, 512) is None      # tail 100 not a power of two
    assert orc.block_layout(4096, 3000) is None           # block not a power of two
    assert orc.block_layout(768, 512) == (1, 256)


def test_fp16_rotation_is_f64_rotation_rounded_once(orc):
    wl = inputs.llama2_7b_decode()
    x = inputs.activations(wl, 3, 4096)
    y = orc.rotate(x, 4096)
    for m in range(3):
        ref = orc.rotate_row_f64(x[m].astype(np.float64), 4096).astype(np.float32)
        assert np.array_equal(y[m], ref)


def test_rotation_equivalence_eq5(orc):
    # X W^T = (X R)(W R)^T: the same R on both operands leaves the product unchanged
    rng = np.random.default_rng(2)
    K, B = 1536, 512
    x = rng.standard_normal((3, K))
    w = rng.standard_normal((5, K))
    xr = np.stack([orc.rotate_row_f64(r, B) for r in x])
    wr = np.stack([orc.rotate_row_f64(r, B) for r in w])
    assert np.allclose(xr @ wr.T, x @ w.T, rtol=1e-12, atol=1e-10)


# ---------------------------------------------------------------- quantizer (Eq. 2, Eq. 3)
def test_quantizer_golden_worked_examples(orc):
    for ln in _rows("quant_worked.txt"):
        bits, ys, s, cs = [p.strip() for p in ln.split("|")]
        y = np.array([[float(v) for v in ys.split()]], dtype=np.float32)
        c, sc = orc.quant_rows(y, int(bits))
        assert sc[0] == np.float32(float(s))
        assert c[0].tolist() == [int(v) for v in cs.split()]


@pytest.mark.parametrize("bits", [4, 8])
def test_quantizer_error_bound_range_and_extremes(orc, bits):
    wl = inputs.llama2_13b_prefill()
    x = inputs.activations(wl, 16, 5120)
    y = orc.rotate(x, 1024)
    c, s = orc.quant_rows(y, bits)
    qmax = (1 << (bits - 1)) - 1
    assert c.min() >= -(qmax + 1) and c.max() <= qmax
    err = np.abs(y.astype(np.float64) - s[:, None].astype(np.float64) * c)        # Eq. 3
    assert np.all(err <= s[:, None] * (0.5 + 1e-6))
    arg = np.argmax(np.abs(y), axis=1)
    assert np.array_equal(np.abs(c[np.arange(16), arg]), np.full(16, qmax))


@pytest.mark.parametrize("bits", [4, 8])
def test_one_hot_closed_form(orc, bits):
    # x = alpha e_j in one block: |y| = |alpha| / sqrt(B) everywhere, codes = +-qmax with
    # the signs of Hadamard row j, zero quantization error
    B, j, alpha = 256, 77, -3.0
    x = np.zeros((1, B), dtype=np.float16)
    x[0, j] = alpha
    c, s = orc.rotate_quant_act(x, B, bits)
    qmax = (1 << (bits - 1)) - 1
    assert np.array_equal(c[0], (np.sign(alpha) * qmax * sylvester(B)[j]).astype(np.int8))
    y = orc.rotate(x, B)
    assert np.allclose(s[0] * c[0].astype(np.float64), y[0], rtol=1e-6, atol=0)


def test_a8_error_below_a4_error_and_step_ratio(orc):
    # Section 3.3 Eq. 22: the step shrinks ~2^-(8-4); with symmetric qmax the ratio is 7/127
    wl = inputs.single_linear()
    x = inputs.activations(wl, 16, 256)
    y = orc.rotate(x, 256).astype(np.float64)
    c4, s4 = orc.quant_rows(y, 4)
    c8, s8 = orc.quant_rows(y, 8)
    e4 = np.sum((y - s4[:, None] * c4) ** 2)
    e8 = np.sum((y - s8[:, None] * c8) ** 2)
    assert e8 < e4
    assert np.allclose(s8 / s4, 7.0 / 127.0, rtol=1e-6)
    assert 1.0 / 20 < 7.0 / 127.0 < 1.0 / 14          # "approximately 2^-4"


def test_uniform_noise_model_mse(orc):
    # Eq. 17: uniform rounding noise, E[e^2] = s^2 / 12 per element (statistical, +-10%)
    rng = np.random.default_rng(9)
    y = rng.standard_normal((64, 4096)).astype(np.float32)
    for bits in (4, 8):
        c, s = orc.quant_rows(y, bits)
        mse = np.mean((y.astype(np.float64) - s[:, None] * c) ** 2 / (s[:, None] ** 2))
        assert abs(mse - 1.0 / 12.0) < 0.1 / 12.0


def test_zero_row_and_bad_bits(orc):
    c, s = orc.quant_rows(np.zeros((2, 64), dtype=np.float32), 4)
    assert np.all(c == 0) and np.all(s == 0)
    with pytest.raises(ValueError):
        orc.quant_rows(np.ones((1, 8), dtype=np.float32), 5)


# ---------------------------------------------------------------- GEMM and epilogue
def test_gemm_brute_force_tiny(orc):
    rng = np.random.default_rng(4)
    for M, N, K in [(1, 1, 1), (3, 5, 7), (17, 9, 64), (64, 48, 33)]:
        a = rng.integers(-128, 128, size=(M, K), dtype=np.int8)
        w = rng.integers(-8, 8, size=(N, K), dtype=np.int8)
        ref = a.astype(np.int64) @ w.astype(np.int64).T
        assert np.array_equal(orc.gemm_i32(a, w), ref.astype(np.int32))
    a = rng.integers(-128, 128, size=(2, 3), dtype=np.int8)
    w = rng.integers(-8, 8, size=(4, 3), dtype=np.int8)
    got = orc.gemm_i32(a, w)
    # element by element, written out: acc[m][n] = sum_k a[m][k] w[n][k]
    for m in range(2):
        for n in range(4):
            assert got[m, n] == sum(int(a[m, k]) * int(w[n, k]) for k in range(3))


def test_gemm_closed_forms_and_int32_range(orc):
    K = 28672
    a = np.full((1, K), -8, dtype=np.int8)
    w = np.full((2, K), -8, dtype=np.int8)
    assert np.all(orc.gemm_i32(a, w) == 64 * K)
    a8 = np.full((1, K), 127, dtype=np.int8)
    w7 = np.full((1, K), -7, dtype=np.int8)
    assert orc.gemm_i32(a8, w7)[0, 0] == -127 * 7 * K
    big = 140000
    with pytest.raises(OverflowError):
        orc.gemm_i32(np.full((1, big), 127, dtype=np.int8), np.full((1, big), 127, dtype=np.int8))


def test_epilogue_golden(orc):
    for ln in _rows("epilogue_worked.txt"):
        acc, sa, sw, hx, _ = [p.strip() for p in ln.split("|")]
        out = orc.epilogue(np.array([[int(acc)]]), np.array([float(sa)]), np.array([float(sw)]))
        assert out.view(np.uint16)[0, 0] == int(hx, 16), ln


def test_epilogue_matches_numpy_fp32_then_fp16(orc):
    rng = np.random.default_rng(6)
    acc = rng.integers(-3_000_000, 3_000_000, size=(7, 33)).astype(np.int32)
    sa = (rng.random(7) * 0.05).astype(np.float32)
    sw = (rng.random(33) * 0.01).astype(np.float32)
    ref = ((acc.astype(np.float32) * sa[:, None]) * sw[None, :]).astype(np.float16)
    got = orc.epilogue(acc, sa, sw)
    assert np.array_equal(got.view(np.uint16), ref.view(np.uint16))


# ---------------------------------------------------------------- whole layer
def test_qlinear_composition_and_accuracy_order(orc):
    wl = inputs.single_linear()
    x = inputs.activations(wl, 16, 256)
    W = inputs.weights(512, 256)
    q, sw = orc.pack_weights(W, 256)
    assert q.min() >= -8 and q.max() <= 7
    ref = x.astype(np.float64) @ W.astype(np.float64).T
    errs = {}
    for bits in (4, 8):
        r = orc.qlinear(x, 256, bits, q, sw)
        c, sa = orc.rotate_quant_act(x, 256, bits)
        assert np.array_equal(r["codes"], c) and np.array_equal(r["sa"], sa)
        acc = orc.gemm_i32(c, q)
        assert np.array_equal(r["acc"], acc)
        assert np.array_equal(r["out"].view(np.uint16), orc.epilogue(acc, sa, sw).view(np.uint16))
        errs[bits] = np.linalg.norm(r["out"].astype(np.float64) - ref) / np.linalg.norm(ref)
    # Eq. 5 makes the rotated product equal X W^T; only quantization error remains
    assert errs[8] < errs[4] < 0.35
    assert errs[8] < 0.2


def test_weight_codes_never_reach_minus_eight(orc):
    # symmetric RTN with s = absmax / 7 keeps |W'/s| <= 7: the -8 code is never produced
    W = inputs.weights(64, 4096, layer=3, proj=2)
    q, _ = orc.pack_weights(W, 4096)
    assert q.min() >= -7


def test_nibble_golden_and_roundtrip(orc):
    for ln in _rows("nibbles.txt"):
        cs, bs = [p.strip() for p in ln.split("|")]
        codes = np.array([[int(v) for v in cs.split()]], dtype=np.int8)
        packed = orc.pack_nibbles(codes)
        assert packed[0].tolist() == [int(b, 16) for b in bs.split()]
        assert np.array_equal(orc.unpack_nibbles(packed, codes.shape[1]), codes)


# ---------------------------------------------------------------- residual statistics (Eqs. 8-13)
def test_jump_ratio_rotation_invariant_and_closed_forms(orc):
    rng = np.random.default_rng(12)
    T, d, B = 8, 1024, 1024
    x = rng.standard_normal((T, d)).astype(np.float32)
    dx = (3.0 * rng.standard_normal((T, d))).astype(np.float32)
    jr, snr = orc.residual_stats(x, dx, 4)
    xr = np.stack([orc.rotate_row_f64(r.astype(np.float64), B) for r in x]).astype(np.float32)
    dr = np.stack([orc.rotate_row_f64(r.astype(np.float64), B) for r in dx]).astype(np.float32)
    jr_r, _ = orc.residual_stats(xr, dr, 4)
    assert abs(jr_r - jr) < 1e-5 * jr                                    # Eq. 13
    ref = np.mean(np.linalg.norm(dx.astype(np.float64), axis=1) /
                  (np.linalg.norm(x.astype(np.float64), axis=1) + 1e-6))
    assert abs(jr - ref) < 1e-9 * ref                                    # Eqs. 8-9
    jr0, _ = orc.residual_stats(x, np.zeros_like(x), 8)
    assert jr0 == 0.0
    # larger update => lower historical SNR at the same bit width (Eq. 19 trend)
    _, snr_small = orc.residual_stats(x, (0.1 * dx).astype(np.float32), 4)
    assert snr < snr_small
    # 8 bits preserve history better than 4 bits
    _, snr8 = orc.residual_stats(x, dx, 8)
    assert snr8 > snr


def test_historical_snr_exact_grid(orc):
    # x + dx on the 4-bit grid with s = 1: quantization is exact, so SNR = 10 log10(|x|^2/eps)
    x = np.array([[1.0, -2.0, 3.0, 0.0]], dtype=np.float32)
    dx = np.array([[6.0, 0.0, -1.0, 2.0]], dtype=np.float32)     # x + dx = [7, -2, 2, 2]
    _, snr = orc.residual_stats(x, dx, 4, eps=1e-6)
    assert abs(snr - 10 * math.log10(14.0 / 1e-6)) < 1e-9


def test_historical_snr_and_jump_ratio_two_token_closed_form(orc):
    # Token A: x + dx = [7, 3.5, 0, 0], so s = 1 at 4 bits and the tie 3.5 rounds to 4;
    # xhat - x = Q(x + dx) - (x + dx) = [0, 0.5, 0, 0]: the numerator is |x|^2 = 30 (not
    # |xhat|^2 = 32.25), the error 0.25.  Token B: x + dx = [7, 0, 0, 0] is on the grid.
    # The layer value is the mean of the per-token values in dB (Eq. 11), and JR the mean
    # of the per-token ratios (Eq. 9).
    eps = 1e-6
    x = np.array([[1.0, 2.0, 3.0, 4.0], [2.0, 0.0, 0.0, 0.0]], dtype=np.float32)
    dx = np.array([[6.0, 1.5, -3.0, -4.0], [5.0, 0.0, 0.0, 0.0]], dtype=np.float32)
    jr, snr = orc.residual_stats(x, dx, 4, eps=eps)
    snr_a = 10 * math.log10(30.0 / (0.25 + eps))
    snr_b = 10 * math.log10(4.0 / eps)
    assert abs(snr - (snr_a + snr_b) / 2) < 1e-9
    jr_ref = (math.sqrt(63.25) / (math.sqrt(30.0) + eps) + 5.0 / (2.0 + eps)) / 2
    assert abs(jr - jr_ref) < 1e-12


def test_sensitive_set_golden():
    # Eq. 21 instantiated for the layer counts of the workloads (0-indexed masks)
    gold = {int(a): [int(v) for v in b.split()] for a, b in
            (ln.split("|") for ln in _rows("sensitive_set.txt"))}
    for L, layers in gold.items():
        assert layers == [0, 1, 2, L - 1]


# ---------------------------------------------------------------- randomized Hadamard
def _signs(K, seed):
    return np.where(np.random.default_rng(seed).random(K) < 0.5, -1, 1).astype(np.int8)


def test_randomized_hadamard_all_plus_signs_is_plain(orc):
    x = inputs.to_f16(np.random.default_rng(40).standard_normal((5, 768)).astype(np.float32))
    assert np.array_equal(orc.rotate(x, 256, signs=np.ones(768, np.int8)), orc.rotate(x, 256))
    c0, s0 = orc.rotate_quant_act(x, 256, 4)
    c1, s1 = orc.rotate_quant_act(x, 256, 4, signs=np.ones(768, np.int8))
    assert np.array_equal(c0, c1) and np.array_equal(s0, s1)


def test_randomized_hadamard_brute_force(orc):
    # y = (x * d) blockdiag(H_8, H_8, H_4) / sqrt(block) with the textbook Sylvester matrix:
    # the fp16 inputs make every fp64 sum exact, so the fp32 results agree bit for bit.
    K, B = 20, 8
    x = inputs.to_f16(np.random.default_rng(41).standard_normal((3, K)).astype(np.float32))
    d = _signs(K, 42)
    xs = x.astype(np.float64) * d
    R = np.zeros((K, K))
    R[0:8, 0:8] = sylvester(8) / math.sqrt(8)
    R[8:16, 8:16] = sylvester(8) / math.sqrt(8)
    R[16:20, 16:20] = sylvester(4) / math.sqrt(4)
    ref = (xs @ R).astype(np.float32)
    assert np.array_equal(orc.rotate(x, B, signs=d), ref)
    # a sign flip is a sign flip of the input element (and nothing else)
    d2 = d.copy()
    d2[5] = -d2[5]
    x2 = x.copy()
    x2[:, 5] = -x2[:, 5]
    assert np.array_equal(orc.rotate(x2, B, signs=d2), orc.rotate(x, B, signs=d))


def test_randomized_hadamard_is_orthogonal_and_folds_into_weights(orc):
    K, B = 512, 128
    rng = np.random.default_rng(43)
    d = _signs(K, 44)
    x = inputs.to_f16(rng.standard_normal((4, K)).astype(np.float32))
    W = inputs.to_f16((0.02 * rng.standard_normal((6, K))).astype(np.float32))
    y = orc.rotate(x, B, signs=d).astype(np.float64)
    yw = orc.rotate(W, B, signs=d).astype(np.float64)
    xf, wf = x.astype(np.float64), W.astype(np.float64)
    assert np.allclose(np.linalg.norm(y, axis=1), np.linalg.norm(xf, axis=1), rtol=1e-6)   # (DR)^T DR = I
    assert np.allclose(y @ yw.T, xf @ wf.T, rtol=1e-5, atol=1e-6)                          # Eq. 5 with R' = DR
    # a different sign vector gives a different rotation
    assert not np.array_equal(orc.rotate(x, B, signs=_signs(K, 45)), orc.rotate(x, B, signs=d))


def test_randomized_hadamard_weights_and_layer(orc):
    K, B, N, M = 256, 64, 32, 5
    rng = np.random.default_rng(46)
    d = _signs(K, 47)
    W = inputs.to_f16((0.02 * rng.standard_normal((N, K))).astype(np.float32))
    x = inputs.to_f16(rng.standard_normal((M, K)).astype(np.float32))
    q, sw = orc.pack_weights(W, B, signs=d)
    qc, sc = orc.rotate_quant_act(W, B, 4, signs=d)
    assert np.array_equal(q, qc) and np.array_equal(sw, sc)
    r = orc.qlinear(x, B, 8, q, sw, signs=d)
    codes, sa = orc.rotate_quant_act(x, B, 8, signs=d)
    assert np.array_equal(r["codes"], codes) and np.array_equal(r["sa"], sa)
    assert np.array_equal(r["acc"], codes.astype(np.int64) @ q.astype(np.int64).T)
    assert np.array_equal(r["out"].view(np.uint16), orc.epilogue(r["acc"], sa, sw).view(np.uint16))


# ---------------------------------------------------------------- KV4 quantizer
def test_kv4_golden_worked_examples(orc):
    for ln in _rows("kv4_worked.txt"):
        g, xs, s, cs = [p.strip() for p in ln.split("|")]
        x = inputs.to_f16(np.array([[float(v) for v in xs.split()]], dtype=np.float32))
        codes, scales = orc.kv4_quantize(x, int(g))
        assert scales[0, 0] == np.float32(float(s))
        assert codes[0].tolist() == [int(v) for v in cs.split()]


def test_kv4_groups_are_independent_and_bounded(orc):
    rng = np.random.default_rng(48)
    x = inputs.to_f16((rng.standard_normal((6, 512)) * np.float32(3.0) ** rng.integers(-3, 4, (6, 1))).astype(np.float32))
    x[2, 128:256] = 0                                          # an all-zero group
    codes, scales = orc.kv4_quantize(x, 128)
    assert codes.shape == (6, 512) and scales.shape == (6, 4)
    xf = x.astype(np.float32).reshape(6, 4, 128)
    c = codes.reshape(6, 4, 128).astype(np.float32)
    assert np.all(np.abs(codes) <= 7)                          # symmetric: -8 is never produced
    assert np.all(scales == np.max(np.abs(xf), axis=2) / np.float32(7))
    err = np.abs(xf - scales[:, :, None] * c)
    assert np.all(err <= scales[:, :, None] * 0.5 * (1 + 1e-6))   # round-trip error <= s/2
    assert scales[2, 1] == 0 and np.all(codes[2, 128:256] == 0)
    # each group is the per-token quantizer of Eq. 2 applied to that group alone
    for gi in range(4):
        cg, sg = orc.quant_rows(xf[:, gi, :], 4)
        assert np.array_equal(cg, codes[:, gi * 128:(gi + 1) * 128]) and np.array_equal(sg, scales[:, gi])
    with pytest.raises(ValueError):
        orc.kv4_quantize(x[:, :200], 128)


# ---------------------------------------------------------------- sensitive-layer policy
def test_policy_mask_closed_form(orc):
    jr = np.array([0.9, 0.9, 0.1, 0.5, 0.5, 0.3], dtype=np.float64)
    snr = np.array([5.0, 25.0, 5.0, 20.0, 19.0, 10.0], dtype=np.float64)
    bits = orc.policy_mask(jr, snr, tau_jr=0.3, tau_snr=20.0)
    # Eq. 20: JR > tau_JR and SNR < tau_SNR, both strict (layer 3 has SNR == tau, layer 5 JR == tau)
    assert bits.tolist() == [8, 4, 4, 4, 8, 4]
    assert orc.policy_mask(jr, snr, tau_jr=-1.0, tau_snr=1e9).tolist() == [8] * 6
    assert orc.policy_mask(jr, snr, tau_jr=1.0, tau_snr=1e9).tolist() == [4] * 6


# ---------------------------------------------------------------- non-power-of-two tail blocks
def test_paley_h12_golden(orc):
    """Rows 0 and 1 of Paley's H_12 and the quadratic character mod 11, worked by hand."""
    chi, row0, row1 = ([int(v) for v in ln.split()] for ln in _rows("paley_q11.txt"))
    assert [orc.paley_entry(12, 0, j) for j in range(12)] == row0
    assert [orc.paley_entry(12, 1, j) for j in range(12)] == row1
    assert [orc.paley_entry(12, 1, 1 + a) for a in range(1, 11)] == chi


@pytest.mark.parametrize("p", [12, 20, 24, 44, 48, 60, 68, 72, 80, 84])
def test_paley_matrices_are_hadamard(orc, p):
    """H_p H_p^T = p I exactly, H_p = I + S with S skew-symmetric, first row all ones
    (Paley's first construction for the prime p - 1 = 3 mod 4)."""
    H = np.array([[orc.paley_entry(p, i, j) for j in range(p)] for i in range(p)], dtype=np.int64)
    assert np.array_equal(H @ H.T, p * np.eye(p, dtype=np.int64))
    S = H - np.eye(p, dtype=np.int64)
    assert np.array_equal(S.T, -S)
    assert np.all(H[0] == 1) and np.all(np.abs(H) == 1)


def test_paley_entry_rejects_other_orders(orc):
    for p in (10, 16, 28, 36, 52):   # not a multiple of 4, or p - 1 composite (15, 27, 35, 51)
        assert orc.paley_entry(p, 1, 2) == 0


@pytest.mark.parametrize("r,expect", [(2816, (44, 6)), (1536, (12, 7)), (512, (1, 9)), (96, (12, 3)),
                                      (160, (20, 3)), (6, None), (3, None), (44, (44, 0))])
def test_tail_factor(orc, r, expect):
    assert orc.tail_factor(r) == expect


@pytest.mark.parametrize("r", [12 * 16, 44 * 4, 20 * 8, 2816])
def test_tail_block_is_kronecker_and_orthogonal(orc, r):
    """The tail block's matrix is H_p (x) H_(2^k) (numpy's kron of the two factors) and is a
    Hadamard matrix of order r."""
    p, k = orc.tail_factor(r)
    Hp = np.array([[orc.paley_entry(p, i, j) for j in range(p)] for i in range(p)], dtype=np.int64)
    ref = np.kron(Hp, sylvester(1 << k))
    idx = range(r) if r <= 256 else np.random.default_rng(r).choice(r, 96, replace=False)
    for i in idx:
        assert [orc.tail_entry(r, int(i), j) for j in range(r)] == ref[int(i)].tolist()
    assert np.array_equal(ref @ ref.T, r * np.eye(r, dtype=np.int64))


@pytest.mark.parametrize("K,B", [(256 + 192, 256), (1024 + 176, 1024), (4096 + 2816, 4096)])
def test_rotation_with_paley_tail_is_orthogonal(orc, K, B):
    """R^T R = I (Section 2 Eq. 4) with a non-power-of-two tail: the rotated basis rows are
    orthonormal, norms are kept, and the tail block equals x_tail H_r / sqrt(r)."""
    q, r = orc.block_layout(K, B)
    assert r == K - q * B and orc.tail_factor(r)[0] > 1
    rng = np.random.default_rng(K)
    for _ in range(3):
        x = rng.standard_normal(K)
        y = orc.rotate_row_f64(x, B)
        assert abs(np.linalg.norm(y) - np.linalg.norm(x)) < 1e-10 * np.linalg.norm(x)
    p, k = orc.tail_factor(r)
    Hp = np.array([[orc.paley_entry(p, i, j) for j in range(p)] for i in range(p)], dtype=np.float64)
    Hr = np.kron(Hp, sylvester(1 << k).astype(np.float64))
    x = rng.standard_normal(K)
    y = orc.rotate_row_f64(x, B)
    assert np.allclose(y[q * B:], x[q * B:] @ Hr / math.sqrt(r), rtol=0, atol=1e-12)
    if K <= 1200:
        R = np.array([orc.rotate_row_f64(e, B) for e in np.eye(K)])
        assert np.allclose(R @ R.T, np.eye(K), atol=1e-12)


def test_fold_equivalence_with_paley_tail(orc):
    """Eq. 5 with a non-power-of-two tail: (X R)(W R)^T = X W^T."""
    K, B = 256 + 96, 256
    rng = np.random.default_rng(5)
    X = rng.standard_normal((3, K))
    W = rng.standard_normal((4, K))
    XR = np.array([orc.rotate_row_f64(x, B) for x in X])
    WR = np.array([orc.rotate_row_f64(w, B) for w in W])
    assert np.allclose(XR @ WR.T, X @ W.T, atol=1e-10)


def test_randomized_hadamard_with_paley_tail(orc):
    """QuaRot's randomized Hadamard D R (Sections 1 and 4.2) over a non-power-of-two tail
    block: D R is still orthogonal (norms kept, Eq. 4), it equals the plain rotation of
    x * d, it folds into the weights (Eq. 5), and the packed weights are the activation
    quantizer applied to W with the same D R."""
    K, B = 256 + 96, 256        # tail 96 = 12 x 8: H_12 (x) H_8
    rng = np.random.default_rng(48)
    d = _signs(K, 49)
    x = inputs.to_f16(rng.standard_normal((3, K)).astype(np.float32))
    W = inputs.to_f16((0.02 * rng.standard_normal((5, K))).astype(np.float32))
    y = orc.rotate(x, B, signs=d).astype(np.float64)
    xd = (x.astype(np.float64) * d).astype(np.float16)   # exact: a sign flip of binary16 values
    assert np.array_equal(orc.rotate(xd, B), orc.rotate(x, B, signs=d))
    xf, wf = x.astype(np.float64), W.astype(np.float64)
    assert np.allclose(np.linalg.norm(y, axis=1), np.linalg.norm(xf, axis=1), rtol=1e-6)
    yw = orc.rotate(W, B, signs=d).astype(np.float64)
    assert np.allclose(y @ yw.T, xf @ wf.T, rtol=1e-5, atol=1e-6)
    q, sw = orc.pack_weights(W, B, signs=d)
    qc, sc = orc.rotate_quant_act(W, B, 4, signs=d)
    assert np.array_equal(q, qc) and np.array_equal(sw, sc)
