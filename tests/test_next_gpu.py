"""Parity of the CUDA path with the oracle for the three items beyond the plain layer:
the randomized Hadamard rotation (QuaRot's diagonal, Sections 1 and 4.2), the
group-wise 4-bit KV-cache quantizer (Section 4.2) and the sensitive-layer policy
(Section 3.1 Eqs. 8-11, Section 3.3 Eq. 20)."""
import numpy as np
import pytest

import parity
from paper_2606_12487_gb300 import inputs

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu
DEV = "cuda"


@pytest.fixture(scope="module")
def dp():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2606_12487_gb300 import dptq
    dptq.load()
    return dptq


def _signs(K, seed):
    return np.where(np.random.default_rng(seed).random(K) < 0.5, -1, 1).astype(np.int8)


# ---------------------------------------------------------------- randomized Hadamard
@pytest.mark.parametrize("K,B,M", [(256, 256, 8), (4096, 4096, 4), (11008, 256, 3), (768, 512, 3)])
def test_randomized_rotation_and_codes(dp, orc, K, B, M):
    wl = inputs.llama2_7b_decode()
    x = inputs.activations(wl, M, K)
    d = _signs(K, K + B)
    xd = torch.from_numpy(x).to(DEV)
    sd = torch.from_numpy(d).to(DEV)
    y = torch.empty((M, K), dtype=torch.float32, device=DEV)
    dp.dptq_rotate_act_rh(xd, B, sd, y)
    y_ref = orc.rotate(x, B, signs=d)
    parity.check_rotation(y.cpu().numpy(), y_ref)
    for bits in (4, 8):
        codes = torch.empty((M, K // 2) if bits == 4 else (M, K), dtype=torch.uint8 if bits == 4 else torch.int8,
                            device=DEV)
        s = torch.empty((M,), dtype=torch.float32, device=DEV)
        dp.dptq_rotate_quant_act_rh(xd, B, bits, sd, codes, s)
        c = codes.cpu().numpy()
        c = orc.unpack_nibbles(c, K) if bits == 4 else c
        c_ref, s_ref = orc.rotate_quant_act(x, B, bits, signs=d)
        parity.check_scales(s.cpu().numpy(), s_ref)
        parity.check_codes(c, c_ref, y_ref, s_ref, bits)
    # plain signs reproduce the plain rotation bit for bit
    y1 = torch.empty_like(y)
    dp.dptq_rotate_act_rh(xd, B, torch.ones(K, dtype=torch.int8, device=DEV), y1)
    y0 = torch.empty_like(y)
    dp.dptq_rotate_act(xd, B, y0)
    torch.cuda.synchronize()
    assert torch.equal(y0, y1)


@pytest.mark.parametrize("M,N,K,B", [(16, 512, 256, 256), (32, 128, 4096, 4096), (5, 384, 11008, 256),
                                     (130, 256, 1024, 1024)])
def test_randomized_qlinear(dp, orc, M, N, K, B):
    wl = inputs.llama2_7b_decode()
    x = inputs.activations(wl, M, K)
    W = inputs.weights(N, K, layer=3, proj=2)
    d = _signs(K, 7 * K + M)
    layer = dp.dptq_pack_weights_rh(torch.from_numpy(W).to(DEV), B, d)
    q_ref, sw_ref = orc.pack_weights(W, B, signs=d)
    wq, sw = dp.dptq_get_packed(layer)
    assert np.array_equal(orc.unpack_nibbles(wq, K), q_ref) and np.array_equal(sw, sw_ref)
    xd = torch.from_numpy(x).to(DEV)
    for bits in (4, 8):
        out = torch.empty((M, N), dtype=torch.float16, device=DEV)
        dp.dptq_qlinear(layer, xd, bits, out)                  # fused launch for small M
        two = torch.empty_like(out)
        dp.dptq_qlinear_quantize(layer, xd, bits)
        dp.dptq_qlinear_gemm(layer, M, bits, two)              # rotate-quantize + GEMM launches
        torch.cuda.synchronize()
        assert torch.equal(out.view(torch.int16), two.view(torch.int16))
        r = orc.qlinear(x, B, bits, q_ref, sw_ref, signs=d)
        cg = torch.empty((M, K // 2) if bits == 4 else (M, K), dtype=torch.uint8 if bits == 4 else torch.int8,
                         device=DEV)
        sg = torch.empty((M,), dtype=torch.float32, device=DEV)
        dp.dptq_rotate_quant_act_rh(xd, B, bits, torch.from_numpy(d).to(DEV), cg, sg)
        c = cg.cpu().numpy()
        c = orc.unpack_nibbles(c, K) if bits == 4 else c
        ok = np.all(c == r["codes"], axis=1)
        parity.check_out(out.cpu().numpy()[ok], r["out"][ok])
    layer.close()


def test_randomized_pack_rejects_bad_signs(dp):
    W = torch.from_numpy(inputs.weights(128, 256)).to(DEV)
    d = np.ones(256, np.int8)
    d[7] = 0
    with pytest.raises(dp.DptqError):
        dp.dptq_pack_weights_rh(W, 256, d)


# ---------------------------------------------------------------- KV4
# (5, 384): 15 groups of 128, a ragged last set of four for the group-128 kernel
@pytest.mark.parametrize("rows,cols,group", [(1, 128, 128), (37, 1024, 128), (64, 4096, 128), (9, 2048, 256),
                                             (3, 3072, 1024), (5, 384, 128)])
def test_kv4_bit_exact(dp, orc, rows, cols, group):
    rng = np.random.default_rng(rows * cols + group)
    x = (rng.standard_normal((rows, cols)) * np.float32(4.0) ** rng.integers(-4, 4, (rows, 1))).astype(np.float32)
    x[0, :group] = 0                                       # an all-zero group
    if rows > 2:
        x[2, 5] = 65504.0                                  # fp16 maximum
        x[1, group:2 * group] = np.float32(1e-6) * rng.standard_normal(group).astype(np.float32)   # subnormal range
    if rows > 3:
        # a group with s = 1 exactly and x / s on half-integers: every code is a tie
        # (round half to even), e.g. 0.5 -> 0, 1.5 -> 2, -2.5 -> -2
        x[3, :group] = (rng.integers(-7, 7, group) + np.float32(0.5)).astype(np.float32)
        x[3, 0] = 7.0
    xh = inputs.to_f16(x)
    kv = torch.from_numpy(xh).to(DEV)
    codes = torch.empty((rows, cols // 2), dtype=torch.uint8, device=DEV)
    scales = torch.empty((rows, cols // group), dtype=torch.float32, device=DEV)
    dp.dptq_kv4_quantize(kv, group, codes, scales)
    torch.cuda.synchronize()
    c_ref, s_ref = orc.kv4_quantize(xh, group)
    assert np.array_equal(scales.cpu().numpy(), s_ref)
    assert np.array_equal(orc.unpack_nibbles(codes.cpu().numpy(), cols), c_ref)


def test_kv4_llama_cache_shape(dp, orc):
    # one layer's K cache of LLaMA-2-7B decode: 32 heads x 128 dims, 1024 tokens, viewed
    # as [tokens * heads, 128] groups; sampled rows compared
    T, H, D = 1024, 32, 128
    x = inputs.to_f16(np.random.default_rng(5).standard_normal((T * H, D)).astype(np.float32))
    kv = torch.from_numpy(x).to(DEV)
    codes = torch.empty((T * H, D // 2), dtype=torch.uint8, device=DEV)
    scales = torch.empty((T * H, 1), dtype=torch.float32, device=DEV)
    dp.dptq_kv4_quantize(kv, 128, codes, scales)
    torch.cuda.synchronize()
    rows = np.random.default_rng(6).choice(T * H, 512, replace=False)
    c_ref, s_ref = orc.kv4_quantize(x[rows], 128)
    assert np.array_equal(scales.cpu().numpy()[rows], s_ref)
    assert np.array_equal(orc.unpack_nibbles(codes.cpu().numpy()[rows], D), c_ref)


# ---------------------------------------------------------------- sensitivity policy
def _residual_streams(L, T, d, seed):
    """Synthetic residual states and updates with a few large-update layers (massive
    activations appearing in early and late layers, Section 3.1)."""
    rng = np.random.default_rng(seed)
    x = rng.standard_normal((L, T, d)).astype(np.float32)
    dx = (0.05 * rng.standard_normal((L, T, d))).astype(np.float32)
    for l in (0, 1, L - 1):
        dx[l, :, :4] += np.float32(40.0) * rng.standard_normal((T, 4)).astype(np.float32)
    x[0, 3] = 0
    dx[0, 3] = 0                                           # a zero token (s = 0)
    return x, dx


# Small cases (one token per CTA), ranges of several tokens per CTA that wrap the
# kernel's ring of token stages and cross layer boundaries (8 x 300 and 4 x 300 tokens),
# and a token wider than 4096 (the unstaged kernel).
@pytest.mark.parametrize("L,T,d,bits", [(6, 16, 256, 4), (4, 8, 4096, 4), (3, 5, 1000, 8),
                                        (8, 300, 512, 4), (4, 300, 4096, 8), (3, 7, 5120, 4)])
def test_policy_stats_and_mask(dp, orc, L, T, d, bits):
    x, dx = _residual_streams(L, T, d, L * T + d)
    jr_ref = np.empty(L)
    snr_ref = np.empty(L)
    for l in range(L):
        jr_ref[l], snr_ref[l] = orc.residual_stats(x[l], dx[l], bits, 1e-6)
    tau_jr = float(np.median(jr_ref))
    tau_snr = float(np.median(snr_ref)) + 0.5
    xd, dd = torch.from_numpy(x).to(DEV), torch.from_numpy(dx).to(DEV)
    jr = torch.empty((L,), dtype=torch.float64, device=DEV)
    snr = torch.empty((L,), dtype=torch.float64, device=DEV)
    bits_out = torch.empty((L,), dtype=torch.uint8, device=DEV)
    dp.dptq_sensitivity_policy(xd, dd, bits, 1e-6, tau_jr, tau_snr, jr, snr, bits_out)
    torch.cuda.synchronize()
    jr_g, snr_g, m_g = jr.cpu().numpy(), snr.cpu().numpy(), bits_out.cpu().numpy()
    # fp32 per element, fp64 per token: JR within 1e-5 relative, SNR within 1e-3 dB
    assert np.all(np.abs(jr_g - jr_ref) <= 1e-5 * np.abs(jr_ref) + 1e-12)
    # a token with x = dx = 0 makes its layer's SNR -inf on both sides
    assert np.array_equal(np.isinf(snr_g), np.isinf(snr_ref)) and np.array_equal(snr_g[np.isinf(snr_g)],
                                                                                 snr_ref[np.isinf(snr_ref)])
    fin = np.isfinite(snr_ref)
    assert np.all(np.abs(snr_g[fin] - snr_ref[fin]) <= 1e-3)
    m_ref = orc.policy_mask(jr_ref, snr_ref, tau_jr, tau_snr)
    clear = (np.abs(jr_ref - tau_jr) > 1e-5 * np.abs(tau_jr)) & ~(np.abs(snr_ref - tau_snr) <= 1e-3)
    assert np.array_equal(m_g[clear], m_ref[clear])
    assert set(m_g.tolist()) <= {4, 8}
