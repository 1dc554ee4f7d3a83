"""Parity of the CUDA path (through the C ABI) with the CPU oracle, on seeded synthetic
inputs: the rotation, the codes and scales, the packed weights, the exact integer
accumulators, the fp16 outputs, edge cases, and full-size workloads on sampled outputs."""
import numpy as np
import pytest

import parity
from paper_2606_12487_gb300 import inputs

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def dp():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2606_12487_gb300 import dptq
    dptq.load()
    return dptq


DEV = "cuda"


def gpu_rotate(dp, x, B):
    xd = torch.from_numpy(x).to(DEV)
    y = torch.empty(x.shape, dtype=torch.float32, device=DEV)
    dp.dptq_rotate_act(xd, B, y)
    return y.cpu().numpy()


def gpu_codes(dp, x, B, bits, orc):
    M, K = x.shape
    xd = torch.from_numpy(x).to(DEV)
    codes = torch.empty((M, K // 2) if bits == 4 else (M, K), dtype=torch.uint8 if bits == 4 else torch.int8,
                        device=DEV)
    s = torch.empty((M,), dtype=torch.float32, device=DEV)
    dp.dptq_rotate_quant_act(xd, B, bits, codes, s)
    c = codes.cpu().numpy()
    c = orc.unpack_nibbles(c, K) if bits == 4 else c
    return c, s.cpu().numpy()


def edge_rows(K):
    rng = np.random.default_rng(21)
    rows = np.zeros((6, K), dtype=np.float32)
    rows[1, K // 3] = 2.5                       # single nonzero
    rows[2] = rng.standard_normal(K)
    rows[2, 5] = 65504.0                        # saturated fp16 outlier
    rows[3] = -65504.0 * (rng.random(K) < 0.01)
    rows[4] = rng.standard_normal(K) * 1e-6     # fp16 subnormal range
    rows[5] = 1.0                               # constant row
    return inputs.to_f16(rows)


# Pairs (a, b): a row with a at position i and b at position j of every Hadamard block
# rotates to +-(a + b) / sqrt(B) and +-(a - b) / sqrt(B), so y / s = qmax (a - b) / (a + b)
# wherever H[i][k] != H[j][k].  For (3k, k) that is 3.5 at 4 bits and 63.5 at 8 bits;
# (27, 1) gives 6.5 at 4 bits: exact rounding ties (Eq. 2, round half to even), half of
# every row.
TIE_PAIRS = [(3, 1), (27, 1), (381, 127), (9, 3), (6, 2), (15, 5), (33, 11), (27, 9)]


def tie_rows(K, B, n=8):
    """n fp16 rows whose rotated values sit exactly on half-integers of the code grid."""
    rows = np.zeros((n, K), dtype=np.float32)
    for r in range(n):
        a, b = TIE_PAIRS[r % len(TIE_PAIRS)]
        i = (7 * r + 3) % B
        j = (i + 1 + 13 * r) % B
        for k0 in range(0, K - B + 1, B):
            rows[r, k0 + i] = a
            rows[r, k0 + j] = b
    return inputs.to_f16(rows)


def oracle_ties(y_ref, s_ref):
    """Number of values whose oracle quotient y / s (fp32, as the oracle forms it) is
    exactly k + 1/2."""
    s = np.asarray(s_ref, dtype=np.float32)[:, None]
    ok = s != 0
    t = np.where(ok, np.asarray(y_ref, dtype=np.float32) / np.where(ok, s, np.float32(1)), np.float32(0))
    t = np.abs(t.astype(np.float32))
    return int(np.sum(t - np.floor(t) == 0.5))


TIE_CASES = [(256, 256), (4096, 256), (4096, 4096), (2048, 512), (4096, 2048), (11008, 256), (1024, 128)]


@pytest.mark.parametrize("bits", [4, 8])
@pytest.mark.parametrize("K,B", TIE_CASES)
def test_exact_ties_round_half_even(dp, orc, K, B, bits):
    """Rows built so that half of their rotated values land exactly on a half-integer of
    the code grid (Section 2 Eq. 2: the rounding of y / s; Section 4.2 per-token
    symmetric scale).  The oracle rounds them half to even; the GPU's exact rotation and
    IEEE-quotient fallback must give the same codes.  For even log2 B the GPU's rotated
    values are bit-identical to the oracle's, so no mismatch at all is allowed; for odd
    log2 B the parity contract (tie mismatches off by one, at most 1e-5 of the codes)."""
    x = tie_rows(K, B)
    c_ref, s_ref = orc.rotate_quant_act(x, B, bits)
    y_ref = orc.rotate(x, B)
    ties = oracle_ties(y_ref, s_ref)
    assert ties >= x.shape[0] * K // 4, f"only {ties} exact ties in the oracle's quotients"
    # the oracle's tie codes are the even neighbours
    t = y_ref.astype(np.float32) / s_ref.astype(np.float32)[:, None]
    at = np.abs(t) - np.floor(np.abs(t)) == 0.5
    assert np.all(c_ref[at] % 2 == 0)
    c, s = gpu_codes(dp, x, B, bits, orc)
    parity.check_scales(s, s_ref)
    n = parity.check_codes(c, c_ref, y_ref, s_ref, bits)
    log2b = B.bit_length() - 1
    if log2b % 2 == 0:
        assert n == 0 and np.array_equal(s, s_ref), f"{n} tie mismatches on an even-log2 block"


ROT_CASES = [(256, 256, 16), (4096, 4096, 8), (11008, 256, 6), (13824, 1024, 5), (14336, 2048, 4),
             (28672, 4096, 2), (160, 32, 3), (768, 512, 3), (96, 64, 2), (5120, 1024, 4)]


@pytest.mark.parametrize("K,B,M", ROT_CASES)
def test_rotation_within_tolerance(dp, orc, K, B, M):
    wl = inputs.llama2_7b_decode()
    x = np.concatenate([inputs.activations(wl, M, K), edge_rows(K)])
    y_ref = orc.rotate(x, B)
    y = gpu_rotate(dp, x, B)
    parity.check_rotation(y, y_ref)


@pytest.mark.parametrize("bits", [4, 8])
@pytest.mark.parametrize("K,B,M", ROT_CASES)
def test_rotate_quant_codes_and_scales(dp, orc, K, B, M, bits):
    wl = inputs.llama2_13b_prefill()
    x = np.concatenate([inputs.activations(wl, M, K), edge_rows(K)])
    c_ref, s_ref = orc.rotate_quant_act(x, B, bits)
    y_ref = orc.rotate(x, B)
    c, s = gpu_codes(dp, x, B, bits, orc)
    parity.check_scales(s, s_ref)
    parity.check_codes(c, c_ref, y_ref, s_ref, bits)
    assert np.all(c[M] == 0) and s[M] == 0.0      # the all-zero edge row


@pytest.mark.parametrize("N,K,B", [(512, 256, 256), (64, 4096, 4096), (128, 11008, 256), (48, 13824, 1024),
                                   (16, 160, 32), (272, 768, 512)])
def test_pack_weights_matches_oracle(dp, orc, N, K, B):
    W = inputs.weights(N, K, layer=2, proj=5)
    q_ref, sw_ref = orc.pack_weights(W, B)
    layer = dp.dptq_pack_weights(torch.from_numpy(W).to(DEV), B)
    wq, sw = dp.dptq_get_packed(layer)
    q = orc.unpack_nibbles(wq, K)
    parity.check_scales(sw, sw_ref)
    y_ref = orc.rotate(W, B)
    parity.check_codes(q, q_ref, y_ref, sw_ref, 4)
    # the same packing from host memory
    layer_h = dp.dptq_pack_weights(torch.from_numpy(W), B)
    wq_h, sw_h = dp.dptq_get_packed(layer_h)
    assert np.array_equal(wq_h, wq) and np.array_equal(sw_h, sw)


def run_codes_gemm(dp, orc, layer, codes, sa, bits):
    M, K = codes.shape
    cd = torch.from_numpy(orc.pack_nibbles(codes) if bits == 4 else codes).to(DEV)
    sd = torch.from_numpy(sa).to(DEV)
    out = torch.empty((M, layer.N), dtype=torch.float16, device=DEV)
    acc = torch.empty((M, layer.N), dtype=torch.int32, device=DEV)
    dp.dptq_qgemm_codes(layer, cd, sd, bits, out, acc)
    return out.cpu().numpy(), acc.cpu().numpy()


# The GEMM does not depend on the Hadamard block; small blocks keep the oracle's dense
# rotation of the weights cheap.
GEMM_CASES = [(16, 512, 256, 32), (1, 4096, 4096, 64), (8, 1024, 4096, 64), (33, 1024, 4096, 64),
              (130, 256, 1024, 32), (300, 384, 512, 32), (64, 128, 11008, 256), (17, 48, 160, 32),
              (2048, 5120, 256, 32),
              # 192-token tiles with an odd number of k-blocks: one k-block per stage
              (200, 256, 384, 128)]


@pytest.mark.parametrize("bits", [4, 8])
@pytest.mark.parametrize("M,N,K,B", GEMM_CASES)
def test_gemm_accumulators_exact(dp, orc, M, N, K, B, bits):
    W = inputs.weights(N, K, layer=1, proj=3)
    q_ref, sw_ref = orc.pack_weights(W, B)
    layer = dp.dptq_pack_weights(torch.from_numpy(W).to(DEV), B)
    q = orc.unpack_nibbles(dp.dptq_get_packed(layer)[0], K)
    same_w = np.all(q == q_ref, axis=1)          # weight rows without a rounding tie
    codes = inputs.random_codes(M, K, bits, seed=M + N)
    sa = (np.random.default_rng(M).random(M) * 0.1 + 0.01).astype(np.float32)
    out, acc = run_codes_gemm(dp, orc, layer, codes, sa, bits)
    acc_ref = orc.gemm_i32(codes, q_ref)
    assert np.array_equal(acc[:, same_w], acc_ref[:, same_w])
    out_ref = orc.epilogue(acc_ref, sa, sw_ref)
    parity.check_out(out[:, same_w], out_ref[:, same_w])
    # a second call must give the same result (split-tile scratch left clean)
    out2, acc2 = run_codes_gemm(dp, orc, layer, codes, sa, bits)
    assert np.array_equal(acc2, acc) and np.array_equal(out2.view(np.uint16), out.view(np.uint16))


@pytest.mark.parametrize("K,B", [(28672, 256), (14336, 512)])
def test_exact_accumulation_beyond_2_24(dp, orc, K, B):
    """A row with one equal nonzero per Hadamard block rotates to +-|v|/sqrt(B) everywhere:
    8-bit codes +-127 and weight codes +-7 with the signs of Hadamard row j.  Rows that
    share j multiply to 127*7*K (> 2^24 at K = 28672), others cancel exactly to 0."""
    M, N = 16, 128
    x = np.zeros((M, K), dtype=np.float16)
    W = np.zeros((N, K), dtype=np.float16)
    jm = [(m * 37) % B for m in range(M)]
    for m in range(M):
        x[m, jm[m]::B] = 1.0 + m
    for n in range(N):
        j = jm[n % 16] if n < 32 else (n * 53) % B
        W[n, j::B] = -0.5 if n % 3 else 0.25
    q_ref, sw_ref = orc.pack_weights(W, B)
    c_ref, s_ref = orc.rotate_quant_act(x, B, 8)
    assert np.all(np.abs(c_ref) == 127) and np.all(np.abs(q_ref) == 7)
    layer = dp.dptq_pack_weights(torch.from_numpy(W).to(DEV), B)
    q = orc.unpack_nibbles(dp.dptq_get_packed(layer)[0], K)
    assert np.array_equal(q, q_ref)
    out, acc = run_codes_gemm(dp, orc, layer, c_ref, s_ref, 8)
    acc_ref = orc.gemm_i32(c_ref, q_ref)
    assert np.abs(acc_ref).max() == 127 * 7 * K
    if K > 20000:
        assert np.abs(acc_ref).max() > 2 ** 24
    assert np.array_equal(acc, acc_ref)
    parity.check_out(out, orc.epilogue(acc_ref, s_ref, sw_ref))


def check_qlinear(dp, orc, x, W, B, bits, rows=None, cols=None):
    """Full-size GPU run; oracle on the sampled rows/cols (all when None)."""
    M, K = x.shape
    N = W.shape[0]
    layer = dp.dptq_pack_weights(torch.from_numpy(W).to(DEV), B)
    xd = torch.from_numpy(x).to(DEV)
    out = torch.empty((M, N), dtype=torch.float16, device=DEV)
    dp.dptq_qlinear(layer, xd, bits, out)
    codes = torch.empty((M, K // 2) if bits == 4 else (M, K), dtype=torch.uint8 if bits == 4 else torch.int8,
                        device=DEV)
    sgpu = torch.empty((M,), dtype=torch.float32, device=DEV)
    dp.dptq_rotate_quant_act(xd, B, bits, codes, sgpu)
    torch.cuda.synchronize()
    rows = np.arange(M) if rows is None else np.asarray(rows)
    cols = np.arange(N) if cols is None else np.asarray(cols)
    got = out.cpu().numpy()[np.ix_(rows, cols)]
    cg = codes.cpu().numpy()[rows]
    cg = orc.unpack_nibbles(cg, K) if bits == 4 else cg
    # oracle on the sample
    xs = np.ascontiguousarray(x[rows])
    Ws = np.ascontiguousarray(W[cols])
    q_ref, sw_ref = orc.pack_weights(Ws, B)
    r = orc.qlinear(xs, B, bits, q_ref, sw_ref)
    y_ref = orc.rotate(xs, B)
    parity.check_scales(sgpu.cpu().numpy()[rows], r["sa"])
    parity.check_codes(cg, r["codes"], y_ref, r["sa"], bits, total=M * K)
    wq, _ = dp.dptq_get_packed(layer)
    qg = orc.unpack_nibbles(wq[cols], K)
    ok_r = np.all(cg == r["codes"], axis=1)
    ok_c = np.all(qg == q_ref, axis=1)
    parity.check_out(got[np.ix_(ok_r, ok_c)], r["out"][np.ix_(ok_r, ok_c)])
    layer.close()
    return got, r


@pytest.mark.parametrize("bits", [4, 8])
def test_qlinear_single_layer_config(dp, orc, bits):
    wl = inputs.single_linear()
    x = inputs.activations(wl, 16, 256)
    W = inputs.weights(512, 256)
    got, r = check_qlinear(dp, orc, x, W, 256, bits)
    assert np.array_equal(got.view(np.uint16), r["out"].view(np.uint16))


@pytest.mark.parametrize("M", [1, 2, 17, 31, 63, 65, 129, 257])
def test_qlinear_ragged_token_counts(dp, orc, M):
    wl = inputs.llama2_7b_decode()
    K, N, B = 1024, 272, 1024
    x = inputs.activations(wl, M, K)
    if M >= 17:   # exact rounding ties inside a ragged token tile
        x = np.concatenate([x[:M - 4], tie_rows(K, B, 4)])
    W = inputs.weights(N, K, layer=4, proj=1)
    for bits in (4, 8):
        check_qlinear(dp, orc, x, W, B, bits)


def test_qlinear_edge_inputs(dp, orc):
    K, N, B = 512, 128, 256
    x = edge_rows(K)
    W = inputs.weights(N, K, layer=9, proj=0)
    W[3] = 0                                    # an all-zero weight row
    for bits in (4, 8):
        got, r = check_qlinear(dp, orc, x, W, B, bits)
        assert np.all(got[0] == 0) and np.all(got[:, 3] == 0)


@pytest.mark.parametrize("M,N,K,B", [(17, 272, 1024, 1024), (32, 4096, 4096, 4096)])
def test_qlinear_unaligned_output(dp, M, N, K, B):
    """An output pointer that is not 16-byte aligned takes the scalar-store epilogue;
    it must give the same bits as an aligned one (split tiles included)."""
    wl = inputs.llama2_7b_decode()
    x = torch.from_numpy(inputs.activations(wl, M, K)).to(DEV)
    W = inputs.weights(N, K, layer=2, proj=3)
    layer = dp.dptq_pack_weights(torch.from_numpy(W).to(DEV), B)
    for bits in (4, 8):
        ref = torch.empty((M, N), dtype=torch.float16, device=DEV)
        dp.dptq_qlinear(layer, x, bits, ref)
        flat = torch.zeros(M * N + 8, dtype=torch.float16, device=DEV)
        out = flat[1:1 + M * N].view(M, N)
        assert out.data_ptr() % 16 != 0
        dp.dptq_qlinear(layer, x, bits, out)
        torch.cuda.synchronize()
        assert torch.equal(out.view(torch.int16), ref.view(torch.int16))
        assert flat[0].item() == 0 and torch.all(flat[1 + M * N:] == 0)
    layer.close()


@pytest.mark.parametrize("M,N,K,B", [(64, 128, 256, 256), (16, 512, 256, 256), (5, 4096, 4096, 4096),
                                     (32, 4096, 11008, 256), (33, 1024, 2048, 512), (1, 22016, 4096, 4096)])
def test_fused_qlinear_equals_two_launches(dp, M, N, K, B):
    """dptq_qlinear (one launch for small M: the GEMM kernel rotates and quantizes the rows
    itself) gives the same bits as the rotate-quantize launch followed by the GEMM launch.
    (64, 128, 256): one CTA quantizes all 64 rows; (16, 512, 256): 4 CTAs, 4 rows each."""
    wl = inputs.llama2_7b_decode()
    x = torch.from_numpy(inputs.activations(wl, M, K)).to(DEV)
    W = inputs.weights(N, K, layer=7, proj=1)
    layer = dp.dptq_pack_weights(torch.from_numpy(W).to(DEV), B)
    for bits in (4, 8):
        fused = torch.empty((M, N), dtype=torch.float16, device=DEV)
        two = torch.empty((M, N), dtype=torch.float16, device=DEV)
        for _ in range(3):   # repeated launches reuse the grid counters
            dp.dptq_qlinear(layer, x, bits, fused)
        dp.dptq_qlinear_quantize(layer, x, bits)
        dp.dptq_qlinear_gemm(layer, M, bits, two)
        torch.cuda.synchronize()
        assert torch.equal(fused.view(torch.int16), two.view(torch.int16)), (M, N, K, bits)
    layer.close()


# How the fused launch splits each row over its parts (np per row, from the planner):
# slices of one block (1024 or 2048 elements per part) when a row has fewer blocks than
# parts, else whole 128-aligned groups of blocks per part.
FUSED_SPLIT_CASES = [
    (5, 4096, 4096, 4096, False, 4),     # slices of 1024, four per block
    (8, 4096, 4096, 2048, True, 4),      # slices of 1024, two per block; randomized signs
    (64, 4096, 4096, 4096, False, 2),    # slices of 2048, two per block
    (32, 12288, 4096, 4096, True, 4),    # q|k|v at M = 32: all SMs (split tiles), slices of 1024; signs
    (64, 12288, 4096, 4096, True, 2),    # q|k|v at M = 64: slices of 2048; signs
    (64, 4096, 8192, 256, True, 2),      # whole blocks, two parts of 4096; signs
    (64, 4096, 11008, 256, False, 4),    # whole blocks, four parts, two rounds of rows
    (32, 4096, 14336, 2048, False, 4),   # whole blocks of 2048: 1 / 2 / 2 / 2 per part
    (32, 4096, 6144, 4096, True, 4),     # one block, the 2048 tail block, two empty parts
    (4, 4096, 224, 64, False, 2),        # a part holding a block of 64 and the 32-element tail
    (16, 4096, 256, 256, False, 2),      # one part rotates the row, the other is empty
]


@pytest.mark.parametrize("M,N,K,B,rh,np_", FUSED_SPLIT_CASES)
def test_fused_row_split_equals_two_launches(dp, M, N, K, B, rh, np_):
    """Every row split of the fused launch (each part rotating only its own outputs, the
    parts exchanging their maxima) gives the bits of the rotate-quantize launch and the
    GEMM launch, which are compared with the oracle elsewhere."""
    sms = torch.cuda.get_device_properties(0).multi_processor_count
    info = dp.dptq_plan_info(M, N, K, 4, sms, fused=True)
    assert info["fused"] == 1 and info["rq_np"] == np_
    wl = inputs.llama2_7b_decode()
    x = torch.from_numpy(inputs.activations(wl, M, K)).to(DEV)
    W = torch.from_numpy(inputs.weights(N, K, layer=5, proj=4)).to(DEV)
    if rh:
        d = np.where(np.random.default_rng(K + M).random(K) < 0.5, -1, 1).astype(np.int8)
        layer = dp.dptq_pack_weights_rh(W, B, d)
    else:
        layer = dp.dptq_pack_weights(W, B)
    for bits in (4, 8):
        fused = torch.empty((M, N), dtype=torch.float16, device=DEV)
        two = torch.empty((M, N), dtype=torch.float16, device=DEV)
        for _ in range(3):   # repeated launches reuse the grid counters and the row-maximum slots
            dp.dptq_qlinear(layer, x, bits, fused)
        dp.dptq_qlinear_quantize(layer, x, bits)
        dp.dptq_qlinear_gemm(layer, M, bits, two)
        torch.cuda.synchronize()
        assert torch.equal(fused.view(torch.int16), two.view(torch.int16)), (M, N, K, B, bits)
    layer.close()
    dp.dptq_last_device_error()


def test_qlinear_m_zero_is_noop(dp):
    W = inputs.weights(128, 256)
    layer = dp.dptq_pack_weights(torch.from_numpy(W).to(DEV), 256)
    x = torch.empty((0, 256), dtype=torch.float16, device=DEV)
    out = torch.empty((0, 128), dtype=torch.float16, device=DEV)
    dp.dptq_qlinear(layer, x, 4, out)
    torch.cuda.synchronize()


def test_bad_arguments_raise(dp):
    W = inputs.weights(128, 256)
    layer = dp.dptq_pack_weights(torch.from_numpy(W).to(DEV), 256)
    x = torch.zeros((4, 256), dtype=torch.float16, device=DEV)
    out = torch.empty((4, 128), dtype=torch.float16, device=DEV)
    with pytest.raises(dp.DptqError):
        dp.dptq_qlinear(layer, x, 6, out)
    with pytest.raises(dp.DptqError):
        dp.dptq_pack_weights(torch.zeros((128, 100), dtype=torch.float16, device=DEV), 64)


def test_graph_capture_and_repeat(dp, orc):
    wl = inputs.llama2_7b_decode()
    K, N, B, M = 4096, 1024, 4096, 32
    x = torch.from_numpy(inputs.activations(wl, M, K)).to(DEV)
    W = inputs.weights(N, K, layer=0, proj=0)
    layer = dp.dptq_pack_weights(torch.from_numpy(W).to(DEV), B)
    dp.dptq_reserve(M, K, N)
    eager = {}
    for bits in (4, 8):
        out = torch.empty((M, N), dtype=torch.float16, device=DEV)
        dp.dptq_qlinear(layer, x, bits, out)
        eager[bits] = out.clone()
    s = torch.cuda.Stream()
    outs = {b: torch.empty((M, N), dtype=torch.float16, device=DEV) for b in (4, 8)}
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=s):
        for bits in (4, 8):
            dp.dptq_qlinear(layer, x, bits, outs[bits])
    for _ in range(3):
        g.replay()
        torch.cuda.synchronize()
        for bits in (4, 8):
            assert torch.equal(outs[bits], eager[bits])


def test_no_device_error_left(dp):
    dp.dptq_last_device_error()


# ----------------------------------------------------------------------------- full-size workloads
def tile_sample(N, seed):
    """One output channel from every 128-channel weight tile (a random one per tile), and
    the first and last channel: every tile's epilogue, and every split-tile reduction of
    the stream-K work split, is compared with the oracle."""
    rng = np.random.default_rng(seed)
    cols = {min(N - 1, t * 128 + int(rng.integers(128))) for t in range((N + 127) // 128)}
    cols.update({0, N - 1})
    return np.array(sorted(cols))


def sample(n, k, seed, must=()):
    rng = np.random.default_rng(seed)
    pick = set(int(v) for v in rng.choice(n, min(k, n), replace=False))
    pick.update(int(v) for v in must if v < n)
    pick.update({0, n - 1})
    return np.array(sorted(pick))


@pytest.mark.parametrize("M", [1, 8, 32])
@pytest.mark.parametrize("proj", ["q", "gate", "down"])
def test_llama2_7b_decode_shapes(dp, orc, M, proj):
    wl = inputs.llama2_7b_decode()
    p = {pp.name: pp for pp in wl.projs}[proj]
    x = inputs.activations(wl, M, p.K)
    W = inputs.weights(p.N, p.K, layer=0, proj=[pp.name for pp in wl.projs].index(proj))
    if M >= 8:   # two rows of exact rounding ties
        x = np.concatenate([x[:M - 2], tie_rows(p.K, p.had_block, 2)])
    cols = tile_sample(p.N, 5)
    for bits in (4, 8):
        check_qlinear(dp, orc, x, W, p.had_block, bits, cols=cols)


@pytest.mark.parametrize("wl_name,proj,M,bits", [
    ("llama3-8b-prefill", "q", 2048, 4), ("llama3-8b-prefill", "down", 2048, 8),
    ("llama2-13b-prefill", "o", 4096, 8), ("llama2-13b-prefill", "down", 4096, 4),
    ("llama2-70b", "q", 512, 4), ("llama2-70b", "down", 64, 8), ("llama2-70b", "down", 8192, 8),
])
def test_prefill_and_70b_shapes_sampled(dp, orc, wl_name, proj, M, bits):
    wl = inputs.WORKLOADS[wl_name]()
    p = {pp.name: pp for pp in wl.projs}[proj]
    x = inputs.activations(wl, M, p.K)
    W = inputs.weights(p.N, p.K, layer=1, proj=[pp.name for pp in wl.projs].index(proj))
    hot = [t for t in range(M) if np.abs(x[t].astype(np.float32)).max() > 50]
    rows = sample(M, 24, 7, must=hot[:8])
    cols = tile_sample(p.N, 8)
    check_qlinear(dp, orc, x, W, p.had_block, bits, rows=rows, cols=cols)


@pytest.mark.parametrize("wl_name,proj,M,bits", [
    ("llama2-70b", "q", 1, 4), ("llama2-70b", "q", 1, 8), ("llama2-70b", "down", 1, 4),
    ("llama2-70b", "gate", 64, 4), ("llama3-8b-prefill", "k", 2048, 4), ("llama3-8b-prefill", "v", 2048, 8),
])
def test_more_workload_shapes(dp, orc, wl_name, proj, M, bits):
    """LLaMA-2-70B at one token (the fused decode launch for K = 8192, the two-launch path
    for the 28672-long down row) and at 64 tokens, and LLaMA-3-8B's GQA k / v projections
    (N = 1024) in prefill; one channel per weight tile."""
    wl = inputs.WORKLOADS[wl_name]()
    p = {pp.name: pp for pp in wl.projs}[proj]
    x = inputs.activations(wl, M, p.K)
    W = inputs.weights(p.N, p.K, layer=5, proj=[pp.name for pp in wl.projs].index(proj))
    hot = [t for t in range(M) if np.abs(x[t].astype(np.float32)).max() > 50]
    rows = None if M <= 64 else sample(M, 24, 9, must=hot[:8])
    check_qlinear(dp, orc, x, W, p.had_block, bits, rows=rows, cols=tile_sample(p.N, 10))


@pytest.mark.parametrize("wl_name,group,M", [("llama2-7b-decode", "qkv", 32), ("llama2-7b-decode", "gateup", 32),
                                             ("llama3-8b-prefill", "gateup", 2048)])
@pytest.mark.parametrize("bits", [4, 8])
def test_concatenated_group_handles(dp, orc, wl_name, group, M, bits):
    """The benchmark's concatenated handles: q|k|v (N = 12288) and gate|up (N = 22016) of
    LLaMA-2-7B at 32 tokens, and LLaMA-3-8B's gate|up (N = 28672) in prefill, packed as one
    weight matrix (the rows of the group's projections stacked), against the oracle on one
    channel of every 128-channel tile.  One quantization of x feeds the whole group."""
    wl = inputs.WORKLOADS[wl_name]()
    names = [pp.name for pp in wl.projs]
    projs = [pp for pp in wl.projs if pp.group == group]
    K, B = projs[0].K, projs[0].had_block
    W = np.concatenate([inputs.weights(pp.N, pp.K, layer=3, proj=names.index(pp.name)) for pp in projs])
    x = inputs.activations(wl, M, K)
    if M <= 64:
        x = np.concatenate([x[:M - 2], tie_rows(K, B, 2)])
    hot = [t for t in range(M) if np.abs(x[t].astype(np.float32)).max() > 50]
    rows = None if M <= 64 else sample(M, 16, 11, must=hot[:4])
    check_qlinear(dp, orc, x, W, B, bits, rows=rows, cols=tile_sample(W.shape[0], 12))


# ----------------------------------------------------------------------------- non-power-of-two tails
# K = 11008 with blocks of 4096 leaves a tail of 2816 = 44 x 64 (LLaMA-2-7B's down input),
# K = 13824 leaves 1536 = 12 x 128 (LLaMA-2-13B's), 448 = 256 + 12 x 16: the tail block's
# Hadamard matrix is Paley's H_p (x) the Sylvester H_(2^k) (Section 2 Eq. 4, R^T R = I).
PALEY_CASES = [(11008, 4096, 4), (13824, 4096, 3), (256 + 192, 256, 6)]


@pytest.mark.parametrize("K,B,M", PALEY_CASES)
def test_paley_tail_rotation_and_codes(dp, orc, K, B, M):
    assert orc.tail_factor(K % B)[0] > 1
    wl = inputs.llama2_7b_decode()
    x = np.concatenate([inputs.activations(wl, M, K), edge_rows(K)])
    y_ref = orc.rotate(x, B)
    parity.check_rotation(gpu_rotate(dp, x, B), y_ref)
    for bits in (4, 8):
        c_ref, s_ref = orc.rotate_quant_act(x, B, bits)
        c, s = gpu_codes(dp, x, B, bits, orc)
        parity.check_scales(s, s_ref)
        parity.check_codes(c, c_ref, y_ref, s_ref, bits)


@pytest.mark.parametrize("K,B", [(11008, 4096), (448, 256)])
def test_paley_tail_pack_and_qlinear(dp, orc, K, B):
    """Weight packing folds the same R (Eq. 5), and the qlinear layer (two launches: the
    fused decode launch takes power-of-two tails only) matches the oracle, at 8 tokens
    and at 130; the oracle's dense fp64 rotation costs about 0.3 s per row at K = 11008,
    so it checks sampled rows and one channel per weight tile."""
    N = 384
    W = inputs.weights(N, K, layer=6, proj=6)
    cols = tile_sample(N, 13)
    q_ref, sw_ref = orc.pack_weights(np.ascontiguousarray(W[cols]), B)
    layer = dp.dptq_pack_weights(torch.from_numpy(W).to(DEV), B)
    wq, sw = dp.dptq_get_packed(layer)
    parity.check_scales(sw[cols], sw_ref)
    parity.check_codes(orc.unpack_nibbles(wq[cols], K), q_ref, orc.rotate(np.ascontiguousarray(W[cols]), B),
                       sw_ref, 4)
    layer.close()
    wl = inputs.llama2_7b_decode()
    for M in (8, 130):
        x = inputs.activations(wl, M, K)
        rows = sample(M, 6, M, must=(127, 128))
        for bits in (4, 8):
            check_qlinear(dp, orc, x, W, B, bits, rows=rows, cols=cols)
