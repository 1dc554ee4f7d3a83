"""Host-side invariants of the GEMM launch planner (dptq_plan_info: no GPU needed).

The plans must fit the hardware (shared memory, tensor-memory columns), keep the fp32
accumulation of integer products exact (Section 4.2 integer GEMM: every partial sum an
integer multiple of 2^-9 below 2^24 units), cover every tile exactly once, and choose
the tile shapes the kernels are built for."""
import itertools

import pytest

from paper_2606_12487_gb300 import dptq

SMEM_LIMIT = 232448          # 227 KB opt-in dynamic shared memory per CTA
TMEM_COLS = 512

# (N, K) of every projection in the workloads: LLaMA-2-7B, LLaMA-3-8B, LLaMA-2-13B,
# LLaMA-2-70B, plus small and ragged shapes.
SHAPES = [(12288, 4096), (4096, 4096), (22016, 4096), (4096, 11008), (1024, 4096), (28672, 4096),
          (4096, 14336), (5120, 5120), (27648, 5120), (5120, 13824), (8192, 8192), (1024, 8192),
          (57344, 8192), (8192, 28672), (512, 256), (272, 1024), (128, 128), (4096, 128)]
TOKENS = [1, 2, 8, 16, 17, 31, 32, 33, 63, 64, 65, 128, 129, 191, 192, 193, 257, 512, 2048, 4096, 8192]


def _plans():
    for (N, K), M, bits, sms in itertools.product(SHAPES, TOKENS, (4, 8), (148, 152)):
        yield N, K, M, bits, sms


def _check_plan(p, M, N, K, bits, sms):
    nt, kps = p["nt"], p["kps"]
    assert nt in (16, 32, 64, 128, 192, 256) and kps in (1, 2)
    assert p["smem_bytes"] <= SMEM_LIMIT
    assert p["stages"] >= 2 and p["grid"] <= sms
    # token padding and tiling
    assert p["M_pad"] % nt == 0 and M <= p["M_pad"] < M + nt
    assert p["m_tiles"] == p["M_pad"] // nt and p["n_wtiles"] == -(-N // 128)
    kb = -(-K // 128)
    assert kb % kps == 0 and p["KI"] == kb // kps
    # tensor memory: accumulators (and the weight slots when they live there) fit
    acc = p["nbuf"] * nt * p["segs"]
    assert p["acc_cols"] == acc
    a_cols = p["conv_slots"] * kps * 32 if p["a_tmem"] else 0
    assert acc + a_cols <= p["tmem_cols"] <= TMEM_COLS
    assert p["tmem_cols"] in (32, 64, 128, 256, 512)
    # exact fp32 accumulation: largest |code x weight| sum of one segment below 2^24
    qa = 128 if bits == 8 else 8
    assert p["seg_iters"] * kps * 128 * qa * 7 < 2 ** 24
    assert p["segs"] * p["seg_iters"] >= p["KI"]
    # work split: whole tiles round-robin, then stream-K over the rest, every tile once
    tiles = p["n_wtiles"] * p["m_tiles"]
    assert p["dp_tiles"] % p["grid"] == 0
    assert p["sk_iters"] % p["KI"] == 0 and p["dp_tiles"] + p["sk_iters"] // p["KI"] == tiles


@pytest.mark.parametrize("N,K,M,bits,sms", list(_plans()))
def test_split_plans_fit_and_cover(N, K, M, bits, sms):
    p = dptq.dptq_plan_info(M, N, K, bits, sms)
    _check_plan(p, M, N, K, bits, sms)
    assert p["fused"] == 0
    # tile shapes the kernels are built for
    even_kb = (-(-K // 128)) % 2 == 0
    if M <= 64:
        # two-block stages with the weights in tensor memory, unless K has an odd number
        # of k-blocks
        assert nt_expected_decode(M) == p["nt"]
        assert p["kps"] == (2 if even_kb else 1) and p["a_tmem"] == (1 if even_kb else 0)
    elif bits == 4 and M > 128:
        assert p["nt"] == 192 and p["a_tmem"] == 1
        assert p["kps"] == (2 if even_kb else 1)
    elif bits == 8 and M > 128:
        # two 24 KB activation planes per k-block: one k-block per stage, at least 4 stages
        assert p["nt"] == 192 and p["a_tmem"] == 1 and p["kps"] == 1 and p["stages"] >= 4
    else:
        assert p["nt"] == 128 and p["kps"] == 1 and p["a_tmem"] == 0


def nt_expected_decode(M):
    return 16 if M <= 16 else 32 if M <= 32 else 64


@pytest.mark.parametrize("N,K", SHAPES)
@pytest.mark.parametrize("M", [1, 8, 16, 32, 33, 64])
@pytest.mark.parametrize("bits", [4, 8])
def test_fused_decode_plans(N, K, M, bits):
    if (-(-K // 128)) % 2:
        # the fused kernel needs two-block stages; dptq_qlinear then takes two launches
        with pytest.raises(dptq.DptqError):
            dptq.dptq_plan_info(M, N, K, bits, 152, fused=True)
        return
    split = dptq.dptq_plan_info(M, N, K, bits, 152)
    M_pad = split["M_pad"]
    tiles = split["n_wtiles"] * split["m_tiles"]
    # the largest grid a decode plan takes: every SM, at most four CTAs per weight tile
    g_max = min(152, 4 * tiles, tiles * split["KI"])
    if M_pad * 4 > 2 * g_max and (M_pad * 2 > g_max or K > 8192):
        # too few CTAs for the rows' parts: dptq_qlinear takes the two-launch path
        with pytest.raises(dptq.DptqError):
            dptq.dptq_plan_info(M, N, K, bits, 152, fused=True)
        return
    p = dptq.dptq_plan_info(M, N, K, bits, 152, fused=True)
    # whole tiles (one CTA each) only when they leave a CTA for each of four parts per row
    if p["grid"] == tiles and tiles < g_max:
        assert M_pad * 4 <= tiles
    _check_plan(p, M, N, K, bits, 152)
    assert p["fused"] == 1 and p["kps"] == 2 and p["nt"] <= 64 and p["stages"] >= 3
    assert p["smem_bytes"] <= SMEM_LIMIT
    # each token row is split into 4 parts, each with a CTA of its own; else into 2 parts
    # (rows of at most two 4096-element chunks); else 4 parts with at most two per CTA
    np_ = p["rq_np"]
    assert np_ in (2, 4)
    if np_ == 2:
        assert M_pad * 4 > p["grid"] and M_pad * 2 <= p["grid"] and K <= 8192
    else:
        assert M_pad * 4 <= 2 * p["grid"]
        assert M_pad * 4 <= p["grid"] or M_pad * 2 > p["grid"] or K > 8192


def test_fused_plan_refused_beyond_64_tokens():
    with pytest.raises(dptq.DptqError):
        dptq.dptq_plan_info(65, 4096, 4096, 4, 152, fused=True)


@pytest.mark.parametrize("args", [(0, 128, 128, 4, 152), (1, 0, 128, 4, 152), (1, 128, 0, 4, 152),
                                  (1, 128, 128, 6, 152), (1, 128, 128, 4, 0)])
def test_plan_info_rejects_bad_arguments(args):
    with pytest.raises(dptq.DptqError):
        dptq.dptq_plan_info(*args)
