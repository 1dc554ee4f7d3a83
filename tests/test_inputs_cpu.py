"""The seeded input generators follow the workload recipe (synthetic stand-ins for the
paper's calibration activations and LLaMA weights): outlier channels and their scales,
outlier token positions, heavy tails, per-layer masks, weight distribution, saturation,
and sampled rows equal to the full draw."""
import numpy as np
import pytest

from paper_2606_12487_gb300 import inputs


def _col_rms(x):
    return np.sqrt(np.mean(x.astype(np.float64) ** 2, axis=0))


def test_llama2_7b_outlier_channels_scaled_by_100():
    wl = inputs.llama2_7b_decode()
    x = inputs.activations(wl, 256, 4096)
    ch = inputs.outlier_channels(4096, 4)
    assert len(set(ch.tolist())) == 4
    rms = _col_rms(x)
    assert np.all(np.abs(rms[ch] / 100.0 - 1.0) < 0.15)
    others = np.delete(rms, ch)
    assert np.all(others < 1.5) and abs(np.mean(others) - 1.0) < 0.02
    # the same channels for every K-sized row set and every call
    assert np.array_equal(inputs.outlier_channels(4096, 4), ch)


def test_llama3_8b_outliers_on_one_percent_of_tokens():
    wl = inputs.llama3_8b_prefill()
    x = inputs.activations(wl, 2048, 1024).astype(np.float64)
    ch = inputs.outlier_channels(1024, 3)
    hot = np.where(np.max(np.abs(x[:, ch]), axis=1) > 30.0)[0]
    assert len(hot) == 20                                     # 1 % of 2048, rounded
    cold = np.setdiff1d(np.arange(2048), hot)
    assert np.max(np.abs(x[np.ix_(cold, ch)])) < 7.0           # no scaling off the hot tokens
    assert abs(np.sqrt(np.mean(x[np.ix_(hot, ch)] ** 2)) / 300.0 - 1.0) < 0.3


def test_llama2_13b_student_t_tails():
    wl = inputs.llama2_13b_prefill()
    x = inputs.activations(wl, 512, 5120).astype(np.float64).ravel()
    # Student-t with 3 degrees of freedom: P(|t| > 5) = 0.0154; a Gaussian gives 6e-7
    frac = np.mean(np.abs(x) > 5.0)
    assert 0.012 < frac < 0.019
    assert abs(np.median(np.abs(x)) - 0.765) < 0.02           # median |t_3| = 0.7649


def test_llama2_70b_outliers_on_the_first_token_of_each_sequence():
    wl = inputs.llama2_70b()
    x = inputs.activations(wl, 4100, 256).astype(np.float64)
    ch = inputs.outlier_channels(256, 2)
    big = np.where(np.max(np.abs(x[:, ch]), axis=1) > 50.0)[0]
    assert big.tolist() == [0, 2048, 4096]


def test_sampled_rows_equal_the_full_draw():
    for wl in (inputs.llama3_8b_prefill(), inputs.llama2_13b_prefill(), inputs.llama2_70b()):
        full = inputs.activations(wl, 2100, 256)
        part = inputs.activations(wl, 60, 256, row_offset=2040)
        assert np.array_equal(full[2040:2100].view(np.uint16), part.view(np.uint16))


def test_masks_follow_the_workloads():
    assert inputs.llama2_7b_decode().mask_a8 == (0, 1, 30, 31)
    assert inputs.llama2_13b_prefill().mask_a8 == (0, 1, 2, 38, 39)
    m8 = inputs.llama3_8b_prefill().mask_a8
    m70 = inputs.llama2_70b().mask_a8
    assert len(m8) == 6 and len(set(m8)) == 6 and all(0 <= v < 32 for v in m8)
    assert len(m70) == 8 and len(set(m70)) == 8 and all(0 <= v < 80 for v in m70)
    assert inputs.llama3_8b_prefill().mask_a8 == m8           # seeded, reproducible
    wl = inputs.llama2_7b_decode()
    assert [wl.bits(l) for l in (0, 1, 2, 29, 30, 31)] == [8, 8, 4, 4, 8, 8]


def test_projection_shapes():
    g7 = {p.name: (p.K, p.N, p.had_block) for p in inputs.llama2_7b_decode().projs}
    assert g7["q"] == (4096, 4096, 4096) and g7["gate"] == (4096, 11008, 4096) and g7["down"] == (11008, 4096, 256)
    g8 = {p.name: (p.K, p.N) for p in inputs.llama3_8b_prefill().projs}
    assert g8["k"] == (4096, 1024) and g8["down"] == (14336, 4096)
    g13 = {p.name: (p.K, p.N, p.had_block) for p in inputs.llama2_13b_prefill().projs}
    assert g13["down"] == (13824, 5120, 1024)                  # 13 x 1024 + a 512 tail
    g70 = {p.name: (p.K, p.N) for p in inputs.llama2_70b().projs}
    assert g70["gate"] == (8192, 28672) and g70["down"] == (28672, 8192)


def test_weights_distribution_seed_and_row_subsets():
    w = inputs.weights(512, 1024, layer=3, proj=2).astype(np.float64)
    assert abs(np.std(w) / 0.02 - 1.0) < 0.01 and abs(np.mean(w)) < 1e-3
    assert np.array_equal(inputs.weights(512, 1024, layer=3, proj=2), w.astype(np.float16))
    assert not np.array_equal(inputs.weights(512, 1024, layer=3, proj=1), w.astype(np.float16))
    rows = [5, 77, 400]
    assert np.array_equal(inputs.weights(512, 1024, 3, 2, rows=rows), w.astype(np.float16)[rows])
    assert inputs.weight_seed(3, 2) == 1 + 16 * 3 + 2


def test_fp16_saturation_and_random_codes():
    a = np.array([1e6, -1e6, 65504.0, 70000.0, 1.5], dtype=np.float32)
    h = inputs.to_f16(a)
    assert h.tolist() == [65504.0, -65504.0, 65504.0, 65504.0, 1.5]
    for bits, qmax in ((4, 7), (8, 127)):
        c = inputs.random_codes(64, 256, bits)
        assert c.min() >= -qmax and c.max() <= qmax and c.dtype == np.int8


@pytest.mark.parametrize("name", sorted(inputs.WORKLOADS))
def test_every_workload_draws_finite_fp16(name):
    wl = inputs.WORKLOADS[name]()
    K = wl.projs[0].K if wl.projs[0].K <= 4096 else 4096
    x = inputs.activations(wl, 8, K)
    assert x.dtype == np.float16 and x.shape == (8, K) and np.all(np.isfinite(x.astype(np.float32)))
