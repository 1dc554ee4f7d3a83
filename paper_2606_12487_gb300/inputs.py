"""Seeded synthetic inputs for the quantized-linear workloads.

This module holds no quantization, rotation or GEMM arithmetic: it only draws
activations, weights and per-layer bit masks with the shapes and value structure of
the LLaMA projection workloads (massive-activation outlier channels, Section 1 and
Section 2 "Massive Activations"; per-layer 4/8-bit masks, Section 3.3 Algorithm 1
step 2).  Both the CUDA path's tests and the oracle's tests draw from here.

Seeds: activations 0, weights 1 + 16 * layer + projection index, masks and outlier
choices 1234.  Values are drawn in fp32 and cast to fp16 with saturation to +-65504.
"""
from __future__ import annotations

from dataclasses import dataclass, field

import numpy as np

ACT_SEED = 0
MASK_SEED = 1234
FP16_MAX = 65504.0
W_STD = 0.02


def weight_seed(layer: int, proj: int) -> int:
    return 1 + 16 * layer + proj


def to_f16(a: np.ndarray) -> np.ndarray:
    return np.clip(a, -FP16_MAX, FP16_MAX).astype(np.float16)


@dataclass(frozen=True)
class Proj:
    """One quantized linear of a transformer layer: K inputs -> N outputs."""
    name: str
    K: int
    N: int
    had_block: int
    group: str          # projections of one group share the same quantized input


@dataclass
class Workload:
    name: str
    layers: int
    projs: tuple
    mask_a8: tuple       # 0-indexed layers that run 8-bit activations
    act_kind: str        # "gauss_channels" | "gauss_tokens" | "student_t" | "gauss_first_token"
    outlier_scale: float = 1.0
    outlier_channels: int = 0
    outlier_token_frac: float = 0.0
    seq_len: int = 2048
    m_values: tuple = field(default_factory=tuple)

    def bits(self, layer: int) -> int:
        return 8 if layer in self.mask_a8 else 4

    def groups(self):
        """Projections grouped by shared input, in execution order."""
        out = []
        for p in self.projs:
            if not out or out[-1][0] != p.group:
                out.append((p.group, []))
            out[-1][1].append(p)
        return out


def _seeded_mask(layers: int, count: int) -> tuple:
    rng = np.random.default_rng(MASK_SEED)
    return tuple(sorted(int(v) for v in rng.choice(layers, count, replace=False)))


def llama2_7b_decode() -> Workload:
    d, f = 4096, 11008
    projs = (Proj("q", d, d, 4096, "qkv"), Proj("k", d, d, 4096, "qkv"),
             Proj("v", d, d, 4096, "qkv"), Proj("o", d, d, 4096, "o"),
             Proj("gate", d, f, 4096, "gateup"), Proj("up", d, f, 4096, "gateup"),
             Proj("down", f, d, 256, "down"))
    return Workload("llama2-7b-decode", 32, projs, (0, 1, 30, 31), "gauss_channels",
                    outlier_scale=100.0, outlier_channels=4, m_values=(1, 8, 32))


def llama3_8b_prefill() -> Workload:
    d, kv, f = 4096, 1024, 14336
    projs = (Proj("q", d, d, 2048, "qkv"), Proj("k", d, kv, 2048, "qkv"),
             Proj("v", d, kv, 2048, "qkv"), Proj("o", d, d, 2048, "o"),
             Proj("gate", d, f, 2048, "gateup"), Proj("up", d, f, 2048, "gateup"),
             Proj("down", f, d, 2048, "down"))
    return Workload("llama3-8b-prefill", 32, projs, _seeded_mask(32, 6), "gauss_tokens",
                    outlier_scale=300.0, outlier_channels=3, outlier_token_frac=0.01,
                    m_values=(2048,))


def llama2_13b_prefill() -> Workload:
    d, f = 5120, 13824
    projs = (Proj("q", d, d, 1024, "qkv"), Proj("k", d, d, 1024, "qkv"),
             Proj("v", d, d, 1024, "qkv"), Proj("o", d, d, 1024, "o"),
             Proj("gate", d, f, 1024, "gateup"), Proj("up", d, f, 1024, "gateup"),
             Proj("down", f, d, 1024, "down"))
    return Workload("llama2-13b-prefill", 40, projs, (0, 1, 2, 38, 39), "student_t",
                    m_values=(4096,))


def llama2_70b() -> Workload:
    d, kv, f = 8192, 1024, 28672
    projs = (Proj("q", d, d, 4096, "qkv"), Proj("k", d, kv, 4096, "qkv"),
             Proj("v", d, kv, 4096, "qkv"), Proj("o", d, d, 4096, "o"),
             Proj("gate", d, f, 4096, "gateup"), Proj("up", d, f, 4096, "gateup"),
             Proj("down", f, d, 4096, "down"))
    return Workload("llama2-70b", 80, projs, _seeded_mask(80, 8), "gauss_first_token",
                    outlier_scale=1000.0, outlier_channels=2, m_values=(1, 64, 512, 8192))


def single_linear() -> Workload:
    return Workload("single-256x512", 1, (Proj("lin", 256, 512, 256, "lin"),), (), "fixed_channels",
                    outlier_scale=50.0, m_values=(16,))


WORKLOADS = {w().name: w for w in (single_linear, llama2_7b_decode, llama3_8b_prefill,
                                   llama2_13b_prefill, llama2_70b)}


def outlier_channels(K: int, count: int) -> np.ndarray:
    rng = np.random.default_rng(MASK_SEED)
    return np.sort(rng.choice(K, count, replace=False))


def activations(wl: Workload, M: int, K: int, seed: int = ACT_SEED,
                row_offset: int = 0) -> np.ndarray:
    """fp16 [M, K] activations with the workload's outlier structure.

    ``row_offset`` places the rows at token positions row_offset.. of the sequence, so a
    sample of rows reproduces exactly what the full matrix holds at those positions.
    """
    rng = np.random.default_rng(seed)
    if row_offset:
        # draw the full prefix so that sampled rows equal the full draw at those tokens
        full = rng.standard_t(3, size=(row_offset + M, K)) if wl.act_kind == "student_t" \
            else rng.standard_normal((row_offset + M, K), dtype=np.float32)
        x = np.asarray(full[row_offset:], dtype=np.float32)
    elif wl.act_kind == "student_t":
        x = rng.standard_t(3, size=(M, K)).astype(np.float32)
    else:
        x = rng.standard_normal((M, K), dtype=np.float32)
    tok = np.arange(row_offset, row_offset + M)
    if wl.act_kind == "fixed_channels":
        x[:, [3, 77]] *= wl.outlier_scale
    elif wl.act_kind == "gauss_channels":
        x[:, outlier_channels(K, wl.outlier_channels)] *= wl.outlier_scale
    elif wl.act_kind == "gauss_tokens":
        rng_t = np.random.default_rng(MASK_SEED)
        n_tok = max(1, int(round(wl.outlier_token_frac * 2048)))
        hot = set(int(t) for t in rng_t.choice(2048, n_tok, replace=False))
        ch = outlier_channels(K, wl.outlier_channels)
        rows = [i for i, t in enumerate(tok) if int(t) % 2048 in hot]
        if rows:
            x[np.ix_(rows, ch)] *= wl.outlier_scale
    elif wl.act_kind == "gauss_first_token":
        ch = outlier_channels(K, wl.outlier_channels)
        rows = [i for i, t in enumerate(tok) if int(t) % wl.seq_len == 0]
        if rows:
            x[np.ix_(rows, ch)] *= wl.outlier_scale
    return to_f16(x)


def weights(N: int, K: int, layer: int = 0, proj: int = 0, rows=None) -> np.ndarray:
    """fp16 [N, K] weights ~ N(0, 0.02^2).  ``rows`` selects a subset of output channels
    (drawn from the same full matrix)."""
    rng = np.random.default_rng(weight_seed(layer, proj))
    w = rng.standard_normal((N, K), dtype=np.float32) * np.float32(W_STD)
    if rows is not None:
        w = w[np.asarray(rows)]
    return to_f16(w)


def random_codes(M: int, K: int, bits: int, seed: int = 7) -> np.ndarray:
    """Uniform integer codes in the symmetric range, for GEMM-only tests and timing."""
    qmax = (1 << (bits - 1)) - 1
    rng = np.random.default_rng(seed)
    return rng.integers(-qmax, qmax + 1, size=(M, K), dtype=np.int8)


def torch_weights(N: int, K: int, layer: int, proj: int, device):
    """Device-side fp16 weights N(0, 0.02^2) from a seeded torch generator (large stacks)."""
    import torch
    g = torch.Generator(device=device)
    g.manual_seed(weight_seed(layer, proj))
    w = torch.randn((N, K), generator=g, device=device, dtype=torch.float32) * W_STD
    return w.clamp_(-FP16_MAX, FP16_MAX).to(torch.float16)
