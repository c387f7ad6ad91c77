"""Seeded synthetic inputs for the UniSVQ linear layer.

This module is the ONLY code shared by the CUDA path's tests/bench and the
CPU oracle. It draws random inputs and nothing else: it holds none of the
method's arithmetic (no dequantisation, no fold, no matmul).

Workload recipe (stand-in for the paper's Llama/Qwen layers, whose weights and
calibration data are not available):

* codes z: uint8 [N][K], each coordinate i.i.d. in {0,1,2,3} with
  probabilities (0.15, 0.35, 0.35, 0.15) (a rounded-Gaussian-like 2-bit
  lattice occupancy);
* affine (A, B), one per weight matrix (the paper attaches 20 parameters,
  a 4x4 A and a 4-vector B, to each weight matrix; Fig. 1 caption and
  Sec. 4.2): A = s (I + 0.1 G) with G ~ N(0,1)^{d x d} and s ~ |N(0.02, 0.005)|,
  B = -1.5 s 1; both stored as IEEE fp16 bit patterns;
* activations x: bf16 [M][K] drawn N(0,1) with a fixed 1% of the K channels
  scaled by 20 (outlier channels), stored as bf16 bit patterns (uint16).

Every stream is a numpy PCG64 generator seeded from (seed, *stream_ids), so a
given (config, layer, projection) always yields the same tensors.
"""
from __future__ import annotations

import numpy as np

CODE_PROBS = (0.15, 0.35, 0.35, 0.15)


def rng(seed: int, *stream) -> np.random.Generator:
    """Counter-free seeded generator for one named input stream."""
    return np.random.Generator(np.random.PCG64(np.random.SeedSequence([int(seed), *[int(s) for s in stream]])))


def gen_codes(g: np.random.Generator, N: int, K: int, probs=CODE_PROBS) -> np.ndarray:
    """uint8 [N][K] lattice coordinates in {0..3} drawn i.i.d. from `probs`.

    Drawn by thresholding 16-bit uniforms at the cumulative probabilities,
    which reproduces `probs` to within 2^-16.
    """
    cum = np.cumsum(np.asarray(probs, dtype=np.float64))[:-1]
    thr = np.round(cum * 65536.0).astype(np.uint32)
    out = np.empty((N, K), dtype=np.uint8)
    rows_per_chunk = max(1, (1 << 24) // max(K, 1))
    for r0 in range(0, N, rows_per_chunk):
        r1 = min(N, r0 + rows_per_chunk)
        u = g.integers(0, 65536, size=(r1 - r0, K), dtype=np.uint16)
        c = (u >= thr[0]).astype(np.uint8)
        c += u >= thr[1]
        c += u >= thr[2]
        out[r0:r1] = c
    return out


def gen_affine(g: np.random.Generator, d: int, s_mean: float = 0.02, s_std: float = 0.005,
               mix: float = 0.1):
    """(A, B) as fp16 arrays: A = s (I + mix*G), B = -1.5 s 1."""
    s = abs(g.normal(s_mean, s_std))
    G = g.standard_normal((d, d))
    A = (s * (np.eye(d) + mix * G)).astype(np.float16)
    B = np.full((d,), -1.5 * s).astype(np.float16)
    return A, B


def gen_affine_grouped(g: np.random.Generator, N: int, G: int, d: int, s_mean: float = 0.02,
                       s_std: float = 0.005, mix: float = 0.1):
    """(A [N][G][d][d], B [N][G][d]) fp16: one independent draw of the
    `gen_affine` distribution per (output row, column group)."""
    s = np.abs(g.normal(s_mean, s_std, size=(N, G)))
    Gm = g.standard_normal((N, G, d, d))
    A = (s[:, :, None, None] * (np.eye(d) + mix * Gm)).astype(np.float16)
    B = np.repeat((-1.5 * s)[:, :, None], d, axis=2).astype(np.float16)
    return A, B


def f32_to_bf16_bits(v: np.ndarray) -> np.ndarray:
    """Round fp32 values to bf16 (round to nearest even); returns uint16 bits."""
    v = np.ascontiguousarray(v, dtype=np.float32)
    u = v.view(np.uint32).astype(np.uint64)
    rounding = ((u >> 16) & 1) + 0x7FFF
    r = ((u + rounding) >> 16).astype(np.uint16)
    nan = np.isnan(v)
    if nan.any():
        r[nan] = 0x7FC0
    return r


def outlier_channels(K: int, seed: int = 0, frac: float = 0.01) -> np.ndarray:
    """Fixed seeded set of round(frac*K) channel indices (at least one)."""
    n = max(1, int(round(frac * K)))
    return np.sort(rng(seed, 0x0A11E5, K).permutation(K)[:n])


def gen_activations(g: np.random.Generator, M: int, K: int, outlier_frac: float = 0.01,
                    outlier_scale: float = 20.0, seed: int = 0) -> np.ndarray:
    """bf16 bits (uint16 [M][K]) of N(0,1) activations with outlier channels."""
    x = g.standard_normal((M, K), dtype=np.float32)
    if outlier_frac > 0 and K > 0:
        x[:, outlier_channels(K, seed, outlier_frac)] *= np.float32(outlier_scale)
    return f32_to_bf16_bits(x)


def layer_inputs(seed: int, config: int, layer: int, proj: int, N: int, K: int, d: int):
    """(codes, A, B) for one projection of one layer of a synthetic config."""
    gc = rng(seed, config, layer, proj, 1)
    ga = rng(seed, config, layer, proj, 2)
    codes = gen_codes(gc, N, K)
    A, B = gen_affine(ga, d)
    return codes, A, B


def layer_inputs_grouped(seed: int, config: int, layer: int, proj: int, N: int, K: int, d: int,
                         group_cols: int = 128):
    """(codes, A, B) with one affine map per (output row, `group_cols` input
    columns), for one projection of one layer of a synthetic config."""
    gc = rng(seed, config, layer, proj, 1)
    ga = rng(seed, config, layer, proj, 4)
    codes = gen_codes(gc, N, K)
    A, B = gen_affine_grouped(ga, N, -(-K // group_cols), d)
    return codes, A, B


# 3-bit codes: a unit Gaussian weight on the grid of Eq. (def:affine) with
# b = 3 (step s = sqrt(12/63), centre 3.5), probability of each of 0..7.
_Z3 = np.arange(8) - 3.5
_P3 = np.exp(-0.5 * (_Z3 * np.sqrt(12.0 / 63.0)) ** 2)
CODE_PROBS_3BIT = tuple(_P3 / _P3.sum())


def layer_inputs_bits(seed: int, config: int, layer: int, proj: int, N: int, K: int, d: int, bits: int):
    """(codes, A, B) with codes of `bits` bits: 2 as `layer_inputs`; 3 draws
    codes i.i.d. from CODE_PROBS_3BIT and centres B at (2^3 - 1)/2 = 3.5 steps."""
    if bits == 2:
        return layer_inputs(seed, config, layer, proj, N, K, d)
    gc = rng(seed, config, layer, proj, 5)
    ga = rng(seed, config, layer, proj, 6)
    codes = gc.choice(8, size=(N, K), p=CODE_PROBS_3BIT).astype(np.uint8)
    s = abs(ga.normal(0.02, 0.005)) / 2.0
    G = ga.standard_normal((d, d))
    A = (s * (np.eye(d) + 0.1 * G)).astype(np.float16)
    B = np.full((d,), -3.5 * s).astype(np.float16)
    return codes, A, B


def activations(seed: int, config: int, stream: int, M: int, K: int) -> np.ndarray:
    """bf16 bits [M][K] for one activation stream of a synthetic config."""
    return gen_activations(rng(seed, config, stream, 3), M, K, seed=seed)


# Projection shapes (out N, in K) of the synthetic workloads, after the public
# model shapes named in the workload descriptions.
LLAMA2_7B = [("q", 4096, 4096), ("k", 4096, 4096), ("v", 4096, 4096), ("o", 4096, 4096),
             ("gate", 11008, 4096), ("up", 11008, 4096), ("down", 4096, 11008)]
LLAMA3_8B = [("q", 4096, 4096), ("k", 1024, 4096), ("v", 1024, 4096), ("o", 4096, 4096),
             ("gate", 14336, 4096), ("up", 14336, 4096), ("down", 4096, 14336)]
LLAMA2_70B = [("q", 8192, 8192), ("k", 1024, 8192), ("v", 1024, 8192), ("o", 8192, 8192),
              ("gate", 28672, 8192), ("up", 28672, 8192), ("down", 8192, 28672)]
