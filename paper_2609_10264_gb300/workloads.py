"""Seeded synthetic inputs for tests and benchmarks.

This module only draws random arrays (numpy PCG64 seeded generators); it holds
none of the pvMVMD arithmetic, so both the CUDA path and the oracle can be fed
from it.  Shapes follow LLM projection layers; weights stand in for int8
quantised model weights (the paper quantises FP8 weights to integers, Sec.
7.2.1; real weights are not used).
"""
from __future__ import annotations

import numpy as np

Q = 2013265921

# Projection shapes (m, K) of one decoder layer.
LAYER_8B = {"q": (4096, 4096), "k": (1024, 4096), "v": (1024, 4096), "o": (4096, 4096),
            "gate": (14336, 4096), "up": (14336, 4096), "down": (4096, 14336)}
LAYER_70B = {"q": (8192, 8192), "kv": (1024, 8192), "gate_up": (28672, 8192), "down": (8192, 28672)}
# Qwen3-4B transformer block (the paper's evaluation model, Sec. 7.3 table
# of projection dimensions), as (output m, input K); weights stay synthetic
LAYER_QWEN3_4B = {"q": (4096, 2560), "k": (1024, 2560), "v": (1024, 2560), "o": (2560, 4096),
                  "gate": (9728, 2560), "up": (9728, 2560), "down": (2560, 9728)}


def _rng(seed) -> np.random.Generator:
    return np.random.default_rng(np.random.SeedSequence(seed))


def weights_uniform(m: int, K: int, seed) -> np.ndarray:
    """int8 m x K, uniform in [-127, 127]."""
    return _rng(seed).integers(-127, 128, size=(m, K), dtype=np.int8)


def weights_gaussian(m: int, K: int, seed, sigma: float = 32.0) -> np.ndarray:
    """int8 m x K: a Gaussian with standard deviation sigma, rounded and
    clipped to [-127, 127]."""
    out = np.empty((m, K), dtype=np.int8)
    rng = _rng(seed)
    step = max(1, (1 << 24) // max(K, 1))  # generate in row blocks to bound memory
    for r0 in range(0, m, step):
        r1 = min(m, r0 + step)
        g = rng.standard_normal(size=(r1 - r0, K), dtype=np.float32) * np.float32(sigma)
        np.clip(np.rint(g), -127, 127, out=g)
        out[r0:r1] = g.astype(np.int8)
    return out


def int8_vectors(B: int, K: int, seed) -> np.ndarray:
    """B x K signed integers uniform in [-127, 127] (int64), before embedding."""
    return _rng(seed).integers(-127, 128, size=(B, K), dtype=np.int64)


def field_vectors(B: int, K: int, seed) -> np.ndarray:
    """B x K uint32 uniform in [0, q)."""
    return _rng(seed).integers(0, Q, size=(B, K), dtype=np.uint32)
