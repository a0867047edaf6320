"""Seeded synthetic inputs shared by the tests and the benchmark.

Holds random generators only -- none of the transfer's arithmetic -- so that
the CUDA path and the CPU oracle can be fed identical bytes without sharing
any of the method's code.

The value recipe follows the workloads this path serves: bf16 KV ~ N(0, 1)
from a fixed seed (the paper's request seed is 314159, Sec. 4.2), block tables
that scatter a context over a larger pool by a seeded random permutation, and
a poison byte for destination buffers so untouched bytes stay recognisable.
"""
from __future__ import annotations

import numpy as np

SEED = 314159
POISON = 0xA5


def rng(seed: int) -> np.random.Generator:
    return np.random.Generator(np.random.PCG64(seed))


def permuted_table(num_blocks: int, n_used: int, seed: int) -> np.ndarray:
    """n_used distinct page ids drawn from range(num_blocks) in seeded random order (int32)."""
    if n_used > num_blocks:
        raise ValueError("table longer than the pool")
    return rng(seed).permutation(num_blocks)[:n_used].astype(np.int32)


def random_bytes(n: int, seed: int) -> np.ndarray:
    """n uniformly random bytes (uint8)."""
    return rng(seed).integers(0, 256, size=n, dtype=np.uint8)


def normal_bf16_(tensor, seed: int):
    """Fill a tensor (any dtype, any device, byte size even) in place with bf16 ~ N(0,1) bit patterns."""
    import torch
    flat = tensor.view(torch.uint8).view(-1)
    assert flat.numel() % 2 == 0
    dst = flat.view(torch.bfloat16)
    g = torch.Generator(device=tensor.device)
    g.manual_seed(seed)
    step = 1 << 28  # elements per draw keeps the temporary bounded
    for start in range(0, dst.numel(), step):
        n = min(step, dst.numel() - start)
        dst[start:start + n].copy_(torch.randn(n, generator=g, device=tensor.device, dtype=torch.float32))
    return tensor


_GOLDEN = np.uint64(0x9E3779B97F4A7C15)


def splitmix64_bytes(n: int, seed: int) -> np.ndarray:
    """n bytes of the counter-based SplitMix64 stream (Steele, Lea & Flood, OOPSLA 2014).

    Output i is the SplitMix64 finaliser applied to seed + (i + 1) * 0x9E3779B97F4A7C15
    (mod 2^64), written little-endian.  Unlike library RNG streams it is fixed
    by its published definition, so stored fixtures stay valid across NumPy and
    PyTorch versions.
    """
    words = (n + 7) // 8
    with np.errstate(over="ignore"):
        z = np.uint64(seed) + (np.arange(1, words + 1, dtype=np.uint64) * _GOLDEN)
        z = (z ^ (z >> np.uint64(30))) * np.uint64(0xBF58476D1CE4E5B9)
        z = (z ^ (z >> np.uint64(27))) * np.uint64(0x94D049BB133111EB)
        z = z ^ (z >> np.uint64(31))
    return z.astype("<u8").view(np.uint8)[:n].copy()


def normal_bf16_bytes(n_elems: int, seed: int) -> np.ndarray:
    """Bytes of n_elems bf16 values distributed approximately N(0, 1), portably.

    Each value is an Irwin-Hall sum: 12 uniforms on (0, 1) from the SplitMix64
    stream (16 bits each, u -> (u + 1/2) / 2^16), minus 6, which has mean 0 and
    variance 1.  The sum is an integer over 2^16, exact in float32, and is
    rounded to bf16 (round to nearest, ties to even) with integer operations,
    so the bytes are the same on every machine and library version.
    """
    u = splitmix64_bytes(n_elems * 24, seed).view("<u2").reshape(n_elems, 12).astype(np.int64)
    k = u.sum(axis=1) - 393210          # sum of (u + 1/2) minus 6 * 2^16, over 2^16
    f32 = (k.astype(np.float32) / np.float32(65536.0)).view(np.uint32).astype(np.uint64)
    bf16 = ((f32 + 0x7FFF + ((f32 >> 16) & 1)) >> 16).astype("<u2")
    return bf16.view(np.uint8).copy()


def portable_table(num_blocks: int, n_used: int, seed: int) -> np.ndarray:
    """Like permuted_table, but fixed by the SplitMix64 definition: page ids in the
    order of num_blocks SplitMix64 words (stable sort), first n_used (int32)."""
    if n_used > num_blocks:
        raise ValueError("table longer than the pool")
    keys = splitmix64_bytes(8 * num_blocks, seed).view("<u8")
    return np.argsort(keys, kind="stable")[:n_used].astype(np.int32)
