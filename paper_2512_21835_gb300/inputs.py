"""Seeded synthetic inputs shared by the tests, the bench and the oracle side.

Holds none of the method's arithmetic: only random token ids, context lengths
and test vectors drawn from numpy's PCG64 generator.  (Model weights are not
drawn here: each side implements the counter-based SplitMix64 generator from
its published definition.)
"""
import numpy as np


def token_ids(seed: int, n: int, vocab: int) -> np.ndarray:
    """n uniform token ids in [0, vocab), int32."""
    return np.random.default_rng(seed).integers(0, vocab, size=n, dtype=np.int64).astype(np.int32)


def prompts(seed: int, n_prompts: int, length: int, vocab: int) -> np.ndarray:
    """[n_prompts, length] uniform token ids."""
    return token_ids(seed, n_prompts * length, vocab).reshape(n_prompts, length)


def context_lengths(seed: int, batch: int, lo: int, hi: int) -> np.ndarray:
    """Per-request context lengths, uniform integers in [lo, hi]."""
    return np.random.default_rng(seed).integers(lo, hi + 1, size=batch, dtype=np.int64).astype(np.int32)


def normal_f32(seed: int, shape, scale: float = 1.0) -> np.ndarray:
    """fp32 test vector, N(0, scale^2)."""
    return (np.random.default_rng(seed).standard_normal(shape) * scale).astype(np.float32)


def bf16_bits(seed: int, shape, scale: float = 0.02) -> np.ndarray:
    """Random bf16 values (as uint16 bit patterns) of N(0, scale^2), truncated
    from fp32 -- any bf16 pattern is a valid input."""
    f = normal_f32(seed, shape, scale)
    return (f.view(np.uint32) >> 16).astype(np.uint16)


def batched_prompts(ctx_seed: int, tok_seed: int, batch: int, lo: int, hi: int, vocab: int):
    """Requests with context lengths uniform in [lo, hi] (seed ctx_seed), each a
    prompt of uniform token ids (seed tok_seed + request index)."""
    lens = context_lengths(ctx_seed, batch, lo, hi)
    return [token_ids(tok_seed + 1000 * (i + 1), int(n), vocab) for i, n in enumerate(lens)]
