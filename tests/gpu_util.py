"""Helpers shared by the GPU parity tests (no method arithmetic here)."""
import numpy as np
import pytest

U = 2.0 ** -24  # fp32 unit roundoff


def need_gpu():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.fail("GPU test run without a CUDA device")
    from paper_2512_21835_gb300 import build
    build.build()
    return torch


def dev_bits(a: np.ndarray):
    """uint16 bf16 bit patterns -> contiguous int16 CUDA tensor (same bits)."""
    import torch
    return torch.from_numpy(np.ascontiguousarray(a).view(np.int16)).cuda()


def dev_f32(a: np.ndarray):
    import torch
    return torch.from_numpy(np.ascontiguousarray(a, dtype=np.float32)).cuda()


def dot_bound(W_f64: np.ndarray, y: np.ndarray, K: int, extra: int = 16) -> np.ndarray:
    """A-priori bound of an fp32 sum of K products: (K + extra) u sum |w||y|."""
    return (K + extra) * U * (np.abs(W_f64) @ np.abs(y))


def argmax_agrees(gpu_tok: int, gpu_logits: np.ndarray, ref_logits: np.ndarray) -> bool:
    """Greedy token parity: equal to the oracle's fp32 argmax (lowest index on
    ties), unless the oracle's top two are closer than 4x the largest logit
    error seen, in which case any token within that band of the top is valid."""
    ref32 = ref_logits.astype(np.float32)
    want = int(np.argmax(ref32))
    if gpu_tok == want:
        return True
    tau = 4.0 * float(np.max(np.abs(gpu_logits.astype(np.float64) - ref_logits)))
    return float(ref32[want]) - float(ref32[gpu_tok]) <= tau
