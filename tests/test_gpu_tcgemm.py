"""Parity of the tensor-core prefill GEMM (tcgen05 + TMA) through the C ABI:
x += A W^T against the oracle's fp64 products, with the fp32 summation bound
(K + 16) u sum|a||w| per output.  Shapes cover ragged M, N and K tails, the
tiny model's projections and a full 70B-layer-sized product (sampled rows); the
split-pair operand (fp32 activations as hi + lo bf16 planes) against the fp64
product of the fp32 activations."""
import numpy as np
import pytest

from gpu_util import dev_bits, dev_f32, dot_bound, need_gpu
from paper_2512_21835_gb300 import inputs

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("M,N,K,rows", [
    (1, 256, 256, None), (32, 512, 256, None), (62, 256, 688, None), (130, 1000, 4096, None),
    (300, 8192, 1024, [0, 1, 127, 128, 299]), (2048, 8192, 8192, [0, 127, 128, 1000, 2047])])
def test_tc_gemm_parity(orc, M, N, K, rows):
    torch = need_gpu()
    from paper_2512_21835_gb300 import loip as L
    A = inputs.bf16_bits(100 + M, (M, K), 1.0)
    W = orc.gen_tensor(7, 90, N * K, 0).reshape(N, K)
    x0 = inputs.normal_f32(200 + N, (M, N), 1.0)
    x = dev_f32(x0)
    L.loip_k_gemm_bf16(dev_bits(A), dev_bits(W), x)
    torch.cuda.synchronize()
    assert L.loip_k_tc_status() == 0
    got = x.cpu().numpy().astype(np.float64)
    W64 = orc.bf16_bits_to_f64(W)
    check = range(M) if rows is None else rows
    for m in check:
        a = orc.bf16_bits_to_f64(A[m])
        want = x0[m].astype(np.float64) + orc.gemv(W, K, a)
        tol = dot_bound(W64, a, K) + 4 * 2.0 ** -24 * np.abs(want)
        assert np.all(np.abs(got[m] - want) <= tol), (m, float(np.max(np.abs(got[m] - want) / tol)))


def _bf16_rne(x):
    """fp64 -> nearest bf16 value (ties to even), in fp64."""
    x = np.asarray(x, dtype=np.float64)
    _, e = np.frexp(x)
    ulp = np.ldexp(1.0, e - 8)
    return np.where(x == 0, 0.0, np.rint(x / ulp) * ulp)


def _bits(v64):
    return (v64.astype(np.float32).view(np.uint32) >> 16).astype(np.uint16)  # exact: v64 is a bf16 value


@pytest.mark.parametrize("M,N,K,rows", [
    (1, 256, 256, None), (62, 256, 688, None), (130, 1000, 4096, None), (300, 8192, 1024, [0, 1, 127, 128, 299]),
    (2048, 8192, 8192, [0, 127, 128, 1000, 2047])])
def test_tc_gemm_split_parity(orc, M, N, K, rows):
    """x += A W^T with A fp32 given as the pair (bf16(A), bf16(A - bf16(A))): within
    the fp32 summation bound plus the pair's residue sum |w| |A - hi - lo|, i.e.
    at fp32-activation accuracy (a single bf16 plane would be ~2^8 x further off)."""
    torch = need_gpu()
    from paper_2512_21835_gb300 import loip as L
    A = inputs.normal_f32(300 + M, (M, K), 1.0).astype(np.float64)
    hi = _bf16_rne(A)
    lo = _bf16_rne(A - hi)
    A2 = np.stack([_bits(hi), _bits(lo)])
    W = orc.gen_tensor(7, 91, N * K, 0).reshape(N, K)
    x0 = inputs.normal_f32(400 + N, (M, N), 1.0)
    x = dev_f32(x0)
    L.loip_k_gemm_split(dev_bits(A2), dev_bits(W), x)
    torch.cuda.synchronize()
    assert L.loip_k_tc_status() == 0
    got = x.cpu().numpy().astype(np.float64)
    W64 = orc.bf16_bits_to_f64(W)
    check = range(M) if rows is None else rows
    worst = 0.0
    for m in check:
        want = x0[m].astype(np.float64) + orc.gemv(W, K, A[m])
        resid = np.abs(W64) @ np.abs(A[m] - hi[m] - lo[m])
        tol = dot_bound(W64, A[m], K, extra=2 * K + 16) + resid + 4 * 2.0 ** -24 * np.abs(want)
        assert np.all(np.abs(got[m] - want) <= tol), (m, float(np.max(np.abs(got[m] - want) / tol)))
        # and far inside what one bf16 plane allows: the lo plane is really used
        worst = max(worst, float(np.max(np.abs(got[m] - want) / (np.abs(W64) @ np.abs(A[m] - hi[m]) + 1e-30))))
    assert worst < 0.25
