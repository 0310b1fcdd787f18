"""Parity of the tensor-core prefill GEMM (tcgen05 + TMA) through the C ABI:
x += A W^T against the oracle's fp64 products, with the fp32 summation bound
(K + 16) u sum|a||w| per output.  Shapes cover ragged M, N and K tails, the
tiny model's projections and a full 70B-layer-sized product (sampled rows)."""
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
