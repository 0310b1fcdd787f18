"""loip_k_attention_noalloc: the split-K attention for callers that cannot
allocate device memory (its partial states live in the library's own
file-scope device array).  Checked through the C ABI against the allocating
entry point, loip_k_attention, on two calls in a row with different shapes.
Collected last so that a stop-at-first-failure run has run everything else."""
import numpy as np
import pytest

from gpu_util import U, dev_f32, need_gpu
from paper_2512_21835_gb300 import inputs

pytestmark = pytest.mark.gpu


def _paged_inputs(torch, orc, Hq, Hkv, d, ctx, max_ctx, seed):
    P = 64
    B = len(ctx)
    max_pages = max_ctx // P
    lpb = 2 * Hkv * P * d * 2
    order = np.random.default_rng(seed).permutation(B * max_pages)
    pt = order.reshape(B, max_pages).astype(np.int64) * lpb
    Kall = inputs.bf16_bits(seed + 1, (B, max_ctx, Hkv, d), 1.0)
    Vall = inputs.bf16_bits(seed + 2, (B, max_ctx, Hkv, d), 1.0)
    host = np.zeros(B * max_pages * lpb, dtype=np.uint8)
    for b in range(B):
        for pg in range(max_pages):
            base = pt[b, pg]
            kp = Kall[b, pg * P:(pg + 1) * P].transpose(1, 0, 2).copy()
            vp = Vall[b, pg * P:(pg + 1) * P].transpose(1, 0, 2).copy()
            host[base:base + kp.nbytes] = kp.view(np.uint8).ravel()
            host[base + kp.nbytes:base + 2 * kp.nbytes] = vp.view(np.uint8).ravel()
    q = inputs.normal_f32(seed + 3, (B, Hq * d), 0.5)
    vmax = float(np.max(np.abs(orc.bf16_bits_to_f64(Vall))))
    return (dev_f32(q), torch.from_numpy(host).cuda(), torch.from_numpy(pt).cuda(), max_pages,
            dev_f32(np.asarray(ctx, dtype=np.int32)).int(), P, lpb, vmax)


def test_noalloc_attention_matches_allocating_entry_point(orc):
    torch = need_gpu()
    from paper_2512_21835_gb300 import loip as L
    cases = [(64, 8, 128, [1, 70, 200, 64], 256, 101), (8, 2, 64, [130, 5, 17], 192, 202)]
    for Hq, Hkv, d, ctx, max_ctx, seed in cases:  # two calls in a row, different shapes
        q, kv, pt, max_pages, cl, P, lpb, vmax = _paged_inputs(torch, orc, Hq, Hkv, d, ctx, max_ctx, seed)
        B = len(ctx)
        scratch = torch.empty(L.loip_k_attention_scratch_floats(B, Hq, d, max_ctx, P), dtype=torch.float32,
                              device="cuda")
        o_ref = torch.empty(B, Hq * d, dtype=torch.float32, device="cuda")
        L.loip_k_attention(q, kv, pt, max_pages, cl, Hq, Hkv, d, P, 0, lpb, max_ctx, scratch, o_ref)
        o = torch.full((B, Hq * d), float("nan"), dtype=torch.float32, device="cuda")
        L.loip_k_attention_noalloc(q, kv, pt, max_pages, cl, Hq, Hkv, d, P, 0, lpb, max_ctx, o)
        torch.cuda.synchronize()
        got, want = o.cpu().numpy().astype(np.float64), o_ref.cpu().numpy().astype(np.float64)
        for b in range(B):
            tol = (d + ctx[b] + 64) * U * 8.0 * vmax + 1e-6  # the attention tolerance of the parity tests
            assert np.max(np.abs(got[b] - want[b])) <= tol
    # a problem larger than the fixed scratch is refused, not run
    q = torch.zeros(8, 64 * 128, dtype=torch.float32, device="cuda")
    with pytest.raises(L.LoipError) as e:
        L.loip_k_attention_noalloc(q, kv, pt, 128, cl, 64, 8, 128, 64, 0, lpb, 8192,
                                   torch.empty_like(q))
    assert e.value.code == L.ERR_INVALID
