"""loip_k_attention_noalloc: the split-K attention for callers that cannot
allocate device memory (its partial states live in the library's own
file-scope device array).  Checked through the C ABI against the allocating
entry point, loip_k_attention, on calls in a row with different shapes (every
GQA ratio the kernel is built for, contexts crossing page boundaries), at the
largest problem the fixed array holds, and on refusals: a problem one page past
that size and a misaligned query, each with buffers sized to the declared shape.
Collected last so that a stop-at-first-failure run has run everything else."""
import numpy as np
import pytest

from gpu_util import U, dev_f32, need_gpu
from paper_2512_21835_gb300 import inputs

pytestmark = pytest.mark.gpu
P = 64


def _paged_inputs(torch, orc, Hq, Hkv, d, ctx, max_pages, seed):
    B = len(ctx)
    max_ctx = max_pages * P
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
    return (dev_f32(q), torch.from_numpy(host).cuda(), torch.from_numpy(pt).cuda(),
            dev_f32(np.asarray(ctx, dtype=np.int32)).int(), lpb, vmax)


def _compare(torch, L, orc, Hq, Hkv, d, ctx, max_pages, max_ctx, seed):
    q, kv, pt, cl, lpb, vmax = _paged_inputs(torch, orc, Hq, Hkv, d, ctx, max_pages, seed)
    B = len(ctx)
    scratch = torch.empty(L.loip_k_attention_scratch_floats(B, Hq, d, max_ctx, P), dtype=torch.float32,
                          device="cuda")
    o_ref = torch.empty(B, Hq * d, dtype=torch.float32, device="cuda")
    L.loip_k_attention(q, kv, pt, max_pages, cl, Hq, Hkv, d, P, 0, lpb, max_ctx, scratch, o_ref)
    o = torch.full((B, Hq * d), float("nan"), dtype=torch.float32, device="cuda")
    L.loip_k_attention_noalloc(q, kv, pt, max_pages, cl, Hq, Hkv, d, P, 0, lpb, max_ctx, o)
    torch.cuda.synchronize()
    got, want = o.cpu().numpy().astype(np.float64), o_ref.cpu().numpy().astype(np.float64)
    assert np.all(np.isfinite(got))
    for b in range(B):
        tol = (d + ctx[b] + 64) * U * 8.0 * vmax + 1e-6  # the attention tolerance of the parity tests
        assert np.max(np.abs(got[b] - want[b])) <= tol, (Hq, Hkv, d, b)
    return q, kv, pt, cl, lpb


def test_noalloc_attention_matches_allocating_entry_point(orc):
    torch = need_gpu()
    from paper_2512_21835_gb300 import loip as L
    # (Hq, Hkv, d, contexts, max_pages, seed): G = 8, 4, 1, 2 in a row, ragged
    # contexts on and across page boundaries
    cases = [(64, 8, 128, [1, 70, 200, 64], 4, 101), (8, 2, 64, [130, 5, 17], 3, 202),
             (4, 4, 64, [65, 128, 3], 3, 303), (8, 4, 128, [190, 1, 64, 129], 3, 404)]
    for Hq, Hkv, d, ctx, max_pages, seed in cases:
        _compare(torch, L, orc, Hq, Hkv, d, ctx, max_pages, max_pages * P, seed)


def test_noalloc_attention_at_the_scratch_limit_and_refusals(orc):
    torch = need_gpu()
    from paper_2512_21835_gb300 import loip as L
    B, Hq, Hkv, d, max_pages = 8, 64, 8, 128, 64
    # the largest context this shape can take in the fixed array: 63 pages
    at = 63 * P
    assert L.loip_k_attention_scratch_floats(B, Hq, d, at, P) <= L.NOALLOC_SCRATCH_FLOATS
    assert L.loip_k_attention_scratch_floats(B, Hq, d, at + 1, P) > L.NOALLOC_SCRATCH_FLOATS
    ctx = [at, 1, 4000, 64, 2017, at - 1, 700, 3000]
    q, kv, pt, cl, lpb = _compare(torch, L, orc, Hq, Hkv, d, ctx, max_pages, at, 505)
    o = torch.full((B, Hq * d), float("nan"), dtype=torch.float32, device="cuda")
    # one position more needs a 64th page of partial states: refused, and the
    # buffers (64 pages per request) are sized to that declared shape
    with pytest.raises(L.LoipError) as e:
        L.loip_k_attention_noalloc(q, kv, pt, max_pages, cl, Hq, Hkv, d, P, 0, lpb, at + 1, o)
    assert e.value.code == L.ERR_INVALID
    # a query 4 bytes off its 16-byte alignment: refused before any launch
    qbuf = torch.zeros(B * Hq * d + 4, dtype=torch.float32, device="cuda")
    q_off = qbuf[1:1 + B * Hq * d].view(B, Hq * d)
    assert q_off.data_ptr() % 16 == 4
    with pytest.raises(L.LoipError) as e:
        L.loip_k_attention_noalloc(q_off, kv, pt, max_pages, cl, Hq, Hkv, d, P, 0, lpb, at, o)
    assert e.value.code == L.ERR_INVALID
    torch.cuda.synchronize()
    assert torch.isnan(o).all()  # neither refused call wrote anything
