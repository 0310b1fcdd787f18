"""Per-kernel parity: each fused CUDA kernel, called through the C ABI, against
the oracle on the same seeded inputs.  Floating-point tolerances are the
a-priori fp32 summation bound (K + c) u sum|w||y| derived from the arithmetic;
generator, embedding and argmax are compared exactly."""
import numpy as np
import pytest

from gpu_util import U, argmax_agrees, dev_bits, dev_f32, dot_bound, need_gpu
from paper_2512_21835_gb300 import inputs

pytestmark = pytest.mark.gpu
SEED = 0x10A1B


@pytest.fixture(scope="module")
def torch():
    return need_gpu()


@pytest.fixture(scope="module")
def L(torch):
    from paper_2512_21835_gb300 import loip
    return loip


def test_generator_bit_exact(torch, L, orc):
    for tid, kind, n, first in [(17, 0, 100_003, 0), (16, 1, 4096, 0), (1, 0, 50_000, 123_456_789),
                                (16 + 16 * 79 + 6, 0, 7, (1 << 32) + 5)]:
        out = torch.empty(n, dtype=torch.int16, device="cuda")
        L.loip_k_generate(out, first, SEED, tid, kind)
        got = out.cpu().numpy().view(np.uint16)
        want = orc.gen_tensor(SEED, tid, n, kind, first=first)
        assert np.array_equal(got, want), (tid, kind)


def test_embed_exact(torch, L, orc):
    V, H = 300, 520
    E = orc.gen_tensor(5, 1, V * H, 0).reshape(V, H)
    toks = np.array([0, 299, 17, 17, 100], dtype=np.int32)
    x = torch.empty(len(toks), H, dtype=torch.float32, device="cuda")
    L.loip_k_embed(dev_bits(E), dev_f32(toks).int(), x)
    assert np.array_equal(x.cpu().numpy().astype(np.float64), orc.bf16_bits_to_f64(E[toks]))


# batch 1: block-tile kernel up to 16384 gate + up rows, persistent kernel above (1, 512, 9000)
@pytest.mark.parametrize("B,H,F", [(1, 1000, 300), (3, 4096, 1000), (8, 2048, 700), (1, 13000, 64),
                                   (5, 4096, 129), (2, 256, 688), (1, 512, 9000)])
def test_gate_up_parity(torch, L, orc, B, H, F):
    eps = 1e-5
    x = inputs.normal_f32(B * 7 + H, (B, H), 1.5)
    g = orc.gen_tensor(SEED, 21, H, 1)
    Wg = orc.gen_tensor(SEED, 22, F * H, 0).reshape(F, H)
    Wu = orc.gen_tensor(SEED, 23, F * H, 0).reshape(F, H)
    a = torch.empty(B, F, dtype=torch.float32, device="cuda")
    L.loip_k_gate_up(dev_f32(x), dev_bits(g), dev_bits(Wg), dev_bits(Wu), eps, a)
    got = a.cpu().numpy().astype(np.float64)
    Wg64, Wu64 = orc.bf16_bits_to_f64(Wg), orc.bf16_bits_to_f64(Wu)
    for b in range(B):
        y = orc.rmsnorm(x[b].astype(np.float64), g, eps)
        gt, ut = orc.gemv(Wg, H, y), orc.gemv(Wu, H, y)
        want = np.array([orc.silu(v) for v in gt]) * ut
        dg, du = dot_bound(Wg64, y, H), dot_bound(Wu64, y, H)
        silu = want / np.where(ut == 0, 1, ut)
        tol = 1.1 * dg * np.abs(ut) + np.abs(silu) * du + dg * du + 8 * U * np.abs(want) + 1e-30
        assert np.all(np.abs(got[b] - want) <= tol), (b, np.max(np.abs(got[b] - want) / tol))


# batch 1: block-tile kernel up to 16384 rows, persistent kernel above (1, 17000, 256)
@pytest.mark.parametrize("B,N,K", [(1, 300, 1000), (2, 777, 4096), (8, 100, 14336), (1, 4096, 14336),
                                   (3, 513, 2048), (1, 256, 256), (1, 17000, 256)])
def test_residual_projection_parity(torch, L, orc, B, N, K):
    a = inputs.normal_f32(11 + K, (B, K), 0.7)
    x0 = inputs.normal_f32(12 + N, (B, N), 1.0)
    W = orc.gen_tensor(SEED, 40, N * K, 0).reshape(N, K)
    x = dev_f32(x0)
    L.loip_k_down(dev_f32(a), dev_bits(W), x)  # same kernel family as the o-projection
    got = x.cpu().numpy().astype(np.float64)
    W64 = orc.bf16_bits_to_f64(W)
    for b in range(B):
        want = x0[b].astype(np.float64) + orc.gemv(W, K, a[b].astype(np.float64))
        tol = dot_bound(W64, a[b].astype(np.float64), K) + 4 * U * np.abs(want)
        assert np.all(np.abs(got[b] - want) <= tol)
    # the o-projection entry point is the same product (at batch 1 its first-wave
    # blocks also prefetch the later tiles into L2: (1, 4096, 14336) has 512 tiles)
    x2 = dev_f32(x0)
    L.loip_k_oproj(dev_f32(a), dev_bits(W), x2)
    assert np.array_equal(x2.cpu().numpy(), x.cpu().numpy())


def _paged_cache(torch, n_pages, Hkv, P, d, seed):
    """One-layer paged cache with pages scattered in reverse order."""
    layer_page_bytes = 2 * Hkv * P * d * 2
    buf = torch.zeros(n_pages * layer_page_bytes + 4096, dtype=torch.uint8, device="cuda")
    order = np.random.default_rng(seed).permutation(n_pages)
    return buf, order, layer_page_bytes


# max_ctx 256: one cluster of 4 blocks per (request, kv head); 1088: 16 blocks
# of up to two pages each, some left without a page; 2112 (33 pages): split-K
# blocks with the last-block combine
@pytest.mark.parametrize("max_ctx,ctx_list", [(256, (1, 70, 200, 64)), (1088, (1, 700, 1088, 129)),
                                              (2112, (1, 2112, 999, 64))])
# G = Hq / Hkv from 1 to 8 at head_dim 64 and 128: with fewer than 512 outputs per kv
# head (G x d) the value sums are split over position groups
@pytest.mark.parametrize("Hq,Hkv,d", [(8, 2, 128), (4, 2, 64), (32, 8, 128), (64, 8, 128), (8, 8, 128),
                                      (4, 4, 64), (16, 4, 64)])
def test_attention_parity(torch, L, orc, Hq, Hkv, d, max_ctx, ctx_list):
    _attention_case(torch, L, orc, Hq, Hkv, d, max_ctx, ctx_list)


# the batched decode workload's shape: 8 requests, contexts up to 4096 + 256 decode
# steps (68 pages, the combine's sixteen-pages-in-flight loop runs five rounds),
# ragged on and off page boundaries; 70B heads (G = 8) and G = 2
@pytest.mark.parametrize("Hq,Hkv,d", [(64, 8, 128), (16, 8, 128)])
def test_attention_parity_batch8_many_pages(torch, L, orc, Hq, Hkv, d):
    _attention_case(torch, L, orc, Hq, Hkv, d, 4352, (4352, 128, 4097, 1, 2600, 64, 3333, 4290))


def _attention_case(torch, L, orc, Hq, Hkv, d, max_ctx, ctx_list):
    P = 64
    ctx = np.array(ctx_list, dtype=np.int32)
    B = len(ctx)
    max_pages = max_ctx // P
    n_pages = B * max_pages
    buf, order, lpb = _paged_cache(torch, n_pages, Hkv, P, d, 3)
    pt = (order.reshape(B, max_pages).astype(np.int64)) * lpb
    Kall = inputs.bf16_bits(31 + d, (B, max_ctx, Hkv, d), 1.0)
    Vall = inputs.bf16_bits(32 + d, (B, max_ctx, Hkv, d), 1.0)
    host = np.zeros(buf.numel(), dtype=np.uint8)
    for b in range(B):
        for pg in range(max_pages):
            base = pt[b, pg]
            kp = Kall[b, pg * P:(pg + 1) * P].transpose(1, 0, 2).copy()  # [Hkv][P][d]
            vp = Vall[b, pg * P:(pg + 1) * P].transpose(1, 0, 2).copy()
            host[base:base + kp.nbytes] = kp.view(np.uint8).ravel()
            host[base + kp.nbytes:base + 2 * kp.nbytes] = vp.view(np.uint8).ravel()
    buf.copy_(torch.from_numpy(host))
    q = inputs.normal_f32(33 + d, (B, Hq * d), 0.5)
    scratch = torch.empty(L.loip_k_attention_scratch_floats(B, Hq, d, max_ctx, P), dtype=torch.float32,
                          device="cuda")
    o = torch.empty(B, Hq * d, dtype=torch.float32, device="cuda")
    L.loip_k_attention(dev_f32(q), buf, torch.from_numpy(pt).cuda(), max_pages, dev_f32(ctx).int(), Hq, Hkv, d, P,
                       0, lpb, max_ctx, scratch, o)
    got = o.cpu().numpy().astype(np.float64)
    for b in range(B):
        T = ctx[b]
        K64 = orc.bf16_bits_to_f64(Kall[b, :T])
        V64 = orc.bf16_bits_to_f64(Vall[b, :T])
        want = orc.attention(q[b].reshape(Hq, d).astype(np.float64), K64, V64, Hkv).ravel()
        # softmax weights carry ~ (d + 8) u relative error through the scores; the
        # weighted sum adds T u; bound by the value magnitude
        tol = (d + T + 64) * U * 8.0 * np.max(np.abs(V64)) + 1e-6
        assert np.max(np.abs(got[b] - want)) <= tol, (b, np.max(np.abs(got[b] - want)), tol)


# one row (batch-1 decode) runs the block-tile kernel up to 8192 QKV rows and the
# persistent kernel above (64 x 128 query + 2 x 8 x 128 kv rows = 10240)
# "batch8": the batched decode shape, 8 rows at positions up to 4351 (68 pages)
@pytest.mark.parametrize("single", [False, True, "batch8"])
@pytest.mark.parametrize("Hq,Hkv,d,H", [(4, 2, 64, 256), (32, 8, 128, 4096), (8, 8, 128, 1024), (64, 8, 128, 1024)])
def test_qkv_rope_parity(torch, L, orc, Hq, Hkv, d, H, single):
    P, eps, theta = 64, 1e-5, 500000.0
    pos = np.array([0, 5, 130, 1000], dtype=np.int32)[: 3 if Hq == 8 else 4]
    if single is True:
        pos = np.array([1000], dtype=np.int32)
    elif single == "batch8":
        pos = np.array([4351, 0, 4096, 64, 2599, 127, 3333, 4289], dtype=np.int32)
    B = len(pos)
    max_pages = int(pos.max()) // P + 1
    buf, order, lpb = _paged_cache(torch, B * max_pages, Hkv, P, d, 4)
    pt = (order.reshape(B, max_pages).astype(np.int64)) * lpb
    x = inputs.normal_f32(41 + H, (B, H), 1.0)
    g = orc.gen_tensor(SEED, 50, H, 1)
    N = (Hq + 2 * Hkv) * d
    W = orc.gen_tensor(SEED, 51, N * H, 0).reshape(N, H)
    q = torch.empty(B, Hq * d, dtype=torch.float32, device="cuda")
    L.loip_k_qkv_rope(dev_f32(x), dev_bits(g), dev_bits(W), Hq, Hkv, d, eps, theta, dev_f32(pos).int(), q, buf,
                      torch.from_numpy(pt).cuda(), max_pages, P, 0, lpb)
    host = buf.cpu().numpy()
    gq = q.cpu().numpy().astype(np.float64)
    W64 = orc.bf16_bits_to_f64(W)
    for b in range(B):
        y = orc.rmsnorm(x[b].astype(np.float64), g, eps)
        raw = orc.gemv(W, H, y)
        bound = dot_bound(W64, y, H)
        qkv = raw.copy()
        for h in range(Hq + Hkv):
            qkv[h * d:(h + 1) * d] = orc.rope(raw[h * d:(h + 1) * d], int(pos[b]), theta)
        # rotation mixes the pair: bound of the pair, plus fp32 rotation rounding
        pb = bound.copy()
        for h in range(Hq + Hkv):
            blk = bound[h * d:(h + 1) * d]
            pb[h * d:(h + 1) * d] = np.concatenate([blk[: d // 2] + blk[d // 2:]] * 2)
        tol = pb + 8 * U * np.abs(raw).max()
        assert np.all(np.abs(gq[b] - qkv[: Hq * d]) <= tol[: Hq * d])
        page, t = pos[b] // P, pos[b] % P
        base = pt[b, page]
        kv = host[base:base + lpb].view(np.uint16).reshape(2, Hkv, P, d)[:, :, t, :]
        k_got = orc.bf16_bits_to_f64(kv[0]).ravel()
        v_got = orc.bf16_bits_to_f64(kv[1]).ravel()
        k_ref = qkv[Hq * d:(Hq + Hkv) * d]
        v_ref = qkv[(Hq + Hkv) * d:]
        # bf16 storage: within one bf16 ulp (2^-8 relative) plus the fp32 bound
        for got, ref, tl in ((k_got, k_ref, tol[Hq * d:(Hq + Hkv) * d]), (v_got, v_ref, tol[(Hq + Hkv) * d:])):
            assert np.all(np.abs(got - ref) <= 2.0 ** -8 * np.abs(ref) + tl)


@pytest.mark.parametrize("B,H,V", [(1, 256, 1024), (4, 4096, 1000), (3, 512, 128256)])
def test_lm_head_parity(torch, L, orc, B, H, V):
    eps = 1e-5
    x = inputs.normal_f32(61 + V, (B, H), 2.0)
    g = orc.gen_tensor(SEED, 3, H, 1)
    W = orc.gen_tensor(SEED, 2, V * H, 0).reshape(V, H)
    z = torch.empty(B, H, dtype=torch.float32, device="cuda")
    lg = torch.empty(B, V, dtype=torch.float32, device="cuda")
    tok = torch.empty(B, dtype=torch.int32, device="cuda")
    scratch = torch.empty(L.loip_k_lm_head_scratch_bytes(B, V), dtype=torch.uint8, device="cuda")
    L.loip_k_lm_head(dev_f32(x), dev_bits(g), dev_bits(W), eps, z, lg, tok, scratch)
    gz, glg, gt = z.cpu().numpy(), lg.cpu().numpy(), tok.cpu().numpy()
    W64 = orc.bf16_bits_to_f64(W)
    for b in range(B):
        zr = orc.rmsnorm(x[b].astype(np.float64), g, eps)
        assert np.max(np.abs(gz[b] - zr)) <= 16 * U * np.max(np.abs(zr))
        ref = orc.gemv(W, H, zr)
        assert np.all(np.abs(glg[b] - ref) <= dot_bound(W64, zr, H))
        assert argmax_agrees(int(gt[b]), glg[b], ref)
        # the token is the argmax of the logits the kernel wrote (lowest index on ties)
        assert int(gt[b]) == int(np.argmax(glg[b]))


def _split_to_f64(orc, o2):
    """[2, M, n] bf16 pair (hi, lo) -> fp64 hi + lo."""
    a = o2.cpu().numpy().view(np.uint16)
    return orc.bf16_bits_to_f64(a[0]) + orc.bf16_bits_to_f64(a[1])


# Tensor-core causal prefill attention: G = 8, 4, 2, 1 at d = 128 and 64; prompts of
# one row, several query tiles and page boundaries; the last prompt continues a
# request whose first 64 or 128 positions are already cached (first_pos > 0)
@pytest.mark.parametrize("Hq,Hkv,d", [(64, 8, 128), (16, 4, 64), (8, 4, 128), (4, 4, 64), (8, 2, 64), (4, 2, 64),
                                      (8, 1, 64), (4, 4, 128)])
@pytest.mark.parametrize("lens,first", [([1, 70, 200, 37], [0, 0, 0, 128]), ([32], [0])])
def test_prefill_attention_tc_parity(torch, L, orc, Hq, Hkv, d, lens, first):
    P = 64
    B = len(lens)
    max_pages = max(f + n for f, n in zip(first, lens)) // P + 1
    buf, order, lpb = _paged_cache(torch, B * max_pages, Hkv, P, d, 5)
    pt = (order.reshape(B, max_pages).astype(np.int64)) * lpb
    T = max_pages * P
    Kall = inputs.bf16_bits(71 + d, (B, T, Hkv, d), 1.0)
    Vall = inputs.bf16_bits(72 + d, (B, T, Hkv, d), 1.0)
    # positions past each request's last row hold no key yet: NaN there, which the
    # kernel must never let into a result
    for b in range(B):
        Kall[b, first[b] + lens[b]:] = 0x7FC0
        Vall[b, first[b] + lens[b]:] = 0x7FC0
    host = np.zeros(buf.numel(), dtype=np.uint8)
    for b in range(B):
        for pg in range(max_pages):
            base = pt[b, pg]
            kp = Kall[b, pg * P:(pg + 1) * P].transpose(1, 0, 2).copy()
            vp = Vall[b, pg * P:(pg + 1) * P].transpose(1, 0, 2).copy()
            host[base:base + kp.nbytes] = kp.view(np.uint8).ravel()
            host[base + kp.nbytes:base + 2 * kp.nbytes] = vp.view(np.uint8).ravel()
    buf.copy_(torch.from_numpy(host))
    M = sum(lens)
    q = inputs.normal_f32(73 + d, (M, Hq * d), 0.5)
    tiles = torch.empty((M + B) * 4, dtype=torch.int32, device="cuda")
    o2 = torch.full((2, M, Hq * d), -1, dtype=torch.int16, device="cuda")
    L.loip_k_prefill_attention(dev_f32(q), buf, torch.from_numpy(pt).cuda(), max_pages, lens, first, Hq, Hkv, d, P, 0,
                               lpb, tiles, o2)
    torch.cuda.synchronize()
    assert L.loip_k_attention_tc_status() == 0
    got = _split_to_f64(orc, o2)
    row = 0
    worst = 0.0
    for b in range(B):
        for i in range(lens[b]):
            pos = first[b] + i
            K64 = orc.bf16_bits_to_f64(Kall[b, :pos + 1])
            V64 = orc.bf16_bits_to_f64(Vall[b, :pos + 1])
            want = orc.attention(q[row].reshape(Hq, d).astype(np.float64), K64, V64, Hkv).ravel()
            vmax = np.max(np.abs(V64))
            # fp32 scores and sums as in decode, plus the split pairs' 2^-17 residues
            tol = (d + pos + 64) * U * 8.0 * vmax + 2.0 ** -15 * vmax + 1e-6
            err = np.max(np.abs(got[row] - want))
            worst = max(worst, err / tol)
            assert err <= tol, (b, i, err, tol)
            row += 1
    print("worst err / tol", worst)
